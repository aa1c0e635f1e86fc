"""The in-kernel Philox4x64-10 against numpy's (an independent implementation of
the same published generator, Salmon et al., SC 2011), bit for bit.

The verification kernels draw their uniforms from this generator; the oracle
reads uniforms that numpy's Philox produced (workloads.philox_uniforms).  So
the pin is: the device words equal numpy's words on over a million counter
blocks, and the device's (u_acc, u_res) pairs equal the generator's host
copies exactly.
"""
import numpy as np
import pytest
import torch

from workloads import make_batch, make_config, philox_uniforms

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed,uid", [(0, 0), (0, 7), (12345, 3), (2 ** 63 + 17, 2 ** 31 - 1)])
def test_device_words_equal_numpy_philox(cuda_lib, seed, uid):
    n_blocks = 1 << 18  # 262144 counter blocks per stream, 1,048,576 over the four streams
    got = cuda_lib.dipsd_philox_words(seed, uid, n_blocks)
    torch.cuda.synchronize()
    got = got.cpu().numpy().view(np.uint64)
    ref = np.random.Philox(key=np.array([seed, uid], dtype=np.uint64)).random_raw(4 * n_blocks)
    mism = np.flatnonzero(got != ref)
    assert mism.size == 0, f"{mism.size} words differ, first at {mism[:4].tolist()}"


def test_keys_give_distinct_streams(cuda_lib):
    a = cuda_lib.dipsd_philox_words(5, 1, 1024).cpu()
    b = cuda_lib.dipsd_philox_words(5, 2, 1024).cpu()
    c = cuda_lib.dipsd_philox_words(6, 1, 1024).cpu()
    assert not torch.equal(a, b) and not torch.equal(a, c)


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_verify_uniforms_equal_the_generators(cuda_lib, cfg):
    b = make_config(cfg, seed=3, spec_only=True)
    got = cuda_lib.dipsd_verify_uniforms(b.L, b.user_ids, b.seed).cpu().numpy()
    assert got.dtype == np.float32
    np.testing.assert_array_equal(got, b.uniforms.numpy())


def test_verify_uniforms_ragged_ids_and_max_draft(cuda_lib):
    rng = np.random.default_rng(4)
    L = rng.integers(0, 32, size=300)
    uid = rng.permutation(100000)[:300]
    b = make_batch(L, np.zeros_like(L), Hq=8, Hkv=1, D=64, V=16, seed=99, user_ids=uid, spec_only=True)
    got = cuda_lib.dipsd_verify_uniforms(b.L, b.user_ids, b.seed).cpu().numpy()
    np.testing.assert_array_equal(got, b.uniforms.numpy())
    # exact fp32 values (k + 1/2) 2^-23 in (0, 1)
    k = got.astype(np.float64) * 2.0 ** 23 - 0.5
    assert np.all(k == np.round(k)) and got.min() > 0 and got.max() < 1
    # position t of user i takes words 2t and 2t+1 of its stream
    i = 17
    q0 = int((b.L[:i] + 1).sum())
    ref = philox_uniforms(b.seed, int(uid[i]), 2 * (int(b.L[i]) + 1)).reshape(-1, 2)
    np.testing.assert_array_equal(got[q0:q0 + int(b.L[i]) + 1], ref)
