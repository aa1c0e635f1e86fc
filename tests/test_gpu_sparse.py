"""dipsd_spec_verify_sparse (sparse draft payload) through the C ABI vs
oracle.spec_verify_sparse, with the same parity reading as the dense path."""
import dataclasses

import numpy as np
import pytest
import scipy.special
import torch

import oracle
from parity import check_spec
from workloads import make_batch, make_config, make_sparse_draft

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _run(dipsd, b, sd, ws=None):
    g = lambda t: t.to(DEV)
    res = dipsd.dipsd_spec_verify_sparse(b.L, b.user_ids, b.seed, g(b.target_logits), g(sd.draft_tokens),
                                         g(sd.draft_logq), g(sd.topk_idx), g(sd.topk_q), ws=ws)
    torch.cuda.synchronize()
    return res


def _check(b, sd, res):
    ref = oracle.spec_verify_sparse(b.L, b.target_logits.double().numpy(), sd.draft_tokens.numpy(),
                                    sd.draft_logq.numpy(), sd.topk_idx.numpy(), sd.topk_q.numpy(), b.uniforms.numpy())
    bs = dataclasses.replace(b, draft_tokens=sd.draft_tokens)
    return check_spec(bs, *res, ref=ref)


@pytest.mark.parametrize("cfg,K", [(1, 8), (2, 64), (2, 1), (3, 16)])
def test_sparse_workloads(cuda_lib, cfg, K):
    b = make_config(cfg, seed=1, spec_only=True)
    sd = make_sparse_draft(b, K, seed=cfg)
    print(f"workload {cfg} K={K}: {_check(b, sd, _run(cuda_lib, b, sd))}")


def test_sparse_ragged_lengths(cuda_lib):
    """L = 0 users (bonus only), long drafts, V not a multiple of the segment size."""
    b = make_batch([0, 7, 0, 31, 2], [0] * 5, Hq=8, Hkv=1, D=64, V=32008, logit_std=2.0, seed=51, spec_only=True)
    sd = make_sparse_draft(b, 32, seed=5, rank_noise=0.3)
    _check(b, sd, _run(cuda_lib, b, sd))


def test_sparse_full_table_matches_dense_reading(cuda_lib):
    """A table over the whole (small) vocabulary holding q = softmax(w): the
    sparse path and the dense path agree with their oracles on the same inputs."""
    b = make_batch([3, 5, 0, 2], [0] * 4, Hq=8, Hkv=1, D=64, V=64, logit_std=1.0, noise_sigma=0.5, seed=52,
                   spec_only=True, logit_dtype="f32")
    w = b.draft_logits.double().numpy()
    q = scipy.special.softmax(w, axis=-1)
    d = b.draft_tokens.numpy()
    sd = dataclasses.replace(make_sparse_draft(b, 8, seed=6),
                             topk_idx=torch.from_numpy(np.tile(np.arange(64, dtype=np.int32), (len(w), 1))),
                             topk_q=torch.from_numpy(q.astype(np.float32)),
                             draft_tokens=b.draft_tokens.clone(),
                             draft_logq=torch.from_numpy(np.log(q[np.arange(len(w)), d]).astype(np.float32)))
    _check(b, sd, _run(cuda_lib, b, sd))


def test_sparse_flags_table_entries_outside_the_vocabulary(cuda_lib):
    b = make_batch([2, 3], [0, 0], Hq=8, Hkv=1, D=64, V=4096, seed=53, spec_only=True)
    sd = make_sparse_draft(b, 4, seed=7)
    sd.topk_idx[0, 3] = 4096 + 9  # out of range: ignored, flagged
    ws = cuda_lib.workspace(cuda_lib.dipsd_spec_verify_sparse_workspace_size(b.L, b.V), DEV)
    _run(cuda_lib, b, sd, ws=ws)
    assert cuda_lib.device_status(ws) & cuda_lib.DEVERR_BAD_TOKEN
