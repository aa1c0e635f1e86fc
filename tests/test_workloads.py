"""The synthetic-input recipe hits the acceptance levels the workloads name."""
import numpy as np

from oracle import softmax
from workloads import config_shape, make_batch, offsets, philox_uniforms


def test_uniforms_are_exact_fp32_in_open_interval_and_keyed():
    u = philox_uniforms(0, 3, 10_000)
    assert u.dtype == np.float32 and u.min() > 0 and u.max() < 1
    assert np.all(u.astype(np.float64) * 2 ** 23 % 1 == 0.5)
    np.testing.assert_array_equal(u, philox_uniforms(0, 3, 10_000))
    assert not np.array_equal(u, philox_uniforms(0, 4, 10_000))
    assert abs(u.mean() - 0.5) < 0.01


def test_acceptance_calibration_per_user():
    """sum_v min(p, q) per draft row lands within 0.01 of the user's alpha."""
    alpha = np.array([0.5, 0.7, 0.9])
    from workloads import sigma_for_alpha
    b = make_batch([2, 2, 2], [16, 16, 16], Hq=8, Hkv=1, D=16, V=151936, logit_std=1.0,
                   noise_sigma=sigma_for_alpha(alpha), alpha=alpha, seed=7)
    p = softmax(b.target_logits.double().numpy())
    q = softmax(b.draft_logits.double().numpy())
    qo, lo = offsets(b.T), offsets(b.L)
    for i in range(3):
        acc = [np.minimum(p[qo[i] + t], q[lo[i] + t]).sum() for t in range(b.L[i])]
        assert abs(np.mean(acc) - alpha[i]) < 0.01, (i, acc)


def test_workload_shapes():
    s = config_shape(3)
    assert s["L"].min() >= 0 and s["L"].max() <= 10
    assert s["ctx"].min() >= 512 and s["ctx"].max() <= 8192
    s = config_shape(4)
    assert np.all(s["ctx"] == 32768) and s["L"].min() >= 2 and s["L"].max() <= 6
    s = config_shape(5)
    assert len(s["L"]) == 128 and s["L"].min() >= 1 and s["L"].max() <= 10


def test_block_tables_scatter_pages_and_mark_unused():
    b = make_batch([1, 5, 0], [40, 3, 17], Hq=4, Hkv=1, D=8, V=32, seed=2)
    bt = b.block_table.numpy()
    used = bt[bt >= 0]
    assert len(np.unique(used)) == len(used)          # no page shared
    for i, n in enumerate(b.kv_len):
        pages = -(-int(n) // 16)
        assert np.all(bt[i, :pages] >= 0) and np.all(bt[i, pages:] == -1)
