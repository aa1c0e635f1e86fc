"""spec_verify through the C ABI vs the fp64 oracle, on the workloads and edge cases."""
import math

import numpy as np
import pytest
import scipy.stats
import torch

from parity import check_spec, valid_spec_outputs
from workloads import make_batch, make_config

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _run(dipsd, b, stream=None):
    g = lambda t: t.to(DEV)
    out = dipsd.dipsd_spec_verify(b.L, b.user_ids, b.seed, g(b.target_logits), g(b.draft_logits),
                                  g(b.draft_tokens), stream=stream)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_spec_verify_workloads(cuda_lib, cfg):
    b = make_config(cfg, seed=0)
    stats = check_spec(b, *_run(cuda_lib, b))
    print(f"workload {cfg}: {stats}")


def test_spec_verify_long_context_workload(cuda_lib):
    b = make_config(4, seed=0, spec_only=True)
    stats = check_spec(b, *_run(cuda_lib, b))
    print(f"workload 4 (spec): {stats}")


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_spec_verify_many_positions(cuda_lib, seed):
    """A few thousand positions over a mid-size vocabulary (several slices, ragged L)."""
    rng = np.random.default_rng(seed)
    L = rng.integers(0, 16, size=160)
    b = make_batch(L, np.zeros_like(L), Hq=8, Hkv=1, D=64, V=32000 + 8 * seed, logit_std=2.0,
                   noise_sigma=0.8, seed=seed)
    stats = check_spec(b, *_run(cuda_lib, b))
    print(stats)


def test_spec_verify_all_bonus(cuda_lib):
    """L_i = 0 for every user: a plain autoregressive step, one token from p each."""
    b = make_batch([0] * 7, [3] * 7, Hq=8, Hkv=1, D=64, V=50000, logit_std=1.5, seed=4)
    acc, offs, toks, probs = _run(cuda_lib, b)
    check_spec(b, acc, offs, toks, probs)
    assert acc.sum().item() == 0 and offs[-1].item() == 7


def test_spec_verify_max_draft_and_unaligned_vocab(cuda_lib):
    """L = 31 (one full warp ballot) and V not a multiple of 8 (scalar path)."""
    b = make_batch([31, 5, 0, 31], [0] * 4, Hq=8, Hkv=1, D=64, V=1001, logit_std=1.0, noise_sigma=0.3, seed=5)
    check_spec(b, *_run(cuda_lib, b))


def test_spec_verify_fp32_logits(cuda_lib):
    b = make_batch([3, 1, 7], [0] * 3, Hq=8, Hkv=1, D=64, V=20000, logit_dtype="f32", logit_std=1.0,
                   noise_sigma=0.6, seed=6)
    check_spec(b, *_run(cuda_lib, b))


def test_spec_verify_many_users(cuda_lib):
    """B = 500 users (the large parameter block) over a small vocabulary."""
    rng = np.random.default_rng(7)
    L = rng.integers(0, 6, size=500)
    b = make_batch(L, np.zeros_like(L), Hq=8, Hkv=1, D=64, V=256, logit_std=1.0, noise_sigma=0.8, seed=7)
    check_spec(b, *_run(cuda_lib, b))


def test_spec_verify_identical_and_disjoint(cuda_lib):
    b = make_batch([4, 4], [0, 0], Hq=8, Hkv=1, D=64, V=4096, logit_std=1.0, noise_sigma=0.5, seed=8)
    # user 0: draft logits equal the target logits -> every draft accepted, bonus from p
    z = b.target_logits.clone()
    w = b.draft_logits.clone()
    w[0:4] = z[0:4]
    # user 1: disjoint supports -> the first draft is always rejected, residual = p
    V = b.V
    w[4:8] = -1e4
    w[4:8, : V // 2] = 0
    z[5:10, : V // 2] = -1e4
    d = b.draft_tokens.clone()
    d[4:8] = torch.randint(0, V // 2, (4,), dtype=torch.int32)
    b.target_logits, b.draft_logits, b.draft_tokens = z, w, d
    acc, offs, toks, probs = _run(cuda_lib, b)
    check_spec(b, acc, offs, toks, probs)
    assert acc[0].item() == 4 and acc[1].item() == 0
    assert toks[offs[1].item()].item() >= V // 2


def test_spec_verify_is_deterministic(cuda_lib):
    b = make_config(2, seed=3)
    r1 = [t.clone() for t in valid_spec_outputs(*_run(cuda_lib, b))]
    r2 = valid_spec_outputs(*_run(cuda_lib, b))
    for x, y in zip(r1, r2):
        assert torch.equal(x, y)


def test_spec_verify_mismatch_rate_at_scale(cuda_lib):
    """~10^4 verify positions: mismatches with the oracle stay under 1e-4 of positions."""
    rng = np.random.default_rng(12)
    total = dict(positions=0, near=0, mismatches=0)
    for k in range(4):
        L = rng.integers(0, 11, size=420)
        b = make_batch(L, np.zeros_like(L), Hq=8, Hkv=1, D=64, V=24000, logit_std=1.0,
                       noise_sigma=0.9, seed=100 + k, spec_only=True)
        st = check_spec(b, *_run(cuda_lib, b))
        for key in total:
            total[key] += st[key]
    print(total)
    assert total["positions"] >= 10_000
    assert total["mismatches"] <= 1e-4 * total["positions"]


def test_spec_verify_output_law_monte_carlo(cuda_lib):
    """Emitted tokens at a reached position follow p (chi-square), independent of the oracle."""
    rng = np.random.default_rng(9)
    V, L, users, calls = 24, 3, 500, 24
    zl = rng.normal(0, 1.2, size=(L + 1, V))
    wl = zl[:L] + rng.normal(0, 0.9, size=(L, V))
    p = scipy.special.softmax(zl, axis=-1)
    q = scipy.special.softmax(wl, axis=-1)
    z = torch.tensor(np.tile(zl, (users, 1)), dtype=torch.float32, device=DEV)
    w = torch.tensor(np.tile(wl, (users, 1)), dtype=torch.float32, device=DEV)
    counts = np.zeros((L + 1, V))
    reached = np.zeros(L + 1)
    acc_hits = np.zeros(L)
    for c in range(calls):
        d = np.stack([rng.choice(V, size=users, p=q[t]) for t in range(L)], axis=1).reshape(-1)
        # a fresh seed per call: the in-kernel Philox uniforms are the only randomness
        acc, offs, toks, _ = cuda_lib.dipsd_spec_verify(
            [L] * users, np.arange(users), 1000 + c, z, w, torch.tensor(d, dtype=torch.int32, device=DEV))
        a = acc.cpu().numpy()
        o = offs.cpu().numpy()
        tk = toks.cpu().numpy()
        for k in range(L + 1):
            sel = np.flatnonzero(a >= k)
            reached[k] += sel.size
            np.add.at(counts[k], tk[o[sel] + k], 1)
            if k < L:
                acc_hits[k] += np.sum(a[sel] > k)
    for k in range(L + 1):
        pv = scipy.stats.chisquare(counts[k], p[k] * reached[k]).pvalue
        assert pv > 1e-4, (k, pv)
        if k < L:
            alpha = np.minimum(p[k], q[k]).sum()
            sd = math.sqrt(alpha * (1 - alpha) / reached[k])
            assert abs(acc_hits[k] / reached[k] - alpha) < 4 * sd


@pytest.mark.parametrize("nk1,nk2", [(4, 2), (8, 4), (16, 8)])
def test_spec_verify_segment_sizes(cuda_lib, nk1, nk2):
    """Every segment size of the two passes (16-byte vectors per lane): more or
    fewer segments per row, ragged last segments, L = 0 and L = 31 users."""
    rng = np.random.default_rng(30 + nk1)
    L = np.concatenate([[0, 31], rng.integers(0, 9, size=40)])
    b = make_batch(L, np.zeros_like(L), Hq=8, Hkv=1, D=64, V=20008, logit_std=1.5, noise_sigma=0.7,
                   seed=30 + nk1, spec_only=True)
    with cuda_lib.plan_override(spec_nk1=nk1, spec_nk2=nk2):
        st = check_spec(b, *_run(cuda_lib, b))
    print(f"segments {nk1}/{nk2}: {st}")


@pytest.mark.parametrize("grid1,nk1", [(1, 16), (3, 8), (40, 4), (97, 16)])
def test_spec_verify_persistent_statistics_grid(cuda_lib, grid1, nk1):
    """The statistics pass on a capped grid, so every warp sums many segments
    in turn (each refilled while the previous one is summed); three calls in a
    row, so the decision words and arrival counters must come back to zero."""
    rng = np.random.default_rng(50 + grid1)
    L = np.concatenate([[0, 31, 0], rng.integers(0, 11, size=37)])
    b = make_batch(L, np.zeros_like(L), Hq=8, Hkv=1, D=64, V=30016, logit_std=2.0, noise_sigma=0.8,
                   seed=50 + grid1, spec_only=True)
    g = lambda t: t.to(DEV)
    ws = cuda_lib.workspace(cuda_lib.dipsd_spec_verify_workspace_size(b.L, b.V), DEV)
    with cuda_lib.plan_override(spec_grid1=grid1, spec_nk1=nk1):
        for _ in range(3):
            out = cuda_lib.dipsd_spec_verify(b.L, b.user_ids, b.seed, g(b.target_logits), g(b.draft_logits),
                                             g(b.draft_tokens), ws=ws)
            torch.cuda.synchronize()
            st = check_spec(b, *out)
            assert cuda_lib.device_status(ws) == 0
    print(f"statistics grid {grid1} x {nk1}: {st}")
