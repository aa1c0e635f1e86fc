"""The attention parity check has the power to catch one-key mistakes at
long contexts (CPU only: the mistakes are planted in copies of the oracle).

With N(0, 1) queries and keys over ~1000 keys the softmax is spread thin, so
a key counted that should not be (a causal off-by-one) or a page missed moves
outputs by ~1e-3, well inside the stated 2e-2 / 1e-2 bar.  On peaked inputs
(Q x4, V of mean 1) and with the arithmetic bound TIGHT x (attention of |V|),
both mistakes fail the check on workload 2's shapes (ctx 1024, 64/8/128),
while the oracle itself, rounded to bf16 as the kernel's output is, passes.
"""
import numpy as np
import pytest

from oracle.attention import gather_pages
from parity import attention_reference, check_attention, peaked_attention
from workloads import make_batch

PAGE = 16


def _planted(b, mistake):
    """The oracle's causal attention with one planted mistake:
    'off_by_one': verify token t also sees key C_i + t + 1 (when it exists);
    'last_page':  every token misses the keys of its user's last page."""
    q = b.q.double().numpy()
    kc, vc, bt = b.k_cache.double().numpy(), b.v_cache.double().numpy(), b.block_table.numpy()
    G = b.Hq // b.Hkv
    out = np.empty_like(q)
    n0 = 0
    for i in range(b.B):
        T = int(b.L[i]) + 1
        kv_len = int(b.ctx[i]) + T
        K = gather_pages(kc, bt[i], kv_len)
        V = gather_pages(vc, bt[i], kv_len)
        last_page_start = (kv_len - 1) // PAGE * PAGE
        for t in range(T):
            visible = int(b.ctx[i]) + t + 1
            if mistake == "off_by_one":
                visible = min(visible + 1, kv_len)
            elif mistake == "last_page":
                visible = min(visible, last_page_start)
            for h in range(b.Hq):
                s = (K[h // G, :visible] @ q[n0 + t, h]) * b.scale
                w = np.exp(s - s.max())
                out[n0 + t, h] = (w @ V[h // G, :visible]) / w.sum()
        n0 += T
    return out


def _bf16(x):
    import torch
    return torch.from_numpy(x).to(torch.bfloat16).double().numpy()


@pytest.fixture(scope="module")
def peaked_batch():
    rng = np.random.default_rng(6)
    L = rng.integers(1, 9, size=8)
    b = peaked_attention(make_batch(L, [1024] * 8, Hq=64, Hkv=8, D=128, V=64, seed=6))
    ref, ref_abs = attention_reference(b)
    return b, ref, ref_abs


def test_oracle_rounded_to_bf16_passes(peaked_batch):
    b, ref, ref_abs = peaked_batch
    check_attention(_bf16(ref), ref, ref_abs)


@pytest.mark.parametrize("mistake", ["off_by_one", "last_page"])
def test_planted_mistake_fails(peaked_batch, mistake):
    b, ref, ref_abs = peaked_batch
    with pytest.raises(AssertionError):
        check_attention(_bf16(_planted(b, mistake)), ref, ref_abs)


def test_planted_copy_without_mistake_is_the_oracle(peaked_batch):
    b, ref, _ = peaked_batch
    np.testing.assert_allclose(_planted(b, None), ref, rtol=1e-12, atol=1e-12)
