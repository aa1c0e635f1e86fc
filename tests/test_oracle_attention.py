"""Pins for the verify-attention oracle (CPU only).

The reference answer comes from torch's scaled_dot_product_attention (a
library routine) in fp64 on a logically contiguous cache that the test
scatters into pages itself, plus special cases with closed forms:
kv_len = 1 gives v_0; identical keys give the running mean of the values.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import verify_attention

PAGE = 16


def _paged_problem(rng, L, ctx, Hq, Hkv, D, spare=5):
    """Logical per-user K/V plus a scattered paged copy built independently."""
    B = len(L)
    kv_len = [c + l + 1 for c, l in zip(ctx, L)]
    pages = [-(-n // PAGE) for n in kv_len]
    nb = sum(pages) + spare
    perm = rng.permutation(nb)
    k_cache = rng.normal(size=(nb, Hkv, PAGE, D))
    v_cache = rng.normal(size=(nb, Hkv, PAGE, D))
    bt = np.full((B, max(pages)), -1, dtype=np.int64)
    Ks, Vs = [], []
    o = 0
    for i in range(B):
        K = rng.normal(size=(Hkv, kv_len[i], D))
        Vv = rng.normal(size=(Hkv, kv_len[i], D))
        for j in range(kv_len[i]):
            blk = perm[o + j // PAGE]
            k_cache[blk, :, j % PAGE] = K[:, j]
            v_cache[blk, :, j % PAGE] = Vv[:, j]
        bt[i, :pages[i]] = perm[o:o + pages[i]]
        o += pages[i]
        Ks.append(K)
        Vs.append(Vv)
    q = rng.normal(size=(sum(l + 1 for l in L), Hq, D))
    return q, k_cache, v_cache, bt, Ks, Vs


def _sdpa_reference(q, Ks, Vs, ctx, L, scale, G):
    outs = []
    n0 = 0
    for i in range(len(L)):
        T = L[i] + 1
        qi = torch.from_numpy(q[n0:n0 + T]).permute(1, 0, 2)            # [Hq, T, D]
        K = torch.from_numpy(Ks[i]).repeat_interleave(G, dim=0)          # [Hq, kv, D]
        V = torch.from_numpy(Vs[i]).repeat_interleave(G, dim=0)
        kv = K.shape[1]
        mask = torch.arange(kv)[None, :] <= (ctx[i] + torch.arange(T))[:, None]
        o = F.scaled_dot_product_attention(qi, K, V, attn_mask=mask, scale=scale)
        outs.append(o.permute(1, 0, 2).numpy())
        n0 += T
    return np.concatenate(outs)


@pytest.mark.parametrize("Hq,Hkv,D", [(8, 2, 16), (4, 1, 64), (16, 2, 32)])
def test_matches_torch_sdpa_on_ragged_paged_batch(Hq, Hkv, D):
    rng = np.random.default_rng(Hq * 100 + D)
    L = [0, 2, 5, 1, 3]
    ctx = [0, 17, 40, 15, 64]
    q, kc, vc, bt, Ks, Vs = _paged_problem(rng, L, ctx, Hq, Hkv, D)
    scale = D ** -0.5
    got = verify_attention(q, kc, vc, bt, ctx, L, scale)
    ref = _sdpa_reference(q, Ks, Vs, ctx, L, scale, Hq // Hkv)
    np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-12)


def test_single_key_returns_v0_of_its_kv_head():
    rng = np.random.default_rng(3)
    Hq, Hkv, D = 6, 3, 8
    q, kc, vc, bt, Ks, Vs = _paged_problem(rng, [0, 0], [0, 0], Hq, Hkv, D)
    got = verify_attention(q, kc, vc, bt, [0, 0], [0, 0], 0.7)
    for i in range(2):
        for h in range(Hq):
            np.testing.assert_allclose(got[i, h], Vs[i][h // 2, 0], rtol=0, atol=1e-14)


def test_equal_keys_give_running_mean_of_values():
    rng = np.random.default_rng(4)
    Hq, Hkv, D = 4, 2, 8
    L, ctx = [3], [9]
    q, kc, vc, bt, Ks, Vs = _paged_problem(rng, L, ctx, Hq, Hkv, D)
    kc[:] = 0.37  # every key identical -> uniform attention over the visible keys
    got = verify_attention(q, kc, vc, bt, ctx, L, 0.5)
    for t in range(L[0] + 1):
        for h in range(Hq):
            np.testing.assert_allclose(got[t, h], Vs[0][h // 2, :ctx[0] + t + 1].mean(0),
                                       rtol=1e-12, atol=1e-13)


def test_page_permutation_invariance():
    rng = np.random.default_rng(5)
    Hq, Hkv, D = 8, 2, 16
    L, ctx = [4, 1], [30, 50]
    q, kc, vc, bt, _, _ = _paged_problem(rng, L, ctx, Hq, Hkv, D)
    perm = rng.permutation(kc.shape[0])
    inv = np.argsort(perm)
    kc2, vc2 = kc[perm], vc[perm]          # block b moves to slot inv[b]
    bt2 = np.where(bt >= 0, inv[np.maximum(bt, 0)], -1)
    a = verify_attention(q, kc, vc, bt, ctx, L, 0.3)
    b = verify_attention(q, kc2, vc2, bt2, ctx, L, 0.3)
    np.testing.assert_array_equal(a, b)


def test_members_select_block_table_rows():
    rng = np.random.default_rng(6)
    Hq, Hkv, D = 4, 1, 8
    L, ctx = [1, 2, 0], [20, 5, 33]
    q, kc, vc, bt, _, _ = _paged_problem(rng, L, ctx, Hq, Hkv, D)
    full = verify_attention(q, kc, vc, bt, ctx, L, 0.4)
    # batch = users 2 and 0 of the table, in that order
    q_sub = np.concatenate([q[5:6], q[0:2]])
    sub = verify_attention(q_sub, kc, vc, bt, [33, 20], [0, 1], 0.4, members=[2, 0])
    np.testing.assert_array_equal(sub, np.concatenate([full[5:6], full[0:2]]))


def _new_rows(Ks, ctx, L):
    """[sum T, Hkv, D]: each user's verify-token rows, read from the logical K/V."""
    return np.concatenate([Ks[i][:, ctx[i]:ctx[i] + L[i] + 1].transpose(1, 0, 2) for i in range(len(L))])


def test_kv_append_restores_poisoned_slots_exactly():
    """Poison the verify tokens' slots, append their rows: the cache the test
    scattered itself comes back bit for bit, and attention on it still matches
    torch's SDPA."""
    from oracle import kv_append
    rng = np.random.default_rng(31)
    L, ctx = [3, 0, 5], [17, 0, 40]
    q, kc, vc, bt, Ks, Vs = _paged_problem(rng, L, ctx, 8, 2, 16)
    pk, pv = kc.copy(), vc.copy()
    for i in range(len(L)):
        for t in range(L[i] + 1):
            pos = ctx[i] + t
            pk[bt[i, pos // PAGE], :, pos % PAGE] = np.nan
            pv[bt[i, pos // PAGE], :, pos % PAGE] = np.nan
    k2, v2 = kv_append(pk, pv, bt, ctx, L, _new_rows(Ks, ctx, L), _new_rows(Vs, ctx, L))
    assert np.array_equal(k2, kc) and np.array_equal(v2, vc)
    o = verify_attention(q, k2, v2, bt, ctx, L, 0.25)
    np.testing.assert_allclose(o, _sdpa_reference(q, Ks, Vs, ctx, L, 0.25, 4), rtol=0, atol=1e-12)


def test_kv_append_touches_only_the_verify_slots():
    from oracle import kv_append
    rng = np.random.default_rng(32)
    L, ctx = [2, 4], [30, 3]
    _, kc, vc, bt, Ks, Vs = _paged_problem(rng, L, ctx, 4, 1, 8)
    nk = rng.normal(size=(sum(l + 1 for l in L), 1, 8))
    nv = rng.normal(size=nk.shape)
    k2, v2 = kv_append(kc, vc, bt, ctx, L, nk, nv)
    touched = np.zeros(kc.shape[:1] + kc.shape[2:3], dtype=bool)  # [block, slot]
    n = 0
    for i in range(len(L)):
        for t in range(L[i] + 1):
            pos = ctx[i] + t
            blk, slot = bt[i, pos // PAGE], pos % PAGE
            touched[blk, slot] = True
            assert np.array_equal(k2[blk, :, slot], nk[n]) and np.array_equal(v2[blk, :, slot], nv[n])
            n += 1
    untouched = ~touched
    assert np.array_equal(k2.transpose(0, 2, 1, 3)[untouched], kc.transpose(0, 2, 1, 3)[untouched])
    assert np.array_equal(v2.transpose(0, 2, 1, 3)[untouched], vc.transpose(0, 2, 1, 3)[untouched])


def test_kv_append_follows_members():
    """With members, user i writes through block-table row members[i]."""
    from oracle import kv_append
    rng = np.random.default_rng(33)
    L, ctx = [1, 2], [5, 20]
    _, kc, vc, bt, Ks, Vs = _paged_problem(rng, L, ctx, 2, 1, 8)
    bt_perm = bt[::-1].copy()  # table rows in the other order
    nk, nv = _new_rows(Ks, ctx, L), _new_rows(Vs, ctx, L)
    a = kv_append(kc, vc, bt, ctx, L, nk, nv)
    b = kv_append(kc, vc, bt_perm, ctx, L, nk, nv, members=[1, 0])
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
