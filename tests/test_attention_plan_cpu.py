"""The attention planner (host code of the C-ABI library) on the CPU, through
dipsd_verify_attention_plan: every key of every user is covered by its KV
splits, the work-item count and the grid follow from them, and the persistent
grid, the cluster merge and the merge kernel are chosen only where the kernel
supports them."""

import numpy as np
import pytest

from workloads import config_shape

PAGE = 16
ROWS_PER_ITEM = 128


@pytest.fixture(scope="module")
def dipsd():
    from paper_2604_20919_gb300 import build, dipsd as d
    build.build()
    d.load()
    return d


def _page_streams(L, ctx, G, Hkv):
    """(user, pages, rows) of every (user, row block, KV head) stream, in the
    order the persistent grid lays them back to back."""
    pages = -(-(np.asarray(ctx) + np.asarray(L) + 1) // PAGE)
    M = G * (np.asarray(L) + 1)
    rb = -(-M // ROWS_PER_ITEM)
    return [(i, int(pages[i]), int(min(ROWS_PER_ITEM, M[i] - r * ROWS_PER_ITEM)))
            for i in range(len(L)) for r in range(int(rb[i])) for _ in range(Hkv)]


def _check_plan(p, L, ctx, Hq, Hkv, D, num_sms, append, forced_cluster=False):
    L, ctx = np.asarray(L), np.asarray(ctx)
    G = Hq // Hkv
    kv_len = ctx + L + 1
    ns, sl = p["nsplit"], p["split_len"]
    assert (sl % PAGE == 0).all() and (sl >= PAGE).all()
    assert (ns >= 1).all()
    if p["stream_chunks"]:
        # persistent grid over page streams, modelled here independently: the
        # streams back to back, chunk b = pages [bound[b], bound[b + 1]) for
        # CTA b; a stream has one split per chunk it touches
        assert not append and not p["cluster"]
        bound = np.asarray(p["chunk_bound"])
        streams = _page_streams(L, ctx, G, Hkv)
        total = sum(n for _, n, _ in streams)
        assert p["grid"] == p["stream_chunks"] == len(bound) - 1 <= min(num_sms, 256)
        assert bound[0] == 0 and bound[-1] == total and (np.diff(bound) > 0).all()
        chunk_of = lambda pos: int(np.searchsorted(bound, pos, side="right")) - 1
        pieces, ns_user, pos, cut_rows = 0, np.ones(len(L), dtype=int), 0, 0
        for i, n, rows in streams:
            c = chunk_of(pos + n - 1) - chunk_of(pos) + 1
            pieces += c
            ns_user[i] = max(ns_user[i], c)
            cut_rows += rows if c > 1 else 0
            pos += n
        assert p["n_items"] == pieces
        np.testing.assert_array_equal(ns, ns_user)
        split_users = ns_user > 1
        # the merge visits the rows of the streams cut by a chunk bound
        assert p["n_merge"] == cut_rows
    else:
        # every key of a user lies in exactly one split; only cluster plans may
        # carry trailing empty splits (every user then has exactly `cluster`)
        assert (ns * sl >= kv_len).all()
        if p["cluster"]:
            assert p["cluster"] <= (3 if D == 128 else 6)
            assert (ns == p["cluster"]).all()
            assert p["n_merge"] == 0
            # chosen by cost only when every cluster is resident at once
            assert forced_cluster or p["n_items"] <= num_sms
        else:
            assert ((ns - 1) * sl < kv_len).all()
        row_blocks = -(-(G * (L + 1)) // ROWS_PER_ITEM)
        assert p["n_items"] == int((ns * row_blocks * Hkv).sum())
        assert p["grid"] == p["n_items"]  # one CTA per item
        split_users = (ns > 1) if not p["cluster"] else np.zeros_like(ns, dtype=bool)
    # split users without a cluster go through the merge kernel: (one CTA
    # per item) it visits one row per (verify token, query head); (m, l) and
    # D partial outputs per (split, head, row) in the workspace
    if not p["stream_chunks"]:
        assert p["n_merge"] == int(((L + 1) * Hq)[split_users].sum())
    part_rows = int((ns * Hkv * G * (L + 1))[split_users].sum())
    assert p["ws_bytes"] >= part_rows * (8 + 4 * D)
    assert (p["ws_bytes"] == 0) == (part_rows == 0)


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("num_sms", [1, 8, 152])
def test_plan_invariants_on_random_batches(dipsd, seed, num_sms):
    rng = np.random.default_rng([seed, num_sms])
    B = int(rng.integers(1, 40))
    L = rng.integers(0, 32, B)
    ctx = np.exp(rng.uniform(0, np.log(40000), B)).astype(int)
    ctx = np.where(rng.random(B) < 0.1, rng.integers(0, 20, B), ctx)  # some near-empty contexts
    Hkv = int(rng.choice([1, 2, 8]))
    G = int(rng.choice([1, 4, 8, 16]))
    D = int(rng.choice([64, 128]))
    for append in (False, True):
        p = dipsd.dipsd_verify_attention_plan(L, ctx, G * Hkv, Hkv, D, num_sms, append)
        _check_plan(p, L, ctx, G * Hkv, Hkv, D, num_sms, append)


def test_plan_of_the_workloads(dipsd):
    """Workload 2 (8 users x 1024 tokens): 2 splits per (user, head) merged in
    a 2-CTA cluster, 128 CTAs, no merge launch.  Workload 3 (32 ragged users):
    a persistent grid of one CTA per SM over the page streams; the append
    variant keeps one CTA per item."""
    s = config_shape(2, 0)
    p = dipsd.dipsd_verify_attention_plan(s["L"], s["ctx"], s["Hq"], s["Hkv"], s["D"], 152)
    assert (p["cluster"], p["n_items"], p["grid"], p["n_merge"]) == (2, 128, 128, 0)
    s = config_shape(3, 0)
    p = dipsd.dipsd_verify_attention_plan(s["L"], s["ctx"], s["Hq"], s["Hkv"], s["D"], 152)
    assert p["cluster"] == 0 and p["stream_chunks"] > 0 and 140 <= p["grid"] <= 152
    pa = dipsd.dipsd_verify_attention_plan(s["L"], s["ctx"], s["Hq"], s["Hkv"], s["D"], 152, append=True)
    assert pa["grid"] == pa["n_items"]
    for cfg in (1, 2, 3, 4):
        s = config_shape(cfg, 0)
        for append in (False, True):
            p = dipsd.dipsd_verify_attention_plan(s["L"], s["ctx"], s["Hq"], s["Hkv"], s["D"], 152, append)
            _check_plan(p, s["L"], s["ctx"], s["Hq"], s["Hkv"], s["D"], 152, append)


def test_plan_overrides(dipsd):
    L, ctx = [5, 0, 8, 2, 20, 1], [1500, 3000, 333, 64, 700, 0]
    with dipsd.plan_override(attn_persist=1, attn_grid=7, attn_split_tiles=2):
        p = dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152)
        assert p["grid"] == 7 and p["n_items"] > 7 and p["n_merge"] > 0
        _check_plan(p, L, ctx, 64, 8, 128, 152, False)
        pa = dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152, append=True)
        assert pa["grid"] == pa["n_items"]  # the append keeps one item per CTA
    with dipsd.plan_override(attn_persist=2):
        s = config_shape(3, 0)
        p = dipsd.dipsd_verify_attention_plan(s["L"], s["ctx"], s["Hq"], s["Hkv"], s["D"], 152)
        assert p["grid"] == p["n_items"]
    with dipsd.plan_override(attn_cluster=3):
        p = dipsd.dipsd_verify_attention_plan(L, ctx, 64, 8, 128, 152)
        assert p["cluster"] == 3 and (p["nsplit"] == 3).all()
        _check_plan(p, L, ctx, 64, 8, 128, 152, False, forced_cluster=True)


def test_plan_rejects_bad_arguments(dipsd):
    from paper_2604_20919_gb300.dipsd import DipsdError
    cases = [([], [], 8, 2, 128, 152, 1),        # empty batch
             ([1, 32], [4, 4], 8, 2, 128, 152, 1),  # draft length above 31
             ([1], [4], 8, 3, 128, 152, 1),      # Hq not a multiple of Hkv
             ([1], [4], 8, 2, 96, 152, 2),       # head_dim not built
             ([1], [4], 8, 2, 128, 0, 1)]        # no SMs
    for L, ctx, Hq, Hkv, D, sms, want in cases:
        with pytest.raises(DipsdError) as e:
            dipsd.dipsd_verify_attention_plan(L, ctx, Hq, Hkv, D, sms)
        assert e.value.status == want
