"""The persistent attention grid's walk over its chunk, modelled on the CPU on
plans the library's planner makes (dipsd_verify_attention_plan).

A CTA of the persistent grid does not search for its work: its first piece
comes from three facts the host records per chunk (the user of the chunk's
first page, how many chunks back the stream of that page starts, how many
chunks ahead the stream of the chunk's last page ends), and every later piece
is the next stream from its first page (csrc/attention.cuh: first_piece,
next_piece).  Here that walk runs over each chunk and must visit exactly the
pieces a plain search of the chunk bounds and user offsets finds, with the
same KV range, split index and split count; the streams it marks for the
merge (one that starts in a chunk and runs past its end) must be exactly the
streams cut by a chunk bound."""

import bisect

import numpy as np
import pytest

from workloads import config_shape

PAGE = 16
ROWS = 128


@pytest.fixture(scope="module")
def dipsd():
    from paper_2604_20919_gb300 import build, dipsd as d
    build.build()
    d.load()
    return d


def _walk_matches_search(dipsd, L, ctx, Hq, Hkv, D, grid):
    with dipsd.plan_override(attn_persist=1, attn_grid=grid):
        pl = dipsd.dipsd_verify_attention_plan(L, ctx, Hq, Hkv, D, 152)
    cb = pl["chunk_bound"]
    if cb is None:  # a cluster plan (the persistent grid does not apply)
        return False
    G, B = Hq // Hkv, len(L)
    T = np.asarray(L) + 1
    kv = np.asarray(ctx) + T
    npg = (kv + PAGE - 1) // PAGE
    nrb = (G * T + ROWS - 1) // ROWS
    page_off = np.concatenate([[0], np.cumsum(npg * nrb * Hkv)])
    nc = len(cb) - 1
    chunk_at = lambda pos: bisect.bisect_right(list(cb[:-1]), pos) - 1

    def stream_at(pos):  # the stream holding page pos: (user, its first page)
        ui = bisect.bisect_right(list(page_off[:B]), pos) - 1
        k = min((pos - page_off[ui]) // npg[ui], nrb[ui] * Hkv - 1)
        return ui, page_off[ui] + k * npg[ui]

    # the host's per-chunk facts, and the rows of the streams cut by a bound
    first_user, c0_back, c1_fwd, starts_cut = [0] * nc, [0] * nc, [0] * nc, [False] * nc
    cut_rows = 0
    for b in range(nc):
        lo, hi = cb[b], cb[b + 1]
        ui, s0 = stream_at(lo)
        first_user[b], c0_back[b] = ui, b - chunk_at(s0)
        ui, s0 = stream_at(hi - 1)
        c1 = chunk_at(s0 + npg[ui] - 1)
        c1_fwd[b] = c1 - b
        starts_cut[b] = c1 > b and chunk_at(s0) == b
        if starts_cut[b]:
            rb = (s0 - page_off[ui]) // npg[ui] // Hkv
            cut_rows += min(ROWS, G * T[ui] - rb * ROWS)
        assert 0 <= c0_back[b] < 256 and 0 <= c1_fwd[b] < 256

    def piece(ui, sidx, pos, c0, cta, hi):  # the kernel's piece_of_stream
        s0 = page_off[ui] + sidx * npg[ui]
        nxt = min(hi, s0 + npg[ui])
        c1 = cta if s0 + npg[ui] <= hi else cta + c1_fwd[cta]
        return dict(ui=ui, h=sidx % Hkv, rb=sidx // Hkv, next=nxt, kv_begin=(pos - s0) * PAGE,
                    kv_end=min((nxt - s0) * PAGE, kv[ui]), nsplit=c1 - c0 + 1, split=cta - c0)

    def searched(pos, cta, hi):  # the same piece found by searching
        ui = bisect.bisect_right(list(page_off[:B]), pos) - 1
        sidx = (pos - page_off[ui]) // npg[ui]
        s0 = page_off[ui] + sidx * npg[ui]
        nxt = min(hi, s0 + npg[ui])
        c0, c1 = chunk_at(s0), chunk_at(s0 + npg[ui] - 1)
        return dict(ui=ui, h=sidx % Hkv, rb=sidx // Hkv, next=nxt, kv_begin=(pos - s0) * PAGE,
                    kv_end=min((nxt - s0) * PAGE, kv[ui]), nsplit=c1 - c0 + 1, split=cta - c0)

    pieces, marked = 0, 0
    for b in range(nc):
        lo, hi = cb[b], cb[b + 1]
        ui, pos = first_user[b], lo
        w = piece(ui, (lo - page_off[ui]) // npg[ui], lo, b - c0_back[b], b, hi)
        while True:
            assert w == searched(pos, b, hi)
            pieces += 1
            if w["nsplit"] > 1 and w["split"] == 0:
                assert starts_cut[b]  # the piece that writes the merge descriptor
                marked += 1
            if w["next"] >= hi:
                break
            ui, sidx = w["ui"], w["rb"] * Hkv + w["h"] + 1
            if sidx == nrb[ui] * Hkv:
                ui, sidx = ui + 1, 0
            pos = w["next"]
            w = piece(ui, sidx, pos, b, b, hi)
    assert pieces == pl["n_items"]
    assert marked == sum(starts_cut)
    assert cut_rows == pl["n_merge"]  # the rows the merge combines
    return True


@pytest.mark.parametrize("grid", [7, 31, 100, 152])
@pytest.mark.parametrize("wl", [3, 4, 5])
def test_walk_on_the_workloads(dipsd, wl, grid):
    s = config_shape(wl)
    L, ctx = np.asarray(s["L"])[:64], np.asarray(s["ctx"])[:64]
    assert _walk_matches_search(dipsd, L, ctx, s["Hq"], s["Hkv"], s["D"], grid)


def test_walk_on_random_batches(dipsd):
    walked = 0
    for seed in range(60):
        rng = np.random.default_rng(seed)
        B = int(rng.integers(1, 60))
        L = rng.integers(0, 32, B)
        ctx = rng.integers(0, 3000, B)
        Hkv = int(rng.choice([1, 2, 8]))
        G = int(rng.choice([1, 4, 8, 16]))
        walked += _walk_matches_search(dipsd, L, ctx, G * Hkv, Hkv, int(rng.choice([64, 128])),
                                       int(rng.integers(1, 200)))
    assert walked >= 40  # most draws get a persistent grid
