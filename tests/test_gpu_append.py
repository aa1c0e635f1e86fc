"""KV append inside verification (dipsd_*_append) through the C ABI.

The verify tokens' own K/V rows are taken out of a batch's cache, their
slots are poisoned with NaN, and the append entry point gets the rows as
inputs: its attention must match the oracle on the untouched cache, and the
cache must come back bit for bit (oracle.kv_append on the poisoned cache
gives the same bytes)."""

import numpy as np
import pytest
import torch

import oracle
from parity import attention_reference, check_attention, valid_spec_outputs
from workloads import make_batch, make_config

pytestmark = pytest.mark.gpu
DEV = "cuda"
PAGE = 16


def _split_new_rows(b):
    """(new_k, new_v [sum T][Hkv][D], poisoned k/v caches) of a batch."""
    bt = b.block_table.numpy()
    nk, nv = [], []
    kc, vc = b.k_cache.clone(), b.v_cache.clone()
    for i in range(b.B):
        for t in range(int(b.L[i]) + 1):
            pos = int(b.ctx[i]) + t
            blk, slot = int(bt[i, pos // PAGE]), pos % PAGE
            nk.append(b.k_cache[blk, :, slot].clone())
            nv.append(b.v_cache[blk, :, slot].clone())
            kc[blk, :, slot] = float("nan")
            vc[blk, :, slot] = float("nan")
    return torch.stack(nk), torch.stack(nv), kc, vc


def _reference(b):
    """(oracle output, oracle attention of |V|) on the untouched cache."""
    return attention_reference(b)


def _append_run(dipsd, b):
    nk, nv, kc, vc = _split_new_rows(b)
    g = lambda t: t.to(DEV)
    kc_d, vc_d = g(kc), g(vc)
    out = dipsd.dipsd_verify_attention_append(b.L, b.ctx, g(b.q), g(nk), g(nv), kc_d, vc_d, g(b.block_table), b.scale)
    torch.cuda.synchronize()
    # the oracle's own scatter of the same rows into the poisoned cache
    ko, vo = oracle.kv_append(kc.view(torch.int16).numpy(), vc.view(torch.int16).numpy(), b.block_table.numpy(),
                              b.ctx, b.L, nk.view(torch.int16).numpy(), nv.view(torch.int16).numpy())
    assert np.array_equal(kc_d.cpu().view(torch.int16).numpy(), ko)
    assert np.array_equal(vc_d.cpu().view(torch.int16).numpy(), vo)
    assert torch.equal(kc_d.cpu().view(torch.int16), b.k_cache.view(torch.int16))
    return out


@pytest.mark.parametrize("cfg", [1, 2])
def test_append_attention_workloads(cuda_lib, cfg):
    b = make_config(cfg, seed=3)
    check_attention(_append_run(cuda_lib, b), *_reference(b))


@pytest.mark.parametrize("L,ctx,Hq,Hkv,D", [
    ([0, 0, 0], [0, 1, 15], 8, 2, 128),            # every token new at position 0; one page
    ([3, 0, 7, 31], [16, 47, 60, 40], 64, 8, 128),  # new rows across page and tile edges
    ([4, 1, 2], [129, 1, 700], 4, 1, 64),          # head_dim 64
])
def test_append_attention_edges(cuda_lib, L, ctx, Hq, Hkv, D):
    b = make_batch(L, ctx, Hq=Hq, Hkv=Hkv, D=D, V=64, seed=40 + sum(L))
    check_attention(_append_run(cuda_lib, b), *_reference(b))


@pytest.mark.parametrize("override,val", [("attn_split_tiles", 1), ("attn_split_tiles", 3), ("attn_cluster", 3),
                                          ("attn_persist", 1)])
def test_append_with_splits(cuda_lib, override, val):
    """Splits of one tile each put the new rows of a user into two CTAs."""
    b = make_batch([31, 5, 0, 12], [50, 1000, 63, 200], Hq=64, Hkv=8, D=128, V=64, seed=47)
    with cuda_lib.plan_override(**{override: val}):
        out = _append_run(cuda_lib, b)
    check_attention(out, *_reference(b))


def test_batch_append_matches_batch(cuda_lib):
    """dipsd_verify_batch_append on a poisoned cache == dipsd_verify_batch on the full one."""
    b = make_config(2, seed=6)
    nk, nv, kc, vc = _split_new_rows(b)
    g = lambda t: t.to(DEV)
    q, bt = g(b.q), g(b.block_table)
    z, w, d = g(b.target_logits), g(b.draft_logits), g(b.draft_tokens)
    ref = cuda_lib.dipsd_verify_batch(b.members, b.L, b.ctx, q, g(b.k_cache), g(b.v_cache), bt, b.scale, z, w, d,
                                      b.seed)
    kc_d, vc_d = g(kc), g(vc)
    res = cuda_lib.dipsd_verify_batch_append(b.members, b.L, b.ctx, q, g(nk), g(nv), kc_d, vc_d, bt, b.scale,
                                             z, w, d, b.seed)
    torch.cuda.synchronize()
    assert torch.equal(res[0], ref[0])
    for x, y in zip(valid_spec_outputs(*res[1:]), valid_spec_outputs(*ref[1:])):
        assert torch.equal(x, y)
    assert torch.equal(kc_d.cpu().view(torch.int16), b.k_cache.view(torch.int16))
    assert torch.equal(vc_d.cpu().view(torch.int16), b.v_cache.view(torch.int16))


def test_append_flags_page_ids_outside_the_cache(cuda_lib):
    """A page id past the cache at an appended position: that row is not written
    (the status word says so); the other users' rows still land."""
    b = make_batch([2, 3], [10, 100], Hq=8, Hkv=2, D=128, V=64, seed=48)
    nk, nv, kc, vc = _split_new_rows(b)
    bt = b.block_table.clone()
    nb = b.k_cache.shape[0]
    bt[0, 0] = nb + 3  # user 0's only page (positions 0..12)
    g = lambda t: t.to(DEV)
    kc_d, vc_d = g(kc), g(vc)
    ws = cuda_lib.workspace(cuda_lib.dipsd_verify_attention_workspace_size(b.L, b.ctx, b.Hq, b.Hkv, b.D), DEV)
    cuda_lib.dipsd_verify_attention_append(b.L, b.ctx, g(b.q), g(nk), g(nv), kc_d, vc_d, g(bt), b.scale, ws=ws)
    assert cuda_lib.device_status(ws) & cuda_lib.DEVERR_BAD_BLOCK
    btn = b.block_table.numpy()
    for t in range(4):  # user 1's rows are in place
        pos = 100 + t
        blk, slot = int(btn[1, pos // PAGE]), pos % PAGE
        assert torch.equal(kc_d[blk, :, slot].cpu().view(torch.int16), b.k_cache[blk, :, slot].view(torch.int16))
