"""verify_attention through the C ABI vs the fp64 oracle."""

import pytest
import torch

import oracle
from parity import attention_reference, attention_subset_reference, check_attention, peaked_attention
from workloads import make_batch, make_config

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _run(dipsd, b, ws=None):
    g = lambda t: t.to(DEV)
    out = dipsd.dipsd_verify_attention(b.L, b.ctx, g(b.q), g(b.k_cache), g(b.v_cache), g(b.block_table),
                                       b.scale, ws=ws)
    torch.cuda.synchronize()
    return out


def _full_reference(b):
    """(oracle output, oracle attention of |V|) of the whole batch."""
    return attention_reference(b)


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_attention_workloads(cuda_lib, cfg):
    b = make_config(cfg, seed=0)
    err = check_attention(_run(cuda_lib, b), *_full_reference(b))
    print(f"workload {cfg}: max abs err {err:.3e}")


def test_attention_long_context_sampled_users(cuda_lib):
    """Workload 4 (64 users x 32768 context, 8.6 GB of KV) at full size; oracle on sampled users."""
    b = make_config(4, seed=0, device="cpu", kv_device=DEV)
    out = _run(cuda_lib, b)
    for users in ([0, 37], [63]):
        rows, ref, ref_abs = attention_subset_reference(b, users, with_abs=True)
        err = check_attention(out[torch.from_numpy(rows).to(DEV)], ref, ref_abs)
        print(f"workload 4 users {users}: max abs err {err:.3e}")
    del b, out
    torch.cuda.empty_cache()


def test_attention_peaked_headline_shapes(cuda_lib):
    """Workload 2's shapes (ctx 1024, 64/8/128) with peaked attention (Q x4,
    V of mean 1): a single key counted or missed moves outputs by O(0.1 .. 1),
    far outside both bounds (the CPU test of the parity check shows a causal
    off-by-one and a dropped last page failing on these shapes)."""
    b = peaked_attention(make_config(2, seed=6))
    err = check_attention(_run(cuda_lib, b), *_full_reference(b))
    print(f"peaked workload 2: max abs err {err:.3e}")


def test_attention_peaked_long_context_sampled_users(cuda_lib):
    """Workload 4 (ctx 32768) with peaked attention; oracle on sampled users."""
    b = peaked_attention(make_config(4, seed=0, device="cpu", kv_device=DEV))
    out = _run(cuda_lib, b)
    rows, ref, ref_abs = attention_subset_reference(b, [5, 50], with_abs=True)
    err = check_attention(out[torch.from_numpy(rows).to(DEV)], ref, ref_abs)
    print(f"peaked workload 4: max abs err {err:.3e}")
    del b, out
    torch.cuda.empty_cache()


@pytest.mark.parametrize("L,ctx,Hq,Hkv,D", [
    ([0, 0, 0], [0, 1, 15], 8, 2, 128),          # kv_len 1, 2, 16: single page, tiny
    ([3, 0, 7, 1], [16, 47, 63, 64], 64, 8, 128),  # page and tile edges
    ([0, 2, 5, 0], [127, 126, 250, 383], 64, 8, 128),  # kv_len 128, 129, 256, 384: 128-key tile edges
    ([31, 16], [5, 200], 64, 8, 128),            # G*T = 256 and 136: two row blocks
    ([9, 2], [300, 1000], 64, 8, 128),           # G*T = 80: eight consumer warps
    ([4, 1, 2], [129, 1, 700], 4, 1, 64),        # head_dim 64, G = 4
    ([2, 5], [90, 33], 16, 16, 128),             # G = 1 (multi-head)
    ([3, 6], [150, 77], 32, 2, 64),              # G = 16
])
def test_attention_edge_shapes(cuda_lib, L, ctx, Hq, Hkv, D):
    b = make_batch(L, ctx, Hq=Hq, Hkv=Hkv, D=D, V=64, seed=sum(L) + sum(ctx))
    check_attention(_run(cuda_lib, b), *_full_reference(b))


@pytest.mark.parametrize("split_tiles", [1, 2, 7])
def test_attention_forced_splits(cuda_lib, split_tiles):
    """Many KV splits per (user, head) exercise the partial/merge path."""
    b = make_batch([5, 0, 8, 2], [1500, 3000, 333, 64], Hq=64, Hkv=8, D=128, V=64, seed=21)
    with cuda_lib.plan_override(attn_split_tiles=split_tiles):
        out = _run(cuda_lib, b)
    check_attention(out, *_full_reference(b))


@pytest.mark.parametrize("cluster,D", [(2, 128), (3, 128), (6, 64)])
def test_attention_cluster_merge(cuda_lib, cluster, D):
    """KV splits merged inside a thread-block cluster, including empty splits
    (a user with fewer 64-key tiles than splits)."""
    b = make_batch([5, 0, 8, 2, 1], [1500, 3000, 333, 64, 0], Hq=64 if D == 128 else 16, Hkv=8 if D == 128 else 2,
                   D=D, V=64, seed=23)
    with cuda_lib.plan_override(attn_cluster=cluster):
        out = _run(cuda_lib, b)
    check_attention(out, *_full_reference(b))


@pytest.mark.parametrize("grid,split_tiles,D", [(1, 0, 128), (3, 0, 128), (7, 2, 128), (5, 1, 64), (152, 1, 128)])
def test_attention_persistent_grid(cuda_lib, grid, split_tiles, D):
    """A grid smaller than the item count: each CTA walks several items (row
    blocks with and without padding rows, ragged last tiles, KV splits and
    their merge), the K/V ring and every barrier phase running on across
    items."""
    b = make_batch([5, 0, 8, 2, 20, 1], [1500, 3000, 333, 64, 700, 0], Hq=64 if D == 128 else 16,
                   Hkv=8 if D == 128 else 2, D=D, V=64, seed=24)
    with cuda_lib.plan_override(attn_persist=1, attn_grid=grid, attn_split_tiles=split_tiles):
        ws = cuda_lib.workspace(cuda_lib.dipsd_verify_attention_workspace_size(b.L, b.ctx, b.Hq, b.Hkv, b.D), DEV)
        out = _run(cuda_lib, b, ws)
        assert cuda_lib.device_status(ws) == 0
    check_attention(out, *_full_reference(b))


def test_attention_ignores_slots_past_kv_len(cuda_lib):
    """NaN in cache slots past each user's kv_len and in unused pages never reaches the output."""
    b = make_batch([2, 5, 0], [30, 500, 1], Hq=64, Hkv=8, D=128, V=64, seed=22)
    ref = _full_reference(b)
    kc, vc = b.k_cache.clone(), b.v_cache.clone()
    bt = b.block_table.numpy()
    used = set()
    for i, n in enumerate(b.kv_len):
        pages = -(-int(n) // 16)
        used.update(bt[i, :pages].tolist())
        last = bt[i, pages - 1]
        kc[last, :, int(n) % 16 or 16:] = float("nan")
        vc[last, :, int(n) % 16 or 16:] = float("nan")
    for blk in range(kc.shape[0]):
        if blk not in used:
            kc[blk] = float("nan")
            vc[blk] = float("nan")
    b.k_cache, b.v_cache = kc, vc
    check_attention(_run(cuda_lib, b), *ref)


def test_attention_status_word_stays_clear(cuda_lib):
    b = make_config(2, seed=1)
    ws = cuda_lib.workspace(cuda_lib.dipsd_verify_attention_workspace_size(b.L, b.ctx, b.Hq, b.Hkv, b.D), DEV)
    _run(cuda_lib, b, ws=ws)
    assert cuda_lib.device_status(ws) == 0


def test_attention_is_deterministic(cuda_lib):
    b = make_config(3, seed=2)
    o1 = _run(cuda_lib, b).clone()
    o2 = _run(cuda_lib, b)
    assert torch.equal(o1, o2)
