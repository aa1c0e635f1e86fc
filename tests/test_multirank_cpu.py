"""The multi-GPU path's host logic on CPU ranks (gloo, world size 2).

Users are independent in both verification stages, so a batch shards by
users with no collective on the data path (shard.partition_users); each rank
verifies its members and the per-user results are gathered on the host and
packed in batch order (shard.merge_outputs).  Here each rank runs the fp64
oracle on its shard (the GPU path needs a GPU), the results travel through a
gloo all_gather, and rank 0 checks that the packed result equals one
unsharded oracle call exactly; the bench's timing aggregation
(shard.aggregate_timing: slowest rank's time, all ranks' units) is checked
on the same ranks.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2604_20919_gb300 import shard
from workloads import make_batch, make_config, offsets

WORLD = 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _host(b):
    return dict(q=b.q.double().numpy(), k=b.k_cache.double().numpy(), v=b.v_cache.double().numpy(),
                bt=b.block_table.numpy(), z=b.target_logits.double().numpy(), w=b.draft_logits.double().numpy(),
                d=b.draft_tokens.numpy(), u=b.uniforms.numpy())


def _verify_users(b, h, users):
    """Oracle verification of a subset of the batch's users (one rank's share)."""
    users = np.asarray(users, dtype=np.int64)
    rows = shard.position_rows(b.T, users)
    drows = shard.position_rows(b.L, users)
    attn = oracle.verify_attention(h["q"][rows], h["k"], h["v"], h["bt"][users], b.ctx[users], b.L[users], b.scale)
    r = oracle.spec_verify(b.L[users], h["z"][rows], h["w"][drows], h["d"][drows], h["u"][rows])
    return dict(users=users.tolist(), rows=rows.tolist(), attn=attn, accept_len=r["accept_len"],
                out_offsets=r["out_offsets"], out_tokens=r["out_tokens"])


def _rank_main(rank, port, cfg, result_path):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        b = cfg()
        h = _host(b)
        parts = shard.partition_users(b.kv_len, WORLD)
        mine = _verify_users(b, h, parts[rank])
        gathered = [None] * WORLD
        dist.all_gather_object(gathered, mine)
        # timing aggregation: rank r reports (10 + r) ms, 100 * (r + 1) units, (20 - r) ms end to end
        t, n, e = shard.aggregate_timing(10.0 + rank, 100.0 * (rank + 1), 20.0 - rank)
        if rank == 0:
            torch.save(dict(gathered=gathered, parts=parts, timing=(t, n, e)), result_path)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def _tiny():
    return make_config(1, seed=3)


def _ragged():
    return make_batch([0, 5, 2, 7, 1], [40, 300, 17, 129, 64], Hq=8, Hkv=2, D=64, V=96, logit_std=1.5,
                      noise_sigma=0.7, seed=12)


@pytest.mark.parametrize("cfg", [_tiny, _ragged], ids=["workload1", "ragged"])
def test_sharded_verification_matches_unsharded(cfg, tmp_path):
    path = str(tmp_path / "res.pt")
    mp.spawn(_rank_main, args=(_free_port(), cfg, path), nprocs=WORLD, join=True)
    res = torch.load(path, weights_only=False)
    b = cfg()
    h = _host(b)
    ref = _verify_users(b, h, list(range(b.B)))
    # every user verified exactly once, packed in batch order
    acc, offs, toks = shard.merge_outputs(b.B, res["parts"], res["gathered"])
    np.testing.assert_array_equal(acc, ref["accept_len"])
    np.testing.assert_array_equal(offs, ref["out_offsets"])
    np.testing.assert_array_equal(toks, ref["out_tokens"])
    attn = np.zeros_like(ref["attn"])
    for g in res["gathered"]:
        attn[np.asarray(g["rows"], dtype=np.int64)] = g["attn"]
    np.testing.assert_array_equal(attn, ref["attn"])
    assert res["timing"] == (11.0, 300.0, 20.0)


def test_partition_balances_kv():
    kv = [1000, 10, 990, 20, 500, 500, 30]
    parts = shard.partition_users(kv, 2)
    assert sorted(sum(parts, [])) == list(range(len(kv)))
    loads = [sum(kv[i] for i in p) for p in parts]
    assert abs(loads[0] - loads[1]) <= max(kv)
    assert parts == shard.partition_users(kv, 2)  # deterministic
    assert shard.partition_users(kv, 1) == [list(range(len(kv)))]
    four = shard.partition_users([5, 5], 4)
    assert sorted(sum(four, [])) == [0, 1] and sum(1 for p in four if not p) == 2


def test_merge_rejects_missing_or_duplicate_users():
    res = dict(accept_len=[1], out_offsets=[0, 2], out_tokens=[3, 4])
    with pytest.raises(ValueError):
        shard.merge_outputs(2, [[0], []], [res, dict(accept_len=[], out_offsets=[0], out_tokens=[])])
    with pytest.raises(ValueError):
        shard.merge_outputs(1, [[0], [0]], [res, res])


def test_position_rows():
    T = [2, 3, 1]
    assert shard.position_rows(T, [1]).tolist() == [2, 3, 4]
    assert shard.position_rows(T, [2, 0]).tolist() == [5, 0, 1]
    assert shard.position_rows(T, []).tolist() == []
    assert offsets(T).tolist() == [0, 2, 5, 6]
