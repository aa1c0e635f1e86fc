"""Sharding one verification batch over several GPUs, one process per GPU.

Users are independent in both stages of batch verification (Sec. II-A, the
server's stage 2): a user's attention reads only its own KV cache pages and
its own verify tokens, and speculative sampling decides a user's drafts from
that user's logit rows alone.  A batch therefore shards by users with no
collective on the data path: each rank verifies the members assigned to it
(`dipsd_verify_batch` takes batch membership as an argument), and the ranks'
per-user results (accept lengths and emitted tokens, a few KB) are gathered
on the host and packed in batch order.

Host-side logic only (plain Python and NumPy); the verification itself runs
in the library's kernels on each rank's GPU.
"""
from __future__ import annotations

from typing import List, Sequence

import numpy as np


def partition_users(kv_len: Sequence[int], world: int) -> List[List[int]]:
    """Assigns users (batch positions) to `world` ranks, balancing KV length.

    Longest first, each user to the rank with the least KV so far (ties to the
    lower rank), so the ranks' attention bytes differ by at most one user's KV.
    Each rank's list is in batch order; a rank may get no user.
    """
    if world < 1:
        raise ValueError("world must be >= 1")
    kv = np.asarray(kv_len, dtype=np.int64)
    load = np.zeros(world, dtype=np.int64)
    parts: List[List[int]] = [[] for _ in range(world)]
    for i in sorted(range(len(kv)), key=lambda u: (-int(kv[u]), u)):
        r = int(np.argmin(load))
        parts[r].append(i)
        load[r] += kv[i]
    return [sorted(p) for p in parts]


def position_rows(T: Sequence[int], users: Sequence[int]) -> np.ndarray:
    """Rows of the per-position tensors ([sum T] ...) that belong to `users`,
    in the given user order (T[i] = L_i + 1 verify positions of user i)."""
    off = np.concatenate([[0], np.cumsum(np.asarray(T, dtype=np.int64))])
    if len(users) == 0:
        return np.zeros(0, dtype=np.int64)
    return np.concatenate([np.arange(off[i], off[i + 1]) for i in users])


def merge_outputs(B: int, parts: Sequence[Sequence[int]], results: Sequence[dict]):
    """Packs per-rank results into the unsharded layout.

    parts[r] lists the batch positions rank r verified (in its own batch
    order) and results[r] holds that rank's `accept_len` [n_r],
    `out_offsets` [n_r + 1] and `out_tokens` [>= out_offsets[-1]].  Returns
    (accept_len [B], out_offsets [B + 1], out_tokens [sum (a_i + 1)]) with
    users in batch order, as one unsharded call would have produced.
    """
    acc = np.full(B, -1, dtype=np.int64)
    toks: List[np.ndarray] = [np.zeros(0, dtype=np.int64)] * B
    for users, res in zip(parts, results):
        a = np.asarray(res["accept_len"], dtype=np.int64)
        o = np.asarray(res["out_offsets"], dtype=np.int64)
        t = np.asarray(res["out_tokens"], dtype=np.int64)
        if len(users) != len(a) or len(o) != len(users) + 1:
            raise ValueError("result sizes do not match the rank's users")
        for k, i in enumerate(users):
            if acc[i] >= 0:
                raise ValueError(f"user {i} verified by two ranks")
            acc[i] = a[k]
            toks[i] = t[o[k]:o[k + 1]]
    if (acc < 0).any():
        raise ValueError("a user was verified by no rank")
    offs = np.concatenate([[0], np.cumsum([len(x) for x in toks])]).astype(np.int64)
    return acc, offs, np.concatenate(toks) if B else np.zeros(0, dtype=np.int64)


def aggregate_timing(total_ms: float, units: float, e2e_ms: float, device=None):
    """Whole-job figures over the ranks of the default process group: the
    slowest rank's device time and end-to-end time, and the units (emitted
    tokens) of all ranks.  Returns (total_ms_max, units_sum, e2e_ms_max)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(total_ms), float(units), float(e2e_ms)
    t = torch.tensor([total_ms, units, e2e_ms], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(t[1]), float(mx[2])
