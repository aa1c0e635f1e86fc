"""Oracle for the verify-attention step (test infrastructure only).

In one verification round the target model runs one forward pass over each
user's draft tokens (Sec. II-A, stage 2 "Batch Verification"; the cost
model Eq. (Fv) carries the matching I*L attention term).  Inside every
decoder block, user i's T_i = L_i + 1 verify tokens (the last emitted token
of the previous round plus the L_i drafts) attend causally to the C_i cached
tokens and to each other: verify token t sits at absolute position C_i + t
and sees keys 0 .. C_i + t.  Query head h reads KV head floor(h / G),
G = Hq / Hkv (grouped-query attention, consecutive query heads share a KV
head as in Qwen3).

The KV cache is paged: page p of user i holds tokens 16p .. 16p+15 of that
user and lives at cache block block_table[i][p].  The round's state update
writes the verify tokens' own keys and values into the pages (kv_append);
verify_attention reads the cache as it stands after that write.

Pins (tests/test_oracle_attention.py): torch's scaled_dot_product_attention
in fp64 on the gathered, GQA-expanded tensors; kv_len = 1 gives v_0; equal
keys give the running mean of the values; page-permutation invariance.
"""
from __future__ import annotations

import numpy as np

PAGE = 16


def gather_pages(cache: np.ndarray, table_row: np.ndarray, n_tokens: int) -> np.ndarray:
    """[num_blocks, Hkv, PAGE, D] cache + one block-table row -> [Hkv, n_tokens, D]."""
    n_pages = -(-n_tokens // PAGE)
    blocks = np.asarray(table_row[:n_pages], dtype=np.int64)
    x = cache[blocks]                                  # [n_pages, Hkv, PAGE, D]
    x = x.transpose(1, 0, 2, 3).reshape(cache.shape[1], n_pages * PAGE, cache.shape[3])
    return x[:, :n_tokens]


def kv_append(k_cache, v_cache, block_table, ctx, L, new_k, new_v, members=None):
    """Writes every user's T_i new key/value rows into its pages (the verify
    tokens join the cache in the same round, Sec. II-A stage 2).

    new_k, new_v  [sum_i T_i, Hkv, D], users concatenated in batch order;
                  verify token t of user i lands at position C_i + t, i.e.
                  block block_table[members[i]][(C_i + t) // 16], slot
                  (C_i + t) % 16.
    returns       updated copies of k_cache and v_cache
    """
    k = np.array(k_cache, copy=True)
    v = np.array(v_cache, copy=True)
    members = np.arange(len(L)) if members is None else np.asarray(members)
    n = 0
    for i in range(len(L)):
        row = np.asarray(block_table[int(members[i])])
        for t in range(int(L[i]) + 1):
            pos = int(ctx[i]) + t
            blk, slot = int(row[pos // PAGE]), pos % PAGE
            k[blk, :, slot, :] = new_k[n + t]
            v[blk, :, slot, :] = new_v[n + t]
        n += int(L[i]) + 1
    return k, v


def verify_attention(q, k_cache, v_cache, block_table, ctx, L, scale, members=None):
    """Causal GQA attention of every verify token over its user's paged cache.

    q           [sum_i T_i, Hq, D]  float64, users concatenated in batch order
    k_cache     [num_blocks, Hkv, PAGE, D] float64 (v_cache alike)
    block_table [rows, max_blocks] int; user i uses row members[i] (default i)
    ctx, L      [B] context length C_i and draft length L_i
    scale       softmax scale (D^-1/2 for the target model)
    returns     o [sum_i T_i, Hq, D] float64 with
                o[n, h] = sum_{j <= C_i + t} softmax_j(scale * q[n,h] . k_j) v_j
    """
    q = np.asarray(q, dtype=np.float64)
    B = len(L)
    Hq, Hkv = q.shape[1], k_cache.shape[1]
    G = Hq // Hkv
    members = np.arange(B) if members is None else np.asarray(members)
    out = np.empty_like(q)
    n0 = 0
    for i in range(B):
        T = int(L[i]) + 1
        kv_len = int(ctx[i]) + T
        row = np.asarray(block_table[int(members[i])])
        K = gather_pages(k_cache, row, kv_len).astype(np.float64)
        V = gather_pages(v_cache, row, kv_len).astype(np.float64)
        for t in range(T):
            visible = int(ctx[i]) + t + 1
            for h in range(Hq):
                kh = h // G
                s = (K[kh, :visible] @ q[n0 + t, h]) * scale
                w = np.exp(s - s.max())
                out[n0 + t, h] = (w @ V[kh, :visible]) / w.sum()
        n0 += T
    return out
