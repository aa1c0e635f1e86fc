"""Seeded synthetic batches for DiP-SD edge-server verification.

This module only draws random numbers and lays them out in the storage
formats both implementations consume (bf16 / fp32 tensors, int32 tables).
It holds none of the verification arithmetic: no softmax, no acceptance
test, no residual, no inverse CDF.  The CUDA path and the CPU oracle both
read the very tensors produced here.

Shapes follow the paper's verifier, Qwen3-32B (Sec. IV-A, Table 2: 64
decoder blocks, hidden 5120), whose attention has 64 query heads, 8 KV
heads and head_dim 128, vocabulary 151936.  Per-user quantities follow the
paper's problem statement (Sec. II-A, Table 1): prefix (context) length
i_m, integer draft length l_m, acceptance parameter alpha_m.

Recipe (seeded, reproducible):
  * block tables: every user's pages come from one seeded permutation of the
    page pool, so a user's pages are scattered, as in a real paged cache;
    unused table entries are -1.
  * K/V caches and Q: N(0,1) drawn by a seeded torch generator on the chosen
    device, rounded to bf16 (round-to-nearest-even).
  * target logits z: N(0, var) in fp64 (numpy), stored bf16 (or fp32).
  * draft logits w = z_stored + N(0, sigma_i^2), stored the same way.  For
    i.i.d. Gaussian logits and a large vocabulary the expected acceptance
    sum_v min(p_v, q_v) tends to 2*Phi(-sigma/2) whatever the logit scale,
    so sigma_i = -2 * Phi^{-1}(alpha_i / 2) targets alpha_i in closed form.
  * draft tokens d ~ softmax(w_stored), drawn with the Gumbel-max trick in
    fp64 from a seeded numpy stream (the drafting device's job, Sec. II-A
    step 1; not the verifier's arithmetic).
  * uniforms: two per verify position (acceptance, resample) from numpy's
    Philox4x64-10 stream keyed on (seed, user id): position t takes words 2t
    and 2t + 1, each mapped to ((w >> 41) + 0.5) * 2^-23, an exact fp32 in
    (0, 1).  The CUDA library draws the same words with its own Philox; the
    oracle reads these host copies.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch
from scipy.special import ndtri

PAGE = 16
QWEN3_32B = dict(Hq=64, Hkv=8, D=128, V=151936)


def round_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp64/fp32 -> bf16 bit patterns (uint16), round-to-nearest-even."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    b = b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))
    return (b >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_torch(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


def store_logits(x: np.ndarray, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        return bf16_bits_to_torch(round_bf16_bits(x))
    if dtype == "f32":
        return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    raise ValueError(dtype)


def philox_uniforms(seed: int, user_id: int, n: int) -> np.ndarray:
    """n uniforms in (0,1), exact fp32, from Philox keyed on (seed, user_id)."""
    bg = np.random.Philox(key=np.array([seed, user_id], dtype=np.uint64))
    raw = bg.random_raw(n) if n > 0 else np.zeros(0, dtype=np.uint64)
    k = (raw >> np.uint64(41)).astype(np.float64)
    return ((k + 0.5) * 2.0 ** -23).astype(np.float32)


def sigma_for_alpha(alpha):
    """Noise std that gives expected acceptance alpha for Gaussian logits."""
    return -2.0 * ndtri(np.asarray(alpha, dtype=np.float64) / 2.0)


def draft_len_for_alpha(alpha, lo: int, hi: int):
    """Draft length from the expected run of accepted drafts alpha/(1-alpha)."""
    a = np.asarray(alpha, dtype=np.float64)
    return np.clip(np.floor(a / (1.0 - a)), lo, hi).astype(np.int32)


def offsets(lengths) -> np.ndarray:
    """Exclusive prefix of lengths with the total appended ([B+1])."""
    o = np.zeros(len(lengths) + 1, dtype=np.int64)
    o[1:] = np.cumsum(np.asarray(lengths, dtype=np.int64))
    return o


@dataclass
class Batch:
    """One verification batch (one pipeline stage's users)."""
    L: np.ndarray            # int32 [B] draft length per batch user
    ctx: np.ndarray          # int32 [B] context (prefix) length before this round
    members: np.ndarray      # int32 [B] row of each batch user in block_table
    Hq: int
    Hkv: int
    D: int
    V: int
    logit_dtype: str         # "bf16" | "f32"
    q: torch.Tensor          # bf16 [sum T, Hq, D], T = L + 1
    k_cache: torch.Tensor    # bf16 [num_blocks, Hkv, PAGE, D]
    v_cache: torch.Tensor    # bf16 [num_blocks, Hkv, PAGE, D]
    block_table: torch.Tensor  # int32 [rows, max_blocks], -1 = unused
    target_logits: torch.Tensor  # [sum T, V]
    draft_logits: torch.Tensor   # [sum L, V]
    draft_tokens: torch.Tensor   # int32 [sum L]
    uniforms: torch.Tensor       # fp32 [sum T, 2]: (u_accept, u_resample), host, for the oracle
    alpha: np.ndarray = field(default=None)  # design acceptance per user
    seed: int = 0                # Philox key word 0
    user_ids: np.ndarray = field(default=None)  # int32 [B]: Philox key word 1 per batch user

    @property
    def B(self) -> int:
        return int(self.L.shape[0])

    @property
    def T(self) -> np.ndarray:
        return (self.L + 1).astype(np.int32)

    @property
    def kv_len(self) -> np.ndarray:
        return (self.ctx + self.L + 1).astype(np.int32)

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.D)

    @property
    def sum_T(self) -> int:
        return int(self.T.sum())

    @property
    def sum_L(self) -> int:
        return int(self.L.sum())

    def kv_bytes(self) -> int:
        return int(self.kv_len.sum()) * self.Hkv * self.D * 2 * 2


def _block_tables(rng, kv_len, spare):
    pages = [-(-int(n) // PAGE) for n in kv_len]
    total = int(sum(pages))
    num_blocks = total + spare
    perm = rng.permutation(num_blocks).astype(np.int32)
    max_blocks = max(pages) if pages else 1
    bt = np.full((len(pages), max_blocks), -1, dtype=np.int32)
    o = 0
    for i, n in enumerate(pages):
        bt[i, :n] = perm[o:o + n]
        o += n
    return bt, num_blocks


def _randn_bf16(shape, seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


def make_spec_inputs(rng, L, user_ids, V, logit_std, noise_sigma, logit_dtype, seed):
    """Target/draft logits, draft tokens and uniforms for one batch."""
    L = np.asarray(L, dtype=np.int32)
    T = L + 1
    sT, sL = int(T.sum()), int(L.sum())
    z = rng.normal(0.0, logit_std, size=(sT, V))
    zt = store_logits(z, logit_dtype)
    z_stored = zt.double().numpy()
    qo, lo = offsets(T), offsets(L)
    w = np.empty((sL, V), dtype=np.float64)
    sig = np.broadcast_to(np.asarray(noise_sigma, dtype=np.float64), L.shape)
    for i in range(len(L)):
        for t in range(int(L[i])):
            w[lo[i] + t] = z_stored[qo[i] + t] + rng.normal(0.0, sig[i], size=V)
    wt = store_logits(w, logit_dtype)
    w_stored = wt.double().numpy()
    # Gumbel-max: argmax(w + G) is an exact draw from softmax(w).
    d = np.empty(sL, dtype=np.int32)
    for r in range(sL):
        u = rng.random(V)
        np.clip(u, 1e-300, None, out=u)
        d[r] = int(np.argmax(w_stored[r] - np.log(-np.log(u))))
    uni = np.empty((sT, 2), dtype=np.float32)
    for i in range(len(L)):
        u = philox_uniforms(seed, int(user_ids[i]), 2 * int(T[i]))
        uni[qo[i]:qo[i + 1]] = u.reshape(int(T[i]), 2)
    return zt, wt, torch.from_numpy(d), torch.from_numpy(uni)


@dataclass
class SparseDraft:
    """A sparse draft payload: per draft row, K support tokens with their draft
    probabilities, the draft token drawn from them, and its log-probability."""
    topk_idx: torch.Tensor     # int32 [sum L, K], distinct tokens
    topk_q: torch.Tensor       # fp32 [sum L, K], >= 0, summing to ~1 per row
    draft_tokens: torch.Tensor  # int32 [sum L]
    draft_logq: torch.Tensor   # fp32 [sum L]: log of the stored q of the draft token


def make_sparse_draft(b: "Batch", K: int, seed: int = 0, rank_noise: float = 1.0, device="cpu") -> SparseDraft:
    """The device's side of a sparse payload for batch b: per draft row the K
    tokens ranked highest by (stored target logit + Gaussian noise), Dirichlet(1)
    probabilities sorted so the best-ranked token gets the largest, and a draft
    token drawn from them (numpy's categorical sampler, the device's job)."""
    rng = np.random.default_rng([seed, 77])
    z = b.target_logits.double().cpu().numpy()
    qo, lo = offsets(b.T), offsets(b.L)
    sL = int(b.L.sum())
    idx = np.zeros((sL, K), dtype=np.int32)
    qv = np.zeros((sL, K), dtype=np.float32)
    d = np.zeros(sL, dtype=np.int32)
    logq = np.zeros(sL, dtype=np.float32)
    for i in range(b.B):
        for t in range(int(b.L[i])):
            r = lo[i] + t
            score = z[qo[i] + t] + rng.normal(0.0, rank_noise, size=z.shape[1])
            top = np.argpartition(-score, K - 1)[:K]
            top = top[np.argsort(-score[top])]
            idx[r] = top
            qv[r] = np.sort(rng.dirichlet(np.ones(K)))[::-1].astype(np.float32)
            pr = qv[r].astype(np.float64)
            j = int(rng.choice(K, p=pr / pr.sum()))
            d[r] = top[j]
            logq[r] = np.float32(np.log(np.float64(qv[r, j])))
    return SparseDraft(topk_idx=torch.from_numpy(idx).to(device), topk_q=torch.from_numpy(qv).to(device),
                       draft_tokens=torch.from_numpy(d).to(device), draft_logq=torch.from_numpy(logq).to(device))


def make_batch(L, ctx, *, Hq, Hkv, D, V, logit_std=1.0, noise_sigma=1.0,
               logit_dtype="bf16", seed=0, device="cpu", kv_device=None,
               alpha=None, spare_pages=3, user_ids=None, spec_only=False) -> Batch:
    """Build one batch from explicit per-user draft and context lengths.

    spec_only=True skips the KV cache, block table and Q (the speculative
    sampling inputs are identical either way).
    """
    L = np.asarray(L, dtype=np.int32)
    ctx = np.asarray(ctx, dtype=np.int32)
    B = int(L.shape[0])
    kv_device = kv_device or device
    rng = np.random.default_rng([seed, 1])
    kv_len = ctx + L + 1
    bt, num_blocks = _block_tables(rng, kv_len, spare_pages)
    if spec_only:
        k_cache = v_cache = q = None
    else:
        k_cache = _randn_bf16((num_blocks, Hkv, PAGE, D), seed * 7919 + 11, kv_device)
        v_cache = _randn_bf16((num_blocks, Hkv, PAGE, D), seed * 7919 + 13, kv_device)
        q = _randn_bf16((int((L + 1).sum()), Hq, D), seed * 7919 + 17, "cpu").to(device)
    uid = np.arange(B, dtype=np.int32) if user_ids is None else np.asarray(user_ids, np.int32)
    srng = np.random.default_rng([seed, 2])
    zt, wt, d, uni = make_spec_inputs(srng, L, uid, V, logit_std, noise_sigma, logit_dtype, seed)
    return Batch(L=L, ctx=ctx, members=np.arange(B, dtype=np.int32), Hq=Hq, Hkv=Hkv, D=D, V=V,
                 logit_dtype=logit_dtype, q=q, k_cache=k_cache, v_cache=v_cache,
                 block_table=torch.from_numpy(bt).to(device),
                 target_logits=zt.to(device), draft_logits=wt.to(device),
                 draft_tokens=d.to(device), uniforms=uni,
                 alpha=None if alpha is None else np.asarray(alpha, np.float64), seed=seed, user_ids=uid)


# ----------------------------------------------------------------------------
# The five workloads.  Gaussian parameters are written N(mean, variance).
# ----------------------------------------------------------------------------

CONFIG_NAMES = {
    1: "tiny: B=4, L=[1,2,3,4], ctx 128, 4/1/64 heads, V=1024, fp32 logits",
    2: "qwen3-32b verify: B=8, L~U{1..8}, ctx 1024, 64/8/128, V=151936, bf16 paged KV",
    3: "ragged: B=32, L from alpha~U(0.5,0.9), ctx log-U[512,8192], Qwen3-32B shapes",
    4: "long context: B=64, L~U{2..6}, ctx 32768, Qwen3-32B shapes",
    5: "pipelined: 4 batches x 32 users, L from alpha~U(0.4,0.95), ctx log-U[256,16384]",
}


def config_shape(cfg: int, seed: int = 0):
    """Per-user lengths and generator parameters of a workload (no tensors)."""
    rng = np.random.default_rng([seed, 0])
    if cfg == 1:
        return dict(L=np.array([1, 2, 3, 4], np.int32), ctx=np.full(4, 128, np.int32),
                    Hq=4, Hkv=1, D=64, V=1024, logit_std=1.0,
                    noise_sigma=math.sqrt(0.5), logit_dtype="f32",
                    alpha=np.full(4, float(2 * _ndtr(-math.sqrt(0.5) / 2))))
    if cfg == 2:
        L = rng.integers(1, 9, size=8).astype(np.int32)
        return dict(L=L, ctx=np.full(8, 1024, np.int32), **QWEN3_32B,
                    logit_std=math.sqrt(3.0), noise_sigma=1.0, logit_dtype="bf16",
                    alpha=np.full(8, float(2 * _ndtr(-0.5))))
    if cfg == 3:
        alpha = rng.uniform(0.5, 0.9, size=32)
        L = draft_len_for_alpha(alpha, 0, 10)
        ctx = np.exp(rng.uniform(math.log(512), math.log(8192), size=32)).astype(np.int32)
        return dict(L=L, ctx=ctx, **QWEN3_32B, logit_std=1.0,
                    noise_sigma=sigma_for_alpha(alpha), logit_dtype="bf16", alpha=alpha)
    if cfg == 4:
        L = rng.integers(2, 7, size=64).astype(np.int32)
        return dict(L=L, ctx=np.full(64, 32768, np.int32), **QWEN3_32B,
                    logit_std=math.sqrt(3.0), noise_sigma=1.0, logit_dtype="bf16",
                    alpha=np.full(64, float(2 * _ndtr(-0.5))))
    if cfg == 5:
        alpha = rng.uniform(0.4, 0.95, size=128)
        L = draft_len_for_alpha(alpha, 1, 10)
        ctx = np.exp(rng.uniform(math.log(256), math.log(16384), size=128)).astype(np.int32)
        return dict(L=L, ctx=ctx, **QWEN3_32B, logit_std=1.0,
                    noise_sigma=sigma_for_alpha(alpha), logit_dtype="bf16", alpha=alpha,
                    n_batches=4)
    raise ValueError(f"unknown workload {cfg}")


def _ndtr(x):
    return 0.5 * math.erfc(-x / math.sqrt(2.0))


def make_config(cfg: int, seed: int = 0, device="cpu", kv_device=None, spec_only=False):
    """Workload 1-4 as one Batch; workload 5 as a list of 4 Batches sharing one KV pool."""
    s = config_shape(cfg, seed)
    if cfg != 5:
        return make_batch(s["L"], s["ctx"], Hq=s["Hq"], Hkv=s["Hkv"], D=s["D"], V=s["V"],
                          logit_std=s["logit_std"], noise_sigma=s["noise_sigma"],
                          logit_dtype=s["logit_dtype"], seed=seed, device=device,
                          kv_device=kv_device, alpha=s["alpha"], spec_only=spec_only)
    return make_pipeline(s, seed, device, kv_device)


def make_pipeline(s, seed, device, kv_device):
    """128 users in one KV pool; the users are dealt into n_batches stages."""
    kv_device = kv_device or device
    L, ctx, alpha = s["L"], s["ctx"], s["alpha"]
    M = int(L.shape[0])
    nb = s["n_batches"]
    rng = np.random.default_rng([seed, 1])
    bt, num_blocks = _block_tables(rng, ctx + L + 1, 3)
    k_cache = _randn_bf16((num_blocks, s["Hkv"], PAGE, s["D"]), seed * 7919 + 11, kv_device)
    v_cache = _randn_bf16((num_blocks, s["Hkv"], PAGE, s["D"]), seed * 7919 + 13, kv_device)
    bt_t = torch.from_numpy(bt).to(device)
    order = np.random.default_rng([seed, 3]).permutation(M).astype(np.int32)
    batches = []
    for n in range(nb):
        mem = np.sort(order[n * (M // nb):(n + 1) * (M // nb)])
        Lb, cb = L[mem], ctx[mem]
        q = _randn_bf16((int((Lb + 1).sum()), s["Hq"], s["D"]), seed * 7919 + 101 + n, "cpu")
        srng = np.random.default_rng([seed, 10 + n])
        zt, wt, d, uni = make_spec_inputs(srng, Lb, mem, s["V"], s["logit_std"],
                                          s["noise_sigma"][mem], s["logit_dtype"], seed)
        batches.append(Batch(L=Lb, ctx=cb, members=mem, Hq=s["Hq"], Hkv=s["Hkv"], D=s["D"],
                             V=s["V"], logit_dtype=s["logit_dtype"], q=q.to(device),
                             k_cache=k_cache, v_cache=v_cache, block_table=bt_t,
                             target_logits=zt.to(device), draft_logits=wt.to(device),
                             draft_tokens=d.to(device), uniforms=uni,
                             alpha=alpha[mem], seed=seed, user_ids=mem.astype(np.int32)))
    return batches
