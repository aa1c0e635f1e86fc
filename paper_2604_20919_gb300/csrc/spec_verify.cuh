// spec_verify: speculative sampling over the vocabulary for a batch of users
// (Sec. II-A stage 2: accept/reject every draft, truncate at the first
// rejection, emit one more token from the residual or, at the bonus position,
// from the target distribution).  Staged path for 16-byte aligned rows.
//
// Pass 1 (spec_stats_kernel) -- one thread-block cluster per verify position.
// Each CTA owns a slice of the target-logit row (and of the draft-logit row at
// draft positions); each of its warps bulk-copies one contiguous chunk of the
// slice into shared memory (TMA bulk engine, one mbarrier per warp) and starts
// as soon as its chunk lands.  A lane takes its maximum m, picks the integer
// reference c = ceil(m log2 e) and sums 2^(x log2 e - c) (one FFMA and one
// ex2 per logit, compensated per 8-logit vector).  Because references are
// integers, every rescale between lanes, warps, CTAs and cluster ranks is an
// exact power of two; partial sums combine as float-float pairs and the row
// normaliser is kept in fp64.  Rank 0 then forms p_t(d), q_t(d) with an
// accurate exp and takes the acceptance decision u_acc * q_t(d) < p_t(d).
//
// Pass 2 (spec_sample_kernel) -- one cluster per user.  Warp ballots over the
// acceptance bits give a_i and the packed output offset.  The slices of the
// rows at position a_i are staged the same way; weights (max(0, p - q) up to a
// common factor, or p at the bonus position) use an accurate exp against the
// pass-1 references.  Each warp scans its chunk in groups of 32 vectors (256
// tokens), keeping every group total; slice totals are exchanged through
// distributed shared memory, and the CTA holding u * total descends slice ->
// warp -> group -> lane -> token using the very same fp32 partial sums, so the
// descent always lands in the cell the totals point to.
#pragma once

#include "spec_common.cuh"

namespace dipsd {

constexpr float kLog2e = 1.4426950408889634f;
// log2(e) = kLog2eHi + kLog2eLo (the fp32 rounding and its remainder).
constexpr float kLog2eHi = 1.44269502162933349609375f;
constexpr float kLog2eLo = 1.925963033500651e-8f;
// ln 2 = kLn2Hi + kLn2Lo; kLn2Hi has 16 significant bits, so c * kLn2Hi is
// exact for integers |c| < 2^8 (Cody and Waite's argument reduction).
constexpr float kLn2Hi = 0.693145751953125f;
constexpr float kLn2Lo = 1.42860682030941723212e-6f;
constexpr int kEmptyRef = -(1 << 29);
constexpr int kMaxGroups = 32;  // 32-vector groups per warp chunk
constexpr int kStagedThreads = 512;
constexpr int kStagedWarps = kStagedThreads / 32;

// Row statistics of one verify position, relative to integer references:
// sz = sum_v 2^(z_v log2 e - cz), sw likewise for the draft row.
struct SpecStat {
  double sz, sw;
  int cz, cw;
  int pad0, pad1;
};

// --------------------------------------------------------- float-float sums
struct FF {
  float hi, lo;
};
__device__ __forceinline__ FF ff_add(FF a, FF b) {
  const float s = __fadd_rn(a.hi, b.hi);
  const float bb = __fsub_rn(s, a.hi);
  const float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, bb)), __fsub_rn(b.hi, bb));
  const float lo = __fadd_rn(__fadd_rn(a.lo, b.lo), e);
  const float hi = __fadd_rn(s, lo);
  return FF{hi, __fsub_rn(lo, __fsub_rn(hi, s))};
}
__device__ __forceinline__ FF ff_scale(FF a, int k) { return FF{scalbnf(a.hi, k), scalbnf(a.lo, k)}; }

// (reference, float-float sum) pairs combine by exact power-of-two rescaling.
struct RefSum {
  int c;
  FF s;
};
__device__ __forceinline__ RefSum refsum_add(RefSum a, RefSum b) {
  const int c = max(a.c, b.c);
  FF x = a.c == kEmptyRef ? FF{0.f, 0.f} : ff_scale(a.s, a.c - c);
  FF y = b.c == kEmptyRef ? FF{0.f, 0.f} : ff_scale(b.s, b.c - c);
  return RefSum{c, ff_add(x, y)};
}
__device__ __forceinline__ RefSum warp_refsum(RefSum v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    RefSum w;
    w.c = __shfl_xor_sync(0xffffffffu, v.c, o);
    w.s.hi = __shfl_xor_sync(0xffffffffu, v.s.hi, o);
    w.s.lo = __shfl_xor_sync(0xffffffffu, v.s.lo, o);
    v = refsum_add(v, w);
  }
  return v;
}

__device__ __forceinline__ float fast_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 2^(x log2 e - c) = e^(x - c ln 2) for an integer reference c: the one form
// used for the row sums, the acceptance test and the sampling weights, so
// every normalised probability sees the same function of x.
__device__ __forceinline__ float ex2_ref(float x, float cf) {
  return fast_ex2(__fmaf_rn(x, kLog2eLo, __fmaf_rn(x, kLog2eHi, -cf)));
}
__device__ __forceinline__ float ex2_ref(float x, int c) { return ex2_ref(x, static_cast<float>(c)); }

// ---------------------------------------------------------- slice staging
// Slice of CTA `rank` in units of 16-byte vectors, and the chunk of warp w.
__device__ __forceinline__ void slice_bounds(int nvec, uint32_t rank, uint32_t csize, int& sb, int& se) {
  sb = static_cast<int>((static_cast<long long>(rank) * nvec) / csize);
  se = static_cast<int>((static_cast<long long>(rank + 1) * nvec) / csize);
}
__device__ __forceinline__ void chunk_bounds(int sb, int se, int w, int& cb, int& ce) {
  cb = sb + static_cast<int>((static_cast<long long>(w) * (se - sb)) / kStagedWarps);
  ce = sb + static_cast<int>((static_cast<long long>(w + 1) * (se - sb)) / kStagedWarps);
}

// Lane 0 of each warp stages its chunk of up to two rows and arms the warp's
// barrier; returns after the lane's copies are issued (not completed).
// Number of 32-vector groups in warp w's chunk of slice [sb, se).
__device__ __forceinline__ int ngroups_of(int sb, int se, int w) {
  int cb, ce;
  chunk_bounds(sb, se, w, cb, ce);
  return (ce - cb + 31) / 32;
}

template <typename T>
__device__ __forceinline__ void stage_chunk(uint64_t* bar, uint8_t* zbuf, uint8_t* wbuf, const T* zrow,
                                            const T* wrow, bool two, int sb, int cb, int ce) {
  const uint32_t bytes = static_cast<uint32_t>(ce - cb) * 16u;
  const uint32_t off = static_cast<uint32_t>(cb - sb) * 16u;
  mbar_init(bar, 1);
  fence_mbar_init();
  mbar_arrive_expect_tx(bar, two ? 2 * bytes : bytes);
  if (bytes) {
    bulk_load(zbuf + off, reinterpret_cast<const uint8_t*>(zrow) + static_cast<size_t>(cb) * 16, bytes, bar);
    if (two) bulk_load(wbuf + off, reinterpret_cast<const uint8_t*>(wrow) + static_cast<size_t>(cb) * 16, bytes, bar);
  }
}

template <typename T>
struct Vec16;
template <>
struct Vec16<__nv_bfloat16> {
  static constexpr int N = 8;
  static __device__ __forceinline__ void load(const uint8_t* p, float (&x)[8]) {
    const uint4 r = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      x[2 * k] = __uint_as_float(w[k] << 16);
      x[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
    }
  }
};
template <>
struct Vec16<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void load(const uint8_t* p, float (&x)[4]) {
    const float4 r = *reinterpret_cast<const float4*>(p);
    x[0] = r.x; x[1] = r.y; x[2] = r.z; x[3] = r.w;
  }
};

// Lane partial sum of 2^(x log2 e - c) over its vectors of a staged chunk
// (vectors lane, lane + 32, ...; two in flight per step).
template <typename T>
__device__ __forceinline__ float vec_ex2_sum(const float (&x)[Vec16<T>::N], float cf) {
  constexpr int N = Vec16<T>::N;
  float e[N];
#pragma unroll
  for (int k = 0; k < N; ++k) e[k] = ex2_ref(x[k], cf);
  if constexpr (N == 8) {
    return ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
  } else {
    return (e[0] + e[1]) + (e[2] + e[3]);
  }
}

template <typename T>
__device__ __forceinline__ RefSum lane_refsum(const uint8_t* buf, int n_local, int lane) {
  constexpr int N = Vec16<T>::N;
  float m0 = -INFINITY, m1 = -INFINITY;
  int v = lane;
  for (; v + 32 < n_local; v += 64) {
    float x[N], y[N];
    Vec16<T>::load(buf + v * 16, x);
    Vec16<T>::load(buf + (v + 32) * 16, y);
#pragma unroll
    for (int e = 0; e < N; ++e) {
      m0 = fmaxf(m0, x[e]);
      m1 = fmaxf(m1, y[e]);
    }
  }
  if (v < n_local) {
    float x[N];
    Vec16<T>::load(buf + v * 16, x);
#pragma unroll
    for (int e = 0; e < N; ++e) m0 = fmaxf(m0, x[e]);
  }
  const float m = fmaxf(m0, m1);
  if (!(m > -INFINITY)) return RefSum{kEmptyRef, FF{0.f, 0.f}};
  const float cf = fminf(fmaxf(ceilf(m * kLog2e), -1048576.f), 1048576.f);
  KahanSum acc;
  v = lane;
  for (; v + 32 < n_local; v += 64) {
    float x[N], y[N];
    Vec16<T>::load(buf + v * 16, x);
    Vec16<T>::load(buf + (v + 32) * 16, y);
    const float sx = vec_ex2_sum<T>(x, cf);
    const float sy = vec_ex2_sum<T>(y, cf);
    acc.add(sx + sy);
  }
  if (v < n_local) {
    float x[N];
    Vec16<T>::load(buf + v * 16, x);
    acc.add(vec_ex2_sum<T>(x, cf));
  }
  return RefSum{static_cast<int>(cf), FF{acc.s, -acc.c}};
}

// ------------------------------------------------------------------ pass 1
template <typename T, int CAP>
__global__ void __launch_bounds__(kStagedThreads)
spec_stats_kernel(const __grid_constant__ SpecParams<CAP> p, int slice_bytes) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ uint64_t bars[kStagedWarps];
  __shared__ RefSum red[2][kStagedWarps];
  __shared__ float4 cl_slot[kMaxCluster][2];
  const uint32_t crank = cluster_ctarank();
  const uint32_t csize = cluster_nctarank();
  cluster_arrive_relaxed();  // phase A: every CTA of the cluster has started

  const int n = blockIdx.x / csize;  // verify position
  const int ui = spec_find_user<CAP>(p.q_off, p.B, n);
  const int t = n - p.q_off[ui];
  const int Li = p.q_off[ui + 1] - p.q_off[ui] - 1;
  const bool has_q = t < Li;
  const int wrow = p.l_off[ui] + t;
  const T* zrow = static_cast<const T*>(p.z) + static_cast<size_t>(n) * p.V;
  const T* wrow_p = static_cast<const T*>(p.w) + static_cast<size_t>(has_q ? wrow : 0) * p.V;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int sb, se, cb, ce;
  slice_bounds(p.nvec, crank, csize, sb, se);
  chunk_bounds(sb, se, warp, cb, ce);
  uint8_t* zbuf = smem;
  uint8_t* wbuf = smem + slice_bytes;

  pdl_wait_prior_grid();
  pdl_launch_dependents();
  if (lane == 0) stage_chunk<T>(&bars[warp], zbuf, wbuf, zrow, wrow_p, has_q, sb, cb, ce);
  __syncwarp();
  // rank 0 fetches the draft token's two logits now; they are used at the end
  int d = -1;
  float zd = 0.f, wd = 0.f;
  if (crank == 0 && threadIdx.x == 0 && has_q) {
    d = p.draft_tokens[wrow];
    if (d >= 0 && d < p.V) {
      zd = load_elem<T>(zrow, d);
      wd = load_elem<T>(wrow_p, d);
    }
  }
  const bool ok = mbar_wait(&bars[warp], 0, p.status);

  RefSum rz{kEmptyRef, FF{0.f, 0.f}}, rw{kEmptyRef, FF{0.f, 0.f}};
  if (ok) {
    const int off = (cb - sb) * 16;
    rz = lane_refsum<T>(zbuf + off, ce - cb, lane);
    if (has_q) rw = lane_refsum<T>(wbuf + off, ce - cb, lane);
  }
  rz = warp_refsum(rz);
  rw = warp_refsum(rw);
  if (lane == 0) {
    red[0][warp] = rz;
    red[1][warp] = rw;
  }
  __syncthreads();
  cluster_wait_acquire();  // phase A complete: rank 0 is running
  if (threadIdx.x == 0) {
    RefSum az = red[0][0], aw = red[1][0];
    for (int k = 1; k < kStagedWarps; ++k) {
      az = refsum_add(az, red[0][k]);
      aw = refsum_add(aw, red[1][k]);
    }
    const uint32_t dst = dsmem_map(&cl_slot[crank][0], 0);
    dsmem_st_f32x4(dst, __int_as_float(az.c), az.s.hi, az.s.lo, 0.f);
    dsmem_st_f32x4(dst + 16, __int_as_float(aw.c), aw.s.hi, aw.s.lo, 0.f);
  }
  cluster_arrive_release();  // phase B: slices delivered to rank 0
  cluster_wait_acquire();
  if (crank != 0 || threadIdx.x != 0) return;

  RefSum az{kEmptyRef, FF{0.f, 0.f}}, aw{kEmptyRef, FF{0.f, 0.f}};
  for (uint32_t k = 0; k < csize; ++k) {
    const float4 a = cl_slot[k][0], b = cl_slot[k][1];
    az = refsum_add(az, RefSum{__float_as_int(a.x), FF{a.y, a.z}});
    aw = refsum_add(aw, RefSum{__float_as_int(b.x), FF{b.y, b.z}});
  }
  SpecStat st;
  st.sz = static_cast<double>(az.s.hi) + static_cast<double>(az.s.lo);
  st.sw = static_cast<double>(aw.s.hi) + static_cast<double>(aw.s.lo);
  st.cz = az.c;
  st.cw = aw.c;
  st.pad0 = st.pad1 = 0;
  static_cast<SpecStat*>(p.stats)[n] = st;
  float pd = 0.f, qd = 0.f;
  unsigned char flag = 0;
  if (has_q) {
    if (d >= 0 && d < p.V) {
      const float ez = ex2_ref(zd, st.cz);
      const float ew = ex2_ref(wd, st.cw);
      pd = ez * (1.f / static_cast<float>(st.sz));
      qd = ew * (1.f / static_cast<float>(st.sw));
      // u * q(d) < p(d), i.e. u * ew * sz < ez * sw (products in fp64, no division)
      flag = static_cast<double>(p.uniforms[2 * n]) * static_cast<double>(ew) * st.sz <
                     static_cast<double>(ez) * st.sw ? 1 : 0;
    } else {
      atomicOr(p.status, kDevErrBadToken);
    }
  }
  p.flags[n] = flag;
  if (p.draft_probs) reinterpret_cast<float2*>(p.draft_probs)[n] = make_float2(pd, qd);
}

// Sampling weight of one 16-byte vector: (p - q)^+ up to the common factor
// 1/sz (residual), or p up to 1/sz (bonus).  Written with explicit rounding
// so every evaluation of the same vector yields the same bits.
template <typename T>
__device__ __forceinline__ void vec_weights(const uint8_t* zb, const uint8_t* wb, int v, bool residual, int cz,
                                            int cw, float khi, float klo, float (&wt)[Vec16<T>::N]) {
  constexpr int N = Vec16<T>::N;
  float xz[N];
  Vec16<T>::load(zb + v * 16, xz);
  if (residual) {
    float xw[N];
    Vec16<T>::load(wb + v * 16, xw);
#pragma unroll
    for (int e = 0; e < N; ++e) {
      const float ez = ex2_ref(xz[e], cz);
      const float ew = ex2_ref(xw[e], cw);
      const float q = __fmaf_rn(ew, khi, __fmul_rn(ew, klo));
      wt[e] = fmaxf(__fsub_rn(ez, q), 0.f);
    }
  } else {
#pragma unroll
    for (int e = 0; e < N; ++e) wt[e] = ex2_ref(xz[e], cz);
  }
}

// ------------------------------------------------------------------ pass 2
template <typename T, int CAP>
__global__ void __launch_bounds__(kStagedThreads)
spec_sample_kernel(const __grid_constant__ SpecParams<CAP> p, int slice_bytes) {
  constexpr int N = Vec16<T>::N;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ uint64_t bars[kStagedWarps];
  __shared__ float gsum[kStagedWarps][kMaxGroups];
  __shared__ double wsum[kStagedWarps];
  __shared__ double slice_sum[2][kMaxCluster];
  __shared__ int s_off, s_a, s_cnt[kStagedWarps];
  __shared__ int s_sel[4];
  __shared__ double s_before, s_target;
  __shared__ float s_k[2];
  const uint32_t crank = cluster_ctarank();
  const uint32_t csize = cluster_nctarank();
  cluster_arrive_relaxed();  // phase A: every CTA has started

  const int ui = blockIdx.x / csize;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait_prior_grid();
  pdl_launch_dependents();

  // a_i and the packed offset sum_{j<i} (a_j + 1), by warp ballots
  int cnt = 0;
  for (int j = warp; j < ui; j += kStagedWarps) cnt += accepted_prefix<CAP>(p, j, lane) + 1;
  if (lane == 0) s_cnt[warp] = cnt;
  if (warp == 0) {
    const int a = accepted_prefix<CAP>(p, ui, lane);
    if (lane == 0) s_a = a;
  }
  __syncthreads();
  const int q0 = p.q_off[ui], l0 = p.l_off[ui];
  const int Li = p.q_off[ui + 1] - q0 - 1;
  if (threadIdx.x == 0) {
    int o = 0;
    for (int k = 0; k < kStagedWarps; ++k) o += s_cnt[k];
    s_off = o;
    // scale of q relative to p in the residual, split into two floats
    const SpecStat st0 = static_cast<const SpecStat*>(p.stats)[q0 + s_a];
    const double kd = s_a < Li ? st0.sz / st0.sw : 0.0;
    const float kh = static_cast<float>(kd);
    s_k[0] = kh;
    s_k[1] = static_cast<float>(kd - static_cast<double>(kh));
  }
  __syncthreads();
  const int a = s_a, off = s_off;
  if (crank == 0) {
    for (int k = threadIdx.x; k < a; k += kStagedThreads) p.out_tokens[off + k] = p.draft_tokens[l0 + k];
    if (threadIdx.x == 0) {
      p.accept_len[ui] = a;
      p.out_offsets[ui] = off;
      if (ui == p.B - 1) p.out_offsets[p.B] = off + a + 1;
    }
  }

  // stage the rows of position a
  const int n = q0 + a;
  bool residual = a < Li;
  const SpecStat st = static_cast<const SpecStat*>(p.stats)[n];
  const T* zrow = static_cast<const T*>(p.z) + static_cast<size_t>(n) * p.V;
  const T* wrow = static_cast<const T*>(p.w) + static_cast<size_t>(residual ? l0 + a : 0) * p.V;
  int sb, se, cb, ce;
  slice_bounds(p.nvec, crank, csize, sb, se);
  chunk_bounds(sb, se, warp, cb, ce);
  uint8_t* zbuf = smem;
  uint8_t* wbuf = smem + slice_bytes;
  if (lane == 0) stage_chunk<T>(&bars[warp], zbuf, wbuf, zrow, wrow, residual, sb, cb, ce);
  __syncwarp();
  const bool ok = mbar_wait(&bars[warp], 0, p.status);

  const float khi = s_k[0], klo = s_k[1];
  const float u = p.uniforms[2 * n + 1];
  const int nloc = ce - cb;
  const uint8_t* zc = zbuf + (cb - sb) * 16;
  const uint8_t* wc = wbuf + (cb - sb) * 16;
  const int ngroups = (nloc + 31) / 32;

  // one pass per candidate distribution: the residual, then p if it is empty
  for (int round = 0; round < 2; ++round) {
    FF wtot{0.f, 0.f};
    if (ok) {
      for (int g = 0; g < ngroups; ++g) {
        const int v = g * 32 + lane;
        float ls = 0.f;
        if (v < nloc) {
          float wt[N];
          vec_weights<T>(zc, wc, v, residual, st.cz, st.cw, khi, klo, wt);
#pragma unroll
          for (int e = 0; e < N; ++e) ls = __fadd_rn(ls, wt[e]);
        }
        float incl = ls;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl = __fadd_rn(incl, y);
        }
        const float gt = __shfl_sync(0xffffffffu, incl, 31);
        if (lane == 0 && g < kMaxGroups) gsum[warp][g] = gt;
        wtot = ff_add(wtot, FF{gt, 0.f});
      }
    }
    if (lane == 0) wsum[warp] = static_cast<double>(wtot.hi) + static_cast<double>(wtot.lo);
    __syncthreads();
    if (round == 0) cluster_wait_acquire();  // phase A complete: all CTAs running
    if (threadIdx.x == 0) {
      double s = 0.0;
      for (int k = 0; k < kStagedWarps; ++k) s += wsum[k];
      for (uint32_t r = 0; r < csize; ++r) dsmem_st_f64(dsmem_map(&slice_sum[round][crank], r), s);
    }
    cluster_arrive_release();
    cluster_wait_acquire();

    // One thread finds the slice, warp and group holding u * total (if
    // rounding leaves none: the last positive weight at every level) and
    // publishes them; the other threads wait at the barrier.
    if (threadIdx.x == 0) {
      double total = 0.0;
      for (uint32_t r = 0; r < csize; ++r) total += slice_sum[round][r];
      int mode = 0;  // 0: crossing, 1: last positive weight, 2: empty distribution
      int cs = static_cast<int>(csize) - 1, ws = kStagedWarps - 1, gs = ngroups - 1;
      double before = 0.0, target = 0.0;
      if (!(total > 0.0)) {
        mode = 2;
      } else {
        target = static_cast<double>(u) * total;
        mode = 1;
        for (uint32_t r = 0; r < csize; ++r) {
          if (before + slice_sum[round][r] > target) { cs = static_cast<int>(r); mode = 0; break; }
          before += slice_sum[round][r];
        }
        if (mode == 1) {
          while (cs > 0 && !(slice_sum[round][cs] > 0.0)) --cs;
          before = 0.0;
        }
        if (cs == static_cast<int>(crank)) {
          if (mode == 0) {
            mode = 1;
            for (int k = 0; k < kStagedWarps; ++k) {
              if (before + wsum[k] > target) { ws = k; mode = 0; break; }
              before += wsum[k];
            }
          }
          if (mode == 1) {
            while (ws > 0 && !(wsum[ws] > 0.0)) --ws;
          } else {
            const int wng = min(ngroups_of(sb, se, ws), kMaxGroups);
            mode = 1;
            for (int g = 0; g < wng; ++g) {
              if (before + static_cast<double>(gsum[ws][g]) > target) { gs = g; mode = 0; break; }
              before += static_cast<double>(gsum[ws][g]);
            }
          }
          if (mode == 1) {
            gs = min(ngroups_of(sb, se, ws), kMaxGroups) - 1;
            while (gs > 0 && !(gsum[ws][gs] > 0.f)) --gs;
          }
        }
      }
      s_sel[0] = mode;
      s_sel[1] = cs;
      s_sel[2] = ws;
      s_sel[3] = gs;
      s_before = before;
      s_target = target;
    }
    __syncthreads();
    const int mode = s_sel[0];
    if (mode == 2) {
      if (residual) {  // no residual mass left: fall back to p at this position
        residual = false;
        continue;
      }
      return;  // p always has mass for finite logits
    }
    if (s_sel[1] != static_cast<int>(crank) || s_sel[2] != warp) return;
    bool last = mode == 1;
    const int gs = s_sel[3];
    const double before = s_before, target = s_target;

    // recompute group gs exactly as in the totals and descend to the token
    const int v = gs * 32 + lane;
    float wt[N];
    float ls = 0.f;
    if (v < nloc) {
      vec_weights<T>(zc, wc, v, residual, st.cz, st.cw, khi, klo, wt);
#pragma unroll
      for (int e = 0; e < N; ++e) ls = __fadd_rn(ls, wt[e]);
    } else {
#pragma unroll
      for (int e = 0; e < N; ++e) wt[e] = 0.f;
    }
    float incl = ls;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl = __fadd_rn(incl, y);
    }
    int ln;
    if (!last) {
      const unsigned hit = __ballot_sync(0xffffffffu, before + static_cast<double>(incl) > target);
      ln = hit ? __ffs(hit) - 1 : -1;
      if (ln < 0) last = true;
    }
    if (last) {
      const unsigned pos = __ballot_sync(0xffffffffu, ls > 0.f);
      ln = pos ? 31 - __clz(pos) : 0;
    }
    float ex = __shfl_up_sync(0xffffffffu, incl, 1);
    if (lane == 0) ex = 0.f;
    if (lane == ln) {
      const double lb = before + static_cast<double>(ex);
      int k = -1;
      float c = 0.f;
      if (!last) {
#pragma unroll
        for (int e = 0; e < N; ++e) {
          c = __fadd_rn(c, wt[e]);
          if (k < 0 && lb + static_cast<double>(c) > target) k = e;
        }
      }
      if (k < 0) {
        for (int e = N - 1; e >= 0; --e)
          if (wt[e] > 0.f) { k = e; break; }
        if (k < 0) k = 0;
      }
      p.out_tokens[off + a] = (cb + v) * N + k;
    }
    return;
  }
}

}  // namespace dipsd
