// spec_verify: speculative sampling over the vocabulary for a batch of users
// (Sec. II-A stage 2: accept/reject every draft, truncate at the first
// rejection, emit one more token from the residual or, at the bonus position,
// from the target distribution).  Register path for 16-byte aligned rows.
//
// Rows are read once, with every 16-byte load of a thread issued up front and
// kept in registers (a slice of 256 threads x up to NK vectors per row), so a
// CTA has its whole slice in flight at once; no shared-memory staging.
//
// Pass 1 (spec_stats_kernel) -- one thread-block cluster per verify position.
// Each CTA owns a slice of the target-logit row (and of the draft-logit row at
// draft positions).  A thread takes its maximum m, picks the integer reference
// c = ceil(m log2 e) and sums 2^(x log2 e - c) (two FFMA and one ex2 per
// logit).  Because references are integers, every rescale between threads,
// warps, CTAs and cluster ranks is an exact power of two; partial sums combine
// as float-float pairs and the row normaliser is kept in fp64.  Rank 0 forms
// p_t(d), q_t(d) and takes the acceptance decision u_acc * q_t(d) < p_t(d).
//
// Pass 2 (spec_sample_kernel) -- one cluster per user.  Warp ballots over the
// acceptance bits give a_i and the packed output offset.  The slices of the
// rows at position a_i are loaded the same way; weights (max(0, p - q) up to a
// common factor, or p at the bonus position) use the pass-1 exponential.  Each
// warp covers 32 consecutive vectors (256 tokens) per step -- a group -- and
// keeps every group total; slice totals are exchanged through distributed
// shared memory, and the CTA holding u * total descends slice -> group ->
// lane -> token on the very same fp32 partial sums, so the descent always
// lands in the cell the totals point to.
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
constexpr int kRegThreads = 256;
constexpr int kRegWarps = kRegThreads / 32;

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
__device__ __forceinline__ FF ff_neg(FF a) { return FF{-a.hi, -a.lo}; }
__device__ __forceinline__ FF ff_sub(FF a, FF b) { return ff_add(a, ff_neg(b)); }
// a > b for float-float values
__device__ __forceinline__ bool ff_gt(FF a, FF b) {
  const FF d = ff_sub(a, b);
  return d.hi > 0.f || (d.hi == 0.f && d.lo > 0.f);
}
// a * u with the product's rounding error kept (u a float)
__device__ __forceinline__ FF ff_mul_f(FF a, float u) {
  const float p = __fmul_rn(a.hi, u);
  const float e = __fmaf_rn(a.hi, u, -p);
  return ff_add(FF{p, 0.f}, FF{e, __fmul_rn(a.lo, u)});
}
// inclusive warp scan of float-float values
__device__ __forceinline__ FF warp_ff_scan(FF v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    FF y;
    y.hi = __shfl_up_sync(0xffffffffu, v.hi, o);
    y.lo = __shfl_up_sync(0xffffffffu, v.lo, o);
    if (lane >= o) v = ff_add(y, v);
  }
  return v;
}

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

// ------------------------------------------------------ register slices
template <typename T>
struct Vec16;
template <>
struct Vec16<__nv_bfloat16> {
  static constexpr int N = 8;
  static __device__ __forceinline__ void unpack(const uint4& r, float (&x)[8]) {
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
  static __device__ __forceinline__ void unpack(const uint4& r, float (&x)[4]) {
    x[0] = __uint_as_float(r.x); x[1] = __uint_as_float(r.y);
    x[2] = __uint_as_float(r.z); x[3] = __uint_as_float(r.w);
  }
};

// Largest element of one 16-byte vector (bf16 pairs compared packed).
template <typename T>
__device__ __forceinline__ float vec_max(const uint4& r) {
  if constexpr (sizeof(T) == 2) {
    uint32_t a, b, c;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(r.x), "r"(r.y));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(r.z), "r"(r.w));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(c) : "r"(a), "r"(b));
    return fmaxf(__uint_as_float(c << 16), __uint_as_float(c & 0xFFFF0000u));
  } else {
    return fmaxf(fmaxf(__uint_as_float(r.x), __uint_as_float(r.y)), fmaxf(__uint_as_float(r.z), __uint_as_float(r.w)));
  }
}

// Slice of CTA `rank` in units of 16-byte vectors.
__device__ __forceinline__ void slice_bounds(int nvec, uint32_t rank, uint32_t csize, int& sb, int& se) {
  sb = static_cast<int>((static_cast<long long>(rank) * nvec) / csize);
  se = static_cast<int>((static_cast<long long>(rank + 1) * nvec) / csize);
}

// Loads this thread's vectors of a slice: vector sb + k*kRegThreads + tid.
template <int NK>
__device__ __forceinline__ void load_slice(const uint8_t* row, int sb, int se, int tid, uint4 (&r)[NK]) {
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    const int v = sb + k * kRegThreads + tid;
    r[k] = v < se ? ldg_stream_v4(row + static_cast<size_t>(v) * 16) : make_uint4(0, 0, 0, 0);
  }
}

// Thread partial sum of 2^(x log2 e - c) over its loaded vectors.
template <typename T, int NK>
__device__ __forceinline__ RefSum thread_refsum(const uint4 (&r)[NK], int sb, int se, int tid) {
  constexpr int N = Vec16<T>::N;
  float m = -INFINITY;
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    if (sb + k * kRegThreads + tid < se) m = fmaxf(m, vec_max<T>(r[k]));
  }
  if (!(m > -INFINITY)) return RefSum{kEmptyRef, FF{0.f, 0.f}};
  const float cf = fminf(fmaxf(ceilf(m * kLog2e), -1048576.f), 1048576.f);
  KahanSum acc;
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    if (sb + k * kRegThreads + tid < se) {
      float x[N];
      Vec16<T>::unpack(r[k], x);
      float e[N];
#pragma unroll
      for (int q = 0; q < N; ++q) e[q] = ex2_ref(x[q], cf);
      float sv;
      if constexpr (N == 8) {
        sv = ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
      } else {
        sv = (e[0] + e[1]) + (e[2] + e[3]);
      }
      acc.add(sv);
    }
  }
  return RefSum{static_cast<int>(cf), FF{acc.s, -acc.c}};
}

// ------------------------------------------------------------------ pass 1
template <typename T, int NK, int CAP>
__global__ void __launch_bounds__(kRegThreads, NK >= 20 ? 1 : 2)
spec_stats_kernel(const __grid_constant__ SpecParams<CAP> p) {
  __shared__ RefSum red[2][kRegWarps];
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
  int sb, se;
  slice_bounds(p.nvec, crank, csize, sb, se);

  pdl_wait_prior_grid();
  pdl_launch_dependents();
  uint4 rz[NK], rw[NK];
  load_slice<NK>(reinterpret_cast<const uint8_t*>(zrow), sb, se, threadIdx.x, rz);
  if (has_q) load_slice<NK>(reinterpret_cast<const uint8_t*>(wrow_p), sb, se, threadIdx.x, rw);
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

  RefSum az = thread_refsum<T, NK>(rz, sb, se, threadIdx.x);
  RefSum aw{kEmptyRef, FF{0.f, 0.f}};
  if (has_q) aw = thread_refsum<T, NK>(rw, sb, se, threadIdx.x);
  az = warp_refsum(az);
  aw = warp_refsum(aw);
  if (lane == 0) {
    red[0][warp] = az;
    red[1][warp] = aw;
  }
  __syncthreads();
  cluster_wait_acquire();  // phase A complete: rank 0 is running
  if (threadIdx.x == 0) {
    RefSum bz = red[0][0], bw = red[1][0];
    for (int k = 1; k < kRegWarps; ++k) {
      bz = refsum_add(bz, red[0][k]);
      bw = refsum_add(bw, red[1][k]);
    }
    const uint32_t dst = dsmem_map(&cl_slot[crank][0], 0);
    dsmem_st_f32x4(dst, __int_as_float(bz.c), bz.s.hi, bz.s.lo, 0.f);
    dsmem_st_f32x4(dst + 16, __int_as_float(bw.c), bw.s.hi, bw.s.lo, 0.f);
  }
  cluster_arrive_release();  // phase B: slices delivered to rank 0
  cluster_wait_acquire();
  if (crank != 0 || threadIdx.x != 0) return;

  RefSum fz{kEmptyRef, FF{0.f, 0.f}}, fw{kEmptyRef, FF{0.f, 0.f}};
  for (uint32_t k = 0; k < csize; ++k) {
    const float4 a = cl_slot[k][0], b = cl_slot[k][1];
    fz = refsum_add(fz, RefSum{__float_as_int(a.x), FF{a.y, a.z}});
    fw = refsum_add(fw, RefSum{__float_as_int(b.x), FF{b.y, b.z}});
  }
  SpecStat st;
  st.sz = static_cast<double>(fz.s.hi) + static_cast<double>(fz.s.lo);
  st.sw = static_cast<double>(fw.s.hi) + static_cast<double>(fw.s.lo);
  st.cz = fz.c;
  st.cw = fw.c;
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

// Sampling weights of one vector: (p - q)^+ up to the common factor 1/sz
// (residual), or p up to 1/sz (bonus).  Explicit rounding, so every
// evaluation of the same vector yields the same bits.
template <typename T>
__device__ __forceinline__ void vec_weights(const uint4& rz, const uint4& rw, bool residual, int cz, int cw,
                                            float khi, float klo, float (&wt)[Vec16<T>::N]) {
  constexpr int N = Vec16<T>::N;
  float xz[N];
  Vec16<T>::unpack(rz, xz);
  if (residual) {
    float xw[N];
    Vec16<T>::unpack(rw, xw);
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

// Sum of one vector's weights, left to right (the order the descent replays).
template <int N>
__device__ __forceinline__ float vec_sum(const float (&wt)[N]) {
  float s = 0.f;
#pragma unroll
  for (int e = 0; e < N; ++e) s = __fadd_rn(s, wt[e]);
  return s;
}

// ------------------------------------------------------------------ pass 2
template <typename T, int NK, int CAP>
__global__ void __launch_bounds__(kRegThreads, 1)
spec_sample_kernel(const __grid_constant__ SpecParams<CAP> p) {
  constexpr int N = Vec16<T>::N;
  __shared__ float gsum[NK * kRegWarps];      // group totals, group g = step k * warps + warp
  __shared__ float gpre[NK * kRegWarps][2];   // float-float inclusive prefix of the groups
  __shared__ float slice_sum[2][kMaxCluster][2];
  __shared__ int s_off, s_a, s_cnt[kRegWarps];
  __shared__ int s_sel[3];
  __shared__ float s_rem[2];
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
  for (int j = warp; j < ui; j += kRegWarps) cnt += accepted_prefix<CAP>(p, j, lane) + 1;
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
    for (int k = 0; k < kRegWarps; ++k) o += s_cnt[k];
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
    for (int k = threadIdx.x; k < a; k += kRegThreads) p.out_tokens[off + k] = p.draft_tokens[l0 + k];
    if (threadIdx.x == 0) {
      p.accept_len[ui] = a;
      p.out_offsets[ui] = off;
      if (ui == p.B - 1) p.out_offsets[p.B] = off + a + 1;
    }
  }

  // the rows of position a, this CTA's slice, into registers
  const int n = q0 + a;
  bool residual = a < Li;
  const SpecStat st = static_cast<const SpecStat*>(p.stats)[n];
  const uint8_t* zrow = reinterpret_cast<const uint8_t*>(static_cast<const T*>(p.z) + static_cast<size_t>(n) * p.V);
  const uint8_t* wrow =
      reinterpret_cast<const uint8_t*>(static_cast<const T*>(p.w) + static_cast<size_t>(residual ? l0 + a : 0) * p.V);
  int sb, se;
  slice_bounds(p.nvec, crank, csize, sb, se);
  uint4 rz[NK], rw[NK];
  load_slice<NK>(zrow, sb, se, threadIdx.x, rz);
  if (residual) load_slice<NK>(wrow, sb, se, threadIdx.x, rw);
  const float khi = s_k[0], klo = s_k[1];
  const float u = p.uniforms[2 * n + 1];

  // one pass per candidate distribution: the residual, then p if it is empty
  constexpr int G = NK * kRegWarps;  // groups of this CTA, in token order (step k, warp)
  for (int round = 0; round < 2; ++round) {
#pragma unroll
    for (int k = 0; k < NK; ++k) {
      float ls = 0.f;
      if (sb + k * kRegThreads + static_cast<int>(threadIdx.x) < se) {
        float wt[N];
        vec_weights<T>(rz[k], rw[k], residual, st.cz, st.cw, khi, klo, wt);
        ls = vec_sum<N>(wt);
      }
      float incl = ls;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl = __fadd_rn(incl, y);
      }
      if (lane == 31) gsum[k * kRegWarps + warp] = incl;
    }
    __syncthreads();
    // warp 0: float-float prefix over the groups; the last one is the slice total
    if (warp == 0) {
      FF carry{0.f, 0.f};
      for (int g0 = 0; g0 < G; g0 += 32) {
        const int g = g0 + lane;
        FF v{g < G ? gsum[g] : 0.f, 0.f};
        v = ff_add(warp_ff_scan(v, lane), carry);
        if (g < G) {
          gpre[g][0] = v.hi;
          gpre[g][1] = v.lo;
        }
        carry.hi = __shfl_sync(0xffffffffu, v.hi, 31);
        carry.lo = __shfl_sync(0xffffffffu, v.lo, 31);
      }
      if (lane == 0) {
        if (round == 0) cluster_wait_acquire();  // phase A complete: all CTAs running
        for (uint32_t r = 0; r < csize; ++r)
          dsmem_st_f32x2(dsmem_map(&slice_sum[round][crank][0], r), carry.hi, carry.lo);
      }
    }
    if (round == 0 && warp != 0) cluster_wait_acquire();
    if (round == 0 && warp == 0 && lane != 0) cluster_wait_acquire();
    cluster_arrive_release();
    cluster_wait_acquire();

    // thread 0 finds the slice and group holding u * total (if rounding
    // leaves none: the last positive weight at every level) and publishes
    // them with the remainder below the group; all in float-float
    if (threadIdx.x == 0) {
      FF total{0.f, 0.f};
      for (uint32_t r = 0; r < csize; ++r) total = ff_add(total, FF{slice_sum[round][r][0], slice_sum[round][r][1]});
      int mode = 0;  // 0: crossing, 1: last positive weight, 2: empty distribution
      int cs = static_cast<int>(csize) - 1;
      FF rem{0.f, 0.f};
      if (!(total.hi > 0.f)) {
        mode = 2;
      } else {
        rem = ff_mul_f(total, u);
        mode = 1;
        for (uint32_t r = 0; r < csize; ++r) {
          const FF sl{slice_sum[round][r][0], slice_sum[round][r][1]};
          if (ff_gt(sl, rem)) { cs = static_cast<int>(r); mode = 0; break; }
          rem = ff_sub(rem, sl);
        }
        if (mode == 1)
          while (cs > 0 && !(slice_sum[round][cs][0] > 0.f)) --cs;
      }
      s_sel[0] = mode;
      s_sel[1] = cs;
      s_rem[0] = rem.hi;
      s_rem[1] = rem.lo;
    }
    __syncthreads();
    int mode = s_sel[0];
    if (mode == 2) {
      if (residual) {  // no residual mass left: fall back to p at this position
        residual = false;
        continue;
      }
      return;  // p always has mass for finite logits
    }
    if (s_sel[1] != static_cast<int>(crank)) return;
    // warp 0 of the chosen slice: first group whose prefix exceeds the remainder
    if (warp == 0) {
      const FF rem{s_rem[0], s_rem[1]};
      int gsel = -1;
      if (mode == 0) {
        for (int g0 = 0; g0 < G && gsel < 0; g0 += 32) {
          const int g = g0 + lane;
          const bool hit = g < G && ff_gt(FF{gpre[g][0], gpre[g][1]}, rem);
          const unsigned bal = __ballot_sync(0xffffffffu, hit);
          if (bal) gsel = g0 + __ffs(bal) - 1;
        }
      }
      if (gsel < 0) {  // rounding: the last group with mass
        mode = 1;
        int lastg = 0;
        for (int g0 = 0; g0 < G; g0 += 32) {
          const int g = g0 + lane;
          const unsigned bal = __ballot_sync(0xffffffffu, g < G && gsum[g] > 0.f);
          if (bal) lastg = g0 + 31 - __clz(bal);
        }
        gsel = lastg;
      }
      if (lane == 0) {
        FF rg = rem;
        if (gsel > 0) rg = ff_sub(rem, FF{gpre[gsel - 1][0], gpre[gsel - 1][1]});
        s_sel[0] = mode;
        s_sel[2] = gsel;
        s_rem[0] = rg.hi;
        s_rem[1] = rg.lo;
      }
    }
    __syncthreads();
    mode = s_sel[0];
    const int gk = s_sel[2] / kRegWarps, gw = s_sel[2] % kRegWarps;
    if (gw != warp) return;
    bool last = mode == 1;
    const FF remg{s_rem[0], s_rem[1]};

    // recompute group (gk, gw) exactly as in the totals and descend to the token
    const int v = sb + gk * kRegThreads + static_cast<int>(threadIdx.x);
    float wt[N];
#pragma unroll
    for (int e = 0; e < N; ++e) wt[e] = 0.f;
    uint4 mz = rz[0], mw = rw[0];
#pragma unroll
    for (int k = 1; k < NK; ++k)
      if (k == gk) { mz = rz[k]; mw = rw[k]; }
    if (v < se) vec_weights<T>(mz, mw, residual, st.cz, st.cw, khi, klo, wt);
    const float ls = vec_sum<N>(wt);
    float incl = ls;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl = __fadd_rn(incl, y);
    }
    int ln = 0;
    if (!last) {
      const unsigned hit = __ballot_sync(0xffffffffu, ff_gt(FF{incl, 0.f}, remg));
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
      const FF reml = ff_sub(remg, FF{ex, 0.f});
      int k = -1;
      float c = 0.f;
      if (!last) {
#pragma unroll
        for (int e = 0; e < N; ++e) {
          c = __fadd_rn(c, wt[e]);
          if (k < 0 && ff_gt(FF{c, 0.f}, reml)) k = e;
        }
      }
      if (k < 0) {
        for (int e = N - 1; e >= 0; --e)
          if (wt[e] > 0.f) { k = e; break; }
        if (k < 0) k = 0;
      }
      p.out_tokens[off + a] = v * N + k;
    }
    return;
  }
}

}  // namespace dipsd
