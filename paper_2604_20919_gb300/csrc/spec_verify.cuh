// spec_verify: speculative sampling over the vocabulary for a batch of users
// (Sec. II-A stage 2: accept/reject every draft, truncate at the first
// rejection, emit one more token from the residual or, at the bonus position,
// from the target distribution).  Register path for 16-byte aligned rows.
//
// Three kernels, chained by programmatic dependent launch.  A work item of
// the two streaming passes is one warp-sized segment of one row: 32 lanes x
// NK 16-byte vectors, lane-interleaved so that every load instruction of the
// warp reads 512 contiguous bytes.  Items spread evenly over the SMs whatever
// the mix of draft lengths.
//
// spec_stats_kernel: the segments of every target row z_t and every draft row
// w_t, persistent over warps.  A warp takes the integer reference
// c = ceil(m log2 e) of a group's maximum m and sums 2^(x log2 e - c) (two
// FFMA and one ex2 per logit).  References are integers, so partial sums
// combine by exact power-of-two rescaling as float-float pairs.  Each segment
// leaves its partial; no atomics, no waits.
//
// spec_decide_kernel: one warp per position combines its rows' partials,
// forms p_t(d), q_t(d) and decides u_acc * q_t(d) < p_t(d); the last decided
// position of user i (a 64-bit decision word per user) counts the leading
// accepts a_i.
//
// spec_sample_kernel: the segments of the rows at position a_i of every
// user.  A warp computes the sampling weights (max(0, p - q) up to a common
// factor, or p at the bonus position) and stores its segment's total, summed
// in token order: fp32 scans over 32-vector groups, float-float across
// groups.  The warp that delivers the last segment of user i (an arrival
// counter) locates u * total: segment, group, lane and token, replaying the
// very sums that produced the totals, so the descent lands in the cell the
// totals point to.
#pragma once

#include "spec_common.cuh"

namespace dipsd {

constexpr float kLog2e = 1.4426950408889634f;
// log2(e) = kLog2eHi + kLog2eLo (the fp32 rounding and its remainder).
constexpr float kLog2eHi = 1.44269502162933349609375f;
constexpr float kLog2eLo = 1.925963033500651e-8f;
constexpr int kEmptyRef = -(1 << 29);
constexpr int kRegThreads = 256;
constexpr int kRegWarps = kRegThreads / 32;

// Row statistics of one verify position, relative to integer references:
// sz = sum_v 2^(z_v log2 e - cz), sw likewise for the draft row, each a
// float-float pair; sz / sw, the scale of q against p in the residual, split
// into two floats.
struct SpecStat {
  float szh, szl, swh, swl;
  int cz, cw;
  float khi, klo;
};
// The part of SpecStat the sampling weights need (its second 16 bytes).
struct WRef {
  int cz, cw;
  float khi, klo;
};

// --------------------------------------------------------- float-float sums
struct FF {
  float hi, lo;
};
// Commutative bit for bit: the TwoSum error term is exact.
__device__ __forceinline__ FF ff_add(FF a, FF b) {
  const float s = __fadd_rn(a.hi, b.hi);
  const float bb = __fsub_rn(s, a.hi);
  const float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, bb)), __fsub_rn(b.hi, bb));
  const float lo = __fadd_rn(__fadd_rn(a.lo, b.lo), e);
  const float hi = __fadd_rn(s, lo);
  return FF{hi, __fsub_rn(lo, __fsub_rn(hi, s))};
}
// 2^k for k <= 0 as an exact float (0 below the normal range).
__device__ __forceinline__ float pow2_nonpos(int k) {
  return k < -126 ? 0.f : __int_as_float((k + 127) << 23);
}
// a * 2^k for k <= 0 (exact for normal results)
__device__ __forceinline__ FF ff_scale(FF a, int k) {
  const float f = pow2_nonpos(k);
  return FF{__fmul_rn(a.hi, f), __fmul_rn(a.lo, f)};
}
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
__device__ __forceinline__ FF ff_shfl(FF v, int src) {
  return FF{__shfl_sync(0xffffffffu, v.hi, src), __shfl_sync(0xffffffffu, v.lo, src)};
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
// the scan value of the previous lane (0 at lane 0)
__device__ __forceinline__ FF warp_ff_exclusive(FF incl, int lane) {
  FF e;
  e.hi = __shfl_up_sync(0xffffffffu, incl.hi, 1);
  e.lo = __shfl_up_sync(0xffffffffu, incl.lo, 1);
  return lane == 0 ? FF{0.f, 0.f} : e;
}
// warp total of float-float values (every lane gets the same bits)
__device__ __forceinline__ FF warp_ff_sum(FF v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    FF y;
    y.hi = __shfl_xor_sync(0xffffffffu, v.hi, o);
    y.lo = __shfl_xor_sync(0xffffffffu, v.lo, o);
    v = ff_add(v, y);
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

// ------------------------------------------------------ arrival counters
// Counters are zero between calls: the last arrival of a call stores 0.
// Returns the arrival number (1-based).  The add is a release of the calling
// thread's earlier writes and an acquire of those of earlier arrivals; the
// arriving lane passes them on to its warp with __syncwarp.
__device__ __forceinline__ unsigned counter_arrive(unsigned* ctr) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], 1;" : "=r"(old) : "l"(ctr) : "memory");
  return old + 1u;
}

// ------------------------------------------------------ register segments
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

// A lane's vectors in the segment that starts at vector vb:
// vb + k * 32 + lane < nvec for k < the returned count (at most nk).
__device__ __forceinline__ int lane_vectors(int nvec, int vb, int lane, int nk) {
  const int n = nvec - vb - lane;
  return n > 0 ? min(nk, (n + 31) >> 5) : 0;
}

// Loads a lane's nv vectors of a segment (the rest of r is zeroed).
template <int NK>
__device__ __forceinline__ void load_segment(const void* row, int vb, int lane, int nv, uint4 (&r)[NK]) {
  const uint8_t* q = static_cast<const uint8_t*>(row) + (static_cast<size_t>(vb) + lane) * 16;
#pragma unroll
  for (int k = 0; k < NK; ++k)
    r[k] = k < nv ? ldg_stream_v4(q + static_cast<size_t>(k) * 512) : make_uint4(0u, 0u, 0u, 0u);
}

// Largest logit among a lane's vectors k0 <= k < k0 + KG, k < nv (bf16 pairs
// compared packed).
template <typename T, int NK, int KG>
__device__ __forceinline__ float lane_max(const uint4 (&r)[NK], int k0, int nv) {
  if constexpr (sizeof(T) == 2) {
    uint32_t pm = 0xFF80FF80u;  // packed -inf, -inf
#pragma unroll
    for (int k = k0; k < k0 + KG; ++k) {
      if (k < nv) {
        uint32_t a, b;
        asm("max.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(r[k].x), "r"(r[k].y));
        asm("max.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(r[k].z), "r"(r[k].w));
        asm("max.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(a), "r"(b));
        asm("max.bf16x2 %0, %1, %2;" : "=r"(pm) : "r"(pm), "r"(a));
      }
    }
    return fmaxf(__uint_as_float(pm << 16), __uint_as_float(pm & 0xFFFF0000u));
  } else {
    float m = -INFINITY;
#pragma unroll
    for (int k = k0; k < k0 + KG; ++k)
      if (k < nv)
        m = fmaxf(m, fmaxf(fmaxf(__uint_as_float(r[k].x), __uint_as_float(r[k].y)),
                           fmaxf(__uint_as_float(r[k].z), __uint_as_float(r[k].w))));
    return m;
  }
}

// ------------------------------------------ packed fp32 pairs (f32x2)
// Each op is two IEEE round-to-nearest operations in one instruction.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "sub.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
// ex2_ref on a pair: the same two roundings as ex2_ref, so the same bits
__device__ __forceinline__ float2 ex2_ref2(float2 x, float2 ncf) {
  const float2 a = fma2(x, make_float2(kLog2eHi, kLog2eHi), ncf);
  const float2 b = fma2(x, make_float2(kLog2eLo, kLog2eLo), a);
  return make_float2(fast_ex2(b.x), fast_ex2(b.y));
}

// Sum of 2^(x log2 e - c) over a lane's vectors k0 <= k < k0 + KG, k < nv:
// pairs of logits in f32x2 arithmetic, Kahan over vectors on the pair.
template <typename T, int NK, int KG>
__device__ __forceinline__ FF lane_expsum(const uint4 (&r)[NK], int k0, int nv, float cf) {
  const float2 ncf = make_float2(-cf, -cf);
  float2 s = make_float2(0.f, 0.f), c = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = k0; k < k0 + KG; ++k) {
    if (k < nv) {
      const uint32_t w[4] = {r[k].x, r[k].y, r[k].z, r[k].w};
      float2 v;
      if constexpr (sizeof(T) == 2) {
        float2 e[4];
#pragma unroll
        for (int j = 0; j < 4; ++j)
          e[j] = ex2_ref2(make_float2(__uint_as_float(w[j] << 16), __uint_as_float(w[j] & 0xFFFF0000u)), ncf);
        v = add2(add2(e[0], e[1]), add2(e[2], e[3]));
      } else {
        const float2 e0 = ex2_ref2(make_float2(__uint_as_float(w[0]), __uint_as_float(w[1])), ncf);
        const float2 e1 = ex2_ref2(make_float2(__uint_as_float(w[2]), __uint_as_float(w[3])), ncf);
        v = add2(e0, e1);
      }
      // Kahan step on both halves
      const float2 y = sub2(v, c);
      const float2 t = add2(s, y);
      c = sub2(sub2(t, s), y);
      s = t;
    }
  }
  // the two halves' compensated sums, added exactly
  return ff_add(FF{s.x, -c.x}, FF{s.y, -c.y});
}

// Sampling weights of one vector: (p - q)^+ up to the common factor 1/sz
// (residual), or p up to 1/sz.  Explicit rounding, so every evaluation of the
// same vector yields the same bits.
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

// inclusive fp32 scan over the lanes
__device__ __forceinline__ float warp_scan_f32(float v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v = __fadd_rn(v, y);
  }
  return v;
}

// Totals of one segment's weights in token order: step k covers the 32
// consecutive vectors vb + k * 32 + (0..31) (a group); a group total is the
// last lane of an fp32 scan over the lanes, groups add up in float-float.  tr
// is the residual's total (p's when not residual) and tp p's.  Bit-identical
// to the descent's recomputation from vec_weights and vec_sum.
template <typename T, int NK>
__device__ __forceinline__ void segment_totals(const uint4 (&rz)[NK], const uint4 (&rw)[NK], int nv, bool residual,
                                               const WRef& st, int lane, FF& tr, FF& tp) {
  constexpr int N = Vec16<T>::N;
  tr = FF{0.f, 0.f};
  tp = FF{0.f, 0.f};
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    float sr = 0.f, sp = 0.f;
    if (k < nv) {
      float xz[N];
      Vec16<T>::unpack(rz[k], xz);
      if (residual) {
        float xw[N];
        Vec16<T>::unpack(rw[k], xw);
#pragma unroll
        for (int e = 0; e < N; ++e) {
          const float ez = ex2_ref(xz[e], st.cz);
          const float ew = ex2_ref(xw[e], st.cw);
          const float q = __fmaf_rn(ew, st.khi, __fmul_rn(ew, st.klo));
          sr = __fadd_rn(sr, fmaxf(__fsub_rn(ez, q), 0.f));
          sp = __fadd_rn(sp, ez);
        }
      } else {
#pragma unroll
        for (int e = 0; e < N; ++e) sp = __fadd_rn(sp, ex2_ref(xz[e], st.cz));
      }
    }
    const float gp = __shfl_sync(0xffffffffu, warp_scan_f32(sp, lane), 31);
    tp = ff_add(tp, FF{gp, 0.f});
    if (residual) {
      const float gr = __shfl_sync(0xffffffffu, warp_scan_f32(sr, lane), 31);
      tr = ff_add(tr, FF{gr, 0.f});
    }
  }
  if (!residual) tr = tp;
}

// segment_totals for a sparse draft table: q of each element from qx.
template <typename T, int NK>
__device__ __forceinline__ void segment_totals_table(const uint4 (&rz)[NK], const float (&qx)[NK][Vec16<T>::N],
                                                     int nv, bool residual, const WRef& st, int lane, FF& tr,
                                                     FF& tp) {
  constexpr int N = Vec16<T>::N;
  tr = FF{0.f, 0.f};
  tp = FF{0.f, 0.f};
#pragma unroll
  for (int k = 0; k < NK; ++k) {
    float sr = 0.f, sp = 0.f;
    if (k < nv) {
      float xz[N];
      Vec16<T>::unpack(rz[k], xz);
#pragma unroll
      for (int e = 0; e < N; ++e) {
        const float ez = ex2_ref(xz[e], st.cz);
        sr = __fadd_rn(sr, residual && qx[k][e] > 0.f
                               ? fmaxf(__fsub_rn(ez, __fmaf_rn(qx[k][e], st.khi, __fmul_rn(qx[k][e], st.klo))), 0.f)
                               : ez);
        sp = __fadd_rn(sp, ez);
      }
    }
    const float gp = __shfl_sync(0xffffffffu, warp_scan_f32(sp, lane), 31);
    tp = ff_add(tp, FF{gp, 0.f});
    if (residual) {
      const float gr = __shfl_sync(0xffffffffu, warp_scan_f32(sr, lane), 31);
      tr = ff_add(tr, FF{gr, 0.f});
    }
  }
  if (!residual) tr = tp;
}

// ------------------------------------------------------ sparse draft table
// The draft row's table entries, two per lane (entry j in lane j % 32).
__device__ __forceinline__ void load_table(const int* idx_row, const float* q_row, int K, int lane, int (&sidx)[2],
                                           float (&sq)[2]) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int j = h * 32 + lane;
    sidx[h] = j < K ? idx_row[j] : -1;
    sq[h] = j < K ? q_row[j] : 0.f;
  }
}

// q of every element of a lane's vectors vb + k * 32 + lane (k < nv) from
// the table: 0 off the table.  Warp-uniform: each lane tests its two entries
// against the segment's token range, and only the entries that fall inside
// (a ballot) go round by shuffle.
template <int NK, int N>
__device__ __forceinline__ void table_q(const int (&sidx)[2], const float (&sq)[2], int K, int V, int vb, int lane,
                                        int nv, float (&qx)[NK][N], unsigned* status) {
#pragma unroll
  for (int k = 0; k < NK; ++k)
#pragma unroll
    for (int e = 0; e < N; ++e) qx[k][e] = 0.f;
  const int lo = vb * N, hi = (vb + 32 * NK) * N;  // tokens of the segment
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int j = h * 32 + lane;
    if (j < K && (sidx[h] < 0 || sidx[h] >= V)) atomicOr(status, kDevErrBadToken);
    unsigned hits = __ballot_sync(0xffffffffu, j < K && sidx[h] >= lo && sidx[h] < hi && sidx[h] < V);
    while (hits) {
      const int src = __ffs(hits) - 1;
      hits &= hits - 1;
      const int idx = __shfl_sync(0xffffffffu, sidx[h], src);
      const float qv = __shfl_sync(0xffffffffu, sq[h], src);
      const int dv = idx / N - vb - lane;
      if (dv < 0 || (dv & 31) != 0 || (dv >> 5) >= nv) continue;
      const int kk = dv >> 5, ee = idx % N;
#pragma unroll
      for (int k = 0; k < NK; ++k)
#pragma unroll
        for (int e = 0; e < N; ++e)
          if (k == kk && e == ee) qx[k][e] = qv;
    }
  }
}

// Sampling weights of one vector from a sparse table: max(0, p - q) up to
// the factor 1/sz (e_z - q sz, sz as khi + klo) where q > 0, else p's e_z
// (residual), or p's e_z.  Same rounding wherever it is evaluated.
template <typename T>
__device__ __forceinline__ void vec_weights_table(const uint4& rz, const float (&qx)[Vec16<T>::N], bool residual,
                                                  int cz, float khi, float klo, float (&wt)[Vec16<T>::N]) {
  constexpr int N = Vec16<T>::N;
  float xz[N];
  Vec16<T>::unpack(rz, xz);
#pragma unroll
  for (int e = 0; e < N; ++e) {
    const float ez = ex2_ref(xz[e], cz);
    wt[e] = residual && qx[e] > 0.f ? fmaxf(__fsub_rn(ez, __fmaf_rn(qx[e], khi, __fmul_rn(qx[e], klo))), 0.f) : ez;
  }
}

// ----------------------------------------------------- position decision
// The decision of position q0 + t of user ui from the row sums (integer
// reference, float-float sum) of z_t and w_t and the draft token's logits zd,
// wd (NaN: the token lies outside [0, V)) or, for a sparse payload, log q(d):
// SpecStat, p_t(d) and q_t(d), and the acceptance bit, added to the user's
// decision word (arrivals in the high half); the user's last decided
// position writes a_i.  One thread.
template <int CAP, bool SP>
__device__ __forceinline__ void decide_from_sums(const SpecParams<CAP>& p, int ui, int t, RefSum az, RefSum aw,
                                                 float zd, float wd, float logq, float u) {
  const int q0 = p.q_off[ui];
  const int Li = p.q_off[ui + 1] - q0 - 1;
  const int n = q0 + t;
  const bool has_q = t < Li;
  {
    // float-float throughout (FP64 is slow on this part): the acceptance
    // products carry ~2^-45 relative error, far inside the 1e-6 band
    SpecStat st;
    st.szh = az.s.hi;
    st.szl = az.s.lo;
    st.cz = az.c;
    st.swh = st.swl = 0.f;
    st.cw = kEmptyRef;
    st.khi = st.klo = 0.f;
    float pd = 0.f, qd = 0.f;
    unsigned char flag = 0;
    if (has_q && SP) {
      // sparse payload: q(d) is given; the residual scales q by sz, kept as
      // a float-float pair
      st.khi = az.s.hi;
      st.klo = az.s.lo;
      if (zd == zd) {
        const float ez = ex2_ref(zd, st.cz);
        const float q_d = expf(logq);
        pd = __fdividef(ez, az.s.hi);
        qd = q_d;
        // u * q(d) < p(d) = ez / sz, i.e. u * q(d) * sz < ez
        flag = ff_gt(FF{ez, 0.f}, ff_mul_f(ff_mul_f(az.s, u), q_d)) ? 1 : 0;
      } else {
        atomicOr(p.status, kDevErrBadToken);
      }
    } else if (has_q) {
      st.swh = aw.s.hi;
      st.swl = aw.s.lo;
      st.cw = aw.c;
      // sz / sw in float-float: q1 = zh / wh, then the remainder's quotient
      const float q1 = __fdiv_rn(az.s.hi, aw.s.hi);
      float r = __fmaf_rn(-q1, aw.s.hi, az.s.hi);
      r = __fmaf_rn(-q1, aw.s.lo, __fadd_rn(r, az.s.lo));
      const float q2 = __fdiv_rn(r, aw.s.hi);
      st.khi = __fadd_rn(q1, q2);
      st.klo = __fsub_rn(q2, __fsub_rn(st.khi, q1));
      if (zd == zd && wd == wd) {
        const float ez = ex2_ref(zd, st.cz);
        const float ew = ex2_ref(wd, st.cw);
        pd = __fdividef(ez, az.s.hi);
        qd = __fdividef(ew, aw.s.hi);
        // u * q(d) < p(d), i.e. u * ew * sz < ez * sw (no division)
        flag = ff_gt(ff_mul_f(aw.s, ez), ff_mul_f(ff_mul_f(az.s, u), ew)) ? 1 : 0;
      } else {
        atomicOr(p.status, kDevErrBadToken);
      }
    }
    static_cast<SpecStat*>(p.stats)[n] = st;
    if (p.draft_probs) reinterpret_cast<float2*>(p.draft_probs)[n] = make_float2(pd, qd);
    // the user's decision word: one arrival, and bit t if d_{t+1} is accepted;
    // the last of the user's L_i + 1 positions reads a_i off the sum
    unsigned long long* word = reinterpret_cast<unsigned long long*>(p.counters + kCntUser1) + ui;
    const unsigned long long add = (1ull << 32) | (flag ? (1ull << t) : 0ull);
    const unsigned long long now = atomicAdd(word, add) + add;
    if (static_cast<int>(now >> 32) == Li + 1) {
      p.accept_len[ui] = min(__ffs(~static_cast<unsigned>(now)) - 1, Li);
      *word = 0ull;
    }
  }
}

// Row sums, p_t(d), q_t(d) and the acceptance decision of position q0 + t of
// user ui (one warp); the user's last decided position also writes a_i.
template <int CAP, bool SP>
__device__ __forceinline__ void decide_position(const SpecParams<CAP>& p, int ui, int t, int lane) {
  const int q0 = p.q_off[ui];
  const int Li = p.q_off[ui + 1] - q0 - 1;
  const int n = q0 + t, l = p.l_off[ui] + t;
  const bool has_q = t < Li;
  const float4* pz = p.part1 + static_cast<size_t>(n) * p.nseg1;
  const float4* pw = p.part1 + static_cast<size_t>(p.sum_t + l) * p.nseg1;
  // every load first: the draft token's logits, left by the rows' first
  // segments (NaN: d outside [0, V)), and both rows' segment partials
  float zd = 0.f, wd = 0.f, logq = 0.f;
  if (has_q && lane == 0) {
    zd = __ldcg(&pz->w);
    if constexpr (SP) logq = p.draft_logq[l];
    else wd = __ldcg(&pw->w);
  }
  RefSum az{kEmptyRef, FF{0.f, 0.f}}, aw{kEmptyRef, FF{0.f, 0.f}};
  // the position's two uniforms (independent of the loads, so they overlap
  // them): the acceptance one here, the resample one kept for the descent
  const float2 u = verify_uniforms(p.seed, static_cast<unsigned>(p.uid[ui]), t);
  const float u_acc = has_q ? u.x : 0.f;
  if (lane == 0) p.u_res[n] = u.y;
#pragma unroll 2
  for (int sg = lane; sg < p.nseg1; sg += 32) {
    const float4 vz = __ldcg(pz + sg);
    const float4 vw = has_q && !SP ? __ldcg(pw + sg) : make_float4(__int_as_float(kEmptyRef), 0.f, 0.f, 0.f);
    az = refsum_add(az, RefSum{__float_as_int(vz.x), FF{vz.y, vz.z}});
    aw = refsum_add(aw, RefSum{__float_as_int(vw.x), FF{vw.y, vw.z}});
  }
  az = warp_refsum(az);
  if (has_q && !SP) aw = warp_refsum(aw);
  if (lane == 0) decide_from_sums<CAP, SP>(p, ui, t, az, aw, zd, wd, logq, u_acc);
}

// ------------------------------------------------------------------ pass 1
// One segment of one logit row: z_t of user ui, or w_t.
template <typename T>
struct StatSeg {
  const T* row;
  int item, vb, nv, l;
  bool has_q;
};

// Segment `item` of the flat item list (rows: every z_t, then every w_t; no
// w rows when the draft payload is sparse).
template <typename T, int NK, int CAP, bool SP>
__device__ __forceinline__ StatSeg<T> stat_seg(const SpecParams<CAP>& p, int item, int lane) {
  const int row = item / p.nseg1;
  const int s = item - row * p.nseg1;
  const bool is_w = !SP && row >= p.sum_t;
  const int ui = is_w ? spec_find_user<CAP>(p.l_off, p.B, row - p.sum_t) : spec_find_user<CAP>(p.q_off, p.B, row);
  const int q0 = p.q_off[ui];
  const int t = is_w ? row - p.sum_t - p.l_off[ui] : row - q0;
  StatSeg<T> g;
  g.item = item;
  g.l = p.l_off[ui] + t;
  g.has_q = t < p.q_off[ui + 1] - q0 - 1;
  g.row = is_w ? static_cast<const T*>(p.w) + static_cast<size_t>(g.l) * p.V
               : static_cast<const T*>(p.z) + static_cast<size_t>(q0 + t) * p.V;
  g.vb = s * (32 * NK);
  g.nv = lane_vectors(p.nvec, g.vb, lane, NK);
  return g;
}

// The draft token's logit in the row, fetched by lane 0 of the row's first
// segment (NaN: the token lies outside [0, V)); 0 elsewhere.
template <typename T, int CAP>
__device__ __forceinline__ float stat_draft_logit(const SpecParams<CAP>& p, const StatSeg<T>& g, int lane) {
  if (g.vb != 0 || lane != 0 || !g.has_q) return 0.f;
  const int d = p.draft_tokens[g.l];
  return d >= 0 && d < p.V ? load_elem<T>(g.row, d) : __int_as_float(0x7fc00000);
}

// Loads a lane's vectors k0 .. k0 + KG - 1 of a segment (zero past nv).
template <int NK, int KG>
__device__ __forceinline__ void load_group(const void* row, int vb, int lane, int nv, int k0, uint4 (&r)[NK]) {
  const uint8_t* q = static_cast<const uint8_t*>(row) + (static_cast<size_t>(vb) + lane) * 16;
#pragma unroll
  for (int k = k0; k < k0 + KG; ++k)
    r[k] = k < nv ? ldg_stream_v4(q + static_cast<size_t>(k) * 512) : make_uint4(0u, 0u, 0u, 0u);
}

// Row sums of every segment, persistent over warps: warp w of the W in the
// grid takes items w, w + W, w + 2W, ...  A segment's vectors go in groups of
// four, each group with its own warp reference, so the first group's
// exponentials overlap the later groups' loads; once a group is summed its
// registers are refilled with the same group of the warp's next segment, so
// the warp keeps about one segment of loads in flight from its first segment
// to its last.  Each segment's partial (reference, float-float sum, draft
// logit) goes to part1; no warp waits for another, and nothing here orders
// the partials: the decision kernel reads them once this grid is complete.
template <typename T, int NK, int CAP, bool SP>
__global__ void __launch_bounds__(kRegThreads, 2)
spec_stats_kernel(const __grid_constant__ SpecParams<CAP> p) {
  const int lane = threadIdx.x & 31;
  const int W = gridDim.x * kRegWarps;
  int item = blockIdx.x * kRegWarps + (threadIdx.x >> 5);
  pdl_wait_prior_grid();
  // (the dependent grid is released as each CTA finishes its segments: the
  // decision kernel's CTAs then take no SM slot while this pass streams)
  if (item >= p.n_items1) {
    pdl_launch_dependents();
    return;
  }
  constexpr int KG = NK < 4 ? NK : 4;
  StatSeg<T> g = stat_seg<T, NK, CAP, SP>(p, item, lane);
  uint4 r[NK];
  load_segment<NK>(g.row, g.vb, lane, g.nv, r);
  float xd = stat_draft_logit<T, CAP>(p, g, lane);
  for (;;) {
    const int nxt = item + W;
    const bool more = nxt < p.n_items1;
    StatSeg<T> ng = g;
    float nxd = 0.f;
    if (more) {
      ng = stat_seg<T, NK, CAP, SP>(p, nxt, lane);
      nxd = stat_draft_logit<T, CAP>(p, ng, lane);
    }
    RefSum tot{kEmptyRef, FF{0.f, 0.f}};
#pragma unroll
    for (int k0 = 0; k0 < NK; k0 += KG) {
      const float m = lane_max<T, NK, KG>(r, k0, g.nv);
      int c = m > -INFINITY ? static_cast<int>(fminf(fmaxf(ceilf(m * kLog2e), -1048576.f), 1048576.f)) : kEmptyRef;
      c = __reduce_max_sync(0xffffffffu, c);
      if (c != kEmptyRef) tot = refsum_add(tot, RefSum{c, lane_expsum<T, NK, KG>(r, k0, g.nv, static_cast<float>(c))});
      if (more) load_group<NK, KG>(ng.row, ng.vb, lane, ng.nv, k0, r);
    }
    const FF sum = warp_ff_sum(tot.s);
    if (lane == 0) p.part1[g.item] = make_float4(__int_as_float(tot.c), sum.hi, sum.lo, xd);
    if (!more) break;
    item = nxt;
    g = ng;
    xd = nxd;
  }
  pdl_launch_dependents();
}

// One warp per verify position: the row sums from the statistics pass's
// partials, p_t(d), q_t(d) and the acceptance decision; the user's last
// decided position writes a_i.
template <int CAP, bool SP>
__global__ void __launch_bounds__(kRegThreads)
spec_decide_kernel(const __grid_constant__ SpecParams<CAP> p) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kRegWarps + (threadIdx.x >> 5);
  pdl_wait_prior_grid();
  pdl_launch_dependents();
  if (n >= p.sum_t) return;
  const int ui = spec_find_user<CAP>(p.q_off, p.B, n);
  decide_position<CAP, SP>(p, ui, n - p.q_off[ui], lane);
}

// ------------------------------------------------------------------ pass 2
// Run by the warp that delivered the last segment of user ui: packed output
// offset, accepted drafts, then the inverse-CDF descent to the emitted token.
template <typename T, int NK, int CAP, bool SP>
__device__ __forceinline__ void descend(const SpecParams<CAP>& p, int ui, int a, bool residual, const WRef& st,
                                        const T* zrow, const T* wrow, const int (&sidx)[2], const float (&sq)[2],
                                        int lane) {
  constexpr int N = Vec16<T>::N;
  const int l0 = p.l_off[ui];
  const float4* part = p.part2 + static_cast<size_t>(ui) * p.nseg2;
  const int per = (p.nseg2 + 31) >> 5;  // lane j owns segments [j per, (j + 1) per)
  const int s0 = lane * per;
  // a run of up to kRun segments per lane is held in registers as its
  // running float-float sums (the same additions in the same order as the
  // lane's total), so the walk below compares them all at once
  constexpr int kRun = 16;
  const bool in_regs = per <= kRun;
  auto load_run = [&](int mode, float2 (&v)[kRun]) {
#pragma unroll
    for (int i = 0; i < kRun; ++i) {
      const int sg = s0 + i;
      v[i] = in_regs && i < per && sg < p.nseg2 ? __ldcg(reinterpret_cast<const float2*>(part + sg) + mode)
                                                : make_float2(0.f, 0.f);
    }
  };
  // every independent load first: the first mode's segment totals, the
  // uniform, the accepted drafts and the earlier users' accept lengths
  const int mode0 = residual ? 0 : 1;
  float2 v[kRun];
  load_run(mode0, v);
  const float u = __ldcg(p.u_res + p.q_off[ui] + a);  // drawn by the decision kernel
  const int dtok = lane < a ? p.draft_tokens[l0 + lane] : 0;  // a <= L_i <= 31
  int o = 0;
  for (int j = lane; j < ui; j += 32)
    o += min(max(p.accept_len[j], 0), p.q_off[j + 1] - p.q_off[j] - 1) + 1;
  const int off = __reduce_add_sync(0xffffffffu, o);
  if (lane < a) p.out_tokens[off + lane] = dtok;
  if (lane == 0) {
    p.counters[kCntUser2 + ui] = 0u;
    p.out_offsets[ui] = off;
    if (ui == p.B - 1) p.out_offsets[p.B] = off + a + 1;
  }
  // mode 0: the residual; mode 1: p (the bonus position, or an empty residual)
  for (int mode = mode0; mode < 2; ++mode) {
    FF pre[kRun];
    FF ls{0.f, 0.f};
    if (in_regs) {
      if (mode != mode0) load_run(mode, v);
#pragma unroll
      for (int i = 0; i < kRun; ++i) {
        ls = ff_add(ls, FF{v[i].x, v[i].y});
        pre[i] = ls;
      }
    } else {
      for (int i = 0; i < per; ++i) {
        const int sg = s0 + i;
        if (sg < p.nseg2) {
          const float2 w = __ldcg(reinterpret_cast<const float2*>(part + sg) + mode);
          ls = ff_add(ls, FF{w.x, w.y});
        }
      }
    }
    const FF incl = warp_ff_scan(ls, lane);
    const FF total = ff_shfl(incl, 31);
    if (!(total.hi > 0.f)) continue;
    const FF target = ff_mul_f(total, u);
    // level 1: the lane whose run of segments holds the target (if rounding
    // leaves none: the last positive mass at every level)
    const unsigned hit = __ballot_sync(0xffffffffu, ff_gt(incl, target));
    bool last = hit == 0;
    const int ln = last ? 31 - __clz(__ballot_sync(0xffffffffu, ls.hi > 0.f)) : __ffs(hit) - 1;
    const FF rem = ff_sub(target, ff_shfl(warp_ff_exclusive(incl, lane), ln));
    int sel = -1;
    FF rs{0.f, 0.f};
    if (lane == ln) {
      int lastpos = -1;
      if (in_regs) {
        FF prev{0.f, 0.f};
#pragma unroll
        for (int i = 0; i < kRun; ++i) {
          if (sel < 0 && !last && ff_gt(pre[i], rem)) {
            sel = s0 + i;
            rs = ff_sub(rem, prev);
          }
          if (pre[i].hi != prev.hi || pre[i].lo != prev.lo) lastpos = s0 + i;
          prev = pre[i];
        }
      } else {
        FF run{0.f, 0.f};
        for (int i = 0; i < per; ++i) {
          const int sg = s0 + i;
          if (sg >= p.nseg2) break;
          const float2 v = __ldcg(reinterpret_cast<const float2*>(part + sg) + mode);
          const FF x{v.x, v.y};
          const FF nx = ff_add(run, x);
          if (!last && ff_gt(nx, rem)) {
            sel = sg;
            rs = ff_sub(rem, run);
            break;
          }
          if (x.hi > 0.f) lastpos = sg;
          run = nx;
        }
      }
      if (sel < 0) {
        sel = lastpos;
        last = true;
      }
    }
    sel = min(max(__shfl_sync(0xffffffffu, sel, ln), 0), p.nseg2 - 1);
    last = __shfl_sync(0xffffffffu, last ? 1 : 0, ln) != 0;
    rs = ff_shfl(rs, ln);
    // level 2: the segment's groups, recomputed exactly as in its totals
    const int vb = sel * (32 * NK);
    const int nv = lane_vectors(p.nvec, vb, lane, NK);
    uint4 rz[NK], rw[NK];
    load_segment<NK>(zrow, vb, lane, nv, rz);
    load_segment<NK>(wrow, vb, lane, residual && !SP ? nv : 0, rw);
    float qx[NK][N];
    if constexpr (SP) {
      if (residual) table_q<NK, N>(sidx, sq, p.topk, p.V, vb, lane, nv, qx, p.status);
      else
#pragma unroll
        for (int k = 0; k < NK; ++k)
#pragma unroll
          for (int e = 0; e < N; ++e) qx[k][e] = 0.f;
    }
    float vs[NK], gin[NK];
#pragma unroll
    for (int k = 0; k < NK; ++k) {
      vs[k] = 0.f;
      if (k < nv) {
        float wt[N];
        if constexpr (SP) vec_weights_table<T>(rz[k], qx[k], mode == 0, st.cz, st.khi, st.klo, wt);
        else vec_weights<T>(rz[k], rw[k], mode == 0, st.cz, st.cw, st.khi, st.klo, wt);
        vs[k] = vec_sum<N>(wt);
      }
      gin[k] = warp_scan_f32(vs[k], lane);
    }
    int kk = -1, lastk = -1;
    FF rg{0.f, 0.f}, run{0.f, 0.f};
#pragma unroll
    for (int k = 0; k < NK; ++k) {
      const float g = __shfl_sync(0xffffffffu, gin[k], 31);
      const FF nx = ff_add(run, FF{g, 0.f});
      if (kk < 0 && !last && ff_gt(nx, rs)) {
        kk = k;
        rg = ff_sub(rs, run);
      }
      if (g > 0.f) lastk = k;
      run = nx;
    }
    if (kk < 0) {
      kk = max(lastk, 0);
      last = true;
    }
    // level 3: the lane of group kk, then the token inside its vector
    float ik = 0.f, vk = 0.f;
    uint4 mz = rz[0], mw = rw[0];
    float mq[N];
#pragma unroll
    for (int e = 0; e < N; ++e) mq[e] = 0.f;
#pragma unroll
    for (int k = 0; k < NK; ++k)
      if (k == kk) {
        ik = gin[k];
        vk = vs[k];
        mz = rz[k];
        mw = rw[k];
        if constexpr (SP)
#pragma unroll
          for (int e = 0; e < N; ++e) mq[e] = qx[k][e];
      }
    int ln2 = -1;
    if (!last) {
      const unsigned h2 = __ballot_sync(0xffffffffu, ff_gt(FF{ik, 0.f}, rg));
      if (h2) ln2 = __ffs(h2) - 1;
      else last = true;
    }
    if (last) {
      const unsigned pos = __ballot_sync(0xffffffffu, vk > 0.f);
      ln2 = pos ? 31 - __clz(pos) : 0;
    }
    float ex = __shfl_up_sync(0xffffffffu, ik, 1);
    if (lane == 0) ex = 0.f;
    const FF rl = ff_sub(rg, FF{__shfl_sync(0xffffffffu, ex, ln2), 0.f});
    if (lane == ln2) {
      float wt[N];
#pragma unroll
      for (int e = 0; e < N; ++e) wt[e] = 0.f;
      if (kk < nv) {
        if constexpr (SP) vec_weights_table<T>(mz, mq, mode == 0, st.cz, st.khi, st.klo, wt);
        else vec_weights<T>(mz, mw, mode == 0, st.cz, st.cw, st.khi, st.klo, wt);
      }
      int es = -1;
      if (!last) {
        float cum = 0.f;
#pragma unroll
        for (int e = 0; e < N; ++e) {
          cum = __fadd_rn(cum, wt[e]);
          if (es < 0 && ff_gt(FF{cum, 0.f}, rl)) es = e;
        }
      }
      if (es < 0) {
#pragma unroll
        for (int e = 0; e < N; ++e)
          if (wt[e] > 0.f) es = e;
      }
      if (es < 0) es = 0;
      p.out_tokens[off + a] = min((vb + kk * 32 + lane) * N + es, p.V - 1);
    }
    return;
  }
  if (lane == 0) p.out_tokens[off + a] = 0;  // no mass at all: every logit -inf
}

template <typename T, int NK, int CAP, bool SP>
__global__ void __launch_bounds__(kRegThreads, 2)
spec_sample_kernel(const __grid_constant__ SpecParams<CAP> p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int item = blockIdx.x * kRegWarps + warp;
  pdl_wait_prior_grid();
  pdl_launch_dependents();
  if (item >= p.n_items2) return;
  const int ui = item / p.nseg2;
  const int s = item - ui * p.nseg2;
  const int q0 = p.q_off[ui], l0 = p.l_off[ui];
  const int Li = p.q_off[ui + 1] - q0 - 1;
  // a_i and the weight references of all the user's positions, fetched together
  const int a_raw = p.accept_len[ui];
  int4 ref4 = make_int4(0, 0, 0, 0);
  if (lane <= Li) ref4 = reinterpret_cast<const int4*>(static_cast<const SpecStat*>(p.stats) + q0 + lane)[1];
  const int a = min(max(a_raw, 0), Li);  // (clamped: written by the stats kernel)
  const int n = q0 + a;
  const bool residual = a < Li;
  WRef st;
  st.cz = __shfl_sync(0xffffffffu, ref4.x, a);
  st.cw = __shfl_sync(0xffffffffu, ref4.y, a);
  st.khi = __int_as_float(__shfl_sync(0xffffffffu, ref4.z, a));
  st.klo = __int_as_float(__shfl_sync(0xffffffffu, ref4.w, a));
  const T* zrow = static_cast<const T*>(p.z) + static_cast<size_t>(n) * p.V;
  const T* wrow = residual && !SP ? static_cast<const T*>(p.w) + static_cast<size_t>(l0 + a) * p.V : zrow;
  const int vb = s * (32 * NK);
  const int nv = lane_vectors(p.nvec, vb, lane, NK);
  uint4 rz[NK], rw[NK];
  load_segment<NK>(zrow, vb, lane, nv, rz);
  load_segment<NK>(wrow, vb, lane, residual && !SP ? nv : 0, rw);
  int sidx[2] = {-1, -1};
  float sq[2] = {0.f, 0.f};
  FF R, P;
  if constexpr (SP) {
    constexpr int N = Vec16<T>::N;
    float qx[NK][N];
    if (residual) {
      load_table(p.topk_idx + static_cast<size_t>(l0 + a) * p.topk, p.topk_q + static_cast<size_t>(l0 + a) * p.topk,
                 p.topk, lane, sidx, sq);
      table_q<NK, N>(sidx, sq, p.topk, p.V, vb, lane, nv, qx, p.status);
    } else {
#pragma unroll
      for (int k = 0; k < NK; ++k)
#pragma unroll
        for (int e = 0; e < N; ++e) qx[k][e] = 0.f;
    }
    segment_totals_table<T, NK>(rz, qx, nv, residual, st, lane, R, P);
  } else {
    segment_totals<T, NK>(rz, rw, nv, residual, st, lane, R, P);
  }
  unsigned cnt = 0;
  if (lane == 31) {
    p.part2[item] = make_float4(R.hi, R.lo, P.hi, P.lo);
    cnt = counter_arrive(p.counters + kCntUser2 + ui);
  }
  __syncwarp();
  cnt = __shfl_sync(0xffffffffu, cnt, 31);
  if (cnt != static_cast<unsigned>(p.nseg2)) return;
  descend<T, NK, CAP, SP>(p, ui, a, residual, st, zrow, wrow, sidx, sq, lane);
}

}  // namespace dipsd
