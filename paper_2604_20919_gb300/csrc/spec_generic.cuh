// spec_verify, generic path: used when a logit row is not 16-byte aligned
// (V times the element size not a multiple of 16 bytes, or a row pointer off
// a 16-byte boundary), where the register path's 16-byte vector loads do not
// apply, or when a row has more segments than its arrival counters can count.
// Same arithmetic contract (speculative sampling, Sec. II-A stage 2); rows are
// streamed with per-thread loads instead of staged.
//
// Pass 1 (spec_stats_generic_kernel): one thread-block cluster per verify position;
// each CTA streams a slice of the target-logit row (and of the draft-logit row
// at draft positions) with 16-byte loads, keeps a per-thread online max and a
// compensated sum of exp(x - max), reduces them over the block and then over
// the cluster through distributed shared memory.  The cluster's rank 0 turns
// the row statistics into p_t(d), q_t(d) and the acceptance bit
// u_acc * q_t(d) < p_t(d).
//
// Pass 2 (spec_sample_generic_kernel): one cluster per user.  A warp ballot over the
// user's acceptance bits gives a_i; ballots over the earlier users give the
// packed output offset.  The cluster then draws the extra token at position
// a_i by inverse CDF: every CTA sums the sampling weights of its slice, the
// slice sums are broadcast through distributed shared memory, and the CTA
// whose slice holds the crossing finds the warp, the 256-token group, the lane
// and finally the token.
#pragma once

#include "spec_common.cuh"

namespace dipsd {

// Online (max, compensated sum of exp(x - max)) over a stream of values.
struct OnlineSoftmaxStat {
  float m = -INFINITY;
  KahanSum s;
  template <int N>
  __device__ __forceinline__ void add(const float (&x)[N]) {
    float cm = x[0];
#pragma unroll
    for (int k = 1; k < N; ++k) cm = fmaxf(cm, x[k]);
    if (cm > m) {
      if (m != -INFINITY) s.scale(expf(m - cm));
      m = cm;
    }
    if (m == -INFINITY) return;
#pragma unroll
    for (int k = 0; k < N; ++k) s.add(expf(x[k] - m));
  }
};

__device__ __forceinline__ void combine_stat(float& m, float& s, float m2, float s2) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) { m = mn; s = 0.f; return; }
  s = (m == -INFINITY ? 0.f : s * expf(m - mn)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - mn));
  m = mn;
}

__device__ __forceinline__ void warp_combine_stat(float& m, float& s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    combine_stat(m, s, m2, s2);
  }
}

// ------------------------------------------------------------------ pass 1
template <typename T, int VEC, int CAP>
__global__ void __launch_bounds__(kSpecThreads)
spec_stats_generic_kernel(const __grid_constant__ SpecParams<CAP> p) {
  __shared__ float4 red[kSpecWarps];
  __shared__ float4 cl_slot[kMaxCluster];
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
  const int vbeg = static_cast<int>((static_cast<long long>(crank) * p.nvec) / csize);
  const int vend = static_cast<int>((static_cast<long long>(crank + 1) * p.nvec) / csize);

  pdl_wait_prior_grid();
  pdl_launch_dependents();

  OnlineSoftmaxStat sz, sw;
  constexpr int U = 4;
  for (int v0 = vbeg + threadIdx.x; v0 < vend; v0 += U * kSpecThreads) {
    float xz[U][VEC], xw[U][VEC];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int v = v0 + k * kSpecThreads;
      if (v < vend) {
        RowLoader<T, VEC>::load(zrow, v, xz[k]);
        if (has_q) RowLoader<T, VEC>::load(wrow_p, v, xw[k]);
      } else {
#pragma unroll
        for (int e = 0; e < VEC; ++e) xz[k][e] = xw[k][e] = -INFINITY;
      }
    }
#pragma unroll
    for (int k = 0; k < U; ++k) {
      sz.add(xz[k]);
      if (has_q) sw.add(xw[k]);
    }
  }
  float mz = sz.m, vz = sz.s.value(), mw = sw.m, vw = sw.s.value();
  warp_combine_stat(mz, vz);
  warp_combine_stat(mw, vw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = make_float4(mz, vz, mw, vw);
  __syncthreads();
  cluster_wait_acquire();  // phase A complete: rank 0 is running
  if (threadIdx.x == 0) {
    float4 a = red[0];
    for (int k = 1; k < kSpecWarps; ++k) {
      combine_stat(a.x, a.y, red[k].x, red[k].y);
      combine_stat(a.z, a.w, red[k].z, red[k].w);
    }
    dsmem_st_f32x4(dsmem_map(&cl_slot[crank], 0), a.x, a.y, a.z, a.w);
  }
  cluster_arrive_release();  // phase B: slices delivered to rank 0
  cluster_wait_acquire();
  if (crank != 0 || threadIdx.x != 0) return;

  float4 a = cl_slot[0];
  for (uint32_t k = 1; k < csize; ++k) {
    combine_stat(a.x, a.y, cl_slot[k].x, cl_slot[k].y);
    combine_stat(a.z, a.w, cl_slot[k].z, cl_slot[k].w);
  }
  static_cast<float4*>(p.stats)[n] = a;
  float pd = 0.f, qd = 0.f;
  unsigned char flag = 0;
  if (has_q) {
    const int d = p.draft_tokens[wrow];
    if (d >= 0 && d < p.V) {
      pd = expf(load_elem<T>(zrow, d) - a.x) / a.y;
      qd = expf(load_elem<T>(wrow_p, d) - a.z) / a.w;
      flag = verify_uniforms(p.seed, static_cast<unsigned>(p.uid[ui]), t).x * qd < pd ? 1 : 0;
    } else {
      atomicOr(p.status, kDevErrBadToken);
    }
  }
  p.flags[n] = flag;
  if (p.draft_probs) reinterpret_cast<float2*>(p.draft_probs)[n] = make_float2(pd, qd);
}

// ------------------------------------------------------------------ pass 2
template <typename T, int VEC, int CAP>
__global__ void __launch_bounds__(kSpecThreads)
spec_sample_generic_kernel(const __grid_constant__ SpecParams<CAP> p) {
  __shared__ double slice_sum[2][kMaxCluster];
  __shared__ double warp_sum[kSpecWarps];
  __shared__ int s_off, s_a;
  __shared__ int s_cnt[kSpecWarps];
  const uint32_t crank = cluster_ctarank();
  const uint32_t csize = cluster_nctarank();
  cluster_arrive_relaxed();  // phase A: every CTA has started

  const int ui = blockIdx.x / csize;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait_prior_grid();
  pdl_launch_dependents();

  // a_i and the packed offset sum_{j<i} (a_j + 1), by warp ballots
  int cnt = 0;
  for (int j = warp; j < ui; j += kSpecWarps) cnt += accepted_prefix<CAP>(p, j, lane) + 1;
  if (lane == 0) s_cnt[warp] = cnt;
  if (warp == 0) {
    const int a = accepted_prefix<CAP>(p, ui, lane);
    if (lane == 0) s_a = a;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int o = 0;
    for (int k = 0; k < kSpecWarps; ++k) o += s_cnt[k];
    s_off = o;
  }
  __syncthreads();
  const int a = s_a, off = s_off;
  const int q0 = p.q_off[ui], l0 = p.l_off[ui];
  const int Li = p.q_off[ui + 1] - q0 - 1;
  if (crank == 0) {
    for (int k = threadIdx.x; k < a; k += kSpecThreads) p.out_tokens[off + k] = p.draft_tokens[l0 + k];
    if (threadIdx.x == 0) {
      p.accept_len[ui] = a;
      p.out_offsets[ui] = off;
      if (ui == p.B - 1) p.out_offsets[p.B] = off + a + 1;
    }
  }

  // sampling distribution at position a
  const int n = q0 + a;
  const float4 st = static_cast<const float4*>(p.stats)[n];
  const T* zrow = static_cast<const T*>(p.z) + static_cast<size_t>(n) * p.V;
  const T* wrow = static_cast<const T*>(p.w) + static_cast<size_t>(a < Li ? l0 + a : 0) * p.V;
  const float u = verify_uniforms(p.seed, static_cast<unsigned>(p.uid[ui]), a).y;
  const float inv_z = 1.f / st.y, inv_w = 1.f / st.w;
  bool residual = a < Li;

  const int sbeg = static_cast<int>((static_cast<long long>(crank) * p.nvec) / csize);
  const int send = static_cast<int>((static_cast<long long>(crank + 1) * p.nvec) / csize);
  const int wbeg = sbeg + static_cast<int>((static_cast<long long>(warp) * (send - sbeg)) / kSpecWarps);
  const int wend = sbeg + static_cast<int>((static_cast<long long>(warp + 1) * (send - sbeg)) / kSpecWarps);

  auto weights = [&](int v, float (&wt)[VEC]) {
    float xz[VEC];
    RowLoader<T, VEC>::load(zrow, v, xz);
    if (residual) {
      float xw[VEC];
      RowLoader<T, VEC>::load(wrow, v, xw);
#pragma unroll
      for (int e = 0; e < VEC; ++e)
        wt[e] = fmaxf(expf(xz[e] - st.x) * inv_z - expf(xw[e] - st.z) * inv_w, 0.f);
    } else {
#pragma unroll
      for (int e = 0; e < VEC; ++e) wt[e] = expf(xz[e] - st.x);
    }
  };

  bool phase_a_done = false;
  for (int round = 0; round < 2; ++round) {
    // slice sum: lane-strided compensated sums, warp tree, block in fp64
    KahanSum acc;
    for (int v = wbeg + lane; v < wend; v += 32) {
      float wt[VEC];
      weights(v, wt);
      float ls = 0.f;
#pragma unroll
      for (int e = 0; e < VEC; ++e) ls += wt[e];
      acc.add(ls);
    }
    double ws = acc.value();
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ws += __shfl_xor_sync(0xffffffffu, ws, o);
    if (lane == 0) warp_sum[warp] = ws;
    __syncthreads();
    if (!phase_a_done) cluster_wait_acquire();  // phase A complete: all CTAs running
    phase_a_done = true;
    if (threadIdx.x == 0) {
      double s = 0.0;
      for (int k = 0; k < kSpecWarps; ++k) s += warp_sum[k];
      for (uint32_t r = 0; r < csize; ++r) dsmem_st_f64(dsmem_map(&slice_sum[round][crank], r), s);
    }
    cluster_arrive_release();
    cluster_wait_acquire();

    double total = 0.0;
    for (uint32_t r = 0; r < csize; ++r) total += slice_sum[round][r];
    if (!(total > 0.0)) {
      if (residual) { residual = false; continue; }  // empty residual: fall back to p
      return;                                         // cannot happen for finite logits
    }
    const double target = static_cast<double>(u) * total;
    // slice holding the crossing; if rounding leaves none, the last slice with mass
    double before = 0.0;
    int cs = -1;
    for (uint32_t r = 0; r < csize; ++r) {
      if (before + slice_sum[round][r] > target) { cs = static_cast<int>(r); break; }
      before += slice_sum[round][r];
    }
    bool take_last = false;
    if (cs < 0) {
      take_last = true;
      for (int r = static_cast<int>(csize) - 1; r >= 0; --r)
        if (slice_sum[round][r] > 0.0) { cs = r; break; }
      before = 0.0;
      for (int r = 0; r < cs; ++r) before += slice_sum[round][r];
    }
    if (cs != static_cast<int>(crank)) return;

    // warp holding the crossing
    double rem = target - before;
    int wsel = -1;
    double wbefore = 0.0;
    if (!take_last) {
      for (int k = 0; k < kSpecWarps; ++k) {
        if (wbefore + warp_sum[k] > rem) { wsel = k; break; }
        wbefore += warp_sum[k];
      }
    }
    if (wsel < 0) {  // the last warp with mass, and its last positive weight
      take_last = true;
      for (int k = kSpecWarps - 1; k >= 0; --k)
        if (warp_sum[k] > 0.0) { wsel = k; break; }
    }
    if (warp != wsel) return;
    rem -= wbefore;

    // scan the warp's range in groups of 32 consecutive vectors
    int token = -1, last_pos = -1;
    double run = 0.0;
    for (int g = wbeg; g < wend; g += 32) {
      const int v = g + lane;
      float wt[VEC];
      if (v < wend) weights(v, wt);
      else {
#pragma unroll
        for (int e = 0; e < VEC; ++e) wt[e] = 0.f;
      }
      float ls = 0.f;
#pragma unroll
      for (int e = 0; e < VEC; ++e) ls += wt[e];
      float incl = ls;  // inclusive scan over lanes
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const float gsum = __shfl_sync(0xffffffffu, incl, 31);
      // last positive weight seen so far (for the rounding fallback)
      int lp = -1;
#pragma unroll
      for (int e = 0; e < VEC; ++e)
        if (wt[e] > 0.f) lp = v * VEC + e;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, o));
      if (lp >= 0) last_pos = lp;
      if (!take_last && run + gsum > rem) {
        const unsigned hit = __ballot_sync(0xffffffffu, run + static_cast<double>(incl) > rem);
        const int ln = __ffs(hit) - 1;
        if (lane == ln) {
          double c = run + static_cast<double>(incl - ls);
          int k = -1;
#pragma unroll
          for (int e = 0; e < VEC; ++e) {
            c += wt[e];
            if (k < 0 && c > rem) k = e;
          }
          if (k < 0) {  // rounding inside the lane: its last positive weight
            for (int e = VEC - 1; e >= 0; --e)
              if (wt[e] > 0.f) { k = e; break; }
          }
          token = v * VEC + k;
        }
        token = __shfl_sync(0xffffffffu, token, ln);
        break;
      }
      run += gsum;
    }
    if (token < 0) token = last_pos;
    if (lane == 0) p.out_tokens[off + a] = token;
    return;
  }
}

}  // namespace dipsd
