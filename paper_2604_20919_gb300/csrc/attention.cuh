// verify_attention: causal GQA attention of each user's L_i + 1 verify tokens
// over that user's paged bf16 KV cache (the target model's attention during
// batch verification, Sec. II-A stage 2; the I*L term of Eq. (Fv)).
//
// Work item = (user i, KV head h, row block, KV split).  The G query heads
// that share KV head h, times the T_i verify tokens, form the rows of one
// tile (row r = t*G + g), so every K/V byte brought on chip serves all G*T_i
// query rows.  K/V pages stream through a shared-memory ring filled by TMA
// (4-D tensor maps over [block][head][slot][dim], 128-byte swizzle), guarded
// by mbarriers; a producer warp issues the copies, consumer warps (one per
// 16 query rows) run QK^T and PV on the tensor cores with an online softmax.
// Splits of one (user, head) are combined by verify_attention_merge_kernel.
#pragma once

#include "common.cuh"

namespace dipsd {

constexpr int kAttnTile = 64;  // KV tokens per pipeline stage (4 pages)

struct AttnUser {
  int q_off;      // first verify token of the user in q / out
  int ctx;        // C_i
  int T;          // L_i + 1
  int kv_len;     // C_i + T
  int bt_row;     // block-table row of the user
  int nsplit;     // KV splits
  int split_len;  // KV tokens per split (multiple of kAttnTile)
  int n_rb;       // row blocks
};

template <int CAP>
struct AttnParams {
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  const int* block_table;
  float2* part_ml;  // per partial row: (running max in log2 units, sum)
  float* part_o;    // per partial row: D unnormalised outputs
  unsigned* status;
  int cluster;  // > 1: the nsplit == cluster splits of a row block and head
                // form one thread-block cluster and merge in shared memory
  int B, Hq, Hkv, G, max_blocks;
  int n_items, n_merge;
  float scale_log2;  // softmax_scale * log2(e)
  int item_off[CAP + 1];
  int merge_off[CAP + 1];
  long long part_off[CAP];  // first partial row of the user (multi-split users)
  AttnUser u[CAP];
};

template <int CAP>
__device__ __forceinline__ int find_user(const int* off, int B, int idx) {
  int lo = 0, hi = B - 1;  // last i with off[i] <= idx
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= idx) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Byte offset of element (row, col) of a [kAttnTile][D] bf16 tile stored as
// D/64 column halves of [kAttnTile][64], each with the TMA 128-byte swizzle
// (16-byte chunk index XOR row mod 8).
template <int D>
__device__ __forceinline__ uint32_t tile_off(int row, int col) {
  const int half = col >> 6;
  const int chunk = (col & 63) >> 3;
  return half * (kAttnTile * 128) + row * 128 + ((chunk ^ (row & 7)) << 4) + ((col & 7) << 1);
}

template <int D, int NW, int STAGES, int CAP>
__global__ void __launch_bounds__((NW + 1) * 32, NW == 4 ? 2 : 1)
verify_attention_kernel(const __grid_constant__ AttnParams<CAP> p,
                        const __grid_constant__ CUtensorMap tm_k,
                        const __grid_constant__ CUtensorMap tm_v) {
  constexpr int kTileBytes = kAttnTile * D * 2;
  constexpr int kHalves = D / 64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * 2 * kTileBytes);
  uint64_t* empty = full + STAGES;

  // ---- decode the work item
  const int item = blockIdx.x;
  const int ui = find_user<CAP>(p.item_off, p.B, item);
  const AttnUser U = p.u[ui];
  int local = item - p.item_off[ui];
  const int split = local % U.nsplit;
  local /= U.nsplit;
  const int h = local % p.Hkv;
  const int rb = local / p.Hkv;
  const int M = p.G * U.T;
  const int row0 = rb * NW * 16;
  const int mtiles = min((M - row0 + 15) >> 4, NW);
  const int kv_begin = split * U.split_len;
  const int kv_end = min(kv_begin + U.split_len, U.kv_len);
  const int ntiles = (kv_end - kv_begin + kAttnTile - 1) / kAttnTile;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], mtiles);
    }
    fence_mbar_init();
  }
  if (warp == NW && lane == 0) {
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  __syncthreads();
  pdl_wait_prior_grid();
  pdl_launch_dependents();

  if (warp == NW) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const int* bt = p.block_table + static_cast<size_t>(U.bt_row) * p.max_blocks;
      const int n_pages = (U.kv_len + kPage - 1) / kPage;
      int issued = 0;
      for (int j = 0; j < ntiles; ++j) {
        const int st = j % STAGES;
        if (j >= STAGES && !mbar_wait(&empty[st], ((j / STAGES) - 1) & 1, p.status)) break;
        mbar_arrive_expect_tx(&full[st], 2 * kTileBytes);
        uint8_t* kd = smem + st * 2 * kTileBytes;
        uint8_t* vd = kd + kTileBytes;
        const int page0 = (kv_begin + j * kAttnTile) / kPage;
#pragma unroll
        for (int pg = 0; pg < kAttnTile / kPage; ++pg) {
          const int page = page0 + pg;
          const int blk = page < n_pages ? __ldg(bt + page) : 0;
#pragma unroll
          for (int hf = 0; hf < kHalves; ++hf) {
            const uint32_t off = hf * (kAttnTile * 128) + pg * kPage * 128;
            tma_load_4d(kd + off, &tm_k, hf * 64, 0, h, blk, &full[st]);
            tma_load_4d(vd + off, &tm_v, hf * 64, 0, h, blk, &full[st]);
          }
        }
        ++issued;
      }
      // Do not leave while copies into this CTA's shared memory are in flight.
      for (int j = max(0, issued - STAGES); j < issued; ++j)
        mbar_wait(&full[j % STAGES], (j / STAGES) & 1, p.status);
    }
    return;
  }
  if (warp >= mtiles) return;

  // -------------------------------------------------------------- consumer
  const int r_lo = row0 + warp * 16 + (lane >> 2);  // rows held by this thread
  const int r_hi = r_lo + 8;
  const int t_lo = r_lo / p.G, t_hi = r_hi / p.G;
  const int cpair = 2 * (lane & 3);

  // Q fragments (A operand) for all of D, kept in registers.
  uint32_t qa[D / 16][4];
  {
    const __nv_bfloat16* q_lo = p.q + (static_cast<size_t>(U.q_off + t_lo) * p.Hq + h * p.G + r_lo % p.G) * D;
    const __nv_bfloat16* q_hi = p.q + (static_cast<size_t>(U.q_off + t_hi) * p.Hq + h * p.G + r_hi % p.G) * D;
    const bool ok_lo = r_lo < M, ok_hi = r_hi < M;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const int c = kk * 16 + cpair;
      qa[kk][0] = ok_lo ? __ldg(reinterpret_cast<const uint32_t*>(q_lo + c)) : 0u;
      qa[kk][1] = ok_hi ? __ldg(reinterpret_cast<const uint32_t*>(q_hi + c)) : 0u;
      qa[kk][2] = ok_lo ? __ldg(reinterpret_cast<const uint32_t*>(q_lo + c + 8)) : 0u;
      qa[kk][3] = ok_hi ? __ldg(reinterpret_cast<const uint32_t*>(q_hi + c + 8)) : 0u;
    }
  }

  float o[D / 8][4];
#pragma unroll
  for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_lo = -INFINITY, m_hi = -INFINITY, l_lo = 0.f, l_hi = 0.f;
  const int vis_lo = U.ctx + t_lo, vis_hi = U.ctx + t_hi;  // last visible key

  // ldmatrix lane roles
  const int lm = lane >> 3, lr = lane & 7;

  for (int j = 0; j < ntiles; ++j) {
    const int st = j % STAGES;
    if (!mbar_wait(&full[st], (j / STAGES) & 1, p.status)) return;
    const uint32_t kbase = smem_addr(smem + st * 2 * kTileBytes);
    const uint32_t vbase = kbase + kTileBytes;
    const int key0 = kv_begin + j * kAttnTile;

    // S = Q K^T for 16 rows x 64 keys
    float s[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
      for (int jp = 0; jp < 4; ++jp) {
        const int key = jp * 16 + (lm >> 1) * 8 + lr;
        const int col = kk * 16 + (lm & 1) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kbase + tile_off<D>(key, col), b0, b1, b2, b3);
        mma_bf16_16816(s[2 * jp], qa[kk], b0, b1);
        mma_bf16_16816(s[2 * jp + 1], qa[kk], b2, b3);
      }
    }

    // scale to log2 units, apply the causal rule key <= C_i + t
    const bool need_mask = key0 + kAttnTile - 1 > U.ctx;
#pragma unroll
    for (int n = 0; n < 8; ++n) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float v = s[n][e] * p.scale_log2;
        if (need_mask) {
          const int key = key0 + n * 8 + cpair + (e & 1);
          if (key > ((e < 2) ? vis_lo : vis_hi)) v = -INFINITY;
        }
        s[n][e] = v;
      }
    }

    // online softmax
    float mx_lo = -INFINITY, mx_hi = -INFINITY;
#pragma unroll
    for (int n = 0; n < 8; ++n) {
      mx_lo = fmaxf(mx_lo, fmaxf(s[n][0], s[n][1]));
      mx_hi = fmaxf(mx_hi, fmaxf(s[n][2], s[n][3]));
    }
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 1));
    mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, 2));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 1));
    mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, 2));
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
    const float base_lo = mn_lo == -INFINITY ? 0.f : mn_lo;
    const float base_hi = mn_hi == -INFINITY ? 0.f : mn_hi;
    const float corr_lo = fast_exp2(m_lo - base_lo), corr_hi = fast_exp2(m_hi - base_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    l_lo *= corr_lo;
    l_hi *= corr_hi;
#pragma unroll
    for (int n = 0; n < D / 8; ++n) {
      o[n][0] *= corr_lo; o[n][1] *= corr_lo;
      o[n][2] *= corr_hi; o[n][3] *= corr_hi;
    }
    uint32_t pa[4][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) {
      const float p0 = fast_exp2(s[n][0] - base_lo), p1 = fast_exp2(s[n][1] - base_lo);
      const float p2 = fast_exp2(s[n][2] - base_hi), p3 = fast_exp2(s[n][3] - base_hi);
      l_lo += p0 + p1;
      l_hi += p2 + p3;
      pa[n >> 1][(n & 1) * 2 + 0] = pack_bf16x2(p0, p1);
      pa[n >> 1][(n & 1) * 2 + 1] = pack_bf16x2(p2, p3);
    }

    // O += P V; V rows past kv_len are zeroed in registers (they may hold
    // anything, and 0 * NaN would poison the row).
    const bool tail = key0 + kAttnTile > U.kv_len;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int dp = 0; dp < D / 16; ++dp) {
        const int key = kk * 16 + (lm & 1) * 8 + lr;
        const int col = dp * 16 + (lm >> 1) * 8;
        uint32_t b0, b1, b2, b3;
        ldsm_x4_trans(vbase + tile_off<D>(key, col), b0, b1, b2, b3);
        if (tail) {
          const int k_a = key0 + kk * 16 + cpair;  // keys of b0/b2: k_a, k_a+1; b1/b3: +8
          const uint32_t m0 = (k_a < U.kv_len ? 0xFFFFu : 0u) | (k_a + 1 < U.kv_len ? 0xFFFF0000u : 0u);
          const uint32_t m1 = (k_a + 8 < U.kv_len ? 0xFFFFu : 0u) | (k_a + 9 < U.kv_len ? 0xFFFF0000u : 0u);
          b0 &= m0; b2 &= m0; b1 &= m1; b3 &= m1;
        }
        mma_bf16_16816(o[2 * dp], pa[kk], b0, b1);
        mma_bf16_16816(o[2 * dp + 1], pa[kk], b2, b3);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);
  }

  // ---- epilogue
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 1);
  l_lo += __shfl_xor_sync(0xffffffffu, l_lo, 2);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 1);
  l_hi += __shfl_xor_sync(0xffffffffu, l_hi, 2);
  if (U.nsplit == 1) {
    const float inv_lo = 1.f / l_lo, inv_hi = 1.f / l_hi;
    __nv_bfloat16* out_lo = p.out + (static_cast<size_t>(U.q_off + t_lo) * p.Hq + h * p.G + r_lo % p.G) * D;
    __nv_bfloat16* out_hi = p.out + (static_cast<size_t>(U.q_off + t_hi) * p.Hq + h * p.G + r_hi % p.G) * D;
#pragma unroll
    for (int n = 0; n < D / 8; ++n) {
      const int c = n * 8 + cpair;
      if (r_lo < M) *reinterpret_cast<uint32_t*>(out_lo + c) = pack_bf16x2(o[n][0] * inv_lo, o[n][1] * inv_lo);
      if (r_hi < M) *reinterpret_cast<uint32_t*>(out_hi + c) = pack_bf16x2(o[n][2] * inv_hi, o[n][3] * inv_hi);
    }
  } else {
    const long long base = p.part_off[ui] + static_cast<long long>(split * p.Hkv + h) * M;
    if (r_lo < M) {
      if ((lane & 3) == 0) p.part_ml[base + r_lo] = make_float2(m_lo, l_lo);
      float* po = p.part_o + (base + r_lo) * D;
#pragma unroll
      for (int n = 0; n < D / 8; ++n)
        *reinterpret_cast<float2*>(po + n * 8 + cpair) = make_float2(o[n][0], o[n][1]);
    }
    if (r_hi < M) {
      if ((lane & 3) == 0) p.part_ml[base + r_hi] = make_float2(m_hi, l_hi);
      float* po = p.part_o + (base + r_hi) * D;
#pragma unroll
      for (int n = 0; n < D / 8; ++n)
        *reinterpret_cast<float2*>(po + n * 8 + cpair) = make_float2(o[n][2], o[n][3]);
    }
  }
}

// Combines the KV splits of every (verify token, query head) row of users
// with more than one split: m = max_s m_s, w_s = 2^(m_s - m),
// out = sum_s w_s o_s / sum_s w_s l_s.  One warp per row.
template <int D, int CAP>
__global__ void __launch_bounds__(128)
verify_attention_merge_kernel(const __grid_constant__ AttnParams<CAP> p) {
  pdl_wait_prior_grid();
  pdl_launch_dependents();
  const int row = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= p.n_merge) return;
  const int ui = find_user<CAP>(p.merge_off, p.B, row);
  const AttnUser U = p.u[ui];
  const int local = row - p.merge_off[ui];
  const int t = local / p.Hq, hq = local % p.Hq;
  const int h = hq / p.G, g = hq % p.G;
  const int M = p.G * U.T;
  const int r = t * p.G + g;
  float m = -INFINITY;
  for (int s = 0; s < U.nsplit; ++s) {
    const long long pr = p.part_off[ui] + static_cast<long long>(s * p.Hkv + h) * M + r;
    m = fmaxf(m, p.part_ml[pr].x);
  }
  constexpr int kPer = D / 32;
  float acc[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) acc[k] = 0.f;
  float l = 0.f;
  for (int s = 0; s < U.nsplit; ++s) {
    const long long pr = p.part_off[ui] + static_cast<long long>(s * p.Hkv + h) * M + r;
    const float2 ml = p.part_ml[pr];
    const float w = ml.x == -INFINITY ? 0.f : fast_exp2(ml.x - m);
    l += w * ml.y;
    const float* po = p.part_o + pr * D + lane * kPer;
    if constexpr (kPer == 4) {
      const float4 v = *reinterpret_cast<const float4*>(po);
      acc[0] += w * v.x; acc[1] += w * v.y; acc[2] += w * v.z; acc[3] += w * v.w;
    } else {
      const float2 v = *reinterpret_cast<const float2*>(po);
      acc[0] += w * v.x; acc[1] += w * v.y;
    }
  }
  const float inv = 1.f / l;
  __nv_bfloat16* out = p.out + (static_cast<size_t>(U.q_off + t) * p.Hq + hq) * D + lane * kPer;
#pragma unroll
  for (int k = 0; k < kPer; k += 2)
    *reinterpret_cast<uint32_t*>(out + k) = pack_bf16x2(acc[k] * inv, acc[k + 1] * inv);
}

}  // namespace dipsd
