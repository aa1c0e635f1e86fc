// verify_attention: causal GQA attention of each user's L_i + 1 verify tokens
// over that user's paged bf16 KV cache (the target model's attention during
// batch verification, Sec. II-A stage 2; the I*L term of Eq. (Fv)).
//
// This header holds what the attention kernel (attention_tc.cuh) shares with
// the host: the work-item parameters (work item = user i, KV head h, row
// block, KV split; rows r = t*G + g), and verify_attention_merge_kernel,
// which combines the splits of one (user, head) through global memory when
// they do not run as one cluster.
#pragma once

#include "common.cuh"

namespace dipsd {

constexpr unsigned kDevErrBadBlock = 4u;  // an appended row's page id outside [0, num_blocks)

struct AttnUser {
  int q_off;      // first verify token of the user in q / out
  int ctx;        // C_i
  int T;          // L_i + 1
  int kv_len;     // C_i + T
  int bt_row;     // block-table row of the user
  int nsplit;     // KV splits
  int split_len;  // KV tokens per split (a whole number of kernel tiles)
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
  // KV append (null: the verify tokens' rows are already in the cache):
  // [sum T][Hkv][D] rows written into the pages and used by this launch
  const __nv_bfloat16* new_k;
  const __nv_bfloat16* new_v;
  __nv_bfloat16* k_cache;  // [num_blocks][Hkv][16][D], written only when new_k is set
  __nv_bfloat16* v_cache;
  int num_blocks;          // cache blocks (bound for the append writes)
  // 1: the kernel reads nothing the preceding grid writes (it runs after the
  // spec_verify kernels of the same batch, whose own wait covered everything
  // before the call), so it waits for that grid only before it exits: the
  // launch then completes only after both stages have
  int wait_at_end;
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
