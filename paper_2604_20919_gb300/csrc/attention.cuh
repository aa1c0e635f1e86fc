// verify_attention: causal GQA attention of each user's L_i + 1 verify tokens
// over that user's paged bf16 KV cache (the target model's attention during
// batch verification, Sec. II-A stage 2; the I*L term of Eq. (Fv)).
//
// This header holds what the attention kernel (attention_tc.cuh) shares with
// the host: the work parameters (rows r = t*G + g of user i pack its verify
// tokens and the G query heads of KV head h; a row block is 128 rows), the
// decoding of a CTA's work, and the two kernels that combine the KV splits of
// one (user, row block, head) through global memory when they do not run as
// one cluster: verify_attention_merge_kernel (one CTA per item plans) and
// verify_attention_merge_streams_kernel (the streams a persistent grid cut).
//
// Two ways to cut the work:
//   * items (one per CTA): (user, row block, KV head, split), every split of
//     a user `split_len` keys long;
//   * page streams (a persistent grid of at most one CTA per SM): the keys of
//     every (user, row block, KV head) as one stream of whole pages, the
//     streams of all users back to back, cut into chunks [chunk_bound[b],
//     chunk_bound[b + 1]), one per CTA.  A CTA takes the pieces of the
//     streams its chunk covers, in order; the host cuts the chunks so that
//     every CTA carries about the same pages plus a fixed cost per piece.  A
//     stream cut by a chunk boundary is merged afterwards, its split s being
//     its piece in the s-th chunk it touches.  A CTA finds its first piece
//     from per-chunk facts the host records and walks to each later one
//     directly (the next stream), without searching.
#pragma once

#include "common.cuh"

namespace dipsd {

constexpr unsigned kDevErrBadBlock = 4u;  // an appended row's page id outside [0, num_blocks)
constexpr int kMaxChunks = 256;           // CTAs of a grid over page streams

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

// A page stream cut by chunk bounds (persistent grid), as its merge reads
// it: written by the CTA that runs the stream's first split, read by the
// merge kernel after the grid.  Partial row of split s and row r of the
// stream's row block: part_row0 + s * step + r; output row of row rg =
// row0 + r (t = rg / G, g = rg % G): out_base + t * Hq + g.
struct MergeDesc {
  long long part_row0;
  long long out_base;
  int step, nsplit, nrows, row0;
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
  int n_chunks, total_pages;  // page streams (n_chunks > 0): chunks (CTAs), all pages
  float scale_log2;  // softmax_scale * log2(e)
  int item_off[CAP + 1];
  int page_off[CAP + 1];  // page streams: first page of user i's streams
  int chunk_bound[kMaxChunks + 1];  // page streams: chunk b is [chunk_bound[b], chunk_bound[b + 1])
  // page streams, per chunk b: the user of its first page, how many chunks
  // back the stream of its first page starts, and how many chunks ahead the
  // stream of its last page ends (so no CTA searches the chunk bounds)
  short chunk_user[kMaxChunks];
  unsigned char chunk_c0_back[kMaxChunks];
  unsigned char chunk_c1_fwd[kMaxChunks];
  // page streams: per chunk, the index of the cut stream that starts in it
  // (255: none); its merge descriptor goes to merge_desc[index]
  unsigned char chunk_cut[kMaxChunks];
  MergeDesc* merge_desc;
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

// One unit of a CTA's work: keys [kv_begin, kv_end) of the stream of user
// ui, row block rb and KV head h, which is split `split` of the stream's
// `nsplit`; `next` is where the CTA's next unit starts (page streams).
struct Work {
  int ui, h, rb, split, nsplit, kv_begin, kv_end, next;
};

__device__ __forceinline__ int pages_of(const AttnUser& U) { return (U.kv_len + kPage - 1) / kPage; }

// Item decoding: item = ((user, row block), head, split), split innermost.
template <int CAP>
__device__ __forceinline__ Work work_of_item(const AttnParams<CAP>& p, int item) {
  Work w;
  w.ui = find_user<CAP>(p.item_off, p.B, item);
  const AttnUser& U = p.u[w.ui];
  int local = item - p.item_off[w.ui];
  w.split = local % U.nsplit;
  local /= U.nsplit;
  w.h = local % p.Hkv;
  w.rb = local / p.Hkv;
  w.nsplit = U.nsplit;
  w.kv_begin = w.split * U.split_len;
  w.kv_end = min(w.kv_begin + U.split_len, U.kv_len);
  w.next = 0;
  return w;
}

// Page-stream decoding.  Streams of user i: index sidx = rb * Hkv + h, each
// pages_of(U) pages, from page page_off[i].  The piece of stream (ui, sidx)
// that starts at page `pos` in chunk `cta` (which ends at page `hi`), the
// stream starting in chunk c0: its splits run from chunk c0 to the chunk
// where it ends, which is `cta` unless the stream runs past `hi` (then this
// is the chunk's last piece, and the host recorded that chunk).
template <int CAP>
__device__ __forceinline__ Work piece_of_stream(const AttnParams<CAP>& p, int ui, int sidx, int pos, int c0,
                                                int cta, int hi) {
  Work w;
  const AttnUser& U = p.u[ui];
  const int np = pages_of(U);
  const int s0 = p.page_off[ui] + sidx * np;
  w.ui = ui;
  w.h = sidx % p.Hkv;
  w.rb = sidx / p.Hkv;
  w.next = min(hi, s0 + np);
  w.kv_begin = (pos - s0) * kPage;
  w.kv_end = min((w.next - s0) * kPage, U.kv_len);
  const int c1 = s0 + np <= hi ? cta : cta + p.chunk_c1_fwd[cta];
  w.nsplit = c1 - c0 + 1;
  w.split = cta - c0;
  return w;
}
// The first piece of chunk `cta`: it starts at the chunk's first page.
template <int CAP>
__device__ __forceinline__ Work first_piece(const AttnParams<CAP>& p, int cta, int hi) {
  const int pos = p.chunk_bound[cta];
  const int ui = p.chunk_user[cta];
  const int sidx = (pos - p.page_off[ui]) / pages_of(p.u[ui]);
  return piece_of_stream<CAP>(p, ui, sidx, pos, cta - p.chunk_c0_back[cta], cta, hi);
}
// The piece after w in chunk `cta` (w.next < hi): the next stream, from its
// first page, in this chunk.
template <int CAP>
__device__ __forceinline__ Work next_piece(const AttnParams<CAP>& p, const Work& w, int cta, int hi) {
  int ui = w.ui, sidx = w.rb * p.Hkv + w.h + 1;
  if (sidx == p.u[ui].n_rb * p.Hkv) {
    ++ui;
    sidx = 0;
  }
  return piece_of_stream<CAP>(p, ui, sidx, w.next, cta, cta, hi);
}

// Combines the KV splits of every (verify token, query head) row of users
// with more than one split (one CTA per item plans): m = max_s m_s, w_s = 2^(m_s - m),
// out = sum_s w_s o_s / sum_s w_s l_s.  One warp per row: lane k holds the
// (m, l) of splits k, k + 32, ..., the weights reach every lane by shuffle,
// and the O rows of eight splits are loaded before any is used.
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
  const int ns = U.nsplit;
  // partial row of split s: base + s * stride
  const long long base = p.part_off[ui] + static_cast<long long>(h) * M + t * p.G + g;
  const long long stride = static_cast<long long>(p.Hkv) * M;
  float m = -INFINITY;
  for (int s = lane; s < ns; s += 32) m = fmaxf(m, p.part_ml[base + s * stride].x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  constexpr int kPer = D / 32;
  float acc[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) acc[k] = 0.f;
  float l = 0.f;
  for (int c0 = 0; c0 < ns; c0 += 32) {
    // lane k: the weight of split c0 + k
    float w = 0.f;
    if (c0 + lane < ns) {
      const float2 ml = p.part_ml[base + (c0 + lane) * stride];
      w = ml.x == -INFINITY ? 0.f : fast_exp2(ml.x - m);
      l += w * ml.y;
    }
    const int nc = min(32, ns - c0);
    for (int k0 = 0; k0 < nc; k0 += 8) {
      float v[8][kPer];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float* po = p.part_o + (base + (c0 + k0 + k) * stride) * D + lane * kPer;
        if (k0 + k < nc) {
          if constexpr (kPer == 4) {
            const float4 x = *reinterpret_cast<const float4*>(po);
            v[k][0] = x.x; v[k][1] = x.y; v[k][2] = x.z; v[k][3] = x.w;
          } else {
            const float2 x = *reinterpret_cast<const float2*>(po);
            v[k][0] = x.x; v[k][1] = x.y;
          }
        } else {
#pragma unroll
          for (int e = 0; e < kPer; ++e) v[k][e] = 0.f;
        }
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float wk = __shfl_sync(0xffffffffu, w, (k0 + k) & 31);
#pragma unroll
        for (int e = 0; e < kPer; ++e) acc[e] += wk * v[k][e];
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
  const float inv = 1.f / l;
  __nv_bfloat16* out = p.out + (static_cast<size_t>(U.q_off + t) * p.Hq + hq) * D + lane * kPer;
#pragma unroll
  for (int k = 0; k < kPer; k += 2)
    *reinterpret_cast<uint32_t*>(out + k) = pack_bf16x2(acc[k] * inv, acc[k + 1] * inv);
}

// Combines the splits of the cut page streams of a persistent grid (the
// same formula as above, as a running merge: the weights are rescaled when a
// later split raises the maximum): CTA (k, c) takes cut stream k and its
// 32-column slice c, one thread per row of the stream's row block.  A round
// of loads brings the (m, l) and the O slices of two splits, so a stream cut
// once costs the descriptor load and one round.
template <int D, int CAP>
__global__ void __launch_bounds__(128)
verify_attention_merge_streams_kernel(const __grid_constant__ AttnParams<CAP> p) {
  pdl_wait_prior_grid();
  pdl_launch_dependents();
  const MergeDesc* dp = p.merge_desc + blockIdx.x;
  const int nrows = __ldcg(&dp->nrows);
  const int r = static_cast<int>(threadIdx.x);
  if (r >= nrows) return;
  const long long row = __ldcg(&dp->part_row0) + r;
  const long long step = __ldcg(&dp->step);
  const int ns = __ldcg(&dp->nsplit);
  const int col = blockIdx.y * 32;
  float m = -INFINITY, l = 0.f;
  float acc[32];
#pragma unroll
  for (int k = 0; k < 32; ++k) acc[k] = 0.f;
  for (int s0 = 0; s0 < ns; s0 += 2) {
    float2 ml[2];
    float4 v[2][8];
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      ml[b] = make_float2(-INFINITY, 0.f);
      if (s0 + b < ns) {
        const long long rs = row + (s0 + b) * step;
        ml[b] = __ldcg(p.part_ml + rs);
        const float4* po = reinterpret_cast<const float4*>(p.part_o + rs * D + col);
#pragma unroll
        for (int k = 0; k < 8; ++k) v[b][k] = __ldcg(po + k);
      }
    }
    // an empty split (no visible key: m = -inf, l = 0) weighs nothing
    const bool ok0 = ml[0].x > -INFINITY && ml[0].y > 0.f, ok1 = ml[1].x > -INFINITY && ml[1].y > 0.f;
    const float mn = fmaxf(m, fmaxf(ok0 ? ml[0].x : -INFINITY, ok1 ? ml[1].x : -INFINITY));
    if (mn > m) {
      const float f = m == -INFINITY ? 0.f : fast_exp2(m - mn);
#pragma unroll
      for (int k = 0; k < 32; ++k) acc[k] *= f;
      l *= f;
      m = mn;
    }
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      if (b == 0 ? ok0 : ok1) {
        const float w = fast_exp2(ml[b].x - m);
        l += w * ml[b].y;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          acc[4 * k] += w * v[b][k].x;
          acc[4 * k + 1] += w * v[b][k].y;
          acc[4 * k + 2] += w * v[b][k].z;
          acc[4 * k + 3] += w * v[b][k].w;
        }
      }
    }
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
  const int rg = __ldcg(&dp->row0) + r;
  const int t = rg / p.G, g = rg % p.G;
  uint4* dst = reinterpret_cast<uint4*>(p.out + (__ldcg(&dp->out_base) + static_cast<long long>(t) * p.Hq + g) * D + col);
#pragma unroll
  for (int k = 0; k < 4; ++k)
    dst[k] = make_uint4(pack_bf16x2(acc[8 * k] * inv, acc[8 * k + 1] * inv),
                        pack_bf16x2(acc[8 * k + 2] * inv, acc[8 * k + 3] * inv),
                        pack_bf16x2(acc[8 * k + 4] * inv, acc[8 * k + 5] * inv),
                        pack_bf16x2(acc[8 * k + 6] * inv, acc[8 * k + 7] * inv));
}

}  // namespace dipsd
