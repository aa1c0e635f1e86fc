// Pieces shared by the two speculative-sampling paths (staged and generic):
// launch constants, the parameter block, row element loaders, the user
// lookup and the ballot that counts a user's leading accepted drafts.
#pragma once

#include "common.cuh"
#include "philox.cuh"

namespace dipsd {

constexpr int kSpecThreads = 256;
constexpr int kSpecWarps = kSpecThreads / 32;
constexpr int kMaxCluster = 8;
constexpr unsigned kDevErrBadToken = 2u;
constexpr int kMaxTopK = 64;  // sparse payload: table entries per draft row
// Counters of the register path, in 32-bit words: one 64-bit word per user
// for the decisions (arrivals in the high half, acceptance bit t of position
// t in the low half); then one per user for the sampling segments.
constexpr int kCntUser1 = 0;
constexpr int kCntUser2 = kCntUser1 + 2 * kMaxUsers;
constexpr int kCounterWords = kCntUser2 + kMaxUsers;

template <int CAP>
struct SpecParams {
  const void* z;              // target logits [sum T][V]
  const void* w;              // draft logits  [sum L][V]
  const int* draft_tokens;    // [sum L]
  void* stats;                // [sum T] row statistics (layout private to each path)
  unsigned char* flags;       // [sum T]: acceptance bit
  float* u_res;               // [sum T]: resample uniform of each position (register path)
  float* draft_probs;         // optional [sum T][2]
  int* accept_len;            // [B]
  int* out_offsets;           // [B+1]
  int* out_tokens;            // [sum T]
  unsigned* status;
  // register path only: segment partial sums and arrival counters
  // sparse draft payload (spec_verify_sparse): per draft row, log q(d) and
  // a table of topk (token, q) entries; q is 0 off the table
  const float* draft_logq;  // [sum L]
  const int* topk_idx;      // [sum L][topk]
  const float* topk_q;      // [sum L][topk]
  int topk;
  float4* part1;       // [n_items1] one per segment of every row
  float4* part2;       // [n_items2] one per segment of the sampled rows
  unsigned* counters;  // [kCounterWords], zero between calls
  int sum_t, nseg1, nseg2, n_items1, n_items2;
  int B, V, nvec;             // nvec = V / VEC
  unsigned long long seed;    // Philox key word 0 (the caller's seed)
  int q_off[CAP + 1];         // first verify position of user i
  int l_off[CAP + 1];         // first draft row of user i
  int uid[CAP];               // Philox key word 1 of user i (its user id)
};

// ----------------------------------------------------- row element access
template <typename T, int VEC>
struct RowLoader;

template <>
struct RowLoader<__nv_bfloat16, 8> {
  static __device__ __forceinline__ void load(const __nv_bfloat16* row, int v, float (&x)[8]) {
    const uint4 r = ldg_stream_v4(row + static_cast<size_t>(v) * 8);
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      x[2 * k] = __uint_as_float(w[k] << 16);
      x[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
    }
  }
};
template <>
struct RowLoader<float, 4> {
  static __device__ __forceinline__ void load(const float* row, int v, float (&x)[4]) {
    const uint4 r = ldg_stream_v4(row + static_cast<size_t>(v) * 4);
    x[0] = __uint_as_float(r.x); x[1] = __uint_as_float(r.y);
    x[2] = __uint_as_float(r.z); x[3] = __uint_as_float(r.w);
  }
};
template <>
struct RowLoader<__nv_bfloat16, 1> {
  static __device__ __forceinline__ void load(const __nv_bfloat16* row, int v, float (&x)[1]) {
    x[0] = __bfloat162float(row[v]);
  }
};
template <>
struct RowLoader<float, 1> {
  static __device__ __forceinline__ void load(const float* row, int v, float (&x)[1]) { x[0] = row[v]; }
};

template <typename T>
__device__ __forceinline__ float load_elem(const T* row, int k) {
  if constexpr (sizeof(T) == 2) return __bfloat162float(row[k]);
  else return row[k];
}

template <int CAP>
__device__ __forceinline__ int spec_find_user(const int* off, int B, int idx) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= idx) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Leading accepted drafts of user j (ballot over its acceptance bits).
template <int CAP>
__device__ __forceinline__ int accepted_prefix(const SpecParams<CAP>& p, int j, int lane) {
  const int q0 = p.q_off[j];
  const int Lj = p.q_off[j + 1] - q0 - 1;
  const bool acc = lane < Lj && p.flags[q0 + lane] != 0;
  const unsigned rejected = ~__ballot_sync(0xffffffffu, acc);
  return min(__ffs(rejected) - 1, Lj);
}

}  // namespace dipsd
