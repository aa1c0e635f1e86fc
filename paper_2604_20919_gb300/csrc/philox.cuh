// The verifier's uniforms, drawn in the kernels from a counter-based
// generator: Philox4x64-10 (Salmon, Moraes, Dror and Shaw, "Parallel random
// numbers: as easy as 1, 2, 3", SC 2011), keyed on (seed, user id).
//
// The paper leaves the random numbers of speculative sampling unspecified
// (Sec. II-A, stage 2 only states the accept / truncate / extra-token
// behaviour).  The reading taken here: user u's stream is the sequence of
// 64-bit words of Philox4x64-10 under key (seed, u) with counter blocks
// (1, 0, 0, 0), (2, 0, 0, 0), ... (four words per block, block b at counter
// b + 1); verify position t of the user takes words 2t and 2t + 1 (block t/2,
// words 2(t%2) and 2(t%2)+1): the first is its acceptance uniform, the second
// its resample uniform.  A word w maps to the exact fp32 value
// ((w >> 41) + 1/2) * 2^-23 in (0, 1).
#pragma once

#include "common.cuh"

namespace dipsd {

// Round multipliers and key increments of Philox4x64 (the SC 2011 paper's
// published constants).
constexpr unsigned long long kPhiloxM0 = 0xD2E7470EE14C6C93ull;
constexpr unsigned long long kPhiloxM1 = 0xCA5A826395121157ull;
constexpr unsigned long long kPhiloxW0 = 0x9E3779B97F4A7C15ull;
constexpr unsigned long long kPhiloxW1 = 0xBB67AE8584CAA73Bull;

struct PhiloxBlock {
  unsigned long long w[4];
};

// One 4 x 64-bit output block: ten rounds of the Philox S-P network on the
// counter c, the key bumped by (W0, W1) after every round.
__device__ __forceinline__ PhiloxBlock philox4x64_10(unsigned long long c0, unsigned long long c1,
                                                     unsigned long long c2, unsigned long long c3,
                                                     unsigned long long k0, unsigned long long k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const unsigned long long hi0 = __umul64hi(kPhiloxM0, c0), lo0 = kPhiloxM0 * c0;
    const unsigned long long hi1 = __umul64hi(kPhiloxM1, c2), lo1 = kPhiloxM1 * c2;
    c0 = hi1 ^ c1 ^ k0;
    c1 = lo1;
    c2 = hi0 ^ c3 ^ k1;
    c3 = lo0;
    k0 += kPhiloxW0;
    k1 += kPhiloxW1;
  }
  return PhiloxBlock{{c0, c1, c2, c3}};
}

// The exact fp32 uniform of one word: the top 23 bits plus one half, times 2^-23.
__device__ __forceinline__ float philox_word_to_uniform(unsigned long long w) {
  return __fmul_rn(static_cast<float>(static_cast<unsigned>(w >> 41)) + 0.5f, 1.1920928955078125e-7f);
}

// (u_acc, u_res) of verify position t of the user with Philox key (seed, uid).
__device__ __forceinline__ float2 verify_uniforms(unsigned long long seed, unsigned long long uid, int t) {
  const PhiloxBlock b = philox4x64_10(static_cast<unsigned long long>(t >> 1) + 1ull, 0ull, 0ull, 0ull, seed, uid);
  const unsigned long long wa = (t & 1) ? b.w[2] : b.w[0];
  const unsigned long long wr = (t & 1) ? b.w[3] : b.w[1];
  return make_float2(philox_word_to_uniform(wa), philox_word_to_uniform(wr));
}

// Words of counter blocks 0 .. n_blocks - 1 of the stream with key
// (seed, uid): out[4 b + j] = word j of block b.  One thread per block.
__global__ void __launch_bounds__(256) philox_words_kernel(unsigned long long seed, unsigned long long uid,
                                                           long long n_blocks, unsigned long long* __restrict__ out) {
  const long long b = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (b >= n_blocks) return;
  const PhiloxBlock r = philox4x64_10(static_cast<unsigned long long>(b) + 1ull, 0ull, 0ull, 0ull, seed, uid);
  ulonglong2* o = reinterpret_cast<ulonglong2*>(out + b * 4);
  o[0] = make_ulonglong2(r.w[0], r.w[1]);
  o[1] = make_ulonglong2(r.w[2], r.w[3]);
}

// A batch's users for verify_uniforms_kernel.
struct UniformParams {
  unsigned long long seed;
  int B;
  int q_off[kMaxUsers + 1];  // first verify position of user i; q_off[B] = sum T
  int uid[kMaxUsers];        // Philox key word of user i
};

// The (u_acc, u_res) pairs of every verify position of a batch, as the
// verification kernels draw them: out[q_off[i] + t] for t = 0 .. T_i - 1.
// One thread per position.
__global__ void __launch_bounds__(256) verify_uniforms_kernel(const __grid_constant__ UniformParams p,
                                                              float2* __restrict__ out) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= p.q_off[p.B]) return;
  int lo = 0, hi = p.B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.q_off[mid] <= n) lo = mid; else hi = mid - 1;
  }
  out[n] = verify_uniforms(p.seed, static_cast<unsigned>(p.uid[lo]), n - p.q_off[lo]);
}

}  // namespace dipsd
