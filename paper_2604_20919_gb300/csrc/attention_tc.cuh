// verify_attention on the 5th-generation tensor cores (tcgen05 + TMEM).
//
// Same work decomposition and output contract as verify_attention_kernel
// (attention.cuh): one CTA per (user i, KV head h, row block, KV split);
// rows r = t*G + g pack the G query heads of the KV group and the T_i verify
// tokens (Sec. II-A stage 2: all L_i+1 tokens of a user are verified in one
// pass), so each K/V byte brought on chip serves every row.
//
// Roles (6 warps):
//   warp 0      TMA producer: 4-D tensor-map loads of the user's pages into
//               a 4-stage ring of 64-token K and V tiles (128-byte swizzle);
//               page ids are fetched 32 at a time, one per lane, a group
//               ahead, and a tile's 16 boxes go out from 16 lanes at once.
//   warp 1      allocates TMEM; one thread issues tcgen05.mma:
//                 S[b] = Q K^T   (M=128 rows, N=64 keys, K=16 per instruction)
//                 O   += P V     (two N=64 column halves of head_dim)
//               and commits completions to mbarriers.
//   warps 2..5  one query row per thread (TMEM lane = row): load S with
//               tcgen05.ld, causal mask, online softmax in log2 units with a
//               lazy rescale (O in TMEM is rescaled only when a row maximum
//               grows by more than 2^8), write P as bf16 into a swizzled
//               shared buffer, and finally read O back for the output.
// TMEM columns: S double buffer [0,64) [64,128), O [128, 128+D).
#pragma once

#include "attention.cuh"
#include "tcgen05.cuh"

namespace dipsd {

constexpr int kTcThreads = 192;
constexpr int kTcStages = 4;
constexpr int kTcTile = 64;                // keys per tile
constexpr uint32_t kTmemCols = 256;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct TcSmem {
  static constexpr int kHalves = D / 64;
  static constexpr int kQBytes = kHalves * 128 * 128;         // 128 rows x D bf16
  static constexpr int kTileBytes = kHalves * kTcTile * 128;  // 64 keys x D bf16 (K or V)
  static constexpr int kStageBytes = 2 * kTileBytes;
  static constexpr int kPBytes = 128 * 128;                   // 128 rows x 64 keys bf16
  static constexpr int kQOff = 0;
  static constexpr int kKVOff = kQOff + kQBytes;
  static constexpr int kPOff = kKVOff + kTcStages * kStageBytes;
  static constexpr int kBarOff = kPOff + 2 * kPBytes;
  static constexpr int kBytes = kBarOff + 256;
  static constexpr int kAlloc = kBytes + 1024;  // slack for 1024-byte alignment
};

template <int D, int CAP>
__global__ void __launch_bounds__(kTcThreads, 1)
verify_attention_tc_kernel(const __grid_constant__ AttnParams<CAP> p, const __grid_constant__ CUtensorMap tm_k,
                           const __grid_constant__ CUtensorMap tm_v) {
  using L = TcSmem<D>;
  constexpr int kHalves = L::kHalves;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem + L::kQOff;
  uint8_t* sKV = smem + L::kKVOff;
  uint8_t* sP = smem + L::kPOff;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  uint64_t* kv_full = bars;                // [kTcStages]
  uint64_t* kv_empty = bars + kTcStages;   // [kTcStages]
  uint64_t* s_full = bars + 2 * kTcStages;  // [2]
  uint64_t* s_empty = s_full + 2;           // [2]
  uint64_t* p_full = s_empty + 2;           // [2]
  uint64_t* pv_done = p_full + 2;           // [2]
  uint64_t* o_final = pv_done + 2;
  uint64_t* q_ready = o_final + 1;
  uint64_t* mma_done = q_ready + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);

  // ---- work item (same decode as the mma.sync kernel)
  const int item = blockIdx.x;
  const int ui = find_user<CAP>(p.item_off, p.B, item);
  const AttnUser U = p.u[ui];
  int local = item - p.item_off[ui];
  const int split = local % U.nsplit;
  local /= U.nsplit;
  const int h = local % p.Hkv;
  const int rb = local / p.Hkv;
  const int M = p.G * U.T;
  const int row0 = rb * 128;
  const int kv_begin = split * U.split_len;
  const int kv_end = min(kv_begin + U.split_len, U.kv_len);
  const int ntiles = (kv_end - kv_begin + kTcTile - 1) / kTcTile;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_empty[b], 4);
      mbar_init(&p_full[b], 4);
      mbar_init(&pv_done[b], 1);
    }
    mbar_init(o_final, 1);
    mbar_init(q_ready, 4);
    mbar_init(mma_done, 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS0 = tmem, tO = tmem + 128;
  pdl_wait_prior_grid();
  pdl_launch_dependents();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // Page ids come from the block table 32 at a time (one per lane, one
    // group of 8 tiles ahead) so no TMA waits on a dependent global load.
    const int* bt = p.block_table + static_cast<size_t>(U.bt_row) * p.max_blocks;
    const int n_pages = (U.kv_len + kPage - 1) / kPage;
    const int page_base = kv_begin / kPage;
    auto fetch = [&](int group) {
      const int page = page_base + group * 32 + lane;
      return page < n_pages ? __ldg(bt + page) : 0;
    };
    int cur = fetch(0);
    int nxt = fetch(1);
    int issued = 0;
    for (int j = 0; j < ntiles; ++j) {
      const int st = j % kTcStages;
      if ((j & 7) == 0 && j > 0) {
        cur = nxt;
        nxt = fetch((j >> 3) + 1);
      }
      bool go = true;
      if (j >= kTcStages && lane == 0) go = mbar_wait(&kv_empty[st], ((j / kTcStages) - 1) & 1, p.status);
      go = __shfl_sync(0xffffffffu, go, 0);
      if (!go) break;
      int blk[kTcTile / kPage];
#pragma unroll
      for (int pg = 0; pg < kTcTile / kPage; ++pg) blk[pg] = __shfl_sync(0xffffffffu, cur, (j & 7) * 4 + pg);
      // one box (one page, one 64-column half, K or V) per lane: a tile's
      // boxes go out in a single warp-wide TMA instruction
      if (lane == 0) mbar_arrive_expect_tx(&kv_full[st], L::kStageBytes);
      __syncwarp();
      {
        constexpr int kBoxes = (kTcTile / kPage) * kHalves;  // per K tile (and per V tile)
        if (lane < 2 * kBoxes) {
          const int isv = lane >= kBoxes;
          const int bx = isv ? lane - kBoxes : lane;
          const int pg = bx / kHalves, hf = bx % kHalves;
          int bk = blk[0];
#pragma unroll
          for (int q = 1; q < kTcTile / kPage; ++q)
            if (pg == q) bk = blk[q];
          uint8_t* dst = sKV + st * L::kStageBytes + (isv ? L::kTileBytes : 0) + hf * (kTcTile * 128) +
                         pg * kPage * 128;
          tma_load_4d(dst, isv ? &tm_v : &tm_k, hf * 64, 0, h, bk, &kv_full[st]);
        }
      }
      ++issued;
    }
    if (lane == 0)
      for (int j = max(0, issued - kTcStages); j < issued; ++j)
        mbar_wait(&kv_full[j % kTcStages], (j / kTcStages) & 1, p.status);
  } else if (warp == 1) {
    // ----------------------------------------------------- MMA issuer (1 thread)
    if (lane == 0) {
      constexpr uint32_t kIdQK = idesc_bf16_f32(128, kTcTile, false, false);
      constexpr uint32_t kIdPV = idesc_bf16_f32(128, 64, false, true);
      const uint32_t q_addr = smem_addr(sQ);
      const uint32_t kv_addr = smem_addr(sKV);
      const uint32_t p_addr = smem_addr(sP);
      bool ok = mbar_wait(q_ready, 0, p.status);
      auto issue_pv = [&](int jj) -> bool {
        const int st = jj % kTcStages, b = jj & 1;
        if (!mbar_wait(&p_full[b], (jj >> 1) & 1, p.status)) return false;
        tc_fence_after();
        const uint32_t v_addr = kv_addr + st * L::kStageBytes + L::kTileBytes;
#pragma unroll
        for (int hf = 0; hf < kHalves; ++hf) {
#pragma unroll
          for (int kk = 0; kk < kTcTile / 16; ++kk) {
            const uint64_t a = smem_desc_sw128(p_addr + b * L::kPBytes + kk * 32, 0, 1024);
            const uint64_t bd = smem_desc_sw128(v_addr + hf * (kTcTile * 128) + kk * 16 * 128, 1024, 1024);
            tc_mma(tO + hf * 64, a, bd, kIdPV, (jj > 0 || kk > 0) ? 1u : 0u);
          }
        }
        tc_commit(&pv_done[b]);
        tc_commit(&kv_empty[st]);
        return true;
      };
      for (int j = 0; ok && j < ntiles; ++j) {
        const int st = j % kTcStages, b = j & 1;
        if (!mbar_wait(&kv_full[st], (j / kTcStages) & 1, p.status)) { ok = false; break; }
        if (j >= 2 && !mbar_wait(&s_empty[b], ((j - 2) >> 1) & 1, p.status)) { ok = false; break; }
        tc_fence_after();
        const uint32_t k_addr = kv_addr + st * L::kStageBytes;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t hoff = (kk >> 2) * (128 * 128), koff = (kk >> 2) * (kTcTile * 128);
          const uint64_t a = smem_desc_sw128(q_addr + hoff + (kk & 3) * 32, 0, 1024);
          const uint64_t bd = smem_desc_sw128(k_addr + koff + (kk & 3) * 32, 0, 1024);
          tc_mma(tS0 + b * kTcTile, a, bd, kIdQK, kk > 0 ? 1u : 0u);
        }
        tc_commit(&s_full[b]);
        if (j >= 1 && !issue_pv(j - 1)) { ok = false; break; }
      }
      if (ok && ntiles > 0) ok = issue_pv(ntiles - 1);
      tc_commit(o_final);
      tc_commit(mma_done);
      mbar_wait(mma_done, 0, p.status);
    }
  } else {
    // ----------------------------------------- softmax / epilogue (row per thread)
    const int quad = warp & 3;
    const int r = quad * 32 + lane;  // row within the block == TMEM lane
    const int rg = row0 + r;         // row within the user
    const bool valid = rg < M;
    const int t = rg / p.G, g = rg % p.G;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;

    // Q row -> shared memory (K-major, 128-byte swizzle); padding rows are zero
    {
      const __nv_bfloat16* qrow = p.q + (static_cast<size_t>(U.q_off + t) * p.Hq + h * p.G + g) * D;
#pragma unroll
      for (int c = 0; c < D / 8; ++c) {
        uint4 v = make_uint4(0, 0, 0, 0);
        if (valid) v = __ldg(reinterpret_cast<const uint4*>(qrow) + c);
        const int hf = c >> 3, ch = c & 7;
        *reinterpret_cast<uint4*>(sQ + hf * (128 * 128) + r * 128 + ((ch ^ (r & 7)) << 4)) = v;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_ready);
    }

    const int last_vis = U.ctx + t;  // last visible key of this row
    // warps whose 32 rows are all padding only keep the barrier phases in step
    const bool active = row0 + quad * 32 < M;
    const float sl2 = p.scale_log2;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      const int b = j & 1, st = j % kTcStages;
      const int key0 = kv_begin + j * kTcTile;
      ok = __all_sync(0xffffffffu, mbar_wait(&s_full[b], (j >> 1) & 1, p.status));
      if (!ok) break;
      uint32_t sr[2][32];
      if (active) {
        tc_fence_after();
        tmem_ld32(tS0 + b * kTcTile + lane_base, sr[0]);
        tmem_ld32(tS0 + b * kTcTile + 32 + lane_base, sr[1]);
        tc_fence_before();
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[b]);

      if (active) {
        // raw scores; the causal rule key <= C_i + t only bites near the end
        float s[kTcTile];
        float mr = -INFINITY;
        const bool need_mask = key0 + kTcTile - 1 > U.ctx;
#pragma unroll
        for (int c = 0; c < kTcTile; ++c) {
          float v = __uint_as_float(sr[c >> 5][c & 31]);
          if (need_mask && key0 + c > last_vis) v = -INFINITY;
          s[c] = v;
          mr = fmaxf(mr, v);
        }
        const float mt = mr * sl2;  // tile maximum in log2 units (scale > 0)
        // lazy rescale: keep the old maximum unless this tile exceeds it by 2^8
        const bool grow = m == -INFINITY ? (mt > -INFINITY) : (mt > m + kRescaleThreshold);
        float factor = 1.f;
        if (grow) {
          factor = m == -INFINITY ? 1.f : fast_exp2(m - mt);
          m = mt;
        }
        if (j > 0 && __any_sync(0xffffffffu, grow && factor != 1.f)) {
          ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[(j - 1) & 1], ((j - 1) >> 1) & 1, p.status));
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int cc = 0; cc < D / 32; ++cc) {
            uint32_t o[32];
            tmem_ld32(tO + cc * 32 + lane_base, o);
#pragma unroll
            for (int k = 0; k < 32; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * factor);
            tmem_st32(tO + cc * 32 + lane_base, o);
          }
          tc_fence_before();
        }
        l *= factor;
        const float nb = m == -INFINITY ? 0.f : -m;
        uint32_t pk[kTcTile / 2];
#pragma unroll
        for (int c = 0; c < kTcTile; c += 2) {
          const float p0 = fast_exp2(__fmaf_rn(s[c], sl2, nb));
          const float p1 = fast_exp2(__fmaf_rn(s[c + 1], sl2, nb));
          l += p0 + p1;
          pk[c >> 1] = pack_bf16x2(p0, p1);
        }
        // P buffer b was last read by the PV of tile j-2
        if (j >= 2) {
          ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[b], ((j - 2) >> 1) & 1, p.status));
          if (!ok) break;
        }
        uint8_t* prow = sP + b * L::kPBytes + r * 128;
#pragma unroll
        for (int ch = 0; ch < 8; ++ch)
          *reinterpret_cast<uint4*>(prow + ((ch ^ (r & 7)) << 4)) =
              make_uint4(pk[4 * ch], pk[4 * ch + 1], pk[4 * ch + 2], pk[4 * ch + 3]);
      }
      // V rows past kv_len may hold anything; zero them before P V reads them
      if (key0 + kTcTile > U.kv_len) {
        ok = __all_sync(0xffffffffu, mbar_wait(&kv_full[st], (j / kTcStages) & 1, p.status));
        if (!ok) break;
        uint8_t* vt = sKV + st * L::kStageBytes + L::kTileBytes;
        const int first = U.kv_len - key0;  // first key row to clear
        const int nchunks = (kTcTile - first) * kHalves * 8;
        for (int c = threadIdx.x - 64; c < nchunks; c += 128) {
          const int row = first + c / (kHalves * 8);
          const int rem = c % (kHalves * 8);
          *reinterpret_cast<uint4*>(vt + (rem >> 3) * (kTcTile * 128) + row * 128 + ((rem & 7) << 4)) =
              make_uint4(0, 0, 0, 0);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[b]);
    }

    // ---- epilogue: O row from TMEM
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_final, 0, p.status));
    if (ok && active) {
      tc_fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      __nv_bfloat16* orow = p.out + (static_cast<size_t>(U.q_off + t) * p.Hq + h * p.G + g) * D;
      const long long prow_idx = p.part_off[ui] + static_cast<long long>(split * p.Hkv + h) * M + rg;
#pragma unroll
      for (int cc = 0; cc < D / 32; ++cc) {
        uint32_t o[32];
        tmem_ld32(tO + cc * 32 + lane_base, o);
        if (!valid) continue;
        if (U.nsplit == 1) {
          uint4* dst = reinterpret_cast<uint4*>(orow + cc * 32);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            dst[k] = make_uint4(pack_bf16x2(__uint_as_float(o[8 * k]) * inv, __uint_as_float(o[8 * k + 1]) * inv),
                                pack_bf16x2(__uint_as_float(o[8 * k + 2]) * inv, __uint_as_float(o[8 * k + 3]) * inv),
                                pack_bf16x2(__uint_as_float(o[8 * k + 4]) * inv, __uint_as_float(o[8 * k + 5]) * inv),
                                pack_bf16x2(__uint_as_float(o[8 * k + 6]) * inv, __uint_as_float(o[8 * k + 7]) * inv));
        } else {
          float4* dst = reinterpret_cast<float4*>(p.part_o + prow_idx * D + cc * 32);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            dst[k] = make_float4(__uint_as_float(o[4 * k]), __uint_as_float(o[4 * k + 1]),
                                 __uint_as_float(o[4 * k + 2]), __uint_as_float(o[4 * k + 3]));
        }
      }
      if (valid && U.nsplit > 1) p.part_ml[prow_idx] = make_float2(m, l);
      tc_fence_before();
    }
  }

  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace dipsd
