// verify_attention on the 5th-generation tensor cores (tcgen05 + TMEM).
//
// Work decomposition: rows r = t*G + g pack the G query heads of a KV group
// and the T_i verify tokens of user i (Sec. II-A stage 2: all L_i+1 tokens of
// a user are verified in one pass), so each K/V byte brought on chip serves
// every row.  One CTA per work item (user, row block, KV head, KV split), or
// (PERSIST) a grid of at most one CTA per SM over the page streams of every
// (user, row block, KV head) laid back to back and cut into equal chunks of
// pages (attention.cuh): CTA b takes the pieces of the streams its chunk
// covers.  The rings, the S/P buffers and every barrier phase then run on
// across pieces, so the producer streams the next piece's tiles while the
// softmax warps finish the current one; every CTA carries the same pages.
//
// Roles (6 warps):
//   warp 0      TMA producer into a ring of kStages 128-token K tiles and
//               a ring of as many V tiles (128-byte swizzle).  K: one box per
//               page and 64-column half (2 KB), stored half after half, so a
//               half is 128 rows at the uniform 1024-byte stride one N=128
//               product needs.  V: one box per page (4 KB at D = 128, both
//               halves through a 5-D tensor map whose third dimension steps
//               128 bytes), stored page after page.  K and V stages are
//               released separately: K once its Q K^T has run, V after its
//               P V.  Page ids are fetched 32 at a time, one per lane, a
//               group ahead.  A split's last tile loads only the pages up
//               to the split's end.  The K/V loads carry an evict-first L2
//               policy (each page is read once); in a persistent grid the
//               next two pieces' Q rows are prefetched into L2.
//   warp 1      allocates TMEM; one thread issues tcgen05.mma as operands
//               become ready (no fixed order between the two products):
//                 S[b] = Q K^T      (A = Q from tensor memory, M=128, N=128)
//                 O   += P[b] V     (A = P from tensor memory; a 16-key step
//                                    is one page of V, N = D: the
//                                    descriptor's leading offset steps to
//                                    the page's second 64-column half)
//               A tile costs 16 MMAs and 4 commits whatever D is; the
//               issuing thread, not the tensor core, is what bounds the
//               tile rate, so tiles are as long as the rings allow.
//   warps 2..5  one query row per thread (TMEM lane = row): put the Q row
//               in TMEM, then per tile read S[b] in 32-column chunks with
//               tcgen05.ld twice (tile maximum, then P), causal mask, online
//               softmax in log2 units with a lazy rescale (O in TMEM is
//               rescaled only when a row maximum grows by more than 2^8),
//               write P as bf16 pairs into the first 64 columns of S[b] with
//               tcgen05.st, and finally read O back.
// KV append (p.new_k set): the T_i new rows are not read from the cache.
// The producer patches them into every K/V tile that covers positions
// C_i .. C_i + T_i - 1 once the tile has landed, and signals the tile on
// k_patch / v_patch instead of k_full / v_full; the CTA with the last split
// and the first row block of each (user, head) also writes them into the
// pages (the round's state update).
// KV splits: either each split writes (m, l, O) rows to global memory for a
// merge kernel (in a persistent grid the CTA running a cut stream's first
// split also writes the stream's merge descriptor), or (p.cluster > 1) the
// splits of one row
// block and head run as one thread-block cluster and merge through
// distributed shared memory: each rank owns a share of the 32-column chunks
// of O, receives the other ranks' (m, l) rows and their rows of its chunks in
// its drained K ring, and writes those columns of the output.
// TMEM columns: S/P double buffer [0,128) [128,256), O [256, 256+D), Q
// double buffer [384, 384 + D/2) [448, 448 + D/2) (item n's Q in buffer
// n & 1, written one item ahead).  Shared memory holds only the two rings (Q and P live in
// tensor memory, so no product re-reads an operand from shared memory every
// tile), which leaves room for kStages tiles of K and of V in flight.
#pragma once

#include "attention.cuh"
#include "tcgen05.cuh"

namespace dipsd {

constexpr int kTcThreads = 192;
constexpr int kTcTile = 128;               // keys per tile (8 pages)
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units
constexpr uint32_t kQCols = 64;            // TMEM columns of one Q buffer (D / 2 bf16 pairs at most)

template <int D>
struct TcSmem {
  static constexpr int kHalves = D / 64;
  static constexpr int kStages = D == 128 ? 3 : 7;
  static constexpr int kPageBytes = kHalves * kPage * 128;           // V: [half][16 rows][128 B]
  static constexpr int kTileBytes = (kTcTile / kPage) * kPageBytes;  // 128 keys x D bf16 (K or V)
  static constexpr int kKOff = 0;
  static constexpr int kVOff = kKOff + kStages * kTileBytes;
  static constexpr int kBarOff = kVOff + kStages * kTileBytes;
  static constexpr int kBytes = kBarOff + 1024;  // barriers (6 kStages + 8) and the TMEM slot
  static constexpr int kAlloc = kBytes + 1024;  // slack for 1024-byte alignment
  // cluster merge: rank r finalises the 32-column chunks cc with cc % C == r;
  // every other rank's (m, l) rows and its O rows of those chunks land in one
  // slot of r's drained K ring, up to kMaxCluster - 1 slots
  static constexpr int kChunks = D / 32;
  static constexpr int kMaxCluster = D == 128 ? 3 : 6;
  static constexpr int kChunkBytes = 128 * 32 * 4;
  static constexpr int kSlotBytes = 128 * 8 + ((kChunks + 1) / 2) * kChunkBytes;
};
static_assert((TcSmem<128>::kMaxCluster - 1) * TcSmem<128>::kSlotBytes <= TcSmem<128>::kVOff, "exchange fits");
static_assert((TcSmem<64>::kMaxCluster - 1) * TcSmem<64>::kSlotBytes <= TcSmem<64>::kVOff, "exchange fits");
static_assert(TcSmem<128>::kAlloc <= 232448 && TcSmem<64>::kAlloc <= 232448, "shared memory per CTA");

// tm_k: 4-D {64 columns, 16 rows, heads, blocks}, one 64-column half of a
// page per box; tm_v: 5-D {64 columns, 16 rows, halves, heads, blocks}, a
// whole page per box.
// PERSIST: every CTA walks the pieces of its chunk of the page streams;
// otherwise every CTA runs exactly one item (the single-pass code).
template <int D, int CAP, bool PERSIST>
__global__ void __launch_bounds__(kTcThreads, 1)
verify_attention_tc_kernel(const __grid_constant__ AttnParams<CAP> p, const __grid_constant__ CUtensorMap tm_k,
                           const __grid_constant__ CUtensorMap tm_v) {
  using L = TcSmem<D>;
  constexpr int kHalves = L::kHalves;
  constexpr int S = L::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = smem + L::kKOff;
  uint8_t* sV = smem + L::kVOff;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  uint64_t* k_full = bars;             // [S]
  uint64_t* k_empty = bars + S;        // [S]
  uint64_t* v_full = bars + 2 * S;     // [S]
  uint64_t* v_empty = bars + 3 * S;    // [S]
  uint64_t* s_full = bars + 4 * S;     // [2]
  uint64_t* p_full = s_full + 2;       // [2]
  uint64_t* pv_done = p_full + 2;      // [2]
  uint64_t* o_final = pv_done + 2;
  uint64_t* q_ready = o_final + 1;   // [2]: one per Q buffer
  uint64_t* k_patch = q_ready + 2;   // [S] (each used at most once: new rows span <= 2 tiles)
  uint64_t* v_patch = k_patch + S;   // [S]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(v_patch + S);

  // ---- work: item blockIdx.x (one per CTA), or (PERSIST) the pieces of the
  // page streams in this CTA's chunk [chunk_lo, chunk_hi), in order.  Every
  // role walks the same pieces in the same order; ring slots and barrier
  // phases run on across them (global tile index g0 + j).
  const int chunk_lo = PERSIST ? p.chunk_bound[blockIdx.x] : static_cast<int>(blockIdx.x);
  const int chunk_hi = PERSIST ? p.chunk_bound[blockIdx.x + 1] : 0;
  // (pieces after a CTA's first follow from the one before: the next stream)
  int ui, split, nsplit, h, rb, M, row0, kv_begin, kv_end, ntiles, split_pages_n, next_w;
  AttnUser U;
  Work unit = PERSIST ? first_piece<CAP>(p, blockIdx.x, chunk_hi) : work_of_item<CAP>(p, blockIdx.x);
  auto following = [&]() { return next_piece<CAP>(p, unit, blockIdx.x, chunk_hi); };
  auto set_item = [&](const Work& W) {
    unit = W;
    ui = W.ui;
    U = p.u[ui];
    split = W.split;
    nsplit = W.nsplit;
    h = W.h;
    rb = W.rb;
    M = p.G * U.T;
    row0 = rb * 128;
    kv_begin = W.kv_begin;
    kv_end = W.kv_end;
    next_w = W.next;
    ntiles = max(0, (kv_end - kv_begin + kTcTile - 1) / kTcTile);  // 0: an empty split
    // Splits start on a page.  A split's last tile holds only the pages up
    // to kv_end: only those are loaded, multiplied (Q K^T with N = 16 per
    // page, one P V step per page) and run through the softmax.
    split_pages_n = (kv_end + kPage - 1) / kPage - kv_begin / kPage;
  };
  // is there work after the current unit (the loop tests it before set_item)
  auto more = [&]() { return PERSIST && next_w < chunk_hi; };
  set_item(unit);
  auto tile_pages = [&](int j) { return min(kTcTile / kPage, split_pages_n - j * (kTcTile / kPage)); };
  // tile j holds new (appended) rows: keys [max(key0, C_i), min(key0 + 128, kv_end)).
  // The patch barriers are single-use: a launch that appends runs one item per CTA.
  auto patched = [&](int j) {
    const int key0 = kv_begin + j * kTcTile;
    return p.new_k != nullptr && max(key0, U.ctx) < min(key0 + kTcTile, kv_end);
  };

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], 4);
      mbar_init(&pv_done[b], 1);
    }
    mbar_init(o_final, 1);
    mbar_init(&q_ready[0], 4);
    mbar_init(&q_ready[1], 4);
    for (int s = 0; s < S; ++s) {
      mbar_init(&k_patch[s], 1);
      mbar_init(&v_patch[s], 1);
    }
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
  // Q of item n in buffer n & 1 (kQCols columns each)
  const uint32_t tS0 = tmem, tO = tmem + 2 * kTcTile, tQ = tmem + 384;
  float fin_m = -INFINITY, fin_l = 0.f;  // softmax threads: row state after the last tile
  bool fin_ok = false;
  if (!p.wait_at_end) pdl_wait_prior_grid();
  pdl_launch_dependents();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // Page ids come from the block table 32 at a time (one per lane, one
    // group of 8 tiles ahead) so no TMA waits on a dependent global load.
    constexpr int kPages = kTcTile / kPage;
    constexpr int kTilesPerGroup = 32 / kPages;
    constexpr int kKBoxes = kPages * kHalves;  // K boxes per tile; V: kPages
    // lane -> its box: K (page, half) for lanes < kKBoxes, V page for the next kPages
    const int kb = lane < kKBoxes ? lane : 0;
    const int vb = lane - kKBoxes;
    const int my_pg = lane < kKBoxes ? kb / kHalves : (vb & (kPages - 1));
    const int my_hf = kb % kHalves;
    int issued = 0;  // tiles issued over all items (the global tile index of the next)
    // every K/V page is read once per launch (per row block): evict first, so
    // the stream keeps the split partials and other reused lines in L2
    const uint64_t kv_pol = l2_evict_first_policy();
    bool alive = true;
    // block ids of page group `group` of the split [kv_begin, kv_end) of the
    // user whose block-table row is `row` (lane = page in the group)
    auto fetch_of = [&](int row, int kb, int ke, int group) {
      const int page = kb / kPage + group * 32 + lane;
      return page < (ke + kPage - 1) / kPage ? __ldg(p.block_table + static_cast<size_t>(row) * p.max_blocks + page)
                                             : p.num_blocks;  // past the split's end: never requested
    };
    int ahead = 0;  // the next unit's first page group, loaded one unit early
    for (int n = 0; alive && (n == 0 || more()); ++n) {
      if (n > 0) set_item(following());
      const int g0 = issued;
      const int* bt = p.block_table + static_cast<size_t>(U.bt_row) * p.max_blocks;
      auto fetch = [&](int group) { return fetch_of(U.bt_row, kv_begin, kv_end, group); };
      int cur = n == 0 ? fetch(0) : ahead;
      int nxt = fetch(1);
      if (more()) {
        // the next unit's first page group, so its first loads do not wait
        // on a dependent block-table read at the boundary
        const Work Wn = following();
        ahead = fetch_of(p.u[Wn.ui].bt_row, Wn.kv_begin, Wn.kv_end, 0);
        // and the Q rows of the next two units into L2: the softmax warps
        // read a unit's Q one unit ahead, and a read that went to DRAM would
        // queue behind this SM's K/V stream (~4 us) while they wait on it
        auto prefetch_q = [&](const Work& W) {
          const AttnUser& Un = p.u[W.ui];
          if (lane < Un.T)
            bulk_prefetch_l2(p.q + (static_cast<size_t>(Un.q_off + lane) * p.Hq + W.h * p.G) * D, p.G * D * 2);
        };
        prefetch_q(Wn);
        if (Wn.next < chunk_hi) prefetch_q(next_piece<CAP>(p, Wn, blockIdx.x, chunk_hi));
      }
      for (int j = 0; j < ntiles; ++j) {
        const int gj = g0 + j;
        const int st = gj % S;
        if (j % kTilesPerGroup == 0 && j > 0) {
          cur = nxt;
          nxt = fetch(j / kTilesPerGroup + 1);
        }
        const int bk = __shfl_sync(0xffffffffu, cur, (j % kTilesPerGroup) * kPages + my_pg);
        const uint32_t ph = ((gj / S) - 1) & 1;
        const uint32_t koff = st * L::kTileBytes + my_hf * (kTcTile * 128) + my_pg * (kPage * 128);
        const uint32_t voff = st * L::kTileBytes + my_pg * L::kPageBytes;
        const int tp = tile_pages(j);  // pages of this tile (kPages except in a split's last tile)
        // K tile
        bool go = true;
        if (gj >= S && lane == 0) go = mbar_wait(&k_empty[st], ph, p.status);
        if (!__shfl_sync(0xffffffffu, go, 0)) {
          alive = false;
          break;
        }
        if (lane == 0) mbar_arrive_expect_tx(&k_full[st], tp * L::kPageBytes);
        __syncwarp();
        if (lane < kKBoxes && my_pg < tp) tma_load_4d_hint(sK + koff, &tm_k, my_hf * 64, 0, h, bk, &k_full[st], kv_pol);
        // V tile
        if (gj >= S && lane == 0) go = mbar_wait(&v_empty[st], ph, p.status);
        if (!__shfl_sync(0xffffffffu, go, 0)) {
          alive = false;
          break;
        }
        if (lane == 0) mbar_arrive_expect_tx(&v_full[st], tp * L::kPageBytes);
        __syncwarp();
        if (lane >= kKBoxes && lane < kKBoxes + kPages && my_pg < tp)
          tma_load_5d_hint(sV + voff, &tm_v, 0, 0, 0, h, bk, &v_full[st], kv_pol);
        ++issued;
        if (patched(j)) {
          // the appended rows of this tile, straight from the input, over what
          // the pages held (generic writes, then a proxy fence for the MMA)
          const int key0 = kv_begin + j * kTcTile;
          const int lo = max(key0, U.ctx), hi = min(key0 + kTcTile, kv_end);
          const int n16 = (hi - lo) * (D / 8);
          go = true;
          if (lane == 0) go = mbar_wait(&k_full[st], (gj / S) & 1, p.status);
          if (!__shfl_sync(0xffffffffu, go, 0)) {
            alive = false;
            break;
          }
          for (int e = lane; e < n16; e += 32) {
            const int key = lo + e / (D / 8), c = e % (D / 8), r = key - key0;
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(
                p.new_k + (static_cast<size_t>(U.q_off + key - U.ctx) * p.Hkv + h) * D) + c);
            *reinterpret_cast<uint4*>(sK + st * L::kTileBytes + (c >> 3) * (kTcTile * 128) + r * 128 +
                                      (((c & 7) ^ (r & 7)) << 4)) = v;
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&k_patch[st]);
          if (lane == 0) go = mbar_wait(&v_full[st], (gj / S) & 1, p.status);
          if (!__shfl_sync(0xffffffffu, go, 0)) {
            alive = false;
            break;
          }
          for (int e = lane; e < n16; e += 32) {
            const int key = lo + e / (D / 8), c = e % (D / 8), r = key - key0;
            const int r16 = r % kPage;
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(
                p.new_v + (static_cast<size_t>(U.q_off + key - U.ctx) * p.Hkv + h) * D) + c);
            *reinterpret_cast<uint4*>(sV + st * L::kTileBytes + (r / kPage) * L::kPageBytes +
                                      (c >> 3) * (kPage * 128) + r16 * 128 + (((c & 7) ^ (r16 & 7)) << 4)) = v;
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&v_patch[st]);
        }
      }
      // state update: the last split of the first row block writes the user's
      // new rows of head h into the pages
      if (alive && p.new_k != nullptr && rb == 0 && split == nsplit - 1) {
        const int n16 = U.T * (D / 8);
        for (int e = lane; e < n16; e += 32) {
          const int tt = e / (D / 8), c = e % (D / 8);
          const int pos = U.ctx + tt;
          const int blk = __ldg(bt + pos / kPage);
          if (blk < 0 || blk >= p.num_blocks) {
            atomicOr(p.status, kDevErrBadBlock);
            continue;
          }
          const size_t dst = ((static_cast<size_t>(blk) * p.Hkv + h) * kPage + pos % kPage) * D;
          const size_t src = (static_cast<size_t>(U.q_off + tt) * p.Hkv + h) * D;
          reinterpret_cast<uint4*>(p.k_cache + dst)[c] = __ldg(reinterpret_cast<const uint4*>(p.new_k + src) + c);
          reinterpret_cast<uint4*>(p.v_cache + dst)[c] = __ldg(reinterpret_cast<const uint4*>(p.new_v + src) + c);
        }
      }
    }
    // copies still in flight must land before the CTA can exit
    if (lane == 0)
      for (int j = max(0, issued - S); j < issued; ++j) {
        mbar_wait(&k_full[j % S], (j / S) & 1, p.status);
        mbar_wait(&v_full[j % S], (j / S) & 1, p.status);
      }
  } else if (warp == 1) {
    // ----------------------------------------------------- MMA issuer (1 thread)
    if (lane == 0) {
      constexpr uint32_t kIdQK = idesc_bf16_f32(128, kTcTile, false, false);
      constexpr uint32_t kIdPV = idesc_bf16_f32(128, D, false, true);
      const uint32_t k_addr = smem_addr(sK);
      const uint32_t v_addr = smem_addr(sV);
      bool ok = true;
      int g0 = 0;  // global index of the item's first tile
      for (int n = 0; ok && (n == 0 || more()); ++n) {
        if (n > 0) set_item(following());
        // Q of this unit is in TMEM buffer n & 1 (written one unit ahead)
        ok = mbar_wait(&q_ready[n & 1], (n >> 1) & 1, p.status);
        const uint32_t tQn = tQ + (n & 1) * kQCols;
        int jq = 0, jp = 0;  // next Q K^T, next P V (within the item)
        uint64_t idle_since = 0;
        uint32_t idle_polls = 0;
        while (ok && jp < ntiles) {
          bool did = false;
          const int gq = g0 + jq, gp = g0 + jp;
          // S[gq & 1] is free once P V of tile gq - 2 has been issued (the
          // tensor core runs one thread's MMAs in issue order)
          if (jq < ntiles && jp >= jq - 1 &&
              (patched(jq) ? mbar_test_wait(&k_patch[gq % S], 0) : mbar_test_wait(&k_full[gq % S], (gq / S) & 1))) {
            tc_fence_after();
            const uint32_t kt = k_addr + (gq % S) * L::kTileBytes;
            // N = 16 keys per loaded page
            const uint32_t id_qk = jq + 1 < ntiles ? kIdQK : idesc_bf16_f32(128, tile_pages(jq) * kPage, false, false);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint64_t bd = smem_desc_sw128(kt + (kk >> 2) * (kTcTile * 128) + (kk & 3) * 32, 0, 1024);
              tc_mma_ts(tS0 + (gq & 1) * kTcTile, tQn + kk * 8, bd, id_qk, kk > 0 ? 1u : 0u);
            }
            tc_commit(&s_full[gq & 1]);
            tc_commit(&k_empty[gq % S]);
            ++jq;
            did = true;
          }
          if (jp < jq && mbar_test_wait(&p_full[gp & 1], (gp >> 1) & 1) &&
              (patched(jp) ? mbar_test_wait(&v_patch[gp % S], 0) : mbar_test_wait(&v_full[gp % S], (gp / S) & 1))) {
            tc_fence_after();
            const uint32_t vt = v_addr + (gp % S) * L::kTileBytes;
            const uint32_t pt = tS0 + (gp & 1) * kTcTile;  // P: 64 columns of bf16 pairs
            const int np = tile_pages(jp);
#pragma unroll
            for (int kk = 0; kk < kTcTile / kPage; ++kk) {
              if (kk >= np) break;
              // MN-major V page: 64-column halves kPage * 128 bytes apart
              // (leading offset), 8-key groups 1024 bytes apart (stride offset);
              // the item's first product overwrites O
              const uint64_t bd = smem_desc_sw128(vt + kk * L::kPageBytes, kPage * 128, 1024);
              tc_mma_ts(tO, pt + kk * 8, bd, kIdPV, (jp > 0 || kk > 0) ? 1u : 0u);
            }
            tc_commit(&pv_done[gp & 1]);
            tc_commit(&v_empty[gp % S]);
            ++jp;
            did = true;
          }
          // the wait stays bounded, but the timer is read once per 256 idle
          // polls: a %globaltimer read costs far more than a test_wait
          if (did) {
            idle_polls = 0;
            idle_since = 0;
          } else if ((++idle_polls & 255u) == 0) {
            const uint64_t now = global_timer_ns();
            if (idle_since == 0) {
              idle_since = now;
            } else if (now - idle_since > kWaitLimitNs) {
              atomicOr(p.status, kDevErrWaitTimeout);
              ok = false;
            }
          }
        }
        tc_commit(o_final);
        g0 += ntiles;
      }
    }
  } else {
    // ----------------------------------------- softmax / epilogue (row per thread)
    const int quad = warp & 3;
    const int r = quad * 32 + lane;  // row within the block == TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    bool ok = true;
    int g0 = 0;  // global index of the item's first tile
    // Q row of the unit starting at w -> TMEM buffer qb, lane r, as bf16
    // pairs (column c holds elements 2c, 2c+1); padding rows are zero
    auto write_q = [&](const Work& Wj, int qb) {
      const AttnUser Uj = p.u[Wj.ui];
      const int hj = Wj.h, rgj = Wj.rb * 128 + r;
      const bool validj = rgj < p.G * Uj.T;
      tc_fence_after();
      const uint4* qrow = reinterpret_cast<const uint4*>(
          p.q + (static_cast<size_t>(Uj.q_off + rgj / p.G) * p.Hq + hj * p.G + rgj % p.G) * D);
#pragma unroll
      for (int cc = 0; cc < D / 64; ++cc) {
        uint32_t w[32];
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          uint4 v = make_uint4(0, 0, 0, 0);
          if (validj) v = __ldg(qrow + cc * 8 + c);
          w[4 * c] = v.x;
          w[4 * c + 1] = v.y;
          w[4 * c + 2] = v.z;
          w[4 * c + 3] = v.w;
        }
        tmem_st32(tQ + qb * kQCols + cc * 32 + lane_base, w);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&q_ready[qb]);
    };
    for (int n = 0; ok && (n == 0 || more()); ++n) {
      if (n > 0) set_item(following());
      const int rg = row0 + r;  // row within the user
      const bool valid = rg < M;
      const int t = rg / p.G, g = rg % p.G;

      // Q is written one item ahead, so the next item's Q K^T products can
      // run while this item's last tiles and epilogue finish: item n + 1's Q
      // goes to buffer (n + 1) & 1 once this item's first tile is softmaxed
      // (off the path from this item's start to its first P V); the buffer's
      // previous user, item n - 1, has its products done: its o_final was
      // waited for.
      if (n == 0) write_q(unit, 0);
      const bool prefetch = more();
      const Work w_next = prefetch ? following() : unit;
      if (prefetch && ntiles == 0) write_q(w_next, (n + 1) & 1);

      const int last_vis = min(U.ctx + t, kv_end - 1);  // last key of this row in this split
      // warps whose 32 rows are all padding write zero P, so every lane of P
      // the tensor core reads is defined
      const bool active = row0 + quad * 32 < M;
      const float sl2 = p.scale_log2;
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < ntiles; ++j) {
        const int gj = g0 + j;
        const int b = gj & 1, st = gj % S;
        const int key0 = kv_begin + j * kTcTile;
        ok = __all_sync(0xffffffffu, mbar_wait(&s_full[b], (gj >> 1) & 1, p.status));
        if (!ok) break;
        tc_fence_after();
        const uint32_t tSb = tS0 + b * kTcTile + lane_base;
        if (active) {
          // two passes over the tile's loaded columns in 32-column chunks (a
          // small loop body: this code runs once per tile and per CTA, so its
          // instruction fetch counts); the second pass overwrites S with P as it
          // goes (P pairs of keys 32c..32c+31 land in columns 16c..16c+15, which
          // this thread has already read)
          const int nch = (tile_pages(j) * kPage + 31) / 32;
          float mr = -INFINITY;
#pragma unroll 1
          for (int ch = 0; ch < nch; ++ch) {
            uint32_t sr[32];
            tmem_ld32(tSb + ch * 32, sr);
            // raw scores; the causal rule key <= C_i + t only bites near the end
            // (columns past the tile's pages are keys past kv_end: masked too)
            const int kb = key0 + ch * 32;
            const bool need_mask = kb + 31 > last_vis;
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float v = __uint_as_float(sr[c]);
              mr = fmaxf(mr, need_mask && kb + c > last_vis ? -INFINITY : v);
            }
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
            // every earlier P V has to be done before O is touched
            ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[(gj - 1) & 1], ((gj - 1) >> 1) & 1, p.status));
            if (!ok) break;
            tc_fence_after();
#pragma unroll 1
            for (int cc = 0; cc < D / 32; ++cc) {
              uint32_t o[32];
              tmem_ld32(tO + cc * 32 + lane_base, o);
#pragma unroll
              for (int k = 0; k < 32; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * factor);
              tmem_st32(tO + cc * 32 + lane_base, o);
            }
          }
          l *= factor;
          const float nb = m == -INFINITY ? 0.f : -m;
#pragma unroll 1
          for (int ch = 0; ch < nch; ++ch) {
            uint32_t sr[32];
            tmem_ld32(tSb + ch * 32, sr);
            const int kb = key0 + ch * 32;
            const bool need_mask = kb + 31 > last_vis;
            uint32_t pk[16];
#pragma unroll
            for (int c = 0; c < 32; c += 2) {
              const float s0 = need_mask && kb + c > last_vis ? -INFINITY : __uint_as_float(sr[c]);
              const float s1 = need_mask && kb + c + 1 > last_vis ? -INFINITY : __uint_as_float(sr[c + 1]);
              const float p0 = fast_exp2(__fmaf_rn(s0, sl2, nb));
              const float p1 = fast_exp2(__fmaf_rn(s1, sl2, nb));
              l += p0 + p1;
              pk[c >> 1] = pack_bf16x2(p0, p1);
            }
            tmem_st16(tSb + ch * 16, pk);
          }
        } else {
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) pk[c] = 0u;
#pragma unroll
          for (int hh = 0; hh < kTcTile / 64; ++hh) tmem_st32(tSb + hh * 32, pk);
        }
        // V rows past kv_len may hold anything; zero them before P V reads them
        if (key0 + kTcTile > U.kv_len) {
          ok = __all_sync(0xffffffffu, mbar_wait(&v_full[st], (gj / S) & 1, p.status));
          if (!ok) break;
          uint8_t* vt = sV + st * L::kTileBytes;
          const int first = U.kv_len - key0;  // first key row to clear, up to the tile's loaded pages
          const int nchunks = max(0, tile_pages(j) * kPage - first) * kHalves * 8;
          for (int c = threadIdx.x - 64; c < nchunks; c += 128) {
            const int row = first + c / (kHalves * 8);
            const int rem = c % (kHalves * 8);  // every 16-byte chunk of the row, in any order
            *reinterpret_cast<uint4*>(vt + (row / kPage) * L::kPageBytes + (rem >> 3) * (kPage * 128) +
                                      (row % kPage) * 128 + ((rem & 7) << 4)) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[b]);
        if (prefetch && j == 0) write_q(w_next, (n + 1) & 1);
      }

      // ---- epilogue: O row from TMEM
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_final, n & 1, p.status));
      fin_m = m;
      fin_l = l;
      fin_ok = ok;
      if (ok && active && p.cluster <= 1) {
        tc_fence_after();
        const float inv = l > 0.f ? 1.f / l : 0.f;
        __nv_bfloat16* orow = p.out + (static_cast<size_t>(U.q_off + t) * p.Hq + h * p.G + g) * D;
        const long long prow_idx = p.part_off[ui] + static_cast<long long>(split * p.Hkv + h) * M + rg;
#pragma unroll
        for (int cc = 0; cc < D / 32; ++cc) {
          uint32_t o[32];
          tmem_ld32(tO + cc * 32 + lane_base, o);
          if (!valid) continue;
          if (nsplit == 1) {
            uint4* dst = reinterpret_cast<uint4*>(orow + cc * 32);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              auto on = [&](int i) { return __uint_as_float(o[8 * k + i]) * inv; };
              dst[k] = make_uint4(pack_bf16x2(on(0), on(1)), pack_bf16x2(on(2), on(3)), pack_bf16x2(on(4), on(5)),
                                  pack_bf16x2(on(6), on(7)));
            }
          } else {
            float4* dst = reinterpret_cast<float4*>(p.part_o + prow_idx * D + cc * 32);
#pragma unroll
            for (int k = 0; k < 8; ++k)
              dst[k] = make_float4(__uint_as_float(o[4 * k]), __uint_as_float(o[4 * k + 1]),
                                   __uint_as_float(o[4 * k + 2]), __uint_as_float(o[4 * k + 3]));
          }
        }
        if (valid && nsplit > 1) p.part_ml[prow_idx] = make_float2(m, l);
      }
      if constexpr (PERSIST) {
        // the first split of a cut stream leaves the stream's merge descriptor
        // (chunk_cut: 255 = no cut stream starts in this chunk; the host
        // marks exactly the streams this test finds)
        if (nsplit > 1 && split == 0 && threadIdx.x == 64 && p.chunk_cut[blockIdx.x] != 255) {
          MergeDesc dsc;
          dsc.part_row0 = p.part_off[ui] + static_cast<long long>(h) * M + row0;
          dsc.out_base = static_cast<long long>(U.q_off) * p.Hq + h * p.G;
          dsc.step = p.Hkv * M;
          dsc.nsplit = nsplit;
          dsc.nrows = min(128, M - row0);
          dsc.row0 = row0;
          p.merge_desc[p.chunk_cut[blockIdx.x]] = dsc;
        }
      }
      tc_fence_before();
      g0 += ntiles;
    }
  }

  if (p.cluster > 1) {
    // ---- split merge inside the cluster (every thread takes both barriers).
    // Rank r finalises the 32-column chunks cc with cc % C == r.  Every rank
    // pushes its (m, l) rows to all others and each chunk it does not own to
    // the owner; the owner weighs the C partial rows by 2^(m_s - max m) and
    // writes its columns of the output.
    constexpr int kSlot = L::kSlotBytes;  // (m, l) per row, then the owner's chunks as [8][128] float4
    constexpr int kCh = L::kChunks;
    const int C = p.cluster;
    const int crank = static_cast<int>(cluster_ctarank());
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const int rg = row0 + r;
    const bool valid = rg < M;
    const bool active = warp >= 2 && row0 + quad * 32 < M;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    uint8_t* xbuf = sK;  // every rank's K ring, drained once all ranks are here
    // slot of source rank `src` at receiving rank `dst`
    auto slot_of = [&](int src, int dst) { return (src < dst ? src : src - 1) * kSlot; };
    cluster_arrive_release();
    cluster_wait_acquire();
    if (active && fin_ok) {
      for (int dst = 0; dst < C; ++dst)
        if (dst != crank && valid) dsmem_st_f32x2(dsmem_map(xbuf + slot_of(crank, dst), dst) + r * 8, fin_m, fin_l);
      tc_fence_after();
#pragma unroll 1
      for (int cc = 0; cc < kCh; ++cc) {
        const int dst = cc % C;
        if (dst == crank) continue;
        uint32_t o[32];
        tmem_ld32(tO + cc * 32 + lane_base, o);
        if (valid && fin_l > 0.f) {
          const uint32_t base = dsmem_map(xbuf + slot_of(crank, dst), dst) + 1024 + (cc / C) * L::kChunkBytes;
#pragma unroll
          for (int k = 0; k < 8; ++k)
            dsmem_st_f32x4(base + (k * 128 + r) * 16, __uint_as_float(o[4 * k]), __uint_as_float(o[4 * k + 1]),
                           __uint_as_float(o[4 * k + 2]), __uint_as_float(o[4 * k + 3]));
        }
      }
    }
    cluster_arrive_release();
    cluster_wait_acquire();
    if (active && fin_ok && crank < kCh) {
      const int t = rg / p.G, g = rg % p.G;
      float mx = fin_m;
      for (int s = 0; s < C; ++s)
        if (s != crank) mx = fmaxf(mx, reinterpret_cast<const float2*>(xbuf + slot_of(s, crank))[r].x);
      // weights 2^(m_s - mx) (log2 units); an empty split weighs 0
      const float w0 = fin_m == -INFINITY ? 0.f : fast_exp2(fin_m - mx);
      float l = w0 * fin_l;
      for (int s = 0; s < C; ++s) {
        if (s == crank) continue;
        const float2 ml = reinterpret_cast<const float2*>(xbuf + slot_of(s, crank))[r];
        l += ml.x == -INFINITY ? 0.f : fast_exp2(ml.x - mx) * ml.y;
      }
      const float inv = l > 0.f ? 1.f / l : 0.f;
      __nv_bfloat16* orow = p.out + (static_cast<size_t>(U.q_off + t) * p.Hq + h * p.G + g) * D;
      tc_fence_after();
#pragma unroll 1
      for (int cc = crank; cc < kCh; cc += C) {
        uint32_t o[32];
        tmem_ld32(tO + cc * 32 + lane_base, o);
        float acc[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) acc[k] = w0 > 0.f ? w0 * __uint_as_float(o[k]) : 0.f;
        for (int s = 0; s < C; ++s) {
          if (s == crank) continue;
          const float2 ml = reinterpret_cast<const float2*>(xbuf + slot_of(s, crank))[r];
          if (!(ml.x > -INFINITY) || !(ml.y > 0.f)) continue;
          const float w = fast_exp2(ml.x - mx);
          const float4* os =
              reinterpret_cast<const float4*>(xbuf + slot_of(s, crank) + 1024 + (cc / C) * L::kChunkBytes);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float4 v = os[k * 128 + r];
            acc[4 * k] += w * v.x;
            acc[4 * k + 1] += w * v.y;
            acc[4 * k + 2] += w * v.z;
            acc[4 * k + 3] += w * v.w;
          }
        }
        if (valid) {
          uint4* dst = reinterpret_cast<uint4*>(orow + cc * 32);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            dst[k] = make_uint4(pack_bf16x2(acc[8 * k] * inv, acc[8 * k + 1] * inv),
                                pack_bf16x2(acc[8 * k + 2] * inv, acc[8 * k + 3] * inv),
                                pack_bf16x2(acc[8 * k + 4] * inv, acc[8 * k + 5] * inv),
                                pack_bf16x2(acc[8 * k + 6] * inv, acc[8 * k + 7] * inv));
        }
      }
    }
    tc_fence_before();
  }

  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (p.wait_at_end && threadIdx.x == 0) pdl_wait_prior_grid();
}

}  // namespace dipsd
