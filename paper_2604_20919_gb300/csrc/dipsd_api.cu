// Host side of the C ABI declared in include/dipsd.h: argument validation,
// work planning (KV split sizes, cluster sizes, workspace layout), TMA tensor
// map encoding and kernel launches.  No entry point allocates or synchronises.
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "dipsd.h"
#include "attention.cuh"
#include "attention_tc.cuh"
#include "philox.cuh"
#include "spec_generic.cuh"
#include "spec_verify.cuh"

namespace dipsd {
namespace {

constexpr size_t kStatusBytes = 256;
// Arrival counters of the spec register path, at a fixed place right after
// the status word whatever the entry point, so that every call finds them as
// the last call left them (all zero).
constexpr size_t kCounterBytes = (kCounterWords * sizeof(unsigned) + 255) / 256 * 256;
constexpr size_t kHeaderBytes = kStatusBytes + kCounterBytes;
constexpr int kCapSmall = 64;
constexpr int kCapLarge = kMaxUsers;
// kernel parameters are limited to 32764 bytes (the attention grid also
// takes its two tensor maps)
static_assert(sizeof(AttnParams<kCapLarge>) + 2 * sizeof(CUtensorMap) <= 32764, "attention parameters");

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Plan overrides set through dipsd_test_set_override (0 = the planner's own
// choice); indexed by the DIPSD_TEST_* codes of dipsd.h.
constexpr int kNumOverrides = 9;
std::atomic<int> g_override[kNumOverrides];
int plan_override(int which) { return g_override[which].load(std::memory_order_relaxed); }
bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// ------------------------------------------------------------ device facts
struct DeviceFacts {
  int sms = 0;
  int max_smem_optin = 0;
};

bool device_facts(DeviceFacts& f) {
  static std::mutex mu;
  static DeviceFacts cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev].sms == 0) {
    if (cudaDeviceGetAttribute(&cache[dev].sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return false;
    cudaDeviceGetAttribute(&cache[dev].max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  }
  f = cache[dev];
  return f.sms > 0;
}

// ------------------------------------------------------ TMA tensor maps
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Paged cache [num_blocks][Hkv][16][D] bf16 as tensor maps with the 128-byte
// swizzle.  K (4-D: D columns, 16 rows, heads, blocks): one box = one
// 64-column half of one page of one head.  V (5-D: 64 columns, 16 rows of
// 2*D bytes, D/64 halves 128 bytes apart, heads, blocks): one box = a whole
// page of one head, stored half after half.
bool encode_cache_map(CUtensorMap* map, const void* base, int num_blocks, int Hkv, int D, bool whole_page) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t row = static_cast<cuuint64_t>(D) * 2;
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  if (!whole_page) {
    cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)kPage, (cuuint64_t)Hkv, (cuuint64_t)num_blocks};
    cuuint64_t strides[3] = {row, kPage * row, (cuuint64_t)Hkv * kPage * row};
    cuuint32_t box[4] = {64, (cuuint32_t)kPage, 1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }
  cuuint64_t dims[5] = {64, (cuuint64_t)kPage, (cuuint64_t)(D / 64), (cuuint64_t)Hkv, (cuuint64_t)num_blocks};
  cuuint64_t strides[4] = {row, 128, kPage * row, (cuuint64_t)Hkv * kPage * row};
  cuuint32_t box[5] = {64, (cuuint32_t)kPage, (cuuint32_t)(D / 64), 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// --------------------------------------------------------------- launching
thread_local long long g_launches = 0;

template <typename... KArgs, typename... Args>
cudaError_t launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                   int cluster, bool pdl, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (cluster > 0) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
  if (e == cudaSuccess) ++g_launches;
  return e;
}

// Raises a kernel's dynamic shared memory limit once per device.
template <typename K>
bool allow_smem(K kernel, int bytes, bool* done) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (done[dev]) return true;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
    return false;
  done[dev] = true;
  return true;
}

// =================================================================== attention
struct AttnPlan {
  int B = 0, Hq = 0, Hkv = 0, G = 0, D = 0;
  int n_items = 0, n_merge = 0;
  int n_chunks = 0, total_pages = 0;  // page streams (persistent grid): chunks, all pages
  std::vector<int> chunk_bound;        // chunk b: pages [chunk_bound[b], chunk_bound[b + 1])
  // per chunk: the user of its first page; chunks back to where the stream of
  // its first page starts; chunks ahead to where the stream of its last ends
  std::vector<short> chunk_user;
  std::vector<unsigned char> chunk_c0_back, chunk_c1_fwd;
  // page streams cut by chunk bounds (merged after the grid): per chunk the
  // index of the cut stream that starts in it (255: none), and their count
  std::vector<unsigned char> chunk_cut;
  int n_cut = 0;
  int grid = 0;     // CTAs launched: n_items, or fewer that each walk several items
  int cluster = 0;  // > 1: splits merged inside a thread-block cluster of this size
  long long part_rows = 0;
  std::vector<AttnUser> u;
  std::vector<int> item_off, merge_off, page_off;
  std::vector<long long> part_off;
  size_t ws_bytes = 0;  // attention region only (excludes the status word)
};


// Validates the per-user attention arguments.
int check_attn_users(int B, const int* L, const int* ctx, int Hq, int Hkv, int D) {
  if (B < 1 || B > kMaxUsers || !L || !ctx) return DIPSD_ERR_INVALID_ARG;
  if (Hkv < 1 || Hq < Hkv || Hq % Hkv != 0 || Hq > 4096) return DIPSD_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return D > 0 ? DIPSD_ERR_UNSUPPORTED : DIPSD_ERR_INVALID_ARG;
  long long sum_t = 0;
  for (int i = 0; i < B; ++i) {
    if (L[i] < 0 || L[i] > kMaxDraft || ctx[i] < 0) return DIPSD_ERR_INVALID_ARG;
    if (static_cast<long long>(ctx[i]) + L[i] + 1 > (1ll << 30)) return DIPSD_ERR_INVALID_ARG;
    sum_t += L[i] + 1;
  }
  if (sum_t * Hq * D > (1ll << 40)) return DIPSD_ERR_INVALID_ARG;
  return DIPSD_OK;
}

// Chooses how many KV splits each user gets, minimising a list-scheduling
// estimate of the makespan over the resident CTA slots: total work / slots +
// the largest item, with a per-item overhead (prologue, pipeline fill,
// epilogue) and the merge traffic.  A user's splits are as even as whole
// 16-token pages allow (the kernel masks a split's last tile at its end).
// Costs are in units of 64 tokens of one (user, head) stream.
// Pages per split when `pages` pages are cut into `ns` near-equal splits.
static int split_pages(int pages, int ns) { return (pages + ns - 1) / ns; }

// Chunks of the page streams (stream k holds np[k] pages; the streams back to
// back) for at most `grid` CTAs, cut so that every CTA carries about the same
// cost: a page costs 1, each piece (a stream or the part of one a chunk
// holds) kPiecePages more.  A stream that would start with less than a piece's
// cost of room left goes whole to the next chunk.  Cut points come from the
// smallest per-chunk cost that needs at most `grid` chunks (bisection).
constexpr long long kPiecePages = 18;  // ~3.5 us per piece at ~0.2 us per page
static std::vector<int> cut_chunks(const std::vector<int>& np, int grid) {
  auto cut = [&](long long cap, std::vector<int>* out) {
    long long acc = 0, pos = 0;
    int n = 1;
    if (out) out->assign(1, 0);
    for (int pages : np) {
      if (acc > 0 && acc + kPiecePages >= cap) {  // start this stream in a new chunk
        ++n;
        if (out) out->push_back(static_cast<int>(pos));
        acc = 0;
      }
      acc += kPiecePages;
      long long rem = pages;
      for (;;) {
        const long long room = std::max<long long>(1, cap - acc);
        if (rem <= room) {
          acc += rem;
          pos += rem;
          break;
        }
        pos += room;
        rem -= room;
        ++n;
        if (out) out->push_back(static_cast<int>(pos));
        acc = kPiecePages;  // the rest of the stream: a new piece in the next chunk
      }
    }
    if (out) out->push_back(static_cast<int>(pos));
    return n;
  };
  long long total = 0;
  for (int pages : np) total += pages + kPiecePages;
  // Every chunk carries at most `cap`, so the smallest feasible cap is at
  // least total / grid; every chunk but the last carries at least cap minus
  // one piece's charge of the streams' own cost, and each cut adds one piece
  // charge, so total / grid + 2 kPiecePages is feasible.  Search that narrow
  // range first; the whole range only if it fails.
  long long lo = std::max<long long>(1, total / std::max(1, grid));
  long long hi = lo + 4 * kPiecePages + 64;
  if (cut(hi, nullptr) > grid) {
    lo = hi + 1;
    hi = total + kPiecePages;  // cut(hi) gives one chunk
  }
  while (lo < hi) {
    const long long mid = (lo + hi) / 2;
    if (cut(mid, nullptr) <= grid) hi = mid; else lo = mid + 1;
  }
  std::vector<int> bounds;
  cut(lo, &bounds);
  return bounds;
}

void plan_attention(int B, const int* L, const int* ctx, const int* bt_rows, int Hq, int Hkv, int D,
                    int sms, AttnPlan& pl, bool persist_ok = true) {
  pl.B = B; pl.Hq = Hq; pl.Hkv = Hkv; pl.G = Hq / Hkv; pl.D = D;
  // tcgen05 kernel: 128 rows per CTA, one CTA per SM (its shared memory and
  // all of tensor memory)
  const int rows_cta = 128;
  const int slots = sms;

  const int forced = plan_override(DIPSD_TEST_ATTN_SPLIT_TILES);
  const int forced_cluster = plan_override(DIPSD_TEST_ATTN_CLUSTER);
  const int cands[] = {1, 2, 3, 4, 5, 6, 8, 10, 12, 16, 20, 24, 32, 40, 48, 64, 96, 128, 192, 256, 384, 512, 1 << 30};
  // Costs in tile units: an item pays its tiles plus ~2 of prologue and
  // epilogue; splits merged by the separate merge kernel pay ~3 more (its
  // launch behind the attention grid), splits merged in a cluster ~0.5.
  double best = 1e300;
  int best_c = 1 << 30;
  for (int c : cands) {
    if (forced > 0) c = forced;
    double total = 0, max_item = 0;
    long long items = 0;
    bool any_split = false;
    for (int i = 0; i < B; ++i) {
      const int tiles = (ctx[i] + L[i] + 1 + kTcTile - 1) / kTcTile;
      const int pages = (ctx[i] + L[i] + 1 + kPage - 1) / kPage;
      const int cc = std::max(1, std::min(c, tiles));
      int ns = (tiles + cc - 1) / cc;
      const int sp = split_pages(pages, ns);
      ns = (pages + sp - 1) / sp;
      const int rb = (pl.G * (L[i] + 1) + rows_cta - 1) / rows_cta;
      const double item = sp * kPage / 64.0 + 2.0 + (ns > 1 ? 0.5 : 0.0);
      total += item * ns * rb * Hkv;
      items += static_cast<long long>(ns) * rb * Hkv;
      max_item = std::max(max_item, item);
      any_split = any_split || ns > 1;
    }
    if (items > (1ll << 30)) continue;
    // items are near-uniform (one split length): waves x longest item, but
    // never better than perfect balance plus one item
    const double waves = std::ceil(static_cast<double>(items) / slots);
    const double cost = std::max(waves * max_item, total / slots + 0.5 * max_item) + (any_split ? 3.0 : 0.0);
    if (cost < best - 1e-9) { best = cost; best_c = c; }
    if (forced > 0) break;
  }

  // Cluster merge: every user's KV in the same number C of splits (one wave,
  // the exchange buffer of C - 1 ranks fitting rank 0's rings).
  const int max_cluster = D == 128 ? TcSmem<128>::kMaxCluster : TcSmem<64>::kMaxCluster;
  int best_cl = 0;
  double best_b = 1e300;
  for (int C = 2; C <= max_cluster && forced == 0; ++C) {
    if (forced_cluster > 0) C = std::min(forced_cluster, max_cluster);
    long long items = 0;
    double max_item = 0;
    for (int i = 0; i < B; ++i) {
      const int pages = (ctx[i] + L[i] + 1 + kPage - 1) / kPage;
      const int rb = (pl.G * (L[i] + 1) + rows_cta - 1) / rows_cta;
      items += static_cast<long long>(C) * rb * Hkv;
      max_item = std::max(max_item, split_pages(pages, C) * kPage / 64.0 + 2.5);
    }
    if (items <= slots || forced_cluster > 0) {
      if (max_item < best_b) { best_b = max_item; best_cl = C; }
    }
    if (forced_cluster > 0) break;
  }
  pl.cluster = (forced_cluster > 0 || best_b < best) && best_cl > 1 ? best_cl : 0;

  // Persistent grid over page streams: the pages of every (user, row block,
  // KV head) as one stream, the streams back to back, cut into equal chunks
  // of pages, one chunk per CTA (one CTA per SM).  Taken whenever one CTA per
  // item would need more than one wave of CTAs (each wave pays its own ramp
  // and drain, and the cost model above undercounts them: measured on the
  // ragged 32-user batch, 87 us over six waves against 76 us for the same
  // work as a persistent grid), or when a test forces it.  Not with the KV
  // append (single-use patch barriers) nor the cluster merge.
  int persist_mode = -1;  // -1: by cost, 0: never, 1: whenever allowed
  int grid_cap = slots;
  if (const int v = plan_override(DIPSD_TEST_ATTN_PERSIST)) persist_mode = v == 1 ? 1 : 0;
  if (const int v = plan_override(DIPSD_TEST_ATTN_GRID)) grid_cap = std::max(1, std::min(slots, v));
  long long total_pages = 0;
  for (int i = 0; i < B; ++i) {
    const int rb = (pl.G * (L[i] + 1) + rows_cta - 1) / rows_cta;
    total_pages += static_cast<long long>(rb) * Hkv * ((ctx[i] + L[i] + 1 + kPage - 1) / kPage);
  }
  // items of the best one-item-per-CTA plan
  long long best_items = 0;
  for (int i = 0; i < B; ++i) {
    const int tiles = (ctx[i] + L[i] + 1 + kTcTile - 1) / kTcTile;
    const int pages = (ctx[i] + L[i] + 1 + kPage - 1) / kPage;
    const int cc = std::max(1, std::min(best_c, tiles));
    const int sp = split_pages(pages, (tiles + cc - 1) / cc);
    best_items += static_cast<long long>((pages + sp - 1) / sp) * ((pl.G * (L[i] + 1) + rows_cta - 1) / rows_cta) * Hkv;
  }
  int sk_grid = 0;
  std::vector<int> sk_bound;
  if (persist_ok && pl.cluster <= 1 && persist_mode != 0 && total_pages < (1ll << 30)) {
    std::vector<int> np;
    for (int i = 0; i < B; ++i) {
      const int streams = ((pl.G * (L[i] + 1) + rows_cta - 1) / rows_cta) * Hkv;
      np.insert(np.end(), streams, (ctx[i] + L[i] + 1 + kPage - 1) / kPage);
    }
    sk_bound = cut_chunks(np, static_cast<int>(std::min<long long>(std::min(grid_cap, kMaxChunks), total_pages)));
    sk_grid = static_cast<int>(sk_bound.size()) - 1;
  }
  const bool persist = sk_grid > 0 && (persist_mode > 0 || best_items > slots);

  pl.u.assign(B, AttnUser{});
  pl.item_off.assign(B + 1, 0);
  pl.merge_off.assign(B + 1, 0);
  pl.page_off.assign(B + 1, 0);
  pl.n_chunks = persist ? sk_grid : 0;
  pl.total_pages = persist ? static_cast<int>(total_pages) : 0;
  if (persist) pl.chunk_bound = sk_bound;
  pl.part_off.assign(B, -1);
  long long items = 0, merge = 0, part = 0, pos_pages = 0;
  for (int i = 0; i < B; ++i) {
    AttnUser& U = pl.u[i];
    U.q_off = i == 0 ? 0 : pl.u[i - 1].q_off + pl.u[i - 1].T;
    U.ctx = ctx[i];
    U.T = L[i] + 1;
    U.kv_len = ctx[i] + U.T;
    U.bt_row = bt_rows ? bt_rows[i] : i;
    const int tiles = (U.kv_len + kTcTile - 1) / kTcTile;
    const int pages = (U.kv_len + kPage - 1) / kPage;
    U.n_rb = (pl.G * U.T + rows_cta - 1) / rows_cta;
    pl.item_off[i] = static_cast<int>(items);
    pl.merge_off[i] = static_cast<int>(merge);
    int ns, sp;
    if (persist) {
      // page streams: the most chunks one of the user's streams touches, and
      // (for the plan query) the user's pages; items = pieces
      pl.page_off[i] = static_cast<int>(pos_pages);
      auto chunk_at = [&](long long pos) {
        return static_cast<int>(std::upper_bound(sk_bound.begin(), sk_bound.end() - 1, static_cast<int>(pos)) -
                                sk_bound.begin()) - 1;
      };
      ns = 1;
      for (int k = 0; k < U.n_rb * Hkv; ++k, pos_pages += pages) {
        const int c = chunk_at(pos_pages + pages - 1) - chunk_at(pos_pages) + 1;
        ns = std::max(ns, c);
        items += c;
      }
      sp = pages;
    } else if (pl.cluster > 1) {
      ns = pl.cluster;  // trailing splits may be empty when pages < C
      sp = split_pages(pages, ns);
      items += static_cast<long long>(ns) * U.n_rb * Hkv;
    } else {
      const int cc = std::max(1, std::min(best_c, tiles));
      ns = (tiles + cc - 1) / cc;
      sp = split_pages(pages, ns);
      ns = (pages + sp - 1) / sp;
      items += static_cast<long long>(ns) * U.n_rb * Hkv;
    }
    U.nsplit = ns;
    U.split_len = sp * kPage;
    if (ns > 1 && pl.cluster <= 1) {
      pl.part_off[i] = part;
      part += static_cast<long long>(ns) * Hkv * pl.G * U.T;
      merge += static_cast<long long>(U.T) * Hq;
    }
  }
  pl.item_off[B] = static_cast<int>(items);
  pl.merge_off[B] = static_cast<int>(merge);
  pl.page_off[B] = static_cast<int>(pos_pages);
  long long merge_rows = 0;
  if (persist) {
    // where the streams at each chunk's two ends start and end (the kernel
    // walks a chunk's later pieces stream by stream, with no search)
    const int nc = pl.n_chunks;
    auto chunk_at = [&](int pos) {
      return static_cast<int>(std::upper_bound(sk_bound.begin(), sk_bound.end() - 1, pos) - sk_bound.begin()) - 1;
    };
    auto stream_at = [&](int pos, int* ui, int* s0, int* np) {  // the stream holding page pos
      *ui = static_cast<int>(std::upper_bound(pl.page_off.begin(), pl.page_off.begin() + B, pos) -
                             pl.page_off.begin()) - 1;
      *np = (pl.u[*ui].kv_len + kPage - 1) / kPage;
      const int k = std::min((pos - pl.page_off[*ui]) / *np, pl.u[*ui].n_rb * Hkv - 1);
      *s0 = pl.page_off[*ui] + k * *np;
    };
    pl.chunk_user.assign(nc, 0);
    pl.chunk_c0_back.assign(nc, 0);
    pl.chunk_c1_fwd.assign(nc, 0);
    pl.chunk_cut.assign(nc, 255);
    for (int b = 0; b < nc; ++b) {
      const int lo = sk_bound[b], hi = sk_bound[b + 1];
      if (lo >= hi) continue;  // an empty chunk runs no piece
      int ui, s0, np;
      stream_at(lo, &ui, &s0, &np);
      pl.chunk_user[b] = static_cast<short>(ui);
      pl.chunk_c0_back[b] = static_cast<unsigned char>(b - chunk_at(s0));
      stream_at(hi - 1, &ui, &s0, &np);
      const int c1 = chunk_at(s0 + np - 1);
      pl.chunk_c1_fwd[b] = static_cast<unsigned char>(c1 - b);
      if (c1 > b && chunk_at(s0) == b) {  // a stream that starts here and runs on: cut
        const int sidx = (s0 - pl.page_off[ui]) / np;
        pl.chunk_cut[b] = static_cast<unsigned char>(pl.n_cut++);
        merge_rows += std::min(rows_cta, pl.G * pl.u[ui].T - (sidx / Hkv) * rows_cta);
      }
    }
  }
  pl.n_items = static_cast<int>(items);
  pl.grid = persist ? sk_grid : pl.n_items;
  // rows whose stream has more than one split: every row of a split user
  // (one CTA per item), the rows of the cut streams (page streams)
  pl.n_merge = static_cast<int>(persist ? merge_rows : merge);
  pl.part_rows = part;
  pl.ws_bytes = part ? align_up(part * sizeof(float2), 256) + align_up(part * D * sizeof(float), 256) +
                           align_up(pl.n_cut * sizeof(MergeDesc), 256)
                     : 0;
}

// KV-append inputs of one call (all null: the cache already holds the rows).
struct KvAppend {
  const void* new_k = nullptr;
  const void* new_v = nullptr;
};

template <int CAP>
void fill_attn_params(AttnParams<CAP>& p, const AttnPlan& pl, const void* q, void* out, const int* bt,
                      int max_blocks, float scale, unsigned* status, uint8_t* region) {
  std::memset(&p, 0, sizeof(p));
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.out = static_cast<__nv_bfloat16*>(out);
  p.block_table = bt;
  p.part_ml = reinterpret_cast<float2*>(region);
  p.part_o = reinterpret_cast<float*>(region + align_up(pl.part_rows * sizeof(float2), 256));
  p.merge_desc = reinterpret_cast<MergeDesc*>(region + align_up(pl.part_rows * sizeof(float2), 256) +
                                              align_up(pl.part_rows * pl.D * sizeof(float), 256));
  p.status = status;
  p.cluster = pl.cluster;
  p.B = pl.B; p.Hq = pl.Hq; p.Hkv = pl.Hkv; p.G = pl.G; p.max_blocks = max_blocks;
  p.n_items = pl.n_items; p.n_merge = pl.n_merge;
  p.n_chunks = pl.n_chunks; p.total_pages = pl.total_pages;
  if (pl.n_chunks > 0) {
    for (int b = 0; b <= pl.n_chunks; ++b) p.chunk_bound[b] = pl.chunk_bound[b];
    for (int b = 0; b < pl.n_chunks; ++b) {
      p.chunk_user[b] = pl.chunk_user[b];
      p.chunk_c0_back[b] = pl.chunk_c0_back[b];
      p.chunk_c1_fwd[b] = pl.chunk_c1_fwd[b];
    }
    for (int b = 0; b < pl.n_chunks; ++b) p.chunk_cut[b] = pl.chunk_cut[b];
  }
  p.scale_log2 = scale * 1.4426950408889634f;
  for (int i = 0; i <= pl.B; ++i) {
    p.item_off[i] = pl.item_off[i];
    p.merge_off[i] = pl.merge_off[i];
    p.page_off[i] = pl.page_off[i];
  }
  for (int i = 0; i < pl.B; ++i) { p.part_off[i] = pl.part_off[i]; p.u[i] = pl.u[i]; }
}

template <int D, int CAP>
int launch_attention_tc_t(const AttnPlan& pl, const AttnParams<CAP>& p, const CUtensorMap& tk,
                          const CUtensorMap& tv, cudaStream_t s, bool pdl) {
  const bool persist = pl.n_chunks > 0;
  auto kern = persist ? verify_attention_tc_kernel<D, CAP, true> : verify_attention_tc_kernel<D, CAP, false>;
  static std::mutex mu;
  static bool attr_done[2][64] = {};
  {
    std::lock_guard<std::mutex> lock(mu);
    if (!allow_smem(kern, TcSmem<D>::kAlloc, attr_done[persist ? 1 : 0])) return DIPSD_ERR_CUDA;
  }
  if (launch(kern, dim3(pl.grid), dim3(kTcThreads), TcSmem<D>::kAlloc, s, pl.cluster > 1 ? pl.cluster : 0, pdl,
             p, tk, tv) != cudaSuccess)
    return DIPSD_ERR_CUDA;
  if (pl.n_merge > 0) {
    const cudaError_t e =
        persist ? launch(verify_attention_merge_streams_kernel<D, CAP>, dim3(static_cast<unsigned>(pl.n_cut), D / 32),
                         dim3(128), 0, s, 0, true, p)
                : launch(verify_attention_merge_kernel<D, CAP>, dim3((pl.n_merge + 3) / 4), dim3(128), 0, s, 0, true, p);
    if (e != cudaSuccess) return DIPSD_ERR_CUDA;
  }
  return DIPSD_OK;
}

template <int CAP>
int run_attention_cap(const AttnPlan& pl, const void* q, const void* kc, const void* vc, int num_blocks,
                      const int* bt, int max_blocks, float scale, void* out, unsigned* status,
                      uint8_t* region, cudaStream_t s, bool pdl, const KvAppend& app, bool wait_at_end) {
  static thread_local AttnParams<CAP> p;
  fill_attn_params<CAP>(p, pl, q, out, bt, max_blocks, scale, status, region);
  p.wait_at_end = wait_at_end ? 1 : 0;
  p.new_k = static_cast<const __nv_bfloat16*>(app.new_k);
  p.new_v = static_cast<const __nv_bfloat16*>(app.new_v);
  p.k_cache = static_cast<__nv_bfloat16*>(const_cast<void*>(kc));
  p.v_cache = static_cast<__nv_bfloat16*>(const_cast<void*>(vc));
  p.num_blocks = num_blocks;
  alignas(64) CUtensorMap tk, tv;
  if (!encode_cache_map(&tk, kc, num_blocks, pl.Hkv, pl.D, false) ||
      !encode_cache_map(&tv, vc, num_blocks, pl.Hkv, pl.D, true))
    return DIPSD_ERR_CUDA;
  return pl.D == 128 ? launch_attention_tc_t<128, CAP>(pl, p, tk, tv, s, pdl)
                     : launch_attention_tc_t<64, CAP>(pl, p, tk, tv, s, pdl);
}

int run_attention(const AttnPlan& pl, const void* q, const void* kc, const void* vc, int num_blocks,
                  const int* bt, int max_blocks, float scale, void* out, unsigned* status, uint8_t* region,
                  cudaStream_t s, bool pdl, const KvAppend& app = KvAppend{}, bool wait_at_end = false) {
  if (pl.B <= kCapSmall)
    return run_attention_cap<kCapSmall>(pl, q, kc, vc, num_blocks, bt, max_blocks, scale, out, status,
                                        region, s, pdl, app, wait_at_end);
  return run_attention_cap<kCapLarge>(pl, q, kc, vc, num_blocks, bt, max_blocks, scale, out, status,
                                      region, s, pdl, app, wait_at_end);
}

int check_append(const void* new_k, const void* new_v, const void* q) {
  if (!new_k || !new_v) return DIPSD_ERR_INVALID_ARG;
  if (!aligned(new_k, 16) || !aligned(new_v, 16)) return DIPSD_ERR_INVALID_ARG;
  if (new_k == new_v || new_k == q || new_v == q) return DIPSD_ERR_INVALID_ARG;
  return DIPSD_OK;
}

int check_attn_buffers(const void* q, const void* kc, const void* vc, int num_blocks, const int* bt,
                       int max_blocks, const void* out, int B, const int* L, const int* ctx, float scale) {
  if (!q || !kc || !vc || !bt || !out) return DIPSD_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(kc, 16) || !aligned(vc, 16) || !aligned(out, 16) || !aligned(bt, 4))
    return DIPSD_ERR_INVALID_ARG;
  if (num_blocks < 1 || max_blocks < 1 || !std::isfinite(scale)) return DIPSD_ERR_INVALID_ARG;
  if (q == out) return DIPSD_ERR_INVALID_ARG;
  for (int i = 0; i < B; ++i)
    if (static_cast<long long>(ctx[i]) + L[i] + 1 > static_cast<long long>(kPage) * max_blocks)
      return DIPSD_ERR_INVALID_ARG;
  return DIPSD_OK;
}

// ===================================================================== spec
struct SpecPlan {
  int B = 0, V = 0, vec = 1, nvec = 0, cl1 = 1, cl2 = 1;
  int nk1 = 0, nk2 = 0;  // register path: vectors per lane and segment (0 = generic path)
  int grid1 = 0;         // register path: CTAs of the (persistent) statistics pass
  int nseg1 = 0, nseg2 = 0, n_items1 = 0, n_items2 = 0;
  int sum_t = 0, sum_l = 0;
  bool sparse = false;  // sparse draft payload: no draft logit rows
  std::vector<int> q_off, l_off;
  size_t off_flags = 0, off_ures = 0, off_part1 = 0, off_part2 = 0;
  size_t ws_bytes = 0;  // spec region only
};

// Register path segment sizes, largest first: a segment is 32 lanes x nk
// 16-byte vectors of one row.
constexpr int kNk1[] = {16, 8, 4};
constexpr int kNk2[] = {8, 4, 2};
// arrivals on one counter must fit its 16-bit count
constexpr int kMaxArrivals = 60000;

int check_spec_users(int B, const int* L, int V) {
  if (B < 1 || B > kMaxUsers || !L || V < 1) return DIPSD_ERR_INVALID_ARG;
  long long st = 0;
  for (int i = 0; i < B; ++i) {
    if (L[i] < 0 || L[i] > kMaxDraft) return DIPSD_ERR_INVALID_ARG;
    st += L[i] + 1;
  }
  if (st * static_cast<long long>(V) > (1ll << 40)) return DIPSD_ERR_INVALID_ARG;
  return DIPSD_OK;
}

int cluster_for(int nvec) { return std::max(1, std::min(kMaxCluster, (nvec + 2047) / 2048)); }

int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Largest segment size whose items still fill three quarters of the resident
// warps (two 8-warp CTAs per SM); the smallest otherwise, or when sms <= 0
// (the workspace bound, which must not depend on the device).
template <size_t K>
int pick_nk(const int (&opts)[K], long long rows, int nvec, int sms) {
  if (sms <= 0) return opts[K - 1];
  const long long want = static_cast<long long>(sms) * 16 * 3 / 4;
  for (int nk : opts)
    if (rows * ceil_div(nvec, 32 * nk) >= want) return nk;
  return opts[K - 1];
}

void plan_spec(int B, const int* L, int V, int elem, bool vec_ok, int sms, SpecPlan& pl, bool sparse = false) {
  pl.B = B; pl.V = V;
  pl.sparse = sparse;
  pl.vec = vec_ok ? 16 / elem : 1;
  pl.nvec = V / pl.vec;
  pl.cl1 = cluster_for(pl.nvec);
  pl.cl2 = cluster_for(pl.nvec);
  pl.q_off.assign(B + 1, 0);
  pl.l_off.assign(B + 1, 0);
  for (int i = 0; i < B; ++i) {
    pl.q_off[i + 1] = pl.q_off[i] + L[i] + 1;
    pl.l_off[i + 1] = pl.l_off[i] + L[i];
  }
  pl.sum_t = pl.q_off[B];
  pl.sum_l = pl.l_off[B];
  pl.nk1 = pl.nk2 = pl.grid1 = 0;
  pl.nseg1 = pl.nseg2 = pl.n_items1 = pl.n_items2 = 0;
  size_t o = align_up(static_cast<size_t>(pl.sum_t) * sizeof(SpecStat), 256);
  pl.off_flags = o;
  o += align_up(pl.sum_t, 256);
  pl.off_ures = o;
  o += align_up(static_cast<size_t>(pl.sum_t) * sizeof(float), 256);
  pl.off_part1 = pl.off_part2 = o;
  if (vec_ok) {
    const int rows = pl.sum_t + (sparse ? 0 : pl.sum_l);
    int nk1 = pick_nk(kNk1, rows, pl.nvec, sms);
    int nk2 = sparse ? std::min(4, pick_nk(kNk2, B, pl.nvec, sms)) : pick_nk(kNk2, B, pl.nvec, sms);
    if (sms > 0) {  // segment sizes set by a test override (never above the workspace bound)
      const int o1 = plan_override(DIPSD_TEST_SPEC_NK1), o2 = plan_override(DIPSD_TEST_SPEC_NK2);
      for (int v : kNk1) if (v == o1) nk1 = v;
      for (int v : kNk2) if (v == o2 && !(sparse && v > 4)) nk2 = v;
    }
    const int nseg1 = ceil_div(pl.nvec, 32 * nk1), nseg2 = ceil_div(pl.nvec, 32 * nk2);
    const long long items1 = static_cast<long long>(rows) * nseg1;
    const long long items2 = static_cast<long long>(B) * nseg2;
    if (2 * nseg1 <= kMaxArrivals && nseg2 <= kMaxArrivals && items1 < (1ll << 31) && items2 < (1ll << 31)) {
      pl.nk1 = nk1; pl.nk2 = nk2;
      pl.nseg1 = nseg1; pl.nseg2 = nseg2;
      pl.n_items1 = static_cast<int>(items1);
      pl.n_items2 = static_cast<int>(items2);
      o += align_up(static_cast<size_t>(items1) * sizeof(float4), 256);
      pl.off_part2 = o;
      o += align_up(static_cast<size_t>(items2) * sizeof(float4), 256);
      // statistics pass: two resident CTAs per SM at most, each warp taking
      // several segments in turn when there are more (or a test's cap)
      pl.grid1 = ceil_div(pl.n_items1, kRegWarps);
      if (sms > 0) pl.grid1 = std::min(pl.grid1, 2 * sms);
      if (const int v = plan_override(DIPSD_TEST_SPEC_GRID1)) pl.grid1 = std::min(pl.grid1, v);
    }
  }
  pl.ws_bytes = o;
}

// Spec workspace that covers every plan a call with these sizes can get
// (either logit type, aligned or not, any device): the smallest segments.
size_t spec_ws_need(int B, const int* L, int V) {
  SpecPlan pl;
  plan_spec(B, L, V, 2, false, 0, pl);
  size_t need = pl.ws_bytes;
  if (V % 8 == 0) {
    plan_spec(B, L, V, 2, true, 0, pl);
    need = std::max(need, pl.ws_bytes);
  }
  if (V % 4 == 0) {
    plan_spec(B, L, V, 4, true, 0, pl);
    need = std::max(need, pl.ws_bytes);
  }
  return need;
}

// Workspace of the sparse-payload path (16-byte aligned rows only).
size_t spec_ws_need_sparse(int B, const int* L, int V) {
  SpecPlan pl;
  size_t need = 0;
  if (V % 8 == 0) {
    plan_spec(B, L, V, 2, true, 0, pl, true);
    need = std::max(need, pl.ws_bytes);
  }
  if (V % 4 == 0) {
    plan_spec(B, L, V, 4, true, 0, pl, true);
    need = std::max(need, pl.ws_bytes);
  }
  return need;
}

template <typename T, int VEC, int CAP>
int launch_spec_t(const SpecPlan& pl, const SpecParams<CAP>& p, cudaStream_t s, bool pdl) {
  if (launch(spec_stats_generic_kernel<T, VEC, CAP>, dim3(pl.sum_t * pl.cl1), dim3(kSpecThreads), 0, s, pl.cl1,
             pdl, p) != cudaSuccess)
    return DIPSD_ERR_CUDA;
  if (launch(spec_sample_generic_kernel<T, VEC, CAP>, dim3(pl.B * pl.cl2), dim3(kSpecThreads), 0, s, pl.cl2,
             true, p) != cudaSuccess)
    return DIPSD_ERR_CUDA;
  return DIPSD_OK;
}

template <typename T, int NK2, int CAP, bool SP>
int launch_spec_sample_t(const SpecPlan& pl, const SpecParams<CAP>& p, cudaStream_t s) {
  return launch(spec_sample_kernel<T, NK2, CAP, SP>, dim3(ceil_div(pl.n_items2, kRegWarps)), dim3(kRegThreads), 0,
                s, 1, true, p) == cudaSuccess ? DIPSD_OK : DIPSD_ERR_CUDA;
}

// A second stream the decision and sampling kernels may move to after the
// statistics pass (aux null: everything on the caller's stream).
struct SpecFork {
  cudaStream_t aux = nullptr;
  cudaEvent_t fork = nullptr;
};

template <typename T, int NK1, int CAP, bool SP>
int launch_spec_reg_t(const SpecPlan& pl, const SpecParams<CAP>& p, cudaStream_t s, bool pdl,
                      const SpecFork& fk) {
  if (launch(spec_stats_kernel<T, NK1, CAP, SP>, dim3(pl.grid1), dim3(kRegThreads), 0, s, 0, pdl, p) !=
      cudaSuccess)
    return DIPSD_ERR_CUDA;
  bool pdl_decide = true;
  if (fk.aux) {  // the rest of the stage behind the statistics pass, on the second stream
    if (cudaEventRecord(fk.fork, s) != cudaSuccess || cudaStreamWaitEvent(fk.aux, fk.fork, 0) != cudaSuccess)
      return DIPSD_ERR_CUDA;
    s = fk.aux;
    pdl_decide = false;
  }
  if (launch(spec_decide_kernel<CAP, SP>, dim3(ceil_div(pl.sum_t, kRegWarps)), dim3(kRegThreads), 0, s, 0,
             pdl_decide, p) != cudaSuccess)
    return DIPSD_ERR_CUDA;
  if constexpr (SP) {  // the table's q of every element stays in registers: at most 4 vectors per lane
    return pl.nk2 == 4 ? launch_spec_sample_t<T, 4, CAP, SP>(pl, p, s) : launch_spec_sample_t<T, 2, CAP, SP>(pl, p, s);
  } else {
    switch (pl.nk2) {
      case 8: return launch_spec_sample_t<T, 8, CAP, SP>(pl, p, s);
      case 4: return launch_spec_sample_t<T, 4, CAP, SP>(pl, p, s);
      default: return launch_spec_sample_t<T, 2, CAP, SP>(pl, p, s);
    }
  }
}

template <typename T, int CAP, bool SP>
int launch_spec_reg(const SpecPlan& pl, const SpecParams<CAP>& p, cudaStream_t s, bool pdl, const SpecFork& fk) {
  switch (pl.nk1) {
    case 16: return launch_spec_reg_t<T, 16, CAP, SP>(pl, p, s, pdl, fk);
    case 8: return launch_spec_reg_t<T, 8, CAP, SP>(pl, p, s, pdl, fk);
    default: return launch_spec_reg_t<T, 4, CAP, SP>(pl, p, s, pdl, fk);
  }
}

// Sparse draft payload of one call (null: dense draft logits).
struct SparseDraft {
  const float* draft_logq = nullptr;
  const int* topk_idx = nullptr;
  const float* topk_q = nullptr;
  int topk = 0;
};

template <int CAP>
int run_spec_cap(const SpecPlan& pl, int dtype, const void* z, const void* w, const int* dt, uint64_t seed,
                 const int* uid, int* acc, int* offs, int* toks, float* probs, unsigned* status, uint8_t* region,
                 cudaStream_t s, bool pdl, const SparseDraft& sd, const SpecFork& fk) {
  static thread_local SpecParams<CAP> p;
  std::memset(&p, 0, sizeof(p));
  p.z = z; p.w = w; p.draft_tokens = dt;
  p.seed = seed;
  for (int i = 0; i < pl.B; ++i) p.uid[i] = uid[i];
  p.stats = region;
  p.flags = region + pl.off_flags;
  p.u_res = reinterpret_cast<float*>(region + pl.off_ures);
  p.part1 = reinterpret_cast<float4*>(region + pl.off_part1);
  p.part2 = reinterpret_cast<float4*>(region + pl.off_part2);
  p.counters = reinterpret_cast<unsigned*>(reinterpret_cast<uint8_t*>(status) + kStatusBytes);
  p.sum_t = pl.sum_t;
  p.nseg1 = pl.nseg1; p.nseg2 = pl.nseg2;
  p.n_items1 = pl.n_items1; p.n_items2 = pl.n_items2;
  p.draft_probs = probs; p.accept_len = acc; p.out_offsets = offs; p.out_tokens = toks;
  p.status = status;
  p.B = pl.B; p.V = pl.V; p.nvec = pl.nvec;
  for (int i = 0; i <= pl.B; ++i) { p.q_off[i] = pl.q_off[i]; p.l_off[i] = pl.l_off[i]; }
  if (pl.sparse) {
    if (!pl.nk1) return DIPSD_ERR_UNSUPPORTED;
    p.draft_logq = sd.draft_logq;
    p.topk_idx = sd.topk_idx;
    p.topk_q = sd.topk_q;
    p.topk = sd.topk;
    return dtype == DIPSD_BF16 ? launch_spec_reg<__nv_bfloat16, CAP, true>(pl, p, s, pdl, fk)
                               : launch_spec_reg<float, CAP, true>(pl, p, s, pdl, fk);
  }
  if (pl.nk1)
    return dtype == DIPSD_BF16 ? launch_spec_reg<__nv_bfloat16, CAP, false>(pl, p, s, pdl, fk)
                               : launch_spec_reg<float, CAP, false>(pl, p, s, pdl, fk);
  if (dtype == DIPSD_BF16)
    return pl.vec == 8 ? launch_spec_t<__nv_bfloat16, 8, CAP>(pl, p, s, pdl)
                       : launch_spec_t<__nv_bfloat16, 1, CAP>(pl, p, s, pdl);
  return pl.vec == 4 ? launch_spec_t<float, 4, CAP>(pl, p, s, pdl) : launch_spec_t<float, 1, CAP>(pl, p, s, pdl);
}

int run_spec(const SpecPlan& pl, int dtype, const void* z, const void* w, const int* dt, uint64_t seed,
             const int* uid, int* acc, int* offs, int* toks, float* probs, unsigned* status, uint8_t* region,
             cudaStream_t s, bool pdl, const SparseDraft& sd = SparseDraft{}, const SpecFork& fk = SpecFork{}) {
  if (pl.B <= kCapSmall)
    return run_spec_cap<kCapSmall>(pl, dtype, z, w, dt, seed, uid, acc, offs, toks, probs, status, region, s, pdl,
                                   sd, fk);
  return run_spec_cap<kCapLarge>(pl, dtype, z, w, dt, seed, uid, acc, offs, toks, probs, status, region, s, pdl,
                                 sd, fk);
}

// The second stream and the two events verify_batch forks onto, one set per
// host thread, device and caller stream (a few kept, made on first use).
// Nothing is made while the caller's stream is being captured: such a call
// runs on the one stream.  They live until the thread exits.
struct ForkSet {
  int dev = -1;
  cudaStream_t caller = nullptr, aux = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};

bool fork_set(cudaStream_t s, ForkSet** out) {
  constexpr int kSets = 8;
  static thread_local ForkSet sets[kSets];
  static thread_local int next_slot = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  for (ForkSet& f : sets)
    if (f.aux && f.dev == dev && f.caller == s) {
      *out = &f;
      return true;
    }
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return false;
  ForkSet& f = sets[next_slot];
  next_slot = (next_slot + 1) % kSets;
  if (f.aux) {  // the oldest set goes to the new caller stream (queued work finishes first)
    cudaStreamDestroy(f.aux);
    cudaEventDestroy(f.fork);
    cudaEventDestroy(f.join);
    f = ForkSet{};
  }
  if (cudaStreamCreateWithFlags(&f.aux, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&f.fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&f.join, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    f = ForkSet{};
    return false;
  }
  f.dev = dev;
  f.caller = s;
  *out = &f;
  return true;
}

// Philox key word 1 of every user: a non-negative user id.
int check_user_ids(int B, const int* uid) {
  if (!uid) return DIPSD_ERR_INVALID_ARG;
  for (int i = 0; i < B; ++i)
    if (uid[i] < 0) return DIPSD_ERR_INVALID_ARG;
  return DIPSD_OK;
}

int check_spec_buffers(int dtype, const void* z, const void* w, const int* dt, int* acc, int* offs, int* toks,
                       float* probs, int sum_l, int V, bool* vec_ok) {
  if (dtype != DIPSD_BF16 && dtype != DIPSD_F32) return DIPSD_ERR_INVALID_ARG;
  if (!z || !acc || !offs || !toks) return DIPSD_ERR_INVALID_ARG;
  if (sum_l > 0 && (!w || !dt)) return DIPSD_ERR_INVALID_ARG;
  const size_t elem = dtype == DIPSD_BF16 ? 2 : 4;
  if (!aligned(z, elem) || (w && !aligned(w, elem)) || !aligned(acc, 4) ||
      !aligned(offs, 4) || !aligned(toks, 4) || (probs && !aligned(probs, 8)) || (dt && !aligned(dt, 4)))
    return DIPSD_ERR_INVALID_ARG;
  *vec_ok = (static_cast<size_t>(V) * elem) % 16 == 0 && aligned(z, 16) && (!w || aligned(w, 16));
  return DIPSD_OK;
}

int check_workspace(const void* ws, size_t have, size_t need) {
  if (!ws || !aligned(ws, 256) || have < need) return DIPSD_ERR_WORKSPACE;
  return DIPSD_OK;
}

int cuda_status() { return cudaGetLastError() == cudaSuccess ? DIPSD_OK : DIPSD_ERR_CUDA; }

// ------------------------------------------------------- no-alloc scratch
// Scratch of dipsd_spec_verify_noalloc: the status word followed by a
// dipsd_spec_verify workspace region (row statistics, acceptance bits,
// segment partial sums and arrival counters).  8 MiB covers bf16 logits with
// V up to about 160k at DIPSD_NOALLOC_MAX_POSITIONS positions.
constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;

}  // namespace
}  // namespace dipsd

static __device__ __align__(256) unsigned char g_noalloc_scratch[dipsd::kNoAllocScratchBytes];

// Device address of g_noalloc_scratch on the current device (looked up once
// per device, with that device current); nullptr if the lookup fails.
static uint8_t* noalloc_scratch() {
  static std::mutex mu;
  static void* addr[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
    addr[dev] = p;
  }
  return static_cast<uint8_t*>(addr[dev]);
}

using namespace dipsd;

extern "C" {

const char* dipsd_status_string(int status) {
  switch (status) {
    case DIPSD_OK: return "ok";
    case DIPSD_ERR_INVALID_ARG: return "invalid argument";
    case DIPSD_ERR_UNSUPPORTED: return "unsupported configuration";
    case DIPSD_ERR_CUDA: return "CUDA error";
    case DIPSD_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    default: return "unknown status";
  }
}

int dipsd_abi_version(void) { return DIPSD_ABI_VERSION; }

long long dipsd_launch_count(void) { return g_launches; }

int dipsd_test_set_override(int which, int value) {
  if (which < 1 || which >= kNumOverrides || value < 0) return DIPSD_ERR_INVALID_ARG;
  g_override[which].store(value, std::memory_order_relaxed);
  return DIPSD_OK;
}

int dipsd_philox_words(uint64_t seed, int user_id, long long n_blocks, uint64_t* d_out, void* stream) {
  if (user_id < 0 || n_blocks < 0 || n_blocks > (1ll << 34) || (n_blocks > 0 && !d_out) || !aligned(d_out, 16))
    return DIPSD_ERR_INVALID_ARG;
  if (n_blocks == 0) return DIPSD_OK;
  const long long grid = (n_blocks + 255) / 256;
  if (launch(philox_words_kernel, dim3(static_cast<unsigned>(grid)), dim3(256), 0, static_cast<cudaStream_t>(stream),
             0, false, static_cast<unsigned long long>(seed), static_cast<unsigned long long>(user_id), n_blocks,
             reinterpret_cast<unsigned long long*>(d_out)) != cudaSuccess)
    return DIPSD_ERR_CUDA;
  return cuda_status();
}

int dipsd_verify_uniforms(int B, const int* h_L, const int* h_user_id, uint64_t seed, float* d_uniforms,
                          void* stream) {
  int st = check_spec_users(B, h_L, 1);
  if (st != DIPSD_OK) return st;
  st = check_user_ids(B, h_user_id);
  if (st != DIPSD_OK) return st;
  if (!d_uniforms || !aligned(d_uniforms, 8)) return DIPSD_ERR_INVALID_ARG;
  static thread_local UniformParams p;
  p.seed = seed;
  p.B = B;
  p.q_off[0] = 0;
  for (int i = 0; i < B; ++i) {
    p.q_off[i + 1] = p.q_off[i] + h_L[i] + 1;
    p.uid[i] = h_user_id[i];
  }
  if (launch(verify_uniforms_kernel, dim3((p.q_off[B] + 255) / 256), dim3(256), 0, static_cast<cudaStream_t>(stream),
             0, false, p, reinterpret_cast<float2*>(d_uniforms)) != cudaSuccess)
    return DIPSD_ERR_CUDA;
  return cuda_status();
}

// Attention workspace that covers the plans of both entry points (with and
// without the KV append, which differ in their split choice).
size_t attn_ws_need(int B, const int* L, const int* ctx, const int* bt_rows, int Hq, int Hkv, int D, int sms) {
  AttnPlan a, b;
  plan_attention(B, L, ctx, bt_rows, Hq, Hkv, D, sms, a, true);
  plan_attention(B, L, ctx, bt_rows, Hq, Hkv, D, sms, b, false);
  return std::max(a.ws_bytes, b.ws_bytes);
}

size_t dipsd_verify_attention_workspace_size(int B, const int* h_L, const int* h_ctx, int Hq, int Hkv, int D) {
  if (check_attn_users(B, h_L, h_ctx, Hq, Hkv, D) != DIPSD_OK) return 0;
  DeviceFacts f;
  if (!device_facts(f)) return 0;
  return kHeaderBytes + attn_ws_need(B, h_L, h_ctx, nullptr, Hq, Hkv, D, f.sms);
}

static int verify_attention_impl(int B, const int* h_L, const int* h_ctx, const void* d_q, const void* d_k_cache,
                                 const void* d_v_cache, int num_blocks, const int* d_block_table, int max_blocks,
                                 int Hq, int Hkv, int D, float softmax_scale, void* d_out, void* d_workspace,
                                 size_t workspace_bytes, void* stream, const KvAppend& app) {
  int st = check_attn_users(B, h_L, h_ctx, Hq, Hkv, D);
  if (st != DIPSD_OK) return st;
  st = check_attn_buffers(d_q, d_k_cache, d_v_cache, num_blocks, d_block_table, max_blocks, d_out, B, h_L,
                          h_ctx, softmax_scale);
  if (st != DIPSD_OK) return st;
  DeviceFacts f;
  if (!device_facts(f)) return DIPSD_ERR_CUDA;
  AttnPlan pl;
  plan_attention(B, h_L, h_ctx, nullptr, Hq, Hkv, D, f.sms, pl, app.new_k == nullptr);
  st = check_workspace(d_workspace, workspace_bytes, kHeaderBytes + pl.ws_bytes);
  if (st != DIPSD_OK) return st;
  uint8_t* ws = static_cast<uint8_t*>(d_workspace);
  st = run_attention(pl, d_q, d_k_cache, d_v_cache, num_blocks, d_block_table, max_blocks, softmax_scale, d_out,
                     reinterpret_cast<unsigned*>(ws), ws + kHeaderBytes, static_cast<cudaStream_t>(stream), true,
                     app);
  return st != DIPSD_OK ? st : cuda_status();
}

int dipsd_verify_attention_plan(int B, const int* h_L, const int* h_ctx, int Hq, int Hkv, int D, int num_sms,
                                int append, dipsd_attention_plan* out, int* h_nsplit, int* h_split_len,
                                int* h_chunk_bound) {
  const int st = check_attn_users(B, h_L, h_ctx, Hq, Hkv, D);
  if (st != DIPSD_OK) return st;
  if (num_sms < 1 || !out) return DIPSD_ERR_INVALID_ARG;
  AttnPlan pl;
  plan_attention(B, h_L, h_ctx, nullptr, Hq, Hkv, D, num_sms, pl, append == 0);
  out->n_items = pl.n_items;
  out->grid = pl.grid;
  out->cluster = pl.cluster > 1 ? pl.cluster : 0;
  out->n_merge = pl.n_merge;
  out->stream_chunks = pl.n_chunks;
  if (h_chunk_bound && pl.n_chunks > 0)
    for (int b = 0; b <= pl.n_chunks; ++b) h_chunk_bound[b] = pl.chunk_bound[b];
  out->ws_bytes = pl.ws_bytes;
  for (int i = 0; i < B; ++i) {
    if (h_nsplit) h_nsplit[i] = pl.u[i].nsplit;
    if (h_split_len) h_split_len[i] = pl.u[i].split_len;
  }
  return DIPSD_OK;
}

int dipsd_verify_attention(int B, const int* h_L, const int* h_ctx, const void* d_q, const void* d_k_cache,
                           const void* d_v_cache, int num_blocks, const int* d_block_table, int max_blocks,
                           int Hq, int Hkv, int D, float softmax_scale, void* d_out, void* d_workspace,
                           size_t workspace_bytes, void* stream) {
  return verify_attention_impl(B, h_L, h_ctx, d_q, d_k_cache, d_v_cache, num_blocks, d_block_table, max_blocks, Hq,
                               Hkv, D, softmax_scale, d_out, d_workspace, workspace_bytes, stream, KvAppend{});
}

int dipsd_verify_attention_append(int B, const int* h_L, const int* h_ctx, const void* d_q, const void* d_new_k,
                                  const void* d_new_v, void* d_k_cache, void* d_v_cache, int num_blocks,
                                  const int* d_block_table, int max_blocks, int Hq, int Hkv, int D,
                                  float softmax_scale, void* d_out, void* d_workspace, size_t workspace_bytes,
                                  void* stream) {
  const int st = check_append(d_new_k, d_new_v, d_q);
  if (st != DIPSD_OK) return st;
  KvAppend app;
  app.new_k = d_new_k;
  app.new_v = d_new_v;
  return verify_attention_impl(B, h_L, h_ctx, d_q, d_k_cache, d_v_cache, num_blocks, d_block_table, max_blocks, Hq,
                               Hkv, D, softmax_scale, d_out, d_workspace, workspace_bytes, stream, app);
}

size_t dipsd_spec_verify_workspace_size(int B, const int* h_L, int V) {
  if (check_spec_users(B, h_L, V) != DIPSD_OK) return 0;
  return kHeaderBytes + spec_ws_need(B, h_L, V);
}

int dipsd_spec_verify(int B, const int* h_L, const int* h_user_id, uint64_t seed, int V, int logit_dtype,
                      const void* d_target_logits, const void* d_draft_logits, const int* d_draft_tokens,
                      int* d_accept_len, int* d_out_offsets, int* d_out_tokens, float* d_draft_probs,
                      void* d_workspace, size_t workspace_bytes, void* stream) {
  int st = check_spec_users(B, h_L, V);
  if (st != DIPSD_OK) return st;
  st = check_user_ids(B, h_user_id);
  if (st != DIPSD_OK) return st;
  long long sum_l = 0;
  for (int i = 0; i < B; ++i) sum_l += h_L[i];
  bool vec_ok = false;
  st = check_spec_buffers(logit_dtype, d_target_logits, d_draft_logits, d_draft_tokens, d_accept_len,
                          d_out_offsets, d_out_tokens, d_draft_probs, static_cast<int>(sum_l), V, &vec_ok);
  if (st != DIPSD_OK) return st;
  st = check_workspace(d_workspace, workspace_bytes, kHeaderBytes + spec_ws_need(B, h_L, V));
  if (st != DIPSD_OK) return st;
  DeviceFacts f;
  if (!device_facts(f)) return DIPSD_ERR_CUDA;
  SpecPlan pl;
  plan_spec(B, h_L, V, logit_dtype == DIPSD_BF16 ? 2 : 4, vec_ok, f.sms, pl);
  uint8_t* ws = static_cast<uint8_t*>(d_workspace);
  st = run_spec(pl, logit_dtype, d_target_logits, d_draft_logits, d_draft_tokens, seed, h_user_id, d_accept_len,
                d_out_offsets, d_out_tokens, d_draft_probs, reinterpret_cast<unsigned*>(ws), ws + kHeaderBytes,
                static_cast<cudaStream_t>(stream), true);
  return st != DIPSD_OK ? st : cuda_status();
}

size_t dipsd_spec_verify_sparse_workspace_size(int B, const int* h_L, int V) {
  if (check_spec_users(B, h_L, V) != DIPSD_OK) return 0;
  const size_t need = spec_ws_need_sparse(B, h_L, V);
  return need ? kHeaderBytes + need : 0;
}

int dipsd_spec_verify_sparse(int B, const int* h_L, const int* h_user_id, uint64_t seed, int V, int K,
                             int logit_dtype, const void* d_target_logits, const int* d_draft_tokens,
                             const float* d_draft_logq, const int* d_topk_idx, const float* d_topk_q,
                             int* d_accept_len, int* d_out_offsets, int* d_out_tokens, float* d_draft_probs,
                             void* d_workspace, size_t workspace_bytes, void* stream) {
  int st = check_spec_users(B, h_L, V);
  if (st != DIPSD_OK) return st;
  st = check_user_ids(B, h_user_id);
  if (st != DIPSD_OK) return st;
  if (K < 1 || K > kMaxTopK) return DIPSD_ERR_INVALID_ARG;
  long long sum_l = 0;
  for (int i = 0; i < B; ++i) sum_l += h_L[i];
  bool vec_ok = false;
  // (the draft-logits slot is checked with the target logits' pointer: the sparse path has none)
  st = check_spec_buffers(logit_dtype, d_target_logits, d_target_logits, d_draft_tokens, d_accept_len,
                          d_out_offsets, d_out_tokens, d_draft_probs, static_cast<int>(sum_l), V, &vec_ok);
  if (st != DIPSD_OK) return st;
  if (sum_l > 0 && (!d_draft_logq || !d_topk_idx || !d_topk_q || !aligned(d_draft_logq, 4) ||
                    !aligned(d_topk_idx, 4) || !aligned(d_topk_q, 4)))
    return DIPSD_ERR_INVALID_ARG;
  if (!vec_ok) return DIPSD_ERR_UNSUPPORTED;
  st = check_workspace(d_workspace, workspace_bytes, kHeaderBytes + spec_ws_need_sparse(B, h_L, V));
  if (st != DIPSD_OK) return st;
  DeviceFacts f;
  if (!device_facts(f)) return DIPSD_ERR_CUDA;
  SpecPlan pl;
  plan_spec(B, h_L, V, logit_dtype == DIPSD_BF16 ? 2 : 4, vec_ok, f.sms, pl, true);
  SparseDraft sd;
  sd.draft_logq = d_draft_logq;
  sd.topk_idx = d_topk_idx;
  sd.topk_q = d_topk_q;
  sd.topk = K;
  uint8_t* ws = static_cast<uint8_t*>(d_workspace);
  st = run_spec(pl, logit_dtype, d_target_logits, nullptr, d_draft_tokens, seed, h_user_id, d_accept_len,
                d_out_offsets, d_out_tokens, d_draft_probs, reinterpret_cast<unsigned*>(ws), ws + kHeaderBytes,
                static_cast<cudaStream_t>(stream), true, sd);
  return st != DIPSD_OK ? st : cuda_status();
}

int dipsd_spec_verify_noalloc(int B, const int* h_L, const int* h_user_id, uint64_t seed, int V, int logit_dtype,
                              const void* d_target_logits, const void* d_draft_logits, const int* d_draft_tokens,
                              int* d_accept_len, int* d_out_offsets, int* d_out_tokens, float* d_draft_probs,
                              void* stream) {
  int st = check_spec_users(B, h_L, V);
  if (st != DIPSD_OK) return st;
  st = check_user_ids(B, h_user_id);
  if (st != DIPSD_OK) return st;
  long long sum_l = 0, sum_t = 0;
  for (int i = 0; i < B; ++i) {
    sum_l += h_L[i];
    sum_t += h_L[i] + 1;
  }
  if (sum_t > DIPSD_NOALLOC_MAX_POSITIONS) return DIPSD_ERR_UNSUPPORTED;
  bool vec_ok = false;
  st = check_spec_buffers(logit_dtype, d_target_logits, d_draft_logits, d_draft_tokens, d_accept_len,
                          d_out_offsets, d_out_tokens, d_draft_probs, static_cast<int>(sum_l), V, &vec_ok);
  if (st != DIPSD_OK) return st;
  DeviceFacts f;
  if (!device_facts(f)) return DIPSD_ERR_CUDA;
  SpecPlan pl;
  plan_spec(B, h_L, V, logit_dtype == DIPSD_BF16 ? 2 : 4, vec_ok, f.sms, pl);
  if (kHeaderBytes + pl.ws_bytes > kNoAllocScratchBytes) return DIPSD_ERR_UNSUPPORTED;
  uint8_t* ws = noalloc_scratch();
  if (!ws) return DIPSD_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the status word and every arrival counter start at zero, whatever an
  // earlier call left there
  if (cudaMemsetAsync(ws, 0, kHeaderBytes, s) != cudaSuccess) return DIPSD_ERR_CUDA;
  st = run_spec(pl, logit_dtype, d_target_logits, d_draft_logits, d_draft_tokens, seed, h_user_id, d_accept_len,
                d_out_offsets, d_out_tokens, d_draft_probs, reinterpret_cast<unsigned*>(ws), ws + kHeaderBytes, s,
                true);
  return st != DIPSD_OK ? st : cuda_status();
}

static int gather_members(int B, const int* members, int M, const int* L_all, const int* ctx_all,
                          std::vector<int>& L, std::vector<int>& ctx) {
  if (B < 1 || B > kMaxUsers || !members || M < 1 || !L_all || !ctx_all) return DIPSD_ERR_INVALID_ARG;
  std::vector<char> seen(M, 0);
  L.resize(B);
  ctx.resize(B);
  for (int b = 0; b < B; ++b) {
    const int m = members[b];
    if (m < 0 || m >= M || seen[m]) return DIPSD_ERR_INVALID_ARG;
    seen[m] = 1;
    L[b] = L_all[m];
    ctx[b] = ctx_all[m];
  }
  return DIPSD_OK;
}

size_t dipsd_verify_batch_workspace_size(int B, const int* h_members, int M, const int* h_L_all,
                                         const int* h_ctx_all, int Hq, int Hkv, int D, int V) {
  std::vector<int> L, ctx;
  if (gather_members(B, h_members, M, h_L_all, h_ctx_all, L, ctx) != DIPSD_OK) return 0;
  if (check_attn_users(B, L.data(), ctx.data(), Hq, Hkv, D) != DIPSD_OK) return 0;
  if (check_spec_users(B, L.data(), V) != DIPSD_OK) return 0;
  DeviceFacts f;
  if (!device_facts(f)) return 0;
  return kHeaderBytes + align_up(attn_ws_need(B, L.data(), ctx.data(), h_members, Hq, Hkv, D, f.sms), 256) +
         spec_ws_need(B, L.data(), V);
}

static int verify_batch_impl(int B, const int* h_members, int M, const int* h_L_all, const int* h_ctx_all,
                             const void* d_q, const void* d_k_cache, const void* d_v_cache, int num_blocks,
                             const int* d_block_table_all, int max_blocks, int Hq, int Hkv, int D,
                             float softmax_scale, void* d_attn_out, int V, int logit_dtype,
                             const void* d_target_logits, const void* d_draft_logits, const int* d_draft_tokens,
                             uint64_t seed, int* d_accept_len, int* d_out_offsets, int* d_out_tokens,
                             float* d_draft_probs, void* d_workspace, size_t workspace_bytes, void* stream,
                             const KvAppend& app) {
  std::vector<int> L, ctx;
  int st = gather_members(B, h_members, M, h_L_all, h_ctx_all, L, ctx);
  if (st != DIPSD_OK) return st;
  st = check_attn_users(B, L.data(), ctx.data(), Hq, Hkv, D);
  if (st != DIPSD_OK) return st;
  st = check_spec_users(B, L.data(), V);
  if (st != DIPSD_OK) return st;
  st = check_attn_buffers(d_q, d_k_cache, d_v_cache, num_blocks, d_block_table_all, max_blocks, d_attn_out, B,
                          L.data(), ctx.data(), softmax_scale);
  if (st != DIPSD_OK) return st;
  long long sum_l = 0;
  for (int b = 0; b < B; ++b) sum_l += L[b];
  bool vec_ok = false;
  st = check_spec_buffers(logit_dtype, d_target_logits, d_draft_logits, d_draft_tokens, d_accept_len,
                          d_out_offsets, d_out_tokens, d_draft_probs, static_cast<int>(sum_l), V, &vec_ok);
  if (st != DIPSD_OK) return st;
  DeviceFacts f;
  if (!device_facts(f)) return DIPSD_ERR_CUDA;
  AttnPlan ap;
  plan_attention(B, L.data(), ctx.data(), h_members, Hq, Hkv, D, f.sms, ap, app.new_k == nullptr);
  SpecPlan sp;
  plan_spec(B, L.data(), V, logit_dtype == DIPSD_BF16 ? 2 : 4, vec_ok, f.sms, sp);
  const size_t attn_region = align_up(ap.ws_bytes, 256);
  st = check_workspace(d_workspace, workspace_bytes, kHeaderBytes + attn_region + sp.ws_bytes);
  if (st != DIPSD_OK) return st;
  uint8_t* ws = static_cast<uint8_t*>(d_workspace);
  unsigned* status = reinterpret_cast<unsigned*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The two stages share no data.  The statistics pass runs first, alone
  // (it wants all of the HBM bandwidth: an attention grid started while it
  // drains measured slower); then the attention grid on the caller's stream
  // and, beside it on a second stream, the decision and sampling kernels,
  // latency-bound chains that need little bandwidth; the call's last
  // operation joins the second stream back into the caller's.
  // Without a second stream (a caller stream first seen inside a capture, the
  // scalar path, or a test's choice) it is one stream: spec_verify, then the
  // attention grid, which starts as soon as the sampling kernel has passed
  // its own wait and waits for that kernel only before it exits.
  // Each member's Philox key word 1 is its index in the per-user tables.
  ForkSet* fs = nullptr;
  const bool forked = sp.nk1 > 0 && plan_override(DIPSD_TEST_BATCH_FORK) != 2 && fork_set(s, &fs);
  st = run_spec(sp, logit_dtype, d_target_logits, d_draft_logits, d_draft_tokens, seed, h_members, d_accept_len,
                d_out_offsets, d_out_tokens, d_draft_probs, status, ws + kHeaderBytes + attn_region, s, true,
                SparseDraft{}, forked ? SpecFork{fs->aux, fs->fork} : SpecFork{});
  if (st != DIPSD_OK) return st;
  st = run_attention(ap, d_q, d_k_cache, d_v_cache, num_blocks, d_block_table_all, max_blocks, softmax_scale,
                     d_attn_out, status, ws + kHeaderBytes, s, !forked, app, !forked);
  if (st != DIPSD_OK) return st;
  if (forked && (cudaEventRecord(fs->join, fs->aux) != cudaSuccess || cudaStreamWaitEvent(s, fs->join, 0) != cudaSuccess))
    return DIPSD_ERR_CUDA;
  return cuda_status();
}

int dipsd_verify_batch(int B, const int* h_members, int M, const int* h_L_all, const int* h_ctx_all,
                       const void* d_q, const void* d_k_cache, const void* d_v_cache, int num_blocks,
                       const int* d_block_table_all, int max_blocks, int Hq, int Hkv, int D, float softmax_scale,
                       void* d_attn_out, int V, int logit_dtype, const void* d_target_logits,
                       const void* d_draft_logits, const int* d_draft_tokens, uint64_t seed,
                       int* d_accept_len, int* d_out_offsets, int* d_out_tokens, float* d_draft_probs,
                       void* d_workspace, size_t workspace_bytes, void* stream) {
  return verify_batch_impl(B, h_members, M, h_L_all, h_ctx_all, d_q, d_k_cache, d_v_cache, num_blocks,
                           d_block_table_all, max_blocks, Hq, Hkv, D, softmax_scale, d_attn_out, V, logit_dtype,
                           d_target_logits, d_draft_logits, d_draft_tokens, seed, d_accept_len, d_out_offsets,
                           d_out_tokens, d_draft_probs, d_workspace, workspace_bytes, stream, KvAppend{});
}

int dipsd_verify_batch_append(int B, const int* h_members, int M, const int* h_L_all, const int* h_ctx_all,
                              const void* d_q, const void* d_new_k, const void* d_new_v, void* d_k_cache,
                              void* d_v_cache, int num_blocks, const int* d_block_table_all, int max_blocks, int Hq,
                              int Hkv, int D, float softmax_scale, void* d_attn_out, int V, int logit_dtype,
                              const void* d_target_logits, const void* d_draft_logits, const int* d_draft_tokens,
                              uint64_t seed, int* d_accept_len, int* d_out_offsets, int* d_out_tokens,
                              float* d_draft_probs, void* d_workspace, size_t workspace_bytes, void* stream) {
  const int st = check_append(d_new_k, d_new_v, d_q);
  if (st != DIPSD_OK) return st;
  KvAppend app;
  app.new_k = d_new_k;
  app.new_v = d_new_v;
  return verify_batch_impl(B, h_members, M, h_L_all, h_ctx_all, d_q, d_k_cache, d_v_cache, num_blocks,
                           d_block_table_all, max_blocks, Hq, Hkv, D, softmax_scale, d_attn_out, V, logit_dtype,
                           d_target_logits, d_draft_logits, d_draft_tokens, seed, d_accept_len, d_out_offsets,
                           d_out_tokens, d_draft_probs, d_workspace, workspace_bytes, stream, app);
}

}  // extern "C"
