/*
 * dipsd.h -- C ABI of the GB300 (sm_103a) batched-verification library for
 * DiP-SD edge servers (arXiv 2604.20919).
 *
 * In every speculative-decoding round each user's device sends L_i draft
 * tokens to the edge server, which verifies a whole batch of users in one
 * target-model pass (Sec. II-A, stage 2 "Batch Verification"): it finds each
 * user's first rejected draft, drops the drafts after it, and emits one more
 * token after the last accepted position, so every user gets at least one
 * token per round.  The per-user arguments follow the paper's problem
 * statement (Sec. II-A, Table 1): draft length l_m (here L_i), prefix length
 * i_m (here the context length C_i), and batch membership B_n(x)
 * (Sec. III-C, the users assigned to stage n).
 *
 * This library implements the data-parallel part of that step:
 *   dipsd_verify_attention  causal GQA attention of each user's L_i+1 verify
 *                           tokens over the user's paged bf16 KV cache;
 *   dipsd_spec_verify       speculative sampling over the vocabulary;
 *   dipsd_verify_batch      both, for one pipeline stage's users;
 *   *_append variants       the same, also writing the verify tokens' own
 *                           K/V rows into their pages in the same launch;
 *   dipsd_spec_verify_sparse  speculative sampling from a sparse draft
 *                           payload (draft-token log-probabilities and a
 *                           top-K draft distribution);
 *   dipsd_verify_attention_plan  the attention's work-item plan for a given
 *                           SM count (host only);
 *   dipsd_philox_words,
 *   dipsd_verify_uniforms   the random numbers speculative sampling draws
 *                           (in-kernel Philox4x64-10), written out.
 *
 * Conventions shared by every entry point
 *   - Pointers named d_* are device pointers, h_* host pointers.  The caller
 *     owns all memory; the library never allocates or frees.
 *   - Calls are asynchronous on `stream` (a cudaStream_t passed as void*;
 *     NULL = legacy default stream).  Outputs are valid once the stream has
 *     reached the end of the call.
 *   - Every argument is validated on the host before anything is launched;
 *     on error nothing is written and a status code is returned.
 *   - Verify token t of user i (t = 0..L_i) is the token at absolute position
 *     C_i + t: t = 0 is the last token emitted in the previous round, t >= 1
 *     are the drafts d_{i,1..L_i}.  Tokens are packed user after user in batch
 *     order: user i's tokens start at row sum_{j<i} (L_j + 1).
 *   - Workspace: caller-allocated device memory of at least the size the
 *     matching *_workspace_size call returns for the same per-user arguments
 *     (on the same device).  Its first 16 bytes hold a device status word:
 *     kernels OR error bits into it (DIPSD_DEVERR_*) instead of trapping; zero
 *     it before a call whose status you want to read.  Zero the whole
 *     workspace once before its first use (cudaMemset): the arrival counters
 *     that follow the status word must start at zero, and every call leaves
 *     them at zero.  Calls that share a workspace must not overlap on the GPU.
 */
#ifndef DIPSD_H
#define DIPSD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DIPSD_ABI_VERSION 2
#define DIPSD_PAGE_SIZE 16    /* tokens per KV page */
#define DIPSD_MAX_USERS 512   /* users per call */
#define DIPSD_MAX_DRAFT 31    /* L_i <= 31: one warp ballot covers a user */

typedef enum {
  DIPSD_OK = 0,
  DIPSD_ERR_INVALID_ARG = 1, /* a size, length or pointer failed validation */
  DIPSD_ERR_UNSUPPORTED = 2, /* valid but not built (e.g. head_dim not 64/128) */
  DIPSD_ERR_CUDA = 3,        /* a CUDA runtime call or launch failed */
  DIPSD_ERR_WORKSPACE = 4    /* workspace NULL, misaligned or too small */
} dipsd_status;

typedef enum { DIPSD_BF16 = 0, DIPSD_F32 = 1 } dipsd_dtype;

/* Device status bits (workspace word 0). */
#define DIPSD_DEVERR_WAIT_TIMEOUT 1u /* a bounded mbarrier wait expired */
#define DIPSD_DEVERR_BAD_TOKEN 2u    /* a draft token outside [0, V): treated as rejected */
#define DIPSD_DEVERR_BAD_BLOCK 4u    /* an appended row's page id outside [0, num_blocks): row not written */

/* Human-readable name of a dipsd_status value (static string). */
const char* dipsd_status_string(int status);

/* DIPSD_ABI_VERSION of the loaded library. */
int dipsd_abi_version(void);

/* Number of CUDA kernels this library has launched from the calling host
 * thread since the library was loaded (a diagnostic counter). */
long long dipsd_launch_count(void);

/* ------------------------------------------------------------------------
 * Verify attention (the target model's attention over the verify tokens,
 * Sec. II-A stage 2; its cost is the I*L term of Eq. (Fv)).
 *
 * For user i, verify token t and query head h (KV head h / G, G = Hq/Hkv):
 *   out[t,h] = sum_{j <= C_i + t} softmax_j(softmax_scale * q[t,h] . k_j) v_j
 * over the user's keys j = 0 .. C_i + L_i.  The K/V rows of the L_i+1 verify
 * tokens must already be written into the cache pages.
 *
 * B             number of users, 1..DIPSD_MAX_USERS
 * h_L, h_ctx    [B] host: draft length L_i in 0..DIPSD_MAX_DRAFT, context C_i >= 0
 * d_q           [sum_i (L_i+1)][Hq][D] bf16, row-major, 16-byte aligned
 * d_k_cache,
 * d_v_cache     [num_blocks][Hkv][DIPSD_PAGE_SIZE][D] bf16, 16-byte aligned
 * d_block_table [B][max_blocks] int32: page p of user i (tokens 16p..16p+15)
 *               is cache block d_block_table[i*max_blocks + p]; entries past
 *               ceil((C_i+L_i+1)/16) are never read.  A block id outside
 *               [0, num_blocks) reads zeros (it cannot fault).
 * Hq, Hkv, D    query heads, KV heads (Hq % Hkv == 0), head_dim in {64, 128}
 * softmax_scale usually D^-1/2
 * d_out         [sum_i (L_i+1)][Hq][D] bf16 (may not alias d_q)
 * Requires C_i + L_i + 1 <= 16 * max_blocks for every user.
 * ---------------------------------------------------------------------- */
size_t dipsd_verify_attention_workspace_size(int B, const int* h_L, const int* h_ctx,
                                             int Hq, int Hkv, int D);
int dipsd_verify_attention(int B, const int* h_L, const int* h_ctx,
                           const void* d_q, const void* d_k_cache, const void* d_v_cache,
                           int num_blocks, const int* d_block_table, int max_blocks,
                           int Hq, int Hkv, int D, float softmax_scale,
                           void* d_out, void* d_workspace, size_t workspace_bytes,
                           void* stream);

/* How a verify_attention launch cuts the batch into work (host only: no
 * CUDA call, no device needed).  The attention entry points make the same
 * plan for a device with num_sms SMs (append = 0: dipsd_verify_attention and
 * dipsd_verify_batch; append = 1: the *_append entry points).
 *
 * Either one CTA per work item: (user, 128-row block of its G*(L_i+1) query
 * rows, KV head, KV split), a user's KV split s covering keys
 * [s*split_len, (s+1)*split_len) of its C_i+L_i+1 (split_len a multiple of
 * DIPSD_PAGE_SIZE); or (stream_chunks > 0) a persistent grid over page
 * streams: the pages of every (user, row block, KV head) as one stream, the
 * streams of users 0..B-1 (row block, then head, in order) back to back, cut
 * into stream_chunks chunks (about equal pages plus a fixed charge per
 * stream piece), CTA b taking chunk b; a stream cut by chunk boundaries has
 * one split per chunk it touches, merged afterwards.
 *
 * B, h_L, h_ctx, Hq, Hkv, D   as for dipsd_verify_attention
 * num_sms       SMs of the device the plan is for (>= 1)
 * append        0 or 1 (see above)
 * out           filled on success (caller-owned)
 * h_nsplit,
 * h_split_len   [B] host, nullable: per user the number of KV splits and the
 *               keys per split (stream_chunks > 0: the most splits one of the
 *               user's streams gets, and the keys of one of its streams)
 * h_chunk_bound [num_sms + 1] host, nullable: stream_chunks > 0: chunk b is
 *               pages [h_chunk_bound[b], h_chunk_bound[b + 1]) of the streams
 * Returns DIPSD_OK; the status dipsd_verify_attention would return for
 * invalid lengths or shapes; DIPSD_ERR_INVALID_ARG for num_sms < 1 or a null
 * out.  Nothing is written on failure.
 * ---------------------------------------------------------------------- */
typedef struct {
  int n_items;     /* work items (page streams: the pieces of all chunks) */
  int grid;        /* CTAs launched: n_items, or (chunk_pages > 0) the chunks */
  int cluster;     /* > 1: every user's KV in `cluster` splits that merge
                      inside one thread-block cluster; 0 otherwise */
  int n_merge;     /* (verify token, query head) rows whose KV stream has
                      more than one split, combined by a merge kernel after
                      the grid (0: no merge launch) */
  int stream_chunks; /* > 0: the persistent grid's chunks (CTAs) */
  size_t ws_bytes; /* workspace bytes of this plan past the status header */
} dipsd_attention_plan;
int dipsd_verify_attention_plan(int B, const int* h_L, const int* h_ctx, int Hq, int Hkv, int D,
                                int num_sms, int append, dipsd_attention_plan* out,
                                int* h_nsplit, int* h_split_len, int* h_chunk_bound);

/* ------------------------------------------------------------------------
 * Speculative verification (Sec. II-A stage 2: first-mismatch truncation and
 * one bonus token; the accept/reject rule is the speculative sampling the
 * paper cites, whose expected output length is Eq. (u_single)).
 *
 * Per user i and draft position t < L_i (draft d = d_{i,t+1}):
 *   p_t = softmax(target_logits[t]), q_t = softmax(draft_logits[t]),
 *   accepted iff u_acc(t) * q_t(d) < p_t(d).
 * a_i = number of leading accepted drafts.  Emitted: d_{i,1..a_i}, then one
 * token drawn with u_res(a_i) by inverse CDF (smallest k whose cumulative
 * weight exceeds u * total, ascending token order) from
 *   max(0, p_a - q_a)  if a_i < L_i (p_a itself if that has no mass),
 *   p_{L_i}            if a_i == L_i (the bonus position).
 *
 * The uniforms are drawn inside the kernels (the paper leaves them
 * unspecified): user i's stream is Philox4x64-10 (Salmon et al., SC 2011)
 * under the 128-bit key (seed, h_user_id[i]), counter blocks (1,0,0,0),
 * (2,0,0,0), ...; verify position t takes the stream's 64-bit words 2t
 * (u_acc) and 2t+1 (u_res), each mapped to ((w >> 41) + 0.5) * 2^-23, an
 * exact fp32 in (0, 1).  The same (seed, user id) always gives the same
 * uniforms; dipsd_verify_uniforms writes them out.
 *
 * B                  1..DIPSD_MAX_USERS;  h_L [B] host, 0..DIPSD_MAX_DRAFT
 * h_user_id          [B] host, >= 0: Philox key word 1 of each user
 * seed               Philox key word 0
 * V                  vocabulary size >= 1
 * logit_dtype        DIPSD_BF16 or DIPSD_F32 (both logit arrays)
 * d_target_logits    [sum_i (L_i+1)][V], user i's rows in position order
 * d_draft_logits     [sum_i L_i][V]
 * d_draft_tokens     [sum_i L_i] int32 in [0, V)
 * d_accept_len       [B] int32 out: a_i
 * d_out_offsets      [B+1] int32 out: exclusive prefix of (a_i + 1)
 * d_out_tokens       [sum_i (L_i+1)] int32 out (capacity); the first
 *                    d_out_offsets[B] entries are the packed emitted tokens
 * d_draft_probs      NULL or [sum_i (L_i+1)][2] fp32 out: (p_t(d), q_t(d)) at
 *                    every draft position, (0, 0) at bonus positions
 * Rows must start 16-byte aligned for the fast path (V*elem % 16 == 0).
 * ---------------------------------------------------------------------- */
size_t dipsd_spec_verify_workspace_size(int B, const int* h_L, int V);
int dipsd_spec_verify(int B, const int* h_L, const int* h_user_id, uint64_t seed, int V,
                      int logit_dtype, const void* d_target_logits, const void* d_draft_logits,
                      const int* d_draft_tokens, int* d_accept_len, int* d_out_offsets,
                      int* d_out_tokens, float* d_draft_probs, void* d_workspace,
                      size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Speculative verification from a sparse draft payload (Sec. II-A: the device
 * sends the drafted tokens and, when the protocol needs it, a small amount of
 * probability information such as the draft tokens' log-probabilities).
 *
 * As dipsd_spec_verify without draft logits.  For draft position t of user i
 * (draft row r = sum_{j<i} L_j + t) the draft distribution q_r is the table
 * (d_topk_idx[r][k], d_topk_q[r][k]), k < K: q_r(idx) = q, 0 for every token
 * not in the table (exact for a device that samples from its own top K).
 *   accepted iff u_acc(t) * exp(d_draft_logq[r]) < p_t(d);
 *   residual max(0, p_a - q_a) over the whole vocabulary.
 * K                 1..64;  d_topk_idx [sum L][K] int32 (distinct tokens;
 *                   entries outside [0, V) are ignored and set
 *                   DIPSD_DEVERR_BAD_TOKEN), d_topk_q [sum L][K] fp32 >= 0,
 *                   d_draft_logq [sum L] fp32.
 * Only the target logit rows are read.  Rows must be 16-byte aligned
 * (V * elem % 16 == 0), else DIPSD_ERR_UNSUPPORTED.  d_draft_probs gets
 * (p_t(d), exp(draft_logq)).
 * ---------------------------------------------------------------------- */
size_t dipsd_spec_verify_sparse_workspace_size(int B, const int* h_L, int V);
int dipsd_spec_verify_sparse(int B, const int* h_L, const int* h_user_id, uint64_t seed, int V,
                             int K, int logit_dtype, const void* d_target_logits,
                             const int* d_draft_tokens, const float* d_draft_logq,
                             const int* d_topk_idx, const float* d_topk_q, int* d_accept_len,
                             int* d_out_offsets, int* d_out_tokens, float* d_draft_probs,
                             void* d_workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * One pipeline stage: the users of batch n (Sec. III-C, B_n(x)) verified
 * together -- attention and speculative verification.  The two stages read
 * disjoint inputs and run overlapped: after the statistics pass of the
 * speculative verification, the attention grid runs on `stream` while the
 * decision and sampling kernels run beside it on a second stream that the
 * library keeps per host thread, device and caller stream (made on the first
 * call from that thread and stream outside a stream capture; it lives until
 * the thread exits) and joins back into `stream` before the call returns.
 * All outputs are complete when the work queued on `stream` completes; a
 * call captured into a CUDA graph captures both streams.  No output buffer
 * may overlap an input buffer.
 *
 * Per-user tables cover all M users being served; h_members[b] (distinct, in
 * [0, M)) names the b-th user of this batch and is also its Philox key word
 * 1 (its user id for dipsd_spec_verify).  Per-batch tensors (d_q,
 * d_attn_out, logits, draft tokens and the outputs) are packed in h_members
 * order exactly as for the two calls above.
 * h_L_all, h_ctx_all  [M] host;  d_block_table_all [M][max_blocks] int32.
 * ---------------------------------------------------------------------- */
size_t dipsd_verify_batch_workspace_size(int B, const int* h_members, int M,
                                         const int* h_L_all, const int* h_ctx_all,
                                         int Hq, int Hkv, int D, int V);
int dipsd_verify_batch(int B, const int* h_members, int M,
                       const int* h_L_all, const int* h_ctx_all,
                       const void* d_q, const void* d_k_cache, const void* d_v_cache,
                       int num_blocks, const int* d_block_table_all, int max_blocks,
                       int Hq, int Hkv, int D, float softmax_scale, void* d_attn_out,
                       int V, int logit_dtype, const void* d_target_logits,
                       const void* d_draft_logits, const int* d_draft_tokens,
                       uint64_t seed, int* d_accept_len, int* d_out_offsets,
                       int* d_out_tokens, float* d_draft_probs,
                       void* d_workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * KV append inside verification (the round's state update, Sec. II-A stage 2:
 * the verify tokens' own keys and values join each user's cache).
 *
 * Same as dipsd_verify_attention / dipsd_verify_batch, with the cache pages
 * at positions C_i .. C_i+L_i (which must be allocated in the block table)
 * not yet holding the verify tokens' rows:
 * d_new_k, d_new_v   [sum_i (L_i+1)][Hkv][D] bf16, 16-byte aligned, users
 *                    packed like d_q: verify token t of user i is written to
 *                    position C_i + t (block d_block_table[i][(C_i+t)/16],
 *                    slot (C_i+t) % 16) of d_k_cache / d_v_cache, and the
 *                    attention of this call uses those rows (whatever the
 *                    pages held before).  Every other cache byte is left as
 *                    it was.
 * Workspaces are sized by the matching *_workspace_size calls.  A page id
 * outside [0, num_blocks) at an appended position sets
 * DIPSD_DEVERR_BAD_BLOCK and that row is not written.
 * ---------------------------------------------------------------------- */
int dipsd_verify_attention_append(int B, const int* h_L, const int* h_ctx,
                                  const void* d_q, const void* d_new_k, const void* d_new_v,
                                  void* d_k_cache, void* d_v_cache, int num_blocks,
                                  const int* d_block_table, int max_blocks, int Hq, int Hkv,
                                  int D, float softmax_scale, void* d_out, void* d_workspace,
                                  size_t workspace_bytes, void* stream);
int dipsd_verify_batch_append(int B, const int* h_members, int M, const int* h_L_all,
                              const int* h_ctx_all, const void* d_q, const void* d_new_k,
                              const void* d_new_v, void* d_k_cache, void* d_v_cache,
                              int num_blocks, const int* d_block_table_all, int max_blocks,
                              int Hq, int Hkv, int D, float softmax_scale, void* d_attn_out,
                              int V, int logit_dtype, const void* d_target_logits,
                              const void* d_draft_logits, const int* d_draft_tokens,
                              uint64_t seed, int* d_accept_len, int* d_out_offsets,
                              int* d_out_tokens, float* d_draft_probs, void* d_workspace,
                              size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Speculative verification without a caller-provided workspace.
 *
 * The paper has no counterpart to this entry point; it exists for callers
 * that cannot allocate device memory themselves: for example a plugin inside
 * a host program whose own pool owns all device memory, or a serving loop
 * that must not call cudaMalloc because it can synchronise the device.  It
 * computes exactly what dipsd_spec_verify computes, with the same arguments
 * minus the workspace, and allocates nothing (no cudaMalloc, no cudaFree, no
 * allocating library routine).
 *
 * Scratch lives in one static device array of the library, sized for at most
 * DIPSD_NOALLOC_MAX_POSITIONS verify positions (sum_i (L_i+1)) and 8 MiB in
 * all (enough for bf16 logits with V up to about 160k at the maximum number of
 * positions); a larger batch is rejected with DIPSD_ERR_UNSUPPORTED before
 * anything is launched.  Every GPU that loads the library holds that 8 MiB
 * array until the process exits.  The first call on a device looks up the
 * array's device address with that device current; make that first call
 * before any stream capture.  All calls share the one array: calls that
 * overlap on the GPU (other streams, other host threads) race and must be
 * serialised by the caller.  Each call clears the array's status word and
 * arrival counters on `stream` before its kernels run, so no call depends
 * on what an earlier one left there.  The device status bits
 * (DIPSD_DEVERR_*) live in that array and cannot be read on this path: a
 * draft token outside [0, V) is still treated as rejected, but unlike the
 * workspace entry points nothing reports it.
 * ---------------------------------------------------------------------- */
#define DIPSD_NOALLOC_MAX_POSITIONS 4096
int dipsd_spec_verify_noalloc(int B, const int* h_L, const int* h_user_id, uint64_t seed,
                              int V, int logit_dtype, const void* d_target_logits,
                              const void* d_draft_logits, const int* d_draft_tokens,
                              int* d_accept_len, int* d_out_offsets, int* d_out_tokens,
                              float* d_draft_probs, void* stream);

/* ------------------------------------------------------------------------
 * The random numbers of speculative sampling, written out (not in the paper:
 * it leaves them unspecified; the generator is Philox4x64-10 of Salmon,
 * Moraes, Dror and Shaw, SC 2011).
 *
 * dipsd_philox_words: words of counter blocks 0 .. n_blocks-1 of the stream
 *   with key (seed, user_id): d_out[4 b + j] = word j of the block at
 *   counter (b + 1, 0, 0, 0).  d_out: [4 n_blocks] uint64, 16-byte aligned;
 *   user_id >= 0; 0 <= n_blocks <= 2^34.
 * dipsd_verify_uniforms: the (u_acc, u_res) pairs dipsd_spec_verify draws
 *   for this batch: d_uniforms [sum_i (L_i+1)][2] fp32, row q_off_i + t =
 *   verify position t of user i (u_acc of a bonus position is drawn but
 *   never used).  Arguments as for dipsd_spec_verify.
 * Both are asynchronous on `stream` and allocate nothing.
 * ---------------------------------------------------------------------- */
int dipsd_philox_words(uint64_t seed, int user_id, long long n_blocks, uint64_t* d_out,
                       void* stream);
int dipsd_verify_uniforms(int B, const int* h_L, const int* h_user_id, uint64_t seed,
                          float* d_uniforms, void* stream);

/* ------------------------------------------------------------------------
 * Test hooks (not for production use): process-wide overrides of the
 * planners' choices, so that tests reach every kernel variant on small
 * inputs.  Each override holds until it is set back to 0 (the planner's own
 * choice).  The *_workspace_size calls plan with the same overrides, so set
 * them before sizing a workspace.  The library never reads the environment.
 *   DIPSD_TEST_ATTN_SPLIT_TILES  KV split length in 128-key tiles
 *   DIPSD_TEST_ATTN_CLUSTER      cluster merge with this many splits (2..)
 *   DIPSD_TEST_ATTN_PERSIST      1: persistent grid whenever allowed, 2: never
 *   DIPSD_TEST_ATTN_GRID         persistent grid of at most this many CTAs
 *   DIPSD_TEST_SPEC_NK1,
 *   DIPSD_TEST_SPEC_NK2          16-byte vectors per lane in a segment of the
 *                                two sampling passes (one of 16/8/4, 8/4/2)
 *   DIPSD_TEST_SPEC_GRID1        at most this many CTAs in the statistics
 *                                pass, so each warp takes several segments
 *   DIPSD_TEST_BATCH_FORK        verify_batch: 1 = decision and sampling on a
 *                                second stream beside the attention grid (the
 *                                default), 2 = everything on the one stream
 * Returns DIPSD_ERR_INVALID_ARG for an unknown code or a negative value.
 * ---------------------------------------------------------------------- */
#define DIPSD_TEST_ATTN_SPLIT_TILES 1
#define DIPSD_TEST_ATTN_CLUSTER 2
#define DIPSD_TEST_ATTN_PERSIST 3
#define DIPSD_TEST_ATTN_GRID 4
#define DIPSD_TEST_SPEC_NK1 5
#define DIPSD_TEST_SPEC_NK2 6
#define DIPSD_TEST_SPEC_GRID1 7
#define DIPSD_TEST_BATCH_FORK 8
int dipsd_test_set_override(int which, int value);

#ifdef __cplusplus
}
#endif
#endif /* DIPSD_H */
