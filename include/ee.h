/*
 * ee.h -- C ABI of the GB300 (sm_103a) verification-step library (libee.so).
 *
 * One verification step of EfficientEdit's edit-oriented speculative decoding
 * (arXiv 2506.02780, Sec. III-A): a draft tree -- a span of the original code
 * reused verbatim plus short generated branches -- is scored in one target
 * pass and the longest draft prefix on which the target's greedy choice agrees
 * is accepted (Eq. (piecewise)).  The entry points are the steps of that pass:
 *
 *   ee_match_reuse       reuse-span lookup in the original code     (Sec. III-A)
 *   ee_tree_prepare      depth / ancestor masks of the draft tree
 *   ee_tree_verify_attn  tree-masked attention over the paged cache (Sec. III-A)
 *   ee_lmhead_accept     LM head + argmax + longest accepted path   (Eq. piecewise)
 *   ee_kv_compact        accepted path's K/V appended to the cache  (Sec. III-A)
 *   ee_tree_verify_attn_inplace / ee_kv_compact_inplace
 *                        the same two steps with the tree's K/V already in
 *                        the cache after the context (in-place speculative K/V)
 *   ee_build_reuse_tree / ee_advance
 *                        the Reuse <-> Generate controller on the device: the
 *                        next draft tree from the match points, the commit of
 *                        a step's result (Sec. III-A)
 *   ee_chain_verify_attn causal attention of linear drafts of up to 2048
 *                        tokens verified in place (long reuse drafts; the LM
 *                        head takes them with anc NULL)
 *   ee_lmhead_pack_weights / ee_lmhead_accept_packed
 *                        the LM-head weights rearranged once into the
 *                        kernel's tile order, and the LM head reading them
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every pointer argument except `ws` in ee_read_errors' output is a DEVICE
 *    pointer owned by the caller.  The library never allocates device memory,
 *    never frees, never synchronises (except ee_read_errors) and enqueues all
 *    work on `stream` (NULL = legacy default stream).
 *  - Integer arrays are int32 unless stated; bf16 arrays are raw bf16 bit
 *    patterns (ee_bf16), row-major, densely packed.
 *  - Tree nodes: sequence s owns global nodes node_off[s] .. node_off[s+1]-1;
 *    their LOCAL ids are 0..T_s-1, local 0 is the root (the last committed
 *    token, whose K/V is computed in this pass), parent[i] holds the LOCAL
 *    parent id, parent[0] = -1 and 0 <= parent[i] < i.  1 <= T_s <= 128.
 *  - Paged KV cache: page = EE_PAGE tokens; one layer is laid out
 *    [num_pages][n_kv][EE_PAGE][head_dim]; position t of sequence s lives in
 *    page block_table[s * max_pages + t / EE_PAGE], row t % EE_PAGE.
 *  - `ws` is a caller-owned device workspace of at least
 *    ee_workspace_size(...) bytes, zeroed once with ee_workspace_init() before
 *    first use: a 16.5 KB head (the error word and the LM head's running
 *    argmax), 3.1 MB of LM-head verification partials and thresholds, then the attention's
 *    per-CTA partial results (65 KB per CTA, B x n_q x 16 CTAs at most).
 *    Its first word is the device error word: kernels never trap;
 *    on a bad index found on the device they set an EE_DEVERR_* bit there,
 *    skip the access and continue.  ee_read_errors() reads (and clears) it.
 *    After any error the workspace must be re-initialised.  Calls that share
 *    one workspace must be ordered on one stream.
 *  - Return value: EE_OK when the work was enqueued.  Host-side argument checks
 *    run before any launch and return EE_ERR_INVALID_ARG / EE_ERR_UNSUPPORTED
 *    without touching memory.  EE_ERR_CUDA reports a launch failure.
 */
#ifndef EE_H_
#define EE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define EE_PAGE 16
#define EE_HEAD_DIM 128
#define EE_MAX_TREE 128
#define EE_MAX_NGRAM 32
#define EE_MAX_MATCHES 1024
#define EE_MAX_LM_NODES 2048
#define EE_MAX_CHAIN 2048   /* nodes of one linear draft (long reuse drafts) */

typedef uint16_t ee_bf16;                 /* raw bfloat16 bits */
typedef struct CUstream_st* ee_stream_t;  /* same type as cudaStream_t */

typedef enum {
  EE_OK = 0,
  EE_ERR_INVALID_ARG = 1,   /* null pointer, bad size or alignment */
  EE_ERR_UNSUPPORTED = 2,   /* valid but outside what the kernels support */
  EE_ERR_CUDA = 3,          /* a CUDA call or launch failed */
  EE_ERR_DEVICE = 4,        /* the device error word was set (ee_read_errors) */
  EE_ERR_WORKSPACE = 5      /* ws_bytes smaller than ee_workspace_size() */
} ee_status;

/* Bits of the device error word. */
#define EE_DEVERR_MATCH_ARGS   0x01  /* cursor < 0 or orig_off decreasing */
#define EE_DEVERR_TREE         0x02  /* parent[] violates 0 <= parent[i] < i, or T outside 1..128 */
#define EE_DEVERR_PAGE         0x04  /* block_table entry outside [0, num_pages) for a needed slot */
#define EE_DEVERR_CTX          0x08  /* ctx_len < 0 or above the max_ctx passed by the host */
#define EE_DEVERR_FP16_RANGE   0x10  /* reserved (no current kernel sets it) */
#define EE_DEVERR_TIMEOUT      0x20  /* a bounded device wait gave up */
#define EE_DEVERR_PATH         0x40  /* path / accept_len inconsistent with the tree */
#define EE_DEVERR_OVERFLOW     0x80  /* ee_advance: the committed-token buffer is full */

const char* ee_version(void);
const char* ee_status_string(ee_status s);

/*
 * Workspace bytes needed by every entry point for problems up to these sizes:
 * B sequences, total_nodes tree nodes in all, n_q query heads, max_ctx cached
 * positions in the longest sequence.  The buffer must be 256-byte aligned.
 * 3,219,968 bytes when max_ctx is 0, else 3,219,968 + max(B * n_q * 16, 304)
 * * 66,816 (the attention's partial slots: one per CTA of a split launch, two
 * per resident CTA of a balanced one; about 30 MB for one sequence with 28
 * heads).
 * Returns 0 for negative arguments.
 */
size_t ee_workspace_size(int32_t B, int32_t total_nodes, int32_t n_q, int32_t head_dim,
                         int32_t max_ctx);

/* Zero `ws` (asynchronously, on `stream`).  Call once after allocating it. */
ee_status ee_workspace_init(void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * Synchronise `stream`, copy the device error word to *bits (host pointer),
 * clear it on the device.  Returns EE_ERR_DEVICE when any bit was set.
 */
ee_status ee_read_errors(void* ws, ee_stream_t stream, int32_t* bits);

/*
 * ee_selftest_timeout -- diagnostic of the device-side failure detection (no
 * step of the verification path calls it).  Launches one 64-thread CTA that
 * makes the two kinds of bounded wait the pipelines use run out, without any
 * fault or trap:
 *   (a) warp 0 waits on a shared-memory mbarrier that nothing arrives at; it
 *       gives up after the device wait limit and raises the CTA's abort flag;
 *   (b) warp 1 starts the same kind of wait half a limit later; it must leave
 *       through the abort flag raised by (a), before its own limit;
 *   (c) thread 0 then waits, with acquire loads, for a global counter in the
 *       workspace head that no launch ever writes (the cross-CTA arrival wait
 *       of the attention merge), and gives up after the limit.
 * Then it sets EE_DEVERR_TIMEOUT in the device error word, as every pipeline
 * does after a wait gave up; ee_read_errors() reports and clears it.  The
 * call runs for about two wait limits (2 x 2e9 SM cycles, ~2 s at 2.07 GHz).
 *   out  device int64[7]: [0] the wait limit in SM cycles, [1] result of (a)
 *        (1 = the wait completed, 0 = it gave up), [2] cycles (a) waited,
 *        [3] result of (b), [4] cycles (b) waited, [5] result of (c),
 *        [6] cycles (c) waited.
 * Errors: EE_ERR_INVALID_ARG for a NULL or misaligned ws or out, or ws_bytes
 * below the fixed workspace head.
 */
ee_status ee_selftest_timeout(void* ws, size_t ws_bytes, int64_t* out, ee_stream_t stream);

/*
 * ee_match_reuse -- reuse-span lookup (Sec. III-A, prefix matching that switches
 * Generate back to Reuse).  For each sequence s, with c = orig_tokens[
 * orig_off[s] .. orig_off[s+1]) and t = tail[s*n .. s*n+n) (the last n generated
 * tokens), finds every position p with cursor[s] <= p and p + n < len(c) and
 * c[p+i] == t[i] for all i < n.  The p + n < len(c) rule keeps at least one
 * token of c after the match to serve as draft.
 *   orig_tokens  int32 [orig_off[B]]   original code of all sequences, CSR
 *   orig_off     int64 [B+1]           non-decreasing offsets
 *   tail         int32 [B][n]          1 <= n <= EE_MAX_NGRAM
 *   cursor       int32 [B]             start of the unverified remainder of c
 *   match_pos    int32 [B][max_matches] out: matches in ascending order, -1 pad
 *   n_matches    int32 [B]             out: total number of matches (may exceed
 *                                      max_matches; 1 <= max_matches <= 1024)
 * A long code is scanned by several CTAs whose hits are concatenated through
 * a region of the workspace (tickets that return to zero, per-CTA records);
 * a workspace of ee_workspace_size() bytes holds it, and one of only the fixed
 * head (EE_ERR_WORKSPACE below that) scans each sequence with one CTA.  The
 * results do not depend on the split.
 * Device errors: EE_DEVERR_MATCH_ARGS (that sequence reports 0 matches).
 */
ee_status ee_match_reuse(const int32_t* orig_tokens, const int64_t* orig_off, int32_t B,
                         const int32_t* tail, int32_t n, const int32_t* cursor,
                         int32_t max_matches, int32_t* match_pos, int32_t* n_matches,
                         void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_tree_prepare -- draft-tree structure.  depth[root] = 0, depth[i] =
 * depth[parent[i]] + 1; anc[i] = anc[parent[i]] U {i}, stored as two uint64
 * words per node (bit j of word j/64 = local node j is on the root-to-i path).
 *   parent    int32 [total_nodes]   local parent ids (see conventions)
 *   node_off  int32 [B+1]
 *   depth     int32 [total_nodes]   out
 *   anc       uint64 [total_nodes][2] out
 * Device errors: EE_DEVERR_TREE (that sequence's depth/anc are zeroed).
 */
ee_status ee_tree_prepare(const int32_t* parent, const int32_t* node_off, int32_t B,
                          int32_t total_nodes, int32_t* depth, uint64_t* anc,
                          void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_tree_verify_attn -- tree-masked attention of every draft node, ONE layer
 * (Sec. III-A: one target pass over (prefix, draft)).  Node i of sequence s,
 * query head h, attends to cached positions 0..ctx_len[s]-1 and to the tree
 * nodes in anc[i] (its own root-to-i path):
 *   out[i][h] = sum_j softmax_j(scale * q[i][h] . k_j) v_j,  KV head h / (n_q/n_kv).
 *   q         bf16 [total_nodes][n_q][head_dim]   (post-RoPE)
 *   k_tree    bf16 [total_nodes][n_kv][head_dim]  K/V of the tree nodes, this layer
 *   v_tree    bf16 [total_nodes][n_kv][head_dim]
 *   k_cache   bf16 [num_pages][n_kv][EE_PAGE][head_dim]  this layer's cache
 *   v_cache   bf16 same
 *   block_table int32 [B][max_pages]; ctx_len int32 [B], 0 <= ctx_len <= max_ctx
 *   node_off  int32 [B+1]; anc uint64 [total_nodes][2] from ee_tree_prepare
 *   out       fp32 [total_nodes][n_q][head_dim]   out
 * head_dim must be 128; n_q a multiple of n_kv; max_T <= 128; max_ctx <= 262144;
 * all bf16 arrays 16-byte aligned.  Q.K^T runs on bf16 tensor cores with fp32
 * accumulation in TMEM; P.V runs on bf16 tensor cores with P carried as two
 * bf16 parts (head + tail, about 2^-14 relative) and V as stored; softmax and
 * the output are fp32.  One launch per call, in one of three forms the host
 * picks from the sizes (ee_attn_plan): the context of each 128 query rows is
 * cut into equal chunks, one CTA each, met at a thread-block cluster barrier
 * or (cooperative launch) a counter; or, balanced, one CTA per SM takes an
 * equal share of all row blocks' 128-key tiles, read from the device's
 * ctx_len and node_off (ragged batches, and row-block counts that do not
 * divide the SM count).  Split work writes partial results to slots in `ws`
 * (L2-resident); once a row block's pieces are all written, each of their
 * CTAs merges a share of its rows.  The plan uses only the partial slots the
 * workspace holds: ee_workspace_size(B, total_nodes, n_q, head_dim, max_ctx)
 * bytes admit every plan for trees; a smaller workspace runs a plan with fewer
 * context chunks (one CTA per row block needs none).  EE_ERR_WORKSPACE when
 * ws_bytes is below the fixed head or no plan fits.
 * Device errors: EE_DEVERR_PAGE (the key is skipped), EE_DEVERR_CTX,
 * EE_DEVERR_TIMEOUT (outputs undefined).
 */
ee_status ee_tree_verify_attn(const ee_bf16* q, const ee_bf16* k_tree, const ee_bf16* v_tree,
                              const ee_bf16* k_cache, const ee_bf16* v_cache, int32_t num_pages,
                              const int32_t* block_table, int32_t max_pages, const int32_t* ctx_len,
                              int32_t max_ctx, const int32_t* node_off, const uint64_t* anc,
                              int32_t B, int32_t total_nodes, int32_t max_T, int32_t n_q,
                              int32_t n_kv, int32_t head_dim, float scale, float* out,
                              void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_tree_verify_attn_inplace -- the same attention when the tree's K/V are
 * already in the cache (in-place speculative K/V): node i of sequence s
 * (local id i) has its keys and values at position ctx_len[s] + i of its
 * pages, where the target's K/V projection wrote them, instead of in
 * k_tree / v_tree.  A node attends to positions 0 .. ctx - 1 and to positions
 * ctx + j for every ancestor j in anc (itself included): out is the same as
 * ee_tree_verify_attn's with k_tree / v_tree read from those positions (Sec.
 * III-A; the paper has no separate tree buffer either).  block_table must hold
 * a page for every position below ctx_len + T: max_ctx + max_T <=
 * max_pages * EE_PAGE (else EE_ERR_INVALID_ARG), and a missing page sets
 * EE_DEVERR_PAGE with its keys skipped.  Other arguments, layouts, precision
 * and errors as ee_tree_verify_attn.  Pair it with ee_kv_compact_inplace.
 */
ee_status ee_tree_verify_attn_inplace(const ee_bf16* q, const ee_bf16* k_cache, const ee_bf16* v_cache,
                                      int32_t num_pages, const int32_t* block_table, int32_t max_pages,
                                      const int32_t* ctx_len, int32_t max_ctx, const int32_t* node_off,
                                      const uint64_t* anc, int32_t B, int32_t total_nodes, int32_t max_T,
                                      int32_t n_q, int32_t n_kv, int32_t head_dim, float scale, float* out,
                                      void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_lmhead_verify -- the LM head with the verification rules the paper
 * compares (Sec. V-C, RQ3), including its entropy-aware dynamic verification
 * (Sec. III-B, Eq. (entropy) and the top_tau rule).  Same inputs, argmax,
 * path, accept_len and bonus as ee_lmhead_accept; what differs is how the edge
 * a -> b (b drafted after a) of edit content is judged on the target
 * distribution at a:
 *   EE_VERIFY_GREEDY   draft_tok[b] is the target's most probable token;
 *   EE_VERIFY_DIRECT   accepted without verification;
 *   EE_VERIFY_TOPK     draft_tok[b] is among the target's k most probable;
 *   EE_VERIFY_ENTROPY  draft_tok[b] is among the first top_tau of them, where
 *                      H_norm = -sum_{i<=k} p_i ln p_i / ln k over the k
 *                      largest probabilities p_i of the full-vocabulary
 *                      softmax (not renormalised) and top_tau =
 *                      max(1, ceil(k * H_norm)), at most k.
 * Probabilities rank by logit, lower token id first among equal logits.
 * gen_mask_or_null uint8 [total_nodes]: 1 = edit content (the mode's rule),
 * 0 = reused code (always greedy, as the paper verifies the Reuse phase);
 * NULL = every node is edit content.  k: 1..8 (2..8 for ENTROPY; unused by
 * GREEDY and DIRECT except as the length of topk_ids).
 * Optional outputs (NULL to skip): topk_ids int32 [total_nodes][k] ranked
 * token ids; top_tau int32 [total_nodes] the number of leading ranks an edit
 * child may hold (greedy 1, top-k k, entropy top_tau, direct 0 = any);
 * h_norm fp32 [total_nodes] (0 when k = 1).  Logits, the log-sum-exp and
 * H_norm are fp32.  The workspace must hold ee_workspace_size(...) bytes
 * (per-CTA partials of the top-k lists live there).  EE_ERR_INVALID_ARG for a
 * bad mode or k; otherwise as ee_lmhead_accept.
 */
typedef enum {
  EE_VERIFY_GREEDY = 0,
  EE_VERIFY_DIRECT = 1,
  EE_VERIFY_TOPK = 2,
  EE_VERIFY_ENTROPY = 3
} ee_verify_mode;

ee_status ee_lmhead_verify(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                           int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                           const int32_t* depth, const uint64_t* anc, const int32_t* node_off,
                           const uint8_t* gen_mask_or_null, int32_t B, int32_t total_nodes,
                           int32_t max_T, int32_t mode, int32_t k, int32_t* argmax,
                           int32_t* topk_ids_or_null, int32_t* top_tau_or_null,
                           float* h_norm_or_null, int32_t* accept_len, int32_t* path,
                           int32_t* bonus, float* logits_or_null, void* ws, size_t ws_bytes,
                           ee_stream_t stream);

/*
 * ee_attn_plan -- the launch plan ee_tree_verify_attn (inplace = 0),
 * ee_tree_verify_attn_inplace (inplace = 1) or ee_chain_verify_attn
 * (inplace = 2, max_T up to EE_MAX_CHAIN) uses for these sizes
 * (introspection only; the paper has no counterpart).  *splits = context
 * chunks per 128 query rows (1..16), *chunk = keys per chunk, *mode = 0
 * (one chunk, no merge), 1 (chunks of a row block form a thread-block
 * cluster) or 2 (cooperative launch, merge counters in the workspace),
 * *ctas = CTAs launched.  Mode 3 (balanced, cooperative, one CTA per SM):
 * *splits = CTAs that share the work at most, *chunk = keys per CTA when
 * every sequence holds max_ctx positions and max_T nodes.  Needs the device (occupancy queries): EE_ERR_CUDA
 * without one; EE_ERR_INVALID_ARG for sizes ee_tree_verify_attn rejects.
 */
ee_status ee_attn_plan(int32_t B, int32_t max_T, int32_t n_q, int32_t n_kv, int32_t max_ctx,
                       int32_t inplace, int32_t* splits, int32_t* chunk, int32_t* mode, int32_t* ctas);

/*
 * ee_lmhead_accept -- LM head fused with greedy decode and acceptance
 * (Eq. (piecewise)).  logits[i][v] = hidden[i] . lm_w[v] (fp32 accumulate of
 * bf16 products, never stored unless logits_or_null is given);
 * argmax[i] = the highest logit, lowest token id on ties.  Node i (i > 0) is
 * accepted when every edge a -> b on its root path has draft_tok[b] ==
 * argmax[a]; the deepest accepted node u* wins (lowest local id among equally
 * deep ones):
 *   accept_len[s] = depth[u*]   (draft tokens accepted, root excluded)
 *   path[s][0..accept_len]      local ids root -> u*, rest of the row -1
 *   bonus[s] = argmax[u*]       the target's next token after the accepted path
 *   hidden    bf16 [total_nodes][hidden_dim]
 *   lm_w      bf16 [vocab][hidden_dim]  (vocab-major)
 *   draft_tok int32 [total_nodes]; parent int32 [total_nodes];
 *   depth int32 / anc uint64[2] from ee_tree_prepare; node_off int32 [B+1]
 *   argmax int32 [total_nodes]; accept_len/bonus int32 [B]; path int32 [B][max_T]
 *   logits_or_null fp32 [total_nodes][vocab] or NULL
 * hidden_dim a multiple of 8; total_nodes <= EE_MAX_LM_NODES; hidden and lm_w
 * 16-byte aligned.  Runs as one persistent tcgen05/TMEM GEMM (vocab rows on
 * the MMA M side) whose epilogue keeps the running argmax; the last CTA to
 * finish runs the acceptance.
 * Linear drafts (long reuse drafts, Sec. III-A): with anc == NULL every
 * sequence is a chain (node i's parent is i - 1; parent and depth may be
 * NULL) of up to EE_MAX_CHAIN nodes (max_T <= EE_MAX_CHAIN): accept_len[s] is
 * the largest j with draft_tok[i] == argmax[i - 1] for all 1 <= i <= j, path
 * is 0 .. j.
 * Device errors: EE_DEVERR_TIMEOUT (outputs undefined).
 */
ee_status ee_lmhead_accept(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                           int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                           const int32_t* depth, const uint64_t* anc, const int32_t* node_off,
                           int32_t B, int32_t total_nodes, int32_t max_T, int32_t* argmax,
                           int32_t* accept_len, int32_t* path, int32_t* bonus,
                           float* logits_or_null, void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_lmhead_accept_static -- ee_lmhead_accept for callers that cannot allocate
 * device memory.  The paper has no counterpart; this is a deployment variant.
 * Some callers have no way to obtain the workspace the other entry points
 * take: code running where cudaMalloc is unavailable or forbidden (host
 * callbacks, a custom allocator's own hooks, processes under a fixed device
 * memory budget).  This entry point takes the same inputs and outputs as
 * ee_lmhead_accept but no `ws`: its scratch lives in a file-scope device array
 * of 16,640 bytes inside libee, which every GPU that loads the library holds
 * until the process exits.  It allocates nothing (no cudaMalloc/cudaFree, no
 * allocating library call).
 *  - total_nodes above EE_MAX_LM_NODES (2048) is rejected with
 *    EE_ERR_UNSUPPORTED; the other argument checks are those of
 *    ee_lmhead_accept.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture.  The array used is the current device's, so
 *    `stream` must belong to the current device (NULL: the current device's
 *    legacy stream); a stream of another device is rejected with
 *    EE_ERR_INVALID_ARG.
 *  - Every call clears the array on `stream` before its launch, because the
 *    array keeps the previous call's contents.  All calls share the one array:
 *    calls that overlap on the GPU (different streams without ordering, or
 *    different host threads) race and corrupt each other's results.
 *  - Device-side failures (the bounded-wait timeout) are recorded only in the
 *    array's own error word, which this entry point does not report; outputs
 *    are then undefined.  Use ee_lmhead_accept with a workspace and
 *    ee_read_errors when that report is needed.
 */
ee_status ee_lmhead_accept_static(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                                  int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                                  const int32_t* depth, const uint64_t* anc, const int32_t* node_off,
                                  int32_t B, int32_t total_nodes, int32_t max_T, int32_t* argmax,
                                  int32_t* accept_len, int32_t* path, int32_t* bonus,
                                  float* logits_or_null, ee_stream_t stream);

/*
 * ee_lmhead_pack_weights -- rearrange the LM-head weights once (at model load:
 * a deployment layout, the paper has no counterpart) into the order the LM
 * head streams them: W is cut into blocks of 128 vocabulary rows x 64 hidden
 * columns, block (vt, kb) = rows 128 vt .. 128 vt + 127, columns 64 kb ..
 * 64 kb + 63, stored row-major as one contiguous 16 KB run at element offset
 * (vt * ceil(hidden_dim / 64) + kb) * 8192; rows past vocab and columns past
 * hidden_dim are zero.  The LM head then reads whole 16 KB runs instead of
 * 128-byte pieces 2 * hidden_dim bytes apart (measured: the 7B-shaped LM head
 * 168 -> 161 us on one GB300).
 *   lm_w   bf16 [vocab][hidden_dim] row-major, in
 *   packed bf16, ee_lmhead_packed_bytes(vocab, hidden_dim) bytes, out
 * hidden_dim a multiple of 8; both arrays 16-byte aligned; packed_bytes at
 * least ee_lmhead_packed_bytes(...).  One kernel launch on `stream`.
 * ee_lmhead_packed_bytes returns 0 for sizes the packing does not take.
 */
size_t ee_lmhead_packed_bytes(int32_t vocab, int32_t hidden_dim);
ee_status ee_lmhead_pack_weights(const ee_bf16* lm_w, int32_t vocab, int32_t hidden_dim, ee_bf16* packed,
                                 size_t packed_bytes, ee_stream_t stream);

/*
 * ee_lmhead_accept_packed -- ee_lmhead_accept (same arguments, results and
 * errors) with the weights in the layout ee_lmhead_pack_weights writes:
 * lm_w_packed is that array for the same vocab and hidden_dim.  The products
 * are the same sums in the same order: argmax, path, accept_len, bonus and the
 * optional logits are bit-identical to ee_lmhead_accept's.
 */
ee_status ee_lmhead_accept_packed(const ee_bf16* hidden, const ee_bf16* lm_w_packed, int32_t hidden_dim,
                                  int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                                  const int32_t* depth, const uint64_t* anc, const int32_t* node_off,
                                  int32_t B, int32_t total_nodes, int32_t max_T, int32_t* argmax,
                                  int32_t* accept_len, int32_t* path, int32_t* bonus,
                                  float* logits_or_null, void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_kv_compact -- append the accepted path's K/V to the paged cache, every
 * layer (Sec. III-A: accepted tokens extend the prefix).  Path entry k
 * (k = 0..accept_len[s], root first) of sequence s goes to position
 * ctx_len_in[s] + k; ctx_len_out[s] = ctx_len_in[s] + accept_len[s] + 1.
 *   k_tree/v_tree  bf16, layer l at + l*tree_layer_stride elements, each layer
 *                  [total_nodes][n_kv][head_dim]
 *   k_cache/v_cache bf16, layer l at + l*cache_layer_stride elements, each layer
 *                  [num_pages][n_kv][EE_PAGE][head_dim]
 *   path int32 [B][max_T], accept_len int32 [B] (from ee_lmhead_accept);
 *                  max_T <= EE_MAX_CHAIN (linear drafts)
 *   dst_slot int32 [B][max_T] out: page*EE_PAGE + row of each appended entry, -1 pad
 *   ctx_len_out must not alias ctx_len_in.
 * Device errors: EE_DEVERR_PAGE (entry skipped), EE_DEVERR_PATH.
 */
ee_status ee_kv_compact(const ee_bf16* k_tree, const ee_bf16* v_tree, int64_t tree_layer_stride,
                        ee_bf16* k_cache, ee_bf16* v_cache, int64_t cache_layer_stride, int32_t L,
                        int32_t num_pages, const int32_t* block_table, int32_t max_pages,
                        const int32_t* ctx_len_in, int32_t* ctx_len_out, const int32_t* node_off,
                        const int32_t* path, const int32_t* accept_len, int32_t B, int32_t max_T,
                        int32_t n_kv, int32_t head_dim, int32_t* dst_slot,
                        void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_chain_verify_attn -- attention of linear drafts verified in place (long
 * reuse drafts: the paper verifies a long span of the original code in one
 * pass, Sec. III-A).  Sequence s's draft of T_s <= EE_MAX_CHAIN tokens has its
 * K/V at cache positions ctx .. ctx + T_s - 1 and draft token i (node i)
 * attends to positions 0 .. ctx + i: ordinary causal attention over prefix +
 * draft, out[i][h] = sum_j softmax_j(scale * q[i][h] . k_j) v_j.  Query rows
 * past a row block's last node never see later keys, so a row block's work
 * ends at its own last position (causal tile skipping).  block_table must
 * cover max_ctx + max_T positions (else EE_ERR_INVALID_ARG); max_T <=
 * EE_MAX_CHAIN.  Arguments, layouts, precision and device errors as
 * ee_tree_verify_attn_inplace without anc.  Pair it with ee_lmhead_accept
 * (anc NULL) and ee_kv_compact_inplace (nothing moves).
 */
ee_status ee_chain_verify_attn(const ee_bf16* q, const ee_bf16* k_cache, const ee_bf16* v_cache,
                               int32_t num_pages, const int32_t* block_table, int32_t max_pages,
                               const int32_t* ctx_len, int32_t max_ctx, const int32_t* node_off, int32_t B,
                               int32_t total_nodes, int32_t max_T, int32_t n_q, int32_t n_kv,
                               int32_t head_dim, float scale, float* out, void* ws, size_t ws_bytes,
                               ee_stream_t stream);

/*
 * ee_build_reuse_tree -- the next step's draft tree on the device (Sec. III-A:
 * match points of the generated suffix in the remaining code are new draft
 * starts, the code after each is a draft).  Every sequence gets
 * T = 1 + n_branches * chain_len + gen_len <= EE_MAX_TREE nodes:
 *   node 0            root: last_tok[s], the last committed token;
 *   nodes 1 + b*chain_len + j  (b < n_branches, j < chain_len)
 *                     branch b, a chain below the root: c[match_pos[s][b] + n + j]
 *                     for b < min(n_matches[s], max_matches); -1 for an absent
 *                     match and past the end of c (never accepted);
 *   last gen_len nodes a chain below the root: gen_tok[s][0 .. gen_len), a
 *                     draft model's proposal for edited content (gen_mask 1).
 *   orig_tokens/orig_off as ee_match_reuse; match_pos int32 [B][max_matches],
 *   n_matches int32 [B] (from ee_match_reuse); last_tok int32 [B];
 *   gen_tok int32 [B][gen_len] or NULL when gen_len == 0.
 *   Outputs: draft_tok, parent (local ids), cpos (position in c of the token,
 *   the root's = match_pos[s][0] + n - 1, -1 for generated or empty nodes)
 *   int32 [B*T]; node_off int32 [B+1] = s*T; gen_mask uint8 [B*T].
 * Device errors: EE_DEVERR_MATCH_ARGS (a negative match position: its branch
 * stays empty).
 */
ee_status ee_build_reuse_tree(const int32_t* orig_tokens, const int64_t* orig_off, int32_t B,
                              const int32_t* match_pos, const int32_t* n_matches, int32_t max_matches,
                              const int32_t* last_tok, int32_t n, int32_t chain_len, int32_t n_branches,
                              const int32_t* gen_tok_or_null, int32_t gen_len, int32_t* draft_tok,
                              int32_t* parent, int32_t* node_off, int32_t* cpos, uint8_t* gen_mask,
                              void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_advance -- commit one verification step on the device (Sec. III-A).  The
 * accepted draft tokens (path nodes 1 .. accept_len; the root was committed
 * before) and the bonus token are appended to the generated sequence
 * out_tok[s][0 .. out_len[s]); then tail[s] = its last n tokens, last_tok[s] =
 * bonus[s], and, when the last accepted node came from the code (cpos q >= 0),
 * cursor[s] = q + 1: the code up to q is consumed and the rest stays the
 * candidate draft; otherwise cursor[s] is unchanged.
 *   out_tok int32 [B][cap], out_len int32 [B] (in/out, out_len >= n after
 *   the commit); draft_tok / cpos / node_off from ee_build_reuse_tree (or any
 *   tree with T <= EE_MAX_TREE); path / accept_len / bonus from the LM head;
 *   tail int32 [B][n], cursor, last_tok int32 [B] (out; cursor in/out).
 * Device errors: EE_DEVERR_PATH (bad path or accept_len), EE_DEVERR_OVERFLOW
 * (out_tok has no room); the sequence is then left unchanged.
 */
ee_status ee_advance(int32_t* out_tok, int32_t* out_len, int32_t cap, const int32_t* draft_tok,
                     const int32_t* cpos, const int32_t* node_off, const int32_t* path,
                     const int32_t* accept_len, const int32_t* bonus, int32_t B, int32_t total_nodes,
                     int32_t max_T, int32_t n, int32_t* tail, int32_t* cursor, int32_t* last_tok,
                     void* ws, size_t ws_bytes, ee_stream_t stream);

/*
 * ee_kv_compact_inplace -- ee_kv_compact's result when the tree's K/V already
 * sit at positions ctx_len_in[s] + i (in-place speculative K/V, see
 * ee_tree_verify_attn_inplace).  Path entry k is node path[k] >= k (a parent's
 * id is below its child's): entries with path[k] == k are already in place --
 * every entry of a reuse chain -- and the others move from position
 * ctx + path[k] down to ctx + k, every layer.  Positions after ctx + accept_len
 * keep the rejected nodes' K/V (they lie beyond the new ctx_len).
 *   k_cache/v_cache bf16, layer l at + l*cache_layer_stride elements, each layer
 *                   [num_pages][n_kv][EE_PAGE][head_dim]
 *   node_off int32 [B+1] with node_off[B] <= total_nodes; path, accept_len,
 *   dst_slot, ctx_len_in / ctx_len_out as ee_kv_compact.  Entries from
 *   EE_MAX_TREE on (linear drafts only) must be in place.
 * HBM traffic: 2 (K, V) x 2 (read, write) x n_kv x 256 bytes per moved entry
 * and layer; a chain moves nothing.
 * Device errors: EE_DEVERR_PATH (path[k] < k or >= T, or a bad accept_len:
 * the sequence is skipped), EE_DEVERR_PAGE (a missing page for a moved entry:
 * the sequence is skipped).
 */
ee_status ee_kv_compact_inplace(ee_bf16* k_cache, ee_bf16* v_cache, int64_t cache_layer_stride, int32_t L,
                                int32_t num_pages, const int32_t* block_table, int32_t max_pages,
                                const int32_t* ctx_len_in, int32_t* ctx_len_out, const int32_t* node_off,
                                const int32_t* path, const int32_t* accept_len, int32_t B,
                                int32_t total_nodes, int32_t max_T, int32_t n_kv, int32_t head_dim,
                                int32_t* dst_slot, void* ws, size_t ws_bytes, ee_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* EE_H_ */
