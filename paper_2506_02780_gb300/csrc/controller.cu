// The Reuse <-> Generate controller on the device (EfficientEdit Sec. III-A):
// between two verification steps, the next draft tree is built from the match
// points of the generated suffix in the remaining original code, and the
// step's result is committed.  With both on the device a whole edit session
// runs as a loop of captured steps, without the host between them.
//
//   ee_build_reuse_tree  root = the last committed token; one reuse chain of
//                        chain_len code tokens after each match point (up to
//                        n_branches); then a generated branch (a draft model's
//                        proposal).  Fixed T nodes per sequence.
//   ee_advance           accepted draft tokens + the bonus token extend the
//                        generated sequence; the tail, the cursor (start of
//                        the code not yet verified) and the root follow.
//
// Both are small integer kernels: one CTA per sequence, one thread per tree
// node (or path entry).  They start before their predecessor ends
// (programmatic dependent launch) and read its outputs only after the wait,
// with plain loads.
#include "ee_common.cuh"

namespace {

constexpr int kThreads = EE_MAX_TREE;   // one thread per node of a tree

__global__ void __launch_bounds__(kThreads)
build_reuse_tree_kernel(const int32_t* orig_tokens, const int64_t* orig_off, const int32_t* match_pos,
                        const int32_t* n_matches, int max_matches, const int32_t* last_tok, int n,
                        int chain_len, int n_branches, const int32_t* gen_tok, int gen_len, int T,
                        int32_t* draft_tok, int32_t* parent, int32_t* node_off, int32_t* cpos,
                        uint8_t* gen_mask, int B, int32_t* err) {
  ee::pdl_allow_next();
  ee::pdl_wait();   // match points and the last committed token are complete
  const int s = blockIdx.x;
  const int i = threadIdx.x;
  if (i >= T) return;
  const int64_t c0 = orig_off[s], c1 = orig_off[s + 1];
  const int nm = min(max(n_matches[s], 0), max_matches);
  const size_t o = (size_t)s * T;
  int tok = -1, par = -1, cp = -1;
  uint8_t gm = 0;
  if (i == 0) {
    tok = last_tok[s];
    if (nm > 0) cp = match_pos[(size_t)s * max_matches] + n - 1;
    node_off[s] = (int32_t)o;
    if (s == B - 1) node_off[B] = (int32_t)(o + T);
  } else if (i <= n_branches * chain_len) {
    const int b = (i - 1) / chain_len, j = (i - 1) - b * chain_len;
    par = j == 0 ? 0 : i - 1;
    if (b < nm) {
      const int p = match_pos[(size_t)s * max_matches + b];
      const int64_t q = (int64_t)p + n + j;
      if (p < 0 || c1 < c0) {
        if (j == 0) ee::flag_error(err, EE_DEVERR_MATCH_ARGS);
      } else if (q < c1 - c0) {
        tok = orig_tokens[c0 + q];
        cp = (int)q;
      }
    }
  } else {
    const int j = i - 1 - n_branches * chain_len;
    par = j == 0 ? 0 : i - 1;
    tok = gen_tok[(size_t)s * gen_len + j];
    gm = 1;
  }
  draft_tok[o + i] = tok;
  parent[o + i] = par;
  cpos[o + i] = cp;
  gen_mask[o + i] = gm;
}

__global__ void __launch_bounds__(kThreads)
advance_kernel(int32_t* out_tok, int32_t* out_len, int cap, const int32_t* draft_tok, const int32_t* cpos,
               const int32_t* node_off, const int32_t* path, const int32_t* accept_len, const int32_t* bonus,
               int max_T, int total_nodes, int n, int32_t* tail, int32_t* cursor, int32_t* last_tok,
               int32_t* err) {
  ee::pdl_allow_next();
  ee::pdl_wait();   // the acceptance's path, accept_len and bonus are complete
  const int s = blockIdx.x;
  const int k = threadIdx.x;
  const int o = node_off[s];
  const int T = node_off[s + 1] - o;
  const int a = accept_len[s];
  const int L = out_len[s];
  const bool seq_ok = T >= 1 && T <= EE_MAX_TREE && o >= 0 && o + T <= total_nodes && a >= 0 && a < T &&
                      a < max_T && L >= 0;
  const bool room = seq_ok && L + a + 1 <= cap && L + a + 1 >= n;
  // path entry k (1 <= k <= a) is committed at L + k - 1, the bonus at L + a
  int node = 0;
  bool bad = false;
  if (seq_ok && k <= a) {
    node = path[(size_t)s * max_T + k];
    bad = node < 0 || node >= T;
  }
  bad = __syncthreads_or(bad);
  if (k == 0) {
    if (!seq_ok || bad) ee::flag_error(err, EE_DEVERR_PATH);
    else if (!room) ee::flag_error(err, EE_DEVERR_OVERFLOW);
  }
  if (!seq_ok || bad || !room) return;     // nothing is committed
  int32_t* row = out_tok + (size_t)s * cap;
  if (k >= 1 && k <= a) row[L + k - 1] = draft_tok[o + node];
  if (k == 0) row[L + a] = bonus[s];
  __syncthreads();                          // the tail reads what was just written
  const int L2 = L + a + 1;
  if (k < n) tail[(size_t)s * n + k] = row[L2 - n + k];
  if (k == a) {                             // the last accepted node
    const int q = cpos[o + node];
    if (q >= 0) cursor[s] = q + 1;
  }
  if (k == 0) {
    out_len[s] = L2;
    last_tok[s] = bonus[s];
  }
}

}  // namespace

extern "C" ee_status ee_build_reuse_tree(const int32_t* orig_tokens, const int64_t* orig_off, int32_t B,
                                         const int32_t* match_pos, const int32_t* n_matches, int32_t max_matches,
                                         const int32_t* last_tok, int32_t n, int32_t chain_len, int32_t n_branches,
                                         const int32_t* gen_tok_or_null, int32_t gen_len, int32_t* draft_tok,
                                         int32_t* parent, int32_t* node_off, int32_t* cpos, uint8_t* gen_mask,
                                         void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (B < 0 || max_matches < 1 || max_matches > EE_MAX_MATCHES || n < 1 || n > EE_MAX_NGRAM || chain_len < 1 ||
      n_branches < 0 || gen_len < 0 || (gen_len > 0 && !gen_tok_or_null))
    return EE_ERR_INVALID_ARG;
  const int64_t T = 1 + (int64_t)n_branches * chain_len + gen_len;
  if (T > EE_MAX_TREE) return EE_ERR_UNSUPPORTED;
  if (B == 0) return EE_OK;
  if (!orig_tokens || !orig_off || !match_pos || !n_matches || !last_tok || !draft_tok || !parent || !node_off ||
      !cpos || !gen_mask || !ws)
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  EE_CUDA_OK(ee::launch_pdl(build_reuse_tree_kernel, dim3(B), dim3(kThreads), 0, (cudaStream_t)stream, 1,
                            orig_tokens, orig_off, match_pos, n_matches, (int)max_matches, last_tok, (int)n,
                            (int)chain_len, (int)n_branches, gen_tok_or_null, (int)gen_len, (int)T, draft_tok,
                            parent, node_off, cpos, gen_mask, (int)B, ee::err_word(ws)));
  return EE_OK;
}

extern "C" ee_status ee_advance(int32_t* out_tok, int32_t* out_len, int32_t cap, const int32_t* draft_tok,
                                const int32_t* cpos, const int32_t* node_off, const int32_t* path,
                                const int32_t* accept_len, const int32_t* bonus, int32_t B, int32_t total_nodes,
                                int32_t max_T, int32_t n, int32_t* tail, int32_t* cursor, int32_t* last_tok,
                                void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (B < 0 || cap < 1 || total_nodes < 0 || max_T < 1 || max_T > EE_MAX_TREE || n < 1 || n > EE_MAX_NGRAM)
    return EE_ERR_INVALID_ARG;
  if (B == 0) return EE_OK;
  if (!out_tok || !out_len || !draft_tok || !cpos || !node_off || !path || !accept_len || !bonus || !tail ||
      !cursor || !last_tok || !ws)
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  EE_CUDA_OK(ee::launch_pdl(advance_kernel, dim3(B), dim3(kThreads), 0, (cudaStream_t)stream, 1, out_tok, out_len,
                            (int)cap, draft_tok, cpos, node_off, path, accept_len, bonus, (int)max_T,
                            (int)total_nodes, (int)n, tail, cursor, last_tok, ee::err_word(ws)));
  return EE_OK;
}
