// ee_match_reuse: reuse-span lookup of the last n generated tokens in the
// original code (EfficientEdit Sec. III-A, prefix matching that switches the
// Generate phase back to Reuse).
//
// One CTA per sequence scans the positions p >= cursor in tiles of
// kTile = 4096: the tile plus an (n-1)-token halo is staged in shared memory
// with coalesced loads, each thread tests 8 consecutive positions against the
// n-token tail, and a block-wide exclusive scan of the per-thread hit counts
// writes the hits in ascending order.  Integer compares only; the kernel is
// bound by reading c once from HBM (4 bytes per position).
#include "ee_common.cuh"

namespace {

constexpr int kThreads = 512;
constexpr int kPer = 8;
constexpr int kTile = kThreads * kPer;
constexpr int kWarps = kThreads / 32;

__global__ void __launch_bounds__(kThreads)
match_reuse_kernel(const int32_t* __restrict__ tok, const int64_t* off, const int32_t* tail, int n,
                   const int32_t* cursor, int max_matches, int32_t* match_pos, int32_t* n_matches,
                   int32_t* err) {
  // tok (the original code) is read-only data for the whole run; the per-step
  // inputs (off, tail, cursor) may come from an earlier kernel and are read
  // with plain loads after the dependent-launch wait (a const __restrict__
  // load may be treated as invariant and issued before the wait)
  __shared__ int32_t s_c[kTile + EE_MAX_NGRAM];
  __shared__ int32_t s_tail[EE_MAX_NGRAM];
  __shared__ int32_t s_wtot[kWarps];
  __shared__ int32_t s_wexcl[kWarps];
  __shared__ int32_t s_tile_total;
  ee::pdl_allow_next();
  ee::pdl_wait();   // no global access before the previous kernel's writes are visible
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;

  for (int i = tid; i < max_matches; i += kThreads) match_pos[(size_t)b * max_matches + i] = -1;
  const int64_t o0 = off[b], o1 = off[b + 1];
  const int cur = cursor[b];
  if (o1 < o0 || cur < 0 || o1 - o0 > INT32_MAX) {
    if (tid == 0) {
      ee::flag_error(err, EE_DEVERR_MATCH_ARGS);
      n_matches[b] = 0;
    }
    return;
  }
  const int len = (int)(o1 - o0);
  const int p_end = len - n;  // valid p satisfy cur <= p < p_end  (p + n < len)
  if (tid < n) s_tail[tid] = tail[(size_t)b * n + tid];
  const int32_t* c = tok + o0;

  int total = 0;  // block-uniform running count
  for (int base = cur; base < p_end; base += kTile) {
    __syncthreads();  // previous tile's readers are done
    const int span = min(kTile + n - 1, len - base);
    for (int i = tid; i < span; i += kThreads) s_c[i] = __ldg(c + base + i);
    __syncthreads();

    unsigned hits = 0;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int pl = tid * kPer + k;
      if (base + pl < p_end) {
        bool ok = true;
        for (int j = 0; j < n; ++j) ok &= (s_c[pl + j] == s_tail[j]);
        hits |= (unsigned)ok << k;
      }
    }
    // block-wide exclusive scan of the per-thread hit counts
    const int cnt = __popc(hits);
    int incl = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      int v = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += v;
    }
    if (lane == 31) s_wtot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const int v = lane < kWarps ? s_wtot[lane] : 0;
      int w = v;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        int u = __shfl_up_sync(0xffffffffu, w, d);
        if (lane >= d) w += u;
      }
      if (lane < kWarps) s_wexcl[lane] = w - v;
      if (lane == kWarps - 1) s_tile_total = w;
    }
    __syncthreads();
    int idx = total + s_wexcl[warp] + incl - cnt;
    unsigned h = hits;
    while (h) {
      const int k = __ffs(h) - 1;
      h &= h - 1;
      if (idx < max_matches) match_pos[(size_t)b * max_matches + idx] = base + tid * kPer + k;
      ++idx;
    }
    total += s_tile_total;
  }
  if (tid == 0) n_matches[b] = total;
}

}  // namespace

extern "C" ee_status ee_match_reuse(const int32_t* orig_tokens, const int64_t* orig_off, int32_t B,
                                    const int32_t* tail, int32_t n, const int32_t* cursor,
                                    int32_t max_matches, int32_t* match_pos, int32_t* n_matches,
                                    void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (B < 0 || n < 1 || n > EE_MAX_NGRAM || max_matches < 1 || max_matches > EE_MAX_MATCHES)
    return EE_ERR_INVALID_ARG;
  if (B == 0) return EE_OK;
  if (!orig_tokens || !orig_off || !tail || !cursor || !match_pos || !n_matches || !ws)
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  EE_CUDA_OK(ee::launch_pdl(match_reuse_kernel, dim3(B), dim3(kThreads), 0, (cudaStream_t)stream, 1,
                             orig_tokens, orig_off, tail, n, cursor, max_matches, match_pos,
                             n_matches, ee::err_word(ws)));
  return EE_OK;
}
