// ee_match_reuse: reuse-span lookup of the last n generated tokens in the
// original code (EfficientEdit Sec. III-A, prefix matching that switches the
// Generate phase back to Reuse).
//
// The positions p >= cursor of a sequence are split into G contiguous ranges,
// one CTA each (G = the launch's grid.x, fewer for a short sequence: at least
// kMinPer positions a CTA).  A CTA scans its range in tiles of kTile = 4096:
// the tile plus an (n-1)-token halo is staged in shared memory with coalesced
// loads (the next tile's loads are issued before the current tile is
// compared), each thread tests 8 consecutive positions against the n-token
// tail, and a block-wide exclusive scan of the per-thread hit counts orders
// the hits.  With G = 1 the CTA writes the outputs directly; otherwise it writes
// its count and first max_matches hits to a workspace record, and the CTA that
// finishes last (a ticket counter taken with one acquire-release add after the
// CTA barrier: nobody waits, no separate fences) concatenates the records in
// range order.  Integer compares only; bound by reading c once (4 bytes per
// position) and, for short codes, by launch latency.
#include "ee_common.cuh"
#include "ee_ptx.cuh"

namespace {

constexpr int kThreads = 512;
constexpr int kPer = 8;
constexpr int kTile = kThreads * kPer;
constexpr int kWarps = kThreads / 32;
constexpr int kMinPer = kTile;        // fewest positions worth a CTA of their own
constexpr int kMaxSplit = 32;         // CTAs per sequence (the merge is one warp wide)
constexpr int kHalo = EE_MAX_NGRAM;

__host__ __device__ inline size_t match_rec_bytes(int max_matches) {
  return ee::align_up(4 * (size_t)(1 + max_matches), 16);
}
__host__ __device__ inline size_t match_seq_bytes(int G, int max_matches) {
  return 16 + (size_t)G * match_rec_bytes(max_matches);
}

__global__ void __launch_bounds__(kThreads)
match_reuse_kernel(const int32_t* __restrict__ tok, const int64_t* off, const int32_t* tail, int n,
                   const int32_t* cursor, int max_matches, int32_t* match_pos, int32_t* n_matches,
                   uint8_t* mws, int32_t* err) {
  // tok (the original code) is read-only data for the whole run; the per-step
  // inputs (off, tail, cursor) may come from an earlier kernel and are read
  // with plain loads after the dependent-launch wait (a const __restrict__
  // load may be treated as invariant and issued before the wait)
  __shared__ __align__(16) int32_t s_c[kTile + kHalo];
  __shared__ int32_t s_tail[EE_MAX_NGRAM];
  __shared__ int32_t s_wtot[kWarps];
  __shared__ int32_t s_wexcl[kWarps];
  __shared__ int32_t s_tile_total;
  __shared__ int s_last;
  ee::pdl_allow_next();
  ee::pdl_wait();   // no global access before the previous kernel's writes are visible
  const int b = blockIdx.x;
  const int g = blockIdx.y, Gl = gridDim.y;
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;

  const int64_t o0 = off[b], o1 = off[b + 1];
  const int cur = cursor[b];
  if (o1 < o0 || cur < 0 || o1 - o0 > INT32_MAX) {
    if (g == 0) {
      for (int i = tid; i < max_matches; i += kThreads) match_pos[(size_t)b * max_matches + i] = -1;
      if (tid == 0) {
        ee::flag_error(err, EE_DEVERR_MATCH_ARGS);
        n_matches[b] = 0;
      }
    }
    return;
  }
  const int len = (int)(o1 - o0);
  const int p_end = len - n;  // valid p satisfy cur <= p < p_end  (p + n < len)
  const int npos = max(p_end - cur, 0);
  // this sequence's CTAs and this CTA's range [r0, r1) (a multiple of kPer long)
  const int G = max(1, min(Gl, (npos + kMinPer - 1) / kMinPer));
  if (g >= G) return;
  const int per = ((npos + G - 1) / G + kPer - 1) / kPer * kPer;
  const int r0 = cur + g * per, r1 = min(p_end, r0 + per);
  int32_t* rec = nullptr;
  if (G > 1) rec = reinterpret_cast<int32_t*>(mws + (size_t)b * match_seq_bytes(Gl, max_matches) + 16 +
                                              (size_t)g * match_rec_bytes(max_matches));
  int32_t* out = G > 1 ? rec + 1 : match_pos + (size_t)b * max_matches;
  if (G == 1)
    for (int i = tid; i < max_matches; i += kThreads) out[i] = -1;
  if (tid < n) s_tail[tid] = tail[(size_t)b * n + tid];
  const int32_t* c = tok + o0;

  // the first tile's tokens, then each tile prefetches the next one's into registers
  constexpr int kLd = (kTile + kHalo + kThreads - 1) / kThreads;
  int32_t nx[kLd];
  auto fetch = [&](int base) {
    const int span = max(0, min(kTile + n - 1, len - base));
#pragma unroll
    for (int k = 0; k < kLd; ++k) {
      const int i = tid + k * kThreads;
      nx[k] = i < span ? __ldg(c + base + i) : 0;
    }
  };
  if (r0 < r1) fetch(r0);
  __syncthreads();   // the tail is in shared memory
  int32_t tl[kPer];
#pragma unroll
  for (int j = 0; j < kPer; ++j) tl[j] = j < n ? s_tail[j] : 0;
  int total = 0;  // block-uniform running count
  for (int base = r0; base < r1; base += kTile) {
    __syncthreads();  // previous tile's readers are done
#pragma unroll
    for (int k = 0; k < kLd; ++k) {
      const int i = tid + k * kThreads;
      if (i < kTile + kHalo) s_c[i] = nx[k];
    }
    __syncthreads();
    if (base + kTile < r1) fetch(base + kTile);

    unsigned hits = 0;
    if (n <= kPer) {
      // the thread's 8 positions and the next 8 tokens, as four 16-byte loads
      // (a warp reads one contiguous kilobyte twice: no bank conflicts)
      int32_t v[2 * kPer];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int4 x = *reinterpret_cast<const int4*>(&s_c[tid * kPer + 4 * q]);
        v[4 * q] = x.x;
        v[4 * q + 1] = x.y;
        v[4 * q + 2] = x.z;
        v[4 * q + 3] = x.w;
      }
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        bool ok = base + tid * kPer + k < r1;
#pragma unroll
        for (int j = 0; j < kPer; ++j)
          if (j < n) ok &= (v[k + j] == tl[j]);
        hits |= (unsigned)ok << k;
      }
    } else {
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const int pl = tid * kPer + k;
        if (base + pl < r1) {
          bool ok = true;
          for (int j = 0; j < n; ++j) ok &= (s_c[pl + j] == s_tail[j]);
          hits |= (unsigned)ok << k;
        }
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
      if (idx < max_matches) out[idx] = base + tid * kPer + k;
      ++idx;
    }
    total += s_tile_total;
  }
  if (G == 1) {
    if (tid == 0) n_matches[b] = total;
    return;
  }
  // publish this range's hits and count; the last of the sequence's CTAs
  // merges.  The ticket is one acquire-release add after the CTA barrier: it
  // releases every thread's record stores and acquires the other CTAs'.
  __syncthreads();
  if (tid == 0) {
    rec[0] = total;
    uint32_t* ticket = reinterpret_cast<uint32_t*>(mws + (size_t)b * match_seq_bytes(Gl, max_matches));
    s_last = ee::atom_add_acq_rel(ticket, 1u) == (uint32_t)(G - 1);
  }
  __syncthreads();
  if (!s_last) return;
  const uint8_t* recs = mws + (size_t)b * match_seq_bytes(Gl, max_matches) + 16;
  // warp 0: the records' counts and their exclusive prefix (range order)
  if (warp == 0) {
    const int v = lane < G ? __ldcg(reinterpret_cast<const int32_t*>(recs + lane * match_rec_bytes(max_matches)))
                           : 0;
    int w = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      int u = __shfl_up_sync(0xffffffffu, w, d);
      if (lane >= d) w += u;
    }
    if (lane < G) s_c[32 + lane] = w - v;   // the tile buffer is free: prefixes at [32, 64)
    if (lane == 31) s_tile_total = w;
  }
  __syncthreads();
  const int all = s_tile_total;
  int32_t* mp = match_pos + (size_t)b * max_matches;
  for (int i = tid; i < max_matches; i += kThreads) {
    int v = -1;
    if (i < all) {
      // the range holding hit i: the last range whose prefix is <= i
      int q = 0;
      for (int r = 1; r < G; ++r)
        if (s_c[32 + r] <= i) q = r;
      const int j = i - s_c[32 + q];
      v = __ldcg(reinterpret_cast<const int32_t*>(recs + q * match_rec_bytes(max_matches)) + 1 + j);
    }
    mp[i] = v;
  }
  if (tid == 0) {
    n_matches[b] = all;
    *reinterpret_cast<uint32_t*>(mws + (size_t)b * match_seq_bytes(Gl, max_matches)) = 0u;   // next call
  }
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
  // CTAs per sequence: about four per SM over the batch (four fit on an SM),
  // as many as the workspace's record region holds (a workspace of only the
  // fixed head: one)
  int G = std::min(kMaxSplit, std::max(1, (4 * ee::kNumSMs + B - 1) / B));
  if (ws_bytes < ee::kMatchOff + ee::kMatchBytes) G = 1;
  while (G > 1 && (size_t)B * match_seq_bytes(G, max_matches) > ee::kMatchBytes) --G;
  EE_CUDA_OK(ee::launch_pdl(match_reuse_kernel, dim3(B, G), dim3(kThreads), 0, (cudaStream_t)stream, 1,
                             orig_tokens, orig_off, tail, n, cursor, max_matches, match_pos, n_matches,
                             static_cast<uint8_t*>(ws) + ee::kMatchOff, ee::err_word(ws)));
  return EE_OK;
}
