// ee_tree_verify_attn: tree-masked attention of every draft node over the
// paged KV cache plus the tree's own K/V, one layer per call (EfficientEdit
// Sec. IV-A: a single target forward pass over (prefix, draft) scores every
// draft token; with a tree, each node sees the prefix and its own root path).
//
// Work decomposition (split-KV):
//   - For a (sequence, KV head) the query rows are the g = n_q / n_kv heads of
//     the group times the T tree nodes, row r = node * g + head_in_group, so
//     one K/V tile feeds g * T rows (GQA packing).  A CTA owns 128 rows: the
//     M side of a tcgen05 MMA.
//   - The context is cut into chunks of `chunk` keys (a multiple of the 16-token
//     page); each (row block, chunk) is one CTA.  The CTA of the last chunk
//     also processes the tree keys, masked by the ancestor bitmask.
//   - Warp 0 streams 64-key K/V tiles with TMA (one 16-row box per page and
//     128-byte half of the head dimension; the tree's own K/V through a 3-D map)
//     into a 3-stage ring.  Warps 2-3 convert each landed V tile to fp16 in
//     place.  Warp 1 issues tcgen05.mma: S = Q K^T (bf16, fp32 in TMEM, double
//     buffered) and O += P V (fp16 P from shared memory, fp16 V read MN-major,
//     fp32 O in TMEM).  Warps 4-7 own one query row per thread: they read S
//     from TMEM, mask, keep the running max/sum, write P, and rescale O in TMEM
//     only when a row's max grows by more than 2^8 (the stale max keeps every
//     P <= 256, exact in fp16, and the final O / l is unchanged).
//   - Partials (unnormalised O, max m, sum l per row) go to the workspace; a
//     second launch merges the chunks with log-sum-exp weights and writes fp32
//     output.  No CTA ever waits on another; every mbarrier wait is bounded.
#include "ee_common.cuh"
#include "ee_ptx.cuh"

namespace {

using namespace ee;

constexpr int kThreads = 256;
constexpr int kRows = 128;                       // query rows per CTA (MMA M)
constexpr int kKT = 64;                          // keys per tile (MMA N of Q K^T)
constexpr int kD = EE_HEAD_DIM;                  // 128
constexpr int kNST = 3;                          // K/V ring depth
constexpr uint32_t kQHalf = kRows * 128;         // 16 KB: one 64-dim half of Q
constexpr uint32_t kKVHalf = kKT * 128;          // 8 KB: one 64-dim half of a K or V tile
constexpr uint32_t kKVBytes = 2 * kKVHalf;       // 16 KB
constexpr uint32_t kStageBytes = 2 * kKVBytes;   // K + V
constexpr uint32_t kPBytes = kRows * kKT * 2;    // 16 KB fp16 P tile
constexpr uint32_t kOffKV = 2 * kQHalf;
constexpr uint32_t kOffP = kOffKV + kNST * kStageBytes;
constexpr uint32_t kOffBar = kOffP + 2 * kPBytes;
constexpr uint32_t kNumBars = 3 * kNST + 3 * 2 + 2;
constexpr uint32_t kSmemBytes = 1024 + kOffBar + 8 * kNumBars + 64;
constexpr uint32_t kTmemCols = 256;              // S0 [0,64) S1 [64,128) O [128,256)
constexpr float kRescaleLog2 = 8.0f;

static_assert(kRows == ee::kAttnRows, "row block size");

struct AttnParams {
  const __nv_bfloat16* q;
  const int32_t* block_table;
  const int32_t* ctx_len;
  const int32_t* node_off;
  const uint64_t* anc;
  float* part_o;
  float2* part_ml;
  int32_t* err;
  int num_pages, max_pages, max_ctx, n_q, n_kv, g, total_nodes, max_T, nrb, chunk;
  float scale_log2;
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi) {
  __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Whether 16-row page block i of a context tile holds loaded keys; the producer,
// the V converter and the softmax all derive the same answer from the inputs.
__device__ __forceinline__ bool page_loaded(const AttnParams& p, int b, int key0, int k_end, int i,
                                            int* page_out) {
  const int pos = key0 + 16 * i;
  if (pos >= k_end) return false;
  const int page = p.block_table[(size_t)b * p.max_pages + (pos >> 4)];
  *page_out = page;
  return page >= 0 && page < p.num_pages;
}

__global__ void __launch_bounds__(kThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmKc, const __grid_constant__ CUtensorMap tmVc,
               const __grid_constant__ CUtensorMap tmKt, const __grid_constant__ CUtensorMap tmVt,
               const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_issued[kNST];

  const int b = blockIdx.z;
  const int hk = blockIdx.y;
  const int rb = blockIdx.x % p.nrb;
  const int split = blockIdx.x / p.nrb;
  const int o = p.node_off[b];
  const int T = p.node_off[b + 1] - o;
  const int R = T * p.g;
  if (T < 1 || T > EE_MAX_TREE || T > p.max_T || o < 0 || o + T > p.total_nodes) {
    if (threadIdx.x == 0 && blockIdx.x == 0 && hk == 0) flag_error(p.err, EE_DEVERR_TREE);
    return;
  }
  if (rb * kRows >= R) return;
  int ctx = p.ctx_len[b];
  if (ctx < 0 || ctx > p.max_ctx) {
    if (threadIdx.x == 0 && blockIdx.x == 0 && hk == 0) flag_error(p.err, EE_DEVERR_CTX);
    ctx = ctx < 0 ? 0 : p.max_ctx;
  }
  const int S = attn_splits_for(ctx, p.chunk);
  if (split >= S) return;
  const int k_begin = split * p.chunk;
  const int k_end = min(ctx, k_begin + p.chunk);
  const int n_ctx_tiles = k_end > k_begin ? (k_end - k_begin + kKT - 1) / kKT : 0;
  const int n_tree_tiles = (split == S - 1) ? (T + kKT - 1) / kKT : 0;
  const int n_tiles = n_ctx_tiles + n_tree_tiles;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase, sKV = sbase + kOffKV, sP = sbase + kOffP;
  const uint32_t bar0 = sbase + kOffBar;
  const uint32_t kv_full = bar0, kv_empty = bar0 + 8 * kNST, v_ready = bar0 + 16 * kNST;
  const uint32_t s_full = bar0 + 24 * kNST, s_free = s_full + 16, p_full = s_free + 16;
  const uint32_t o_done = p_full + 16, drain = o_done + 8;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int i = 0; i < kNST; ++i) {
      mbar_init(kv_full + 8 * i, 1);
      mbar_init(kv_empty + 8 * i, 1);
      mbar_init(v_ready + 8 * i, 64);
      s_issued[i] = -1;
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full + 8 * i, 1);
      mbar_init(s_free + 8 * i, kRows);
      mbar_init(p_full + 8 * i, kRows);
    }
    mbar_init(o_done, 1);
    mbar_init(drain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_async_smem();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&s_tmem)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // Q tile: 128 rows x 128 dims, K-major with 128-byte swizzle, two 64-dim halves
  {
    const int row_base = rb * kRows;
#pragma unroll
    for (int it = 0; it < (kRows * 16) / kThreads; ++it) {
      const int idx = threadIdx.x + it * kThreads;
      const int r = idx >> 4, c = idx & 15;
      const int rr = row_base + r;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (rr < R) {
        const int node = rr / p.g, j = rr - node * p.g;
        const __nv_bfloat16* src = p.q + ((size_t)(o + node) * p.n_q + hk * p.g + j) * kD + c * 8;
        v = __ldg(reinterpret_cast<const uint4*>(src));
      }
      const uint32_t dst = sQ + (c >> 3) * kQHalf + r * 128 + (((c & 7) ^ (r & 7)) << 4);
      asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(v.x), "r"(v.y), "r"(v.z),
                   "r"(v.w)
                   : "memory");
    }
    fence_async_smem();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      for (int t = 0; t < n_tiles; ++t) {
        const int st = t % kNST, use = t / kNST;
        if (!mbar_wait(kv_empty + 8 * st, (uint32_t)(use & 1) ^ 1u, &s_abort)) break;
        const uint32_t full = kv_full + 8 * st;
        const uint32_t sK = sKV + st * kStageBytes, sV = sK + kKVBytes;
        if (t < n_ctx_tiles) {
          const int key0 = k_begin + t * kKT;
          int pages[4];
          uint32_t bytes = 0;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            int pg = -1;
            const bool ok = page_loaded(p, b, key0, k_end, i, &pg);
            if (!ok && key0 + 16 * i < k_end) flag_error(p.err, EE_DEVERR_PAGE);
            pages[i] = ok ? pg : -1;
            bytes += ok ? 4u * 2048u : 0u;
          }
          mbar_expect_tx(full, bytes);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            if (pages[i] < 0) continue;
            const int row0 = (pages[i] * p.n_kv + hk) * EE_PAGE;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              tma_load_2d(sK + h * kKVHalf + i * 2048, &tmKc, full, h * 64, row0);
              tma_load_2d(sV + h * kKVHalf + i * 2048, &tmVc, full, h * 64, row0);
            }
          }
        } else {
          const int key0 = (t - n_ctx_tiles) * kKT;
          mbar_expect_tx(full, 4 * kKVHalf);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            tma_load_3d(sK + h * kKVHalf, &tmKt, full, h * 64, hk, o + key0);
            tma_load_3d(sV + h * kKVHalf, &tmVt, full, h * 64, hk, o + key0);
          }
        }
        s_issued[st] = use;
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t id_qk = idesc_f16(kRows, kKT, 1, 1, 0);
      const uint32_t id_pv = idesc_f16(kRows, kD, 0, 0, 1);
      bool ok = true;
      auto issue_pv = [&](int u) -> bool {
        const int st = u % kNST, sb = u & 1;
        if (!mbar_wait(p_full + 8 * sb, (uint32_t)((u >> 1) & 1), &s_abort)) return false;
        if (!mbar_wait(v_ready + 8 * st, (uint32_t)((u / kNST) & 1), &s_abort)) return false;
        tc_fence_after();
        const uint32_t pa = sP + sb * kPBytes;
        const uint32_t vb = sKV + st * kStageBytes + kKVBytes;
#pragma unroll
        for (int j = 0; j < kKT / 16; ++j)
          tc_mma(tmem + 128, smem_desc_sw128(pa + j * 32), smem_desc_sw128_mn(vb + j * 2048, kKVHalf, 1024),
                 id_pv, (u > 0 || j > 0) ? 1u : 0u);
        tc_commit(kv_empty + 8 * st);
        tc_commit(o_done);
        return true;
      };
      for (int t = 0; t < n_tiles && ok; ++t) {
        const int st = t % kNST, use = t / kNST, sb = t & 1;
        if (!mbar_wait(kv_full + 8 * st, (uint32_t)(use & 1), &s_abort)) break;
        if (t >= 2 && !mbar_wait(s_free + 8 * sb, (uint32_t)((t >> 1) & 1) ^ 1u, &s_abort)) break;
        tc_fence_after();
        const uint32_t kb = sKV + st * kStageBytes;
#pragma unroll
        for (int kk = 0; kk < kD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * 0 + (kk & 3) * 32;
          tc_mma(tmem + sb * kKT, smem_desc_sw128(sQ + (kk >> 2) * kQHalf + off),
                 smem_desc_sw128(kb + (kk >> 2) * kKVHalf + off), id_qk, kk > 0 ? 1u : 0u);
        }
        tc_commit(s_full + 8 * sb);
        if (t >= 1) ok = issue_pv(t - 1);
      }
      if (ok && n_tiles > 0) issue_pv(n_tiles - 1);
    }
  } else if (warp < 4) {
    // ---------------- V converters: bf16 -> fp16 in place ----------------
    const int ct = threadIdx.x - 64;
    bool overflow = false;
    for (int t = 0; t < n_tiles; ++t) {
      const int st = t % kNST, use = t / kNST;
      if (!mbar_wait(kv_full + 8 * st, (uint32_t)(use & 1), &s_abort)) break;
      uint4* sv = reinterpret_cast<uint4*>(smem + kOffKV + st * kStageBytes + kKVBytes);
      // rows of a context tile whose page was not loaded hold stale bytes: zero them
      unsigned loaded = 0xFu;
      if (t < n_ctx_tiles) {
        const int key0 = k_begin + t * kKT;
        loaded = 0u;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          int pg;
          if (page_loaded(p, b, key0, k_end, i, &pg)) loaded |= 1u << i;
        }
      }
#pragma unroll 4
      for (int it = 0; it < (int)(kKVBytes / 16) / 64; ++it) {
        const int idx = ct + it * 64;                 // 16-byte chunk; 8 per 128-byte row
        const int row = (idx >> 3) & (kKT - 1);       // key row within the 64-dim half
        uint4 v = sv[idx];
        if (!((loaded >> (row >> 4)) & 1u)) {
          v = make_uint4(0u, 0u, 0u, 0u);
        } else {
          uint32_t* w = reinterpret_cast<uint32_t*>(&v);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 bb = *reinterpret_cast<__nv_bfloat162*>(&w[e]);
            const float2 f = __bfloat1622float2(bb);
            overflow |= (fabsf(f.x) > 65504.f) || (fabsf(f.y) > 65504.f);
            w[e] = pack_half2(f.x, f.y);
          }
        }
        sv[idx] = v;
      }
      fence_async_smem();
      mbar_arrive(v_ready + 8 * st);
    }
    if (overflow) flag_error(p.err, EE_DEVERR_FP16_RANGE);
  } else {
    // ---------------- softmax: one query row per thread ----------------
    const int r = threadIdx.x - 128;                  // == TMEM lane
    const int rr = rb * kRows + r;
    const bool vrow = rr < R;
    const int node = vrow ? rr / p.g : 0;
    const int head = hk * p.g + (vrow ? rr - node * p.g : 0);
    const uint64_t a0 = vrow ? p.anc[2 * (size_t)(o + node)] : 0ull;
    const uint64_t a1 = vrow ? p.anc[2 * (size_t)(o + node) + 1] : 0ull;
    const uint32_t tl = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < n_tiles; ++t) {
      const int sb = t & 1;
      if (!mbar_wait(s_full + 8 * sb, (uint32_t)((t >> 1) & 1), &s_abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sr[64];
      tc_ld32(tl + sb * kKT, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
      tc_ld32(tl + sb * kKT + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
      tc_fence_before();
      mbar_arrive(s_free + 8 * sb);
      float tmax = -INFINITY;
      if (t < n_ctx_tiles) {
        const int key0 = k_begin + t * kKT;
        unsigned loaded = 0u;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          int pg;
          if (page_loaded(p, b, key0, k_end, i, &pg)) loaded |= 1u << i;
        }
#pragma unroll
        for (int c = 0; c < kKT; ++c) {
          const bool v = vrow && (key0 + c < k_end) && ((loaded >> (c >> 4)) & 1u);
          const float x = v ? __uint_as_float(sr[c]) * p.scale_log2 : -INFINITY;
          sr[c] = __float_as_uint(x);
          tmax = fmaxf(tmax, x);
        }
      } else {
        const int key0 = (t - n_ctx_tiles) * kKT;
        const uint64_t w = key0 == 0 ? a0 : a1;       // key0 is 0 or 64
#pragma unroll
        for (int c = 0; c < kKT; ++c) {
          const bool v = vrow && (key0 + c < T) && ((w >> c) & 1ull);
          const float x = v ? __uint_as_float(sr[c]) * p.scale_log2 : -INFINITY;
          sr[c] = __float_as_uint(x);
          tmax = fmaxf(tmax, x);
        }
      }
      const float m_new = fmaxf(m_used, tmax);
      if (t >= 1 && !mbar_wait(o_done, (uint32_t)((t - 1) & 1), &s_abort)) {
        ok = false;
        break;
      }
      const bool need = m_new > m_used + kRescaleLog2;
      if (t >= 1 && __any_sync(0xffffffffu, need)) {
        tc_fence_after();
        const float f = need ? ex2(m_used - m_new) : 1.f;
#pragma unroll 1
        for (int c4 = 0; c4 < 4; ++c4) {
          uint32_t ov[32];
          tc_ld32(tl + 128 + 32 * c4, ov);
#pragma unroll
          for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * f);
          tc_st32(tl + 128 + 32 * c4, ov);
        }
      }
      if (need) {
        l *= ex2(m_used - m_new);
        m_used = m_new;
      }
      const float mu = m_used == -INFINITY ? 0.f : m_used;
      // P row (fp16) into the K-major, 128-byte-swizzled P tile
      const uint32_t prow = sP + sb * kPBytes + r * 128;
#pragma unroll
      for (int ch = 0; ch < 8; ++ch) {
        uint32_t w4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float p0 = ex2(__uint_as_float(sr[ch * 8 + 2 * e]) - mu);
          const float p1 = ex2(__uint_as_float(sr[ch * 8 + 2 * e + 1]) - mu);
          l += p0 + p1;
          w4[e] = pack_half2(p0, p1);
        }
        asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(prow + ((ch ^ (r & 7)) << 4)),
                     "r"(w4[0]), "r"(w4[1]), "r"(w4[2]), "r"(w4[3])
                     : "memory");
      }
      fence_async_smem();
      tc_fence_before();
      mbar_arrive(p_full + 8 * sb);
    }
    if (ok && n_tiles > 0 && mbar_wait(o_done, (uint32_t)((n_tiles - 1) & 1), &s_abort)) {
      tc_fence_after();
      const size_t pr = ((size_t)split * p.total_nodes + o + node) * p.n_q + head;
#pragma unroll 1
      for (int c4 = 0; c4 < 4; ++c4) {
        uint32_t ov[32];
        tc_ld32(tl + 128 + 32 * c4, ov);
        if (vrow) {
          float4* dst = reinterpret_cast<float4*>(p.part_o + pr * kD + 32 * c4);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            dst[e] = make_float4(__uint_as_float(ov[4 * e]), __uint_as_float(ov[4 * e + 1]),
                                 __uint_as_float(ov[4 * e + 2]), __uint_as_float(ov[4 * e + 3]));
        }
      }
      if (vrow) p.part_ml[pr] = make_float2(m_used, l);
    }
  }

  // ---- teardown: drain on abort, free TMEM ----------------------------------
  tc_fence_before();
  __syncthreads();
  const bool aborted = s_abort != 0;
  if (aborted && threadIdx.x == 0) {
    flag_error(p.err, EE_DEVERR_TIMEOUT);
    for (int st = 0; st < kNST; ++st)   // TMA copies still in flight land before the CTA exits
      if (s_issued[st] >= 0) mbar_wait_plain(kv_full + 8 * st, (uint32_t)(s_issued[st] & 1));
  }
  if (warp == 1) {
    if (aborted && lane == 0) {
      tc_commit(drain);
      mbar_wait_plain(drain, 0);
    }
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols)
                 : "memory");
  }
}

// Merge the split partials of every (node, head) with log-sum-exp weights:
// one warp per (node, head), lane s holds split s's (m, l), lanes own 4 dims.
__global__ void __launch_bounds__(256)
attn_combine_kernel(const float* __restrict__ part_o, const float2* __restrict__ part_ml,
                    const int32_t* __restrict__ ctx_len, const int32_t* __restrict__ node_off,
                    int max_ctx, int chunk, int n_q, int total_nodes, float* __restrict__ out) {
  const int b = blockIdx.z;
  const int i = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y * 8 + warp;
  const int o = node_off[b];
  const int T = node_off[b + 1] - o;
  if (T < 1 || T > EE_MAX_TREE || o < 0 || o + T > total_nodes || i >= T || h >= n_q) return;
  int ctx = ctx_len[b];
  ctx = ctx < 0 ? 0 : (ctx > max_ctx ? max_ctx : ctx);
  const int S = attn_splits_for(ctx, chunk);
  const size_t r0 = (size_t)(o + i) * n_q + h;
  const size_t sstride = (size_t)total_nodes * n_q;
  float m = -INFINITY, lsum = 0.f;
  if (lane < S) {
    const float2 ml = part_ml[lane * sstride + r0];
    m = ml.x;
    lsum = ml.y;
  }
  float M = m;
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, d));
  const float Mu = M == -INFINITY ? 0.f : M;
  const float w = lane < S ? ex2(m - Mu) : 0.f;
  float L = w * lsum;
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) L += __shfl_xor_sync(0xffffffffu, L, d);
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s = 0; s < S; ++s) {
    const float ws = __shfl_sync(0xffffffffu, w, s);
    const float4 v = __ldg(reinterpret_cast<const float4*>(part_o + (s * sstride + r0) * kD) + lane);
    a.x += ws * v.x;
    a.y += ws * v.y;
    a.z += ws * v.z;
    a.w += ws * v.w;
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  reinterpret_cast<float4*>(out + r0 * kD)[lane] = make_float4(a.x * inv, a.y * inv, a.z * inv, a.w * inv);
}

// Context chunk length: the smallest number of splits whose CTA count fills
// the 152 SMs nearly as well as the best choice does.
int choose_chunk(int max_ctx, int per_split_ctas) {
  if (max_ctx <= 0) return EE_PAGE;
  const int cap = std::max(1, std::min(kMaxSplits, (max_ctx + 255) / 256));
  double best = 0.0;
  double eff[kMaxSplits + 1];
  for (int s = 1; s <= cap; ++s) {
    const long n = (long)per_split_ctas * s;
    const long waves = (n + kNumSMs - 1) / kNumSMs;
    eff[s] = (double)n / (double)(waves * kNumSMs);
    best = std::max(best, eff[s]);
  }
  int pick = cap;
  for (int s = 1; s <= cap; ++s)
    if (eff[s] >= 0.9 * best) {
      pick = s;
      break;
    }
  int chunk = (max_ctx + pick - 1) / pick;
  chunk = (chunk + EE_PAGE - 1) / EE_PAGE * EE_PAGE;
  return chunk;
}

}  // namespace

extern "C" ee_status ee_tree_verify_attn(const ee_bf16* q, const ee_bf16* k_tree,
                                         const ee_bf16* v_tree, const ee_bf16* k_cache,
                                         const ee_bf16* v_cache, int32_t num_pages,
                                         const int32_t* block_table, int32_t max_pages,
                                         const int32_t* ctx_len, int32_t max_ctx,
                                         const int32_t* node_off, const uint64_t* anc, int32_t B,
                                         int32_t total_nodes, int32_t max_T, int32_t n_q,
                                         int32_t n_kv, int32_t head_dim, float scale, float* out,
                                         void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (B < 0 || total_nodes < 0 || n_q < 1 || n_kv < 1 || num_pages < 1 || max_pages < 1 ||
      max_ctx < 0 || max_T < 1)
    return EE_ERR_INVALID_ARG;
  if (head_dim != EE_HEAD_DIM || n_q % n_kv != 0 || max_T > EE_MAX_TREE) return EE_ERR_UNSUPPORTED;
  if ((int64_t)max_ctx > (int64_t)max_pages * EE_PAGE) return EE_ERR_INVALID_ARG;
  if (!(scale > 0.f) || !std::isfinite(scale)) return EE_ERR_INVALID_ARG;
  if (B == 0 || total_nodes == 0) return EE_OK;
  if (!q || !k_tree || !v_tree || !k_cache || !v_cache || !block_table || !ctx_len || !node_off ||
      !anc || !out || !ws)
    return EE_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k_tree, 16) || !aligned(v_tree, 16) || !aligned(k_cache, 16) ||
      !aligned(v_cache, 16) || !aligned(out, 16) || !aligned(anc, 8) || !aligned(ws, 256))
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < kAttnOff + attn_partial_bytes(total_nodes, n_q, head_dim)) return EE_ERR_WORKSPACE;
  if ((int64_t)num_pages * n_kv * EE_PAGE >= ((int64_t)1 << 31)) return EE_ERR_UNSUPPORTED;

  static bool attr_set = false;
  if (!attr_set) {
    EE_CUDA_OK(cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)kSmemBytes));
    attr_set = true;
  }
  // tensor maps: cache [pages * n_kv * 16 rows][128], tree [total][n_kv][128]
  CUtensorMap tmKc, tmVc, tmKt, tmVt;
  {
    const uint64_t dims[2] = {(uint64_t)head_dim, (uint64_t)num_pages * n_kv * EE_PAGE};
    const uint64_t strides[1] = {(uint64_t)head_dim * 2};
    const uint32_t box[2] = {64, EE_PAGE};
    if (!encode_bf16_tmap(&tmKc, k_cache, 2, dims, strides, box)) return EE_ERR_CUDA;
    if (!encode_bf16_tmap(&tmVc, v_cache, 2, dims, strides, box)) return EE_ERR_CUDA;
  }
  {
    const uint64_t dims[3] = {(uint64_t)head_dim, (uint64_t)n_kv, (uint64_t)total_nodes};
    const uint64_t strides[2] = {(uint64_t)head_dim * 2, (uint64_t)n_kv * head_dim * 2};
    const uint32_t box[3] = {64, 1, 64};
    if (!encode_bf16_tmap(&tmKt, k_tree, 3, dims, strides, box)) return EE_ERR_CUDA;
    if (!encode_bf16_tmap(&tmVt, v_tree, 3, dims, strides, box)) return EE_ERR_CUDA;
  }
  const int g = n_q / n_kv;
  const int nrb = (max_T * g + kRows - 1) / kRows;
  const int chunk = choose_chunk(max_ctx, nrb * n_kv * B);
  const int S = attn_splits_for(max_ctx, chunk);

  char* wsb = static_cast<char*>(ws);
  AttnParams p;
  p.q = reinterpret_cast<const __nv_bfloat16*>(q);
  p.block_table = block_table;
  p.ctx_len = ctx_len;
  p.node_off = node_off;
  p.anc = anc;
  p.part_o = reinterpret_cast<float*>(wsb + kAttnOff);
  const size_t rows = (size_t)kMaxSplits * total_nodes * n_q;
  p.part_ml = reinterpret_cast<float2*>(wsb + kAttnOff + align_up(rows * head_dim * 4, 256));
  p.err = err_word(ws);
  p.num_pages = num_pages;
  p.max_pages = max_pages;
  p.max_ctx = max_ctx;
  p.n_q = n_q;
  p.n_kv = n_kv;
  p.g = g;
  p.total_nodes = total_nodes;
  p.max_T = max_T;
  p.nrb = nrb;
  p.chunk = chunk;
  p.scale_log2 = scale * 1.4426950408889634f;

  dim3 grid(nrb * S, n_kv, B);
  attn_tc_kernel<<<grid, kThreads, kSmemBytes, (cudaStream_t)stream>>>(tmKc, tmVc, tmKt, tmVt, p);
  EE_LAUNCH_OK();
  attn_combine_kernel<<<dim3(max_T, (n_q + 7) / 8, B), 256, 0, (cudaStream_t)stream>>>(
      p.part_o, p.part_ml, ctx_len, node_off, max_ctx, chunk, n_q, total_nodes, out);
  EE_LAUNCH_OK();
  return EE_OK;
}
