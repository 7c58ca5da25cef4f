// ee_tree_verify_attn: tree-masked attention of every draft node over the
// paged KV cache plus the tree's own K/V, one layer per call (EfficientEdit
// Sec. IV-A: a single target forward pass over (prefix, draft) scores every
// draft token; with a tree, each node sees the prefix and its own root path).
//
// Work decomposition (split-KV):
//   - For a (sequence, KV head) the query rows are the g = n_q / n_kv heads of
//     the group times the T tree nodes, row r = node * g + head_in_group, so
//     one K/V tile feeds g * T rows (GQA packing).  A CTA owns 128 rows
//     (8 warps x 16 rows).
//   - The context is cut into chunks of `chunk` keys (a multiple of the 16-token
//     page); each (row block, chunk) is one CTA.  The CTA of the last chunk
//     also processes the tree keys, masked by the ancestor bitmask.
//   - Each CTA streams 64-key K/V tiles into shared memory with cp.async
//     (double buffered, 16-byte chunks, XOR-swizzled rows), computes S = Q K^T
//     on bf16 tensor cores with fp32 accumulation, keeps an fp32 online softmax
//     in the exp2 domain, and accumulates O += P V with P and V in fp16
//     (V converted in shared memory; bf16 -> fp16 is exact for |v| <= 65504).
//   - Partials (unnormalised O, running max m, running sum l) go to the
//     workspace; a second launch merges the chunks with log-sum-exp weights and
//     writes fp32 output.  No CTA ever waits on another.
#include "ee_common.cuh"

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kRows = 16 * kWarps;          // query rows per CTA
constexpr int kKT = 64;                     // keys per tile
constexpr int kD = EE_HEAD_DIM;             // 128
constexpr int kTileBytes = kKT * kD * 2;    // 16 KB for K or V
constexpr int kSmemBytes = 4 * kTileBytes;  // 2 buffers x (K, V)

static_assert(kRows == ee::kAttnRows, "row block size");

struct AttnParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* kt;
  const __nv_bfloat16* vt;
  const __nv_bfloat16* kc;
  const __nv_bfloat16* vc;
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

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// byte offset of 16-byte chunk `ch` (0..15) of row `row` in a 64 x 256-byte tile
__device__ __forceinline__ uint32_t swz(int row, int ch) {
  return (uint32_t)(row * 256 + ((ch ^ (row & 7)) << 4));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src),
               "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_f16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                        uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_half2(float lo, float hi) {
  __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Issue the cp.async copies of one 64-key tile (K and V) into buffer (sK, sV).
// Context tile: keys are cache positions key0.. (< key_end); tree tile: keys are
// local tree nodes key0.. (< T).  Missing or invalid keys are zero-filled and
// marked invalid in s_valid.
__device__ __forceinline__ void load_tile(const AttnParams& p, int b, int hk, int o, int T,
                                          bool tree, int key0, int key_end, uint32_t sK,
                                          uint32_t sV, int* s_valid) {
#pragma unroll
  for (int it = 0; it < (kKT * 16) / kThreads; ++it) {
    const int idx = threadIdx.x + it * kThreads;
    const int key = idx >> 4, ch = idx & 15;
    const __nv_bfloat16* srck = p.kc;
    const __nv_bfloat16* srcv = p.vc;
    bool ok;
    if (!tree) {
      const int pos = key0 + key;
      ok = pos < key_end;
      if (ok) {
        const int page = p.block_table[(size_t)b * p.max_pages + (pos >> 4)];
        if (page < 0 || page >= p.num_pages) {
          if (ch == 0) ee::flag_error(p.err, EE_DEVERR_PAGE);
          ok = false;
        } else {
          const size_t row = ((size_t)page * p.n_kv + hk) * EE_PAGE + (pos & (EE_PAGE - 1));
          srck = p.kc + row * kD + ch * 8;
          srcv = p.vc + row * kD + ch * 8;
        }
      }
    } else {
      const int j = key0 + key;
      ok = j < T;
      if (ok) {
        const size_t row = (size_t)(o + j) * p.n_kv + hk;
        srck = p.kt + row * kD + ch * 8;
        srcv = p.vt + row * kD + ch * 8;
      }
    }
    const int nb = ok ? 16 : 0;
    cp_async16(sK + swz(key, ch), srck, nb);
    cp_async16(sV + swz(key, ch), srcv, nb);
    if (ch == 0) s_valid[key] = ok ? 1 : 0;
  }
}

// Convert this thread's own V chunks of a landed tile from bf16 to fp16 in place.
__device__ __forceinline__ void convert_v(char* sV, int32_t* err) {
  bool overflow = false;
#pragma unroll
  for (int it = 0; it < (kKT * 16) / kThreads; ++it) {
    const int idx = threadIdx.x + it * kThreads;
    const int key = idx >> 4, ch = idx & 15;
    uint4* ptr = reinterpret_cast<uint4*>(sV + swz(key, ch));
    uint4 v = *ptr;
    uint32_t* w = reinterpret_cast<uint32_t*>(&v);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      __nv_bfloat162 bb = *reinterpret_cast<__nv_bfloat162*>(&w[e]);
      float2 f = __bfloat1622float2(bb);
      overflow |= (fabsf(f.x) > 65504.f) || (fabsf(f.y) > 65504.f);
      w[e] = pack_half2(f.x, f.y);
    }
    *ptr = v;
  }
  if (overflow) ee::flag_error(err, EE_DEVERR_FP16_RANGE);
}

__global__ void __launch_bounds__(kThreads, 1) attn_split_kernel(const AttnParams p) {
  extern __shared__ __align__(1024) char smem[];
  __shared__ int s_valid[2][kKT];

  const int b = blockIdx.z;
  const int hk = blockIdx.y;
  const int rb = blockIdx.x % p.nrb;
  const int split = blockIdx.x / p.nrb;
  const int o = p.node_off[b];
  const int T = p.node_off[b + 1] - o;
  const int R = T * p.g;
  if (T < 1 || T > EE_MAX_TREE || T > p.max_T || o < 0 || o + T > p.total_nodes) {
    if (threadIdx.x == 0 && blockIdx.x == 0 && hk == 0) ee::flag_error(p.err, EE_DEVERR_TREE);
    return;
  }
  if (rb * kRows >= R) return;
  int ctx = p.ctx_len[b];
  if (ctx < 0 || ctx > p.max_ctx) {
    if (threadIdx.x == 0 && rb == 0 && split == 0 && hk == 0) ee::flag_error(p.err, EE_DEVERR_CTX);
    ctx = ctx < 0 ? 0 : p.max_ctx;
  }
  const int S = ee::attn_splits_for(ctx, p.chunk);
  if (split >= S) return;
  const int k_begin = split * p.chunk;
  const int k_end = min(ctx, k_begin + p.chunk);
  const int n_ctx_tiles = k_end > k_begin ? (k_end - k_begin + kKT - 1) / kKT : 0;
  const bool last = (split == S - 1);
  const int n_tree_tiles = last ? (T + kKT - 1) / kKT : 0;
  const int n_tiles = n_ctx_tiles + n_tree_tiles;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row_a = rb * kRows + warp * 16 + (lane >> 2);
  const int row_b = row_a + 8;
  const bool va = row_a < R, vb = row_b < R;
  const int node_a = va ? row_a / p.g : 0, node_b = vb ? row_b / p.g : 0;
  const int head_a = hk * p.g + (va ? row_a % p.g : 0);
  const int head_b = hk * p.g + (vb ? row_b % p.g : 0);

  // Q fragments (A operand, 16 rows x 128 dims per warp) straight from global memory
  uint32_t qa[8][4];
  {
    const uint32_t* qra =
        reinterpret_cast<const uint32_t*>(p.q + ((size_t)(o + node_a) * p.n_q + head_a) * kD);
    const uint32_t* qrb =
        reinterpret_cast<const uint32_t*>(p.q + ((size_t)(o + node_b) * p.n_q + head_b) * kD);
    const int c = (lane & 3);
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      qa[ks][0] = va ? __ldg(qra + ks * 8 + c) : 0u;
      qa[ks][1] = vb ? __ldg(qrb + ks * 8 + c) : 0u;
      qa[ks][2] = va ? __ldg(qra + ks * 8 + 4 + c) : 0u;
      qa[ks][3] = vb ? __ldg(qrb + ks * 8 + 4 + c) : 0u;
    }
  }
  const uint64_t anc_a0 = va ? p.anc[2 * (size_t)(o + node_a)] : 0ull;
  const uint64_t anc_a1 = va ? p.anc[2 * (size_t)(o + node_a) + 1] : 0ull;
  const uint64_t anc_b0 = vb ? p.anc[2 * (size_t)(o + node_b)] : 0ull;
  const uint64_t anc_b1 = vb ? p.anc[2 * (size_t)(o + node_b) + 1] : 0ull;

  float acc[16][4];
#pragma unroll
  for (int i = 0; i < 16; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
  float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;

  const uint32_t sbase = smem_u32(smem);
  auto tile_key0 = [&](int t) { return t < n_ctx_tiles ? k_begin + t * kKT : (t - n_ctx_tiles) * kKT; };

  if (n_tiles > 0) {
    load_tile(p, b, hk, o, T, n_ctx_tiles == 0, tile_key0(0), k_end, sbase, sbase + kTileBytes,
              s_valid[0]);
    cp_async_commit();
  }
  for (int t = 0; t < n_tiles; ++t) {
    const int buf = t & 1;
    if (t + 1 < n_tiles) {
      const int nb = (t + 1) & 1;
      load_tile(p, b, hk, o, T, t + 1 >= n_ctx_tiles, tile_key0(t + 1), k_end,
                sbase + nb * 2 * kTileBytes, sbase + nb * 2 * kTileBytes + kTileBytes,
                s_valid[nb]);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    convert_v(smem + buf * 2 * kTileBytes + kTileBytes, p.err);
    __syncthreads();

    const bool tree = t >= n_ctx_tiles;
    const int key0 = tile_key0(t);
    const uint32_t sK = sbase + buf * 2 * kTileBytes;
    const uint32_t sV = sK + kTileBytes;

    // S = Q K^T : 16 rows x 64 keys per warp
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int kk2 = 0; kk2 < 4; ++kk2) {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sK + swz(nt * 8 + (lane & 7), kk2 * 4 + (lane >> 3)), b0, b1, b2, b3);
        mma_bf16(s[nt], qa[2 * kk2], b0, b1);
        mma_bf16(s[nt], qa[2 * kk2 + 1], b2, b3);
      }
    }
    // mask + scale, row max
    float mx_a = -INFINITY, mx_b = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int col = nt * 8 + (lane & 3) * 2 + (e & 1);
        bool ok = s_valid[buf][col] != 0;
        if (tree) {
          const int j = key0 + col;
          const uint64_t w0 = e < 2 ? anc_a0 : anc_b0;
          const uint64_t w1 = e < 2 ? anc_a1 : anc_b1;
          const uint64_t bit = j < 64 ? (w0 >> j) : (w1 >> (j - 64));
          ok = ok && (bit & 1ull);
        }
        const float v = ok ? s[nt][e] * p.scale_log2 : -INFINITY;
        s[nt][e] = v;
        if (e < 2) mx_a = fmaxf(mx_a, v); else mx_b = fmaxf(mx_b, v);
      }
    }
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
    const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
    const float mu_a = mn_a == -INFINITY ? 0.f : mn_a;
    const float mu_b = mn_b == -INFINITY ? 0.f : mn_b;
    const float al_a = ex2(m_a - mu_a), al_b = ex2(m_b - mu_b);
    m_a = mn_a;
    m_b = mn_b;
    l_a *= al_a;
    l_b *= al_b;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      acc[i][0] *= al_a;
      acc[i][1] *= al_a;
      acc[i][2] *= al_b;
      acc[i][3] *= al_b;
    }
    // P (fp16 A fragments) and row sums
    uint32_t pa[4][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = ex2(s[nt][0] - mu_a), p1 = ex2(s[nt][1] - mu_a);
      const float p2 = ex2(s[nt][2] - mu_b), p3 = ex2(s[nt][3] - mu_b);
      l_a += p0 + p1;
      l_b += p2 + p3;
      pa[nt >> 1][(nt & 1) * 2 + 0] = pack_half2(p0, p1);
      pa[nt >> 1][(nt & 1) * 2 + 1] = pack_half2(p2, p3);
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int ntp = 0; ntp < 8; ++ntp) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sV + swz(kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8, ntp * 2 + (lane >> 4)), b0,
                  b1, b2, b3);
        mma_f16(acc[2 * ntp], pa[kk], b0, b1);
        mma_f16(acc[2 * ntp + 1], pa[kk], b2, b3);
      }
    }
    __syncthreads();  // buffer `buf` is refilled two tiles later
  }

  l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);

  const size_t pra = ((size_t)split * p.total_nodes + o + node_a) * p.n_q + head_a;
  const size_t prb = ((size_t)split * p.total_nodes + o + node_b) * p.n_q + head_b;
  const int c0 = (lane & 3) * 2;
#pragma unroll
  for (int nt = 0; nt < 16; ++nt) {
    if (va)
      *reinterpret_cast<float2*>(p.part_o + pra * kD + nt * 8 + c0) = make_float2(acc[nt][0], acc[nt][1]);
    if (vb)
      *reinterpret_cast<float2*>(p.part_o + prb * kD + nt * 8 + c0) = make_float2(acc[nt][2], acc[nt][3]);
  }
  if ((lane & 3) == 0) {
    if (va) p.part_ml[pra] = make_float2(m_a, l_a);
    if (vb) p.part_ml[prb] = make_float2(m_b, l_b);
  }
}

// Merge the split partials of every (node, head) with log-sum-exp weights.
__global__ void __launch_bounds__(256)
attn_combine_kernel(const float* __restrict__ part_o, const float2* __restrict__ part_ml,
                    const int32_t* __restrict__ ctx_len, const int32_t* __restrict__ node_off,
                    int max_ctx, int chunk, int n_q, int total_nodes, float* __restrict__ out) {
  const int b = blockIdx.y;
  const int i = blockIdx.x;
  const int o = node_off[b];
  const int T = node_off[b + 1] - o;
  if (T < 1 || T > EE_MAX_TREE || o < 0 || o + T > total_nodes || i >= T) return;
  int ctx = ctx_len[b];
  ctx = ctx < 0 ? 0 : (ctx > max_ctx ? max_ctx : ctx);
  const int S = ee::attn_splits_for(ctx, chunk);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int h = warp; h < n_q; h += 8) {
    float M = -INFINITY;
    for (int s = 0; s < S; ++s) M = fmaxf(M, part_ml[((size_t)s * total_nodes + o + i) * n_q + h].x);
    const float Mu = M == -INFINITY ? 0.f : M;
    float L = 0.f;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s = 0; s < S; ++s) {
      const size_t r = ((size_t)s * total_nodes + o + i) * n_q + h;
      const float2 ml = part_ml[r];
      const float w = ex2(ml.x - Mu);
      L += w * ml.y;
      const float4 v = *reinterpret_cast<const float4*>(part_o + r * kD + lane * 4);
      a.x += w * v.x;
      a.y += w * v.y;
      a.z += w * v.z;
      a.w += w * v.w;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    *reinterpret_cast<float4*>(out + ((size_t)(o + i) * n_q + h) * kD + lane * 4) =
        make_float4(a.x * inv, a.y * inv, a.z * inv, a.w * inv);
  }
}

// Context chunk length: the smallest number of splits whose CTA count fills
// the 152 SMs nearly as well as the best choice does.
int choose_chunk(int max_ctx, int per_split_ctas) {
  if (max_ctx <= 0) return EE_PAGE;
  const int cap = std::max(1, std::min(ee::kMaxSplits, (max_ctx + 255) / 256));
  double best = 0.0;
  double eff[ee::kMaxSplits + 1];
  for (int s = 1; s <= cap; ++s) {
    const long n = (long)per_split_ctas * s;
    const long waves = (n + ee::kNumSMs - 1) / ee::kNumSMs;
    eff[s] = (double)n / (double)(waves * ee::kNumSMs);
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
  if (!ee::aligned(q, 16) || !ee::aligned(k_tree, 16) || !ee::aligned(v_tree, 16) ||
      !ee::aligned(k_cache, 16) || !ee::aligned(v_cache, 16) || !ee::aligned(out, 16) ||
      !ee::aligned(anc, 8) || !ee::aligned(ws, 256))
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kAttnOff + ee::attn_partial_bytes(total_nodes, n_q, head_dim))
    return EE_ERR_WORKSPACE;

  static bool attr_set = false;
  if (!attr_set) {
    EE_CUDA_OK(cudaFuncSetAttribute(attn_split_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kSmemBytes));
    attr_set = true;
  }
  const int g = n_q / n_kv;
  const int nrb = (max_T * g + kRows - 1) / kRows;
  const int chunk = choose_chunk(max_ctx, nrb * n_kv * B);
  const int S = ee::attn_splits_for(max_ctx, chunk);

  char* wsb = static_cast<char*>(ws);
  AttnParams p;
  p.q = reinterpret_cast<const __nv_bfloat16*>(q);
  p.kt = reinterpret_cast<const __nv_bfloat16*>(k_tree);
  p.vt = reinterpret_cast<const __nv_bfloat16*>(v_tree);
  p.kc = reinterpret_cast<const __nv_bfloat16*>(k_cache);
  p.vc = reinterpret_cast<const __nv_bfloat16*>(v_cache);
  p.block_table = block_table;
  p.ctx_len = ctx_len;
  p.node_off = node_off;
  p.anc = anc;
  p.part_o = reinterpret_cast<float*>(wsb + ee::kAttnOff);
  const size_t rows = (size_t)ee::kMaxSplits * total_nodes * n_q;
  p.part_ml = reinterpret_cast<float2*>(wsb + ee::kAttnOff + ee::align_up(rows * head_dim * 4, 256));
  p.err = ee::err_word(ws);
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
  attn_split_kernel<<<grid, kThreads, kSmemBytes, (cudaStream_t)stream>>>(p);
  EE_LAUNCH_OK();
  attn_combine_kernel<<<dim3(max_T, B), 256, 0, (cudaStream_t)stream>>>(
      p.part_o, p.part_ml, ctx_len, node_off, max_ctx, chunk, n_q, total_nodes, out);
  EE_LAUNCH_OK();
  return EE_OK;
}
