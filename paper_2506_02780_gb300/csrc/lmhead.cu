// ee_lmhead_accept: LM head fused with greedy decode and path acceptance
// (EfficientEdit Sec. III-A, Eq. (piecewise): a draft token is accepted while the
// target's greedy choice at the previous position equals it).
//
// Design (sm_103a, one persistent CTA per SM):
//   - Swap-AB GEMM on the 5th-generation tensor cores: the vocabulary is the
//     MMA M side (128 rows of W per tile), the tree nodes are the N side
//     (BN = 16..256 columns), K = hidden in 64-element (128-byte) blocks.
//     D[vocab_row][node] accumulates in fp32 in TMEM, never in registers and
//     never in HBM (unless the caller asks for the logits).
//   - Warp 0 (one lane) streams W and X tiles with TMA (128B swizzle) into a
//     STAGES-deep shared-memory ring guarded by mbarriers; warp 1 (one lane)
//     issues tcgen05.mma.kind::f16 (bf16 x bf16 -> fp32) and commits each
//     stage back to the producer; two TMEM accumulators let the epilogue drain
//     tile i while tile i+1 accumulates.
//   - Warps 2..5 (the epilogue) read the accumulator with tcgen05.ld (one TMEM
//     lane = one vocabulary row per thread) and reduce each node's column to
//     (max, lowest index) with a shuffle reduce-scatter; the running best per
//     node stays in shared memory across the CTA's tiles and is published once
//     with a 64-bit atomicMax on an order-preserving key.
//   - The last CTA to finish (ticket counter, no waiting) decodes the keys into
//     argmax[], runs the acceptance for every sequence with one warp each
//     (ancestor masks AND a per-node "edge accepted" mask), and resets the
//     workspace state for the next call.
//   - The kernel is bound by streaming W from HBM when the node count is below
//     the ridge point (~250), by the tensor pipe above it.
// Every mbarrier wait is bounded (2e9 SM cycles, about 1 s); on expiry the CTA sets
// EE_DEVERR_TIMEOUT, drains its own copies and MMAs (again bounded), frees its
// TMEM and returns.
#include <cmath>
#include <mutex>
#include <cuda.h>

#include "ee_common.cuh"
#include "ee_ptx.cuh"

namespace {

using namespace ee;

constexpr int BM = 128;           // vocab rows per tile (MMA M)
constexpr int BK = 64;            // bf16 per 128-byte swizzle row
constexpr int kThreads = 192;     // warp 0 TMA, warp 1 MMA, warps 2..5 epilogue
constexpr int kABytes = BM * BK * 2;

struct LmParams {
  int vocab, hidden, total_nodes, B, max_T;
  int BN, n_nt, n_vt, nkb, stages, tmem_cols;
  const int32_t* draft_tok;
  const int32_t* parent;
  const int32_t* depth;
  const uint64_t* anc;
  const int32_t* node_off;
  int32_t* argmax;
  int32_t* accept_len;
  int32_t* path;
  int32_t* bonus;
  float* logits;
  unsigned long long* keys;   // [EE_MAX_LM_NODES] running argmax keys (workspace)
  unsigned int* ticket;       // CTAs finished (workspace)
  int32_t* err;
};

__device__ __forceinline__ uint32_t ordered(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ unsigned long long make_key(float v, int idx) {
  return ((unsigned long long)ordered(v) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)idx);
}
__device__ __forceinline__ bool better(float v, int i, float w, int j) {
  return v > w || (v == w && i < j);
}

struct BestPair {
  float v;
  int i;
};

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads, 1)
lmhead_accept_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                     const LmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  ee::pdl_allow_next();
  ee::pdl_wait();   // no global access before the previous kernel's writes are visible
  const int S = p.stages, BN = p.BN;
  const uint32_t bBytes = (uint32_t)BN * BK * 2;
  uint8_t* sA = smem;
  uint8_t* sB = smem + (size_t)S * kABytes;
  uint8_t* tail = sB + (size_t)S * bBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(tail);   // full[S], empty[S], tfull[2], tempty[2], drain
  BestPair* s_best = reinterpret_cast<BestPair*>(tail + 8 * (2 * S + 5) + 8);  // [4][BN]
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(tail + 8 * (2 * S + 5));
  __shared__ volatile int s_abort;
  __shared__ int s_last;
  __shared__ int s_issued, s_consumed;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, tfull0 = empty0 + 8 * S;
  const uint32_t tempty0 = tfull0 + 16, drain = tempty0 + 16;

  if (threadIdx.x == 0) {
    s_abort = 0;
    s_issued = 0;
    s_consumed = 0;
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 4);
    }
    mbar_init(drain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(s_tmem)),
                 "r"(p.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  for (int i = threadIdx.x; i < 4 * BN; i += kThreads) s_best[i] = BestPair{-INFINITY, 0x7fffffff};
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;

  const int num_tiles = p.n_vt * p.n_nt;

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmX)) : "memory");
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x) {
        const int vt = t / p.n_nt, nt = t % p.n_nt;
        for (int kb = 0; kb < p.nkb; ++kb) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1, &s_abort)) {
            ok = false;
            break;
          }
          const uint32_t fb = full0 + 8 * stage;
          mbar_expect_tx(fb, kABytes + bBytes);
          tma_load_2d(smem_u32(sA + (size_t)stage * kABytes), &tmW, fb, kb * BK, vt * BM);
          tma_load_2d(smem_u32(sB + (size_t)stage * bBytes), &tmX, fb, kb * BK, nt * BN);
          ++s_issued;
          if (++stage == S) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int lt = 0;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x, ++lt) {
        const int acc = lt & 1;
        const uint32_t acc_phase = (lt >> 1) & 1;
        if (!mbar_wait(tempty0 + 8 * acc, acc_phase ^ 1, &s_abort)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int kb = 0; kb < p.nkb; ++kb) {
          if (!mbar_wait(full0 + 8 * stage, phase, &s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc_sw128(smem_u32(sA + (size_t)stage * kABytes));
          const uint64_t bd = smem_desc_sw128(smem_u32(sB + (size_t)stage * bBytes));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                   (kb | k) != 0 ? 1u : 0u);
          tc_commit(empty0 + 8 * stage);
          ++s_consumed;
          if (++stage == S) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (ok) tc_commit(tfull0 + 8 * acc);
      }
    }
  } else {
    // epilogue warps 2..5: TMEM lane quarter = warp % 4
    const int q = warp & 3;
    const int ew = warp - 2;
    BestPair* mybest = s_best + ew * BN;
    int lt = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++lt) {
      const int vt = t / p.n_nt, nt = t % p.n_nt;
      const int acc = lt & 1;
      const uint32_t acc_phase = (lt >> 1) & 1;
      // warp-uniform outcome: the tcgen05.ld below is warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait(tfull0 + 8 * acc, acc_phase, &s_abort))) break;
      tc_fence_after();
      const int row = vt * BM + q * 32 + lane;
      const bool row_ok = row < p.vocab;
      for (int c0 = 0; c0 < BN; c0 += 16) {
        uint32_t r[16];
        tc_ld16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN + c0), r);
        float v[16];
        int id[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          v[j] = row_ok ? __uint_as_float(r[j]) : -INFINITY;
          id[j] = row;
        }
        if (p.logits != nullptr && row_ok) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int node = nt * BN + c0 + j;
            if (node < p.total_nodes) p.logits[(size_t)node * p.vocab + row] = v[j];
          }
        }
        // reduce-scatter: 16 columns over 32 lanes -> lanes 2c and 2c+1 own column c
#pragma unroll
        for (int half = 8, bit = 16; half >= 1; half >>= 1, bit >>= 1) {
          const bool upper = (lane & bit) != 0;
#pragma unroll
          for (int j = 0; j < half; ++j) {
            const float keep_v = upper ? v[j + half] : v[j];
            const int keep_i = upper ? id[j + half] : id[j];
            const float give_v = upper ? v[j] : v[j + half];
            const int give_i = upper ? id[j] : id[j + half];
            const float ov = __shfl_xor_sync(0xffffffffu, give_v, bit);
            const int oi = __shfl_xor_sync(0xffffffffu, give_i, bit);
            const bool take = better(ov, oi, keep_v, keep_i);
            v[j] = take ? ov : keep_v;
            id[j] = take ? oi : keep_i;
          }
        }
        {
          const float ov = __shfl_xor_sync(0xffffffffu, v[0], 1);
          const int oi = __shfl_xor_sync(0xffffffffu, id[0], 1);
          if (better(ov, oi, v[0], id[0])) {
            v[0] = ov;
            id[0] = oi;
          }
        }
        const int col = ((lane >> 4) & 1) * 8 + ((lane >> 3) & 1) * 4 + ((lane >> 2) & 1) * 2 +
                        ((lane >> 1) & 1);
        if ((lane & 1) == 0) {
          BestPair cur = mybest[c0 + col];
          if (better(v[0], id[0], cur.v, cur.i)) mybest[c0 + col] = BestPair{v[0], id[0]};
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
    }
    // publish this CTA's best per node (every tile of a CTA has the same node tile)
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (blockIdx.x < num_tiles) {
      const int nt = blockIdx.x % p.n_nt;
      for (int c = threadIdx.x - 64; c < BN; c += 128) {
        BestPair b = s_best[c];
        for (int w = 1; w < 4; ++w) {
          const BestPair o = s_best[w * BN + c];
          if (better(o.v, o.i, b.v, b.i)) b = o;
        }
        const int node = nt * BN + c;
        if (node < p.total_nodes && b.i != 0x7fffffff) atomicMax(&p.keys[node], make_key(b.v, b.i));
      }
    }
    __threadfence();
  }

  // ---- teardown: drain on abort, free TMEM --------------------------------
  tc_fence_before();
  __syncthreads();
  const bool aborted = s_abort != 0;
  if (aborted) {
    if (threadIdx.x == 0) {
      ee::flag_error(p.err, EE_DEVERR_TIMEOUT);
      // TMA loads issued but never consumed still land in shared memory: wait for them
      for (int k = s_consumed; k < s_issued; ++k)
        if (!mbar_wait_plain(full0 + 8 * (k % S), (uint32_t)((k / S) & 1))) break;
    }
  }
  if (warp == 1) {
    if (aborted && lane == 0) {
      tc_commit(drain);
      mbar_wait_plain(drain, 0);
    }
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(p.tmem_cols)
                 : "memory");
  }
  if (aborted) return;

  // ---- last CTA: argmax decode + acceptance ---------------------------------
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned int ticket = atomicAdd(p.ticket, 1u);
    s_last = (ticket == gridDim.x - 1) ? 1 : 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  int32_t* s_am = reinterpret_cast<int32_t*>(smem);   // pipeline buffers are idle now
  for (int i = threadIdx.x; i < p.total_nodes; i += kThreads) {
    const unsigned long long k = atomicExch(&p.keys[i], 0ull);
    const int a = k ? (int)(0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFull)) : -1;
    s_am[i] = a;
    p.argmax[i] = a;
  }
  if (threadIdx.x == 0) *p.ticket = 0u;
  __syncthreads();
  for (int s = warp; s < p.B; s += kThreads / 32) {
    const int o = p.node_off[s];
    const int T = p.node_off[s + 1] - o;
    if (T < 1 || T > EE_MAX_TREE || T > p.max_T || o < 0 || o + T > p.total_nodes) {
      if (lane == 0) ee::flag_error(p.err, EE_DEVERR_TREE);
      continue;
    }
    // notok bit i: node i's edge from its parent is rejected
    uint32_t notok[4];
    uint64_t a0[4], a1[4];
    int key_best = -1;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int i = c * 32 + lane;
      bool bad = false;
      if (i < T && i > 0) {
        const int par = p.parent[o + i];
        bad = (par < 0 || par >= i) ? true : (p.draft_tok[o + i] != s_am[o + par]);
      }
      notok[c] = __ballot_sync(0xffffffffu, bad);
      a0[c] = i < T ? p.anc[2 * (size_t)(o + i)] : 0ull;
      a1[c] = i < T ? p.anc[2 * (size_t)(o + i) + 1] : 0ull;
    }
    const uint64_t nz0 = (uint64_t)notok[0] | ((uint64_t)notok[1] << 32);
    const uint64_t nz1 = (uint64_t)notok[2] | ((uint64_t)notok[3] << 32);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int i = c * 32 + lane;
      if (i < T && (a0[c] & nz0) == 0 && (a1[c] & nz1) == 0) {
        const int k = (p.depth[o + i] << 8) | (255 - i);
        key_best = max(key_best, k);
      }
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) key_best = max(key_best, __shfl_xor_sync(0xffffffffu, key_best, d));
    const int u = 255 - (key_best & 255);
    const int du = key_best >> 8;
    const uint64_t w0 = p.anc[2 * (size_t)(o + u)], w1 = p.anc[2 * (size_t)(o + u) + 1];
    for (int j = lane; j < p.max_T; j += 32) p.path[(size_t)s * p.max_T + j] = -1;
    __syncwarp();
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int j = c * 32 + lane;
      const bool on = j < 64 ? ((w0 >> j) & 1ull) : ((w1 >> (j - 64)) & 1ull);
      if (j < T && on) {
        const int pos = j < 64 ? __popcll(w0 & ((1ull << j) - 1ull))
                               : __popcll(w0) + __popcll(w1 & ((1ull << (j - 64)) - 1ull));
        if (pos < p.max_T) p.path[(size_t)s * p.max_T + pos] = j;
      }
    }
    if (lane == 0) {
      p.accept_len[s] = du;
      p.bonus[s] = s_am[o + u];
    }
  }
}

// ---------------------------------------------------------------------------
bool encode_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
               uint32_t box_outer) {
  const uint64_t dims[2] = {inner, outer};
  const uint64_t strides[1] = {inner * 2};
  const uint32_t box[2] = {box_inner, box_outer};
  return ee::encode_bf16_tmap(map, base, 2, dims, strides, box);
}

// Host-side argument checks shared by the LM-head entry points.  Sets *empty
// when there is nothing to launch.
ee_status check_lm_args(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                        int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                        const int32_t* depth, const uint64_t* anc, const int32_t* node_off, int32_t B,
                        int32_t total_nodes, int32_t max_T, const int32_t* argmax,
                        const int32_t* accept_len, const int32_t* path, const int32_t* bonus,
                        bool* empty) {
  *empty = false;
  if (B < 0 || total_nodes < 0 || hidden_dim < 8 || vocab < 1 || max_T < 1)
    return EE_ERR_INVALID_ARG;
  if (hidden_dim % 8 != 0 || max_T > EE_MAX_TREE || total_nodes > EE_MAX_LM_NODES)
    return EE_ERR_UNSUPPORTED;
  if (B == 0 || total_nodes == 0) {
    *empty = true;
    return EE_OK;
  }
  if (!hidden || !lm_w || !draft_tok || !parent || !depth || !anc || !node_off || !argmax ||
      !accept_len || !path || !bonus)
    return EE_ERR_INVALID_ARG;
  if (!ee::aligned(hidden, 16) || !ee::aligned(lm_w, 16)) return EE_ERR_INVALID_ARG;
  return EE_OK;
}

// Encode the tensor maps and launch the persistent LM-head kernel; `keys`
// (EE_MAX_LM_NODES running-argmax words, zero on entry), `ticket` (zero on
// entry) and `err` are the kernel's scratch.
ee_status launch_lmhead(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                        int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                        const int32_t* depth, const uint64_t* anc, const int32_t* node_off, int32_t B,
                        int32_t total_nodes, int32_t max_T, int32_t* argmax, int32_t* accept_len,
                        int32_t* path, int32_t* bonus, float* logits_or_null,
                        unsigned long long* keys, unsigned int* ticket, int32_t* err,
                        ee_stream_t stream, bool pdl) {
  LmParams p;
  p.vocab = vocab;
  p.hidden = hidden_dim;
  p.total_nodes = total_nodes;
  p.B = B;
  p.max_T = max_T;
  p.n_nt = (total_nodes + 255) / 256;
  p.BN = ((total_nodes + p.n_nt - 1) / p.n_nt + 15) / 16 * 16;
  p.n_vt = (vocab + BM - 1) / BM;
  p.nkb = (hidden_dim + BK - 1) / BK;
  const size_t stage_bytes = (size_t)kABytes + (size_t)p.BN * BK * 2;
  const size_t fixed = 1024 /*align slack*/ + 8 * (2 * 8 + 5) + 8 + 4 * (size_t)p.BN * sizeof(BestPair);
  const size_t budget = 227 * 1024 - fixed - 64;
  p.stages = (int)std::min<size_t>(8, budget / stage_bytes);
  if (p.stages < 2) return EE_ERR_UNSUPPORTED;
  int cols = 32;
  while (cols < 2 * p.BN) cols <<= 1;
  p.tmem_cols = cols;
  p.draft_tok = draft_tok;
  p.parent = parent;
  p.depth = depth;
  p.anc = anc;
  p.node_off = node_off;
  p.argmax = argmax;
  p.accept_len = accept_len;
  p.path = path;
  p.bonus = bonus;
  p.logits = logits_or_null;
  p.keys = keys;
  p.ticket = ticket;
  p.err = err;

  CUtensorMap tmW, tmX;
  if (!encode_2d(&tmW, lm_w, (uint64_t)hidden_dim, (uint64_t)vocab, BK, BM)) return EE_ERR_CUDA;
  if (!encode_2d(&tmX, hidden, (uint64_t)hidden_dim, (uint64_t)total_nodes, BK, p.BN))
    return EE_ERR_CUDA;

  const size_t smem = 1024 + (size_t)p.stages * stage_bytes + 8 * (2 * p.stages + 5) + 8 +
                      4 * (size_t)p.BN * sizeof(BestPair);
  const size_t smem_acc = std::max(smem, (size_t)1024 + (size_t)EE_MAX_LM_NODES * 4);
  static size_t attr_bytes = 0;
  if (attr_bytes < smem_acc) {
    EE_CUDA_OK(cudaFuncSetAttribute(lmhead_accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)smem_acc));
    attr_bytes = smem_acc;
  }
  const int num_tiles = p.n_vt * p.n_nt;
  int grid = (ee::kNumSMs / p.n_nt) * p.n_nt;   // multiple of n_nt: each CTA keeps one node tile
  if (grid > num_tiles) grid = num_tiles;
  if (grid < 1) grid = 1;
  if (pdl) {
    EE_CUDA_OK(ee::launch_pdl(lmhead_accept_kernel, dim3(grid), dim3(kThreads), smem_acc,
                              (cudaStream_t)stream, 1, tmW, tmX, p));
  } else {
    lmhead_accept_kernel<<<grid, kThreads, smem_acc, (cudaStream_t)stream>>>(tmW, tmX, p);
    EE_LAUNCH_OK();
  }
  return EE_OK;
}

}  // namespace

extern "C" ee_status ee_lmhead_accept(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                                      int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                                      const int32_t* depth, const uint64_t* anc,
                                      const int32_t* node_off, int32_t B, int32_t total_nodes,
                                      int32_t max_T, int32_t* argmax, int32_t* accept_len,
                                      int32_t* path, int32_t* bonus, float* logits_or_null,
                                      void* ws, size_t ws_bytes, ee_stream_t stream) {
  bool empty = false;
  const ee_status st = check_lm_args(hidden, lm_w, hidden_dim, vocab, draft_tok, parent, depth, anc,
                                     node_off, B, total_nodes, max_T, argmax, accept_len, path,
                                     bonus, &empty);
  if (st != EE_OK || empty) return st;
  if (!ws || !ee::aligned(ws, 256)) return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  char* wsb = static_cast<char*>(ws);
  return launch_lmhead(hidden, lm_w, hidden_dim, vocab, draft_tok, parent, depth, anc, node_off, B,
                       total_nodes, max_T, argmax, accept_len, path, bonus, logits_or_null,
                       reinterpret_cast<unsigned long long*>(wsb + ee::kArgmaxOff),
                       reinterpret_cast<unsigned int*>(wsb + ee::kTicketOff), ee::err_word(ws),
                       stream, true);
}

// ---------------------------------------------------------------------------
// ee_lmhead_accept_static: the same LM head + argmax + acceptance for callers
// that cannot allocate device memory -- code that runs where cudaMalloc is not
// available to it (inside a host callback or a custom allocator's own hooks,
// or under an allocation budget that forbids new device buffers).  Its scratch
// (running-argmax words, finished-CTA ticket, device error word) lives in the
// file-scope array below, 16,640 bytes, which every GPU that loads libee holds
// until the process exits.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kStaticScratchBytes = ee::kArgmaxOff + 8 * (size_t)EE_MAX_LM_NODES;  // 16,640
static __device__ __align__(256) unsigned char g_lm_scratch[kStaticScratchBytes];

// Device address of g_lm_scratch per device ordinal, looked up once per device.
// The host-side symbol `g_lm_scratch` is only a stand-in for the device array:
// it must never be passed to a kernel.
constexpr int kMaxDevices = 64;
void* g_lm_scratch_ptr[kMaxDevices] = {};

std::mutex g_lm_scratch_mu;

ee_status static_scratch(void** out) {
  int dev = -1;
  EE_CUDA_OK(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return EE_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_lm_scratch_mu);
  if (!g_lm_scratch_ptr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_lm_scratch) != cudaSuccess || !ptr) return EE_ERR_CUDA;
    g_lm_scratch_ptr[dev] = ptr;
  }
  *out = g_lm_scratch_ptr[dev];
  return EE_OK;
}

}  // namespace

extern "C" ee_status ee_lmhead_accept_static(const ee_bf16* hidden, const ee_bf16* lm_w,
                                             int32_t hidden_dim, int32_t vocab,
                                             const int32_t* draft_tok, const int32_t* parent,
                                             const int32_t* depth, const uint64_t* anc,
                                             const int32_t* node_off, int32_t B,
                                             int32_t total_nodes, int32_t max_T, int32_t* argmax,
                                             int32_t* accept_len, int32_t* path, int32_t* bonus,
                                             float* logits_or_null, ee_stream_t stream) {
  bool empty = false;
  const ee_status st = check_lm_args(hidden, lm_w, hidden_dim, vocab, draft_tok, parent, depth, anc,
                                     node_off, B, total_nodes, max_T, argmax, accept_len, path,
                                     bonus, &empty);
  if (st != EE_OK || empty) return st;   // total_nodes > EE_MAX_LM_NODES -> EE_ERR_UNSUPPORTED
  void* scratch = nullptr;
  const ee_status ss = static_scratch(&scratch);
  if (ss != EE_OK) return ss;
  // the array keeps the previous call's contents: start from zero every call
  EE_CUDA_OK(cudaMemsetAsync(scratch, 0, kStaticScratchBytes, (cudaStream_t)stream));
  char* base = static_cast<char*>(scratch);
  return launch_lmhead(hidden, lm_w, hidden_dim, vocab, draft_tok, parent, depth, anc, node_off, B,
                       total_nodes, max_T, argmax, accept_len, path, bonus, logits_or_null,
                       reinterpret_cast<unsigned long long*>(base + ee::kArgmaxOff),
                       reinterpret_cast<unsigned int*>(base + ee::kTicketOff),
                       reinterpret_cast<int32_t*>(base + ee::kErrOff), stream, false);
}
