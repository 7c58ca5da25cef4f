// ee_lmhead_accept: LM head fused with greedy decode and path acceptance
// (EfficientEdit Sec. III-A, Eq. (piecewise): a draft token is accepted while the
// target's greedy choice at the previous position equals it).
//
// Design (sm_103a, one persistent CTA per SM):
//   - Swap-AB GEMM on the 5th-generation tensor cores: the vocabulary is the
//     MMA M side (up to 128 rows of W per tile, as many tiles for every CTA:
//     126 rows at V = 152064 on 152 SMs), the tree nodes are the N side
//     (BN = 16..256 columns), K = hidden in 64-element (128-byte) blocks.
//     D[vocab_row][node] accumulates in fp32 in TMEM, never in registers and
//     never in HBM (unless the caller asks for the logits).
//   - Warp 0 (one lane) streams W and X tiles with TMA (128B swizzle) into a
//     STAGES-deep shared-memory ring guarded by mbarriers; warp 1 (one lane)
//     issues tcgen05.mma.kind::f16 (bf16 x bf16 -> fp32) and commits each
//     stage back to the producer; two TMEM accumulators let the epilogue drain
//     tile i while tile i+1 accumulates.
//   - Warps 2..9 (the epilogue, two per TMEM lane quarter taking alternate
//     16-column chunks) read the accumulator with tcgen05.ld (one TMEM lane =
//     one vocabulary row per thread) and reduce each node's column to (max,
//     lowest index) with a shuffle reduce-scatter; the running best per node
//     stays in shared memory across the CTA's tiles and is published once with
//     a 64-bit atomicMax on an order-preserving key.
//   - The LM head waits for the previous kernel before its first weight load:
//     on sm_103a a TMA load issued before griddepcontrol.wait lands only after
//     the previous grid has finished (measured in the attention kernel: 1.3 to
//     1.5 us after the wait, the same as a load issued after it), so streaming
//     W earlier buys nothing.
//   - The last CTA to finish (ticket counter, no waiting) decodes the keys into
//     argmax[], runs the acceptance for every sequence with one warp each
//     (ancestor masks AND a per-node "edge accepted" mask), and resets the
//     workspace state for the next call.  The tail is a chain of global round
//     trips, kept short: the ticket is one acquire-release add after the CTA
//     barrier (no separate fences), the node offsets load beside the key
//     exchange, and the acceptance loads each node's inputs in one round trip.
//   - The producer thread issues the ring's first stages right after it
//     initialises the barriers, before the set-up barrier.
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
constexpr int kThreads = 320;     // warp 0 TMA, warp 1 MMA, warps 2..9 epilogue
constexpr int kEpiWarps = 8;      // two per TMEM lane quarter, alternate 16-column chunks
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kABytes = BM * BK * 2;

struct LmParams {
  int vocab, hidden, total_nodes, B, max_T;
  int BN, n_nt, n_vt, nkb, stages, tmem_cols;
  int BMr;                    // vocabulary rows per tile (<= BM; the MMA's other rows are not used)
  int packed;                 // W in tile order ([V/128][H/64][128][64], ee_lmhead_pack_weights): BMr = BM
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
  // verification rules (ee_lmhead_verify only)
  int mode, K;                // EE_VERIFY_*, list length k
  const uint8_t* gen_mask;    // 1 = edit content (the mode's rule), 0 = reused (greedy); NULL = all 1
  int32_t* topk_ids;          // [total][K] or NULL
  int32_t* tau_out;           // [total] or NULL
  float* h_out;               // [total] or NULL
  uint8_t* part;              // per-CTA partials (workspace), BN * (8 K + 8) bytes per CTA
  unsigned long long* gthr;   // [EE_MAX_LM_NODES] best K-th key published by any CTA (workspace)
};

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// (m1, s1) + (m2, s2): sums of 2^((l - m) log2 e) kept against a running max
__device__ __forceinline__ void lse_add(float& m, float& sm, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    sm = s2;
    return;
  }
  const float mm = fmaxf(m, m2);
  sm = sm * ex2f((m - mm) * kLog2e) + s2 * ex2f((m2 - mm) * kLog2e);
  m = mm;
}
// lane that owns column c after the 16-column reduce-scatter below
__device__ __forceinline__ int lane_of_col(int c) {
  return (((c >> 3) & 1) << 4) | (((c >> 2) & 1) << 3) | (((c >> 1) & 1) << 2) | ((c & 1) << 1);
}

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

__device__ __forceinline__ float unordered(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}
// One round of a warp-wide selection over one (value, id) per lane: the best
// value (order-preserving 32-bit key, one warp reduction), the lowest id among
// lanes holding exactly that value.  Returns the winner in (*wv, *wi).
__device__ __forceinline__ void warp_best(float v, int id, float* wv, int* wi) {
  const uint32_t key = ordered(v);
  const uint32_t mx = __reduce_max_sync(0xffffffffu, key);
  const uint32_t mid = __reduce_min_sync(0xffffffffu, key == mx ? (uint32_t)id : 0xFFFFFFFFu);
  *wv = unordered(mx);
  *wi = (int)mid;
}
struct BestPair {
  float v;
  int i;
};

// ---------------------------------------------------------------------------
// Acceptance for every sequence (one warp each): node i is accepted when every
// edge on its root path is accepted -- a 128-bit "edge rejected" ballot mask
// ANDed with each node's ancestor mask -- and the deepest accepted node (lowest
// local id among equally deep ones) gives the path, accept_len and bonus.
// An edge a -> b of reused code is accepted when draft_tok[b] = argmax[a];
// with kVerify, edit content follows the mode's rule on the ranked ids tk and
// top_tau of a.  kGlobal: am / tk / tau live in global memory (read through L2).
struct AcceptArgs {
  int B, max_T, total, mode, K;
  const int32_t* node_off;
  const int32_t* parent;
  const int32_t* draft_tok;
  const int32_t* depth;
  const uint64_t* anc;
  const uint8_t* gen_mask;
  int32_t* accept_len;
  int32_t* path;
  int32_t* bonus;
  int32_t* err;
};

template <bool kVerify>
__device__ void accept_sequences(const AcceptArgs& a, const int32_t* am, const int32_t* tk,
                                 const int32_t* tau, int warp, int lane, int nwarps) {
  auto ld_i = [](const int32_t* q) -> int {
    if constexpr (kVerify)
      return __ldcg(q);
    else
      return *q;
  };
  const bool chain = a.anc == nullptr;   // linear drafts (greedy only): node i's parent is i - 1
  for (int s = warp; s < a.B; s += nwarps) {
    const int o = a.node_off[s];
    const int T = a.node_off[s + 1] - o;
    if (T < 1 || T > (chain ? EE_MAX_CHAIN : EE_MAX_TREE) || T > a.max_T || o < 0 || o + T > a.total) {
      if (lane == 0) ee::flag_error(a.err, EE_DEVERR_TREE);
      continue;
    }
    if (chain) {
      // Eq. (piecewise) on a linear draft: the first node whose token differs
      // from the argmax at its predecessor ends the accepted prefix
      int first = T;
      for (int base = 1; base < T; base += 32) {
        const int i = base + lane;
        const bool bad = i < T && a.draft_tok[o + i] != ld_i(am + o + i - 1);
        const unsigned m = __ballot_sync(0xffffffffu, bad);
        if (m) {
          first = base + __ffs(m) - 1;
          break;
        }
      }
      const int acc = first - 1;
      for (int j = lane; j < a.max_T; j += 32) a.path[(size_t)s * a.max_T + j] = j <= acc ? j : -1;
      if (lane == 0) {
        a.accept_len[s] = acc;
        a.bonus[s] = ld_i(am + o + acc);
      }
      continue;
    }
    // notok bit i: node i's edge from its parent is rejected.  Each lane's
    // nodes' parent, token, ancestor mask and depth are loaded together (one
    // round trip); the deepest accepted node's mask comes from its lane.
    uint32_t notok[4];
    uint64_t a0[4], a1[4];
    int par_[4], tok_[4], dep_[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int i = c * 32 + lane;
      const bool in = i < T;
      par_[c] = in && i > 0 ? a.parent[o + i] : -1;
      tok_[c] = in && i > 0 ? a.draft_tok[o + i] : 0;
      dep_[c] = in ? a.depth[o + i] : 0;
      a0[c] = in ? a.anc[2 * (size_t)(o + i)] : 0ull;
      a1[c] = in ? a.anc[2 * (size_t)(o + i) + 1] : 0ull;
    }
    int key_best = -1;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int i = c * 32 + lane;
      bool bad = false;
      if (i < T && i > 0) {
        const int par = par_[c];
        if (par < 0 || par >= i) {
          bad = true;
        } else {
          const int tok = tok_[c];
          if (!kVerify || (a.gen_mask && !a.gen_mask[o + i])) {
            bad = tok != ld_i(am + o + par);               // reused code: greedy
          } else if (a.mode == EE_VERIFY_DIRECT) {
            bad = false;
          } else {
            const int lim = a.mode == EE_VERIFY_GREEDY ? 1
                          : (a.mode == EE_VERIFY_TOPK ? a.K : ld_i(tau + o + par));
            bad = true;
            for (int rr = 0; rr < lim; ++rr)
              if (ld_i(tk + (size_t)(o + par) * a.K + rr) == tok) bad = false;
          }
        }
      }
      notok[c] = __ballot_sync(0xffffffffu, bad);
    }
    const uint64_t nz0 = (uint64_t)notok[0] | ((uint64_t)notok[1] << 32);
    const uint64_t nz1 = (uint64_t)notok[2] | ((uint64_t)notok[3] << 32);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int i = c * 32 + lane;
      if (i < T && (a0[c] & nz0) == 0 && (a1[c] & nz1) == 0) {
        const int k = (dep_[c] << 8) | (255 - i);
        key_best = max(key_best, k);
      }
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) key_best = max(key_best, __shfl_xor_sync(0xffffffffu, key_best, d));
    const int u = 255 - (key_best & 255);
    const int du = key_best >> 8;
    uint64_t w0 = 0ull, w1 = 0ull;   // node u's ancestor mask, held by lane u % 32
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const uint64_t x0 = __shfl_sync(0xffffffffu, a0[c], u & 31);
      const uint64_t x1 = __shfl_sync(0xffffffffu, a1[c], u & 31);
      if (c == (u >> 5)) {
        w0 = x0;
        w1 = x1;
      }
    }
    for (int j = lane; j < a.max_T; j += 32) a.path[(size_t)s * a.max_T + j] = -1;
    __syncwarp();
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int j = c * 32 + lane;
      const bool on = j < 64 ? ((w0 >> j) & 1ull) : ((w1 >> (j - 64)) & 1ull);
      if (j < T && on) {
        const int pos = j < 64 ? __popcll(w0 & ((1ull << j) - 1ull))
                               : __popcll(w0) + __popcll(w1 & ((1ull << (j - 64)) - 1ull));
        if (pos < a.max_T) a.path[(size_t)s * a.max_T + pos] = j;
      }
    }
    if (lane == 0) {
      a.accept_len[s] = du;
      a.bonus[s] = ld_i(am + o + u);
    }
  }
}


template <bool kVerify>
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
  const uint32_t aBytes = (uint32_t)p.BMr * BK * 2;   // W rows a stage receives
  uint8_t* sA = smem;
  uint8_t* sB = smem + (size_t)S * kABytes;
  uint8_t* tail = sB + (size_t)S * bBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(tail);   // full[S], empty[S], tfull[2], tempty[2], drain
  BestPair* s_best = reinterpret_cast<BestPair*>(tail + 8 * (2 * S + 5) + 8);  // [4][BN]
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(tail + 8 * (2 * S + 5));
  // verification state per epilogue warp and node: top-K list, (max, sum) of 2^logit
  const int K = kVerify ? p.K : 1;
  float* s_lv = reinterpret_cast<float*>(s_best + 4 * BN);          // [4][BN][K]
  int* s_li = reinterpret_cast<int*>(s_lv + 4 * BN * K);            // [4][BN][K]
  float2* s_lse = reinterpret_cast<float2*>(s_li + 4 * BN * K);     // [4][BN]
  // per node, the best K-th entry over the 4 warps' lists (an order-preserving
  // key): a row below it cannot be among the CTA's K best
  unsigned long long* s_thr = reinterpret_cast<unsigned long long*>(s_lse + 4 * BN);   // [BN]
  unsigned long long* s_pub = s_thr + BN;   // [BN] the key this CTA last published
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
      mbar_init(tempty0 + 8 * a, kEpiWarps);
    }
    mbar_init(drain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // the producer thread fills the ring's first stages now, before the set-up
    // barrier (the ring is free and its barriers are initialised): the weight
    // stream starts while the other warps allocate TMEM and clear their state
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmX)) : "memory");
    if ((int)blockIdx.x < p.n_vt * p.n_nt) {
      const int vt = (int)blockIdx.x / p.n_nt, nt = (int)blockIdx.x % p.n_nt;
      const int pre = min(S, p.nkb);
      for (int kb = 0; kb < pre; ++kb) {
        const uint32_t fb = full0 + 8 * kb;
        mbar_expect_tx(fb, aBytes + bBytes);
        if (p.packed)
          tma_load_2d(smem_u32(sA + (size_t)kb * kABytes), &tmW, fb, 0, (vt * p.nkb + kb) * BM);
        else
          tma_load_2d(smem_u32(sA + (size_t)kb * kABytes), &tmW, fb, kb * BK, vt * p.BMr);
        tma_load_2d(smem_u32(sB + (size_t)kb * bBytes), &tmX, fb, kb * BK, nt * BN);
      }
      s_issued = pre;
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(s_tmem)),
                 "r"(p.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  for (int i = threadIdx.x; i < 4 * BN; i += kThreads) s_best[i] = BestPair{-INFINITY, 0x7fffffff};
  if (kVerify) {
    for (int i = threadIdx.x; i < 4 * BN * K; i += kThreads) {
      s_lv[i] = -INFINITY;
      s_li[i] = 0x7fffffff;
    }
    for (int i = threadIdx.x; i < 4 * BN; i += kThreads) s_lse[i] = make_float2(-INFINITY, 0.f);
    for (int i = threadIdx.x; i < BN; i += kThreads) {
      s_thr[i] = 0ull;
      s_pub[i] = 0ull;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;

  const int num_tiles = p.n_vt * p.n_nt;

  if (warp == 0) {
    if (lane == 0) {
      // the first min(S, nkb) stages of the first tile went out before the set-up barrier
      const int pre = s_issued;
      int stage = pre % S;
      uint32_t phase = pre == S ? 1u : 0u;
      bool ok = true;
      for (int t = blockIdx.x; t < num_tiles && ok; t += gridDim.x) {
        const int vt = t / p.n_nt, nt = t % p.n_nt;
        for (int kb = (t == (int)blockIdx.x ? pre : 0); kb < p.nkb; ++kb) {
          if (!mbar_wait(empty0 + 8 * stage, phase ^ 1, &s_abort)) {
            ok = false;
            break;
          }
          const uint32_t fb = full0 + 8 * stage;
          mbar_expect_tx(fb, aBytes + bBytes);
          if (p.packed)   // one contiguous 16 KB block of W
            tma_load_2d(smem_u32(sA + (size_t)stage * kABytes), &tmW, fb, 0, (vt * p.nkb + kb) * BM);
          else
            tma_load_2d(smem_u32(sA + (size_t)stage * kABytes), &tmW, fb, kb * BK, vt * p.BMr);
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
    const int q = warp & 3;                 // TMEM lane quarter
    const int ew = q;                       // per-quarter state index
    const int half = (warp - 2) >> 2;       // which 16-column chunks: c0 / 16 = half mod 2
    BestPair* mybest = s_best + ew * BN;
    int lt = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x, ++lt) {
      const int vt = t / p.n_nt, nt = t % p.n_nt;
      const int acc = lt & 1;
      const uint32_t acc_phase = (lt >> 1) & 1;
      // warp-uniform outcome: the tcgen05.ld below is warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait(tfull0 + 8 * acc, acc_phase, &s_abort))) break;
      tc_fence_after();
      if (kVerify) {
        // fold the other CTAs' published K-th keys into the shared threshold (a
        // stale value only lets more rows through)
        for (int c = threadIdx.x - 64; c < BN; c += kEpiThreads)
          if (nt * BN + c < p.total_nodes) atomicMax(&s_thr[c], __ldcg(p.gthr + nt * BN + c));
      }
      const int row = vt * p.BMr + q * 32 + lane;
      const bool row_ok = q * 32 + lane < p.BMr && row < p.vocab;
      for (int c0 = 16 * half; c0 < BN; c0 += 32) {
        uint32_t r[16];
        tc_ld16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN + c0), r);
        float v[16];
        int id[16];
        float v0[16];   // this row's logits, kept for the verification state
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          v[j] = row_ok ? __uint_as_float(r[j]) : -INFINITY;
          v0[j] = v[j];
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
        if (kVerify) {
          // (1) log-sum-exp: each column's sum over this warp's rows of
          //     2^((l - colmax) log2 e), reduce-scattered like the maximum, then
          //     folded into the warp's running (max, sum) of the node
          float e[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float cm = __shfl_sync(0xffffffffu, v[0], lane_of_col(j));
            e[j] = cm == -INFINITY ? 0.f : ex2f((v0[j] - cm) * kLog2e);
          }
#pragma unroll
          for (int half = 8, bit = 16; half >= 1; half >>= 1, bit >>= 1) {
            const bool upper = (lane & bit) != 0;
#pragma unroll
            for (int j = 0; j < half; ++j) {
              const float keep = upper ? e[j + half] : e[j];
              const float give = upper ? e[j] : e[j + half];
              e[j] = keep + __shfl_xor_sync(0xffffffffu, give, bit);
            }
          }
          e[0] += __shfl_xor_sync(0xffffffffu, e[0], 1);
          if ((lane & 1) == 0) {
            float2 cur = s_lse[ew * BN + c0 + col];
            lse_add(cur.x, cur.y, v[0], e[0]);
            s_lse[ew * BN + c0 + col] = cur;
          }
          __syncwarp();
          // (2) top-K per node column: a row is a candidate when its key beats the
          //     CTA's shared threshold; up to four candidates are inserted into
          //     the warp's sorted list by lane 0, more re-select the K best of
          //     list + candidates with K rounds of a warp argmax
          const int row0 = vt * p.BMr + q * 32;
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            float* lv = s_lv + (size_t)(ew * BN + c0 + j) * K;
            int* li = s_li + (size_t)(ew * BN + c0 + j) * K;
            const bool cand = row_ok && make_key(v0[j], row) > s_thr[c0 + j];
            unsigned mask = __ballot_sync(0xffffffffu, cand);
            if (mask == 0u) continue;
            if (__popc(mask) <= 4) {
              while (mask) {
                const int src = __ffs(mask) - 1;
                mask &= mask - 1;
                const float cv = __shfl_sync(0xffffffffu, v0[j], src);
                const int ci = row0 + src;
                if (lane == 0 && better(cv, ci, lv[K - 1], li[K - 1])) {
                  int pos = K - 1;
                  while (pos > 0 && better(cv, ci, lv[pos - 1], li[pos - 1])) {
                    lv[pos] = lv[pos - 1];
                    li[pos] = li[pos - 1];
                    --pos;
                  }
                  lv[pos] = cv;
                  li[pos] = ci;
                }
                __syncwarp();
              }
            } else {
              float av = lane < K ? lv[lane] : -INFINITY;
              int ai = lane < K ? li[lane] : 0x7fffffff;
              float bv = cand ? v0[j] : -INFINITY;
              int bi = cand ? row : 0x7fffffff;
              __syncwarp();
              for (int rr = 0; rr < K; ++rr) {
                const bool useA = better(av, ai, bv, bi);
                const float mv = useA ? av : bv;
                const int mi = useA ? ai : bi;
                float xv;
                int xi;
                warp_best(mv, mi, &xv, &xi);
                if (mi == xi && mv == xv) {   // (value, id) pairs are unique: this lane held it
                  if (useA) {
                    av = -INFINITY;
                    ai = 0x7fffffff;
                  } else {
                    bv = -INFINITY;
                    bi = 0x7fffffff;
                  }
                }
                if (lane == 0) {
                  lv[rr] = xv;
                  li[rr] = xi;
                }
              }
              __syncwarp();
            }
            if (lane == 0 && li[K - 1] != 0x7fffffff)
              atomicMax(&s_thr[c0 + j], make_key(lv[K - 1], li[K - 1]));
            __syncwarp();
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
      if (kVerify) {
        // publish this CTA's K-th keys: no row below another CTA's K-th entry
        // can be among the K best of the whole vocabulary
        for (int c = threadIdx.x - 64; c < BN; c += kEpiThreads) {
          const unsigned long long key = s_thr[c];
          if (key > s_pub[c] && nt * BN + c < p.total_nodes) {   // only when it improved
            atomicMax(p.gthr + nt * BN + c, key);
            s_pub[c] = key;
          }
        }
      }
    }
    // publish this CTA's best per node (every tile of a CTA has the same node tile)
    asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
    if (blockIdx.x < num_tiles) {
      const int nt = blockIdx.x % p.n_nt;
      for (int c = threadIdx.x - 64; c < BN; c += kEpiThreads) {
        BestPair b = s_best[c];
        for (int w = 1; w < 4; ++w) {
          const BestPair o = s_best[w * BN + c];
          if (better(o.v, o.i, b.v, b.i)) b = o;
        }
        const int node = nt * BN + c;
        if (node < p.total_nodes && b.i != 0x7fffffff) atomicMax(&p.keys[node], make_key(b.v, b.i));
        if (kVerify) {
          // this CTA's partial for the node: the 4 warps' lists merged, their sums added
          uint8_t* rec = p.part + ((size_t)blockIdx.x * BN + c) * lm_rec_bytes(K);
          float* pv = reinterpret_cast<float*>(rec);
          int* pi = reinterpret_cast<int*>(rec + 4 * K);
          float2* pl = reinterpret_cast<float2*>(rec + 8 * K);
          int hs[4] = {0, 0, 0, 0};   // next entry of each warp's sorted list
          for (int rr = 0; rr < K; ++rr) {
            int wb = -1;
            float bv = -INFINITY;
            int bi = 0x7fffffff;
#pragma unroll
            for (int w = 0; w < 4; ++w) {
              if (hs[w] >= K) continue;   // exhausted
              const float ov = s_lv[(size_t)(w * BN + c) * K + hs[w]];
              const int oi = s_li[(size_t)(w * BN + c) * K + hs[w]];
              if (wb < 0 || better(ov, oi, bv, bi)) {
                bv = ov;
                bi = oi;
                wb = w;
              }
            }
            pv[rr] = bv;
            pi[rr] = bi;
#pragma unroll
            for (int w = 0; w < 4; ++w) hs[w] += wb == w;
          }
          float m = -INFINITY, sm = 0.f;
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            const float2 x = s_lse[w * BN + c];
            lse_add(m, sm, x.x, x.y);
          }
          *pl = make_float2(m, sm);
        }
      }
    }
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

  // ---- last CTA: argmax decode (+ greedy acceptance) -------------------------
  // the CTA's key publications (before the teardown barrier) are released with
  // its ticket; the last CTA's ticket acquires every other CTA's
  if (threadIdx.x == 0) {
    const unsigned int ticket = atom_add_acq_rel(p.ticket, 1u);
    s_last = (ticket == gridDim.x - 1) ? 1 : 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  int32_t* s_am = reinterpret_cast<int32_t*>(smem);   // pipeline buffers are idle now
  int32_t* s_off = s_am + p.total_nodes;              // the sequences' node offsets (greedy acceptance)
  // the node offsets are loaded beside the key exchange (one round trip for both)
  int offv[(EE_MAX_LM_NODES + 1 + kThreads - 1) / kThreads];
  if constexpr (!kVerify) {
#pragma unroll
    for (int k = 0; k < (EE_MAX_LM_NODES + 1 + kThreads - 1) / kThreads; ++k) {
      const int i = threadIdx.x + k * kThreads;
      offv[k] = i <= p.B ? p.node_off[i] : 0;
    }
  }
  for (int i = threadIdx.x; i < p.total_nodes; i += kThreads) {
    const unsigned long long k = atomicExch(&p.keys[i], 0ull);
    const int a = k ? (int)(0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFull)) : -1;
    s_am[i] = a;
    p.argmax[i] = a;
  }
  if (threadIdx.x == 0) *p.ticket = 0u;
  if constexpr (!kVerify) {   // (verification: the finalize kernel ranks, decides top_tau and accepts)
#pragma unroll
    for (int k = 0; k < (EE_MAX_LM_NODES + 1 + kThreads - 1) / kThreads; ++k) {
      const int i = threadIdx.x + k * kThreads;
      if (i <= p.B) s_off[i] = offv[k];
    }
    __syncthreads();
    AcceptArgs aa{p.B, p.max_T, p.total_nodes, EE_VERIFY_GREEDY, 1, s_off, p.parent, p.draft_tok,
                  p.depth, p.anc, nullptr, p.accept_len, p.path, p.bonus, p.err};
    accept_sequences<false>(aa, s_am, nullptr, nullptr, warp, lane, kThreads / 32);
  }
}


// ---------------------------------------------------------------------------
// Verification finalize (second launch of ee_lmhead_verify): one warp per node
// merges the per-CTA partials of the LM head -- its K best (logit, id) over the
// whole vocabulary and the log-sum-exp -- computes H_norm of Eq. (entropy) and
// top_tau, writes the ranked ids and top_tau to the workspace; the last CTA to
// finish runs the acceptance and zeroes the pruning thresholds.
// ---------------------------------------------------------------------------
constexpr int kFinWarps = 8;
constexpr int kSurv = 256;   // per warp: entries that can still be among a node's K best

struct FinParams {
  int total, B, max_T, BN, n_nt, n_src, K, mode;
  const uint8_t* part;
  unsigned long long* gthr;
  int32_t* tk;                // [total][K] (workspace)
  int32_t* tau;               // [total] (workspace)
  int32_t* topk_ids;          // user outputs or NULL
  int32_t* tau_out;
  float* h_out;
  const int32_t* argmax;      // written by the LM head
  unsigned int* ticket;
  AcceptArgs acc;
};

template <int K>
__global__ void __launch_bounds__(32 * kFinWarps, 1) lm_verify_finalize_kernel(const FinParams p) {
  ee::pdl_allow_next();
  ee::pdl_wait();   // the LM head's partials, thresholds and argmax are complete
  __shared__ float s_sv[kFinWarps][kSurv];
  __shared__ int s_svi[kFinWarps][kSurv];
  __shared__ int s_svn[kFinWarps];
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int BN = p.BN;
  const int node = blockIdx.x * kFinWarps + warp;
  if (node < p.total) {
    const int nt = node / BN, c = node - nt * BN;
    constexpr int kRec = lm_rec_bytes(K) / 16;   // 16-byte words per (CTA, node) record
    // the best K-th key any CTA published: at most the node's true K-th best,
    // so only entries reaching it can be among the K best
    const unsigned long long g = __ldcg(p.gthr + node);
    constexpr int kMaxU = (kNumSMsMax + 31) / 32;
    float cv[kMaxU][K];
    int ci[kMaxU][K];
    float2 xs[kMaxU];
    // every record of the node: lane l takes source CTAs l, l + 32, ...; all
    // loads are unconditional (source 0 stands in for absent ones) and in flight
    // together, the absent ones masked afterwards
    uint4 w[kMaxU][kRec];
#pragma unroll
    for (int u = 0; u < kMaxU; ++u) {
      const int q2 = lane + 32 * u;
      const uint4* rec = reinterpret_cast<const uint4*>(
          p.part + ((size_t)(q2 < p.n_src ? q2 * p.n_nt + nt : nt) * BN + c) * lm_rec_bytes(K));
#pragma unroll
      for (int t = 0; t < kRec; ++t) w[u][t] = __ldcg(rec + t);
    }
#pragma unroll
    for (int u = 0; u < kMaxU; ++u) {
      const uint32_t* ww = reinterpret_cast<const uint32_t*>(w[u]);
#pragma unroll
      for (int rr = 0; rr < K; ++rr) {
        cv[u][rr] = __uint_as_float(ww[rr]);
        ci[u][rr] = (int)ww[K + rr];
      }
      xs[u] = make_float2(__uint_as_float(ww[2 * K]), __uint_as_float(ww[2 * K + 1]));
    }
    float m = -INFINITY, sm = 0.f;
#pragma unroll
    for (int u = 0; u < kMaxU; ++u) {
      const bool valid = lane + 32 * u < p.n_src;
      if (valid) lse_add(m, sm, xs[u].x, xs[u].y);
#pragma unroll
      for (int rr = 0; rr < K; ++rr)
        if (!valid) {
          cv[u][rr] = -INFINITY;
          ci[u][rr] = 0x7fffffff;
        }
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
      const float mo = __shfl_xor_sync(0xffffffffu, m, d);
      const float so = __shfl_xor_sync(0xffffffffu, sm, d);
      lse_add(m, sm, mo, so);
    }
    const float lse = m + logf(sm);
    // survivors into the warp's buffer
    float* sv = s_sv[warp];
    int* svi = s_svi[warp];
    if (lane == 0) s_svn[warp] = 0;
    __syncwarp();
#pragma unroll
    for (int u = 0; u < kMaxU; ++u)
#pragma unroll
      for (int rr = 0; rr < K; ++rr)
        if (ci[u][rr] != 0x7fffffff && make_key(cv[u][rr], ci[u][rr]) >= g) {
          const int pos = atomicAdd(&s_svn[warp], 1);
          if (pos < kSurv) {
            sv[pos] = cv[u][rr];
            svi[pos] = ci[u][rr];
          }
        }
    __syncwarp();
    const int n_sv = s_svn[warp];
    const bool few = n_sv <= kSurv;
    // overflow (not seen with a published threshold): each lane merges its own
    // sorted source lists, then the warp takes the K best of the lane heads
    float lv[K];
    int li[K];
#pragma unroll
    for (int t = 0; t < K; ++t) {
      lv[t] = -INFINITY;
      li[t] = 0x7fffffff;
    }
    if (!few) {
#pragma unroll
      for (int rr = 0; rr < K; ++rr) {
        int wu = 0;
        float bv = cv[0][0];
        int bi = ci[0][0];
#pragma unroll
        for (int u = 1; u < kMaxU; ++u)
          if (better(cv[u][0], ci[u][0], bv, bi)) {
            wu = u;
            bv = cv[u][0];
            bi = ci[u][0];
          }
        lv[rr] = bv;
        li[rr] = bi;
#pragma unroll
        for (int u = 0; u < kMaxU; ++u) {
          if (u != wu) continue;
#pragma unroll
          for (int t = 0; t < K - 1; ++t) {
            cv[u][t] = cv[u][t + 1];
            ci[u][t] = ci[u][t + 1];
          }
          cv[u][K - 1] = -INFINITY;
          ci[u][K - 1] = 0x7fffffff;
        }
      }
    }
    float hsum = 0.f;   // -sum p ln p over the K best, with ln p = logit - lse
    for (int rr = 0; rr < K; ++rr) {
      float xv;
      int xi;
      if (few) {
        float bv = -INFINITY;
        int bi = 0x7fffffff, bpos = -1;
        for (int pos = lane; pos < n_sv; pos += 32)
          if (better(sv[pos], svi[pos], bv, bi)) {
            bv = sv[pos];
            bi = svi[pos];
            bpos = pos;
          }
        warp_best(bv, bi, &xv, &xi);
        if (bpos >= 0 && bi == xi && bv == xv) {
          sv[bpos] = -INFINITY;
          svi[bpos] = 0x7fffffff;
        }
        __syncwarp();
      } else {
        warp_best(lv[0], li[0], &xv, &xi);
        if (xi != 0x7fffffff && li[0] == xi && lv[0] == xv) {   // this lane held it: next one up
#pragma unroll
          for (int t = 0; t < K - 1; ++t) {
            lv[t] = lv[t + 1];
            li[t] = li[t + 1];
          }
          lv[K - 1] = -INFINITY;
          li[K - 1] = 0x7fffffff;
        }
      }
      const float pr = ex2f((xv - lse) * kLog2e);
      if (pr > 0.f) hsum += pr * (lse - xv);
      if (lane == 0) {
        p.tk[(size_t)node * K + rr] = xi;
        if (p.topk_ids) p.topk_ids[(size_t)node * K + rr] = xi;
      }
    }
    if (lane == 0) {
      int tau = 1;
      float h = 0.f;
      if (K >= 2) h = hsum / logf((float)K);
      if (p.mode == EE_VERIFY_ENTROPY) tau = min(K, max(1, (int)ceilf((float)K * h)));
      else if (p.mode == EE_VERIFY_TOPK) tau = K;
      else if (p.mode == EE_VERIFY_DIRECT) tau = 0;
      p.tau[node] = tau;
      if (p.tau_out) p.tau_out[node] = tau;
      if (p.h_out) p.h_out[node] = h;
    }
  }
  // the last CTA to finish: acceptance, then zero the thresholds for the next call
  __syncthreads();
  if (threadIdx.x == 0) s_last = atom_add_acq_rel(p.ticket, 1u) == gridDim.x - 1 ? 1 : 0;   // releases the CTA's writes
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int i = threadIdx.x; i < p.total; i += blockDim.x) p.gthr[i] = 0ull;
  if (threadIdx.x == 0) *p.ticket = 0u;
  accept_sequences<true>(p.acc, p.argmax, p.tk, p.tau, warp, lane, kFinWarps);
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
// With allow_chain, anc == NULL selects linear drafts (parent and depth may
// then be NULL, max_T up to EE_MAX_CHAIN).
ee_status check_lm_args(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                        int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                        const int32_t* depth, const uint64_t* anc, const int32_t* node_off, int32_t B,
                        int32_t total_nodes, int32_t max_T, const int32_t* argmax,
                        const int32_t* accept_len, const int32_t* path, const int32_t* bonus,
                        bool* empty, bool allow_chain) {
  *empty = false;
  const bool chain = allow_chain && anc == nullptr;
  if (B < 0 || total_nodes < 0 || hidden_dim < 8 || vocab < 1 || max_T < 1)
    return EE_ERR_INVALID_ARG;
  if (hidden_dim % 8 != 0 || max_T > (chain ? EE_MAX_CHAIN : EE_MAX_TREE) || total_nodes > EE_MAX_LM_NODES)
    return EE_ERR_UNSUPPORTED;
  if (B == 0 || total_nodes == 0) {
    *empty = true;
    return EE_OK;
  }
  if (!hidden || !lm_w || !draft_tok || (!chain && (!parent || !depth || !anc)) || !node_off || !argmax ||
      !accept_len || !path || !bonus)
    return EE_ERR_INVALID_ARG;
  if (!ee::aligned(hidden, 16) || !ee::aligned(lm_w, 16)) return EE_ERR_INVALID_ARG;
  return EE_OK;
}

// Arguments of the verification rules (ee_lmhead_verify).
struct VerifyArgs {
  int mode, k;
  const uint8_t* gen_mask;
  int32_t* topk_ids;
  int32_t* tau;
  float* h_norm;
  uint8_t* part;               // the workspace's verification region (kLmVerifyOff)
  unsigned int* fin_ticket;
};

// Encode the tensor maps and launch the persistent LM-head kernel; `keys`
// (EE_MAX_LM_NODES running-argmax words, zero on entry), `ticket` (zero on
// entry) and `err` are the kernel's scratch.  `va` selects the verification
// variant (NULL: greedy acceptance).
ee_status launch_lmhead(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                        int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                        const int32_t* depth, const uint64_t* anc, const int32_t* node_off, int32_t B,
                        int32_t total_nodes, int32_t max_T, int32_t* argmax, int32_t* accept_len,
                        int32_t* path, int32_t* bonus, float* logits_or_null,
                        unsigned long long* keys, unsigned int* ticket, int32_t* err,
                        ee_stream_t stream, bool pdl, const VerifyArgs* va = nullptr, bool packed = false) {
  LmParams p;
  p.packed = packed ? 1 : 0;
  p.vocab = vocab;
  p.hidden = hidden_dim;
  p.total_nodes = total_nodes;
  p.B = B;
  p.max_T = max_T;
  p.n_nt = (total_nodes + 255) / 256;
  p.BN = ((total_nodes + p.n_nt - 1) / p.n_nt + 15) / 16 * 16;
  // vocabulary tiles: as many per CTA for every CTA (the launch's end is the
  // busiest CTA's), each of ceil(V / tiles) <= 128 rows; the MMA's remaining
  // rows hold stale shared memory and are dropped by the epilogue.  Below 64
  // rows a tile would waste most of its MMA: plain 128-row tiles then.
  {
    const int n_vt0 = (vocab + BM - 1) / BM;
    const int per_group = std::max(1, ee::kNumSMs / p.n_nt);   // CTAs per node tile
    const int k = (n_vt0 + per_group - 1) / per_group;
    const int rows = (vocab + k * per_group - 1) / (k * per_group);
    p.BMr = rows >= 64 && !packed ? rows : BM;
    p.n_vt = (vocab + p.BMr - 1) / p.BMr;
  }
  p.nkb = (hidden_dim + BK - 1) / BK;
  const size_t stage_bytes = (size_t)kABytes + (size_t)p.BN * BK * 2;
  const int K = va ? va->k : 1;
  // epilogue state: running best per warp and node (+ top-K lists and sums)
  const size_t epi = 4 * (size_t)p.BN * sizeof(BestPair) +
                     (va ? 4 * (size_t)p.BN * (8 * K + 8) + 16 * (size_t)p.BN : 0);
  const size_t fixed = 1024 /*align slack*/ + 8 * (2 * 8 + 5) + 8 + epi;
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
  p.mode = va ? va->mode : EE_VERIFY_GREEDY;
  p.K = K;
  p.gen_mask = va ? va->gen_mask : nullptr;
  p.topk_ids = va ? va->topk_ids : nullptr;
  p.tau_out = va ? va->tau : nullptr;
  p.h_out = va ? va->h_norm : nullptr;
  p.part = va ? va->part : nullptr;
  p.gthr = va ? reinterpret_cast<unsigned long long*>(va->part + ee::kLmGthrOff) : nullptr;

  CUtensorMap tmW, tmX;
  if (packed) {
    // the packed W as rows of 64 elements: block (vt, kb) is rows (vt * nkb + kb) * 128 ..
    if (!encode_2d(&tmW, lm_w, (uint64_t)BK, (uint64_t)p.n_vt * p.nkb * BM, BK, (uint32_t)BM)) return EE_ERR_CUDA;
  } else if (!encode_2d(&tmW, lm_w, (uint64_t)hidden_dim, (uint64_t)vocab, BK, (uint32_t)p.BMr)) {
    return EE_ERR_CUDA;
  }
  if (!encode_2d(&tmX, hidden, (uint64_t)hidden_dim, (uint64_t)total_nodes, BK, p.BN))
    return EE_ERR_CUDA;

  const size_t smem = 1024 + (size_t)p.stages * stage_bytes + 8 * (2 * p.stages + 5) + 8 + epi;
  // the last CTA reuses the pipeline buffers: argmax (+ ranked ids and top_tau) per node
  // the last CTA: argmax per node and the node offsets
  const size_t last = 1024 + (size_t)(2 * EE_MAX_LM_NODES + 5) * 4;
  const size_t smem_acc = std::max(smem, last);
  if (smem_acc > 227 * 1024) return EE_ERR_UNSUPPORTED;
  {
    // the dynamic shared memory attribute, raised once per device and kernel
    int dev = 0;
    const ee_status ds = ee::current_device(&dev);
    if (ds != EE_OK) return ds;
    static std::mutex mu;
    static size_t attr_bytes[ee::kMaxDevices][2] = {};
    std::lock_guard<std::mutex> lock(mu);
    if (attr_bytes[dev][va ? 1 : 0] < smem_acc) {
      if (va)
        EE_CUDA_OK(cudaFuncSetAttribute(lmhead_accept_kernel<true>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_acc));
      else
        EE_CUDA_OK(cudaFuncSetAttribute(lmhead_accept_kernel<false>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_acc));
      attr_bytes[dev][va ? 1 : 0] = smem_acc;
    }
  }
  const int num_tiles = p.n_vt * p.n_nt;
  int grid = (ee::kNumSMs / p.n_nt) * p.n_nt;   // multiple of n_nt: each CTA keeps one node tile
  if (grid > num_tiles) grid = num_tiles;
  if (grid < 1) grid = 1;
  if (va && (size_t)grid * p.BN * ee::lm_rec_bytes(K) > ee::kLmPartBytes) return EE_ERR_UNSUPPORTED;
  if (va) {
    EE_CUDA_OK(ee::launch_pdl(lmhead_accept_kernel<true>, dim3(grid), dim3(kThreads), smem_acc,
                              (cudaStream_t)stream, 1, tmW, tmX, p));
    FinParams fp;
    fp.total = total_nodes;
    fp.B = B;
    fp.max_T = max_T;
    fp.BN = p.BN;
    fp.n_nt = p.n_nt;
    fp.n_src = grid / p.n_nt;
    fp.K = K;
    fp.mode = va->mode;
    fp.part = va->part;
    fp.gthr = p.gthr;
    fp.tk = reinterpret_cast<int32_t*>(va->part + ee::kLmTkOff);
    fp.tau = reinterpret_cast<int32_t*>(va->part + ee::kLmTauOff);
    fp.topk_ids = va->topk_ids;
    fp.tau_out = va->tau;
    fp.h_out = va->h_norm;
    fp.argmax = argmax;
    fp.ticket = va->fin_ticket;
    fp.acc = AcceptArgs{B, max_T, total_nodes, va->mode, K, node_off, parent, draft_tok, depth, anc,
                        va->gen_mask, accept_len, path, bonus, err};
    const dim3 fg((total_nodes + kFinWarps - 1) / kFinWarps), fb(32 * kFinWarps);
    cudaError_t fe = cudaErrorInvalidValue;
    switch (K) {
#define EE_FIN_CASE(n) \
  case n:              \
    fe = ee::launch_pdl(lm_verify_finalize_kernel<n>, fg, fb, 0, (cudaStream_t)stream, 1, fp); \
    break;
      EE_FIN_CASE(1) EE_FIN_CASE(2) EE_FIN_CASE(3) EE_FIN_CASE(4)
      EE_FIN_CASE(5) EE_FIN_CASE(6) EE_FIN_CASE(7) EE_FIN_CASE(8)
#undef EE_FIN_CASE
      default:
        break;
    }
    EE_CUDA_OK(fe);
  } else if (pdl) {
    EE_CUDA_OK(ee::launch_pdl(lmhead_accept_kernel<false>, dim3(grid), dim3(kThreads), smem_acc,
                              (cudaStream_t)stream, 1, tmW, tmX, p));
  } else {
    lmhead_accept_kernel<false><<<grid, kThreads, smem_acc, (cudaStream_t)stream>>>(tmW, tmX, p);
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
                                     bonus, &empty, true);
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

namespace {

// ---------------------------------------------------------------------------
// Tile-ordered LM-head weights (ee_lmhead_pack_weights): the 128-row x
// 64-column blocks of W that the kernel loads one per ring stage, each stored
// as one contiguous 16 KB run, so that the weight stream reads whole DRAM
// pages instead of 128-byte pieces 2*H bytes apart.  Block (vt, kb) = rows
// [128 vt, 128 vt + 128) x columns [64 kb, 64 kb + 64) of W, row-major inside
// the block, at element ((vt * nkb + kb) * 128) * 64; rows past V and columns
// past H are zero.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) pack_w_kernel(const uint4* __restrict__ w, int vocab, int hidden,
                                                     int n_vt, int nkb, uint4* __restrict__ out) {
  const size_t total = (size_t)n_vt * nkb * BM * (BK / 8);   // 16-byte words
  for (size_t q = (size_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (size_t)gridDim.x * blockDim.x) {
    const int c8 = (int)(q & 7);
    const size_t rest = q >> 3;
    const int r = (int)(rest & (BM - 1));
    const size_t blk = rest / BM;
    const int kb = (int)(blk % (size_t)nkb), vt = (int)(blk / (size_t)nkb);
    const int row = vt * BM + r, col = kb * BK + c8 * 8;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (row < vocab && col < hidden) v = w[((size_t)row * hidden + col) / 8];
    out[q] = v;
  }
}

size_t packed_w_bytes(int32_t vocab, int32_t hidden_dim) {
  if (vocab < 1 || hidden_dim < 8 || hidden_dim % 8 != 0) return 0;
  return (size_t)((vocab + BM - 1) / BM) * BM * (size_t)((hidden_dim + BK - 1) / BK) * BK * 2;
}

}  // namespace

extern "C" size_t ee_lmhead_packed_bytes(int32_t vocab, int32_t hidden_dim) {
  return packed_w_bytes(vocab, hidden_dim);
}

extern "C" ee_status ee_lmhead_pack_weights(const ee_bf16* lm_w, int32_t vocab, int32_t hidden_dim, ee_bf16* packed,
                                            size_t packed_bytes, ee_stream_t stream) {
  const size_t need = packed_w_bytes(vocab, hidden_dim);
  if (need == 0) return vocab < 1 || hidden_dim < 8 ? EE_ERR_INVALID_ARG : EE_ERR_UNSUPPORTED;
  if (!lm_w || !packed || !ee::aligned(lm_w, 16) || !ee::aligned(packed, 16)) return EE_ERR_INVALID_ARG;
  if (packed_bytes < need) return EE_ERR_INVALID_ARG;
  const int n_vt = (vocab + BM - 1) / BM, nkb = (hidden_dim + BK - 1) / BK;
  const size_t words = need / 16;
  const int grid = (int)std::min<size_t>((words + 255) / 256, (size_t)ee::kNumSMs * 16);
  pack_w_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(reinterpret_cast<const uint4*>(lm_w), vocab, hidden_dim,
                                                        n_vt, nkb, reinterpret_cast<uint4*>(packed));
  EE_CUDA_OK(cudaGetLastError());
  return EE_OK;
}

extern "C" ee_status ee_lmhead_accept_packed(const ee_bf16* hidden, const ee_bf16* lm_w_packed,
                                             int32_t hidden_dim, int32_t vocab, const int32_t* draft_tok,
                                             const int32_t* parent, const int32_t* depth, const uint64_t* anc,
                                             const int32_t* node_off, int32_t B, int32_t total_nodes,
                                             int32_t max_T, int32_t* argmax, int32_t* accept_len,
                                             int32_t* path, int32_t* bonus, float* logits_or_null,
                                             void* ws, size_t ws_bytes, ee_stream_t stream) {
  bool empty = false;
  const ee_status st = check_lm_args(hidden, lm_w_packed, hidden_dim, vocab, draft_tok, parent, depth, anc,
                                     node_off, B, total_nodes, max_T, argmax, accept_len, path,
                                     bonus, &empty, true);
  if (st != EE_OK || empty) return st;
  if (!ws || !ee::aligned(ws, 256)) return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  char* wsb = static_cast<char*>(ws);
  return launch_lmhead(hidden, lm_w_packed, hidden_dim, vocab, draft_tok, parent, depth, anc, node_off, B,
                       total_nodes, max_T, argmax, accept_len, path, bonus, logits_or_null,
                       reinterpret_cast<unsigned long long*>(wsb + ee::kArgmaxOff),
                       reinterpret_cast<unsigned int*>(wsb + ee::kTicketOff), ee::err_word(ws),
                       stream, true, nullptr, true);
}

extern "C" ee_status ee_lmhead_verify(const ee_bf16* hidden, const ee_bf16* lm_w, int32_t hidden_dim,
                                      int32_t vocab, const int32_t* draft_tok, const int32_t* parent,
                                      const int32_t* depth, const uint64_t* anc,
                                      const int32_t* node_off, const uint8_t* gen_mask_or_null,
                                      int32_t B, int32_t total_nodes, int32_t max_T, int32_t mode,
                                      int32_t k, int32_t* argmax, int32_t* topk_ids_or_null,
                                      int32_t* top_tau_or_null, float* h_norm_or_null,
                                      int32_t* accept_len, int32_t* path, int32_t* bonus,
                                      float* logits_or_null, void* ws, size_t ws_bytes,
                                      ee_stream_t stream) {
  if (mode < EE_VERIFY_GREEDY || mode > EE_VERIFY_ENTROPY || k < 1 || k > ee::kLmMaxK ||
      (mode == EE_VERIFY_ENTROPY && k < 2))
    return EE_ERR_INVALID_ARG;
  bool empty = false;
  const ee_status st = check_lm_args(hidden, lm_w, hidden_dim, vocab, draft_tok, parent, depth, anc,
                                     node_off, B, total_nodes, max_T, argmax, accept_len, path,
                                     bonus, &empty, false);
  if (st != EE_OK || empty) return st;
  if (!ws || !ee::aligned(ws, 256)) return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kLmVerifyOff + ee::kLmVerifyBytes) return EE_ERR_WORKSPACE;
  char* wsb = static_cast<char*>(ws);
  VerifyArgs va{mode, k, gen_mask_or_null, topk_ids_or_null, top_tau_or_null, h_norm_or_null,
                reinterpret_cast<uint8_t*>(wsb + ee::kLmVerifyOff),
                reinterpret_cast<unsigned int*>(wsb + ee::kFinTicketOff)};
  return launch_lmhead(hidden, lm_w, hidden_dim, vocab, draft_tok, parent, depth, anc, node_off, B,
                       total_nodes, max_T, argmax, accept_len, path, bonus, logits_or_null,
                       reinterpret_cast<unsigned long long*>(wsb + ee::kArgmaxOff),
                       reinterpret_cast<unsigned int*>(wsb + ee::kTicketOff), ee::err_word(ws),
                       stream, true, &va);
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
void* g_lm_scratch_ptr[ee::kMaxDevices] = {};

std::mutex g_lm_scratch_mu;

// The current device's copy of the array; the launch stream must belong to
// that device (the address, like the kernel attributes, is the current
// device's), else EE_ERR_INVALID_ARG.
ee_status static_scratch(ee_stream_t stream, void** out) {
  int dev = -1;
  const ee_status ds = ee::current_device(&dev);
  if (ds != EE_OK) return ds;
  if (stream) {
    int sdev = -1;
    EE_CUDA_OK(cudaStreamGetDevice((cudaStream_t)stream, &sdev));
    if (sdev != dev) return EE_ERR_INVALID_ARG;
  }
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
                                     bonus, &empty, true);
  if (st != EE_OK || empty) return st;   // total_nodes > EE_MAX_LM_NODES -> EE_ERR_UNSUPPORTED
  void* scratch = nullptr;
  const ee_status ss = static_scratch(stream, &scratch);
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
