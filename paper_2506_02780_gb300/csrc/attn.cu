// ee_tree_verify_attn: tree-masked attention of every draft node over the
// paged KV cache plus the tree's own K/V, one layer per call (EfficientEdit
// Sec. III-A: a single target forward pass over (prefix, draft) scores every
// draft token; with a tree, each node sees the prefix and its own root path).
// ee_tree_verify_attn_inplace and ee_chain_verify_attn are the same kernel
// with the draft's K/V in the cache after the context (see kKV below).
//
// Work decomposition (split-KV):
//   - For a (sequence, KV head) the query rows are the g = n_q / n_kv heads of
//     the group times the T tree nodes, row r = node * g + head_in_group, so
//     one K/V tile feeds g * T rows (GQA packing).  A CTA owns 128 rows: the
//     M side of a tcgen05 MMA.
//   - A CTA processes segments: contiguous 128-key tile ranges of one row
//     block.  Uniform launches cut each row block's context into S <= 16
//     chunks of `chunk` keys (a multiple of the 16-token page, at most 2048
//     pages), one CTA each; the last chunk also processes the tree keys (one
//     128-key tile, masked by the ancestor bitmask).  Balanced launches give
//     each of one CTA per SM an equal share of all row blocks' tiles (a CTA
//     may finish one row block and start the next).  A CTA stages each
//     segment's page ids in shared memory.
//   - Q lives in shared memory (the softmax threads load the block's rows
//     coalesced and store them in the 128-byte-swizzled K-major layout TMA
//     gives the K tiles) and is the A operand of S = Q K^T; TMEM holds three S
//     buffers and O (4 x 128 fp32 columns).
//   - Keys come in 128-key tiles.  Warps 0 and 2 stream K and V tiles with TMA
//     (one 16-row box per page and 64-dim half, spread over 8 lanes; the tree's
//     K/V through a 3-D map) into a 3-stage K ring and a 2-stage V ring.  Warp
//     1 issues tcgen05.mma in a fixed order: S = Q K^T for the first three
//     tiles (bf16, fp32 accumulators in TMEM), then for each tile O += P V
//     followed by the Q K^T three tiles ahead, which overwrites the TMEM
//     columns P lived in (the in-order tensor pipe finishes reading P first).
//     With three S buffers the hand-off chain P(t) -> P.V(t) -> Q.K^T(t+3) ->
//     softmax(t+3) spans three tiles, so it no longer sets the tile period.
//   - P.V runs on bf16 operands: P is split into a bf16 head (the fp32 value
//     rounded to nearest bf16) and a bf16 tail (the exact remainder, rounded
//     to nearest bf16), both written over S in TMEM and used as the MMA A
//     operand; V is read straight from shared memory (MN-major).  P is carried
//     to about 2^-17 relative (fp16 would give 2^-11) and V needs no
//     conversion; per column pair the split is two packing conversions, a
//     shift, a mask and one packed subtraction.
//   - Warps 4-11 own one query row per thread (its TMEM lane), two warps per
//     lane quarter splitting each tile's keys: they read S, mask, keep the
//     running max/sum, write P, and rescale O in TMEM only when a row's max
//     grows by more than 2^8 (the stale max keeps every P <= 256, and the final
//     O / l is unchanged).
//   - Every chunk-CTA writes its unnormalised O rows and (max, sum) from TMEM
//     to its own slot of the workspace (fp32, column-chunk major so that a
//     warp's stores are contiguous; the slots stay in L2).  Once all S slots of
//     a row block are written, chunk k merges the contiguous rows
//     [k * ceil(128 / S), ...) of all S slots with log-sum-exp weights and
//     writes the fp32 output: one launch, no second pass, and L2 moves the
//     partials several times faster than distributed shared memory does.
//     A segment that is a whole row block writes O / l directly.  The CTAs of
//     a row block learn that all slots are written in one of two ways, chosen
//     by the host:
//       cluster: they form a thread-block cluster and meet at one cluster
//         barrier (release / acquire at cluster scope);
//       cooperative: the launch is cooperative (every CTA resident at once);
//         the row block's 64-bit count grows by 720720 = lcm(1..16) per
//         launch: each of its S CTAs reads the count at its start (a
//         multiple of 720720 plus some of this launch's arrivals, never all:
//         its own is missing; a relaxed load whose value is first used at the
//         end), stores its partial, and after a CTA barrier one thread adds
//         720720 / S with a release reduction and waits (acquire) for the next
//         multiple.  One release per CTA orders all its threads'
//         stores, and nothing resets the count at the end of the kernel.  No
//         GPC packing constraint: S can be any value up to 16, so the grid can
//         cover every SM.  Balanced launches count the pieces of each split
//         row block the same way.
//     Every CTA, also one whose chunk is empty for a short sequence, arrives:
//     every wait before the arrival is bounded.
//   - The next kernel in the stream may launch (programmatic dependent launch)
//     once every CTA has drained its pipeline; triggering earlier lets its
//     CTAs hold SMs that a later wave of this grid still needs.
// Shared-memory traffic per 128-key tile: K 64 KB + V 64 KB (TMA write, MMA
// read) + Q 32 KB (MMA read).
#include "ee_common.cuh"
#include "ee_ptx.cuh"

namespace {

using namespace ee;

constexpr int kThreads = 384;                    // 12 warps, roles below
constexpr int kRows = 128;                       // query rows per CTA (MMA M)
constexpr int kKT = 128;                         // keys per tile (MMA N of Q K^T, K of P V)
constexpr int kD = EE_HEAD_DIM;                  // 128
constexpr int kKST = 3;                          // K ring depth
constexpr int kVST = 2;                          // V ring depth
constexpr int kSB = 3;                           // S buffers in TMEM (Q.K^T runs kSB tiles ahead)
constexpr uint32_t kKVHalf = kKT * 128;          // 16 KB: one 64-dim half of a K or V tile
constexpr uint32_t kKVBytes = 2 * kKVHalf;       // 32 KB
constexpr int kMaxCtaPages = 2048;               // context pages one CTA can own (32768 keys)
constexpr uint32_t kOffK = 0;
constexpr uint32_t kOffV = kOffK + kKST * kKVBytes;
constexpr uint32_t kOffQ = kOffV + kVST * kKVBytes;  // Q block, 128 rows x 128 bf16, SW128 K-major
constexpr uint32_t kOffPages = kOffQ + kKVBytes;
constexpr uint32_t kOffBar = kOffPages + 4 * kMaxCtaPages;
constexpr uint32_t kNumBars = 2 * kKST + 2 * kVST + 2 * kSB + 2 + 3;
constexpr uint32_t kSmemBytes = 1024 + kOffBar + 8 * kNumBars + 64;
constexpr uint32_t kTmemCols = 512;              // S0 [0,128) S1 [128,256) S2 [256,384) O [384,512)
constexpr uint32_t kColO = 384;
constexpr float kRescaleLog2 = 8.0f;
constexpr int kMaxCluster = 8;                   // portable thread-block cluster size
constexpr int kMaxSplits = ee::kAttnMaxSplits;   // chunks per row block (cooperative launch)
constexpr int kMaxBalSeqs = 512;                 // sequences of a balanced launch
// warp roles (warp 3 is idle after set-up); softmax warps 4..11, two per TMEM
// lane quarter
constexpr int kWarpK = 0, kWarpMma = 1, kWarpV = 2, kWarpSched = 3, kWarpSoft0 = 4;
constexpr int kSoftThreads = 8 * 32;

static_assert(kRows == ee::kAttnRows, "row block size");
static_assert(kThreads == 32 * kWarpSoft0 + kSoftThreads, "eight softmax warps, two per TMEM lane quarter");
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
static_assert(ee::kAttnMlOff == kRows * kD * 4, "partial slot: O rows, then (m, l), then counters");

struct AttnParams {
  const __nv_bfloat16* q;
  const int32_t* block_table;
  const int32_t* ctx_len;
  const int32_t* node_off;
  const uint64_t* anc;
  float* out;
  uint8_t* part;               // per-CTA partial slots (ee::kAttnPartBytes each), S > 1 only
  int32_t* err;
  int num_pages, max_pages, max_ctx, n_q, n_kv, g, total_nodes, max_T, nrb, chunk, S;
  int coop;                    // 1: cooperative launch, counters; 0: cluster barrier
  int B;                       // sequences (the balanced mode's work list)
  float scale_log2;
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// {hi, lo} rounded to nearest bf16 and packed: lo in bits 0-15, hi in 16-31
__device__ __forceinline__ uint32_t bf16x2_rn(float hi, float lo) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}
// three-input maximum (one instruction on sm_100-family GPUs)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Loaded-page mask of context tile t: bit i set when the tile's 16-row block i
// holds keys below k_end in a valid page.  s_pages holds the CTA's page ids
// (-1 for an out-of-range block-table entry).
__device__ __forceinline__ unsigned tile_mask(const int32_t* s_pages, int t, int k_begin, int k_end) {
  unsigned m = 0u;
#pragma unroll
  for (int i = 0; i < kKT / 16; ++i) {
    const int pos = k_begin + t * kKT + 16 * i;
    m |= (pos < k_end && s_pages[t * (kKT / 16) + i] >= 0) ? (1u << i) : 0u;
  }
  return m;
}

// Merge rows [r0, r0 + nown) of a row block (query rows row0, ...) from its S
// partial slots with log-sum-exp weights (Sec. III-A: the scores of one row
// are normalised over all keys it sees) and write the fp32 output.  Thread t
// takes row t % nown and the 16-byte column chunks t / nown + k * tpr, where
// tpr = 256 / nown threads share a row: the loads of a warp for one chunk are
// contiguous, and every load is issued before the first one is used.  Rows
// without keys have (m, l) = (-inf, 0) and weight 0; their O words, never
// written, are not used.
template <int S>
__device__ __forceinline__ void merge_rows(const AttnParams& p, size_t slot_a, size_t slot_b, int stride,
                                           int row0, int r0, int nown, int o, int hk) {
  // partial s lives in slot slot_a (s = 0) or slot_b + (s - 1) * stride
  auto slot = [&](int s) -> const uint8_t* {
    return p.part + (s == 0 ? slot_a : slot_b + (size_t)(s - 1) * stride) * kAttnPartBytes;
  };
  constexpr int kRpc = (kRows + S - 1) / S;
  constexpr int kTprMin = kThreads / kRpc;
  constexpr int kCh = (kD / 4 + kTprMin - 1) / kTprMin;   // chunks per thread, at most
  const int tpr = kThreads / nown;                        // >= kTprMin, as nown <= kRpc
  const int j = threadIdx.x % nown, cg = threadIdx.x / nown;
  if (cg >= tpr) return;
  float2 ml[S];
#pragma unroll
  for (int s = 0; s < S; ++s)
    ml[s] = __ldcg(reinterpret_cast<const float2*>(slot(s) + kAttnMlOff) + r0 + j);
  float4 v[kCh][S];
#pragma unroll
  for (int k = 0; k < kCh; ++k) {
    const int c = cg + k * tpr;
#pragma unroll
    for (int s = 0; s < S; ++s)
      v[k][s] = c < kD / 4 ? __ldcg(reinterpret_cast<const float4*>(slot(s)) +
                                    (size_t)c * kRows + r0 + j)
                           : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  float M = -INFINITY;
#pragma unroll
  for (int s = 0; s < S; ++s) M = fmaxf(M, ml[s].x);
  float w[S], L = 0.f;
#pragma unroll
  for (int s = 0; s < S; ++s) {
    w[s] = ml[s].x == -INFINITY ? 0.f : ex2(ml[s].x - M);
    L += w[s] * ml[s].y;
  }
  const float il = L > 0.f ? 1.f / L : 0.f;
  const int rrow = row0 + j;
  const int nd = rrow / p.g;
  float4* dst = reinterpret_cast<float4*>(p.out + ((size_t)(o + nd) * p.n_q + hk * p.g + (rrow - nd * p.g)) * kD);
#pragma unroll
  for (int k = 0; k < kCh; ++k) {
    const int c = cg + k * tpr;
    if (c >= kD / 4) break;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int s = 0; s < S; ++s) {
      if (w[s] == 0.f) continue;
      a.x = fmaf(w[s], v[k][s].x, a.x);
      a.y = fmaf(w[s], v[k][s].y, a.y);
      a.z = fmaf(w[s], v[k][s].z, a.z);
      a.w = fmaf(w[s], v[k][s].w, a.w);
    }
    dst[c] = make_float4(a.x * il, a.y * il, a.z * il, a.w * il);
  }
}

// A row block's partial that this CTA merges with the other pieces of the same
// row block (balanced mode): the unit, the number of pieces K, this CTA's
// piece index k, and where the pieces' slots are (piece 0 at slot0, piece
// s >= 1 at slot1 + 2 (s - 1)).
struct BalPiece {
  int hk, rb, o, R, K, k, slot0, slot1;
  unsigned long long target;   // the count the row block's pieces raise it to
};
// A split row block's pieces meet at a 64-bit count in the trailer of its first
// partial slot: every launch raises it by kCountGen in all (kCountGen / K per
// piece, a release reduction after the piece's partial is stored), so a count a
// piece reads at any time before its own arrival is a multiple of kCountGen
// plus fewer than K arrivals, and the piece waits (acquire) for the next
// multiple.  The count is never reset; ee_workspace_init
// zeroes it.
constexpr unsigned long long kCountGen = 720720;   // lcm(1..16): K <= 16 divides it

// Where the draft's K/V are (template kKV):
//   kKVTree  -- k_tree / v_tree, one extra 128-key tile after the context;
//   kKVInPlace -- in the cache at positions ctx .. ctx + T - 1 (in-place
//     speculative K/V): a sequence's keys are positions [0, ctx + T) of its
//     pages, and a key at p >= ctx is visible to a row when bit p - ctx of the
//     row's ancestor mask is set;
//   kKVChain -- as kKVInPlace for a linear draft of up to EE_MAX_CHAIN tokens:
//     node i sees positions 0 .. ctx + i (causal), and a row block's keys end
//     at its last node's position.
constexpr int kKVTree = 0, kKVInPlace = 1, kKVChain = 2;

// Chain drafts: 128-key tiles of row block r (its last node's position + 1 keys).
__host__ __device__ inline int chain_rb_tiles(int ctx, int T, int g, int r) {
  const int n_hi = min(T - 1, ((r + 1) * kRows - 1) / g);
  return (ctx + n_hi + 1 + kKT - 1) / kKT;
}

// kBal: balanced work list (else one (row block, chunk) per CTA).
template <bool kBal, int kKV>
__global__ void __launch_bounds__(kThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tmKc, const __grid_constant__ CUtensorMap tmVc,
               const __grid_constant__ CUtensorMap tmKt, const __grid_constant__ CUtensorMap tmVt,
               const AttnParams p) {
  constexpr bool kIP = kKV != kKVTree;       // draft K/V in the cache
  constexpr bool kChain = kKV == kKVChain;
  constexpr int kMaxT = kChain ? EE_MAX_CHAIN : EE_MAX_TREE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_kissued[kKST], s_vissued[kVST];
  __shared__ float s_xmax[2][2][kRows];             // [tile parity][half][row]: softmax pair exchange
  __shared__ float s_xl[2][kRows];                  // [half][row]: final row sums
  // balanced mode: per sequence (node offset, T, context length, tiles) and the
  // exclusive prefix of the sequences' work in tiles
  __shared__ int4 s_seq[kBal ? kMaxBalSeqs : 1];
  __shared__ int s_wpre[kBal ? kMaxBalSeqs + 1 : 1];
  __shared__ int s_sched[7];   // balanced: range start, range end, W, N, tiles done, segments done, next end
  __shared__ BalPiece s_pc[2];                      // balanced: this CTA's pieces of split units
  __shared__ int s_npc;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sK = sbase + kOffK, sV = sbase + kOffV;
  const uint32_t bar0 = sbase + kOffBar;
  const uint32_t k_full = bar0, k_empty = k_full + 8 * kKST;
  const uint32_t v_full = k_empty + 8 * kKST, v_empty = v_full + 8 * kVST;
  const uint32_t s_full = v_empty + 8 * kVST, p_full = s_full + 8 * kSB, o_done = p_full + 8 * kSB;
  const uint32_t drain = o_done + 16, q_ready = drain + 8, o_final = q_ready + 8;

  // on-chip set-up first: it touches no global memory, so it overlaps the end
  // of the previous kernel in the stream
  if (threadIdx.x == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmKc)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmVc)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmKt)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmVt)) : "memory");
    s_abort = 0;
    s_npc = 0;
    for (int i = 0; i < kKST; ++i) {
      mbar_init(k_full + 8 * i, 1);
      mbar_init(k_empty + 8 * i, 1);
      s_kissued[i] = -1;
    }
    for (int i = 0; i < kVST; ++i) {
      mbar_init(v_full + 8 * i, 1);
      mbar_init(v_empty + 8 * i, 1);
      s_vissued[i] = -1;
    }
    for (int i = 0; i < kSB; ++i) {
      mbar_init(s_full + 8 * i, 1);
      mbar_init(p_full + 8 * i, 2 * kRows);
    }
    for (int i = 0; i < 2; ++i) mbar_init(o_done + 8 * i, 1);
    mbar_init(drain, 1);
    mbar_init(q_ready, 2 * kRows);
    mbar_init(o_final, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_async_smem();
  }
  if (warp == kWarpMma) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&s_tmem)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }

  pdl_wait();   // no global access before the previous kernel's writes are visible
  const int g = p.g;

  // ---- balanced mode: the shared work list ---------------------------------------
  // Work is counted in 128-key tiles: sequence b brings n_kv x nrb_b units (a
  // KV head's row block) of ceil(ctx_b / 128) context tiles + 1 tree tile.
  // Units are ordered sequence, KV head, row block; CTA c takes the tiles
  // [c W / N, (c + 1) W / N) of that order, so a CTA may finish one unit and
  // start the next (at most two of its segments are pieces of split units).
  // N is capped so that every CTA gets at least m = max(2, ceil(t_max / 14))
  // tiles, which bounds the pieces of any unit by 15.
  // Warp 3 (otherwise idle) builds it: lane l takes sequences [16 l, 16 l + 16).
  if constexpr (kBal) {
    if (warp == kWarpSched) {
      constexpr int kPer = kMaxBalSeqs / 32;
      int wl[kPer];
      int wsum = 0, tmax = 0;
#pragma unroll
      for (int k = 0; k < kPer; ++k) {   // loads first (clamped indices), all in flight
        const int bb = min(lane * kPer + k, p.B - 1);
        s_seq[lane * kPer + k] = make_int4(p.node_off[bb], p.node_off[bb + 1], p.ctx_len[bb], 0);
      }
      __syncwarp();
      // chain drafts: one KV head's tiles are a sum over its row blocks; for a
      // few sequences the warp sums each one's row blocks 32 at a time (stored
      // in .w), otherwise each lane walks its own sequences' row blocks
      const bool coop = kChain && p.B <= 64;
      if (coop) {
        for (int bb = 0; bb < p.B; ++bb) {
          const int4 sq = s_seq[bb];
          const int Tb = sq.y - sq.x;
          const bool bad = Tb < 1 || Tb > kMaxT || Tb > p.max_T || sq.x < 0 || sq.x + Tb > p.total_nodes;
          const int c = min(max(sq.z, 0), p.max_ctx);
          int acc = 0;
          if (!bad)
            for (int r = lane; r < (Tb * g + kRows - 1) / kRows; r += 32) acc += chain_rb_tiles(c, Tb, g, r);
          acc = __reduce_add_sync(0xffffffffu, acc);
          __syncwarp();
          if (lane == 0) s_seq[bb].w = acc;
        }
        __syncwarp();
      }
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const int bb = lane * kPer + k;
        wl[k] = 0;
        if (bb < p.B) {
          const int4 sq = s_seq[bb];
          const int Tb = sq.y - sq.x;
          const bool bad = Tb < 1 || Tb > kMaxT || Tb > p.max_T || sq.x < 0 || sq.x + Tb > p.total_nodes;
          if (bad && blockIdx.x == 0) flag_error(p.err, EE_DEVERR_TREE);
          int c = sq.z;
          if (c < 0 || c > p.max_ctx) {
            if (blockIdx.x == 0) flag_error(p.err, EE_DEVERR_CTX);
            c = c < 0 ? 0 : p.max_ctx;
          }
          // tiles of a unit (chain: of one KV head's row blocks, whose lengths differ)
          const int nrb_b = bad ? 1 : (Tb * g + kRows - 1) / kRows;
          int tiles = kIP ? (c + (bad ? 1 : Tb) + kKT - 1) / kKT : (c + kKT - 1) / kKT + 1;
          int unit_max = tiles;
          if constexpr (kChain) {
            tiles = sq.w;
            if (!coop) {
              tiles = 0;
              for (int r = 0; r < nrb_b && !bad; ++r) tiles += chain_rb_tiles(c, Tb, g, r);
            }
            unit_max = bad ? 1 : chain_rb_tiles(c, Tb, g, nrb_b - 1);
          }
          if (!bad) {
            wl[k] = p.n_kv * (kChain ? 1 : nrb_b) * tiles;
            tmax = max(tmax, unit_max);
          }
          s_seq[bb] = make_int4(sq.x, bad ? 0 : Tb, c, tiles);
        }
        wsum += wl[k];
      }
      // warp-wide exclusive scan of the lanes' sums (lane order is sequence order)
      int incl = wsum;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += v;
      }
      const int W = __shfl_sync(0xffffffffu, incl, 31);
      const int tmax_all = __reduce_max_sync(0xffffffffu, tmax);
      int run = incl - wsum;
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const int bb = lane * kPer + k;
        if (bb < p.B) s_wpre[bb] = run;
        run += wl[k];
      }
      if (lane == 0) {
        const int m = max(2, (tmax_all + 13) / 14);
        const int N = W > 0 ? min((int)gridDim.x, max(1, W / m)) : 0;
        const bool mine = (int)blockIdx.x < N;
        s_sched[0] = mine ? (int)blockIdx.x * W / N : 0;
        s_sched[1] = mine ? ((int)blockIdx.x + 1) * W / N : 0;
        s_sched[2] = W;
        s_sched[3] = N;
        s_sched[4] = 0;
        s_sched[5] = 0;
        s_sched[6] = s_sched[1];
        s_wpre[p.B] = W;
      }
    }
    __syncthreads();
  }

  const int qhalf = lane >> 4, qc = lane & 15;
  int32_t* s_pages = reinterpret_cast<int32_t*>(smem + kOffPages);
  uint32_t tmem = 0;
  bool skip = false;          // uniform mode: the row block has no work
  // uniform mode: the (row block, chunk) of this CTA, and the row block's node
  // offset and rows for the merge
  const int split = kBal ? 0 : (int)(blockIdx.x % p.S);   // == cluster rank in the cluster mode
  int u_o = 0, u_R = 0;
  // uniform cooperative mode, thread 0: the row block's count as read at the
  // start (the target is the next multiple of kCountGen)
  unsigned long long u_target = 0;

  for (;;) {
    // ---------------- the next segment of this CTA's work ----------------
    constexpr int kPgPerThread = (kMaxCtaPages + kThreads - 1) / kThreads;
    int b, hk, rb, o, T, ctx, k_begin, k_end;
    bool with_tree, alone;
    size_t slot;
    int32_t pgr[kPgPerThread];
    int x_next = 0;
    int rot = 0;                // tiles run in the order rot, rot + 1, ..., n_tiles - 1, 0, ..., rot - 1
    // tiles this CTA processed before this segment (ring slots and phases count
    // over all segments), and the segments done; kept in shared memory so that
    // no register carries them across the softmax loop
    const int tb = kBal ? s_sched[4] : 0;
    const int nseg = kBal ? s_sched[5] : 0;
    if constexpr (kBal) {
      // The CTA walks its range from the end: its last segment (the head of a
      // row block) first.  Within a segment the tiles run rotated so that the
      // CTA reads tile x of a row block at about its local time x mod P (P =
      // the share): the CTAs holding other row blocks of the same KV head then
      // read the same K/V tiles at about the same time, and L2 serves the
      // repeats (each KV head's tiles are read by all its row blocks).
      const int x_begin = s_sched[0], y = s_sched[6], W = s_sched[2], N = s_sched[3];
      if (y <= x_begin) break;
      int lo = 0, hi = p.B;   // s_wpre[lo] <= y - 1 < s_wpre[hi]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (s_wpre[mid] <= y - 1) lo = mid; else hi = mid;
      }
      b = lo;
      const int4 sq = s_seq[b];
      o = sq.x;
      T = sq.y;
      ctx = sq.z;
      int tiles = sq.w;
      int U0;                                        // the unit's first tile in the work list
      if constexpr (kChain) {
        // sq.w = tiles of one KV head's row blocks; row block r has chain_rb_tiles
        const int local = y - 1 - s_wpre[b];
        hk = local / tiles;
        const int rem = local - hk * tiles;
        // the row block holding tile rem: every warp scans the row blocks' tile
        // counts 32 at a time (a warp prefix sum; all warps reach the same answer)
        const int nrb_b = (T * g + kRows - 1) / kRows;
        int r = nrb_b - 1, cum = 0, tu = 0;
        for (int r0 = 0, base = 0; r0 < nrb_b; r0 += 32) {
          const int rr = r0 + lane;
          const int t = rr < nrb_b ? chain_rb_tiles(ctx, T, g, rr) : 0;
          int incl = t;
#pragma unroll
          for (int dd = 1; dd < 32; dd <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, dd);
            if (lane >= dd) incl += v;
          }
          const int excl = base + incl - t;
          const unsigned hit = __ballot_sync(0xffffffffu, rr < nrb_b && rem >= excl && rem < excl + t);
          if (hit) {
            const int src = __ffs(hit) - 1;
            r = r0 + src;
            cum = __shfl_sync(0xffffffffu, excl, src);
            tu = __shfl_sync(0xffffffffu, t, src);
            break;
          }
          base += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (tu == 0) {   // not reached for a consistent work list
          cum = 0;
          for (int q = 0; q < r; ++q) cum += chain_rb_tiles(ctx, T, g, q);
          tu = chain_rb_tiles(ctx, T, g, r);
        }
        rb = r;
        U0 = s_wpre[b] + hk * tiles + cum;
        tiles = tu;
      } else {
        const int nrb_b = (T * g + kRows - 1) / kRows;
        const int u = (y - 1 - s_wpre[b]) / tiles;
        hk = u / nrb_b;
        rb = u - hk * nrb_b;
        U0 = s_wpre[b] + u * tiles;
      }
      const int seg0 = max(U0, x_begin);
      const int t0 = seg0 - U0;
      const int len = y - seg0;
      const int n_ctx_b = kIP ? tiles : tiles - 1;   // paged tiles of the unit
      k_begin = min(t0, n_ctx_b) * kKT;
      const int unit_span = kChain ? ctx + min(T, ((rb + 1) * kRows - 1) / g + 1) : (kIP ? ctx + T : ctx);
      k_end = t0 < n_ctx_b ? min(unit_span, min(t0 + len, n_ctx_b) * kKT) : k_begin;
      with_tree = !kIP && t0 + len == tiles;
      const int P = (W + N - 1) / N;
      int ph = (tb - t0) % P;
      ph += ph < 0 ? P : 0;
      rot = ph < len ? ph : 0;
      // the CTAs holding the unit's first and last tiles
      const int c0 = ((U0 + 1) * N - 1) / W;
      const int c1 = ((U0 + tiles) * N - 1) / W;
      alone = c0 == c1;
      // a piece starts the CTA's range (slot 2c) or ends it (slot 2c + 1)
      slot = 2 * (size_t)blockIdx.x + (seg0 > x_begin ? 1 : 0);
      if (!alone && threadIdx.x == 0 && s_npc < 2) {
        const int start0 = c0 * W / N;
        const int slot0 = 2 * c0 + (U0 > start0 ? 1 : 0);
        const unsigned long long c = ld_acquire64(
            reinterpret_cast<const unsigned long long*>(p.part + (size_t)slot0 * kAttnPartBytes + kAttnCntOff));
        s_pc[s_npc] = BalPiece{hk, rb, o, T * g, c1 - c0 + 1, (int)blockIdx.x - c0, slot0, 2 * (c0 + 1),
                               (c / kCountGen + 1) * kCountGen};
        s_npc = s_npc + 1;
      }
      x_next = seg0;
      const int pg_first = k_begin / EE_PAGE;
      const int npg = (k_end - k_begin + EE_PAGE - 1) / EE_PAGE;   // <= kMaxCtaPages: see the plan
#pragma unroll
      for (int k = 0; k < kPgPerThread; ++k) {
        const int i = threadIdx.x + k * kThreads;
        pgr[k] = i < npg ? ld_nc_pinned(p.block_table + (size_t)b * p.max_pages + pg_first + i) : -1;
      }
    } else {
      b = blockIdx.z;
      hk = blockIdx.y;
      rb = blockIdx.x / p.S;                     // the S chunks of a row block are consecutive
      // the row block's count, read now beside the node range (any time before
      // this CTA's own arrival will do: it is a multiple of kCountGen plus the
      // arrivals of this launch so far, never all of them)
      if (p.coop && p.S > 1 && threadIdx.x == 0) {
        const size_t cta0 = ((size_t)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + (size_t)rb * p.S;
        u_target = ld_relaxed64(
            reinterpret_cast<const unsigned long long*>(p.part + cta0 * kAttnPartBytes + kAttnCntOff));
      }
      // this chunk's page ids, issued now beside the sequence's node range and
      // context length so that the round trips overlap (validated below)
      const int pg_first = split * (p.chunk / EE_PAGE);
      const int npg_cap = max(0, min(p.chunk / EE_PAGE, p.max_pages - pg_first));
#pragma unroll
      for (int k = 0; k < kPgPerThread; ++k) {
        const int i = threadIdx.x + k * kThreads;
        pgr[k] = i < npg_cap ? ld_nc_pinned(p.block_table + (size_t)b * p.max_pages + pg_first + i) : -1;
      }
      o = p.node_off[b];
      T = p.node_off[b + 1] - o;
      ctx = p.ctx_len[b];
      const bool bad_tree = T < 1 || T > kMaxT || T > p.max_T || o < 0 || o + T > p.total_nodes;
      if (bad_tree && threadIdx.x == 0 && blockIdx.x == 0 && hk == 0) flag_error(p.err, EE_DEVERR_TREE);
      if (bad_tree || rb * kRows >= T * g) {     // uniform over the CTA (and the row block)
        skip = true;
        break;
      }
      if (ctx < 0 || ctx > p.max_ctx) {
        if (threadIdx.x == 0 && blockIdx.x == 0 && hk == 0) flag_error(p.err, EE_DEVERR_CTX);
        ctx = ctx < 0 ? 0 : p.max_ctx;
      }
      // everything above is uniform over the row block's CTAs; from here on every
      // CTA reaches the merge synchronisation
      // paged keys of the row block (chain: up to its last node's position)
      const int span = kChain ? ctx + min(T, ((rb + 1) * kRows - 1) / g + 1) : (kIP ? ctx + T : ctx);
      const int S = attn_splits_for(span, p.chunk);  // chunks this sequence uses, <= p.S
      const bool active = split < S;
      k_begin = split * p.chunk;
      k_end = active ? min(span, k_begin + p.chunk) : k_begin;
      with_tree = !kIP && active && split == S - 1;
      alone = p.S == 1;
      slot = ((size_t)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
      u_o = o;
      u_R = T * g;

    }
    const int R = T * g;
    const int n_ctx_tiles = k_end > k_begin ? (k_end - k_begin + kKT - 1) / kKT : 0;
    const int n_tiles = n_ctx_tiles + (with_tree ? 1 : 0);

    // softmax threads issue the coalesced loads of the block's Q rows now (a
    // half-warp reads one 256-byte row; rows past R read row R - 1 and are
    // zeroed later) so that they leave before the K/V stream starts; the values
    // are consumed after the barrier below
    bool pages_ok = true;
    uint4 qv[kRows / 16];
    if (warp >= kWarpSoft0) {
#pragma unroll
      for (int k = 0; k < kRows / 16; ++k) {
        const int rq = 2 * ((warp - kWarpSoft0) + 8 * k) + qhalf;   // 0..127
        const int rrq = min(rb * kRows + rq, R - 1);
        const int nq = rrq / g;
        qv[k] = __ldg(reinterpret_cast<const uint4*>(
                          p.q + ((size_t)(o + nq) * p.n_q + hk * g + (rrq - nq * g)) * kD) +
                      qc);
      }
    }
    {
      // pages that hold keys of this segment (k_end <= ctx <= max_pages * 16);
      // the previous segment's readers are past the barrier that ended it
      const int npg = (k_end - k_begin + EE_PAGE - 1) / EE_PAGE;
#pragma unroll
      for (int k = 0; k < kPgPerThread; ++k) {
        const int i = threadIdx.x + k * kThreads;
        if (i < npg) {
          const int pg = pgr[k];
          const bool ok = pg >= 0 && pg < p.num_pages;
          if (!ok) flag_error(p.err, EE_DEVERR_PAGE);
          s_pages[i] = ok ? pg : -1;
          pages_ok &= ok;
        }
      }
    }
    tc_fence_before();
    // every page of the segment valid: whole context tiles need no mask
    const bool seg_pages_ok = __syncthreads_and(pages_ok) != 0;
    tc_fence_after();
    tmem = s_tmem;
    // every thread has read the schedule position: advance it for the next segment
    if (kBal && threadIdx.x == 0) {
      s_sched[6] = x_next;
      s_sched[4] = tb + n_tiles;
      s_sched[5] = nseg + 1;
    }

    if (warp == kWarpK || warp == kWarpV) {
      // ---------------- TMA producers: warp 0 streams K, warp 2 streams V ----------------
      // lane 0 waits for the slot and posts the byte count; lane i < 8 then issues
      // the two boxes of the tile's 16-row block i.  Ring slots and phases count
      // the CTA's tiles over all its segments.
      const bool isK = warp == kWarpK;
      const int nst = isK ? kKST : kVST;
      const uint32_t full0 = isK ? k_full : v_full, empty0 = isK ? k_empty : v_empty;
      const uint32_t ring = isK ? sK : sV;
      const CUtensorMap* mc = isK ? &tmKc : &tmVc;
      const CUtensorMap* mt = isK ? &tmKt : &tmVt;
      int* issued = isK ? s_kissued : s_vissued;
      for (int t = 0; t < n_tiles; ++t) {
        const int tg = tb + t;
        const int st = tg % nst, use = tg / nst;
        bool go = true;
        if (lane == 0) go = mbar_wait(empty0 + 8 * st, (uint32_t)(use & 1) ^ 1u, &s_abort);
        if (!__shfl_sync(0xffffffffu, go, 0)) break;
        const uint32_t full = full0 + 8 * st;
        const uint32_t dst = ring + st * kKVBytes;
        if (lane == 0) mbar_expect_tx(full, 2 * kKVHalf);
        __syncwarp();
        const int i = t + rot < n_tiles ? t + rot : t + rot - n_tiles;   // the segment's tile
        if (i < n_ctx_tiles) {
          // every 16-row block is written: blocks without a loaded page are read at
          // row -16, wholly out of range, which the TMA unit fills with zeros (a
          // stale V row would turn 0 * P into NaN)
          if (lane < kKT / 16) {
            const int pos = k_begin + i * kKT + 16 * lane;
            const int pg = pos < k_end ? s_pages[i * (kKT / 16) + lane] : -1;
            const int row0 = pg >= 0 ? (pg * p.n_kv + hk) * EE_PAGE : -EE_PAGE;
            tma_load_2d(dst + lane * 2048, mc, full, 0, row0);
            tma_load_2d(dst + kKVHalf + lane * 2048, mc, full, 64, row0);
          }
        } else if (lane == 0) {
          tma_load_3d(dst, mt, full, 0, hk, o);
          tma_load_3d(dst + kKVHalf, mt, full, 64, hk, o);
        }
        __syncwarp();
        if (lane == 0) issued[st] = use;
      }
    } else if (warp == kWarpMma) {
      // ---------- MMA issuer: Q.K^T(0..kSB-1), then P.V(t), Q.K^T(t+kSB) ----------
      if (lane == 0) {
        tc_fence_after();
        const uint32_t id_qk = idesc_f16(kRows, kKT, 1, 1, 0);
        const uint32_t sQ = sbase + kOffQ;
        const uint32_t id_pv = idesc_f16(kRows, kD, 1, 1, 1);
        auto issue_qk = [&](int t) -> bool {
          const int tg = tb + t;
          if (!mbar_wait(k_full + 8 * (tg % kKST), (uint32_t)((tg / kKST) & 1), &s_abort)) return false;
          tc_fence_after();
          const uint32_t kb = sK + (tg % kKST) * kKVBytes;
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint32_t off = (kk & 3) * 32;
            tc_mma(tmem + (tg % kSB) * kKT, smem_desc_sw128(sQ + (kk >> 2) * kKVHalf + off),
                   smem_desc_sw128(kb + (kk >> 2) * kKVHalf + off), id_qk, kk > 0 ? 1u : 0u);
          }
          tc_commit(k_empty + 8 * (tg % kKST));
          tc_commit(s_full + 8 * (tg % kSB));
          return true;
        };
        bool ok = mbar_wait(q_ready, (uint32_t)(nseg & 1), &s_abort);
        for (int t = 0; t < kSB && t < n_tiles && ok; ++t) ok = issue_qk(t);
        for (int t = 0; t < n_tiles && ok; ++t) {
          const int tg = tb + t;
          if (!mbar_wait(p_full + 8 * (tg % kSB), (uint32_t)((tg / kSB) & 1), &s_abort) ||
              !mbar_wait(v_full + 8 * (tg % kVST), (uint32_t)((tg / kVST) & 1), &s_abort))
            break;
          tc_fence_after();
          const uint32_t pa = tmem + (tg % kSB) * kKT;       // bf16 P head: cols 0..63, tail: 64..127
          const uint32_t vb = sV + (tg % kVST) * kKVBytes;
#pragma unroll
          for (int part = 0; part < 2; ++part)
#pragma unroll
            for (int j = 0; j < kKT / 16; ++j)
              tc_mma_ts(tmem + kColO, pa + 64 * part + 8 * j,
                        smem_desc_sw128_mn(vb + j * 2048, kKVHalf, 1024), id_pv,
                        (t > 0 || part > 0 || j > 0) ? 1u : 0u);
          tc_commit(v_empty + 8 * (tg % kVST));
          tc_commit(o_done + 8 * (tg & 1));
          if (t + kSB < n_tiles) ok = issue_qk(t + kSB);
        }
        // one phase per segment: every product of the segment is complete
        if (n_tiles > 0) tc_commit(o_final);
      }
    } else if (warp >= kWarpSoft0) {
      // ---------------- softmax: one query row and half of every tile per thread ----------------
      // Warps w and w + 4 share TMEM lane quarter w & 3 (32 query rows); half hf
      // of the pair takes keys [64 hf, 64 hf + 64) of every tile and O columns
      // [64 hf, 64 hf + 64).  The pair agrees on each tile's row maximum through
      // shared memory at a 64-thread named barrier, so both halves take the same
      // rescale decisions; each keeps the sum over its own keys, and the two sums
      // are added (half 0 first) at the end.  Two warps per sub-partition hide
      // each other's latencies.  Every exit from the tile loop happens right
      // after the pair barrier and on a decision both warps share.
      const int qd = warp & 3;
      const int hf = (warp - kWarpSoft0) >> 2;
      const uint32_t pair_bar = 2 + qd;
      const int r = qd * 32 + lane;                     // == TMEM lane of this quarter
      const int rr = rb * kRows + r;
      const bool vrow = rr < R;
      const int node = vrow ? rr / g : 0;
      // this half's tree keys (separate tree tile), or the row's whole ancestor
      // mask (in place: tree keys at any offset from a half's first key)
      const uint64_t ancw = (!kChain && vrow) ? p.anc[2 * (size_t)(o + node) + (kIP ? 0 : hf)] : 0ull;
      const uint64_t anc_hi = (kKV == kKVInPlace && vrow) ? p.anc[2 * (size_t)(o + node) + 1] : 0ull;
      const uint32_t tl = tmem + ((uint32_t)(qd * 32) << 16);
      // the block's Q rows into shared memory as the A operand of Q.K^T: 128 rows
      // x 128 bf16 in two 64-column slabs, 128-byte swizzled K-major (the layout
      // TMA gives the K tiles): 16-byte chunk j of row r at slab (j / 8),
      // (r / 8) * 1024 + (r % 8) * 128 + ((j % 8) ^ (r % 8)) * 16; rows past R are
      // zero.  The rows were loaded (coalesced) before the set-up barrier; the
      // previous segment's Q.K^T products completed before its last P.V did.
      {
        uint8_t* qs = smem + kOffQ;
#pragma unroll
        for (int k = 0; k < kRows / 16; ++k) {
          const int rq = 2 * ((warp - kWarpSoft0) + 8 * k) + qhalf;
          const int j = qc & 7;
          *reinterpret_cast<uint4*>(qs + (qc >> 3) * kKVHalf + (rq >> 3) * 1024 + (rq & 7) * 128 +
                                    ((j ^ (rq & 7)) << 4)) =
              rb * kRows + rq < R ? qv[k] : make_uint4(0u, 0u, 0u, 0u);
        }
        fence_async_smem();   // generic-proxy writes, read by the tensor core
        mbar_arrive(q_ready);
      }
      // m_used is kept in raw score units (scale > 0, so the max commutes with it)
      float m_used = -INFINITY, l = 0.f;
      const float sl2 = p.scale_log2;
      const float kFail = __int_as_float(0x7fffffff);   // NaN: "this half's wait failed"
      bool ok = true;
      // the loop runs over the CTA's tile count tg (ring phases), with the
      // segment's first tile at tg = tb; step tg processes the segment's tile
      // tg + d (mod n_tiles)
      const int tg_end = tb + n_tiles;
      const int d = rot - tb;
      for (int tg = tb; tg < tg_end; ++tg) {
        const int sb = tg % kSB;    // S buffer of this tile
        const int xb = tg & 1;      // pair-exchange slot
        // wait outcomes are warp-uniform: the TMEM accesses that follow are
        // warp-collective (.sync.aligned)
        const bool got =
            __all_sync(0xffffffffu, mbar_wait(s_full + 8 * sb, (uint32_t)((tg / kSB) & 1), &s_abort));
        uint32_t sr[64];
        float tmax = -INFINITY;
        if (got) {
          tc_fence_after();
          tc_ld32(tl + sb * kKT + 64 * hf, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
          tc_ld32(tl + sb * kKT + 64 * hf + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
          // visibility of this half's 64 keys as one 64-bit word
          uint64_t kw;
          const int i = tg + d < n_tiles ? tg + d : tg + d - n_tiles;
          if (seg_pages_ok && k_begin + (i + 1) * kKT <= (kIP ? min(k_end, ctx) : k_end)) {
            kw = ~0ull;   // a whole tile of context keys in valid pages: every row sees all of it
          } else if (i < n_ctx_tiles) {
            const unsigned m = tile_mask(s_pages, i, k_begin, k_end);
            const int nv = min(max(k_end - (k_begin + i * kKT) - 64 * hf, 0), 64);
            uint64_t pgw = 0ull;
#pragma unroll
            for (int pb = 0; pb < 4; ++pb) pgw |= ((m >> (4 * hf + pb)) & 1u) ? (0xFFFFull << (16 * pb)) : 0ull;
            kw = pgw & (nv >= 64 ? ~0ull : ((1ull << nv) - 1ull));
            if constexpr (kChain) {
              // causal: node sees positions up to ctx + node
              const int p0 = k_begin + i * kKT + 64 * hf;
              const int nvis = min(max(ctx + node + 1 - p0, 0), 64);
              kw &= nvis >= 64 ? ~0ull : ((1ull << nvis) - 1ull);
            } else if constexpr (kIP) {
              // keys below ctx are context; key p >= ctx is tree node p - ctx
              const int p0 = k_begin + i * kKT + 64 * hf;
              const int nc = min(max(ctx - p0, 0), 64);
              const int sh = p0 - ctx;    // ancestor bit of this half's first key
              uint64_t tm;
              if (sh >= 0)
                tm = sh >= 128 ? 0ull
                     : sh >= 64 ? (anc_hi >> (sh - 64))
                     : sh == 0  ? ancw
                                : ((ancw >> sh) | (anc_hi << (64 - sh)));
              else
                tm = sh <= -64 ? 0ull : (ancw << (-sh));
              kw &= (nc >= 64 ? ~0ull : ((1ull << nc) - 1ull)) | tm;
            }
          } else {
            const int th = min(max(T - 64 * hf, 0), 64);
            kw = ancw & (th >= 64 ? ~0ull : ((1ull << th) - 1ull));
          }
          if (!vrow) kw = 0ull;
          if (!__all_sync(0xffffffffu, kw == ~0ull)) {
#pragma unroll
            for (int c = 0; c < 64; ++c)
              if (!((kw >> c) & 1ull)) sr[c] = __float_as_uint(-INFINITY);
          }
          // 8 independent chains of three-input maxima over the 64 values
          float mx[8];
#pragma unroll
          for (int c = 0; c < 8; ++c) mx[c] = __uint_as_float(sr[c]);
#pragma unroll
          for (int c = 8; c < 56; c += 16)         // values 8 .. 55, two per instruction
#pragma unroll
            for (int k = 0; k < 8; ++k)
              mx[k] = fmax3(mx[k], __uint_as_float(sr[c + k]), __uint_as_float(sr[c + 8 + k]));
#pragma unroll
          for (int k = 0; k < 8; ++k) mx[k] = fmaxf(mx[k], __uint_as_float(sr[56 + k]));   // values 56 .. 63
          tmax = fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
        }
        // the pair swaps its halves' maxima; both S halves are in registers before
        // either warp overwrites S with P
        s_xmax[xb][hf][r] = got ? tmax : kFail;
        tc_fence_before();
        asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
        tc_fence_after();
        const float other = s_xmax[xb][hf ^ 1][r];
        if (!__all_sync(0xffffffffu, got && other == other)) {
          ok = false;
          break;
        }
        tmax = fmaxf(tmax, other);
        const float m_new = fmaxf(m_used, tmax);
        const bool need = (m_new - m_used) * sl2 > kRescaleLog2;   // true when m_used = -inf < m_new
        if (tg > 0 && __any_sync(0xffffffffu, need)) {
          // O must hold P.V(tg-1) before this half's columns are rescaled; a failed
          // wait sets the abort flag, and the pair stops at the next barrier.  At a
          // segment's first tile that product belongs to the previous segment (its
          // completion was already waited for) and the rescale is harmless: the
          // segment's first P.V overwrites O.
          if (__all_sync(0xffffffffu,
                         mbar_wait(o_done + 8 * ((tg - 1) & 1), (uint32_t)(((tg - 1) >> 1) & 1), &s_abort))) {
            tc_fence_after();
            const float f = need ? ex2((m_used - m_new) * sl2) : 1.f;
#pragma unroll 1
            for (int c4 = 0; c4 < 4; ++c4) {
              uint32_t ov[16];
              tc_ld16(tl + kColO + 64 * hf + 16 * c4, ov);
#pragma unroll
              for (int e = 0; e < 16; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * f);
              tc_st16_nowait(tl + kColO + 64 * hf + 16 * c4, ov);
            }
            tc_wait_st();
          } else {
            ok = false;
          }
        }
        if (need) {
          l *= ex2((m_used - m_new) * sl2);
          m_used = m_new;
        }
        const float nms = m_used == -INFINITY ? 0.f : -m_used * sl2;
        // p = 2^(s*scale_log2 - m); P = head + tail, both bf16: this
        // half's head pairs go to columns 32 hf.. of the S buffer, its tail pairs
        // to 64 + 32 hf..
        // (pairs of columns run on packed fp32x2 arithmetic: the scale-and-shift,
        // the running sums and the tail subtraction take one instruction per pair)
        const uint64_t sl2x2 = f2_pack(__float_as_uint(sl2), __float_as_uint(sl2));
        const uint64_t nmsx2 = f2_pack(__float_as_uint(nms), __float_as_uint(nms));
        uint64_t ls2[4];
        // two halves of 16 column pairs: each half's head and tail words go
        // out before the next half is computed (fewer live registers)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t hw[16], tw[16];
#pragma unroll
          for (int e2 = 0; e2 < 16; ++e2) {
            const int e = 16 * hh + e2;
            uint32_t y0, y1;
            f2_unpack(f2_fma(f2_pack(sr[2 * e], sr[2 * e + 1]), sl2x2, nmsx2), y0, y1);
            const uint32_t p0 = __float_as_uint(ex2(__uint_as_float(y0)));
            const uint32_t p1 = __float_as_uint(ex2(__uint_as_float(y1)));
            const uint64_t pp = f2_pack(p0, p1);
            ls2[e & 3] = e < 4 ? pp : f2_add(ls2[e & 3], pp);
            // head = p rounded to bf16; tail = the remainder p - head (exact
            // in fp32) rounded to bf16
            const uint32_t hb = bf16x2_rn(__uint_as_float(p1), __uint_as_float(p0));
            uint32_t t0, t1;
            f2_unpack(f2_sub(pp, f2_pack(hb << 16, hb & 0xFFFF0000u)), t0, t1);
            hw[e2] = hb;
            tw[e2] = bf16x2_rn(__uint_as_float(t1), __uint_as_float(t0));
          }
          tc_st16_nowait(tl + sb * kKT + 32 * hf + 16 * hh, hw);
          tc_st16_nowait(tl + sb * kKT + 64 + 32 * hf + 16 * hh, tw);
        }
        tc_wait_st();
        {
          uint32_t a0, a1, b0, b1, c0, c1, d0, d1;
          f2_unpack(ls2[0], a0, a1);
          f2_unpack(ls2[1], b0, b1);
          f2_unpack(ls2[2], c0, c1);
          f2_unpack(ls2[3], d0, d1);
          l += ((__uint_as_float(a0) + __uint_as_float(a1)) + (__uint_as_float(b0) + __uint_as_float(b1))) +
               ((__uint_as_float(c0) + __uint_as_float(c1)) + (__uint_as_float(d0) + __uint_as_float(d1)));
        }
        tc_fence_before();
        mbar_arrive(p_full + 8 * sb);
      }
      // wait for the last P.V; the pair adds its two sums, then each half writes
      // its 64 columns out: O / l itself when the segment is a whole row block,
      // else the partial (O, m, l) to the segment's slot.  The wait is on a
      // barrier of its own: here the tensor pipe may still owe P.V(n-3) and
      // P.V(n-1), two phases of the same o_done barrier, which a parity wait
      // cannot tell apart (inside the loop at most one phase is pending, since
      // S(t) completes after P.V(t-3))
      const bool fin = ok && n_tiles > 0 && mbar_wait(o_final, (uint32_t)(nseg & 1), &s_abort);
      const bool have = __all_sync(0xffffffffu, fin);
      s_xl[hf][r] = have ? l : kFail;
      asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
      const float l_sum = s_xl[0][r] + s_xl[1][r];     // NaN when either half failed
      const bool both = have && l_sum == l_sum;
      const float row_m = (both && vrow && m_used != -INFINITY) ? m_used * sl2 : -INFINITY;
      const float row_l = (both && vrow && m_used != -INFINITY) ? l_sum : 0.f;
      float4* dst;
      size_t dstride;                                   // float4 between column chunks
      float inv = 1.f;
      if (alone) {
        const size_t orow = (size_t)(o + node) * p.n_q + hk * g + (rr - node * g);
        dst = reinterpret_cast<float4*>(p.out + orow * kD);
        dstride = 1;
        inv = row_l > 0.f ? 1.f / row_l : 0.f;
      } else {
        dst = reinterpret_cast<float4*>(p.part + slot * kAttnPartBytes) + r;
        dstride = kRows;
      }
      const bool store = alone ? vrow : row_l > 0.f;
      // the TMEM read is warp-collective: the whole warp reads when any lane stores
      if (__any_sync(0xffffffffu, store)) {
        tc_fence_after();
#pragma unroll 1
        for (int c4 = 0; c4 < 2; ++c4) {
          uint32_t ov[32];
          tc_ld32(tl + kColO + 64 * hf + 32 * c4, ov);
          if (store) {
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float4 v = make_float4(__uint_as_float(ov[4 * e]) * inv, __uint_as_float(ov[4 * e + 1]) * inv,
                                           __uint_as_float(ov[4 * e + 2]) * inv,
                                           __uint_as_float(ov[4 * e + 3]) * inv);
              __stcg(dst + (size_t)(16 * hf + 8 * c4 + e) * dstride, v);
            }
          }
        }
      }
      if (!alone) {
        if (hf == 0)
          __stcg(reinterpret_cast<float2*>(p.part + slot * kAttnPartBytes + kAttnMlOff) + r,
                 make_float2(row_m, row_l));
      }
    }
    if constexpr (!kBal) break;
    // end of the segment: every role is done with its pages, Q, S buffers and O
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (s_abort) break;
  }

  // ---- CTA teardown: drain on abort, free TMEM --------------------------------
  tc_fence_before();
  __syncthreads();
  pdl_allow_next();   // this grid's pipeline is done: the next kernel may take SMs as they free
  const bool aborted = s_abort != 0;
  if (aborted && threadIdx.x == 0) {
    flag_error(p.err, EE_DEVERR_TIMEOUT);
    // TMA copies still in flight land before the rings are reused
    for (int st = 0; st < kKST; ++st)
      if (s_kissued[st] >= 0) mbar_wait_plain(k_full + 8 * st, (uint32_t)(s_kissued[st] & 1));
    for (int st = 0; st < kVST; ++st)
      if (s_vissued[st] >= 0) mbar_wait_plain(v_full + 8 * st, (uint32_t)(s_vissued[st] & 1));
  }
  if (warp == kWarpMma) {
    if (aborted && lane == 0) {
      tc_commit(drain);
      mbar_wait_plain(drain, 0);
    }
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(s_tmem), "r"(kTmemCols)
                 : "memory");
  }

  __shared__ int s_ready[2];
  if constexpr (kBal) {
    // ---- merge of split row blocks (balanced mode) ----------------------------------
    // every CTA counts all its pieces before it waits for any (the launch is
    // cooperative, so all CTAs are resident and every count arrives)
    const int npieces = s_npc;     // written by thread 0 before the teardown barrier
    if (npieces == 0) return;
    unsigned long long* cnt[2];
#pragma unroll
    for (int i = 0; i < 2; ++i)
      cnt[i] = reinterpret_cast<unsigned long long*>(
          p.part + (size_t)s_pc[i < npieces ? i : 0].slot0 * kAttnPartBytes + kAttnCntOff);
    if (threadIdx.x == 0) {
      // the partials of this CTA's pieces (every thread's stores precede the
      // teardown barrier) are released with the count
      for (int i = 0; i < npieces; ++i) red_add_release64(cnt[i], kCountGen / (unsigned)s_pc[i].K);
      for (int i = 0; i < npieces; ++i) {
        const bool ready = wait_count64_geq(cnt[i], s_pc[i].target);
        if (!ready) flag_error(p.err, EE_DEVERR_TIMEOUT);
        s_ready[i] = ready;
      }
    }
    __syncthreads();
    for (int i = 0; i < npieces; ++i) {
      const BalPiece q = s_pc[i];
      const int rpc = (kRows + q.K - 1) / q.K;
      const int r0 = q.k * rpc;
      const int nown = s_ready[i] ? max(0, min(rpc, min(kRows, q.R - q.rb * kRows) - r0)) : 0;
      if (nown > 0) {
        const int row0 = q.rb * kRows + r0;
        switch (q.K) {
#define EE_MERGE_CASE(n)                                                                   \
  case n:                                                                                  \
    merge_rows<n>(p, (size_t)q.slot0, (size_t)q.slot1, 2, row0, r0, nown, q.o, q.hk); \
    break;
          EE_MERGE_CASE(2) EE_MERGE_CASE(3) EE_MERGE_CASE(4) EE_MERGE_CASE(5) EE_MERGE_CASE(6)
          EE_MERGE_CASE(7) EE_MERGE_CASE(8) EE_MERGE_CASE(9) EE_MERGE_CASE(10) EE_MERGE_CASE(11)
          EE_MERGE_CASE(12) EE_MERGE_CASE(13) EE_MERGE_CASE(14) EE_MERGE_CASE(15) EE_MERGE_CASE(16)
#undef EE_MERGE_CASE
          default:
            break;
        }
      }
    }
    return;
  } else {
    if (skip || p.S == 1) return;

    // ---- merge (uniform modes) -------------------------------------------------------
    // once every slot of the row block is complete and visible, chunk `split`
    // merges rows [r0, r0 + nown) of the row block
    const int R = u_R, o = u_o;
    const int rb = blockIdx.x / p.S;
    const size_t cta0 = ((size_t)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + (size_t)rb * p.S;
    unsigned long long* cnt = reinterpret_cast<unsigned long long*>(p.part + cta0 * kAttnPartBytes + kAttnCntOff);
    if (p.coop) {
      if (threadIdx.x == 0) {
        // this CTA's partial (every thread's stores precede the teardown barrier)
        red_add_release64(cnt, kCountGen / (unsigned)p.S);
        const bool ready = wait_count64_geq(cnt, (u_target / kCountGen + 1) * kCountGen);
        if (!ready) flag_error(p.err, EE_DEVERR_TIMEOUT);
        s_ready[0] = ready;
      }
      __syncthreads();
    } else {
      cluster_sync();
      if (threadIdx.x == 0) s_ready[0] = 1;
      __syncthreads();
    }
    const int rpc = (kRows + p.S - 1) / p.S;
    const int r0 = split * rpc;
    const int nown = s_ready[0] ? max(0, min(rpc, min(kRows, R - rb * kRows) - r0)) : 0;
    if (nown > 0) {
      const int row0 = rb * kRows + r0;
      switch (p.S) {
#define EE_MERGE_CASE(n)                                                                  \
  case n:                                                                                 \
    merge_rows<n>(p, cta0, cta0 + 1, 1, row0, r0, nown, o, (int)blockIdx.y); \
    break;
        EE_MERGE_CASE(2) EE_MERGE_CASE(3) EE_MERGE_CASE(4) EE_MERGE_CASE(5) EE_MERGE_CASE(6)
        EE_MERGE_CASE(7) EE_MERGE_CASE(8) EE_MERGE_CASE(9) EE_MERGE_CASE(10) EE_MERGE_CASE(11)
        EE_MERGE_CASE(12) EE_MERGE_CASE(13) EE_MERGE_CASE(14) EE_MERGE_CASE(15) EE_MERGE_CASE(16)
#undef EE_MERGE_CASE
        default:
          break;
      }
    }
  }
}

// Clusters of `S` CTAs that fit on device `dev` at once (asked once per device
// and size; `dev` is the current device).
int active_clusters(int dev, int S) {
  static std::mutex mu;
  static int cache[kMaxDevices][kMaxCluster + 1] = {};
  std::lock_guard<std::mutex> lock(mu);
  int* cached = &cache[dev][S];
  if (!*cached) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S * 64, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kSmemBytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel<false, kKVTree>, &cfg) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = std::max(1, kNumSMs / S);
    }
    *cached = n;
  }
  return *cached;
}

// CTAs of one instantiation device `dev` (the current device) holds at once
// (asked once per device; -1 if unknown).
template <bool kBal>
int resident_ctas(int dev) {
  static std::mutex mu;
  static int caps[kMaxDevices] = {};
  std::lock_guard<std::mutex> lock(mu);
  int& cap = caps[dev];
  if (!cap) {
    int sms = 0, per = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, attn_tc_kernel<kBal, kKVTree>, kThreads, kSmemBytes) !=
            cudaSuccess ||
        per < 1) {
      cudaGetLastError();
      cap = -1;
    } else {
      cap = sms * per;
    }
  }
  return cap;
}

// Every instantiation takes the full dynamic shared memory (set once per device;
// `dev` is the current device).
cudaError_t set_attrs(int dev) {
  static std::mutex mu;
  static bool done_dev[kMaxDevices] = {};
  std::lock_guard<std::mutex> lock(mu);
  bool& done = done_dev[dev];
  if (done) return cudaSuccess;
  cudaError_t e = cudaSuccess;
  const void* fns[6] = {(const void*)attn_tc_kernel<false, kKVTree>, (const void*)attn_tc_kernel<true, kKVTree>,
                        (const void*)attn_tc_kernel<false, kKVInPlace>, (const void*)attn_tc_kernel<true, kKVInPlace>,
                        (const void*)attn_tc_kernel<false, kKVChain>, (const void*)attn_tc_kernel<true, kKVChain>};
  for (const void* f : fns)
    if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  done = e == cudaSuccess;
  return e;
}

// Chunk length for s chunks of `span` paged keys (with tree_tile, the last one
// also carries the 128-key tree tile), the chunks actually used and the
// 128-key tiles of the busiest CTA.
void chunk_for(int span, bool tree_tile, int s, int* chunk, int* used, int* tiles) {
  int c = (span + (tree_tile ? kKT : 0) + s - 1) / s;
  c = (c + EE_PAGE - 1) / EE_PAGE * EE_PAGE;
  c = std::min(c, kMaxCtaPages * EE_PAGE);          // a CTA stages at most kMaxCtaPages page ids
  *chunk = c;
  *used = attn_splits_for(span, c);
  const int last = span - (*used - 1) * c;
  *tiles = std::max((c + kKT - 1) / kKT, (last + kKT - 1) / kKT + (tree_tile ? 1 : 0));
}

struct Split {
  int S = 1, chunk = EE_PAGE;
  bool coop = false;
  bool bal = false;            // balanced work list (cooperative, one CTA per SM)
  int ctas = 0;                // balanced: grid size; CTAs sharing the work (at most); tiles per CTA
  int bal_ctas = 0, bal_tiles = 0;
};

// Launch plan.  Cost, in half-tiles, = 2 x waves x (tiles of the busiest CTA
// + a fixed per-CTA cost of about 3):
//   cluster mode: S <= 8, waves from the clusters the GPU holds at once (one
//   slot fewer per wave once a second wave is needed);
//   cooperative mode: one wave by construction, S up to 16 with n_rb x S
//   CTAs no more than the GPU holds.  Ties go to the cooperative mode;
//   balanced mode: every resident CTA takes an equal share of all units'
//   tiles (w_max at most, t_max per unit at most) and may cross one unit
//   boundary (about 1.5 tiles more); it needs 2 partial slots per CTA, a
//   share of at most 256 context tiles (the staged page ids) and B <= 512.
Split choose_split(int dev, int span, bool tree_tile, int n_rb, long w_max, int t_max, int B, size_t part_slots) {
  Split best;
  if (span <= 0) return best;                      // the tree tile alone: one chunk
  const int min_splits = (span + kMaxCtaPages * EE_PAGE - 1) / (kMaxCtaPages * EE_PAGE);
  long best_cost = -1;
  for (int s = std::max(1, min_splits); s <= kMaxCluster; ++s) {
    int chunk, used, tiles;
    chunk_for(span, tree_tile, s, &chunk, &used, &tiles);
    // from the second wave on, clusters start as earlier ones finish, and free
    // SMs scattered over the GPCs can leave a slot unusable: plan such launches
    // with one cluster slot fewer
    if (used > 1 && (size_t)n_rb * used > part_slots) continue;   // one partial slot per CTA
    const long act = active_clusters(dev, used);
    long waves = (n_rb + act - 1) / act;
    if (waves >= 2 && act > 1) waves = (n_rb + act - 2) / (act - 1);
    const long cost = 2 * waves * (tiles + 3);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best.S = used;
      best.chunk = chunk;
    }
  }
  const int cap = resident_ctas<false>(dev);
  if (cap > 0) {
    for (int s = std::max(2, min_splits); s <= kMaxSplits && (long)s * n_rb <= cap; ++s) {
      int chunk, used, tiles;
      chunk_for(span, tree_tile, s, &chunk, &used, &tiles);
      if (used < 2 || (size_t)n_rb * used > part_slots) continue;
      const long cost = 2 * (tiles + 3);
      if (cost <= best_cost) {
        best_cost = cost;
        best.S = used;
        best.chunk = chunk;
        best.coop = true;
      }
    }
  }
  const int capb = resident_ctas<true>(dev);
  if (capb > 0 && B <= kMaxBalSeqs && w_max <= (long)(kMaxCtaPages / (kKT / EE_PAGE)) * capb &&
      part_slots >= 2 * (size_t)capb) {
    const long m = std::max(2, (t_max + 13) / 14);
    const long n_eff = std::min<long>(capb, std::max<long>(1, w_max / m));
    const long share = (w_max + n_eff - 1) / n_eff;
    const long cost = 2 * share + 9;
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best.bal = true;
      best.coop = true;
      best.ctas = capb;
      best.bal_ctas = (int)n_eff;
      best.bal_tiles = (int)share;
    }
  }
  if (best_cost < 0) best.S = 0;   // no plan fits the workspace's partial slots
  return best;
}

// The plan for these sizes: span = paged keys of the longest row block
// (max_ctx, or max_ctx + max_T in place), row blocks, work-list bound.
Split plan_for(int dev, int B, int max_T, int n_q, int n_kv, int max_ctx, int kv, size_t slots) {
  const int g = n_q / n_kv;
  const int nrb = (max_T * g + kRows - 1) / kRows;
  const int span = kv != kKVTree ? max_ctx + max_T : max_ctx;
  const int t_max = kv != kKVTree ? (span + kKT - 1) / kKT : (max_ctx + kKT - 1) / kKT + 1;
  long per_seq = (long)n_kv * nrb * t_max;
  if (kv == kKVChain) {
    per_seq = 0;
    for (int r = 0; r < nrb; ++r) per_seq += chain_rb_tiles(max_ctx, max_T, g, r);
    per_seq *= n_kv;
  }
  return choose_split(dev, span, kv == kKVTree, nrb * n_kv * B, (long)B * per_seq, t_max, B, slots);
}

// Shared by ee_tree_verify_attn (tree K/V from k_tree / v_tree) and
// ee_tree_verify_attn_inplace (tree K/V at cache positions ctx .. ctx + T - 1).
ee_status verify_attn(const ee_bf16* q, const ee_bf16* k_tree, const ee_bf16* v_tree, const ee_bf16* k_cache,
                      const ee_bf16* v_cache, int32_t num_pages, const int32_t* block_table, int32_t max_pages,
                      const int32_t* ctx_len, int32_t max_ctx, const int32_t* node_off, const uint64_t* anc,
                      int32_t B, int32_t total_nodes, int32_t max_T, int32_t n_q, int32_t n_kv, int32_t head_dim,
                      float scale, float* out, void* ws, size_t ws_bytes, ee_stream_t stream, int kv) {
  const bool inplace = kv != kKVTree;
  if (B < 0 || total_nodes < 0 || n_q < 1 || n_kv < 1 || num_pages < 1 || max_pages < 1 ||
      max_ctx < 0 || max_T < 1)
    return EE_ERR_INVALID_ARG;
  if (head_dim != EE_HEAD_DIM || n_q % n_kv != 0 || max_T > (kv == kKVChain ? EE_MAX_CHAIN : EE_MAX_TREE))
    return EE_ERR_UNSUPPORTED;
  // every key position must have a block-table entry: the context, and in
  // place the tree's positions after it
  const int64_t span = (int64_t)max_ctx + (inplace ? max_T : 0);
  if (span > (int64_t)max_pages * EE_PAGE) return EE_ERR_INVALID_ARG;
  if (!(scale > 0.f) || !std::isfinite(scale)) return EE_ERR_INVALID_ARG;
  if (B == 0 || total_nodes == 0) return EE_OK;
  if (!q || (!inplace && (!k_tree || !v_tree)) || !k_cache || !v_cache || !block_table || !ctx_len ||
      !node_off || (kv != kKVChain && !anc) || !out || !ws)
    return EE_ERR_INVALID_ARG;
  if (!aligned(q, 16) || (!inplace && (!aligned(k_tree, 16) || !aligned(v_tree, 16))) ||
      !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) || !aligned(anc, 8) ||
      !aligned(ws, 256))
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < kWorkspaceBytes) return EE_ERR_WORKSPACE;
  if ((int64_t)num_pages * n_kv * EE_PAGE >= ((int64_t)1 << 31)) return EE_ERR_UNSUPPORTED;
  // a CTA stages at most kMaxCtaPages page ids, and a cluster holds at most 8 chunks
  if (span > (int64_t)kMaxCluster * kMaxCtaPages * EE_PAGE) return EE_ERR_UNSUPPORTED;

  int dev = 0;
  {
    const ee_status ds = current_device(&dev);
    if (ds != EE_OK) return ds;
  }
  EE_CUDA_OK(set_attrs(dev));
  // tensor maps: cache [pages * n_kv * 16 rows][128], tree [total][n_kv][128]
  // (in place the tree maps are not read: the cache maps stand in)
  CUtensorMap tmKc, tmVc, tmKt, tmVt;
  {
    const uint64_t dims[2] = {(uint64_t)head_dim, (uint64_t)num_pages * n_kv * EE_PAGE};
    const uint64_t strides[1] = {(uint64_t)head_dim * 2};
    const uint32_t box[2] = {64, EE_PAGE};
    if (!encode_bf16_tmap(&tmKc, k_cache, 2, dims, strides, box)) return EE_ERR_CUDA;
    if (!encode_bf16_tmap(&tmVc, v_cache, 2, dims, strides, box)) return EE_ERR_CUDA;
  }
  if (inplace) {
    tmKt = tmKc;
    tmVt = tmVc;
  } else {
    const uint64_t dims[3] = {(uint64_t)head_dim, (uint64_t)n_kv, (uint64_t)total_nodes};
    const uint64_t strides[2] = {(uint64_t)head_dim * 2, (uint64_t)n_kv * head_dim * 2};
    const uint32_t box[3] = {64, 1, (uint32_t)kKT};
    if (!encode_bf16_tmap(&tmKt, k_tree, 3, dims, strides, box)) return EE_ERR_CUDA;
    if (!encode_bf16_tmap(&tmVt, v_tree, 3, dims, strides, box)) return EE_ERR_CUDA;
  }
  const int g = n_q / n_kv;
  const int nrb = (max_T * g + kRows - 1) / kRows;
  const size_t slots = ws_bytes > kAttnPartOff ? (ws_bytes - kAttnPartOff) / kAttnPartBytes : 0;
  const Split sp = plan_for(dev, B, max_T, n_q, n_kv, max_ctx, kv, slots);
  if (sp.S == 0) return EE_ERR_WORKSPACE;
  const int S = sp.bal ? 1 : sp.S, chunk = sp.chunk;
  // a split launch writes one partial slot per CTA after the zeroed part
  if (!sp.bal && S > 1 && ws_bytes < kAttnPartOff + (size_t)nrb * S * n_kv * B * kAttnPartBytes)
    return EE_ERR_WORKSPACE;

  AttnParams p;
  p.q = reinterpret_cast<const __nv_bfloat16*>(q);
  p.block_table = block_table;
  p.ctx_len = ctx_len;
  p.node_off = node_off;
  p.anc = anc;
  p.out = out;
  p.part = static_cast<uint8_t*>(ws) + kAttnPartOff;
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
  p.S = S;
  p.coop = (S > 1 && sp.coop) || sp.bal ? 1 : 0;
  p.B = B;
  p.scale_log2 = scale * 1.4426950408889634f;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = sp.bal ? dim3(sp.ctas, 1, 1) : dim3(nrb * S, n_kv, B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (p.coop) {
    attr[1].id = cudaLaunchAttributeCooperative;
    attr[1].val.cooperative = 1;
    cfg.numAttrs = 2;
  } else if (S > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = S;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
  }
  decltype(&attn_tc_kernel<false, kKVTree>) fn;
  switch (kv * 2 + (sp.bal ? 1 : 0)) {
    case 0: fn = attn_tc_kernel<false, kKVTree>; break;
    case 1: fn = attn_tc_kernel<true, kKVTree>; break;
    case 2: fn = attn_tc_kernel<false, kKVInPlace>; break;
    case 3: fn = attn_tc_kernel<true, kKVInPlace>; break;
    case 4: fn = attn_tc_kernel<false, kKVChain>; break;
    default: fn = attn_tc_kernel<true, kKVChain>; break;
  }
  EE_CUDA_OK(cudaLaunchKernelEx(&cfg, fn, tmKc, tmVc, tmKt, tmVt, p));
  return EE_OK;
}

}  // namespace

extern "C" ee_status ee_attn_plan(int32_t B, int32_t max_T, int32_t n_q, int32_t n_kv,
                                  int32_t max_ctx, int32_t inplace, int32_t* splits, int32_t* chunk,
                                  int32_t* mode, int32_t* ctas) {
  if (B < 1 || max_T < 1 || inplace < 0 || inplace > 2 ||
      max_T > (inplace == kKVChain ? EE_MAX_CHAIN : EE_MAX_TREE) || n_q < 1 || n_kv < 1 || n_q % n_kv != 0 ||
      max_ctx < 0 || !splits || !chunk || !mode || !ctas)
    return EE_ERR_INVALID_ARG;
  int dev = 0;
  {
    const ee_status ds = current_device(&dev);
    if (ds != EE_OK) return ds;
  }
  EE_CUDA_OK(set_attrs(dev));
  const int nrb = (max_T * (n_q / n_kv) + kRows - 1) / kRows;
  // the partial slots of a workspace sized by ee_workspace_size
  const size_t slots = std::max((size_t)B * n_q * kAttnMaxSplits, 2 * (size_t)kNumSMsMax);
  const Split sp = plan_for(dev, B, max_T, n_q, n_kv, max_ctx, inplace, slots);
  if (sp.S == 0) return EE_ERR_UNSUPPORTED;
  if (sp.bal) {
    *splits = sp.bal_ctas;
    *chunk = sp.bal_tiles * kKT;
    *mode = 3;
    *ctas = sp.ctas;
  } else {
    *splits = sp.S;
    *chunk = sp.chunk;
    *mode = sp.S == 1 ? 0 : (sp.coop ? 2 : 1);
    *ctas = nrb * sp.S * n_kv * B;
  }
  return EE_OK;
}

extern "C" ee_status ee_tree_verify_attn(const ee_bf16* q, const ee_bf16* k_tree,
                                         const ee_bf16* v_tree, const ee_bf16* k_cache,
                                         const ee_bf16* v_cache, int32_t num_pages,
                                         const int32_t* block_table, int32_t max_pages,
                                         const int32_t* ctx_len, int32_t max_ctx,
                                         const int32_t* node_off, const uint64_t* anc, int32_t B,
                                         int32_t total_nodes, int32_t max_T, int32_t n_q,
                                         int32_t n_kv, int32_t head_dim, float scale, float* out,
                                         void* ws, size_t ws_bytes, ee_stream_t stream) {
  return verify_attn(q, k_tree, v_tree, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx,
                     node_off, anc, B, total_nodes, max_T, n_q, n_kv, head_dim, scale, out, ws, ws_bytes, stream,
                     kKVTree);
}

extern "C" ee_status ee_tree_verify_attn_inplace(const ee_bf16* q, const ee_bf16* k_cache,
                                                 const ee_bf16* v_cache, int32_t num_pages,
                                                 const int32_t* block_table, int32_t max_pages,
                                                 const int32_t* ctx_len, int32_t max_ctx,
                                                 const int32_t* node_off, const uint64_t* anc, int32_t B,
                                                 int32_t total_nodes, int32_t max_T, int32_t n_q,
                                                 int32_t n_kv, int32_t head_dim, float scale, float* out,
                                                 void* ws, size_t ws_bytes, ee_stream_t stream) {
  return verify_attn(q, nullptr, nullptr, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx,
                     node_off, anc, B, total_nodes, max_T, n_q, n_kv, head_dim, scale, out, ws, ws_bytes, stream,
                     kKVInPlace);
}

extern "C" ee_status ee_chain_verify_attn(const ee_bf16* q, const ee_bf16* k_cache, const ee_bf16* v_cache,
                                          int32_t num_pages, const int32_t* block_table, int32_t max_pages,
                                          const int32_t* ctx_len, int32_t max_ctx, const int32_t* node_off,
                                          int32_t B, int32_t total_nodes, int32_t max_T, int32_t n_q,
                                          int32_t n_kv, int32_t head_dim, float scale, float* out, void* ws,
                                          size_t ws_bytes, ee_stream_t stream) {
  return verify_attn(q, nullptr, nullptr, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx,
                     node_off, nullptr, B, total_nodes, max_T, n_q, n_kv, head_dim, scale, out, ws, ws_bytes,
                     stream, kKVChain);
}
