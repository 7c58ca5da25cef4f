// ee_kv_compact: append the accepted path's K/V rows to the paged cache, for
// every layer (EfficientEdit Sec. III-A: accepted draft tokens extend the
// prefix, so the K/V computed for them in the verification pass become cache
// entries).  Path entry k of sequence s lands at position ctx + k.
//
// Pure data movement: one warp per (sequence, path entry, group of
// kLayersPerWarp layers) copies the n_kv K rows and n_kv V rows (head_dim bf16
// = 256 bytes each) of each of its layers with 16-byte vector loads/stores,
// all of a batch's loads in flight before its stores.  HBM-bound:
// 2 * 2 * n_kv * 256 bytes per entry and layer.
//
// ee_kv_compact_inplace: the same result when the tree's K/V already sit at
// positions ctx + i.  Path entry k is node path[k] >= k: entries with
// path[k] == k are in place (all of a reuse chain's), the others move down
// from ctx + path[k] to ctx + k.  A destination can be a later entry's source,
// so one CTA per (layer, sequence, KV head) first reads every moving row into
// shared memory and, after a barrier, writes them all.
#include "ee_common.cuh"

// Both kernels start before the LM head that produces path / accept_len has
// finished (programmatic dependent launch).  Everything another kernel may
// have written is read after griddepcontrol.wait with plain coherent loads
// (__ldcg), never through const __restrict__ parameters: the compiler may
// treat such loads as invariant and issue them before the wait.

namespace {

constexpr int kWarpsPerBlock = 8;
constexpr int kVecPerRow = EE_HEAD_DIM * 2 / 16;   // uint4 per head row
constexpr int kBatch = 8;                          // uint4 a lane holds between its loads and stores
constexpr int kLayersPerWarp = 4;

// kNkv > 0: the KV head count as a constant (the index arithmetic becomes
// shifts); 0: taken from n_kv_arg
template <int kNkv>
__global__ void __launch_bounds__(32 * kWarpsPerBlock)
kv_compact_kernel(const uint4* k_tree, const uint4* v_tree, int64_t tree_layer_stride, uint4* k_cache,
                  uint4* v_cache, int64_t cache_layer_stride, int num_pages, const int32_t* block_table,
                  int max_pages, const int32_t* ctx_in, int32_t* ctx_out, const int32_t* node_off,
                  const int32_t* path, const int32_t* accept_len, int max_T, int n_kv_arg, int total_nodes,
                  int L, int32_t* dst_slot, int32_t* err) {
  const int n_kv = kNkv > 0 ? kNkv : n_kv_arg;
  ee::pdl_allow_next();
  ee::pdl_wait();   // no global access before the previous kernel's writes are visible
  const int lane = threadIdx.x & 31;
  const int k = blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
  const int b = blockIdx.y;
  const int l = blockIdx.z;      // layer group
  if (k >= max_T) return;
  const int o = __ldcg(node_off + b);
  const int T = __ldcg(node_off + b + 1) - o;
  const int acc = __ldcg(accept_len + b);
  const int ctx = __ldcg(ctx_in + b);
  const bool lead = (l == 0 && lane == 0);
  if (acc < 0 || acc >= T || acc >= max_T || ctx < 0 || o < 0 || o + T > total_nodes) {
    if (lead) {
      if (k == 0) ee::flag_error(err, EE_DEVERR_PATH);
      dst_slot[(size_t)b * max_T + k] = -1;
    }
    return;
  }
  if (k > acc) {
    if (lead) dst_slot[(size_t)b * max_T + k] = -1;
    return;
  }
  if (lead && k == 0) ctx_out[b] = ctx + acc + 1;
  const int node = __ldcg(path + (size_t)b * max_T + k);
  const int pos = ctx + k;
  const int pg = pos / EE_PAGE;
  const int page = pg < max_pages ? __ldcg(block_table + (size_t)b * max_pages + pg) : -1;
  if (node < 0 || node >= T || page < 0 || page >= num_pages) {
    if (lead) {
      ee::flag_error(err, (node < 0 || node >= T) ? EE_DEVERR_PATH : EE_DEVERR_PAGE);
      dst_slot[(size_t)b * max_T + k] = -1;
    }
    return;
  }
  const int row = pos % EE_PAGE;
  if (lead) dst_slot[(size_t)b * max_T + k] = page * EE_PAGE + row;
  // 16 uint4 per head row; K rows then V rows
  const int64_t tl = tree_layer_stride / 8;   // layer strides in uint4 (given in bf16 elements)
  const int64_t cl = cache_layer_stride / 8;
  // the warp's layers [l0, l1): up to kBatch vectors per lane are loaded
  // before any is stored, so a warp has all its reads of a batch in flight
  const int l0 = l * kLayersPerWarp, l1 = min(L, l0 + kLayersPerWarp);
  const int nh = n_kv * kVecPerRow;               // uint4 of one K (or V) entry
  const int nvec = 2 * nh;                        // per layer
  const int tot = (l1 - l0) * nvec;
  for (int v0 = 0; v0 < tot; v0 += 32 * kBatch) {
    uint4 buf[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int v = v0 + 32 * u + lane;
      if (v < tot) {
        const int li = v / nvec, w = v - li * nvec;
        const int which = w / nh;               // 0 = K, 1 = V
        const int64_t src = tl * (l0 + li) + (int64_t)(o + node) * nh + (w - which * nh);
        buf[u] = __ldcg((which ? v_tree : k_tree) + src);
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int v = v0 + 32 * u + lane;
      if (v < tot) {
        const int li = v / nvec, w = v - li * nvec;
        const int which = w / nh;
        const int rem = w - which * nh;
        const int h = rem / kVecPerRow, c = rem % kVecPerRow;
        const int64_t dst = cl * (l0 + li) + (((int64_t)page * n_kv + h) * EE_PAGE + row) * kVecPerRow + c;
        (which ? v_cache : k_cache)[dst] = buf[u];
      }
    }
  }
}

constexpr int kInplaceThreads = 256;
constexpr size_t kInplaceSmem = (size_t)EE_MAX_TREE * 2 * kVecPerRow * 16;   // K and V rows, 64 KB

__global__ void __launch_bounds__(kInplaceThreads)
kv_compact_inplace_kernel(uint4* k_cache, uint4* v_cache, int64_t cache_layer_stride, int num_pages,
                          const int32_t* block_table, int max_pages, const int32_t* ctx_in, int32_t* ctx_out,
                          const int32_t* node_off, const int32_t* path, const int32_t* accept_len, int max_T,
                          int n_kv, int total_nodes, int32_t* dst_slot, int32_t* err) {
  extern __shared__ uint4 stage[];   // [entry][K 16 | V 16] uint4
  ee::pdl_allow_next();
  ee::pdl_wait();   // no global access before the previous kernel's writes are visible
  const int h = blockIdx.x, b = blockIdx.y, l = blockIdx.z;
  const bool lead = h == 0 && l == 0;
  const int o = __ldcg(node_off + b);
  const int T = __ldcg(node_off + b + 1) - o;
  const int acc = __ldcg(accept_len + b);
  const int ctx = __ldcg(ctx_in + b);
  const bool seq_ok = acc >= 0 && acc < T && acc < max_T && ctx >= 0 && o >= 0 && o + T <= total_nodes;
  // entry k: its node, source and destination slots.  Only a tree (at most
  // EE_MAX_TREE nodes) moves entries; a longer path (a linear draft) must be
  // in place.  A bad node or page anywhere stops the whole sequence (every CTA
  // of it decides alike).
  __shared__ int s_src[EE_MAX_TREE], s_dst[EE_MAX_CHAIN];
  bool bad = false;
  for (int k = threadIdx.x; seq_ok && k <= acc; k += kInplaceThreads) {
    const int node = __ldcg(path + (size_t)b * max_T + k);
    const int dpos = ctx + k, spos = ctx + node;
    const int dpg = dpos / EE_PAGE < max_pages ? __ldcg(block_table + (size_t)b * max_pages + dpos / EE_PAGE) : -1;
    const int spg =
        (node >= 0 && spos / EE_PAGE < max_pages) ? __ldcg(block_table + (size_t)b * max_pages + spos / EE_PAGE) : -1;
    if (node < k || node >= T || (k >= EE_MAX_TREE && node != k)) {
      bad = true;
      if (lead) ee::flag_error(err, EE_DEVERR_PATH);
    } else if (dpg < 0 || dpg >= num_pages || spg < 0 || spg >= num_pages) {
      bad = true;
      if (lead) ee::flag_error(err, EE_DEVERR_PAGE);
    } else {
      s_dst[k] = dpg * EE_PAGE + dpos % EE_PAGE;
      if (k < EE_MAX_TREE) s_src[k] = node != k ? spg * EE_PAGE + spos % EE_PAGE : -1;   // -1: in place
    }
  }
  const bool stop = __syncthreads_or(bad) || !seq_ok;
  if (lead)
    for (int k = threadIdx.x; k < max_T; k += kInplaceThreads)
      dst_slot[(size_t)b * max_T + k] = (!stop && k <= acc) ? s_dst[k] : -1;
  if (lead && threadIdx.x == 0) {
    if (!seq_ok) ee::flag_error(err, EE_DEVERR_PATH);
    else ctx_out[b] = ctx + acc + 1;
  }
  if (stop) return;
  const int nm = min(acc, EE_MAX_TREE - 1);   // entries that may move: 0 .. nm
  // row (slot, head h) of layer l starts at uint4 ((slot / PAGE * n_kv + h) * PAGE + slot % PAGE) * 16
  const int64_t cl = cache_layer_stride / 8 * l;
  auto row = [&](int slot) -> int64_t {
    return cl + (((int64_t)(slot / EE_PAGE) * n_kv + h) * EE_PAGE + slot % EE_PAGE) * kVecPerRow;
  };
  const int n = (nm + 1) * 2 * kVecPerRow;
  for (int v = threadIdx.x; v < n; v += kInplaceThreads) {   // gather every moving row
    const int e = v / (2 * kVecPerRow), r = v % (2 * kVecPerRow);
    if (s_src[e] < 0) continue;
    const int64_t a = row(s_src[e]) + (r % kVecPerRow);
    stage[v] = r < kVecPerRow ? __ldcg(k_cache + a) : __ldcg(v_cache + a);
  }
  __syncthreads();
  for (int v = threadIdx.x; v < n; v += kInplaceThreads) {   // then scatter them
    const int e = v / (2 * kVecPerRow), r = v % (2 * kVecPerRow);
    if (s_src[e] < 0) continue;
    const int64_t a = row(s_dst[e]) + (r % kVecPerRow);
    if (r < kVecPerRow) k_cache[a] = stage[v];
    else v_cache[a] = stage[v];
  }
}

}  // namespace

extern "C" ee_status ee_kv_compact(const ee_bf16* k_tree, const ee_bf16* v_tree,
                                   int64_t tree_layer_stride, ee_bf16* k_cache, ee_bf16* v_cache,
                                   int64_t cache_layer_stride, int32_t L, int32_t num_pages,
                                   const int32_t* block_table, int32_t max_pages,
                                   const int32_t* ctx_len_in, int32_t* ctx_len_out,
                                   const int32_t* node_off, const int32_t* path,
                                   const int32_t* accept_len, int32_t B, int32_t max_T, int32_t n_kv,
                                   int32_t head_dim, int32_t* dst_slot, void* ws, size_t ws_bytes,
                                   ee_stream_t stream) {
  if (B < 0 || L < 0 || max_T < 1 || max_T > EE_MAX_CHAIN || n_kv < 1 || num_pages < 1 ||
      max_pages < 1)
    return EE_ERR_INVALID_ARG;
  if (head_dim != EE_HEAD_DIM) return EE_ERR_UNSUPPORTED;
  if (B == 0) return EE_OK;
  if (!k_tree || !v_tree || !k_cache || !v_cache || !block_table || !ctx_len_in || !ctx_len_out ||
      !node_off || !path || !accept_len || !dst_slot || !ws)
    return EE_ERR_INVALID_ARG;
  if (ctx_len_in == ctx_len_out) return EE_ERR_INVALID_ARG;
  if (!ee::aligned(k_tree, 16) || !ee::aligned(v_tree, 16) || !ee::aligned(k_cache, 16) ||
      !ee::aligned(v_cache, 16) || tree_layer_stride % 8 || cache_layer_stride % 8)
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  if (L == 0) return EE_OK;
  if (tree_layer_stride % ((int64_t)n_kv * head_dim)) return EE_ERR_INVALID_ARG;
  const int total_nodes = (int)(tree_layer_stride / ((int64_t)n_kv * head_dim));
  dim3 grid((max_T + kWarpsPerBlock - 1) / kWarpsPerBlock, B, (L + kLayersPerWarp - 1) / kLayersPerWarp);
  auto kern = n_kv == 1   ? kv_compact_kernel<1>
              : n_kv == 2 ? kv_compact_kernel<2>
              : n_kv == 4 ? kv_compact_kernel<4>
              : n_kv == 8 ? kv_compact_kernel<8>
                          : kv_compact_kernel<0>;
  EE_CUDA_OK(ee::launch_pdl(
      kern, grid, dim3(32 * kWarpsPerBlock), 0, (cudaStream_t)stream, 1,
      reinterpret_cast<const uint4*>(k_tree), reinterpret_cast<const uint4*>(v_tree),
      tree_layer_stride, reinterpret_cast<uint4*>(k_cache), reinterpret_cast<uint4*>(v_cache),
      cache_layer_stride, num_pages, block_table, max_pages, ctx_len_in, ctx_len_out, node_off, path,
      accept_len, max_T, n_kv, total_nodes, (int)L, dst_slot, ee::err_word(ws)));
  return EE_OK;
}

extern "C" ee_status ee_kv_compact_inplace(ee_bf16* k_cache, ee_bf16* v_cache, int64_t cache_layer_stride,
                                           int32_t L, int32_t num_pages, const int32_t* block_table,
                                           int32_t max_pages, const int32_t* ctx_len_in, int32_t* ctx_len_out,
                                           const int32_t* node_off, const int32_t* path,
                                           const int32_t* accept_len, int32_t B, int32_t total_nodes,
                                           int32_t max_T, int32_t n_kv, int32_t head_dim, int32_t* dst_slot,
                                           void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (B < 0 || L < 0 || max_T < 1 || max_T > EE_MAX_CHAIN || n_kv < 1 || num_pages < 1 || max_pages < 1 ||
      total_nodes < 0)
    return EE_ERR_INVALID_ARG;
  if (head_dim != EE_HEAD_DIM) return EE_ERR_UNSUPPORTED;
  if (B == 0) return EE_OK;
  if (!k_cache || !v_cache || !block_table || !ctx_len_in || !ctx_len_out || !node_off || !path ||
      !accept_len || !dst_slot || !ws)
    return EE_ERR_INVALID_ARG;
  if (ctx_len_in == ctx_len_out) return EE_ERR_INVALID_ARG;
  if (!ee::aligned(k_cache, 16) || !ee::aligned(v_cache, 16) || cache_layer_stride % 8)
    return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  if (L == 0) return EE_OK;
  {
    // the dynamic shared memory attribute, set once per device
    int dev = 0;
    const ee_status ds = ee::current_device(&dev);
    if (ds != EE_OK) return ds;
    static std::mutex mu;
    static bool attr_set[ee::kMaxDevices] = {};
    std::lock_guard<std::mutex> lock(mu);
    if (!attr_set[dev]) {
      EE_CUDA_OK(cudaFuncSetAttribute(kv_compact_inplace_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)kInplaceSmem));
      attr_set[dev] = true;
    }
  }
  dim3 grid(n_kv, B, L);
  EE_CUDA_OK(ee::launch_pdl(kv_compact_inplace_kernel, grid, dim3(kInplaceThreads), kInplaceSmem,
                            (cudaStream_t)stream, 1, reinterpret_cast<uint4*>(k_cache),
                            reinterpret_cast<uint4*>(v_cache), cache_layer_stride, num_pages, block_table,
                            max_pages, ctx_len_in, ctx_len_out, node_off, path, accept_len, max_T, n_kv,
                            total_nodes, dst_slot, ee::err_word(ws)));
  return EE_OK;
}
