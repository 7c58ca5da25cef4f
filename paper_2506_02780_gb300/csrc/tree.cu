// ee_tree_prepare: depth and root-path (ancestor) bitmask of every draft-tree
// node.  The paper verifies linear drafts (EfficientEdit Sec. III-A); several
// match points and generated branches share a prefix, so the step scores them
// together as a tree whose nodes each see only their own root-to-node path.
//
// One CTA of 128 threads per sequence, thread i for node i.  After a
// block-wide validation that parent[i] < i, the root paths are built by
// pointer jumping in shared memory: node i keeps the nodes from itself up to
// (not including) its current jump target and a jump target that doubles its
// reach every round, so 7 rounds cover any path of a 128-node tree.
#include "ee_common.cuh"

namespace {

__global__ void __launch_bounds__(EE_MAX_TREE)
tree_prepare_kernel(const int32_t* parent, const int32_t* node_off, int32_t* depth, uint64_t* anc,
                    int total_nodes, int32_t* err) {
  // parent / node_off may come from an earlier kernel: plain loads after the
  // dependent-launch wait (no const __restrict__, whose loads may be issued
  // before it)
  __shared__ int32_t s_jmp[2][EE_MAX_TREE];
  __shared__ uint64_t s_a0[2][EE_MAX_TREE], s_a1[2][EE_MAX_TREE];
  ee::pdl_allow_next();
  ee::pdl_wait();   // no global access before the previous kernel's writes are visible
  const int b = blockIdx.x;
  const int i = threadIdx.x;
  const int o = node_off[b];
  const int T = node_off[b + 1] - o;
  if (T < 1 || T > EE_MAX_TREE || o < 0 || o + T > total_nodes) {
    if (i == 0) ee::flag_error(err, EE_DEVERR_TREE);
    return;
  }
  int p = -1;
  bool ok = true;
  if (i < T) {
    p = parent[o + i];
    ok = (i == 0) ? (p == -1) : (p >= 0 && p < i);
  }
  const bool all_ok = __syncthreads_and(ok);
  if (!all_ok) {
    if (i == 0) ee::flag_error(err, EE_DEVERR_TREE);
    if (i < T) {
      depth[o + i] = 0;
      anc[2 * (size_t)(o + i)] = 0;
      anc[2 * (size_t)(o + i) + 1] = 0;
    }
    return;
  }
  // every thread takes part in the rounds (nodes past T are isolated roots)
  int j = i < T ? p : -1;
  uint64_t a0 = i < 64 ? 1ull << i : 0ull, a1 = i < 64 ? 0ull : 1ull << (i - 64);
  s_jmp[0][i] = j;
  s_a0[0][i] = a0;
  s_a1[0][i] = a1;
  __syncthreads();
#pragma unroll
  for (int r = 0; r < 7; ++r) {   // 2^7 = 128 > the longest path
    const int cur = r & 1;
    if (j >= 0) {
      a0 |= s_a0[cur][j];
      a1 |= s_a1[cur][j];
      j = s_jmp[cur][j];
    }
    s_jmp[cur ^ 1][i] = j;
    s_a0[cur ^ 1][i] = a0;
    s_a1[cur ^ 1][i] = a1;
    __syncthreads();
  }
  if (i >= T) return;
  depth[o + i] = __popcll(a0) + __popcll(a1) - 1;   // the path holds the root and the node
  anc[2 * (size_t)(o + i)] = a0;
  anc[2 * (size_t)(o + i) + 1] = a1;
}

}  // namespace

extern "C" ee_status ee_tree_prepare(const int32_t* parent, const int32_t* node_off, int32_t B,
                                     int32_t total_nodes, int32_t* depth, uint64_t* anc,
                                     void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (B < 0 || total_nodes < 0) return EE_ERR_INVALID_ARG;
  if (B == 0) return EE_OK;
  if (!parent || !node_off || !depth || !anc || !ws) return EE_ERR_INVALID_ARG;
  if (!ee::aligned(anc, 8)) return EE_ERR_INVALID_ARG;
  if (ws_bytes < ee::kWorkspaceBytes) return EE_ERR_WORKSPACE;
  EE_CUDA_OK(ee::launch_pdl(tree_prepare_kernel, dim3(B), dim3(EE_MAX_TREE), 0, (cudaStream_t)stream,
                             1, parent, node_off, depth, anc, total_nodes, ee::err_word(ws)));
  return EE_OK;
}
