// Shared device/host helpers of libee (sm_103a).  Internal header.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <utility>

#include "../../include/ee.h"

namespace ee {

// ---------------------------------------------------------------------------
// Workspace layout (bytes from the start of `ws`):
//   [0, 4)              device error word (EE_DEVERR_* bits)
//   [16, 20)            LM-head "CTAs finished" ticket counter
//   [24, 28)            verification finalize "CTAs finished" ticket counter
//   [32, 36)            never-written flag (zero): the self-test's wait target
//   [256, 256+8*EE_MAX_LM_NODES)  LM-head packed running argmax per node
//   [kLmVerifyOff, +kLmVerifyBytes) LM-head verification partials
//   [kMatchOff, +kMatchBytes)     split reuse-span match: tickets and records
//   [kAttnPartOff, ...)           attention partial slots, kAttnPartBytes per
//                                 CTA of a split launch; the trailer of a row
//                                 block's first slot holds its arrival counters
// ---------------------------------------------------------------------------
constexpr size_t kErrOff = 0;
constexpr size_t kTicketOff = 16;
constexpr size_t kNeverSetOff = 32;
constexpr size_t kArgmaxOff = 256;
constexpr size_t kWorkspaceBytes = 256 + 8 * (size_t)EE_MAX_LM_NODES + 256;   // the fixed head
constexpr int kNumSMsMax = 152;       // LM-head grid bound (one persistent CTA per SM)
// LM-head verification partials (ee_lmhead_verify): per CTA and node of its
// node tile, the CTA's top-k (value, id) list and its (max, sum) of 2^logit;
// then the per-node global pruning threshold
constexpr int kLmMaxK = 8;
constexpr int kLmMaxBN = 256;
constexpr size_t kLmVerifyOff = kWorkspaceBytes;
// one (CTA, node) record: K values, K ids, (max, sum), padded to 16 bytes
__host__ __device__ constexpr int lm_rec_bytes(int K) { return (8 * K + 8 + 15) / 16 * 16; }
constexpr size_t kLmPartBytes = (size_t)kNumSMsMax * kLmMaxBN * lm_rec_bytes(kLmMaxK);
// then one u64 per node: the best K-th key any CTA has published (zero between
// calls); then the finalize step's ranked ids [node][K] and top_tau [node]
constexpr size_t kLmGthrOff = kLmPartBytes;
constexpr size_t kLmTkOff = kLmGthrOff + 8 * (size_t)EE_MAX_LM_NODES;
constexpr size_t kLmTauOff = kLmTkOff + 4 * (size_t)EE_MAX_LM_NODES * kLmMaxK;
constexpr size_t kLmVerifyBytes = kLmTauOff + 4 * (size_t)EE_MAX_LM_NODES;
constexpr size_t kFinTicketOff = 24;   // in the head: finalize CTAs finished
// reuse-span match split over several CTAs per sequence: per sequence a 16-byte
// ticket (zero between calls), then one record per CTA (its hit count and its
// first max_matches hits)
constexpr size_t kMatchOff = kLmVerifyOff + kLmVerifyBytes;
constexpr size_t kMatchBytes = (size_t)1 << 20;
constexpr size_t kAttnPartOff = kMatchOff + kMatchBytes;   // attention partial slots
constexpr int kAttnRows = 128;        // query rows (node x head-in-group) per attention CTA
constexpr int kAttnMaxSplits = 16;    // context chunks per row block
// one CTA's partial: 128 rows x 128 fp32 of O (column-chunk major), then
// 128 x (m, l), then a 256-byte trailer whose first 8 bytes are the row
// block's 64-bit arrival count (zeroed by ee_workspace_init; every launch that
// uses it raises it by the same constant, so it is never reset)
constexpr size_t kAttnMlOff = (size_t)kAttnRows * 128 * 4;
constexpr size_t kAttnCntOff = kAttnMlOff + (size_t)kAttnRows * 8;
constexpr size_t kAttnPartBytes = kAttnCntOff + 256;
constexpr int kNumSMs = 152;

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Host-side set-up that CUDA applies per device (kernel attributes, occupancy
// queries, device addresses of symbols) is cached per device ordinal: the
// current device's index, or EE_ERR_UNSUPPORTED beyond kMaxDevices.  Each cache
// is guarded by its own mutex, so host threads may call libee concurrently.
constexpr int kMaxDevices = 64;
inline ee_status current_device(int* dev) {
  if (cudaGetDevice(dev) != cudaSuccess) return EE_ERR_CUDA;
  return (*dev >= 0 && *dev < kMaxDevices) ? EE_OK : EE_ERR_UNSUPPORTED;
}

__device__ __forceinline__ void flag_error(int32_t* err, int bits) { atomicOr(err, bits); }

__host__ __device__ inline int32_t* err_word(void* ws) {
  return reinterpret_cast<int32_t*>(static_cast<char*>(ws) + kErrOff);
}

inline bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Number of context chunks a sequence of `ctx` cached positions uses in the
// split-KV attention.
__host__ __device__ inline int attn_splits_for(int ctx, int chunk) {
  int s = (ctx + chunk - 1) / chunk;
  return s < 1 ? 1 : s;
}

// Encode a TMA tensor map over a bf16 array with 128-byte swizzle and zero
// fill out of bounds.  dims[0] is the contiguous dimension; strides_bytes[i]
// is the byte stride of dimension i+1.  Returns false on failure.
bool encode_bf16_tmap(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                      const uint64_t* strides_bytes, const uint32_t* box);

// Programmatic dependent launch.  A kernel launched with
// launch_pdl() may start while the previous kernel in the stream is still
// running; it must call pdl_wait() before its first read of global memory that
// an earlier kernel may have written.  pdl_allow_next() lets the next kernel
// start early.  Both are no-ops when the kernel was launched normally.
__device__ __forceinline__ void pdl_allow_next() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Launch `kernel` on `stream` with programmatic stream serialisation (and an
// optional cluster size).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, unsigned cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace ee

#define EE_CUDA_OK(call)                                  \
  do {                                                    \
    cudaError_t e_ = (call);                              \
    if (e_ != cudaSuccess) return EE_ERR_CUDA;            \
  } while (0)

#define EE_LAUNCH_OK()                                    \
  do {                                                    \
    cudaError_t e_ = cudaGetLastError();                  \
    if (e_ != cudaSuccess) return EE_ERR_CUDA;            \
  } while (0)
