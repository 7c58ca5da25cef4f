// Library-level entry points of libee: version, status strings, workspace
// sizing/initialisation and the device error word.
#include "ee_common.cuh"
#include "ee_ptx.cuh"

extern "C" const char* ee_version(void) { return "libee 0.1 (sm_103a)"; }

extern "C" const char* ee_status_string(ee_status s) {
  switch (s) {
    case EE_OK: return "ok";
    case EE_ERR_INVALID_ARG: return "invalid argument";
    case EE_ERR_UNSUPPORTED: return "unsupported configuration";
    case EE_ERR_CUDA: return "CUDA error";
    case EE_ERR_DEVICE: return "device error word set";
    case EE_ERR_WORKSPACE: return "workspace too small";
  }
  return "unknown status";
}

extern "C" size_t ee_workspace_size(int32_t B, int32_t total_nodes, int32_t n_q, int32_t head_dim,
                                    int32_t max_ctx) {
  if (B < 0 || total_nodes < 0 || n_q < 0 || head_dim < 0 || max_ctx < 0) return 0;
  if (max_ctx == 0) return ee::kAttnPartOff;      // one chunk per row block: no attention slots
  // attention CTAs of a split launch: B x n_kv x ceil(max_T * g / 128) row
  // blocks (<= B x n_q, as max_T <= 128) x at most 16 chunks; a balanced
  // launch: two slots per resident CTA (one per SM)
  const size_t slots = std::max((size_t)B * n_q * ee::kAttnMaxSplits, 2 * (size_t)ee::kNumSMsMax);
  return ee::kAttnPartOff + slots * ee::kAttnPartBytes;
}

extern "C" ee_status ee_workspace_init(void* ws, size_t ws_bytes, ee_stream_t stream) {
  if (!ws || ws_bytes < ee::kWorkspaceBytes || !ee::aligned(ws, 256)) return EE_ERR_INVALID_ARG;
  EE_CUDA_OK(cudaMemsetAsync(ws, 0, ws_bytes, (cudaStream_t)stream));
  return EE_OK;
}

extern "C" ee_status ee_read_errors(void* ws, ee_stream_t stream, int32_t* bits) {
  if (!ws || !bits) return EE_ERR_INVALID_ARG;
  int32_t h = 0;
  EE_CUDA_OK(cudaMemcpyAsync(&h, ee::err_word(ws), sizeof(int32_t), cudaMemcpyDeviceToHost,
                             (cudaStream_t)stream));
  EE_CUDA_OK(cudaStreamSynchronize((cudaStream_t)stream));
  *bits = h;
  if (h) {
    EE_CUDA_OK(cudaMemsetAsync(ee::err_word(ws), 0, sizeof(int32_t), (cudaStream_t)stream));
    EE_CUDA_OK(cudaStreamSynchronize((cudaStream_t)stream));
    return EE_ERR_DEVICE;
  }
  return EE_OK;
}

namespace ee {
namespace {

// Makes the two kinds of bounded wait of the pipelines run out (an mbarrier
// nothing arrives at, a global counter nothing raises) and records how each
// ended; see ee_selftest_timeout in ee.h.
__global__ void __launch_bounds__(64) selftest_timeout_kernel(int32_t* err, const uint32_t* never_set,
                                                              int64_t* out) {
  __shared__ __align__(8) uint64_t s_bar[2];
  __shared__ volatile int s_abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&s_bar[0]), 1);
    mbar_init(smem_u32(&s_bar[1]), 1);
    s_abort = 0;
  }
  __syncthreads();
  if (lane == 0) {
    if (warp == 1) {   // start half a limit after warp 0
      const long long d0 = cycles();
      while (cycles() - d0 < kWaitLimitCycles / 2) {
      }
    }
    const long long t0 = cycles();
    // phase 0 of a fresh barrier completes only when its one arrival comes
    const bool ok = mbar_wait(smem_u32(&s_bar[warp]), 0u, &s_abort);
    out[1 + 2 * warp] = ok ? 1 : 0;
    out[2 + 2 * warp] = cycles() - t0;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const long long t0 = cycles();
    const bool ok = wait_count_geq(never_set, 1u);
    out[5] = ok ? 1 : 0;
    out[6] = cycles() - t0;
    out[0] = kWaitLimitCycles;
    if (s_abort || !ok) flag_error(err, EE_DEVERR_TIMEOUT);
  }
}

}  // namespace
}  // namespace ee

extern "C" ee_status ee_selftest_timeout(void* ws, size_t ws_bytes, int64_t* out, ee_stream_t stream) {
  if (!ws || !out || ws_bytes < ee::kWorkspaceBytes || !ee::aligned(ws, 256) || !ee::aligned(out, 8))
    return EE_ERR_INVALID_ARG;
  const uint32_t* never_set =
      reinterpret_cast<const uint32_t*>(static_cast<const char*>(ws) + ee::kNeverSetOff);
  ee::selftest_timeout_kernel<<<1, 64, 0, (cudaStream_t)stream>>>(ee::err_word(ws), never_set, out);
  EE_CUDA_OK(cudaGetLastError());
  return EE_OK;
}
