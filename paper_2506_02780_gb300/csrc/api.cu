// Library-level entry points of libee: version, status strings, workspace
// sizing/initialisation and the device error word.
#include "ee_common.cuh"

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
  // blocks (<= B x n_q, as max_T <= 128) x at most 16 chunks
  return ee::kAttnPartOff + (size_t)B * n_q * ee::kAttnMaxSplits * ee::kAttnPartBytes;
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
