// Library-wide entry points: version, error text, workspace sizing and the
// device status word.
#include <cstdio>
#include <string>

#include "rl_host.h"

namespace rl {

static thread_local std::string g_last_error;

rl_status set_error(rl_status st, const std::string& msg) {
  g_last_error = msg;
  return st;
}

rl_status cuda_error(cudaError_t e, const char* what) {
  g_last_error = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
  return RL_ERR_CUDA;
}

void clear_error() { g_last_error.clear(); }

}  // namespace rl

extern "C" {

int32_t rl_version(void) { return 10000; }

const char* rl_last_error_message(void) { return rl::g_last_error.c_str(); }

size_t rl_workspace_size(int64_t max_rows, int64_t V, int64_t D) {
  if (max_rows < 0) max_rows = 0;
  if (D > 0 && V > 0) return rl::head_workspace_bytes(max_rows, V, D);
  const size_t rows_bytes = (static_cast<size_t>(max_rows) * sizeof(double) + 255) & ~size_t(255);
  return rl::kWsHeader + rows_bytes;
}

rl_status rl_workspace_init(void* ws, size_t ws_bytes, rl_stream_t stream) {
  rl::clear_error();
  if (!ws) return rl::set_error(RL_ERR_INVALID_ARG, "rl_workspace_init: ws is NULL");
  if (ws_bytes < rl::kWsHeader)
    return rl::set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_workspace_init: workspace smaller than its header");
  cudaError_t e = cudaMemsetAsync(ws, 0, rl::kWsHeader, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return rl::cuda_error(e, "rl_workspace_init: cudaMemsetAsync");
  return RL_OK;
}

rl_status rl_query_status(const void* ws, rl_stream_t stream, int32_t* device_status_out) {
  rl::clear_error();
  if (!ws || !device_status_out) return rl::set_error(RL_ERR_INVALID_ARG, "rl_query_status: NULL argument");
  int32_t word = 0;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(&word, ws, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return rl::cuda_error(e, "rl_query_status: cudaMemcpyAsync");
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return rl::cuda_error(e, "rl_query_status: cudaStreamSynchronize");
  *device_status_out = word;
  if (word == 0) return RL_OK;
  if (word & RL_DEV_TIMEOUT) {
    rl::set_error(RL_ERR_TIMEOUT, "device status: a bounded wait ran out");
    return RL_ERR_TIMEOUT;
  }
  char buf[160];
  std::snprintf(buf, sizeof(buf), "device status 0x%x:%s%s%s", word,
                (word & RL_DEV_BAD_TOKEN) ? " token id out of range;" : "",
                (word & RL_DEV_BAD_TRAJ) ? " trajectory index out of range;" : "",
                (word & RL_DEV_BAD_OFFSETS) ? " inconsistent offsets;" : "");
  return rl::set_error(RL_ERR_DEVICE_CHECK, buf);
}

}  // extern "C"
