// Library-wide entry points: version, error text, workspace sizing and the
// device status word.
#include <cstdio>
#include <string>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {

// One CTA waits, through the kernels' own bounded waits (plain and cluster-scope), on an
// mbarrier that nothing arrives at; each wait gives up after limit_ns, sets RL_DEV_TIMEOUT and
// the kernel returns, leaving the context usable. waited_ns receives the longest wait seen.
__global__ void __launch_bounds__(32) wait_selftest_kernel(int32_t* status, uint64_t limit_ns,
                                                           unsigned long long* waited_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  const uint64_t t0 = global_timer_ns();
  const bool a = mbar_wait_bounded(&bar, 0, limit_ns);  // phase 0 never completes
  const bool b = mbar_wait_cluster_bounded(&bar, 0, limit_ns);
  const uint64_t dt = global_timer_ns() - t0;
  if (threadIdx.x == 0) {
    if (!a || !b) flag_status(status, RL_DEV_TIMEOUT);
    if (waited_ns) atomicMax(waited_ns, static_cast<unsigned long long>(dt));
  }
}

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

size_t rl_fused_head_workspace_size(int64_t T, int64_t V, int64_t D, int64_t group_tokens) {
  if (T < 0) T = 0;
  if (V < 1 || D < 1) return rl_workspace_size(T, V, D);
  return rl::head_workspace_bytes_grouped(T, V, D, group_tokens);
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

rl_status rl_selftest_bounded_wait(void* ws, size_t ws_bytes, int64_t limit_ns, uint64_t* waited_ns,
                                   rl_stream_t stream) {
  rl::clear_error();
  if (!ws) return rl::set_error(RL_ERR_INVALID_ARG, "rl_selftest_bounded_wait: ws is NULL");
  if (ws_bytes < rl::kWsHeader)
    return rl::set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_selftest_bounded_wait: workspace smaller than its header");
  if (reinterpret_cast<uintptr_t>(ws) % 16 != 0)
    return rl::set_error(RL_ERR_ALIGNMENT, "rl_selftest_bounded_wait: ws not 16-byte aligned");
  if (limit_ns < 1000 || limit_ns > static_cast<int64_t>(rl::kWaitLimitNs))
    return rl::set_error(RL_ERR_INVALID_ARG, "rl_selftest_bounded_wait: limit_ns outside [1e3, 2e9]");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  rl::wait_selftest_kernel<<<1, 32, 0, s>>>(reinterpret_cast<int32_t*>(ws), static_cast<uint64_t>(limit_ns),
                                            reinterpret_cast<unsigned long long*>(waited_ns));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return rl::cuda_error(e, "wait_selftest_kernel launch");
  return RL_OK;
}

}  // extern "C"
