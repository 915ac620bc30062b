// Allocation-free form of rl_policy_loss_fwd_bwd.
//
// Some callers cannot allocate device memory at the point where they compute
// the loss: code running inside a framework's memory pool that forbids
// cudaMalloc during a step, a plugin that only receives pointers from its host
// application, or a process that must not grow its device footprint after
// start-up. They cannot provide the workspace that rl_policy_loss_fwd_bwd needs,
// so this entry point brings its own: a fixed array in device global memory,
// defined below, that every GPU which loads this library holds until the
// process exits.
#include <map>
#include <mutex>

#include "rl_host.h"

namespace rl {

// Largest microbatch (rows) the allocation-free entry point accepts.
constexpr int64_t kNoAllocMaxRows = 131072;

// The workspace of the allocation-free entry point: header (device status word)
// followed by one double per row. 256 + 131,072 * 8 bytes = 1 MiB + 256 bytes.
// In host code this name is only a handle for cudaGetSymbolAddress, never a
// device address.
static __device__ __align__(256) unsigned char g_noalloc_ws[kWsHeader + kNoAllocMaxRows * sizeof(double)];

// Device address of g_noalloc_ws on the current device, looked up once per device (the first
// call on a device) and kept for the life of the process: a cudaDeviceReset, which destroys the
// context that holds the array, makes the kept address stale.
static rl_status noalloc_workspace(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "rl_policy_loss_fwd_bwd_noalloc: cudaGetDevice");
  static std::mutex mu;
  static std::map<int, void*> addr;
  std::lock_guard<std::mutex> lock(mu);
  auto it = addr.find(dev);
  if (it == addr.end()) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_ws);
    if (e != cudaSuccess) return cuda_error(e, "rl_policy_loss_fwd_bwd_noalloc: cudaGetSymbolAddress");
    it = addr.emplace(dev, ptr).first;
  }
  *out = it->second;
  return RL_OK;
}

}  // namespace rl

extern "C" rl_status rl_policy_loss_fwd_bwd_noalloc(
    const void* logits, rl_dtype dtype, int64_t rows, int64_t V, int64_t ld, const int32_t* token_ids,
    const uint8_t* mask, const int32_t* token_traj, int32_t n_traj, const float* adv, const float* coef,
    const float* old_logp, const float* ref_logp, const float* rollout_logp, const rl_loss_params* params,
    void* grad_out, double* loss_accum, float* token_stats, int32_t* device_status, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (rows > kNoAllocMaxRows)
    return set_error(RL_ERR_UNSUPPORTED,
                     "rl_policy_loss_fwd_bwd_noalloc: rows exceeds the 131072-row limit of the built-in workspace; "
                     "split the microbatch or use rl_policy_loss_fwd_bwd with a caller workspace");
  void* ws = nullptr;
  rl_status st = noalloc_workspace(&ws);
  if (st != RL_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // The 256-byte header must start at zero: it holds the status word and the loss kernel's
  // finished-cluster counter, which a call that overlapped another one (or did not run to
  // its end) can leave non-zero; the per-cluster loss slots are written before they are read.
  cudaError_t e = cudaMemsetAsync(ws, 0, kWsHeader, s);
  if (e != cudaSuccess) return cuda_error(e, "rl_policy_loss_fwd_bwd_noalloc: cudaMemsetAsync");
  st = rl_policy_loss_fwd_bwd(logits, dtype, rows, V, ld, token_ids, mask, token_traj, n_traj, adv, coef, old_logp,
                              ref_logp, rollout_logp, params, grad_out, loss_accum, token_stats, ws,
                              kWsHeader + kNoAllocMaxRows * sizeof(double), stream);
  if (st != RL_OK) return st;
  if (device_status) {
    e = cudaMemcpyAsync(device_status, ws, sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_error(e, "rl_policy_loss_fwd_bwd_noalloc: cudaMemcpyAsync");
  }
  return RL_OK;
}
