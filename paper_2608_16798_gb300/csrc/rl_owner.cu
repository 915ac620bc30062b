// Sums over the tokens that a unit owns, for any token order: sequence-level importance
// weights (Sec. 3.2.4) over trajectories or over the deduplicated tokens of a rollout's
// prefix tree (Sec. 3.2.3), where a unit's tokens need not be contiguous.
//
//   owner_logratio_kernel  per token with M_t = 1: d = log pi_old - log pi_rollout in double,
//                          rounded to a fixed-point integer (2^-40 units); lanes of a warp
//                          with the same owner add theirs (__match_any_sync), one 64-bit
//                          integer atomic per owner and warp. Integer addition is associative,
//                          so the sums do not depend on the order of the atomics.
//   seq_weight_kernel      per unit: S = sum * 2^-40, w = min(exp(S), c-bar); optionally
//                          scales the unit's advantage by w.
//   token_scale_kernel     optionally scales per-token advantages by their owner's w.
#include <cstdint>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {
namespace owner {

constexpr double kFix = 1099511627776.0;  // 2^40
constexpr double kMaxTerm = 4194304.0;    // |d| <= 2^22 per token keeps every sum inside int64

__global__ void __launch_bounds__(256) owner_logratio_kernel(int64_t T, const int32_t* __restrict__ token_traj,
                                                             const uint8_t* __restrict__ mask,
                                                             const float* __restrict__ old_logp,
                                                             const float* __restrict__ rollout_logp, int32_t n_traj,
                                                             unsigned long long* __restrict__ acc, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x - lane; base < T; base += stride) {
    const int64_t t = base + lane;
    int32_t who = -1;
    long long q = 0;
    if (t < T && mask[t] != 0) {
      const int32_t i = token_traj[t];
      if (i < 0 || i >= n_traj) {
        flag_status(status, RL_DEV_BAD_TRAJ);
      } else {
        double d = static_cast<double>(old_logp[t]) - static_cast<double>(rollout_logp[t]);
        if (!(fabs(d) <= kMaxTerm)) {
          flag_status(status, RL_DEV_BAD_VALUE);
          d = d != d ? 0.0 : (d > 0 ? kMaxTerm : -kMaxTerm);
        }
        q = __double2ll_rn(d * kFix);
        who = i;
      }
    }
    const unsigned peers = __match_any_sync(0xffffffffu, who);
    long long sum = 0;
#pragma unroll 4
    for (int j = 0; j < 32; ++j) {
      const long long v = __shfl_sync(0xffffffffu, q, j);
      if ((peers >> j) & 1u) sum += v;
    }
    if (who >= 0 && lane == __ffs(peers) - 1) atomicAdd(&acc[who], static_cast<unsigned long long>(sum));
  }
}

__global__ void __launch_bounds__(256) seq_weight_kernel(int32_t n_traj, const unsigned long long* __restrict__ acc,
                                                         float cap, float* __restrict__ weight_out,
                                                         float* __restrict__ log_ratio_out,
                                                         float* __restrict__ traj_adv) {
  const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n_traj) return;
  const double S = static_cast<double>(static_cast<long long>(acc[i])) / kFix;
  double w = exp(S);
  if (cap > 0.f && w > cap) w = cap;
  const float wf = static_cast<float>(w);
  weight_out[i] = wf;
  if (log_ratio_out) log_ratio_out[i] = static_cast<float>(S);
  if (traj_adv) traj_adv[i] *= wf;
}

__global__ void __launch_bounds__(256) token_scale_kernel(int64_t T, const int32_t* __restrict__ token_traj,
                                                          int32_t n_traj, const float* __restrict__ weight,
                                                          float* __restrict__ token_adv) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < T; t += stride) {
    const int32_t i = token_traj[t];
    if (i >= 0 && i < n_traj) token_adv[t] *= weight[i];
  }
}

static int grid_for(int64_t work, int per_block, int cap) {
  int64_t g = (work + per_block - 1) / per_block;
  if (g < 1) g = 1;
  return static_cast<int>(g < cap ? g : cap);
}

}  // namespace owner
}  // namespace rl

extern "C" rl_status rl_sequence_is_weights(int32_t n_traj, int64_t n_tokens, const int32_t* token_traj,
                                            const uint8_t* mask, const float* old_logp, const float* rollout_logp,
                                            float cap, float* weight_out, float* log_ratio_out,
                                            float* traj_adv_inout, float* token_adv_inout, void* ws, size_t ws_bytes,
                                            rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (n_traj < 0 || n_tokens < 0) return set_error(RL_ERR_INVALID_ARG, "rl_sequence_is_weights: negative size");
  if (cap != cap) return set_error(RL_ERR_INVALID_ARG, "rl_sequence_is_weights: cap is NaN");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, "rl_sequence_is_weights: NULL workspace");
  if (ws_bytes < kWsHeader + static_cast<size_t>(n_traj) * sizeof(unsigned long long))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL,
                     "rl_sequence_is_weights: workspace smaller than rl_workspace_size(n_traj, 0, 0)");
  if (n_traj == 0) return RL_OK;
  if (!weight_out || (n_tokens > 0 && (!token_traj || !mask || !old_logp || !rollout_logp)))
    return set_error(RL_ERR_INVALID_ARG, "rl_sequence_is_weights: NULL array argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int32_t* status = reinterpret_cast<int32_t*>(ws);
  unsigned long long* acc =
      reinterpret_cast<unsigned long long*>(static_cast<char*>(ws) + ws_row_loss_offset());
  cudaError_t e = cudaMemsetAsync(acc, 0, static_cast<size_t>(n_traj) * sizeof(unsigned long long), s);
  if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync");
  if (n_tokens > 0) {
    owner::owner_logratio_kernel<<<owner::grid_for(n_tokens, 256, 152 * 8), 256, 0, s>>>(
        n_tokens, token_traj, mask, old_logp, rollout_logp, n_traj, acc, status);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "owner_logratio_kernel launch");
  }
  owner::seq_weight_kernel<<<(n_traj + 255) / 256, 256, 0, s>>>(n_traj, acc, cap, weight_out, log_ratio_out,
                                                                 traj_adv_inout);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "seq_weight_kernel launch");
  if (token_adv_inout && n_tokens > 0) {
    owner::token_scale_kernel<<<owner::grid_for(n_tokens, 256, 152 * 8), 256, 0, s>>>(n_tokens, token_traj, n_traj,
                                                                                      weight_out, token_adv_inout);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "token_scale_kernel launch");
  }
  return RL_OK;
}
