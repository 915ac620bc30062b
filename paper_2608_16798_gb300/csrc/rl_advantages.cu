// Group-relative advantages and loss coefficients over ragged trajectories.
//
//   traj_count_kernel   L_i = sum_t M_t over trajectory i's span of the packed
//                       stream, and token_traj[t] = i (one warp per trajectory).
//                       The 1 / sum_t M_{i,t} normaliser of the masked GRPO
//                       objective (Sec. 2.3.2).
//   group_adv_kernel    one CTA: per group (one warp each) the mean and
//                       population standard deviation of the valid members'
//                       rewards, A_i = (R_i - mu) / (sigma + eps) (Sec. 2.3.2
//                       GRPO advantage; Sec. 3.2.3; discarded rollouts leave
//                       the statistics, Sec. 3.4); then N = #{valid, L_i > 0}
//                       and the coefficients c_i.
//
// Both are latency-bound: they touch ~T + 30 n bytes, well under 0.1% of the
// logits stream of one microbatch.
#include <cstdint>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {

__global__ void __launch_bounds__(256) traj_count_kernel(int32_t n_traj, int64_t n_tokens,
                                                         const int64_t* __restrict__ traj_offsets,
                                                         const uint8_t* __restrict__ mask,
                                                         int32_t* __restrict__ n_tok_out,
                                                         int32_t* __restrict__ token_traj_out,
                                                         int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int64_t i = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  if (i >= n_traj) return;
  int64_t s = traj_offsets[i], e = traj_offsets[i + 1];
  if (s < 0 || e < s || e > n_tokens) {
    if (lane == 0) {
      flag_status(status, RL_DEV_BAD_OFFSETS);
      n_tok_out[i] = 0;
    }
    return;
  }
  int32_t cnt = 0;
  for (int64_t t = s + lane; t < e; t += 32) {
    cnt += mask[t] != 0;
    if (token_traj_out) token_traj_out[t] = static_cast<int32_t>(i);
  }
  cnt = warp_sum(cnt);
  if (lane == 0) n_tok_out[i] = cnt;
}

// L_i by owner, for tokens in any order (tree-packed batches, Sec. 3.2.3: each shared prefix
// token is one token of its rollout): lanes of a warp with the same owner are counted together
// and one integer atomic per owner and warp adds them (the counts are exact in any order).
__global__ void __launch_bounds__(256) owner_count_kernel(int64_t n_tokens, const int32_t* __restrict__ token_traj,
                                                          const uint8_t* __restrict__ mask, int32_t n_traj,
                                                          int32_t* __restrict__ n_tok_out, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x - lane; base < n_tokens;
       base += stride) {
    const int64_t t = base + lane;
    int32_t who = -1;
    if (t < n_tokens && mask[t] != 0) {
      const int32_t i = token_traj[t];
      if (i < 0 || i >= n_traj) flag_status(status, RL_DEV_BAD_TRAJ);
      else who = i;
    }
    const unsigned peers = __match_any_sync(0xffffffffu, who);
    if (who >= 0 && lane == __ffs(peers) - 1) atomicAdd(&n_tok_out[who], __popc(peers));
  }
}

constexpr int kAdvThreads = 1024;

__global__ void __launch_bounds__(kAdvThreads) group_adv_kernel(
    int32_t n_traj, int32_t n_groups, const int32_t* __restrict__ group_offsets,
    const float* __restrict__ rewards, const uint8_t* __restrict__ traj_valid,
    const int32_t* __restrict__ n_tok, double adv_eps, int32_t loss_agg, float* __restrict__ adv_out,
    float* __restrict__ coef_out, int32_t* status) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarps = kAdvThreads / 32;

  // trajectories outside every group keep A = 0
  for (int i = tid; i < n_traj; i += kAdvThreads) adv_out[i] = 0.f;
  __syncthreads();

  for (int g = warp; g < n_groups; g += kWarps) {
    const int b = group_offsets[g], e = group_offsets[g + 1];
    if (b < 0 || e < b || e > n_traj) {
      if (lane == 0) flag_status(status, RL_DEV_BAD_OFFSETS);
      continue;
    }
    // pass 1: count, sum, and min / max (all-equal test) over valid members
    int k = 0;
    double sum = 0.0;
    float lo = __int_as_float(0x7f800000), hi = -__int_as_float(0x7f800000);
    for (int i = b + lane; i < e; i += 32) {
      if (traj_valid && traj_valid[i] == 0) continue;
      const float r = rewards[i];
      ++k;
      sum += static_cast<double>(r);
      lo = fminf(lo, r);
      hi = fmaxf(hi, r);
    }
    k = warp_sum(k);
    sum = warp_sum(sum);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (k == 0 || lo == hi) continue;  // nothing valid, or all valid rewards equal: A = 0
    const double mu = sum / k;
    double sq = 0.0;
    for (int i = b + lane; i < e; i += 32) {
      if (traj_valid && traj_valid[i] == 0) continue;
      const double d = static_cast<double>(rewards[i]) - mu;
      sq += d * d;
    }
    sq = warp_sum(sq);
    const double denom = sqrt(sq / k) + adv_eps;
    for (int i = b + lane; i < e; i += 32) {
      if (traj_valid && traj_valid[i] == 0) continue;
      adv_out[i] = static_cast<float>((static_cast<double>(rewards[i]) - mu) / denom);
    }
  }

  // N = number of valid trajectories with L_i > 0; S = sum of their L_i
  __shared__ long long red_n[kWarps], red_s[kWarps];
  long long cnt = 0, tok = 0;
  for (int i = tid; i < n_traj; i += kAdvThreads) {
    const bool counted = (!traj_valid || traj_valid[i] != 0) && n_tok[i] > 0;
    cnt += counted;
    tok += counted ? n_tok[i] : 0;
  }
  cnt = warp_sum(cnt);
  tok = warp_sum(tok);
  if (lane == 0) {
    red_n[warp] = cnt;
    red_s[warp] = tok;
  }
  __syncthreads();
  long long N = 0, S = 0;
  for (int w = 0; w < kWarps; ++w) {
    N += red_n[w];
    S += red_s[w];
  }
  for (int i = tid; i < n_traj; i += kAdvThreads) {
    const int32_t L = n_tok[i];
    const bool counted = (!traj_valid || traj_valid[i] != 0) && L > 0;
    float c = 0.f;
    if (counted) {
      if (loss_agg == RL_AGG_SEQ_MEAN_TOKEN_MEAN)
        c = static_cast<float>(1.0 / (static_cast<double>(N) * static_cast<double>(L)));
      else if (loss_agg == RL_AGG_TOKEN_MEAN)
        c = static_cast<float>(1.0 / static_cast<double>(S));
      else
        c = 1.f;
    }
    coef_out[i] = c;
  }
}

}  // namespace rl

extern "C" rl_status rl_group_advantages(int32_t n_traj, int32_t n_groups, const int32_t* group_offsets,
                                         const float* rewards, const uint8_t* traj_valid, int64_t n_tokens,
                                         const int64_t* traj_offsets, const uint8_t* mask,
                                         const rl_loss_params* params, float* adv_out, float* coef_out,
                                         int32_t* n_tok_out, int32_t* token_traj_out, void* ws,
                                         size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (n_traj < 0 || n_groups < 0 || n_tokens < 0)
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: negative size");
  if (!params) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: params is NULL");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: ws is NULL");
  if (ws_bytes < rl_workspace_size(0, 0, 0))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_group_advantages: workspace too small");
  if (params->loss_agg < RL_AGG_SEQ_MEAN_TOKEN_MEAN || params->loss_agg > RL_AGG_TOKEN_SUM)
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: unknown loss_agg");
  if (!(params->adv_eps >= 0.f)) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: adv_eps < 0");
  if (n_traj == 0) return RL_OK;
  if (!group_offsets && n_groups > 0) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: group_offsets is NULL");
  if (!rewards || !traj_offsets || !adv_out || !coef_out || !n_tok_out)
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: NULL array argument");
  if (n_tokens > 0 && !mask) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages: mask is NULL");
  if (n_tokens > INT32_MAX) return set_error(RL_ERR_UNSUPPORTED, "rl_group_advantages: more than 2^31 - 1 tokens");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int32_t* status = reinterpret_cast<int32_t*>(ws);
  const int warps_per_block = 256 / 32;
  const unsigned blocks = static_cast<unsigned>((static_cast<int64_t>(n_traj) + warps_per_block - 1) / warps_per_block);
  traj_count_kernel<<<blocks, 256, 0, s>>>(n_traj, n_tokens, traj_offsets, mask, n_tok_out, token_traj_out, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "rl_group_advantages: traj_count_kernel launch");
  group_adv_kernel<<<1, kAdvThreads, 0, s>>>(n_traj, n_groups, group_offsets, rewards, traj_valid, n_tok_out,
                                             static_cast<double>(params->adv_eps), params->loss_agg, adv_out,
                                             coef_out, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "rl_group_advantages: group_adv_kernel launch");
  return RL_OK;
}

extern "C" rl_status rl_group_advantages_by_owner(int32_t n_traj, int32_t n_groups, const int32_t* group_offsets,
                                                  const float* rewards, const uint8_t* traj_valid, int64_t n_tokens,
                                                  const int32_t* token_traj, const uint8_t* mask,
                                                  const rl_loss_params* params, float* adv_out, float* coef_out,
                                                  int32_t* n_tok_out, void* ws, size_t ws_bytes,
                                                  rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (n_traj < 0 || n_groups < 0 || n_tokens < 0)
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: negative size");
  if (!params) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: params is NULL");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: ws is NULL");
  if (ws_bytes < rl_workspace_size(0, 0, 0))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_group_advantages_by_owner: workspace too small");
  if (params->loss_agg < RL_AGG_SEQ_MEAN_TOKEN_MEAN || params->loss_agg > RL_AGG_TOKEN_SUM)
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: unknown loss_agg");
  if (!(params->adv_eps >= 0.f)) return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: adv_eps < 0");
  if (n_traj == 0) return RL_OK;
  if (!group_offsets && n_groups > 0)
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: group_offsets is NULL");
  if (!rewards || !adv_out || !coef_out || !n_tok_out || (n_tokens > 0 && (!token_traj || !mask)))
    return set_error(RL_ERR_INVALID_ARG, "rl_group_advantages_by_owner: NULL array argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int32_t* status = reinterpret_cast<int32_t*>(ws);
  cudaError_t e = cudaMemsetAsync(n_tok_out, 0, static_cast<size_t>(n_traj) * sizeof(int32_t), s);
  if (e != cudaSuccess) return cuda_error(e, "rl_group_advantages_by_owner: cudaMemsetAsync");
  if (n_tokens > 0) {
    int64_t blocks = (n_tokens + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    owner_count_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(n_tokens, token_traj, mask, n_traj, n_tok_out,
                                                                     status);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "rl_group_advantages_by_owner: owner_count_kernel launch");
  }
  group_adv_kernel<<<1, kAdvThreads, 0, s>>>(n_traj, n_groups, group_offsets, rewards, traj_valid, n_tok_out,
                                             static_cast<double>(params->adv_eps), params->loss_agg, adv_out,
                                             coef_out, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "rl_group_advantages_by_owner: group_adv_kernel launch");
  return RL_OK;
}
