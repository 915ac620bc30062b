// Group-relative advantages and loss coefficients over ragged trajectories.
//
//   count_adv_kernel    one launch, two kinds of CTA: the first count L_i, the
//                       trainable tokens of each trajectory (one warp per
//                       trajectory span, writing token_traj[t] = i; or, by owner,
//                       a grid-stride pass over tokens in any order), the 1 /
//                       sum_t M_{i,t} normaliser of the masked GRPO objective
//                       (Sec. 2.3.2); the others form A_i = (R_i - mu_g) /
//                       (sigma_g + eps) per group (one warp per group: mean and
//                       population standard deviation of the valid members'
//                       rewards in double precision; Sec. 2.3.2 GRPO advantage,
//                       Sec. 3.2.3; discarded rollouts leave the statistics and
//                       get A = 0, Sec. 3.4). Counts and advantages do not depend
//                       on each other.
//   coef_kernel         N = #{valid i : L_i > 0} and S = sum of their L_i (every
//                       CTA forms both, integer sums, so any order gives the same
//                       values), then c_i for its share of the trajectories, and
//                       A = 0 for trajectories outside every group.
//
// Every kind of work is spread over the GPU: a batch of many small groups (4,096
// groups of 4) costs no more than a few large ones. Both kernels are
// latency-bound: they touch ~T + 30 n bytes, well under 0.1% of the logits
// stream of one microbatch.
#include <cstdint>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {

constexpr int kAdvThreads = 256;
constexpr int kAdvWarps = kAdvThreads / 32;

// L_i over trajectory i's span [traj_offsets[i], traj_offsets[i + 1]) and the owner of each of
// its tokens (one warp)
__device__ __forceinline__ void count_span(int64_t i, int lane, int64_t n_tokens, const int64_t* traj_offsets,
                                           const uint8_t* mask, int32_t* n_tok_out, int32_t* token_traj_out,
                                           int32_t* status) {
  const int64_t s = traj_offsets[i], e = traj_offsets[i + 1];
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
// Warp w of `warps` takes the 32-token runs w, w + warps, ... (n_tok_out zeroed before).
__device__ __forceinline__ void count_owners(int64_t w, int64_t warps, int lane, int64_t n_tokens,
                                             const int32_t* token_traj, const uint8_t* mask, int32_t n_traj,
                                             int32_t* n_tok_out, int32_t* status) {
  for (int64_t base = w * 32; base < n_tokens; base += warps * 32) {
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

// A_i for the members of group g (one warp): mean and population standard deviation of the
// valid members' rewards in double precision, each A_i rounded once to float. Invalid members,
// and every member of a group with no valid member or whose valid rewards are all equal, get 0.
__device__ __forceinline__ void group_advantage(int64_t g, int lane, int32_t n_traj, const int32_t* group_offsets,
                                                const float* rewards, const uint8_t* traj_valid, double adv_eps,
                                                float* adv_out, int32_t* status) {
  const int b = group_offsets[g], e = group_offsets[g + 1];
  if (b < 0 || e < b || e > n_traj) {
    if (lane == 0) flag_status(status, RL_DEV_BAD_OFFSETS);
    return;
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
  if (k == 0 || lo == hi) {  // nothing valid, or all valid rewards equal: A = 0
    for (int i = b + lane; i < e; i += 32) adv_out[i] = 0.f;
    return;
  }
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
    const bool valid = !traj_valid || traj_valid[i] != 0;
    adv_out[i] = valid ? static_cast<float>((static_cast<double>(rewards[i]) - mu) / denom) : 0.f;
  }
}

struct CountAdvArgs {
  int32_t n_traj, n_groups;
  int64_t n_tokens;
  int64_t count_blocks;            // CTAs [0, count_blocks) count, the rest form advantages
  const int64_t* traj_offsets;     // spans (rl_group_advantages)
  const int32_t* token_traj;       // owners (rl_group_advantages_by_owner)
  const uint8_t* mask;
  const int32_t* group_offsets;
  const float* rewards;
  const uint8_t* traj_valid;
  double adv_eps;
  float* adv_out;
  float* coef_out;
  int32_t* n_tok_out;
  int32_t* token_traj_out;
  int32_t* status;
};

template <bool BY_OWNER>
__global__ void __launch_bounds__(kAdvThreads) count_adv_kernel(const CountAdvArgs a) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (blockIdx.x < a.count_blocks) {
    const int64_t w = static_cast<int64_t>(blockIdx.x) * kAdvWarps + warp;
    if (BY_OWNER) {
      count_owners(w, a.count_blocks * kAdvWarps, lane, a.n_tokens, a.token_traj, a.mask, a.n_traj, a.n_tok_out,
                   a.status);
    } else if (w < a.n_traj) {
      count_span(w, lane, a.n_tokens, a.traj_offsets, a.mask, a.n_tok_out, a.token_traj_out, a.status);
    }
  } else {
    const int64_t g = (static_cast<int64_t>(blockIdx.x) - a.count_blocks) * kAdvWarps + warp;
    if (g < a.n_groups)
      group_advantage(g, lane, a.n_traj, a.group_offsets, a.rewards, a.traj_valid, a.adv_eps, a.adv_out, a.status);
  }
}

// Coefficients c_i (Sec. 2.3.2: 1 / (N L_i) under seq-mean-token-mean; 1 / S under token-mean;
// 1 under token-sum) for valid trajectories with L_i > 0, else 0; A = 0 for trajectories
// before the first group or after the last.
__global__ void __launch_bounds__(kAdvThreads) coef_kernel(int32_t n_traj, int32_t n_groups,
                                                           const int32_t* __restrict__ group_offsets,
                                                           const uint8_t* __restrict__ traj_valid,
                                                           const int32_t* __restrict__ n_tok, int32_t loss_agg,
                                                           float* __restrict__ adv_out, float* __restrict__ coef_out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ long long red_n[kAdvWarps], red_s[kAdvWarps];
  long long cnt = 0, tok = 0;
#pragma unroll 4
  for (int i = tid; i < n_traj; i += kAdvThreads) {
    const int32_t L = n_tok[i];
    const bool counted = (!traj_valid || traj_valid[i] != 0) && L > 0;
    cnt += counted;
    tok += counted ? L : 0;
  }
  cnt = warp_sum(cnt);
  tok = warp_sum(tok);
  if (lane == 0) {
    red_n[warp] = cnt;
    red_s[warp] = tok;
  }
  __syncthreads();
  long long N = 0, S = 0;
  for (int w = 0; w < kAdvWarps; ++w) {
    N += red_n[w];
    S += red_s[w];
  }
  int32_t first = n_traj, last = n_traj;  // trajectories [first, last) belong to groups
  if (n_groups > 0) {
    first = min(max(group_offsets[0], 0), n_traj);
    last = min(max(group_offsets[n_groups], first), n_traj);
  }
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kAdvThreads + tid; i < n_traj;
       i += static_cast<int64_t>(gridDim.x) * kAdvThreads) {
    if (i < first || i >= last) adv_out[i] = 0.f;
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

// Launches count_adv_kernel (count_blocks counting CTAs, then one warp per group) and
// coef_kernel on stream s.
template <bool BY_OWNER>
static rl_status launch_advantages(CountAdvArgs a, int64_t count_blocks, const rl_loss_params* params, const char* fn,
                                   cudaStream_t s) {
  a.count_blocks = count_blocks;
  const int64_t adv_blocks = (static_cast<int64_t>(a.n_groups) + kAdvWarps - 1) / kAdvWarps;
  const int64_t blocks = count_blocks + adv_blocks;
  if (blocks > 0) {
    count_adv_kernel<BY_OWNER><<<static_cast<unsigned>(blocks), kAdvThreads, 0, s>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, (std::string(fn) + ": count_adv_kernel launch").c_str());
  }
  // every CTA reads all n_tok once for N and S: a few CTAs per wave of the GPU at most
  int64_t cb = (static_cast<int64_t>(a.n_traj) + kAdvThreads - 1) / kAdvThreads;
  if (cb > 152) cb = 152;
  coef_kernel<<<static_cast<unsigned>(cb), kAdvThreads, 0, s>>>(a.n_traj, a.n_groups, a.group_offsets, a.traj_valid,
                                                                 a.n_tok_out, params->loss_agg, a.adv_out, a.coef_out);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, (std::string(fn) + ": coef_kernel launch").c_str());
  return RL_OK;
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
  CountAdvArgs a = {};
  a.n_traj = n_traj;
  a.n_groups = n_groups;
  a.n_tokens = n_tokens;
  a.traj_offsets = traj_offsets;
  a.mask = mask;
  a.group_offsets = group_offsets;
  a.rewards = rewards;
  a.traj_valid = traj_valid;
  a.adv_eps = static_cast<double>(params->adv_eps);
  a.adv_out = adv_out;
  a.coef_out = coef_out;
  a.n_tok_out = n_tok_out;
  a.token_traj_out = token_traj_out;
  a.status = reinterpret_cast<int32_t*>(ws);
  const int64_t count_blocks = (static_cast<int64_t>(n_traj) + kAdvWarps - 1) / kAdvWarps;  // a warp per span
  return launch_advantages<false>(a, count_blocks, params, "rl_group_advantages",
                                  reinterpret_cast<cudaStream_t>(stream));
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
  cudaError_t e = cudaMemsetAsync(n_tok_out, 0, static_cast<size_t>(n_traj) * sizeof(int32_t), s);
  if (e != cudaSuccess) return cuda_error(e, "rl_group_advantages_by_owner: cudaMemsetAsync");
  CountAdvArgs a = {};
  a.n_traj = n_traj;
  a.n_groups = n_groups;
  a.n_tokens = n_tokens;
  a.token_traj = token_traj;
  a.mask = mask;
  a.group_offsets = group_offsets;
  a.rewards = rewards;
  a.traj_valid = traj_valid;
  a.adv_eps = static_cast<double>(params->adv_eps);
  a.adv_out = adv_out;
  a.coef_out = coef_out;
  a.n_tok_out = n_tok_out;
  a.status = reinterpret_cast<int32_t*>(ws);
  // grid-stride over 32-token runs: at most 8 CTAs per SM
  int64_t count_blocks = (n_tokens + kAdvThreads - 1) / kAdvThreads;
  if (count_blocks > 152 * 8) count_blocks = 152 * 8;
  return launch_advantages<true>(a, count_blocks, params, "rl_group_advantages_by_owner", s);
}
