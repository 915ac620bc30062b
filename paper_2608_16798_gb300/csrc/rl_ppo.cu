// PPO parts of the method (Sec. 2.3.1, Sec. 2.3.4): the masked generalised advantage
// estimate over packed ragged trajectories and the masked value loss.
//
//   gae_kernel         one CTA per trajectory (grid-stride). The estimate is the backward
//                      affine recurrence x_t = a_t x_{t+1} + b_t inside the trajectory
//                      (x past its end = 0), evaluated chunk by chunk from the end: each
//                      thread composes its 4 tokens' maps, a block-wide suffix scan of the
//                      composed maps gives every thread its entry value, and the chunk's
//                      first value carries into the next chunk down.
//                        printed reading  a_t = gamma lambda,
//                                         b_t = M_t (r_t + gamma M_{t+1} V_{t+1} - V_t)
//                        skip reading     a_t = M_t ? gamma lambda : 1,
//                                         b_t = M_t (r_t + gamma Vn_{t+1} - V_t), with
//                                         Vn_{t+1} the value of the next trainable token,
//                                         itself the suffix scan of the selection map
//                                         x_t = M_t ? V_t : x_{t+1} (exact in fp32)
//   value_loss_kernel  per token: c M (V - G)^2, added per CTA in a fixed order into one
//                      partial per CTA, and dV = 2 c M (V - G); the last CTA to finish adds
//                      the partials, in a fixed order, into the caller's accumulator.
//   rollout_adv_kernel A_t = R_i - V_t, G_t = R_i per token for tokens in any order (the
//                      gamma = lambda = 1 form of Sec. 2.3.4, which also holds on the shared
//                      prefixes of a rollout's prefix tree).
//
// Both touch a few bytes per token (mask, values, rewards, outputs) and are latency- or
// launch-bound next to the logits stream.
#include <cstdint>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {
namespace ppo {

constexpr int kThreads = 256;
constexpr int kPer = 4;                  // consecutive tokens per thread
constexpr int kChunk = kThreads * kPer;  // tokens per block step
constexpr int kWarps = kThreads / 32;

// x -> a x + b
struct Affine {
  float a, b;
};

// outer(inner(x)): inner is applied first (it covers the later positions).
__device__ __forceinline__ Affine compose(Affine outer, Affine inner) {
  return Affine{outer.a * inner.a, fmaf(outer.a, inner.b, outer.b)};
}

// Every thread passes the composition of its own tokens' maps (`mine`, mapping the value
// just above its tokens to the value at its first token) and the value above the whole
// chunk (`top`, the same in every thread). Returns the value just above this thread's
// tokens. `sh` holds kWarps maps.
__device__ __forceinline__ float suffix_entry(Affine mine, float top, Affine* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // inclusive suffix within the warp: S_k = F_k o F_{k+1} o ... o F_31
  Affine s = mine;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float oa = __shfl_down_sync(0xffffffffu, s.a, off);
    const float ob = __shfl_down_sync(0xffffffffu, s.b, off);
    if (lane + off < 32) s = compose(s, Affine{oa, ob});
  }
  if (lane == 0) sh[warp] = s;
  __syncthreads();
  // value above this warp: the later warps' totals applied to `top`, highest first
  float above_warp = top;
  for (int w = kWarps - 1; w > warp; --w) above_warp = fmaf(sh[w].a, above_warp, sh[w].b);
  __syncthreads();  // sh is reused by the caller's next scan
  // exclusive suffix within the warp: S_{k+1} applied to the warp's entry value
  const float na = __shfl_down_sync(0xffffffffu, s.a, 1);
  const float nb = __shfl_down_sync(0xffffffffu, s.b, 1);
  return lane == 31 ? above_warp : fmaf(na, above_warp, nb);
}

struct GaeArgs {
  int32_t n_traj;
  const int64_t* offs;
  int64_t T;
  const uint8_t* mask;
  const float* values;
  const float* token_rewards;  // [T] or null
  const float* traj_rewards;   // [n_traj] or null: R_i at the last trainable token
  float gamma, lam;
  int32_t skip;
  float* adv;
  float* ret;  // or null
  int32_t* status;
};

__global__ void __launch_bounds__(kThreads) gae_kernel(const GaeArgs p) {
  __shared__ Affine sh[kWarps];
  __shared__ int64_t sh_pos[kWarps];
  __shared__ float sh_carry[2];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float gl = p.gamma * p.lam;
  for (int32_t i = blockIdx.x; i < p.n_traj; i += gridDim.x) {
    const int64_t s = p.offs[i], e = p.offs[i + 1];
    if (s < 0 || e < s || e > p.T) {
      if (tid == 0) flag_status(p.status, RL_DEV_BAD_OFFSETS);
      continue;  // uniform across the block
    }
    // last trainable token (for R_i), searched chunk by chunk from the end
    int64_t last = -1;
    if (p.traj_rewards) {
      for (int64_t c1 = e; c1 > s && last < 0; c1 -= kChunk) {
        const int64_t c0 = c1 - kChunk > s ? c1 - kChunk : s;
        int64_t best = -1;
        for (int j = 0; j < kPer; ++j) {
          const int64_t t = c0 + tid * kPer + j;
          if (t < c1 && p.mask[t] != 0) best = t;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const int64_t o = __shfl_down_sync(0xffffffffu, best, off);
          best = o > best ? o : best;
        }
        if (lane == 0) sh_pos[warp] = best;
        __syncthreads();
        for (int w = 0; w < kWarps; ++w) last = sh_pos[w] > last ? sh_pos[w] : last;
        __syncthreads();
      }
    }
    const float Ri = (p.traj_rewards && last >= 0) ? p.traj_rewards[i] : 0.f;

    float carry_x = 0.f;   // recurrence value at the first position above the chunk
    float carry_vn = 0.f;  // skip reading: value of the first trainable token above it
    for (int64_t c1 = e; c1 > s; c1 -= kChunk) {
      const int64_t c0 = c1 - kChunk > s ? c1 - kChunk : s;
      const int64_t t0 = c0 + static_cast<int64_t>(tid) * kPer;
      bool M[kPer];
      float V[kPer], r[kPer], a[kPer], b[kPer];
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        const int64_t t = t0 + j;
        const bool in = t < c1;
        M[j] = in && p.mask[t] != 0;
        V[j] = in ? p.values[t] : 0.f;
        r[j] = (in && p.token_rewards) ? p.token_rewards[t] : 0.f;
        if (t == last) r[j] += Ri;
      }
      if (p.skip) {
        // Vn above each token: suffix scan of the selection maps
        Affine f{1.f, 0.f};
#pragma unroll
        for (int j = kPer - 1; j >= 0; --j) f = compose(M[j] ? Affine{0.f, V[j]} : Affine{1.f, 0.f}, f);
        float vn = suffix_entry(f, carry_vn, sh);
#pragma unroll
        for (int j = kPer - 1; j >= 0; --j) {
          a[j] = M[j] ? gl : 1.f;
          b[j] = M[j] ? (r[j] + fmaf(p.gamma, vn, -V[j])) : 0.f;
          if (M[j]) vn = V[j];
        }
        if (tid == 0) sh_carry[1] = vn;  // the chunk's lowest token's selection value
      } else {
#pragma unroll
        for (int j = 0; j < kPer; ++j) {
          const int64_t t = t0 + j;
          float boot = 0.f;
          if (t + 1 < e && p.mask[t + 1] != 0) boot = p.values[t + 1];
          a[j] = gl;
          b[j] = M[j] ? (r[j] + fmaf(p.gamma, boot, -V[j])) : 0.f;
          if (t >= c1) { a[j] = 1.f; b[j] = 0.f; }  // past the chunk: identity
        }
      }
      Affine f{1.f, 0.f};
#pragma unroll
      for (int j = kPer - 1; j >= 0; --j) f = compose(Affine{a[j], b[j]}, f);
      float x = suffix_entry(f, carry_x, sh);
#pragma unroll
      for (int j = kPer - 1; j >= 0; --j) {
        x = fmaf(a[j], x, b[j]);
        const int64_t t = t0 + j;
        if (t < c1) {
          p.adv[t] = M[j] ? x : 0.f;
          if (p.ret) p.ret[t] = M[j] ? x + V[j] : 0.f;
        }
      }
      if (tid == 0) sh_carry[0] = x;
      __syncthreads();
      carry_x = sh_carry[0];
      if (p.skip) carry_vn = sh_carry[1];
      __syncthreads();
    }
  }
}

struct ValueArgs {
  int64_t rows;
  const float* values;
  const float* returns;
  const uint8_t* mask;
  const int32_t* token_traj;
  int32_t n_traj;
  const float* coef;
  float* d_values;
  double* row_loss;
  double* loss_accum;
  uint32_t* done;  // finished-CTA count in the workspace header
  int32_t* status;
};

// Each CTA adds its rows' terms in a fixed order (thread-strided, then warp and CTA) and leaves
// one partial per CTA in row_loss[blockIdx.x]; the last CTA to finish (a counter in the
// workspace header, which it resets) adds the partials in a fixed order into loss_accum.
__global__ void __launch_bounds__(256) value_loss_kernel(const ValueArgs p) {
  __shared__ double part[8];
  __shared__ uint32_t last;
  double acc = 0.0;
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < p.rows;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float c = 0.f;
    if (p.mask[t] != 0) {
      const int32_t i = p.token_traj[t];
      if (i < 0 || i >= p.n_traj) flag_status(p.status, RL_DEV_BAD_TRAJ);
      else c = p.coef[i];
    }
    const float d = p.values[t] - p.returns[t];
    const float cd = c * d;
    p.d_values[t] = c != 0.f ? 2.f * cd : 0.f;
    if (c != 0.f) acc += static_cast<double>(cd) * static_cast<double>(d);
  }
  acc = warp_sum(acc);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < 8; ++w) t += part[w];
    p.row_loss[blockIdx.x] = t;
    __threadfence();
    last = atomicAdd(p.done, 1u) == gridDim.x - 1 ? 1u : 0u;
    if (last) __threadfence();
  }
  __syncthreads();
  if (last) {  // uniform across the CTA
    double t = 0.0;
    for (uint32_t k = threadIdx.x; k < gridDim.x; k += blockDim.x) t += __ldcg(p.row_loss + k);
    t = warp_sum(t);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = t;
    __syncthreads();
    if (threadIdx.x == 0) {
      double u = 0.0;
      for (int w = 0; w < 8; ++w) u += part[w];
      *p.loss_accum += u;
      *p.done = 0u;
    }
  }
}

// A_t = R_{i(t)} - V_t and G_t = R_{i(t)} on trainable tokens, 0 elsewhere (any token order).
__global__ void __launch_bounds__(256) rollout_adv_kernel(int64_t T, const int32_t* __restrict__ token_traj,
                                                          const uint8_t* __restrict__ mask,
                                                          const float* __restrict__ values,
                                                          const float* __restrict__ rewards, int32_t n_traj,
                                                          float* __restrict__ adv, float* __restrict__ ret,
                                                          int32_t* status) {
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < T;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float a = 0.f, g = 0.f;
    if (mask[t] != 0) {
      const int32_t i = token_traj[t];
      if (i < 0 || i >= n_traj) {
        flag_status(status, RL_DEV_BAD_TRAJ);
      } else {
        g = rewards[i];
        a = g - values[t];
      }
    }
    adv[t] = a;
    if (ret) ret[t] = g;
  }
}

static int grid_for(int64_t work, int per_block, int cap) {
  int64_t g = (work + per_block - 1) / per_block;
  if (g < 1) g = 1;
  return static_cast<int>(g < cap ? g : cap);
}

}  // namespace ppo
}  // namespace rl

extern "C" rl_status rl_masked_gae(int32_t n_traj, const int64_t* traj_offsets, int64_t n_tokens, const uint8_t* mask,
                                   const float* values, const float* token_rewards, const float* traj_rewards,
                                   float gamma, float gae_lambda, int32_t skip_masked, float* adv_out,
                                   float* returns_out, void* ws, size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (n_traj < 0 || n_tokens < 0) return set_error(RL_ERR_INVALID_ARG, "rl_masked_gae: negative size");
  if (!(gamma >= 0.f && gamma <= 1.f) || !(gae_lambda >= 0.f && gae_lambda <= 1.f))
    return set_error(RL_ERR_INVALID_ARG, "rl_masked_gae: gamma and lambda must lie in [0, 1]");
  if (skip_masked != 0 && skip_masked != 1)
    return set_error(RL_ERR_INVALID_ARG, "rl_masked_gae: skip_masked must be 0 or 1");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, "rl_masked_gae: NULL workspace");
  if (ws_bytes < kWsHeader) return set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_masked_gae: workspace too small");
  if (n_traj == 0) return RL_OK;
  if (!traj_offsets || (n_tokens > 0 && (!mask || !values || !adv_out)))
    return set_error(RL_ERR_INVALID_ARG, "rl_masked_gae: NULL array argument");
  ppo::GaeArgs a = {};
  a.n_traj = n_traj;
  a.offs = traj_offsets;
  a.T = n_tokens;
  a.mask = mask;
  a.values = values;
  a.token_rewards = token_rewards;
  a.traj_rewards = traj_rewards;
  a.gamma = gamma;
  a.lam = gae_lambda;
  a.skip = skip_masked;
  a.adv = adv_out;
  a.ret = returns_out;
  a.status = reinterpret_cast<int32_t*>(ws);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  ppo::gae_kernel<<<ppo::grid_for(n_traj, 1, 152 * 8), ppo::kThreads, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "gae_kernel launch");
  return RL_OK;
}

extern "C" rl_status rl_value_loss_fwd_bwd(int64_t rows, const float* values, const float* returns,
                                           const uint8_t* mask, const int32_t* token_traj, int32_t n_traj,
                                           const float* coef, float* d_values, double* loss_accum, void* ws,
                                           size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (rows < 0 || n_traj < 0) return set_error(RL_ERR_INVALID_ARG, "rl_value_loss_fwd_bwd: negative size");
  if (!ws || !loss_accum) return set_error(RL_ERR_INVALID_ARG, "rl_value_loss_fwd_bwd: NULL argument");
  if (ws_bytes < kWsHeader + static_cast<size_t>(rows) * sizeof(double))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL,
                     "rl_value_loss_fwd_bwd: workspace smaller than rl_workspace_size(rows, 0, 0)");
  if (rows == 0) return RL_OK;
  if (!values || !returns || !mask || !token_traj || !d_values || (n_traj > 0 && !coef))
    return set_error(RL_ERR_INVALID_ARG, "rl_value_loss_fwd_bwd: NULL array argument");
  ppo::ValueArgs a = {};
  a.rows = rows;
  a.values = values;
  a.returns = returns;
  a.mask = mask;
  a.token_traj = token_traj;
  a.n_traj = n_traj;
  a.coef = coef;
  a.d_values = d_values;
  double* row_loss = reinterpret_cast<double*>(static_cast<char*>(ws) + ws_row_loss_offset());
  a.row_loss = row_loss;
  a.loss_accum = loss_accum;
  a.done = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + kWsValueDoneOffset);
  a.status = reinterpret_cast<int32_t*>(ws);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int blocks = ppo::grid_for(rows, 256, 152 * 16);  // <= rows: one partial per CTA fits
  ppo::value_loss_kernel<<<blocks, 256, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "value_loss_kernel launch");
  return RL_OK;  // the kernel's last CTA has added the loss into loss_accum
}

extern "C" rl_status rl_rollout_value_advantages(int64_t n_tokens, const int32_t* token_traj, const uint8_t* mask,
                                                 const float* values, const float* rewards, int32_t n_traj,
                                                 float* adv_out, float* returns_out, void* ws, size_t ws_bytes,
                                                 rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (n_tokens < 0 || n_traj < 0) return set_error(RL_ERR_INVALID_ARG, "rl_rollout_value_advantages: negative size");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, "rl_rollout_value_advantages: NULL workspace");
  if (ws_bytes < kWsHeader)
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_rollout_value_advantages: workspace too small");
  if (n_tokens == 0) return RL_OK;
  if (!token_traj || !mask || !values || !adv_out || (n_traj > 0 && !rewards))
    return set_error(RL_ERR_INVALID_ARG, "rl_rollout_value_advantages: NULL array argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  ppo::rollout_adv_kernel<<<ppo::grid_for(n_tokens, 256, 152 * 8), 256, 0, s>>>(
      n_tokens, token_traj, mask, values, rewards, n_traj, adv_out, returns_out, reinterpret_cast<int32_t*>(ws));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "rollout_adv_kernel launch");
  return RL_OK;
}
