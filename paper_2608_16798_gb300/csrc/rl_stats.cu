// Fixed-order reductions: the loss sum behind every loss entry point, and batch summaries of
// the per-token statistics that rl_policy_loss_fwd_bwd and
// rl_fused_head_loss_fwd_bwd write: the number of trained tokens, of clipped ones, and the
// sums of entropy, KL and ratio over them (the clip fraction and the mean policy entropy that
// are tracked during training, Sec. 4). Fixed assignment of rows to threads and a fixed
// reduction order in double precision: the sums are the same on every run.
#include <cstdint>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {

// Fixed-order sum of per-row loss contributions into the caller's accumulator (every loss
// entry point ends with it). Thread k adds rows k, k + 1024, ... into eight accumulators in
// turn, so eight independent loads are in flight per thread (one memory latency per 8,192
// rows instead of per 1,024); the accumulators, the warps and the CTA are then combined in a
// fixed order: the sum is the same on every run.
__global__ void __launch_bounds__(1024) reduce_loss_kernel(const double* __restrict__ row_loss, int64_t rows,
                                                           double* loss_accum) {
  __shared__ double part[32];
  double acc[8] = {0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0};
  int64_t r = threadIdx.x;
  for (; r + 7 * 1024 < rows; r += 8 * 1024) {
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[k] += row_loss[r + k * 1024];
  }
  for (int k = 0; r < rows; r += 1024, ++k) acc[k] += row_loss[r];
  double a = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
  a = warp_sum(a);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = a;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < 32; ++w) t += part[w];
    *loss_accum += t;
  }
}

rl_status launch_reduce_loss(const double* row_loss, int64_t rows, double* loss_accum, cudaStream_t s) {
  reduce_loss_kernel<<<1, 1024, 0, s>>>(row_loss, rows, loss_accum);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "reduce_loss_kernel launch");
  return RL_OK;
}

// Batch summary of the per-token statistics: one cluster of kSumCluster CTAs (one launch, no
// workspace). Global thread g of the cluster takes rows g, g + G, g + 2G, ... (G = all its
// threads) in groups of kSumUnroll rows whose loads are issued together (mask and owner, then
// the coefficients, then the statistics: three dependent round trips per group instead of per
// row); each thread adds its rows in order, then the warps, the CTA and the cluster's CTAs are
// combined in a fixed order (the CTA totals meet in rank 0's shared memory): the sums are the
// same on every run.
constexpr int kSumThreads = 1024;
constexpr int kSumCluster = 8;
constexpr int kSumUnroll = 4;

__device__ __forceinline__ void st_cluster_f64(uint32_t addr, double v) {
  asm volatile("st.shared::cluster.f64 [%0], %1;" :: "r"(addr), "d"(v) : "memory");
}

__global__ void __cluster_dims__(kSumCluster, 1, 1) __launch_bounds__(kSumThreads)
    stats_summary_kernel(int64_t rows, const float* __restrict__ st, const uint8_t* __restrict__ mask,
                         const int32_t* __restrict__ token_traj, int32_t n_traj, const float* __restrict__ coef,
                         double* __restrict__ out, int32_t* status) {
  __shared__ double part[kSumThreads / 32][5];
  __shared__ double cta_total[kSumCluster][5];  // used in rank 0
  const uint32_t rank = cluster_ctarank();
  const int64_t G = static_cast<int64_t>(kSumCluster) * kSumThreads;
  double acc[5] = {0.0, 0.0, 0.0, 0.0, 0.0};
  bool bad = false;
  auto add_rows = [&](int64_t r0, int nr) {  // rows r0, r0 + G, ... (nr <= kSumUnroll of them)
    uint32_t m[kSumUnroll];
    int32_t i[kSumUnroll];
#pragma unroll
    for (int k = 0; k < kSumUnroll; ++k) {
      m[k] = k < nr ? mask[r0 + k * G] : 0u;
      i[k] = k < nr ? token_traj[r0 + k * G] : 0;
    }
    float c[kSumUnroll];
#pragma unroll
    for (int k = 0; k < kSumUnroll; ++k) {
      const bool in = i[k] >= 0 && i[k] < n_traj;
      bad |= m[k] != 0 && !in;
      c[k] = (m[k] != 0 && in) ? coef[i[k]] : 0.f;
    }
    float v[kSumUnroll][4];
#pragma unroll
    for (int k = 0; k < kSumUnroll; ++k) {
      const float* s = st + (r0 + k * G) * 5;
#pragma unroll
      for (int q = 0; q < 4; ++q) v[k][q] = c[k] != 0.f ? s[q + 1] : 0.f;
    }
#pragma unroll
    for (int k = 0; k < kSumUnroll; ++k) {
      if (c[k] == 0.f) continue;
      acc[0] += 1.0;
      acc[1] += static_cast<double>(v[k][1]);  // clipped flag
      acc[2] += static_cast<double>(v[k][2]);  // H
      acc[3] += static_cast<double>(v[k][3]);  // KL
      acc[4] += static_cast<double>(v[k][0]);  // rho
    }
  };
  int64_t r = static_cast<int64_t>(rank) * kSumThreads + threadIdx.x;
  for (; r + (kSumUnroll - 1) * G < rows; r += kSumUnroll * G) add_rows(r, kSumUnroll);
  if (r < rows) add_rows(r, static_cast<int>((rows - r + G - 1) / G));
  if (bad) flag_status(status, RL_DEV_BAD_TRAJ);
#pragma unroll
  for (int k = 0; k < 5; ++k) acc[k] = warp_sum(acc[k]);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0)
    for (int k = 0; k < 5; ++k) part[warp][k] = acc[k];
  cluster_sync_all();  // every CTA of the cluster is running before rank 0's memory is written
  if (threadIdx.x < 5) {
    double sum = 0.0;
    for (int w = 0; w < kSumThreads / 32; ++w) sum += part[w][threadIdx.x];
    st_cluster_f64(map_to_rank(smem_addr(&cta_total[rank][threadIdx.x]), 0), sum);
  }
  cluster_sync_all();
  if (rank == 0 && threadIdx.x < 5) {
    double sum = 0.0;
    for (int k = 0; k < kSumCluster; ++k) sum += cta_total[k][threadIdx.x];
    out[threadIdx.x] += sum;
  }
}

}  // namespace rl

extern "C" rl_status rl_token_stats_summary(int64_t rows, const float* token_stats, const uint8_t* mask,
                                            const int32_t* token_traj, int32_t n_traj, const float* coef,
                                            double* summary_accum, void* ws, size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  if (rows < 0 || n_traj < 0) return set_error(RL_ERR_INVALID_ARG, "rl_token_stats_summary: negative size");
  if (!summary_accum || !ws) return set_error(RL_ERR_INVALID_ARG, "rl_token_stats_summary: NULL argument");
  if (ws_bytes < kWsHeader) return set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_token_stats_summary: workspace too small");
  if (rows == 0) return RL_OK;
  if (!token_stats || !mask || !token_traj || (n_traj > 0 && !coef))
    return set_error(RL_ERR_INVALID_ARG, "rl_token_stats_summary: NULL array argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  stats_summary_kernel<<<kSumCluster, kSumThreads, 0, s>>>(rows, token_stats, mask, token_traj, n_traj, coef, summary_accum,
                                                 reinterpret_cast<int32_t*>(ws));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "stats_summary_kernel launch");
  return RL_OK;
}
