// Backward products of the fused LM head on the tensor cores (tcgen05, CTA pairs), both in
// one persistent launch:
//
//   dH  = dZ W      M = tokens, N = D, K = V        A = dZ   (K-major: V contiguous)
//                                                   B = W    (MN-major: D contiguous)
//   dW += dZ^T H    M = V,      N = D, K = tokens   A = dZ^T (MN-major: V contiguous)
//                                                   B = H    (MN-major: D contiguous)
//
// dZ is the bf16 gradient of the logits of a chunk (or group of chunks) of n tokens, formed
// in the workspace by the loss pass; W and H are the caller's bf16 matrices in their own
// row-major layouts, read in place (the MN-major operands use the transpose bits of the
// instruction descriptor: nothing is transposed in memory).
//
// A 2-CTA cluster computes output tiles of 256 rows x 512 columns: per K step of 16 the even
// CTA issues two cta_group::2 MMAs of 256 x 256 that share the A operand, into one fp32
// accumulator of all 512 TMEM columns (each CTA holds 128 rows of A and, for each MMA, 128 of
// B's 256 columns; 4 shared-memory stages of 48 KB filled by TMA; both CTAs' loads complete on
// the even CTA's barrier and the MMA's commits are multicast to both). Sharing A between two
// MMAs moves a quarter fewer operand bytes through shared memory and L2 per flop than 256 x
// 256 tiles, which is what lets the MMAs run close to their peak rate. The epilogue drains
// TMEM 32 columns at a time into a swizzled shared-memory slab and hands it to the TMA: a
// tiled store into d_hidden (bf16 or fp32) or a tiled reduce-add into the fp32 d_weight.
//
// Work items are dH tiles (each the whole contraction over V: long) followed by dW tiles
// (contraction over the n tokens: short), handed out by a counter in global memory as pairs
// become free: the dW tiles fill the time the last dH tiles leave over, and pairs that run at
// the same time work on neighbouring tiles, sharing operand rows and columns in L2. The even
// CTA's producer thread takes each item and publishes it to both CTAs' roles through a small
// ring guarded by mbarriers. Every output element receives exactly one store (dH) or one
// addition (dW) per launch, so results do not depend on the schedule.
#include <cuda.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <utility>

#include "rl_device.cuh"
#include "rl_host.h"
#include "rl_tc.cuh"
#include "rl_tmap.h"

namespace rl {
namespace grad {

constexpr int BM = 128;                          // output rows per CTA (TMEM lanes)
constexpr int NB = 512;                          // output columns per tile (TMEM columns)
constexpr int NH = NB / 256;                     // MMAs per K step (N = 256 each)
constexpr int BK = 64;                           // contraction elements per stage
constexpr uint32_t A_BYTES = BM * BK * 2;        // this CTA's 128 rows of A
constexpr uint32_t HALF_BYTES = 64 * BK * 2;     // one 64-element MN block of 64 K rows
constexpr uint32_t B_BYTES = NH * 2 * HALF_BYTES;  // this CTA's 128 columns of each MMA's B
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int NS = 4;                            // shared-memory stages
constexpr int NR = 4;                            // slots of the work-item ring
constexpr uint32_t SLAB_BYTES = 4096;            // epilogue slab: 32 rows x 128 bytes
constexpr int kThreads = 192;                    // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr size_t kSmem = NS * STAGE_BYTES + 4 * 2 * SLAB_BYTES + 1024;
static_assert(kSmem <= 232448 - 1024, "shared memory of the backward kernel");
// consumers of each published work item: the MMA thread and 4 epilogue warps of the even CTA,
// the producer thread and 4 epilogue warps of the odd CTA
constexpr uint32_t kItemReaders = 10;

struct GradArgs {
  int32_t n_h;           // dH tiles: row tiles x n_nt
  int32_t n_w;           // dW tiles: row tiles x n_nt
  int32_t n_nt;          // 512-column tiles of D
  int32_t nkb_h, nkb_w;  // 64-element K blocks: over V (dH), over the tokens (dW)
  uint32_t* counter;     // work-item counter (zero at launch)
  int32_t* status;
};

// Element type of the stored d_hidden tiles.
enum HOut { H_F32 = 0, H_BF16 = 1 };

template <int HO>
__global__ void __launch_bounds__(kThreads, 1) head_grad_kernel(
    const __grid_constant__ CUtensorMap tmAh, const __grid_constant__ CUtensorMap tmBh,
    const __grid_constant__ CUtensorMap tmOh, const __grid_constant__ CUtensorMap tmAw,
    const __grid_constant__ CUtensorMap tmBw, const __grid_constant__ CUtensorMap tmOw, const GradArgs p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[NS], empty[NS], accf, acce, ifull[NR], iempty[NR];
  __shared__ int32_t ring[NR];
  __shared__ uint32_t tbase;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* slabs = sm + NS * STAGE_BYTES;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int n_items = p.n_h + p.n_w;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&accf, 1);
    mbar_init(&acce, 8);  // 4 epilogue warps in each CTA of the pair
    for (int r = 0; r < NR; ++r) {
      mbar_init(&ifull[r], 1);
      mbar_init(&iempty[r], kItemReaders);
    }
    fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc_pair(&tbase, NB);
  tc::fence_before_sync();
  cluster_sync_all();
  tc::fence_after_sync();
  const uint32_t tmem = tbase;

  // item -> (dW?, tile row, tile column, K blocks); columns fastest
  const int n_h = p.n_h, n_nt = p.n_nt, nkb_h = p.nkb_h, nkb_w = p.nkb_w;
  auto decode = [n_h, n_nt, nkb_h, nkb_w](int item, bool& w, int& mt, int& nt, int& nkb) {
    w = item >= n_h;
    const int r = w ? item - n_h : item;
    mt = r / n_nt;
    nt = r % n_nt;
    nkb = w ? nkb_w : nkb_h;
  };
  // Read the k-th published item (every role but the even CTA's producer): -1 if the wait
  // ran out.
  auto next_item = [&](uint32_t k) -> int {
    const int r = static_cast<int>(k % NR);
    const bool got = rank == 0 ? mbar_wait_bounded(&ifull[r], (k / NR) & 1)
                               : mbar_wait_cluster_bounded(&ifull[r], (k / NR) & 1);
    if (!got) return -1;
    const int item = ring[r];
    if (rank == 0) mbar_arrive(&iempty[r]);
    else mbar_arrive_remote(map_to_rank(smem_addr(&iempty[r]), 0));
    return item;
  };

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (uint32_t k = 0; ok; ++k) {
        int item;
        if (rank == 0) {
          // take the next item and publish it to both CTAs
          const int r = static_cast<int>(k % NR);
          if (k >= NR && !mbar_wait_cluster_bounded(&iempty[r], ((k / NR) - 1) & 1)) {
            flag_status(p.status, RL_DEV_TIMEOUT);
            break;
          }
          const uint32_t v = atomicAdd(p.counter, 1u);
          item = v < static_cast<uint32_t>(n_items) ? static_cast<int>(v) : n_items;
          ring[r] = item;
          const uint32_t peer_slot = map_to_rank(smem_addr(&ring[r]), 1);
          asm volatile("st.shared::cluster.u32 [%0], %1;" :: "r"(peer_slot), "r"(item) : "memory");
          mbar_arrive(&ifull[r]);
          mbar_arrive_remote(map_to_rank(smem_addr(&ifull[r]), 1));
        } else {
          item = next_item(k);
          if (item < 0) {
            flag_status(p.status, RL_DEV_TIMEOUT);
            break;
          }
        }
        if (item >= n_items) break;
        bool w;
        int mt, nt, nkb;
        decode(item, w, mt, nt, nkb);
        const int m0 = mt * 2 * BM + static_cast<int>(rank) * BM;
        const int n0 = nt * NB + static_cast<int>(rank) * 128;
        const CUtensorMap* mb = w ? &tmBw : &tmBh;
        for (int kb = 0; kb < nkb; ++kb, ++g) {
          const int s = g % NS;
          const uint32_t use = g / NS;
          if (use > 0 && !mbar_wait_bounded(&empty[s], (use - 1) & 1)) {
            flag_status(p.status, RL_DEV_TIMEOUT);
            ok = false;
            break;
          }
          uint8_t* st = sm + s * STAGE_BYTES;
          if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * STAGE_BYTES);  // both CTAs' bytes
          const uint32_t bar = map_to_rank(smem_addr(&full[s]), 0);
          if (w) {
            tc::tma_load_2d_pair(st, &tmAw, m0, kb * BK, bar);
            tc::tma_load_2d_pair(st + HALF_BYTES, &tmAw, m0 + 64, kb * BK, bar);
          } else {
            tc::tma_load_2d_pair(st, &tmAh, kb * BK, m0, bar);
          }
#pragma unroll
          for (int h = 0; h < NH; ++h) {
            uint8_t* sb = st + A_BYTES + h * 2 * HALF_BYTES;
            tc::tma_load_2d_pair(sb, mb, n0 + h * 256, kb * BK, bar);
            tc::tma_load_2d_pair(sb + HALF_BYTES, mb, n0 + h * 256 + 64, kb * BK, bar);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc_h = tc::idesc_bf16_f32_major(2 * BM, 256, false, true);
      constexpr uint32_t idesc_w = tc::idesc_bf16_f32_major(2 * BM, 256, true, true);
      uint32_t g = 0;
      for (uint32_t t = 0;; ++t) {
        const int item = next_item(t);
        if (item < 0) {
          flag_status(p.status, RL_DEV_TIMEOUT);
          break;
        }
        if (item >= n_items) break;
        bool w;
        int mt, nt, nkb;
        decode(item, w, mt, nt, nkb);
        if (t > 0 && !mbar_wait_cluster_bounded(&acce, (t - 1) & 1)) {
          flag_status(p.status, RL_DEV_TIMEOUT);
          break;
        }
        tc::fence_after_sync();
        const uint32_t idesc = w ? idesc_w : idesc_h;
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb, ++g) {
          const int s = g % NS;
          if (!mbar_wait_bounded(&full[s], (g / NS) & 1)) {
            flag_status(p.status, RL_DEV_TIMEOUT);
            ok = false;
            break;
          }
          tc::fence_after_sync();
          const uint32_t a = smem_addr(sm + s * STAGE_BYTES), b = a + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = w ? tc::desc_mnmajor_sw128(a + k * 2048, HALF_BYTES, 1024)
                                  : tc::desc_kmajor_sw128(a + k * 32);
#pragma unroll
            for (int h = 0; h < NH; ++h) {
              const uint64_t bd = tc::desc_mnmajor_sw128(b + h * 2 * HALF_BYTES + k * 2048, HALF_BYTES, 1024);
              tc::mma_bf16_pair(tmem + h * 256, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
            }
          }
          tc::mma_commit_pair(&empty[s], 0x3);
        }
        if (!ok) break;
        tc::mma_commit_pair(&accf, 0x3);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (4 warps)
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    uint8_t* my = slabs + (warp - 2) * 2 * SLAB_BYTES;
    const uint32_t tq = tmem + (static_cast<uint32_t>(32 * q) << 16);
    uint32_t buf = 0;
    for (uint32_t t = 0;; ++t) {
      int item = 0;
      if (lane == 0) item = next_item(t);
      item = __shfl_sync(0xffffffffu, item, 0);
      if (item < 0) {
        if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
        break;
      }
      if (item >= n_items) break;
      bool w;
      int mt, nt, nkb;
      decode(item, w, mt, nt, nkb);
      if (!mbar_wait_sleep_bounded(&accf, t & 1)) {
        if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
        break;
      }
      tc::fence_after_sync();
      const int row0 = mt * 2 * BM + static_cast<int>(rank) * BM + 32 * q;
#pragma unroll 1
      for (int c = 0; c < NB / 32; ++c) {
        float v[32];
        tc::tmem_ld32(tq + c * 32, v);
        if (c == NB / 32 - 1) {
          // the whole accumulator is in registers or slabs: hand it back to the MMA
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) {
            if (rank != 0) mbar_arrive_remote(map_to_rank(smem_addr(&acce), 0));
            else mbar_arrive(&acce);
          }
        }
        uint8_t* sb = my + buf * SLAB_BYTES;
        if (lane == 0) tc::bulk_wait_read_1();  // the slab's previous TMA has read it
        __syncwarp();
        if (!w && HO == H_BF16) {
          // 32 rows x 64 bytes, 64-byte swizzle: 16-byte chunk j of row r at chunk j ^ ((r / 2) % 4)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint4 u = make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                                       pack_bf16x2(v[8 * j + 4], v[8 * j + 5]),
                                       pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
            *reinterpret_cast<uint4*>(sb + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) = u;
          }
        } else {
          // 32 rows x 128 bytes, 128-byte swizzle: 16-byte chunk j of row r at chunk j ^ (r % 8)
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(sb + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          const int col = nt * NB + c * 32;
          if (w) tc::tma_reduce_add_2d(&tmOw, col, row0, sb);
          else tc::tma_store_2d(&tmOh, col, row0, sb);
          bulk_commit();
        }
        buf ^= 1;
      }
    }
    if (lane == 0) tc::bulk_wait_all();
  }
  tc::fence_before_sync();
  cluster_sync_all();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc_pair(tmem, NB);
  }
}

}  // namespace grad

rl_status head_grad(const uint16_t* dz, int64_t ldz, int64_t n, int64_t V, const void* weight, const void* hidden,
                    int64_t D, void* d_hidden, rl_dtype dh_dtype, float* d_weight, uint32_t* counter,
                    int32_t* status, cudaStream_t s) {
  using namespace grad;
  CUtensorMap ah, bh, oh, aw, bw, ow;
  const bool bf16 = dh_dtype == RL_BF16;
  rl_status st = tmap_2d(&ah, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dz, V, n, ldz * 2, BK, BM, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&bh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, weight, D, V, D * 2, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = bf16 ? tmap_2d(&oh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, d_hidden, D, n, D * 2, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B)
              : tmap_2d(&oh, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, d_hidden, D, n, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&aw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dz, V, n, ldz * 2, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&bw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, hidden, D, n, D * 2, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&ow, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, d_weight, D, V, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st != RL_OK) return st;
  GradArgs a = {};
  a.n_nt = static_cast<int32_t>((D + NB - 1) / NB);
  a.n_h = static_cast<int32_t>((n + 2 * BM - 1) / (2 * BM)) * a.n_nt;
  a.n_w = static_cast<int32_t>((V + 2 * BM - 1) / (2 * BM)) * a.n_nt;
  a.nkb_h = static_cast<int32_t>((V + BK - 1) / BK);
  a.nkb_w = static_cast<int32_t>((n + BK - 1) / BK);
  a.counter = counter;
  a.status = status;

  cudaError_t e = cudaMemsetAsync(counter, 0, sizeof(uint32_t), s);
  if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync(work counter)");
  auto kern = bf16 ? head_grad_kernel<H_BF16> : head_grad_kernel<H_F32>;
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  static std::mutex mu;
  static std::map<std::pair<int, bool>, int> resident;  // CTA pairs resident at once
  int max_pairs = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    const auto key = std::make_pair(dev, bf16);
    auto it = resident.find(key);
    if (it == resident.end()) {
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kSmem));
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(head_grad_kernel)");
      int npairs = 0;
      cfg.gridDim = dim3(2);
      e = cudaOccupancyMaxActiveClusters(&npairs, kern, &cfg);
      if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveClusters(head_grad_kernel)");
      if (npairs <= 0) return set_error(RL_ERR_UNSUPPORTED, "head_grad_kernel: no CTA pair fits on the device");
      it = resident.emplace(key, npairs).first;
    }
    max_pairs = it->second;
  }
  // persistent: at most as many pairs as fit on the device at once, and no more than items
  cfg.gridDim = dim3(2 * std::max(1, std::min(a.n_h + a.n_w, max_pairs)));
  e = cudaLaunchKernelEx(&cfg, kern, ah, bh, oh, aw, bw, ow, a);
  if (e != cudaSuccess) return cuda_error(e, "cudaLaunchKernelEx(head_grad_kernel)");
  return RL_OK;
}

}  // namespace rl
