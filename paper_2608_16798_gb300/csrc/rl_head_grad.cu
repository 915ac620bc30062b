// Backward products of the fused LM head on the tensor cores (tcgen05, CTA pairs):
//
//   dH  = dZ W      M = tokens, N = D, K = V        A = dZ   (K-major: V contiguous)
//                                                   B = W    (MN-major: D contiguous)
//   dW += dZ^T H    M = V,      N = D, K = tokens   A = dZ^T (MN-major: V contiguous)
//                                                   B = H    (MN-major: D contiguous)
//
// dZ is the bf16 gradient of the logits for a chunk (or group of chunks) of tokens, formed
// in the workspace by the loss pass; W and H are the caller's bf16 matrices in their own
// row-major layouts. Both products run in one persistent kernel template: a 2-CTA cluster
// computes 256 x 256 output tiles with cta_group::2 MMAs issued by the even CTA (each CTA
// holds 128 rows of A and 128 of B's 256 columns per stage; both CTAs' TMA loads complete on
// the even CTA's barrier; the MMA's commits are multicast to both CTAs), accumulating in two
// TMEM buffers of 256 fp32 columns so that the epilogue of one tile overlaps the MMAs of the
// next. The epilogue drains TMEM 32 columns at a time into a swizzled shared-memory slab and
// hands it to the TMA: a tiled store (dH in bf16 or fp32) or a tiled reduce-add (fp32 dW, and
// dH when the contraction over V is split in two: both halves add onto zeros, so the sum is
// independent of their order). Each dW element receives exactly one addition per launch, so
// dW accumulates deterministically across launches.
//
// The operands use the MN-major shared-memory layout of the tensor cores directly (the
// descriptor's transpose bits), so neither W nor H nor dZ is ever transposed in memory.
#include <cuda.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <tuple>

#include "rl_device.cuh"
#include "rl_host.h"
#include "rl_tc.cuh"
#include "rl_tmap.h"

namespace rl {
namespace grad {

constexpr int BM = 128;                            // output rows per CTA (TMEM lanes)
constexpr int BN = 256;                            // output columns per tile (TMEM columns)
constexpr int BK = 64;                             // contraction elements per stage
constexpr uint32_t A_BYTES = BM * BK * 2;          // this CTA's 128 rows of A
constexpr uint32_t B_BYTES = (BN / 2) * BK * 2;    // this CTA's 128 of B's 256 columns
constexpr uint32_t HALF_BYTES = 64 * BK * 2;       // one 64-element MN block of 64 K rows
constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
#ifndef RL_GRAD_NS
#define RL_GRAD_NS 6
#endif
constexpr int NS = RL_GRAD_NS;
constexpr uint32_t SLAB_BYTES = 4096;              // epilogue slab: 32 rows x 128 bytes
constexpr int kThreads = 192;                      // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr size_t kSmem = NS * STAGE_BYTES + 4 * 2 * SLAB_BYTES + 1024;
static_assert(kSmem <= 232448 - 512, "shared memory of the backward kernel");

struct GradArgs {
  int32_t n_mt, n_nt;   // 256-row and 256-column output tiles
  int32_t nkb;          // 64-element K blocks of the whole contraction
  int32_t kbps;         // K blocks per split (the contraction is cut into ksplit parts)
  int32_t ksplit;
  int32_t* status;
};

// Output of the epilogue.
enum Out { RED_F32 = 0, ST_F32 = 1, ST_BF16 = 2 };

template <bool A_MN, int OUT>
__global__ void __launch_bounds__(kThreads, 1) head_grad_kernel(const __grid_constant__ CUtensorMap tmA,
                                                                const __grid_constant__ CUtensorMap tmB,
                                                                const __grid_constant__ CUtensorMap tmO,
                                                                const GradArgs p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[NS], empty[NS], accf[2], acce[2];
  __shared__ uint32_t tbase;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* slabs = sm + NS * STAGE_BYTES;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int unit = static_cast<int>(blockIdx.x >> 1);
  const int n_units = static_cast<int>(gridDim.x >> 1);
  const int tiles = p.n_mt * p.n_nt;
  const int n_items = tiles * p.ksplit;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&accf[a], 1);
      mbar_init(&acce[a], 8);  // 4 epilogue warps in each CTA of the pair
    }
    fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc_pair(&tbase, 2 * BN);
  tc::fence_before_sync();
  cluster_sync_all();
  tc::fence_after_sync();
  const uint32_t tmem = tbase;

  // work item -> (output tile row, column, K range); column fastest, so that the pairs that
  // run at the same time share their A rows and B columns in L2
  const int n_nt = p.n_nt, kbps = p.kbps, nkb = p.nkb;
  auto decode = [tiles, n_nt, kbps, nkb](int item, int& mt, int& nt, int& kb0, int& kb1) {
    const int sp = item / tiles, rem = item % tiles;
    mt = rem / n_nt;
    nt = rem % n_nt;
    kb0 = sp * kbps;
    kb1 = min(kb0 + kbps, nkb);
  };

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (int item = unit; item < n_items && ok; item += n_units) {
        int mt, nt, kb0, kb1;
        decode(item, mt, nt, kb0, kb1);
        const int m0 = mt * 2 * BM + static_cast<int>(rank) * BM;
        const int n0 = nt * BN + static_cast<int>(rank) * (BN / 2);
        for (int kb = kb0; kb < kb1; ++kb, ++g) {
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
          if constexpr (A_MN) {
            tc::tma_load_2d_pair(st, &tmA, m0, kb * BK, bar);
            tc::tma_load_2d_pair(st + HALF_BYTES, &tmA, m0 + 64, kb * BK, bar);
          } else {
            tc::tma_load_2d_pair(st, &tmA, kb * BK, m0, bar);
          }
          tc::tma_load_2d_pair(st + A_BYTES, &tmB, n0, kb * BK, bar);
          tc::tma_load_2d_pair(st + A_BYTES + HALF_BYTES, &tmB, n0 + 64, kb * BK, bar);
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32_major(2 * BM, BN, A_MN, true);
      uint32_t g = 0, t = 0;
      bool ok = true;
      for (int item = unit; item < n_items && ok; item += n_units, ++t) {
        int mt, nt, kb0, kb1;
        decode(item, mt, nt, kb0, kb1);
        const int acc = t & 1;
        if (t >= 2 && !mbar_wait_cluster_bounded(&acce[acc], ((t >> 1) - 1) & 1)) {
          flag_status(p.status, RL_DEV_TIMEOUT);
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t d = tmem + acc * BN;
        for (int kb = kb0; kb < kb1; ++kb, ++g) {
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
            const uint64_t ad = A_MN ? tc::desc_mnmajor_sw128(a + k * 2048, HALF_BYTES, 1024)
                                     : tc::desc_kmajor_sw128(a + k * 32);
            const uint64_t bd = tc::desc_mnmajor_sw128(b + k * 2048, HALF_BYTES, 1024);
            tc::mma_bf16_pair(d, ad, bd, idesc, (kb != kb0 || k != 0) ? 1u : 0u);
          }
          tc::mma_commit_pair(&empty[s], 0x3);
        }
        if (ok) tc::mma_commit_pair(&accf[acc], 0x3);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (4 warps)
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    uint8_t* my = slabs + (warp - 2) * 2 * SLAB_BYTES;
    uint32_t t = 0, buf = 0;
    bool ok = true;
    for (int item = unit; item < n_items && ok; item += n_units, ++t) {
      int mt, nt, kb0, kb1;
      decode(item, mt, nt, kb0, kb1);
      const int acc = t & 1;
      if (!mbar_wait_bounded(&accf[acc], (t >> 1) & 1)) {
        if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
        ok = false;
        break;
      }
      tc::fence_after_sync();
      const int row0 = mt * 2 * BM + static_cast<int>(rank) * BM + 32 * q;
      const uint32_t tacc = tmem + (static_cast<uint32_t>(32 * q) << 16) + acc * BN;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        tc::tmem_ld32(tacc + c * 32, v);
        if (c == BN / 32 - 1) {
          // the whole accumulator is in registers or slabs: hand it back to the MMA
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) {
            if (rank != 0) mbar_arrive_remote(map_to_rank(smem_addr(&acce[acc]), 0));
            else mbar_arrive(&acce[acc]);
          }
        }
        uint8_t* sb = my + buf * SLAB_BYTES;
        if (lane == 0) tc::bulk_wait_read_1();  // the slab's previous TMA has read it
        __syncwarp();
        if constexpr (OUT == ST_BF16) {
          // 32 rows x 64 bytes, 64-byte swizzle: 16-byte chunk j of row r at chunk j ^ ((r / 2) % 4)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint4 w = make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                                       pack_bf16x2(v[8 * j + 4], v[8 * j + 5]),
                                       pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
            *reinterpret_cast<uint4*>(sb + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) = w;
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
          const int col = nt * BN + c * 32;
          if constexpr (OUT == RED_F32) tc::tma_reduce_add_2d(&tmO, col, row0, sb);
          else tc::tma_store_2d(&tmO, col, row0, sb);
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
    tc::tmem_dealloc_pair(tmem, 2 * BN);
  }
}

template <bool A_MN, int OUT>
static rl_status launch(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mo, const GradArgs& a,
                        cudaStream_t s) {
  auto kern = head_grad_kernel<A_MN, OUT>;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
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
  static std::map<std::tuple<int, bool, int>, int> resident;  // CTA pairs resident at once
  int max_pairs = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    const auto key = std::make_tuple(dev, A_MN, OUT);
    auto it = resident.find(key);
    if (it == resident.end()) {
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kSmem));
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(head_grad_kernel)");
      int n = 0;
      cfg.gridDim = dim3(2);
      e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
      if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveClusters(head_grad_kernel)");
      if (n <= 0) return set_error(RL_ERR_UNSUPPORTED, "head_grad_kernel: no CTA pair fits on the device");
      it = resident.emplace(key, n).first;
    }
    max_pairs = it->second;
  }
  const int items = a.n_mt * a.n_nt * a.ksplit;
  cfg.gridDim = dim3(2 * std::max(1, std::min(items, max_pairs)));
  e = cudaLaunchKernelEx(&cfg, kern, ma, mb, mo, a);
  if (e != cudaSuccess) return cuda_error(e, "cudaLaunchKernelEx(head_grad_kernel)");
  return RL_OK;
}

static int resident_pairs() {
  // the same for every instance (one CTA per SM: shared memory)
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
  return std::max(1, sms / 2);
}

}  // namespace grad

int head_grad_dh_split(int64_t n, int64_t V, int64_t D) {
  using namespace grad;
  const int64_t tiles = ((n + 2 * BM - 1) / (2 * BM)) * ((D + BN - 1) / BN);
  const int64_t nkb = (V + BK - 1) / BK;
  if (nkb < 2) return 1;
  const int64_t P = resident_pairs();
  // fraction of the pairs' time spent on work: items / (waves x pairs)
  auto eff = [&](int64_t items) { return static_cast<double>(items) / (((items + P - 1) / P) * P); };
  return eff(2 * tiles) > eff(tiles) + 0.02 ? 2 : 1;
}

rl_status head_grad_dh(const uint16_t* dz, int64_t ldz, int64_t n, int64_t V, const void* weight, int64_t D,
                       void* out, int out_kind, int ksplit, int32_t* status, cudaStream_t s) {
  using namespace grad;
  CUtensorMap ma, mb, mo;
  rl_status st = tmap_2d(&ma, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dz, V, n, ldz * 2, BK, BM, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&mb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, weight, D, V, D * 2, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK) {
    if (out_kind == ST_BF16)
      st = tmap_2d(&mo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, out, D, n, D * 2, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
    else
      st = tmap_2d(&mo, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, D, n, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
  }
  if (st != RL_OK) return st;
  GradArgs a = {};
  a.n_mt = static_cast<int32_t>((n + 2 * BM - 1) / (2 * BM));
  a.n_nt = static_cast<int32_t>((D + BN - 1) / BN);
  a.nkb = static_cast<int32_t>((V + BK - 1) / BK);
  a.ksplit = ksplit;
  a.kbps = (a.nkb + ksplit - 1) / ksplit;
  a.status = status;
  switch (out_kind) {
    case RED_F32: return launch<false, RED_F32>(ma, mb, mo, a, s);
    case ST_F32: return launch<false, ST_F32>(ma, mb, mo, a, s);
    default: return launch<false, ST_BF16>(ma, mb, mo, a, s);
  }
}

rl_status head_grad_dw(const uint16_t* dz, int64_t ldz, int64_t n, int64_t V, const void* hidden, int64_t D,
                       float* d_weight, int32_t* status, cudaStream_t s) {
  using namespace grad;
  CUtensorMap ma, mb, mo;
  rl_status st = tmap_2d(&ma, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dz, V, n, ldz * 2, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&mb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, hidden, D, n, D * 2, 64, BK, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st == RL_OK)
    st = tmap_2d(&mo, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, d_weight, D, V, D * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
  if (st != RL_OK) return st;
  GradArgs a = {};
  a.n_mt = static_cast<int32_t>((V + 2 * BM - 1) / (2 * BM));
  a.n_nt = static_cast<int32_t>((D + BN - 1) / BN);
  a.nkb = static_cast<int32_t>((n + BK - 1) / BK);
  a.ksplit = 1;
  a.kbps = a.nkb;
  a.status = status;
  return launch<true, RED_F32>(ma, mb, mo, a, s);
}

}  // namespace rl
