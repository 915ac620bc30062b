// Fused LM head: the policy loss and its gradients with respect to the hidden states
// and the output projection, with the logits Z = H W^T never written to memory.
//
// For each chunk of tokens:
//   1. head_kernel<STATS_P> tcgen05 GEMM tiles Z[256 x 256] = H W^T on CTA pairs (2-CTA
//      clusters, cta_group::2 MMAs; TMA-fed shared-memory stages, fp32 accumulators in TMEM,
//      two accumulators so the epilogue of one tile overlaps the MMAs of the next; each CTA
//      holds 128 of the tile's tokens). The epilogue reads each tile twice from TMEM: first
//      its row maximum m_j, then e = exp(z - m_j), which it stores (bf16) in the chunk's
//      dZ buffer, with m_j per token and tile, and folds into per-row online-softmax
//      partials: two per vocabulary block (its even and its odd tiles).
//   2. head_merge_kernel    one thread per token: merges the partials into lse, entropy and
//      logp, evaluates the objective's per-token terms (same readings as the logits path),
//      writes the row's loss contribution and the coefficients of dZ.
//   3. head_dz_kernel       rescales the stored e in place into
//      dZ = c [g (delta_a - p) + alpha p (log p + H)], p = e exp(m_j - lse) (HBM-bound: the
//      logits are formed once, not twice).
// The dZ of one chunk (4,096 tokens x V in bf16) is the only logits-sized buffer; a caller
// that passes more workspace lets a group of several chunks keep their dZ side by side.
// After the group's last chunk (every chunk, with the smallest workspace):
//   4. dH = dZ W and dW += dZ^T H over the group in one persistent launch of
//      head_grad_kernel (rl_head_grad.cu): CTA-pair tcgen05 MMAs on 256 x 512 tiles with the
//      operands in their row-major layouts (dZ K-major for dH, MN-major for dW; W and H
//      MN-major), dH tiles first and dW tiles after them, handed out by a work counter; dH is
//      stored, dW added in fp32 by TMA reduce-add, once per group.
// The forward-only call runs head_wide_kernel<STATS> (256 x 512 tiles, no stores; the same two
// partials per block) and head_logp_merge_kernel.
// The objective (Sec. 2.3.2, Sec. 3.2.4) is the same as for rl_policy_loss_fwd_bwd; here
// pi_theta's logits come from the hidden states times the vocabulary projection.
#include <cuda.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <string>

#include "rl_device.cuh"
#include "rl_host.h"
#include "rl_tc.cuh"
#include "rl_tmap.h"

namespace rl {
namespace head {

constexpr int BM = 128;            // tokens per tile (TMEM lanes)
constexpr int BN = 256;            // vocabulary entries per tile (TMEM columns per accumulator)
constexpr int BK = 64;             // hidden elements per stage (one 128-byte swizzle row)
constexpr int NS = 4;              // shared-memory stages
#ifndef RL_HEAD_VB_TILES
#define RL_HEAD_VB_TILES 16
#endif
constexpr int VB_TILES = RL_HEAD_VB_TILES;  // N tiles per work item (16: a vocabulary block of 4,096)
constexpr uint32_t A_BYTES = BM * BK * 2, B_BYTES = BN * BK * 2, STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int kThreads = 192;      // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr size_t kSmem = NS * STAGE_BYTES + 1024;
// CTA-pair form: each CTA stages its 128 tokens and half of the 256 vocabulary rows
#ifndef RL_HEAD_NS2
#define RL_HEAD_NS2 6
#endif
constexpr int NS2 = RL_HEAD_NS2;
constexpr uint32_t STAGE2_BYTES = A_BYTES + B_BYTES / 2;
constexpr size_t kSmem2 = NS2 * STAGE2_BYTES + 1024;
#ifndef RL_HEAD_PAIR
#define RL_HEAD_PAIR 1
#endif
constexpr bool kPair = RL_HEAD_PAIR != 0;
constexpr uint32_t kWBoxRows = kPair ? BN / 2 : BN;  // rows of W per TMA box
#ifndef RL_HEAD_CHUNK
#define RL_HEAD_CHUNK 4096
#endif
constexpr int64_t kChunk = RL_HEAD_CHUNK;  // tokens per chunk (tuning knob, compile time)
constexpr int64_t kParts = 2;               // partials per token and vocabulary block (even, odd tiles)

enum Mode { STATS = 0, STATS_P = 1 };

// Per-token coefficients of dZ (from head_merge_kernel).
struct RowCoef {
  float nlse2;  // -lse * log2(e)
  float Kp;     // dZ_v = Kp p_v (+ cg at v = a), without the entropy term
  float cg;
  float ca;     // entropy: dZ_v = p_v (ca z_v + Ke) (+ cg at v = a)
  float Ke;
  int32_t a;
  int32_t active;
  float pad;
};

struct HeadArgs {
  int64_t t0;  // first token of the chunk
  int32_t Tc, D, V, n_mt, n_vb, n_nt;
  int32_t ent;
  const int32_t* token_ids;
  float4* partials;        // [2 n_vb][Tc] (m, s, u, z_a): a block's even tiles, then its odd tiles
  uint16_t* dz;            // [Tc x ldz] bf16: e = exp(z - m_j) (STATS_P)
  int64_t ldz;
  float* tmax;             // [Tc x n_nt]: m_j per token and tile (STATS_P)
  int32_t* status;
};

// Two forms share this kernel. PAIR = false: each CTA computes 128 x 256 tiles with
// cta_group::1 MMAs from 48 KB stages (A 16 KB + B 32 KB, 4 stages). PAIR = true: a cluster of
// two CTAs computes 256 x 256 tiles with cta_group::2 MMAs issued by the even CTA; each CTA
// loads its own 128 tokens of H and its own 128 vocabulary rows of W (32 KB stages, 6 of them),
// both CTAs' loads complete on the even CTA's barrier, the MMA's commits are multicast to both
// CTAs, and each CTA's epilogue drains its own 128 TMEM lanes (all 256 columns) and tells the
// even CTA's MMA thread when an accumulator is free. Per pair this halves the W operand each SM
// fetches and stages per MMA.
template <int MODE, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1) head_kernel(const __grid_constant__ CUtensorMap tmH,
                                                           const __grid_constant__ CUtensorMap tmW,
                                                           const HeadArgs p) {
  constexpr int kNS = PAIR ? NS2 : NS;
  constexpr uint32_t kStage = PAIR ? STAGE2_BYTES : STAGE_BYTES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[kNS], empty[kNS], accf[2], acce[2];
  __shared__ uint32_t tbase;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  const int unit = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int n_units = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  constexpr int kMStep = PAIR ? 2 * BM : BM;  // tokens per work item
  const int n_m = (p.Tc + kMStep - 1) / kMStep;
  const int n_items = n_m * p.n_vb;
  const int nkb = p.D / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kNS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&accf[a], 1);
      mbar_init(&acce[a], PAIR ? 8 : 4);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (PAIR) tc::tmem_alloc_pair(&tbase, 2 * BN);
    else tc::tmem_alloc(&tbase, 2 * BN);
  }
  tc::fence_before_sync();
  if constexpr (PAIR) cluster_sync_all();
  else __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (int item = unit; item < n_items && ok; item += n_units) {
        const int vb = item / n_m, m0 = (item % n_m) * kMStep + static_cast<int>(rank) * BM;
        const int nt1 = min((vb + 1) * VB_TILES, p.n_nt);
        for (int nt = vb * VB_TILES; nt < nt1 && ok; ++nt) {
          for (int kb = 0; kb < nkb; ++kb, ++g) {
            const int s = g % kNS;
            const uint32_t use = g / kNS;
            if (use > 0 && !mbar_wait_bounded(&empty[s], (use - 1) & 1)) {
              flag_status(p.status, RL_DEV_TIMEOUT);
              ok = false;
              break;
            }
            uint8_t* st = sm + s * kStage;
            if constexpr (PAIR) {
              if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * kStage);  // both CTAs' bytes
              const uint32_t bar = map_to_rank(smem_addr(&full[s]), 0);
              tc::tma_load_2d_pair(st, &tmH, kb * BK, m0, bar);
              tc::tma_load_2d_pair(st + A_BYTES, &tmW, kb * BK, nt * BN + static_cast<int>(rank) * (BN / 2), bar);
            } else {
              mbar_arrive_expect_tx(&full[s], kStage);
              tc::tma_load_2d(st, &tmH, kb * BK, m0, &full[s]);
              tc::tma_load_2d(st + A_BYTES, &tmW, kb * BK, nt * BN, &full[s]);
            }
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32(kMStep, BN);
      uint32_t g = 0, t = 0;
      bool ok = true;
      for (int item = unit; item < n_items && ok; item += n_units) {
        const int vb = item / n_m;
        const int nt1 = min((vb + 1) * VB_TILES, p.n_nt);
        for (int nt = vb * VB_TILES; nt < nt1 && ok; ++nt, ++t) {
          const int acc = t & 1;
          if (t >= 2) {
            const uint32_t par = ((t >> 1) - 1) & 1;
            const bool got = PAIR ? mbar_wait_cluster_bounded(&acce[acc], par) : mbar_wait_bounded(&acce[acc], par);
            if (!got) {
              flag_status(p.status, RL_DEV_TIMEOUT);
              ok = false;
              break;
            }
          }
          tc::fence_after_sync();
          const uint32_t d = tmem + acc * BN;
          for (int kb = 0; kb < nkb; ++kb, ++g) {
            const int s = g % kNS;
            if (!mbar_wait_bounded(&full[s], (g / kNS) & 1)) {
              flag_status(p.status, RL_DEV_TIMEOUT);
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint32_t a = smem_addr(sm + s * kStage), b = a + A_BYTES;
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              if constexpr (PAIR)
                tc::mma_bf16_pair(d, tc::desc_kmajor_sw128(a + k * 32), tc::desc_kmajor_sw128(b + k * 32), idesc,
                                  (kb | k) != 0);
              else
                tc::mma_bf16(d, tc::desc_kmajor_sw128(a + k * 32), tc::desc_kmajor_sw128(b + k * 32), idesc,
                             (kb | k) != 0);
            }
            if constexpr (PAIR) tc::mma_commit_pair(&empty[s], 0x3);
            else tc::mma_commit(&empty[s]);
          }
          if (ok) {
            if constexpr (PAIR) tc::mma_commit_pair(&accf[acc], 0x3);
            else tc::mma_commit(&accf[acc]);
          }
        }
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (4 warps)
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int rl = 32 * q + lane;
    const float kNegInf = -__int_as_float(0x7f800000);
    uint32_t t = 0;
    bool ok = true;
    for (int item = unit; item < n_items && ok; item += n_units) {
      const int vb = item / n_m, m0 = (item % n_m) * kMStep + static_cast<int>(rank) * BM;
      const int r = m0 + rl;  // token within the chunk
      const bool row_ok = r < p.Tc;
      const int nt1 = min((vb + 1) * VB_TILES, p.n_nt);
      // running partials of the block's even and odd tiles (the halves of its 256 x 512 tiles)
      SoftmaxPartial ps0{kNegInf, 0.f, 0.f}, ps1{kNegInf, 0.f, 0.f};
      float za = 0.f;
      const int32_t a = row_ok ? p.token_ids[p.t0 + r] : -1;
      for (int nt = vb * VB_TILES; nt < nt1; ++nt, ++t) {
        const int acc = t & 1;
        if (!mbar_wait_bounded(&accf[acc], (t >> 1) & 1)) {
          if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const int n0 = nt * BN;
        const uint32_t tbase_acc = tmem + (static_cast<uint32_t>(32 * q) << 16) + acc * BN;
        // sweep 1: the tile's row maximum and the sampled id's logit
        float tm = kNegInf;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int col0 = n0 + c;
          const int nvalid = min(32, p.V - col0);
          if (nvalid <= 0) break;  // past the vocabulary (uniform across the warp)
          float v[32];
          tc::tmem_ld32(tbase_acc + c, v);
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (j < nvalid) tm = fmaxf(tm, v[j]);
          const int ja = a - col0;
          if (ja >= 0 && ja < 32) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j == ja) za = v[j];
          }
        }
        // sweep 2: e = exp(z - m_j), its sums, and (STATS_P) e stored in bf16
        const float nm = -tm * kLog2e;
        float s0 = 0.f, s1 = 0.f, u0 = 0.f;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int col0 = n0 + c;
          const int nvalid = min(32, p.V - col0);
          if (nvalid <= 0) break;
          float v[32];
          tc::tmem_ld32(tbase_acc + c, v);
          uint32_t w[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float e2[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const bool in = j + h < nvalid;
              const float z = in ? v[j + h] : tm;
              const float e = in ? ex2(fmaf(z, kLog2e, nm)) : 0.f;
              if (h) s1 += e; else s0 += e;
              if (p.ent) u0 = fmaf(e, z - tm, u0);
              e2[h] = e;
            }
            w[j / 2] = pack_bf16x2(e2[0], e2[1]);
          }
          if (MODE == STATS_P && row_ok) {
            uint16_t* out = p.dz + static_cast<int64_t>(r) * p.ldz + col0;
            if (nvalid == 32) {
#pragma unroll
              for (int j = 0; j < 4; ++j)
                *reinterpret_cast<uint4*>(out + 8 * j) = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (j < nvalid) out[j] = static_cast<uint16_t>((w[j / 2] >> (16 * (j & 1))) & 0xFFFFu);
            }
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) {
          if (PAIR && rank != 0) mbar_arrive_remote(map_to_rank(smem_addr(&acce[acc]), 0));
          else mbar_arrive(&acce[acc]);
        }
        if (MODE == STATS_P && row_ok) p.tmax[static_cast<int64_t>(r) * p.n_nt + nt] = tm;
        const SoftmaxPartial tile{tm, s0 + s1, u0};
        if (nt & 1) ps1 = merge(ps1, tile);
        else ps0 = merge(ps0, tile);
      }
      if (ok && row_ok) {
        p.partials[static_cast<int64_t>(2 * vb) * p.Tc + r] = make_float4(ps0.m, ps0.s, ps0.u, za);
        p.partials[static_cast<int64_t>(2 * vb + 1) * p.Tc + r] = make_float4(ps1.m, ps1.s, ps1.u, 0.f);
      }
    }
  }
  tc::fence_before_sync();
  if constexpr (PAIR) cluster_sync_all();
  else __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    if constexpr (PAIR) tc::tmem_dealloc_pair(tmem, 2 * BN);
    else tc::tmem_dealloc(tmem, 2 * BN);
  }
}

// ------------------------------------------------------------------ 256 x 512 tiles
//
// Wide form of the pair kernel: a CTA pair computes 256 tokens x 512 vocabulary entries per
// tile with two cta_group::2 MMAs per K step that share the H operand, into one accumulator of
// all 512 TMEM columns (4 stages of 48 KB: this CTA's 128 tokens of H and, per MMA, its 128
// of the 256 W rows). The epilogue treats the tile as two 256-column halves with the same two
// sweeps as the 256 x 256 form (so the tile maxima keep their 256-column granularity), one
// group of four warps per half, each with its own partial (the block's even or odd tiles, as
// in the 256 x 256 form, so both forms give the same bits). It cannot overlap the next
// tile's MMAs: the single accumulator is handed back after both halves; the second group
// halves the time that takes.
constexpr uint32_t W_HALF = (BN / 2) * BK * 2;          // 16 KB
constexpr uint32_t STAGEW_BYTES = A_BYTES + 2 * W_HALF;  // 48 KB
constexpr int NSW = 4;
constexpr size_t kSmemW = NSW * STAGEW_BYTES + 1024;

// One 256-column half of a tile's epilogue: the row maximum of the valid columns and the
// sampled id's logit (za), then e = exp(z - m), its sums and (STATS_P) e in bf16 at `out`.
template <int MODE>
__device__ __forceinline__ SoftmaxPartial epi_half(uint32_t tacc, int n0, int V, int32_t a, int ent, uint16_t* out,
                                                   float& za, float& tm_out) {
  const float kNegInf = -__int_as_float(0x7f800000);
  float tm = kNegInf;
#pragma unroll 1
  for (int c = 0; c < BN; c += 32) {
    const int col0 = n0 + c;
    const int nvalid = min(32, V - col0);
    if (nvalid <= 0) break;  // past the vocabulary (uniform across the warp)
    float v[32];
    tc::tmem_ld32(tacc + c, v);
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < nvalid) tm = fmaxf(tm, v[j]);
    const int ja = a - col0;
    if (ja >= 0 && ja < 32) {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j == ja) za = v[j];
    }
  }
  const float nm = -tm * kLog2e;
  float s0 = 0.f, s1 = 0.f, u0 = 0.f;
#pragma unroll 1
  for (int c = 0; c < BN; c += 32) {
    const int col0 = n0 + c;
    const int nvalid = min(32, V - col0);
    if (nvalid <= 0) break;
    float v[32];
    tc::tmem_ld32(tacc + c, v);
    uint32_t w[16];
#pragma unroll
    for (int j = 0; j < 32; j += 2) {
      float e2[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const bool in = j + h < nvalid;
        const float z = in ? v[j + h] : tm;
        const float e = in ? ex2(fmaf(z, kLog2e, nm)) : 0.f;
        if (h) s1 += e; else s0 += e;
        if (ent) u0 = fmaf(e, z - tm, u0);
        e2[h] = e;
      }
      w[j / 2] = pack_bf16x2(e2[0], e2[1]);
    }
    if (MODE == STATS_P && out) {
      uint16_t* o = out + c;
      if (nvalid == 32) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          *reinterpret_cast<uint4*>(o + 8 * j) = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (j < nvalid) o[j] = static_cast<uint16_t>((w[j / 2] >> (16 * (j & 1))) & 0xFFFFu);
      }
    }
  }
  tm_out = tm;
  return SoftmaxPartial{tm, s0 + s1, u0};
}

// warp 0 TMA, warp 1 MMA, warps 2-9 epilogue: warps 2-5 read the tile's first 256 columns and
// warps 6-9 its second 256, each group with its own running partial (two per vocabulary block)
constexpr int kThreadsW = 320;

template <int MODE>
__global__ void __launch_bounds__(kThreadsW, 1) head_wide_kernel(const __grid_constant__ CUtensorMap tmH,
                                                                const __grid_constant__ CUtensorMap tmW,
                                                                const HeadArgs p) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[NSW], empty[NSW], accf, acce;
  __shared__ uint32_t tbase;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int unit = static_cast<int>(blockIdx.x >> 1);
  const int n_units = static_cast<int>(gridDim.x >> 1);
  constexpr int VB2 = VB_TILES / 2;  // 512-column tiles per vocabulary block
  const int n_m = (p.Tc + 2 * BM - 1) / (2 * BM);
  const int n_nt2 = (p.n_nt + 1) / 2;
  const int n_items = n_m * p.n_vb;
  const int nkb = p.D / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NSW; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&accf, 1);
    mbar_init(&acce, 16);  // 8 epilogue warps in each CTA of the pair
    fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc_pair(&tbase, 2 * BN);
  tc::fence_before_sync();
  cluster_sync_all();
  tc::fence_after_sync();
  const uint32_t tmem = tbase;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (int item = unit; item < n_items && ok; item += n_units) {
        const int vb = item / n_m, m0 = (item % n_m) * 2 * BM + static_cast<int>(rank) * BM;
        const int nt1 = min((vb + 1) * VB2, n_nt2);
        for (int nt = vb * VB2; nt < nt1 && ok; ++nt) {
          for (int kb = 0; kb < nkb; ++kb, ++g) {
            const int s = g % NSW;
            const uint32_t use = g / NSW;
            if (use > 0 && !mbar_wait_bounded(&empty[s], (use - 1) & 1)) {
              flag_status(p.status, RL_DEV_TIMEOUT);
              ok = false;
              break;
            }
            uint8_t* st = sm + s * STAGEW_BYTES;
            if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * STAGEW_BYTES);  // both CTAs' bytes
            const uint32_t bar = map_to_rank(smem_addr(&full[s]), 0);
            tc::tma_load_2d_pair(st, &tmH, kb * BK, m0, bar);
#pragma unroll
            for (int h = 0; h < 2; ++h)
              tc::tma_load_2d_pair(st + A_BYTES + h * W_HALF, &tmW, kb * BK,
                                   nt * 2 * BN + h * BN + static_cast<int>(rank) * (BN / 2), bar);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32(2 * BM, BN);
      uint32_t g = 0, t = 0;
      bool ok = true;
      for (int item = unit; item < n_items && ok; item += n_units) {
        const int vb = item / n_m;
        const int nt1 = min((vb + 1) * VB2, n_nt2);
        for (int nt = vb * VB2; nt < nt1 && ok; ++nt, ++t) {
          if (t > 0 && !mbar_wait_cluster_bounded(&acce, (t - 1) & 1)) {
            flag_status(p.status, RL_DEV_TIMEOUT);
            ok = false;
            break;
          }
          tc::fence_after_sync();
          for (int kb = 0; kb < nkb; ++kb, ++g) {
            const int s = g % NSW;
            if (!mbar_wait_bounded(&full[s], (g / NSW) & 1)) {
              flag_status(p.status, RL_DEV_TIMEOUT);
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint32_t a = smem_addr(sm + s * STAGEW_BYTES), b = a + A_BYTES;
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              const uint64_t ad = tc::desc_kmajor_sw128(a + k * 32);
#pragma unroll
              for (int h = 0; h < 2; ++h)
                tc::mma_bf16_pair(tmem + h * BN, ad, tc::desc_kmajor_sw128(b + h * W_HALF + k * 32), idesc,
                                  (kb | k) != 0);
            }
            tc::mma_commit_pair(&empty[s], 0x3);
          }
          if (ok) tc::mma_commit_pair(&accf, 0x3);
        }
      }
    }
  } else {
    const int q = warp & 3;            // TMEM lane quarter this warp may access
    const int h = (warp - 2) >> 2;     // the 256-column half of each tile this warp reads
    const int rl = 32 * q + lane;
    const float kNegInf = -__int_as_float(0x7f800000);
    const uint32_t tq = tmem + (static_cast<uint32_t>(32 * q) << 16);
    uint32_t t = 0;
    bool ok = true;
    for (int item = unit; item < n_items && ok; item += n_units) {
      const int vb = item / n_m, m0 = (item % n_m) * 2 * BM + static_cast<int>(rank) * BM;
      const int r = m0 + rl;
      const bool row_ok = r < p.Tc;
      const int nt1 = min((vb + 1) * VB2, n_nt2);
      SoftmaxPartial ps{kNegInf, 0.f, 0.f};
      float za = 0.f;
      const int32_t a = row_ok ? p.token_ids[p.t0 + r] : -1;
      uint16_t* dz_row = (MODE == STATS_P && row_ok) ? p.dz + static_cast<int64_t>(r) * p.ldz : nullptr;
      for (int nt = vb * VB2; nt < nt1; ++nt, ++t) {
        if (!mbar_wait_sleep_bounded(&accf, t & 1)) {
          if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const int j = nt * 2 + h;  // 256-column tile
        if (j < p.n_nt) {
          float tm;
          const SoftmaxPartial half =
              epi_half<MODE>(tq + h * BN, j * BN, p.V, a, p.ent, dz_row ? dz_row + j * BN : nullptr, za, tm);
          if (MODE == STATS_P && row_ok) p.tmax[static_cast<int64_t>(r) * p.n_nt + j] = tm;
          ps = merge(ps, half);
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) {
          if (rank != 0) mbar_arrive_remote(map_to_rank(smem_addr(&acce), 0));
          else mbar_arrive(&acce);
        }
      }
      if (ok && row_ok)
        p.partials[static_cast<int64_t>(2 * vb + h) * p.Tc + r] = make_float4(ps.m, ps.s, ps.u, za);
    }
  }
  tc::fence_before_sync();
  cluster_sync_all();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc_pair(tmem, 2 * BN);
  }
}

struct MergeArgs {
  int64_t t0;
  int32_t Tc, V, n_part, n_traj;  // n_part partials per token (two per vocabulary block)
  const float4* partials;
  const int32_t* token_ids;
  const uint8_t* mask;
  const int32_t* token_traj;
  const float* adv;
  const float* coef;
  const float* old_logp;
  const float* ref_logp;
  const float* rollout_logp;
  float clip_lo, clip_hi, beta, alpha, tis_cap;
  int32_t adv_per_row;  // adv holds one A_t per token (else one per trajectory)
  RowCoef* rc;
  double* row_loss;
  float* token_stats;
  int32_t* status;
};

// Token r's partials merged in index order (the same order in both merge kernels, so that the
// forward-only call and the loss call agree bit for bit); the loads run 8 ahead of the merges.
__device__ __forceinline__ void merge_partials(const float4* partials, int64_t Tc, int r, int n_part,
                                               SoftmaxPartial& q, float& za) {
  constexpr int kAhead = 8;
  for (int b0 = 0; b0 < n_part; b0 += kAhead) {
    float4 w[kAhead];
#pragma unroll
    for (int k = 0; k < kAhead; ++k)
      if (b0 + k < n_part) w[k] = partials[static_cast<int64_t>(b0 + k) * Tc + r];
#pragma unroll
    for (int k = 0; k < kAhead; ++k)
      if (b0 + k < n_part) {
        q = merge(q, SoftmaxPartial{w[k].x, w[k].y, w[k].z});
        za += w[k].w;  // nonzero in the one partial whose columns hold the sampled id
      }
  }
}

// threads per CTA of the merge kernels: small CTAs spread a chunk's tokens over many SMs
constexpr int kMergeThreads = 64;

// One thread per token of the chunk: merge the vocabulary blocks' partials (fixed order)
// and evaluate the per-token objective terms.
__global__ void __launch_bounds__(kMergeThreads) head_merge_kernel(const MergeArgs p) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= p.Tc) return;
  const int64_t t = p.t0 + r;
  RowCoef rc = {};
  rc.a = -1;
  bool active = p.mask[t] != 0;
  int32_t i = 0;
  if (active) {
    i = p.token_traj[t];
    if (i < 0 || i >= p.n_traj) {
      flag_status(p.status, RL_DEV_BAD_TRAJ);
      active = false;
    } else if (p.coef[i] == 0.f) {
      active = false;
    }
  }
  const int32_t a = p.token_ids[t];
  if (active && (a < 0 || a >= p.V)) {
    flag_status(p.status, RL_DEV_BAD_TOKEN);
    active = false;
  }
  if (!active) {
    p.rc[r] = rc;
    p.row_loss[t] = 0.0;
    if (p.token_stats)
      for (int k = 0; k < 5; ++k) p.token_stats[t * 5 + k] = 0.f;
    return;
  }
  SoftmaxPartial q{-__int_as_float(0x7f800000), 0.f, 0.f};
  float za = 0.f;
  merge_partials(p.partials, p.Tc, r, p.n_part, q, za);
  const float lnS = logf(q.s);
  const float lse = q.m + lnS;
  const float H = lnS - q.u / q.s;
  const float A = p.adv_per_row ? p.adv[t] : p.adv[i], c = p.coef[i], old = p.old_logp[t];
  const float logp = za - lse;
  const float rho = expf((za - old) - lse);
  const float crho = fminf(fmaxf(rho, p.clip_lo), p.clip_hi);
  const float surr = fminf(rho * A, crho * A);
  const bool cut = (A > 0.f && rho > p.clip_hi) || (A < 0.f && rho < p.clip_lo);
  const float w = (p.tis_cap > 0.f && p.rollout_logp) ? fminf(expf(old - p.rollout_logp[t]), p.tis_cap) : 1.f;
  float kl = 0.f, dkl = 0.f;
  if (p.beta != 0.f && p.ref_logp) {
    const float d = (p.ref_logp[t] - za) + lse;
    const float ed = expf(d);
    kl = ed - d - 1.f;
    dkl = 1.f - ed;
  }
  const float ell = -w * surr + p.beta * kl - p.alpha * H;
  const float g = (cut ? 0.f : -w * A * rho) + p.beta * dkl;
  const float cg = c * g, ca = c * p.alpha;
  rc.nlse2 = -lse * kLog2e;
  rc.Kp = -cg;
  rc.cg = cg;
  rc.ca = ca;
  rc.Ke = -cg + ca * (H - lse);
  rc.a = a;
  rc.active = 1;
  p.rc[r] = rc;
  p.row_loss[t] = static_cast<double>(c) * static_cast<double>(ell);
  if (p.token_stats) {
    float* st = p.token_stats + t * 5;
    st[0] = logp; st[1] = rho; st[2] = cut ? 1.f : 0.f; st[3] = H; st[4] = kl;
  }
}

struct DzArgs {
  int32_t Tc, V, n_nt;
  int32_t ent;
  const RowCoef* rc;
  uint16_t* dz;       // in: e = exp(z - m_j) (bf16); out: dZ (bf16)
  int64_t ldz;
  const float* tmax;  // [Tc x n_nt]
};

constexpr int kDzThreads = 256;
constexpr int kMaxTilesSmem = 2048;  // V up to 524,288 keeps the row's tile factors in shared memory

// One CTA per token row of the chunk (grid-stride): p_v = e_v exp(m_j - lse), then
// dZ_v = Kp p_v (+ cg at v = a), or with the entropy bonus p_v (ca z_v + Ke) (+ cg at v = a),
// z_v = m_j + ln e_v. Rows that are not trained on become zeros. 16-byte loads and stores.
__global__ void __launch_bounds__(kDzThreads) head_dz_kernel(const DzArgs p) {
  __shared__ float fac[kMaxTilesSmem], zoff[kMaxTilesSmem];
  for (int r = blockIdx.x; r < p.Tc; r += gridDim.x) {
    const RowCoef rc = p.rc[r];
    uint16_t* row = p.dz + static_cast<int64_t>(r) * p.ldz;
    const int nvec = p.V / 8;
    if (!rc.active) {
      for (int k = threadIdx.x; k < nvec; k += kDzThreads) reinterpret_cast<uint4*>(row)[k] = make_uint4(0, 0, 0, 0);
      for (int v = nvec * 8 + threadIdx.x; v < p.V; v += kDzThreads) row[v] = 0;
      continue;
    }
    // per tile: Kp exp(m_j - lse) (no entropy) or exp(m_j - lse) and m_j (entropy)
    for (int j = threadIdx.x; j < p.n_nt; j += kDzThreads) {
      const float m = p.tmax[static_cast<int64_t>(r) * p.n_nt + j];
      const float f = ex2(fmaf(m, kLog2e, rc.nlse2));
      fac[j] = p.ent ? f : rc.Kp * f;
      zoff[j] = fmaf(rc.ca, m, rc.Ke);  // ca m_j + Ke
    }
    __syncthreads();
    for (int k = threadIdx.x; k < nvec; k += kDzThreads) {
      uint4 w = reinterpret_cast<const uint4*>(row)[k];
      const int j = (k * 8) / BN;
      const float f = fac[j];
      uint32_t* wp = reinterpret_cast<uint32_t*>(&w);
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        float o[2];
#pragma unroll
        for (int b = 0; b < 2; ++b) {
          const float e = b ? bf16_hi(wp[h]) : bf16_lo(wp[h]);
          float x;
          if (p.ent) {
            // p (ca z + Ke) with z = m_j + ln e; e = 0 contributes 0
            x = e > 0.f ? f * e * fmaf(rc.ca, __logf(e), zoff[j]) : 0.f;
          } else {
            x = f * e;
          }
          if (k * 8 + 2 * h + b == rc.a) x += rc.cg;
          o[b] = x;
        }
        wp[h] = pack_bf16x2(o[0], o[1]);
      }
      reinterpret_cast<uint4*>(row)[k] = w;
    }
    for (int v = nvec * 8 + threadIdx.x; v < p.V; v += kDzThreads) {
      const int j = v / BN;
      const float e = bf16_to_f32(row[v]);
      float x = p.ent ? (e > 0.f ? fac[j] * e * fmaf(rc.ca, __logf(e), zoff[j]) : 0.f) : fac[j] * e;
      if (v == rc.a) x += rc.cg;
      row[v] = f32_to_bf16(x);
    }
    __syncthreads();  // fac / zoff are rewritten for the next row
  }
}

struct LogpMergeArgs {
  int64_t t0;
  int32_t Tc, V, n_part;  // n_part partials per token (two per vocabulary block)
  const float4* partials;
  const int32_t* token_ids;
  float* logp_out;
  float* entropy_out;
  float* lse_out;
  int32_t* status;
};

// Forward-only merge: one thread per token of the chunk writes logp, H and lse.
__global__ void __launch_bounds__(kMergeThreads) head_logp_merge_kernel(const LogpMergeArgs p) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= p.Tc) return;
  const int64_t t = p.t0 + r;
  SoftmaxPartial q{-__int_as_float(0x7f800000), 0.f, 0.f};
  float za = 0.f;
  merge_partials(p.partials, p.Tc, r, p.n_part, q, za);
  const float lnS = logf(q.s);
  const float lse = q.m + lnS;
  const int32_t a = p.token_ids[t];
  const bool a_ok = a >= 0 && a < p.V;
  if (!a_ok) flag_status(p.status, RL_DEV_BAD_TOKEN);
  p.logp_out[t] = a_ok ? za - lse : __int_as_float(0x7fc00000);
  if (p.entropy_out) p.entropy_out[t] = lnS - q.u / q.s;
  if (p.lse_out) p.lse_out[t] = lse;
}

// ------------------------------------------------------------------ host side

// bf16 matrix [rows x inner] (row stride inner), tiles of box_rows x 64 with the 128-byte swizzle.
static rl_status make_map(CUtensorMap* m, const void* base, int64_t inner, int64_t rows, uint32_t box_rows) {
  return tmap_2d(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, base, inner, rows, inner * 2, 64, box_rows,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}

struct Layout {
  int64_t Tc, G, n_nt, n_vb, ldz;  // G chunks per group
  size_t off_partials, off_rc, off_tmax, off_dz, total;
};

static size_t al256(size_t x) { return (x + 255) & ~size_t(255); }

// Workspace of the loss call for up to max_rows tokens. Its smallest form (ws_bytes = 0)
// keeps the dZ of one chunk; every further Tc x ldz x 2 bytes the caller passes keep one more
// chunk's dZ, so that the two products run once per group of G chunks.
static Layout layout(int64_t max_rows, int64_t V, size_t ws_bytes = 0, int64_t want_G = 0) {
  Layout L;
  L.Tc = std::max<int64_t>(1, std::min<int64_t>(max_rows, kChunk));
  const int64_t chunks = (std::max<int64_t>(max_rows, 1) + L.Tc - 1) / L.Tc;
  const int64_t n_nt = (V + BN - 1) / BN;
  L.n_nt = n_nt;
  L.n_vb = (n_nt + VB_TILES - 1) / VB_TILES;
  L.ldz = (V + 7) / 8 * 8;
  auto al = al256;
  size_t off = kWsHeader + al(static_cast<size_t>(std::max<int64_t>(max_rows, 0)) * sizeof(double));
  L.off_partials = off;
  off += al(static_cast<size_t>(kParts * L.n_vb * L.Tc) * sizeof(float4));
  L.off_rc = off;
  off += al(static_cast<size_t>(L.Tc) * sizeof(RowCoef));
  L.off_tmax = off;
  off += al(static_cast<size_t>(L.Tc * n_nt) * sizeof(float));
  L.off_dz = off;
  const size_t chunk_dz = static_cast<size_t>(L.Tc * L.ldz) * 2;
  int64_t G = std::max<int64_t>(want_G, 1);
  if (ws_bytes > off + chunk_dz) G = static_cast<int64_t>((ws_bytes - off) / chunk_dz);
  L.G = std::max<int64_t>(1, std::min<int64_t>(G, chunks));
  off += al(static_cast<size_t>(L.G) * chunk_dz);
  L.total = off;
  return L;
}

// Which passes use the 256 x 512 form: bit 0 the forward-only statistics (STATS), bit 1 the
// loss call's statistics pass (STATS_P). Measured at 32,768 x 4,096 x 151,936 (back to back,
// same box): the forward-only call 24.24-24.36 ms wide (one epilogue group; 23.54-23.65 ms with
// two) against 24.81 ms with 256 x 256 tiles; the loss call 70.9-71.9 ms with wide statistics
// tiles (two epilogue groups) against 69.7-70.1 ms with 256 x 256 ones: its heavier epilogue,
// which stores the exponentials, is hidden behind the MMAs only with two accumulators.
#ifndef RL_HEAD_WIDE
#define RL_HEAD_WIDE 1
#endif

template <int MODE>
static rl_status launch_head(const CUtensorMap& mh, const CUtensorMap& mw, const HeadArgs& a, cudaStream_t s) {
  constexpr bool kWide = ((RL_HEAD_WIDE >> MODE) & 1) != 0;
  auto kern = kWide ? head_wide_kernel<MODE> : head_kernel<MODE, kPair>;
  constexpr size_t smem = kWide ? kSmemW : (kPair ? kSmem2 : kSmem);
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kWide ? kThreadsW : kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  static std::mutex mu;
  static std::map<std::pair<int, int>, int> resident;  // pairs resident at once (pair form)
  int max_pairs = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    auto key = std::make_pair(dev, MODE);
    auto it = resident.find(key);
    if (it == resident.end()) {
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(head_kernel)");
      int n = sms;
      if constexpr (kPair || kWide) {
        cfg.gridDim = dim3(2);
        e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
        if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveClusters(head_kernel)");
        if (n <= 0) return set_error(RL_ERR_UNSUPPORTED, "head_kernel: no CTA pair fits on the device");
      }
      it = resident.emplace(key, n).first;
    }
    max_pairs = it->second;
  }
  if constexpr (kPair || kWide) {
    // persistent: one 2-CTA cluster per resident pair, work items of 256 tokens x one vocabulary block
    const int items = (a.Tc + 2 * BM - 1) / (2 * BM) * a.n_vb;
    const int pairs = std::max(1, std::min(items, max_pairs));
    cfg.gridDim = dim3(2 * pairs);
    e = cudaLaunchKernelEx(&cfg, kern, mh, mw, a);
    if (e != cudaSuccess) return cuda_error(e, "cudaLaunchKernelEx(head_kernel)");
  } else {
    const int items = a.n_mt * a.n_vb;
    kern<<<std::min(items, sms), kThreads, smem, s>>>(mh, mw, a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "head_kernel launch");
  }
  return RL_OK;
}

}  // namespace head

size_t head_workspace_bytes(int64_t max_rows, int64_t V, int64_t D) {
  (void)D;
  return head::layout(max_rows, V).total;
}

size_t head_workspace_bytes_grouped(int64_t max_rows, int64_t V, int64_t D, int64_t group_tokens) {
  const int64_t g = (std::max<int64_t>(group_tokens, 1) + head::kChunk - 1) / head::kChunk;
  (void)D;
  return head::layout(max_rows, V, 0, g).total;
}

// The forward-only call needs the status word and one chunk's partials, which sit at the
// same offset as in the loss layout's header; rl_workspace_size(T, V, D) always suffices.
// It keeps the loss call's chunk of 4,096 tokens: the chunk's hidden states (32 MB at
// D = 4,096) and the W tiles in use then stay in L2 together. Measured at 32,768 x 4,096 x
// 151,936: chunks of 4,096 tokens give 24.8 ms per forward-only call (70.9 ms per loss call),
// 3,072 and 6,144 are within 2%, 8,192 takes 26.7 ms (73.1), and 32,768 takes 31.5 ms: the
// hidden states (256 MB) then evict W's tiles from the 129 MB L2.
static size_t head_logp_workspace_bytes(int64_t T, int64_t V) {
  const head::Layout L = head::layout(T, V);
  return kWsHeader + head::al256(static_cast<size_t>(head::kParts * L.n_vb * L.Tc) * sizeof(float4));
}

}  // namespace rl

extern "C" rl_status rl_fused_head_loss_fwd_bwd(
    const void* hidden, const void* weight, int64_t T, int64_t D, int64_t V, const int32_t* token_ids,
    const uint8_t* mask, const int32_t* token_traj, int32_t n_traj, const float* adv, const float* coef,
    const float* old_logp, const float* ref_logp, const float* rollout_logp, const rl_loss_params* params,
    void* d_hidden, rl_dtype d_hidden_dtype, float* d_weight, double* loss_accum, float* token_stats, void* ws,
    size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  using namespace rl::head;
  clear_error();
  if (T < 0 || D < 64 || V < 1 || n_traj < 0)
    return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_loss_fwd_bwd: need T >= 0, D >= 64, V >= 1, n_traj >= 0");
  if (D % 64 != 0) return set_error(RL_ERR_UNSUPPORTED, "rl_fused_head_loss_fwd_bwd: D must be a multiple of 64");
  if (T > INT32_MAX || V > static_cast<int64_t>(kMaxTilesSmem) * BN || D > 65536)
    return set_error(RL_ERR_UNSUPPORTED, "rl_fused_head_loss_fwd_bwd: T above 2^31 - 1, V above 524,288 or D above 65536");
  if (!params || !loss_accum || !ws) return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_loss_fwd_bwd: NULL argument");
  if (d_hidden_dtype != RL_BF16 && d_hidden_dtype != RL_F32)
    return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_loss_fwd_bwd: unknown d_hidden dtype");
  if (params->kl_estimator != 0 && params->kl_estimator != 3)
    return set_error(RL_ERR_UNSUPPORTED, "rl_fused_head_loss_fwd_bwd: kl_estimator must be 0 or 3");
  if (params->token_level_adv != 0 && params->token_level_adv != 1)
    return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_loss_fwd_bwd: token_level_adv must be 0 or 1");
  if (ws_bytes < rl_workspace_size(T, V, D))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL,
                     "rl_fused_head_loss_fwd_bwd: workspace smaller than rl_workspace_size(T, V, D)");
  if (T == 0) return RL_OK;
  if (!hidden || !weight || !token_ids || !mask || !token_traj || !old_logp || !d_hidden || !d_weight ||
      (n_traj > 0 && (!adv || !coef)) || (params->token_level_adv && !adv))
    return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_loss_fwd_bwd: NULL array argument");
  if (!aligned16(hidden) || !aligned16(weight) || !aligned16(d_hidden) || !aligned16(d_weight) || !aligned16(ws))
    return set_error(RL_ERR_ALIGNMENT,
                     "rl_fused_head_loss_fwd_bwd: hidden, weight, d_hidden, d_weight and ws must be 16-byte aligned");

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const Layout L = layout(T, V, ws_bytes);
  char* wsb = static_cast<char*>(ws);
  int32_t* status = reinterpret_cast<int32_t*>(wsb);
  double* row_loss = reinterpret_cast<double*>(wsb + ws_row_loss_offset());
  float4* partials = reinterpret_cast<float4*>(wsb + L.off_partials);
  RowCoef* rcs = reinterpret_cast<RowCoef*>(wsb + L.off_rc);
  float* tmax = reinterpret_cast<float*>(wsb + L.off_tmax);
  uint16_t* dz_base = reinterpret_cast<uint16_t*>(wsb + L.off_dz);
  rl_status st = RL_OK;
  const bool kl_on = params->kl_estimator == 3 && params->kl_coef != 0.f && ref_logp != nullptr;
  const bool ent = params->entropy_coef != 0.f || token_stats != nullptr;

  CUtensorMap mw;
  st = make_map(&mw, weight, D, V, kWBoxRows);
  if (st != RL_OK) return st;
  const int n_nt = static_cast<int>((V + BN - 1) / BN);
  const int64_t group_rows = L.G * L.Tc;
  for (int64_t t0 = 0; t0 < T; t0 += L.Tc) {
    const int Tc = static_cast<int>(std::min<int64_t>(L.Tc, T - t0));
    const int64_t g0 = t0 - t0 % group_rows;  // first token of this chunk's group
    uint16_t* dz = dz_base + (t0 - g0) * L.ldz;
    const uint16_t* h0 = static_cast<const uint16_t*>(hidden) + t0 * D;
    CUtensorMap mh;
    st = make_map(&mh, h0, D, Tc, BM);
    if (st != RL_OK) return st;
    HeadArgs ha = {};
    ha.t0 = t0;
    ha.Tc = Tc;
    ha.D = static_cast<int>(D);
    ha.V = static_cast<int>(V);
    ha.n_mt = (Tc + BM - 1) / BM;
    ha.n_nt = n_nt;
    ha.n_vb = static_cast<int>(L.n_vb);
    ha.ent = ent ? 1 : 0;
    ha.token_ids = token_ids;
    ha.partials = partials;
    ha.dz = dz;
    ha.ldz = L.ldz;
    ha.tmax = tmax;
    ha.status = status;
    st = launch_head<STATS_P>(mh, mw, ha, s);
    if (st != RL_OK) return st;

    MergeArgs ma = {};
    ma.t0 = t0;
    ma.Tc = Tc;
    ma.V = static_cast<int>(V);
    ma.n_part = ha.n_vb * static_cast<int>(kParts);
    ma.n_traj = n_traj;
    ma.partials = partials;
    ma.token_ids = token_ids;
    ma.mask = mask;
    ma.token_traj = token_traj;
    ma.adv = adv;
    ma.coef = coef;
    ma.old_logp = old_logp;
    ma.ref_logp = kl_on ? ref_logp : nullptr;
    ma.rollout_logp = rollout_logp;
    ma.clip_lo = 1.f - params->clip_eps_low;
    ma.clip_hi = 1.f + params->clip_eps_high;
    ma.beta = kl_on ? params->kl_coef : 0.f;
    ma.alpha = params->entropy_coef;
    ma.tis_cap = rollout_logp ? params->tis_cap : 0.f;
    ma.adv_per_row = params->token_level_adv;
    ma.rc = rcs;
    ma.row_loss = row_loss;
    ma.token_stats = token_stats;
    ma.status = status;
    head_merge_kernel<<<(Tc + kMergeThreads - 1) / kMergeThreads, kMergeThreads, 0, s>>>(ma);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "head_merge_kernel launch");

    DzArgs da = {};
    da.Tc = Tc;
    da.V = static_cast<int>(V);
    da.n_nt = n_nt;
    da.ent = ent && params->entropy_coef != 0.f ? 1 : 0;
    da.rc = rcs;
    da.dz = dz;
    da.ldz = L.ldz;
    da.tmax = tmax;
    head_dz_kernel<<<std::min(Tc, 148 * 16), kDzThreads, 0, s>>>(da);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "head_dz_kernel launch");

    // after the group's last chunk, the two products over the group's n = g1 - g0 tokens
    const int64_t g1 = std::min<int64_t>(g0 + group_rows, T);
    if (t0 + Tc == g1) {
      const int64_t n = g1 - g0;
      void* dh = static_cast<char*>(d_hidden) + g0 * D * (d_hidden_dtype == RL_BF16 ? 2 : 4);
      st = head_grad(dz_base, L.ldz, n, V, weight, static_cast<const uint16_t*>(hidden) + g0 * D, D, dh,
                     d_hidden_dtype, d_weight, reinterpret_cast<uint32_t*>(wsb + kWsHeadCounterOffset), status, s);
      if (st != RL_OK) return st;
    }
  }
  return launch_reduce_loss(row_loss, T, loss_accum, s);
}

extern "C" rl_status rl_fused_head_token_logprobs(const void* hidden, const void* weight, int64_t T, int64_t D,
                                                  int64_t V, const int32_t* token_ids, float* logp_out,
                                                  float* entropy_out, float* lse_out, void* ws, size_t ws_bytes,
                                                  rl_stream_t stream) {
  using namespace rl;
  using namespace rl::head;
  clear_error();
  if (T < 0 || D < 64 || V < 1)
    return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_token_logprobs: need T >= 0, D >= 64, V >= 1");
  if (D % 64 != 0) return set_error(RL_ERR_UNSUPPORTED, "rl_fused_head_token_logprobs: D must be a multiple of 64");
  if (T > INT32_MAX || V > INT32_MAX || D > 65536)
    return set_error(RL_ERR_UNSUPPORTED, "rl_fused_head_token_logprobs: T or V above 2^31 - 1, or D above 65536");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_token_logprobs: NULL workspace");
  if (ws_bytes < head_logp_workspace_bytes(T, V))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL, "rl_fused_head_token_logprobs: workspace too small");
  if (T == 0) return RL_OK;
  if (!hidden || !weight || !token_ids || !logp_out)
    return set_error(RL_ERR_INVALID_ARG, "rl_fused_head_token_logprobs: NULL array argument");
  if (!aligned16(hidden) || !aligned16(weight) || !aligned16(ws))
    return set_error(RL_ERR_ALIGNMENT, "rl_fused_head_token_logprobs: hidden, weight and ws must be 16-byte aligned");

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const Layout L = layout(T, V);
  char* wsb = static_cast<char*>(ws);
  int32_t* status = reinterpret_cast<int32_t*>(wsb);
  float4* partials = reinterpret_cast<float4*>(wsb + kWsHeader);
  CUtensorMap mw;
  rl_status st = make_map(&mw, weight, D, V, kWBoxRows);
  if (st != RL_OK) return st;
  const int n_nt = static_cast<int>((V + BN - 1) / BN);
  for (int64_t t0 = 0; t0 < T; t0 += L.Tc) {
    const int Tc = static_cast<int>(std::min<int64_t>(L.Tc, T - t0));
    CUtensorMap mh;
    st = make_map(&mh, static_cast<const uint16_t*>(hidden) + t0 * D, D, Tc, BM);
    if (st != RL_OK) return st;
    HeadArgs ha = {};
    ha.t0 = t0;
    ha.Tc = Tc;
    ha.D = static_cast<int>(D);
    ha.V = static_cast<int>(V);
    ha.n_mt = (Tc + BM - 1) / BM;
    ha.n_nt = n_nt;
    ha.n_vb = static_cast<int>(L.n_vb);
    ha.ent = entropy_out ? 1 : 0;
    ha.token_ids = token_ids;
    ha.partials = partials;
    ha.status = status;
    st = launch_head<STATS>(mh, mw, ha, s);
    if (st != RL_OK) return st;
    LogpMergeArgs ma = {};
    ma.t0 = t0;
    ma.Tc = Tc;
    ma.V = static_cast<int>(V);
    ma.n_part = ha.n_vb * static_cast<int>(kParts);
    ma.partials = partials;
    ma.token_ids = token_ids;
    ma.logp_out = logp_out;
    ma.entropy_out = entropy_out;
    ma.lse_out = lse_out;
    ma.status = status;
    head_logp_merge_kernel<<<(Tc + kMergeThreads - 1) / kMergeThreads, kMergeThreads, 0, s>>>(ma);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "head_logp_merge_kernel launch");
  }
  return RL_OK;
}
