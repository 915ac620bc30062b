// Streaming log-softmax kernels over logits rows:
//
//   rl_token_logprobs       logp / entropy / lse of the sampled token per row
//                           (pi(a_t | s_t) of Sec. 2.3; the pi_old recompute of
//                           Sec. 3.2.4)
//   rl_policy_loss_fwd_bwd  the masked clipped objective (Sec. 2.3.1, 2.3.2),
//                           k3-KL, entropy bonus and TIS weight (Sec. 3.2.4), and
//                           d loss / d logits
//
// Design (GB300, sm_103a). Each logits row is owned by one thread-block
// cluster of C CTAs; CTA k of the cluster holds the vocabulary slice
// [k * slice, (k + 1) * slice) of the row in shared memory. The slice arrives
// by bulk asynchronous copies (cp.async.bulk, the 1-D TMA) completing on an
// mbarrier, double-buffered so the copy of the cluster's next row overlaps the
// work on the current one. Pass 1 reads the slice once from shared memory and
// forms an online-softmax partial (max m, sum exp(z - m), sum exp(z - m)(z - m));
// the C partials are exchanged through distributed shared memory and merged
// identically in every CTA. Pass 2 re-reads the slice from shared memory and
// writes the gradient with 16-byte stores. Each unmasked row is therefore read
// from HBM exactly once and its gradient written once; masked rows (and rows of
// trajectories with c_i = 0) are not read at all, only zero-filled.
//
// Rows of at most 8 KB (V <= 4,096 bf16 or 2,048 fp32) take a lighter form of the
// loss kernel, a warp per row with the row held in registers (small_rows_kernel).
//
// The kernels are persistent: the grid holds as many clusters as fit on the
// GPU at once, and cluster j processes rows j, j + n_clusters, ... . Each
// cluster adds its rows' loss contributions in row order and leaves one partial
// in the workspace; the last cluster to finish (a counter in the workspace
// header) sums the partials in a fixed order into the caller's total, so the
// loss is bit-reproducible without a second launch.
#include <algorithm>
#include <cstdint>
#include <map>
#include <mutex>
#include <tuple>
#include <type_traits>

#include "rl_device.cuh"
#include "rl_host.h"

namespace rl {

struct RowArgs {
  const void* logits;
  void* grad;
  int64_t rows, V, ld;
  const int32_t* token_ids;
  const uint8_t* mask;
  const int32_t* token_traj;
  int32_t n_traj;
  const float* adv;
  const float* coef;
  const float* old_logp;
  const float* ref_logp;
  const float* rollout_logp;
  float clip_lo, clip_hi;  // 1 - eps_low, 1 + eps_high
  float beta;              // 0 when the KL term is off
  float alpha;             // entropy bonus
  float tis_cap;           // <= 0 when TIS is off
  int32_t adv_per_row;     // adv holds one A_t per row (else one per trajectory)
  double* row_loss;
  double* loss_accum;      // the caller's total (loss kernel: the last cluster adds into it)
  uint32_t* done;          // finished-cluster count in the workspace header
  float* token_stats;
  float* logp_out;
  float* entropy_out;
  float* lse_out;
  int32_t* status;
  int64_t slice;      // elements per CTA slice, a multiple of the 16-byte vector
  int64_t buf_elems;  // element stride between the two shared-memory buffers
  int32_t tma;        // rows 16-byte aligned: bulk copies and 16-byte stores
};

#ifndef RL_STORE_CS
#define RL_STORE_CS 0
#endif

// 16-byte global store; with RL_STORE_CS the line is marked evict-first (streaming)
__device__ __forceinline__ void st_global_16(void* p, uint4 w) {
#if RL_STORE_CS
  asm volatile("st.global.cs.v4.b32 [%0], {%1, %2, %3, %4};" :: "l"(p), "r"(w.x), "r"(w.y), "r"(w.z), "r"(w.w)
               : "memory");
#else
  *reinterpret_cast<uint4*>(p) = w;
#endif
}

template <typename T>
struct Vec;
template <>
struct Vec<uint16_t> {  // bf16
  static constexpr int N = 8;
  static __device__ __forceinline__ void load(const uint16_t* buf, int64_t j, float (&v)[8]) {
    const uint4 w = reinterpret_cast<const uint4*>(buf)[j];
    v[0] = bf16_lo(w.x); v[1] = bf16_hi(w.x); v[2] = bf16_lo(w.y); v[3] = bf16_hi(w.y);
    v[4] = bf16_lo(w.z); v[5] = bf16_hi(w.z); v[6] = bf16_lo(w.w); v[7] = bf16_hi(w.w);
  }
  static constexpr int NP = 4;  // float2 pairs per 16-byte vector
  // pad of register-held vectors past the slice: two bf16 values of about -1.5e38, at or below
  // -1e38 (so they count as -inf for the maximum) yet far enough from -FLT_MAX that
  // z log2(e) - m log2(e) stays finite: its exponential is 0 and, with the entropy on, e x is
  // 0, not 0 x -inf = NaN (which would send every thread holding a pad down the slow path)
  static constexpr uint32_t kPadWord = 0xFEE1FEE1u;
  static __device__ __forceinline__ void pairs(const uint4 w, float2 (&q)[4]) {
    q[0] = make_float2(bf16_lo(w.x), bf16_hi(w.x)); q[1] = make_float2(bf16_lo(w.y), bf16_hi(w.y));
    q[2] = make_float2(bf16_lo(w.z), bf16_hi(w.z)); q[3] = make_float2(bf16_lo(w.w), bf16_hi(w.w));
  }
  static __device__ __forceinline__ uint4 pack_pairs(const float2 (&o)[4]) {
    return make_uint4(pack_bf16x2(o[0].x, o[0].y), pack_bf16x2(o[1].x, o[1].y), pack_bf16x2(o[2].x, o[2].y),
                      pack_bf16x2(o[3].x, o[3].y));
  }
  static __device__ __forceinline__ void unpack(const uint4 w, float (&v)[8]) {
    v[0] = bf16_lo(w.x); v[1] = bf16_hi(w.x); v[2] = bf16_lo(w.y); v[3] = bf16_hi(w.y);
    v[4] = bf16_lo(w.z); v[5] = bf16_hi(w.z); v[6] = bf16_lo(w.w); v[7] = bf16_hi(w.w);
  }
  static __device__ __forceinline__ void store(uint16_t* dst, const float (&g)[8]) {
    uint4 w;
    w.x = pack_bf16x2(g[0], g[1]); w.y = pack_bf16x2(g[2], g[3]);
    w.z = pack_bf16x2(g[4], g[5]); w.w = pack_bf16x2(g[6], g[7]);
    st_global_16(dst, w);
  }
  static __device__ __forceinline__ void store_scalar(uint16_t* dst, float g) { *dst = f32_to_bf16(g); }
  static __device__ __forceinline__ float to_f(uint16_t x) { return bf16_to_f32(x); }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void load(const float* buf, int64_t j, float (&v)[4]) {
    const float4 w = reinterpret_cast<const float4*>(buf)[j];
    v[0] = w.x; v[1] = w.y; v[2] = w.z; v[3] = w.w;
  }
  static constexpr int NP = 2;
  static constexpr uint32_t kPadWord = 0xFEE1B1E6u;  // -1.5e38: see Vec<uint16_t>::kPadWord
  static __device__ __forceinline__ void pairs(const uint4 w, float2 (&q)[2]) {
    q[0] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
    q[1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
  }
  static __device__ __forceinline__ uint4 pack_pairs(const float2 (&o)[2]) {
    return make_uint4(__float_as_uint(o[0].x), __float_as_uint(o[0].y), __float_as_uint(o[1].x),
                      __float_as_uint(o[1].y));
  }
  static __device__ __forceinline__ void unpack(const uint4 w, float (&v)[4]) {
    v[0] = __uint_as_float(w.x); v[1] = __uint_as_float(w.y); v[2] = __uint_as_float(w.z); v[3] = __uint_as_float(w.w);
  }
  static __device__ __forceinline__ void store(float* dst, const float (&g)[4]) {
    st_global_16(dst, make_uint4(__float_as_uint(g[0]), __float_as_uint(g[1]), __float_as_uint(g[2]),
                                 __float_as_uint(g[3])));
  }
  static __device__ __forceinline__ void store_scalar(float* dst, float g) { *dst = g; }
  static __device__ __forceinline__ float to_f(float x) { return x; }
};

#define RL_NEG_INF (-__int_as_float(0x7f800000))

// Pass 1: -inf (and anything below -1e30) becomes -1e30, so that e = 0 and e (z - m) = 0
// instead of NaN; a NaN stays NaN (a comparison, not fmaxf, which would drop it) and poisons
// its row. Pass 2 clamps with fmaxf: there p = 2^(NaN) is NaN already.
__device__ __forceinline__ float clamp_ninf(float z) { return z < -1e30f ? -1e30f : z; }
constexpr uint32_t kBulkChunk = 32768;

// fold one value into a per-thread online-softmax partial whose max is already >= z
template <bool ENT>
__device__ __forceinline__ void accumulate(SoftmaxPartial& ps, float z, float neg_m_l2e) {
  if (ENT) {
    const float t = clamp_ninf(z) - ps.m;  // -inf logits contribute 0, not NaN
    const float e = ex2(t * kLog2e);
    ps.s += e;
    ps.u = fmaf(e, t, ps.u);
  } else {
    ps.s += ex2(fmaf(z, kLog2e, neg_m_l2e));
  }
}

template <bool ENT>
__device__ __forceinline__ void raise_max(SoftmaxPartial& ps, float vm) {
  if (vm > ps.m) {
    const float d = ps.m - vm;
    const float sc = ex2(d * kLog2e);
    if (ENT) ps.u = (ps.s == 0.f) ? 0.f : sc * fmaf(d, ps.s, ps.u);
    ps.s *= sc;
    ps.m = vm;
  }
}

// Shared-memory stages per CTA (tuning knob). The consumer warps per CTA, the 16-byte vectors
// of the slice each consumer thread holds in registers, the CTAs per SM and the slice size that
// picks the cluster width are chosen per path on the host (loss_shape).
#ifndef RL_STAGES
#define RL_STAGES 2
#endif

constexpr int kMaxCluster = 16;
// zero-filled shared region, source of the masked rows' bulk stores (8 KB at 2 CTAs per SM:
// 12.947 against 13.029 ms per benchmark step with 2 KB)
constexpr int kZeroBytesMax = 8192;

// Per-row inputs, staged in shared memory by the producer warp.
struct RowMeta {
  int64_t r;  // row index, -1 = end of the stream
  int32_t a;  // sampled token id
  float A, c, old, ref, roll;
};

// Warp-specialised, cluster-per-row kernel.
//
//   warp NW (producer): walks this cluster's rows cid, cid + ncl, ...; decides which
//     are trained on; zero-fills the others with bulk stores from a zeroed shared
//     region; for a trained row stages its metadata and bulk-copies this CTA's slice
//     into the next free stage (full / empty mbarrier pair per stage).
//   warps 0..NW-1 (consumers): per row, pass 1 over the slice gives one online-softmax
//     partial per warp; every warp pushes its partial to all C CTAs of the cluster
//     with st.async (remote store + complete_tx on the receiver's mailbox mbarrier);
//     each warp then merges all C * NW partials in a fixed order (bit-identical in
//     every warp of every CTA), computes the row's scalars, runs pass 2 (gradient
//     from the on-chip slice) and releases the stage.
// Nothing per row synchronises a whole CTA or the whole cluster.
// Fold EPV values into an online-softmax partial. The reference ps.m is the first
// finite vector maximum and moves only when a vector's exponentials sum above 1e30
// (some value lies far above the reference): the common case needs no per-element
// max. exp(z - m) <= e^88 < FLT_MAX for every z within 88 of m, so before that
// test overflows nothing.
template <bool ENT, int EPV>
__device__ __forceinline__ void fold(SoftmaxPartial& ps, const float (&v)[EPV]) {
  if (ps.m == RL_NEG_INF) {
    float vm = v[0];
#pragma unroll
    for (int k = 1; k < EPV; ++k) vm = fmaxf(vm, v[k]);
    if (vm == RL_NEG_INF) return;
    ps.m = vm;
  }
  float e[EPV], t[EPV];
  auto exps = [&]() {
    const float nm = -ps.m * kLog2e;
#pragma unroll
    for (int k = 0; k < EPV; ++k) {
      if (ENT) {
        t[k] = clamp_ninf(v[k]) - ps.m;  // -inf logits contribute 0, not NaN
        e[k] = ex2(t[k] * kLog2e);
      } else {
        e[k] = ex2(fmaf(v[k], kLog2e, nm));
      }
    }
  };
  auto tree = [&](const float (&x)[EPV]) {
    float a[EPV];
#pragma unroll
    for (int k = 0; k < EPV; ++k) a[k] = x[k];
#pragma unroll
    for (int w = EPV / 2; w > 0; w /= 2)
#pragma unroll
      for (int k = 0; k < w; ++k) a[k] += a[k + w];
    return a[0];
  };
  exps();
  float se = tree(e);
  if (!(se <= 1e30f)) {  // rare: move the reference up to this vector's maximum
    float vm = v[0];
#pragma unroll
    for (int k = 1; k < EPV; ++k) vm = fmaxf(vm, v[k]);
    raise_max<ENT>(ps, vm);
    exps();
    se = tree(e);
  }
  ps.s += se;
  if (ENT) {
    float et[EPV];
#pragma unroll
    for (int k = 0; k < EPV; ++k) et[k] = e[k] * t[k];
    ps.u += tree(et);
  }
}

// Fold NV register-held 16-byte vectors into a partial, branch-free in the common
// case. Vectors past the end of the data hold about -1.5e38 (Vec<T>::kPadWord), whose
// exponential is exactly 0. The reference is the partial's own maximum or, for a
// fresh partial, the first vector's maximum; when the exponentials sum above 1e30
// (a value far above the reference) everything is redone against the exact
// maximum. Values at or below -1e38 count as -inf.
template <typename T, bool ENT, int NV, typename Reload>
__device__ __forceinline__ void fold_block(SoftmaxPartial& ps, const uint4 (&x)[NV], Reload reload) {
  constexpr int NP = Vec<T>::NP;
  auto vmax = [&](const uint4 w) {
    float2 q[NP];
    Vec<T>::pairs(w, q);
    float m = fmaxf(q[0].x, q[0].y);
#pragma unroll
    for (int i = 1; i < NP; ++i) m = fmaxf(m, fmaxf(q[i].x, q[i].y));
    return m;
  };
  // exact maximum, recomputed from shared memory (the rare paths only)
  auto all_max = [&]() {
    float m = vmax(reload(0));
    for (int k = 1; k < NV; ++k) m = fmaxf(m, vmax(reload(k)));
    return m;
  };
  if (!(ps.m > -1e38f)) {
    float m0 = vmax(x[0]);
    if (!(m0 > -1e38f)) m0 = all_max();
    if (!(m0 > -1e38f)) return;
    ps.m = m0;
  }
  // x = (z - m) log2(e) by one fused multiply-add against nm = fl(-m log2(e)); with the
  // entropy, u accumulates e x (log2 units, scaled by ln 2 at the end). A logit at -inf gives
  // e = 0 and e x = NaN: such a block is redone on the clamped path (CLAMP), where z counts as
  // -1e30 (a NaN stays NaN). The rounding of nm shifts every x of the block by the same
  // err = -m log2(e) - nm (exact by one fma); the block's sums are corrected for it once at
  // the end.
  auto exps = [&](auto clamp, const uint4 w, float2& s0, float2& s1, float2& u0) {
    constexpr bool CLAMP = decltype(clamp)::value;
    const float nm = -ps.m * kLog2e;
    const float2 l2 = make_float2(kLog2e, kLog2e), nm2 = make_float2(nm, nm);
    float2 q[NP];
    Vec<T>::pairs(w, q);
#pragma unroll
    for (int i = 0; i < NP; ++i) {
      const float2 qi = CLAMP ? make_float2(clamp_ninf(q[i].x), clamp_ninf(q[i].y)) : q[i];
      const float2 xx = __ffma2_rn(qi, l2, nm2);
      const float2 e = make_float2(ex2(xx.x), ex2(xx.y));
      if (i & 1) s1 = __fadd2_rn(s1, e); else s0 = __fadd2_rn(s0, e);
      if (ENT) u0 = __ffma2_rn(e, xx, u0);
    }
  };
  using Fast = std::integral_constant<bool, false>;
  using Clamped = std::integral_constant<bool, true>;
  const float2 z2 = make_float2(0.f, 0.f);
  float2 s0 = z2, s1 = z2, u0 = z2;
#pragma unroll
  for (int k = 0; k < NV; ++k) exps(Fast{}, x[k], s0, s1, u0);
  float2 sacc = __fadd2_rn(s0, s1);
  float se = sacc.x + sacc.y;
  float ue = ENT ? u0.x + u0.y : 0.f;
  if (!(se <= 1e30f) || (ENT && ue != ue)) {
    // rare: a value far above the reference (move it up to the exact maximum) or a logit at
    // -inf with the entropy on; redo from shared memory on the clamped path
    if (!(se <= 1e30f)) raise_max<ENT>(ps, all_max());
    s0 = z2; s1 = z2; u0 = z2;
    for (int k = 0; k < NV; ++k) exps(Clamped{}, reload(k), s0, s1, u0);
    sacc = __fadd2_rn(s0, s1);
    se = sacc.x + sacc.y;
    ue = ENT ? u0.x + u0.y : 0.f;
  }
  // e_true = e 2^err and x_true = x + err, with |err| <= 2^-24 |m log2(e)|: first order in err
  const float nm = -ps.m * kLog2e;
  const float err = fmaf(-ps.m, kLog2e, -nm);
  const float f = fmaf(err, kLn2, 1.f);
  if (ENT) ps.u = fmaf(fmaf(err, se, ue) * f, kLn2, ps.u);
  ps.s = fmaf(se, f, ps.s);
}

// MINB: CTAs per SM the register budget is sized for (2, or 3 with a smaller zero region).
template <typename T, int NW, bool ENT, bool BWD, int HOLDV, int MINB>
__global__ void __launch_bounds__((NW + 1) * 32, MINB) rows_kernel(const RowArgs p) {
  constexpr int kZeroBytes = MINB >= 3 ? 2048 : kZeroBytesMax;
  constexpr int EPV = Vec<T>::N;
  constexpr int NB = RL_STAGES;
  constexpr int NC = NW * 32;  // consumer threads
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[NB], empty_bar[NB], xbar[2];
  __shared__ RowMeta meta[NB];
  __shared__ __align__(16) float4 mbox[2][kMaxCluster * NW];
  __shared__ __align__(128) uint4 zeros[kZeroBytes / 16];

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t rank = cluster_ctarank(), C = cluster_nctarank();
  const int64_t cid = blockIdx.x / C, ncl = gridDim.x / C;
  const int64_t rows = p.rows, V = p.V, ld = p.ld;
  const int64_t s0 = static_cast<int64_t>(rank) * p.slice;
  const int64_t n_end = (s0 + p.slice < V) ? s0 + p.slice : V;
  const int n = n_end > s0 ? static_cast<int>(n_end - s0) : 0;  // elements of my slice
  const int nv = n / EPV;                                        // full 16-byte vectors
  const int first_scalar = p.tma ? nv * EPV : 0;
  const uint32_t tma_bytes = p.tma ? static_cast<uint32_t>(nv * 16) : 0u;
  const T* logits = static_cast<const T*>(p.logits);
  T* grad = static_cast<T*>(p.grad);
  T* const buf_base = reinterpret_cast<T*>(smem_raw);

  if (tid == 0) {
#pragma unroll
    for (int k = 0; k < NB; ++k) {
      mbar_init(&full_bar[k], 1);
      mbar_init(&empty_bar[k], NW);
    }
    mbar_init(&xbar[0], 1);
    mbar_init(&xbar[1], 1);
    fence_mbar_init();
  }
  for (int k = tid; k < kZeroBytes / 16; k += blockDim.x) zeros[k] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  __syncthreads();
  if (C > 1) cluster_sync_all();  // every peer's mailbox barrier exists before the first st.async

  if (warp == NW) {
    // =============================================================== producer warp
    // Row metadata is fetched 32 rows at a time, one row per lane, and handed row by row to the
    // staging loop with shuffles. The loads of the next batch are issued while the current one
    // is staged (its owners' coefficients once the owners have arrived), so their latency is
    // hidden behind the copies.
    uint32_t it = 0;
    bool failed = false, stored = false;
    struct Batch {
      int32_t a, i;
      uint32_t m;
      float c, A, old, ref, roll;
    };
    auto load_primary = [&](int64_t b0, Batch& q) {
      const int64_t my = b0 + static_cast<int64_t>(lane) * ncl;
      q = Batch{0, -1, 0u, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (my < rows) {
        q.a = p.token_ids[my];
        if (BWD) {
          q.m = p.mask[my];
          q.i = p.token_traj[my];
          q.old = p.old_logp[my];
          if (p.ref_logp) q.ref = p.ref_logp[my];
          if (p.rollout_logp) q.roll = p.rollout_logp[my];
          if (p.adv_per_row) q.A = p.adv[my];
        }
      }
    };
    auto load_dependent = [&](Batch& q) {
      if (BWD && q.m != 0 && q.i >= 0 && q.i < p.n_traj) {
        q.c = p.coef[q.i];
        if (!p.adv_per_row) q.A = p.adv[q.i];
      }
    };
    Batch cur, nxt = Batch{0, -1, 0u, 0.f, 0.f, 0.f, 0.f, 0.f};
    load_primary(cid, cur);
    load_dependent(cur);
    for (int64_t base = cid; base < rows && !failed; base += 32 * ncl) {
      const int64_t next_base = base + 32 * ncl;
      const bool has_next = next_base < rows;
      if (has_next) load_primary(next_base, nxt);
      const int32_t la = cur.a, li = cur.i;
      const uint32_t lm = cur.m;
      const float lc = cur.c, lA = cur.A, lold = cur.old, lref = cur.ref, lroll = cur.roll;
      const int nb = static_cast<int>(min(static_cast<int64_t>(32), (rows - base + ncl - 1) / ncl));
      for (int jr = 0; jr < nb && !failed; ++jr) {
        if (jr == 1 && has_next) load_dependent(nxt);  // the next batch's owners have arrived by now
        const int64_t r = base + static_cast<int64_t>(jr) * ncl;
        RowMeta m;
        bool active = true;
        m.r = r;
        m.a = __shfl_sync(0xffffffffu, la, jr);
        if (BWD) {
          active = __shfl_sync(0xffffffffu, lm, jr) != 0;
          if (active) {
            const int32_t i = __shfl_sync(0xffffffffu, li, jr);
            if (i < 0 || i >= p.n_traj) {
              if (rank == 0 && lane == 0) flag_status(p.status, RL_DEV_BAD_TRAJ);
              active = false;
            } else {
              m.c = __shfl_sync(0xffffffffu, lc, jr);
              m.A = __shfl_sync(0xffffffffu, lA, jr);
              active = m.c != 0.f;
              if (active && (m.a < 0 || m.a >= V)) {
                if (rank == 0 && lane == 0) flag_status(p.status, RL_DEV_BAD_TOKEN);
                active = false;
              }
            }
          }
          if (!active) {
            // zero this CTA's slice of gradient row r
            T* g = grad + r * ld + s0;
            if (p.tma) {
              if (lane == 0) {
                const uint32_t bytes = tma_bytes;
                for (uint32_t off = 0; off < bytes; off += kZeroBytes)
                  bulk_s2g(reinterpret_cast<char*>(g) + off, zeros, min(static_cast<uint32_t>(kZeroBytes), bytes - off));
                bulk_commit();
                stored = true;
              }
              for (int e = nv * EPV + lane; e < n; e += 32) g[e] = T(0);
            } else {
              for (int e = lane; e < n; e += 32) g[e] = T(0);
            }
            if (rank == 0 && lane == 0 && p.token_stats)
              for (int k = 0; k < 5; ++k) p.token_stats[r * 5 + k] = 0.f;
            continue;
          }
          m.old = __shfl_sync(0xffffffffu, lold, jr);
          m.ref = __shfl_sync(0xffffffffu, lref, jr);
          m.roll = __shfl_sync(0xffffffffu, lroll, jr);
        }
        const int b = it % NB;
        const uint32_t use = it / NB;
        if (use > 0 && !mbar_wait_bounded(&empty_bar[b], (use - 1) & 1)) {
          failed = true;
          if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
          break;
        }
        T* buf = buf_base + b * p.buf_elems;
        const T* src = logits + r * ld + s0;
        for (int e = first_scalar + lane; e < n; e += 32) buf[e] = src[e];
        __syncwarp();
        if (lane == 0) {
          meta[b] = m;
          if (tma_bytes > 0) {
            mbar_arrive_expect_tx(&full_bar[b], tma_bytes);
            for (uint32_t off = 0; off < tma_bytes; off += kBulkChunk)
              bulk_g2s(reinterpret_cast<char*>(buf) + off, reinterpret_cast<const char*>(src) + off,
                       min(kBulkChunk, tma_bytes - off), &full_bar[b]);
          } else {
            mbar_arrive(&full_bar[b]);
          }
        }
        ++it;
      }
      if (has_next && nb <= 1) load_dependent(nxt);
      cur = nxt;
    }
    if (!failed) {
      // end of stream
      const int b = it % NB;
      const uint32_t use = it / NB;
      if (use > 0 && !mbar_wait_bounded(&empty_bar[b], (use - 1) & 1)) {
        if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
      } else if (lane == 0) {
        meta[b].r = -1;
        mbar_arrive(&full_bar[b]);
      }
    }
    if (lane == 0 && stored) bulk_wait_read_all();
  } else {
    // =============================================================== consumer warps
    // the cluster's loss contributions, added in the order of its rows (rank 0, warp 0, lane 0
    // keeps the sum; one partial per cluster goes to the workspace at the end)
    double cl_loss = 0.0;
    for (uint32_t it = 0;; ++it) {
      const int b = it % NB;
      if (!mbar_wait_bounded(&full_bar[b], (it / NB) & 1)) {
        if (tid == 0) flag_status(p.status, RL_DEV_TIMEOUT);
        break;
      }
      const RowMeta m = meta[b];
      if (m.r < 0) break;
      const int64_t r = m.r;
      const T* buf = buf_base + b * p.buf_elems;
      const int32_t a = m.a;
      const bool a_ok = a >= 0 && a < V;
      const uint32_t owner = a_ok ? static_cast<uint32_t>(a / p.slice) : 0u;

      // ---- pass 1: online softmax partial over the slice. With HOLDV > 0 the slice moves
      // into registers here (vector j = tid + k * NC in hold[k]) and the stage is released
      // right after, so the next copy lands while the exchange and pass 2 run.
      SoftmaxPartial ps{RL_NEG_INF, 0.f, 0.f};
      uint4 hold[HOLDV > 0 ? HOLDV : 1];
      float tail_z = 0.f;
      if (HOLDV > 0) {
        const uint32_t pad = Vec<T>::kPadWord;
        auto reload = [&](int k) {
          const int j = tid + k * NC;
          return j < nv ? reinterpret_cast<const uint4*>(buf)[j] : make_uint4(pad, pad, pad, pad);
        };
#pragma unroll
        for (int k = 0; k < (HOLDV > 0 ? HOLDV : 1); ++k) hold[k] = reload(k);
        fold_block<T, ENT>(ps, hold, reload);
      } else {
        for (int j = tid; j < nv; j += NC) {
          float v[EPV];
          Vec<T>::load(buf, j, v);
          fold<ENT>(ps, v);
        }
      }
      // ragged tail (fewer than EPV elements): one per thread at most
      if (nv * EPV + tid < n) {
        const float z = Vec<T>::to_f(buf[nv * EPV + tid]);
        tail_z = z;
        if (z != RL_NEG_INF) {
          raise_max<ENT>(ps, z);
          accumulate<ENT>(ps, z, -ps.m * kLog2e);
        }
      }
      ps = warp_merge(ps);
      // lane 0's merge is the warp's partial: broadcast it so every copy sent is identical
      ps.m = __shfl_sync(0xffffffffu, ps.m, 0);
      ps.s = __shfl_sync(0xffffffffu, ps.s, 0);
      ps.u = __shfl_sync(0xffffffffu, ps.u, 0);
      // warp 0 of the CTA holding the sampled token carries z_a; every other partial carries 0
      const float za_part = (warp == 0 && a_ok && rank == owner) ? Vec<T>::to_f(buf[a - s0]) : 0.f;
      if (HOLDV > 0) {  // every read of the stage is done
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[b]);
      }

      // ---- exchange: every warp's partial to every CTA of the cluster
      const int par = it & 1;
      if (warp == 0 && lane == 0) mbar_arrive_expect_tx(&xbar[par], C * NW * 16u);
      if (lane < static_cast<int>(C)) {
        const uint32_t dst = map_to_rank(smem_addr(&mbox[par][rank * NW + warp]), lane);
        const uint32_t bar = map_to_rank(smem_addr(&xbar[par]), lane);
        st_async_f4(dst, make_float4(ps.m, ps.s, ps.u, za_part), bar);
      }
      if (!mbar_wait_cluster_bounded(&xbar[par], (it >> 1) & 1)) {
        if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
        break;
      }
      // ---- merge all C * NW partials in a fixed order
      const int total = static_cast<int>(C) * NW;
      SoftmaxPartial qa{RL_NEG_INF, 0.f, 0.f}, qb{RL_NEG_INF, 0.f, 0.f};
      float zsum = 0.f;
      if (lane < total) {
        const float4 w = mbox[par][lane];
        qa = SoftmaxPartial{w.x, w.y, w.z};
        zsum = w.w;
      }
      if (lane + 32 < total) {
        const float4 w = mbox[par][lane + 32];
        qb = SoftmaxPartial{w.x, w.y, w.z};
        zsum += w.w;
      }
      for (int k = lane + 64; k < total; k += 32) {  // clusters of 16 with more than 4 consumer warps
        const float4 w = mbox[par][k];
        qb = merge(qb, SoftmaxPartial{w.x, w.y, w.z});
        zsum += w.w;
      }
      SoftmaxPartial q = warp_merge(merge(qa, qb));
      const float za = __shfl_sync(0xffffffffu, warp_sum(zsum), 0);
      const float lnS = logf(__shfl_sync(0xffffffffu, q.s, 0));
      const float lse = __shfl_sync(0xffffffffu, q.m, 0) + lnS;
      const float H = lnS - __shfl_sync(0xffffffffu, q.u, 0) / __shfl_sync(0xffffffffu, q.s, 0);

      if (!BWD) {
        if (rank == 0 && warp == 0 && lane == 0) {
          if (!a_ok) flag_status(p.status, RL_DEV_BAD_TOKEN);
          p.logp_out[r] = a_ok ? za - lse : __int_as_float(0x7fc00000);
          if (p.entropy_out) p.entropy_out[r] = H;
          if (p.lse_out) p.lse_out[r] = lse;
        }
      } else {
        // per-token scalars (every lane computes the same values)
        const float A = m.A, c = m.c, old = m.old;
        const float logp = za - lse;
        const float rho = expf((za - old) - lse);   // large operands differenced first
        const float crho = fminf(fmaxf(rho, p.clip_lo), p.clip_hi);
        const float surr = fminf(rho * A, crho * A);
        const bool cut = (A > 0.f && rho > p.clip_hi) || (A < 0.f && rho < p.clip_lo);
        const float w = (p.tis_cap > 0.f && p.rollout_logp) ? fminf(expf(old - m.roll), p.tis_cap) : 1.f;
        float kl = 0.f, dkl = 0.f;
        if (p.beta != 0.f && p.ref_logp) {
          const float d = (m.ref - za) + lse;  // r - logp
          const float ed = expf(d);
          kl = ed - d - 1.f;
          dkl = 1.f - ed;
        }
        const float ell = -w * surr + p.beta * kl - p.alpha * H;
        const float g = (cut ? 0.f : -w * A * rho) + p.beta * dkl;
        const float cg = c * g, ca0 = c * p.alpha;
        // p_v = 2^(z_v log2(e) + nl) with nl = fl(-lse log2(e)); its rounding scales every p_v of
        // the row by 2^errl (errl exact by one fma), folded into the coefficients below
        const float nl = -lse * kLog2e;
        const float fl = fmaf(fmaf(-lse, kLog2e, -nl), kLn2, 1.f);
        const float Kp = -cg * fl;                      // gradient = Kp p_v (+ cg at v = a)
        const float ca = ca0 * fl;                      // entropy: p_v (ca z_v + Ke)
        const float Ke = (-cg + ca0 * (H - lse)) * fl;
        if (rank == 0 && warp == 0 && lane == 0) {
          cl_loss += static_cast<double>(c) * static_cast<double>(ell);
          if (p.token_stats) {
            float* st = p.token_stats + r * 5;
            st[0] = logp; st[1] = rho; st[2] = cut ? 1.f : 0.f; st[3] = H; st[4] = kl;
          }
        }
        // ---- pass 2: gradient from the on-chip slice
        T* g_row = grad + r * ld + s0;
        auto grad_vec = [&](const float (&v)[EPV], int j) {
          float o[EPV];
#pragma unroll
          for (int k = 0; k < EPV; ++k) {
            const float pk = ex2(fmaf(v[k], kLog2e, nl));
            o[k] = ENT ? pk * fmaf(ca, fmaxf(v[k], -1e30f), Ke) : Kp * pk;
          }
          if (p.tma) {
            Vec<T>::store(g_row + j * EPV, o);
          } else {
#pragma unroll
            for (int k = 0; k < EPV; ++k) Vec<T>::store_scalar(g_row + j * EPV + k, o[k]);
          }
        };
        if (HOLDV > 0 && p.tma) {
          constexpr int NP = Vec<T>::NP;
          const float2 l2 = make_float2(kLog2e, kLog2e), nl2 = make_float2(nl, nl);
          const float2 kp2 = make_float2(Kp, Kp), ca2 = make_float2(ca, ca), ke2 = make_float2(Ke, Ke);
#pragma unroll
          for (int k = 0; k < (HOLDV > 0 ? HOLDV : 1); ++k) {
            const int j = tid + k * NC;
            float2 q[NP], o[NP];
            Vec<T>::pairs(hold[k], q);
#pragma unroll
            for (int i = 0; i < NP; ++i) {
              const float2 xx = __ffma2_rn(q[i], l2, nl2);
              const float2 pk = make_float2(ex2(xx.x), ex2(xx.y));
              if (ENT) {
                const float2 zc = make_float2(fmaxf(q[i].x, -1e30f), fmaxf(q[i].y, -1e30f));
                o[i] = __fmul2_rn(pk, __ffma2_rn(ca2, zc, ke2));
              } else {
                o[i] = __fmul2_rn(kp2, pk);
              }
            }
            if (j < nv) st_global_16(g_row + j * EPV, Vec<T>::pack_pairs(o));
          }
        } else if (HOLDV > 0) {
#pragma unroll
          for (int k = 0; k < (HOLDV > 0 ? HOLDV : 1); ++k) {
            const int j = tid + k * NC;
            if (j < nv) {
              float v[EPV];
              Vec<T>::unpack(hold[k], v);
              grad_vec(v, j);
            }
          }
        } else {
          for (int j = tid; j < nv; j += NC) {
            float v[EPV];
            Vec<T>::load(buf, j, v);
            grad_vec(v, j);
          }
        }
        if (nv * EPV + tid < n) {
          const float z = tail_z;
          const float pk = ex2(fmaf(z, kLog2e, nl));
          Vec<T>::store_scalar(g_row + nv * EPV + tid, ENT ? pk * fmaf(ca, fmaxf(z, -1e30f), Ke) : Kp * pk);
        }
        // the sampled token's element gets + c g; rewritten by the thread that stored it
        if (rank == owner) {
          const int ia = static_cast<int>(a - s0);
          const int writer = ia < nv * EPV ? (ia / EPV) % NC : (ia - nv * EPV);
          if (tid == writer) {
            const float pk = ex2(fmaf(za, kLog2e, nl));
            const float ga = (ENT ? pk * fmaf(ca, fmaxf(za, -1e30f), Ke) : Kp * pk) + cg;
            Vec<T>::store_scalar(g_row + ia, ga);
          }
        }
      }
      // ---- release the stage (already released after pass 1 when the slice is held in registers)
      if (HOLDV == 0) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[b]);
      }
    }
    if (BWD && rank == 0 && warp == 0) {
      // one partial per cluster (cid < clusters <= rows); the last cluster to finish adds all
      // of them, in a fixed order, into the caller's total, so no second launch is needed
      __syncwarp();
      uint32_t last = 0;
      if (lane == 0) {
        p.row_loss[cid] = cl_loss;
        __threadfence();
        last = atomicAdd(p.done, 1u) == static_cast<uint32_t>(ncl - 1) ? 1u : 0u;
        if (last) __threadfence();
      }
      __syncwarp();
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        double t = 0.0;
        for (int64_t k = lane; k < ncl; k += 32) t += __ldcg(p.row_loss + k);
        t = warp_sum(t);
        if (lane == 0) {
          *p.loss_accum += t;
          *p.done = 0u;
        }
      }
    }
  }
  __syncthreads();
  // no CTA leaves while a peer may still write into its mailbox
  if (C > 1) cluster_sync_all();
}

// ------------------------------------------------------------------ short rows
//
// For rows of at most kSmallRowBytes (V <= 4,096 bf16 or 2,048 fp32) a cluster of CTAs per row
// costs more in set-up and exchange than the row's own data. Here one warp owns a row: its lanes
// hold the row in registers (vector j = lane + 32 k in x[k]), fold it with the same online
// softmax as the cluster kernel, merge the 32 partials by shuffles, and write the gradient from
// registers. Warps take rows w, w + (all warps), ...; each warp adds its rows' loss terms in row
// order, the CTA adds its warps' sums in warp order into one partial, and the last CTA to finish
// (the same workspace counter as the cluster kernel's) adds the CTAs' partials, in order, into
// the caller's total.
constexpr int64_t kSmallRowBytes = 8192;
constexpr int kSmallWarps = 8;

template <typename T, bool ENT>
__global__ void __launch_bounds__(kSmallWarps * 32, 2) small_rows_kernel(const RowArgs p) {
  constexpr int EPV = Vec<T>::N;
  constexpr int NV = static_cast<int>(kSmallRowBytes / 16 / 32);  // 16-byte vectors a lane holds
  __shared__ double warp_loss[kSmallWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t all_warps = static_cast<int64_t>(gridDim.x) * kSmallWarps;
  const int64_t V = p.V, ld = p.ld;
  const int nv = static_cast<int>(V / EPV);  // full vectors of a row
  const uint32_t pad = Vec<T>::kPadWord;
  const T* logits = static_cast<const T*>(p.logits);
  T* grad = static_cast<T*>(p.grad);
  double w_loss = 0.0;  // lane 0: this warp's rows' c l, in row order
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * kSmallWarps + warp; r < p.rows; r += all_warps) {
    // ---- which rows are trained on (the same tests, in the same order, as the cluster kernel).
    // The row's own words are loaded at once; then its owner's coefficient and advantage together
    // with the row's logits (when the row is masked in and its owner in range), so that a row
    // costs two dependent trips to memory before its arithmetic.
    const int32_t a = p.token_ids[r];
    const uint32_t mk = p.mask[r];
    const int32_t i = p.token_traj[r];
    const float old = p.old_logp[r];
    const float ref = p.ref_logp ? p.ref_logp[r] : 0.f;
    const float roll = p.rollout_logp ? p.rollout_logp[r] : 0.f;
    const float A_row = p.adv_per_row ? p.adv[r] : 0.f;
    const bool owner_ok = i >= 0 && i < p.n_traj;
    const bool fetch = mk != 0 && owner_ok;
    const T* row = logits + r * ld;
    auto reload = [&](int k) {
      const int j = lane + k * 32;
      return j < nv ? reinterpret_cast<const uint4*>(row)[j] : make_uint4(pad, pad, pad, pad);
    };
    uint4 x[NV];
    float c = 0.f, A = 0.f;
    if (fetch) {
      c = p.coef[i];
      A = p.adv_per_row ? A_row : p.adv[i];
#pragma unroll
      for (int k = 0; k < NV; ++k) x[k] = reload(k);
    }
    bool active = fetch && c != 0.f;
    if (mk != 0 && !owner_ok && lane == 0) flag_status(p.status, RL_DEV_BAD_TRAJ);
    if (active && (a < 0 || a >= V)) {
      if (lane == 0) flag_status(p.status, RL_DEV_BAD_TOKEN);
      active = false;
    }
    T* g_row = grad + r * ld;
    if (!active) {
      for (int j = lane; j < nv; j += 32) st_global_16(g_row + j * EPV, make_uint4(0u, 0u, 0u, 0u));
      for (int64_t e = static_cast<int64_t>(nv) * EPV + lane; e < V; e += 32) g_row[e] = T(0);
      if (lane == 0 && p.token_stats)
        for (int k = 0; k < 5; ++k) p.token_stats[r * 5 + k] = 0.f;
      continue;
    }
    const float za = Vec<T>::to_f(row[a]);
    // ---- pass 1: the lane's partial, then the warp's (lane 0's merge, broadcast)
    SoftmaxPartial ps{RL_NEG_INF, 0.f, 0.f};
    fold_block<T, ENT>(ps, x, reload);
    float tail_z = 0.f;
    const int64_t te = static_cast<int64_t>(nv) * EPV + lane;  // ragged tail: one element per lane at most
    if (te < V) {
      const float z = Vec<T>::to_f(row[te]);
      tail_z = z;
      if (z != RL_NEG_INF) {
        raise_max<ENT>(ps, z);
        accumulate<ENT>(ps, z, -ps.m * kLog2e);
      }
    }
    SoftmaxPartial q = warp_merge(ps);
    q.m = __shfl_sync(0xffffffffu, q.m, 0);
    q.s = __shfl_sync(0xffffffffu, q.s, 0);
    q.u = __shfl_sync(0xffffffffu, q.u, 0);
    const float lnS = logf(q.s);
    const float lse = q.m + lnS;
    const float H = lnS - q.u / q.s;
    // ---- per-token scalars (every lane computes the same values)
    const float logp = za - lse;
    const float rho = expf((za - old) - lse);  // large operands differenced first
    const float crho = fminf(fmaxf(rho, p.clip_lo), p.clip_hi);
    const float surr = fminf(rho * A, crho * A);
    const bool cut = (A > 0.f && rho > p.clip_hi) || (A < 0.f && rho < p.clip_lo);
    const float w = (p.tis_cap > 0.f && p.rollout_logp) ? fminf(expf(old - roll), p.tis_cap) : 1.f;
    float kl = 0.f, dkl = 0.f;
    if (p.beta != 0.f && p.ref_logp) {
      const float d = (ref - za) + lse;  // r - logp
      const float ed = expf(d);
      kl = ed - d - 1.f;
      dkl = 1.f - ed;
    }
    const float ell = -w * surr + p.beta * kl - p.alpha * H;
    const float g = (cut ? 0.f : -w * A * rho) + p.beta * dkl;
    const float cg = c * g, ca0 = c * p.alpha;
    // p_v = 2^(z_v log2(e) + nl), the rounding of nl folded into the coefficients (as in the
    // cluster kernel)
    const float nl = -lse * kLog2e;
    const float fl = fmaf(fmaf(-lse, kLog2e, -nl), kLn2, 1.f);
    const float Kp = -cg * fl;
    const float ca = ca0 * fl;
    const float Ke = (-cg + ca0 * (H - lse)) * fl;
    if (lane == 0) {
      w_loss += static_cast<double>(c) * static_cast<double>(ell);
      if (p.token_stats) {
        float* st = p.token_stats + r * 5;
        st[0] = logp; st[1] = rho; st[2] = cut ? 1.f : 0.f; st[3] = H; st[4] = kl;
      }
    }
    __syncwarp();  // every lane has read z_a before any lane overwrites it (in-place gradients)
    // ---- pass 2: gradient from the registers
    constexpr int NP = Vec<T>::NP;
    const float2 l2 = make_float2(kLog2e, kLog2e), nl2 = make_float2(nl, nl);
    const float2 kp2 = make_float2(Kp, Kp), ca2 = make_float2(ca, ca), ke2 = make_float2(Ke, Ke);
#pragma unroll
    for (int k = 0; k < NV; ++k) {
      const int j = lane + k * 32;
      float2 qv[NP], o[NP];
      Vec<T>::pairs(x[k], qv);
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        const float2 xx = __ffma2_rn(qv[i], l2, nl2);
        const float2 pk = make_float2(ex2(xx.x), ex2(xx.y));
        if (ENT) {
          const float2 zc = make_float2(fmaxf(qv[i].x, -1e30f), fmaxf(qv[i].y, -1e30f));
          o[i] = __fmul2_rn(pk, __ffma2_rn(ca2, zc, ke2));
        } else {
          o[i] = __fmul2_rn(kp2, pk);
        }
      }
      if (j < nv) st_global_16(g_row + j * EPV, Vec<T>::pack_pairs(o));
    }
    if (te < V) {
      const float pk = ex2(fmaf(tail_z, kLog2e, nl));
      Vec<T>::store_scalar(g_row + te, ENT ? pk * fmaf(ca, fmaxf(tail_z, -1e30f), Ke) : Kp * pk);
    }
    // the sampled token's element gets + c g; rewritten by the lane that stored it
    const int writer = a < nv * EPV ? (a / EPV) % 32 : (a - nv * EPV);
    if (lane == writer) {
      const float pk = ex2(fmaf(za, kLog2e, nl));
      Vec<T>::store_scalar(g_row + a, (ENT ? pk * fmaf(ca, fmaxf(za, -1e30f), Ke) : Kp * pk) + cg);
    }
  }
  // ---- the loss: warps in order into one partial per CTA; the last CTA adds the partials, all
  // its threads loading them at once (thread k takes partials k, k + 256, ...), then combined
  // by shuffles and the warps in order: a fixed order for a given grid
  __shared__ uint32_t is_last;
  if (lane == 0) warp_loss[warp] = w_loss;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int k = 0; k < kSmallWarps; ++k) t += warp_loss[k];
    p.row_loss[blockIdx.x] = t;
    __threadfence();
    is_last = atomicAdd(p.done, 1u) == gridDim.x - 1 ? 1u : 0u;
  }
  __syncthreads();
  if (is_last) {
    __threadfence();
    double t = 0.0;
    for (unsigned k = threadIdx.x; k < gridDim.x; k += kSmallWarps * 32) t += __ldcg(p.row_loss + k);
    t = warp_sum(t);
    if (lane == 0) warp_loss[warp] = t;
    __syncthreads();
    if (threadIdx.x == 0) {
      double sum = 0.0;
      for (int k = 0; k < kSmallWarps; ++k) sum += warp_loss[k];
      *p.loss_accum += sum;
      *p.done = 0u;
    }
  }
}

// ------------------------------------------------------------------ forward-only stream
//
// rl_token_logprobs reads each row exactly once and keeps nothing on chip, so it
// needs no cluster: one CTA owns a row at a time (persistent over rows). A
// producer warp streams the CTA's rows as back-to-back chunks through a ring of
// shared-memory stages (bulk copies, full / empty mbarriers); consumer warps fold
// each chunk into per-thread online-softmax partials and, at the end of a row,
// merge them (one named barrier among the consumers per row).
// Stages and chunk size per form, chosen by a sweep on the benchmark batch (bf16, V = 151,936):
// without the entropy 3 x 16 KB (3 CTAs per SM, bound by registers) ran in 6.54 ms per batch
// against 6.80 with 6 x 16 KB (2 CTAs per SM, bound by shared memory); with the entropy
// 4 x 12 KB ran in 7.19 against 7.27 ms (3 x 16 KB: 7.55).
template <bool ENT>
struct FwdCfg {
  static constexpr int kStages = ENT ? 4 : 3;
  static constexpr int kChunkKB = ENT ? 12 : 16;
};

struct StreamArgs {
  const void* logits;
  int64_t rows, V, ld;
  const int32_t* token_ids;
  float* logp_out;
  float* entropy_out;
  float* lse_out;
  int32_t* status;
  int64_t chunk;      // elements per chunk (a multiple of the 16-byte vector)
  int64_t buf_elems;  // element stride between stages
  int32_t tma;        // rows 16-byte aligned
};

struct ChunkInfo {
  int64_t r;      // row, -1 = end of stream
  int32_t first;  // first element of the chunk within the row
  int32_t count;  // elements in the chunk
};

template <typename T, int NW, bool ENT>
__global__ void __launch_bounds__((NW + 1) * 32, 2) stream_logprobs_kernel(const StreamArgs p) {
  constexpr int EPV = Vec<T>::N;
  constexpr int NS = FwdCfg<ENT>::kStages;
  constexpr int NC = NW * 32;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[NS], empty_bar[NS];
  __shared__ ChunkInfo info[NS];
  __shared__ SoftmaxPartial red[2][NW];

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t rows = p.rows, V = p.V, ld = p.ld, CH = p.chunk;
  const int64_t nchunk = (V + CH - 1) / CH;
  const T* logits = static_cast<const T*>(p.logits);
  T* const buf_base = reinterpret_cast<T*>(smem_raw);

  if (tid == 0) {
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      mbar_init(&full_bar[k], 1);
      mbar_init(&empty_bar[k], NW);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == NW) {
    // =============================================================== producer warp
    uint32_t q = 0;
    bool failed = false;
    for (int64_t r = blockIdx.x; r < rows && !failed; r += gridDim.x) {
      for (int64_t k = 0; k < nchunk; ++k, ++q) {
        const int st = q % NS;
        const uint32_t use = q / NS;
        if (use > 0 && !mbar_wait_bounded(&empty_bar[st], (use - 1) & 1)) {
          failed = true;
          if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
          break;
        }
        const int64_t first = k * CH;
        const int64_t cnt = (first + CH < V ? first + CH : V) - first;
        const int cv = p.tma ? static_cast<int>(cnt / EPV) : 0;
        T* buf = buf_base + st * p.buf_elems;
        const T* src = logits + r * ld + first;
        for (int e = cv * EPV + lane; e < static_cast<int>(cnt); e += 32) buf[e] = src[e];
        __syncwarp();
        if (lane == 0) {
          info[st] = ChunkInfo{r, static_cast<int32_t>(first), static_cast<int32_t>(cnt)};
          if (cv > 0) {
            mbar_arrive_expect_tx(&full_bar[st], static_cast<uint32_t>(cv * 16));
            bulk_g2s(buf, src, static_cast<uint32_t>(cv * 16), &full_bar[st]);
          } else {
            mbar_arrive(&full_bar[st]);
          }
        }
      }
    }
    if (!failed) {
      const int st = q % NS;
      const uint32_t use = q / NS;
      if (use > 0 && !mbar_wait_bounded(&empty_bar[st], (use - 1) & 1)) {
        if (lane == 0) flag_status(p.status, RL_DEV_TIMEOUT);
      } else if (lane == 0) {
        info[st].r = -1;
        mbar_arrive(&full_bar[st]);
      }
    }
  } else {
    // =============================================================== consumer warps
    SoftmaxPartial ps{RL_NEG_INF, 0.f, 0.f};
    uint32_t row_it = 0;
    for (uint32_t q = 0;; ++q) {
      const int st = q % NS;
      if (!mbar_wait_bounded(&full_bar[st], (q / NS) & 1)) {
        if (tid == 0) flag_status(p.status, RL_DEV_TIMEOUT);
        break;
      }
      const ChunkInfo ci = info[st];
      if (ci.r < 0) break;
      const T* buf = buf_base + st * p.buf_elems;
      const int cv = ci.count / EPV;
      {
        constexpr int KV = (FwdCfg<ENT>::kChunkKB * 1024 / 16 + NC - 1) / NC;  // vectors per thread per chunk
        uint4 x[KV];
        const uint32_t pad = Vec<T>::kPadWord;
        auto reload = [&](int k) {
          const int j = tid + k * NC;
          return j < cv ? reinterpret_cast<const uint4*>(buf)[j] : make_uint4(pad, pad, pad, pad);
        };
#pragma unroll
        for (int k = 0; k < KV; ++k) x[k] = reload(k);
        fold_block<T, ENT>(ps, x, reload);
      }
      if (cv * EPV + tid < ci.count) {
        const float z = Vec<T>::to_f(buf[cv * EPV + tid]);
        if (z != RL_NEG_INF) {
          raise_max<ENT>(ps, z);
          accumulate<ENT>(ps, z, -ps.m * kLog2e);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[st]);
      if (ci.first + ci.count == V) {
        // ---- end of row ci.r: merge the consumers' partials
        const int par = row_it & 1;
        ps = warp_merge(ps);
        if (lane == 0) red[par][warp] = ps;
        asm volatile("bar.sync 1, %0;" :: "n"(NC) : "memory");
        if (warp == 0) {
          SoftmaxPartial qq = lane < NW ? red[par][lane] : SoftmaxPartial{RL_NEG_INF, 0.f, 0.f};
          qq = warp_merge(qq);
          if (lane == 0) {
            const int64_t r = ci.r;
            const float lnS = logf(qq.s);
            const float lse = qq.m + lnS;
            const int32_t a = p.token_ids[r];
            const bool a_ok = a >= 0 && a < V;
            if (!a_ok) flag_status(p.status, RL_DEV_BAD_TOKEN);
            const float za = a_ok ? Vec<T>::to_f(logits[r * ld + a]) : 0.f;
            p.logp_out[r] = a_ok ? za - lse : __int_as_float(0x7fc00000);
            if (p.entropy_out) p.entropy_out[r] = lnS - qq.u / qq.s;
            if (p.lse_out) p.lse_out[r] = lse;
          }
        }
        ps = SoftmaxPartial{RL_NEG_INF, 0.f, 0.f};
        ++row_it;
      }
    }
  }
}

// ------------------------------------------------------------------ host side

constexpr int64_t kMaxSliceBytes = 100 * 1024;

struct Plan {
  int C;
  int64_t slice, buf_elems;
  size_t smem;
};

// Smallest cluster whose slices are at most target_bytes (or, at 16 CTAs, at most 100 KB).
static bool make_plan(int64_t V, int es, Plan* out, int64_t target_bytes = 40 * 1024) {
  const int64_t epv = 16 / es;
  for (int C = 1; C <= 16; ++C) {
    const int64_t per = (V + C - 1) / C;
    const int64_t slice = (per + epv - 1) / epv * epv;
    if (slice * es <= target_bytes || (C == 16 && slice * es <= kMaxSliceBytes)) {
      const int64_t stride_bytes = (slice * es + 127) / 128 * 128;
      out->C = C;
      out->slice = slice;
      out->buf_elems = stride_bytes / es;
      out->smem = static_cast<size_t>(RL_STAGES * stride_bytes);
      return true;
    }
  }
  return false;
}

// Configure a kernel once per (kernel, device): dynamic shared memory up to the
// largest request so far, and non-portable cluster sizes allowed.
static rl_status configure(const void* kern, int dev, size_t smem) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, size_t> smem_attr;
  std::lock_guard<std::mutex> lock(mu);
  auto ka = std::make_pair(kern, dev);
  auto ita = smem_attr.find(ka);
  if (ita == smem_attr.end() || ita->second < smem) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(max dynamic smem)");
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(non-portable cluster)");
    smem_attr[ka] = smem;
  }
  return RL_OK;
}

template <typename T, int NW, bool ENT, int HOLDV, int MINB>
static rl_status launch_rows(const RowArgs& args, const Plan& plan, cudaStream_t s, int64_t* n_clusters_out) {
  auto kern = rows_kernel<T, NW, ENT, true, HOLDV, MINB>;
  constexpr int kRowThreads = (NW + 1) * 32;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  rl_status st = configure(reinterpret_cast<const void*>(kern), dev, plan.smem);
  if (st != RL_OK) return st;

  static std::mutex mu;
  static std::map<std::tuple<const void*, int, int, size_t>, int> cache;
  int max_clusters = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    auto key = std::make_tuple(reinterpret_cast<const void*>(kern), dev, plan.C, plan.smem);
    auto itc = cache.find(key);
    if (itc != cache.end()) {
      max_clusters = itc->second;
    } else {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = plan.C;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(plan.C * 1024, 1, 1);
      cfg.blockDim = dim3(kRowThreads, 1, 1);
      cfg.dynamicSmemBytes = plan.smem;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      e = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
      if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveClusters");
      if (max_clusters <= 0) return set_error(RL_ERR_UNSUPPORTED, "no cluster of this shape fits on the device");
      cache[key] = max_clusters;
    }
  }
  const int64_t n_clusters = std::max<int64_t>(1, std::min<int64_t>(max_clusters, args.rows));
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = plan.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(n_clusters * plan.C), 1, 1);
  cfg.blockDim = dim3(kRowThreads, 1, 1);
  cfg.dynamicSmemBytes = plan.smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, args);
  if (e != cudaSuccess) return cuda_error(e, "cudaLaunchKernelEx(rows_kernel)");
  if (n_clusters_out) *n_clusters_out = n_clusters;
  return RL_OK;
}

// Shape of the loss kernel per path, from sweeps on the GB300 (full-size microbatches):
//   bf16 without the entropy (the benchmark): 8 consumer warps holding up to 10 vectors each,
//     slices up to 40 KB (clusters of 8 at V = 151,936), 2 CTAs per SM: 12.84 ms per benchmark
//     step against 12.96 with 7 warps of 11 vectors; wider clusters or 3 CTAs per SM were
//     slower (13.6-18.5 ms);
//   bf16 with the entropy: the same 8 warps of 10 vectors: 2.72 ms per 32,768-row long-horizon
//     microbatch, against 2.73 with 7 warps of 11 and 3.16 with 11 warps of 7;
//   fp32: slices up to 30 KB (clusters of 5 at V = 32,000), 7 warps of up to 9 vectors, 3 CTAs
//     per SM: 4.15 ms per 131,072-row edge batch against 4.35 with clusters of 4 at 2 per SM.
#ifndef RL_ENT_NW
#define RL_ENT_NW 8
#endif
#ifndef RL_ENT_HOLD
#define RL_ENT_HOLD 10
#endif
template <typename T>
struct LossShape;
template <>
struct LossShape<uint16_t> {
  static constexpr int64_t kSliceBytes[2] = {40 * 1024, 40 * 1024};  // [entropy off, on]
};
template <>
struct LossShape<float> {
  static constexpr int64_t kSliceBytes[2] = {30 * 1024, 30 * 1024};
};

// The plan of the loss kernel for this path (the forward-only kernel has no clusters); false
// if no cluster of at most 16 CTAs of 100 KB holds the row (the callers check that first).
template <typename T>
static bool loss_plan(int64_t V, bool ent, Plan* plan) {
  return make_plan(V, static_cast<int>(sizeof(T)), plan, LossShape<T>::kSliceBytes[ent ? 1 : 0]) ||
         make_plan(V, static_cast<int>(sizeof(T)), plan);
}

// Launches the loss kernel; *n_clusters receives the number of clusters, each of which leaves
// one loss partial at the head of the per-row loss area (the last one also adds them up).
// Registers hold the slice when it fits the path's held vectors; otherwise the slice stays in
// shared memory (7 warps, 2 CTAs per SM, slices up to 40 KB).
// Launches the short-row kernel: as many CTAs as fit on the GPU at once, at most one warp per row.
template <typename T, bool ENT>
static rl_status launch_small(const RowArgs& args, cudaStream_t s) {
  auto kern = small_rows_kernel<T, ENT>;
  constexpr int kThreads = kSmallWarps * 32;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int64_t> grid_cache;
  int64_t grid = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    auto key = std::make_pair(reinterpret_cast<const void*>(kern), dev);
    auto it = grid_cache.find(key);
    if (it != grid_cache.end()) {
      grid = it->second;
    } else {
      int per_sm = 0, sms = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
      if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
      e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
      if (per_sm <= 0) return set_error(RL_ERR_UNSUPPORTED, "small_rows_kernel does not fit on an SM");
      grid = static_cast<int64_t>(per_sm) * sms;
      grid_cache[key] = grid;
    }
  }
  const int64_t blocks = std::min<int64_t>(grid, (args.rows + kSmallWarps - 1) / kSmallWarps);
  kern<<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(args);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "small_rows_kernel launch");
  return RL_OK;
}

template <typename T>
static rl_status dispatch_loss(bool ent, RowArgs args, int64_t V, cudaStream_t s, int64_t* n_clusters) {
  // rows of at most 8 KB (16-byte aligned): a warp per row
  if (args.tma && V * static_cast<int64_t>(sizeof(T)) <= kSmallRowBytes) {
    *n_clusters = 0;
    return ent ? launch_small<T, true>(args, s) : launch_small<T, false>(args, s);
  }
  auto run = [&](const Plan& plan, auto launcher) {
    args.slice = plan.slice;
    args.buf_elems = plan.buf_elems;
    return launcher(args, plan, s, n_clusters);
  };
  Plan plan = {};
  if (!loss_plan<T>(V, ent, &plan)) return set_error(RL_ERR_UNSUPPORTED, "rl_policy_loss_fwd_bwd: row too large");
  const int64_t vecs_per_slice = plan.slice * static_cast<int64_t>(sizeof(T)) / 16;
  if constexpr (sizeof(T) == 2) {
    if (!ent && vecs_per_slice <= 10 * 8 * 32) return run(plan, launch_rows<T, 8, false, 10, 2>);
    if (ent && vecs_per_slice <= RL_ENT_HOLD * RL_ENT_NW * 32)
      return run(plan, launch_rows<T, RL_ENT_NW, true, RL_ENT_HOLD, 2>);
  } else {
    if (vecs_per_slice <= 9 * 7 * 32)
      return ent ? run(plan, launch_rows<T, 7, true, 9, 3>) : run(plan, launch_rows<T, 7, false, 9, 3>);
  }
  Plan big = {};
  if (!make_plan(V, static_cast<int>(sizeof(T)), &big))
    return set_error(RL_ERR_UNSUPPORTED, "rl_policy_loss_fwd_bwd: row too large");
  return ent ? run(big, launch_rows<T, 7, true, 0, 2>) : run(big, launch_rows<T, 7, false, 0, 2>);
}

constexpr int kFwdWarps = 8;

template <typename T, bool ENT>
static rl_status launch_stream(StreamArgs args, cudaStream_t s) {
  auto kern = stream_logprobs_kernel<T, kFwdWarps, ENT>;
  args.chunk = static_cast<int64_t>(FwdCfg<ENT>::kChunkKB) * 1024 / static_cast<int64_t>(sizeof(T));
  args.buf_elems = args.chunk;  // chunk bytes are a multiple of 128
  const size_t smem = static_cast<size_t>(FwdCfg<ENT>::kStages) * args.buf_elems * sizeof(T);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  rl_status st = configure(reinterpret_cast<const void*>(kern), dev, smem);
  if (st != RL_OK) return st;
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> grid_cache;
  int grid = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    auto key = std::make_pair(reinterpret_cast<const void*>(kern), dev);
    auto it = grid_cache.find(key);
    if (it != grid_cache.end()) {
      grid = it->second;
    } else {
      int per_sm = 0, sms = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, (kFwdWarps + 1) * 32, smem);
      if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
      e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
      if (per_sm <= 0) return set_error(RL_ERR_UNSUPPORTED, "stream kernel does not fit on an SM");
      grid = per_sm * sms;
      grid_cache[key] = grid;
    }
  }
  const unsigned blocks = static_cast<unsigned>(std::min<int64_t>(grid, args.rows));
  kern<<<blocks, (kFwdWarps + 1) * 32, smem, s>>>(args);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "stream_logprobs_kernel launch");
  return RL_OK;
}

static rl_status check_rows_args(const char* fn, const void* logits, rl_dtype dt, int64_t rows, int64_t V,
                                 int64_t ld, const void* ws, size_t ws_bytes, Plan* plan, int* es) {
  if (dt != RL_BF16 && dt != RL_F32) return set_error(RL_ERR_INVALID_ARG, std::string(fn) + ": unknown dtype");
  if (rows < 0 || V < 1 || ld < V)
    return set_error(RL_ERR_INVALID_ARG, std::string(fn) + ": need rows >= 0, V >= 1, ld >= V");
  if (!ws) return set_error(RL_ERR_INVALID_ARG, std::string(fn) + ": ws is NULL");
  if (ws_bytes < rl_workspace_size(rows, V, 0))
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL, std::string(fn) + ": workspace smaller than rl_workspace_size(rows, V, 0)");
  if (!aligned16(ws)) return set_error(RL_ERR_ALIGNMENT, std::string(fn) + ": ws not 16-byte aligned");
  if (rows > 0 && !logits) return set_error(RL_ERR_INVALID_ARG, std::string(fn) + ": logits is NULL");
  if (logits && !aligned16(logits)) return set_error(RL_ERR_ALIGNMENT, std::string(fn) + ": logits not 16-byte aligned");
  if (V > INT32_MAX) return set_error(RL_ERR_UNSUPPORTED, std::string(fn) + ": V above 2^31 - 1");
  *es = dt == RL_BF16 ? 2 : 4;
  if (!make_plan(V, *es, plan))
    return set_error(RL_ERR_UNSUPPORTED, std::string(fn) + ": vocabulary row larger than 16 x 100 KB");
  return RL_OK;
}

}  // namespace rl

extern "C" rl_status rl_token_logprobs(const void* logits, rl_dtype dtype, int64_t rows, int64_t V, int64_t ld,
                                       const int32_t* token_ids, float* logp_out, float* entropy_out,
                                       float* lse_out, void* ws, size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  Plan plan;
  int es = 0;
  rl_status st = check_rows_args("rl_token_logprobs", logits, dtype, rows, V, ld, ws, ws_bytes, &plan, &es);
  if (st != RL_OK) return st;
  if (rows == 0) return RL_OK;
  if (!token_ids || !logp_out) return set_error(RL_ERR_INVALID_ARG, "rl_token_logprobs: NULL array argument");
  StreamArgs a = {};
  a.logits = logits;
  a.rows = rows;
  a.V = V;
  a.ld = ld;
  a.token_ids = token_ids;
  a.logp_out = logp_out;
  a.entropy_out = entropy_out;
  a.lse_out = lse_out;
  a.status = reinterpret_cast<int32_t*>(ws);
  a.tma = ((ld * es) % 16) == 0;  // chunk and buf_elems are set per form by launch_stream
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (dtype == RL_BF16)
    return entropy_out ? launch_stream<uint16_t, true>(a, s) : launch_stream<uint16_t, false>(a, s);
  return entropy_out ? launch_stream<float, true>(a, s) : launch_stream<float, false>(a, s);
}

extern "C" rl_status rl_policy_loss_fwd_bwd(const void* logits, rl_dtype dtype, int64_t rows, int64_t V,
                                            int64_t ld, const int32_t* token_ids, const uint8_t* mask,
                                            const int32_t* token_traj, int32_t n_traj, const float* adv,
                                            const float* coef, const float* old_logp, const float* ref_logp,
                                            const float* rollout_logp, const rl_loss_params* params,
                                            void* grad_out, double* loss_accum, float* token_stats, void* ws,
                                            size_t ws_bytes, rl_stream_t stream) {
  using namespace rl;
  clear_error();
  Plan plan;
  int es = 0;
  rl_status st = check_rows_args("rl_policy_loss_fwd_bwd", logits, dtype, rows, V, ld, ws, ws_bytes, &plan, &es);
  if (st != RL_OK) return st;
  if (!params) return set_error(RL_ERR_INVALID_ARG, "rl_policy_loss_fwd_bwd: params is NULL");
  if (!(params->clip_eps_low >= 0.f) || !(params->clip_eps_high >= 0.f))
    return set_error(RL_ERR_INVALID_ARG, "rl_policy_loss_fwd_bwd: clip eps must be >= 0");
  if (params->kl_estimator != 0 && params->kl_estimator != 3)
    return set_error(RL_ERR_UNSUPPORTED, "rl_policy_loss_fwd_bwd: kl_estimator must be 0 or 3");
  if (!loss_accum) return set_error(RL_ERR_INVALID_ARG, "rl_policy_loss_fwd_bwd: loss_accum is NULL");
  if (n_traj < 0) return set_error(RL_ERR_INVALID_ARG, "rl_policy_loss_fwd_bwd: n_traj < 0");
  if (rows == 0) return RL_OK;
  if (!token_ids || !mask || !token_traj || !old_logp || !grad_out || (n_traj > 0 && (!adv || !coef)) ||
      (params->token_level_adv && !adv))
    return set_error(RL_ERR_INVALID_ARG, "rl_policy_loss_fwd_bwd: NULL array argument");
  if (params->token_level_adv != 0 && params->token_level_adv != 1)
    return set_error(RL_ERR_INVALID_ARG, "rl_policy_loss_fwd_bwd: token_level_adv must be 0 or 1");
  if (!aligned16(grad_out)) return set_error(RL_ERR_ALIGNMENT, "rl_policy_loss_fwd_bwd: grad_out not 16-byte aligned");
  const bool kl_on = params->kl_estimator == 3 && params->kl_coef != 0.f && ref_logp != nullptr;
  RowArgs a = {};
  a.logits = logits;
  a.grad = grad_out;
  a.rows = rows;
  a.V = V;
  a.ld = ld;
  a.token_ids = token_ids;
  a.mask = mask;
  a.token_traj = token_traj;
  a.n_traj = n_traj;
  a.adv = adv;
  a.coef = coef;
  a.old_logp = old_logp;
  a.ref_logp = kl_on ? ref_logp : nullptr;
  a.rollout_logp = rollout_logp;
  a.clip_lo = 1.f - params->clip_eps_low;
  a.clip_hi = 1.f + params->clip_eps_high;
  a.beta = kl_on ? params->kl_coef : 0.f;
  a.alpha = params->entropy_coef;
  a.tis_cap = rollout_logp ? params->tis_cap : 0.f;
  a.adv_per_row = params->token_level_adv;
  double* row_loss = reinterpret_cast<double*>(static_cast<char*>(ws) + ws_row_loss_offset());
  a.row_loss = row_loss;
  a.loss_accum = loss_accum;
  a.done = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + kWsDoneOffset);
  a.token_stats = token_stats;
  a.status = reinterpret_cast<int32_t*>(ws);
  a.tma = ((ld * es) % 16) == 0;
  const bool ent = params->entropy_coef != 0.f || token_stats != nullptr;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int64_t n_clusters = 0;
  st = dtype == RL_BF16 ? dispatch_loss<uint16_t>(ent, a, V, s, &n_clusters)
                        : dispatch_loss<float>(ent, a, V, s, &n_clusters);
  return st;  // the kernel's last cluster has added the loss into loss_accum
}
