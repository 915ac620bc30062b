// Host-side internals shared by the library's translation units.
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>

#include <cuda_runtime.h>

#include "rl_loss.h"

namespace rl {

// Workspace layout (offsets in bytes from the caller's workspace pointer):
//   [0, 256)                 header: int32 device status word at offset 0
//   [256, 256 + 8 * rows)    double loss contributions: one per cluster of the logits-path
//                            loss kernel (its rows' c_i * l_t added in row order), one per
//                            row for the fused head and the value loss
constexpr size_t kWsHeader = 256;

inline size_t ws_row_loss_offset() { return kWsHeader; }
// Header word counting the loss kernel's finished clusters (zeroed by rl_workspace_init; the
// last cluster of each launch resets it).
constexpr size_t kWsDoneOffset = 16;
// The same for the value loss kernel's finished CTAs.
constexpr size_t kWsValueDoneOffset = 20;

rl_status set_error(rl_status st, const std::string& msg);
rl_status cuda_error(cudaError_t e, const char* what);
void clear_error();

// Fixed-order sum of `rows` loss contributions into *loss_accum (rl_stats.cu).
rl_status launch_reduce_loss(const double* row_loss, int64_t rows, double* loss_accum, cudaStream_t s);
// Smallest workspace of the fused LM head for up to max_rows tokens (rl_head.cu).
size_t head_workspace_bytes(int64_t max_rows, int64_t V, int64_t D);
// The same, keeping the dZ of up to group_tokens tokens (whole chunks) at once.
size_t head_workspace_bytes_grouped(int64_t max_rows, int64_t V, int64_t D, int64_t group_tokens);

// Backward products of the fused LM head on the tensor cores (rl_head_grad.cu). dz is the
// bf16 gradient of the logits of n tokens ([n x V], rows ldz elements apart).
// out_kind: 0 = add into fp32 (TMA reduce-add), 1 = store fp32, 2 = store bf16.
// dH[n x D] = dZ W; with ksplit = 2 the contraction over V is cut in two halves that are
// both added (out_kind 0) into a zeroed fp32 destination.
rl_status head_grad_dh(const uint16_t* dz, int64_t ldz, int64_t n, int64_t V, const void* weight, int64_t D,
                       void* out, int out_kind, int ksplit, int32_t* status, cudaStream_t s);
// dW[V x D] += dZ^T H[n x D] (fp32, one addition per element).
rl_status head_grad_dw(const uint16_t* dz, int64_t ldz, int64_t n, int64_t V, const void* hidden, int64_t D,
                       float* d_weight, int32_t* status, cudaStream_t s);
// 2 if splitting dH's contraction in two balances the CTA pairs' work better, else 1.
int head_grad_dh_split(int64_t n, int64_t V, int64_t D);

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace rl
