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
// Work-item counter of the fused head's backward products (zeroed before each launch).
constexpr size_t kWsHeadCounterOffset = 24;

rl_status set_error(rl_status st, const std::string& msg);
rl_status cuda_error(cudaError_t e, const char* what);
void clear_error();

// Fixed-order sum of `rows` loss contributions into *loss_accum (rl_stats.cu).
rl_status launch_reduce_loss(const double* row_loss, int64_t rows, double* loss_accum, cudaStream_t s);
// Smallest workspace of the fused LM head for up to max_rows tokens (rl_head.cu).
size_t head_workspace_bytes(int64_t max_rows, int64_t V, int64_t D);
// The same, keeping the dZ of up to group_tokens tokens (whole chunks) at once.
size_t head_workspace_bytes_grouped(int64_t max_rows, int64_t V, int64_t D, int64_t group_tokens);

// Backward products of the fused LM head on the tensor cores (rl_head_grad.cu), one launch:
// d_hidden[n x D] = dZ W (stored, bf16 or fp32) and d_weight[V x D] += dZ^T H[n x D] (fp32),
// with dz the bf16 gradient of the logits of the n tokens ([n x V], rows ldz elements apart).
// counter: a workspace word for the work-item counter (zeroed here, on the stream).
rl_status head_grad(const uint16_t* dz, int64_t ldz, int64_t n, int64_t V, const void* weight, const void* hidden,
                    int64_t D, void* d_hidden, rl_dtype dh_dtype, float* d_weight, uint32_t* counter,
                    int32_t* status, cudaStream_t s);

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace rl
