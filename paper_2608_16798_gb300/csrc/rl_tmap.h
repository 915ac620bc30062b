// Host-side encoding of 2-D TMA tensor maps (cuTensorMapEncodeTiled, fetched from the
// driver at run time so that the library links only the CUDA runtime).
#pragma once

#include <cstdint>

#include <cuda.h>

#include "rl_loss.h"

namespace rl {

// Row-major matrix of `rows` rows of `inner` elements of `dtype`, consecutive rows
// `row_stride_bytes` apart (a multiple of 16, at least inner x element size), cut into
// boxes of box_rows x box_inner elements with the given shared-memory swizzle. Loads past
// the matrix read zeros; stores and reductions past it are dropped.
rl_status tmap_2d(CUtensorMap* map, CUtensorMapDataType dtype, const void* base, int64_t inner, int64_t rows,
                  int64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle swizzle);

}  // namespace rl
