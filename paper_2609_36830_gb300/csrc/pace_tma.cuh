// 2-D bf16 TMA tensor maps shared by the tensor-core kernels.
#pragma once

#include <cuda.h>

#include "pace_internal.cuh"

namespace pace {

// bf16 matrix [rows][cols], row stride ld elements (ld * 2 a multiple of 16
// bytes), boxes of box_inner x box_outer elements with the 128-byte swizzle
// (box_inner * 2 <= 128).  Out-of-range box elements load as zeros.  Returns
// PACE_ERR_UNSUPPORTED_SHAPE when the driver rejects the map, PACE_ERR_CUDA
// when its entry point is unavailable.
pace_status encode_bf16_2d(CUtensorMap* tm, const void* ptr, int64_t rows, int64_t cols,
                           int64_t ld, int box_inner, int box_outer);

}  // namespace pace
