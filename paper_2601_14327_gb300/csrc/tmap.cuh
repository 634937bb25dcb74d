// TMA tensor-map (descriptor) encoding shared by the tensor-core kernels.
#pragma once

#include <cuda.h>
#include <stdint.h>

namespace moe {

// Tensor map of a bf16 row-major [rows, cols] matrix whose tiles are box_cols
// (inner, contiguous) x box_rows elements, with the given shared-memory swizzle.
// Elements outside the matrix read as zero. Returns MOE_OK or an error status
// (recorded for moe_last_error_string).
int make_map(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_cols,
             uint32_t box_rows, const char *what,
             CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B);

}  // namespace moe
