// Host-side TMA tensor-map encoding shared by the tensor-core kernels.
#pragma once

#include <cuda.h>

#include <cstdint>

namespace xs {

// Row-major [outer, inner] matrix of `dtype`, boxes of box_inner x box_outer
// elements, the given swizzle, out-of-range elements read as zero.  Returns
// false if the driver entry point is unavailable or rejects the arguments.
bool encode_tmap_2d(CUtensorMap *m, CUtensorMapDataType dtype, uint32_t elem_bytes,
                    const void *base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                    uint32_t box_outer, CUtensorMapSwizzle swizzle);

}  // namespace xs
