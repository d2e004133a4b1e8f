// tmap.cuh - host-side creation of TMA tensor maps through the driver entry
// point (no link-time dependency on libcuda).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace cover {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// Returns nullptr if the driver does not provide cuTensorMapEncodeTiled.
EncodeTiledFn encode_tiled_fn();

// bf16 tensor viewed as 4-D (d0 fastest) with 128-byte swizzle and a box of
// {64, box1, 1, 1} elements; out-of-range elements read as zero.
bool make_bf16_map_4d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t d3,
                      uint32_t box1);

}  // namespace cover
