// Host-side encoding of TMA tensor maps (shared by the dense-product and attention kernels).
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace jagg {

// Tiled tensor map of `rank` dimensions (innermost first): dims[i] elements, strides[i]
// bytes between consecutive indices of dimension i + 1 (rank - 1 entries, multiples of 16),
// boxes of box[i] elements, bf16 or f32 elements, the given shared-memory swizzle; parts
// of a box outside the tensor read as zero and are not written.
int encode_tmap(CUtensorMap* m, bool f32, int rank, const void* base, const uint64_t* dims, const uint64_t* strides,
                const uint32_t* box, CUtensorMapSwizzle swz);

}  // namespace jagg
