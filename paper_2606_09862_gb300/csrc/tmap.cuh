// tmap.cuh -- host-side construction of TMA tensor maps (bf16, 128-byte swizzle).
#pragma once
#include <cuda.h>
#include <stdint.h>

namespace bla {

// Encode a tiled bf16 tensor map of rank 2..5.  dims[0] is the innermost (contiguous)
// extent; strides_bytes[i] is the byte stride of dimension i+1; box[0] must be 64
// (128 bytes, the swizzle span).  Out-of-bounds box elements read as zero.
// Returns false if the driver entry point is unavailable or the encode fails.
bool make_tmap_bf16(CUtensorMap *map, const void *base, int rank, const uint64_t *dims,
                    const uint64_t *strides_bytes, const uint32_t *box);

}  // namespace bla
