// tmap.cuh -- host-side construction of TMA tensor maps (bf16 with 128-byte swizzle or none; fp32).
#pragma once
#include <cuda.h>
#include <stdint.h>

namespace bla {

// Encode a tiled bf16 tensor map of rank 2..5.  dims[0] is the innermost (contiguous)
// extent; strides_bytes[i] is the byte stride of dimension i+1.  With swizzle128, box[0] is 64
// (128 bytes, the swizzle span) and shared memory holds the 128-byte-swizzled layout; without, box[0]
// is a multiple of 8 (16 bytes) and the box lands densely, row after row.  Out-of-bounds box
// elements read as zero.
// Returns false if the driver entry point is unavailable or the encode fails.
bool make_tmap_bf16(CUtensorMap *map, const void *base, int rank, const uint64_t *dims,
                    const uint64_t *strides_bytes, const uint32_t *box, bool swizzle128 = true);
// The same for fp32 tensors, 128-byte swizzle: box[0] is 32 (128 bytes).
bool make_tmap_f32(CUtensorMap *map, const void *base, int rank, const uint64_t *dims,
                   const uint64_t *strides_bytes, const uint32_t *box);

}  // namespace bla
