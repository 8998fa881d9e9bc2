// Host helper: encode a bf16 TMA tensor map with 128-byte swizzle.
#pragma once
#include <cstdint>

#include <cuda.h>

#include "../../include/cachedsearch.h"

namespace cs {
// dims[0] is the innermost (contiguous) extent; strides_bytes[i] is the byte stride of
// dimension i+1; box[i] the tile extent copied per load (box[0] * 2 bytes <= 128).
cs_status make_tmap_bf16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                         const uint64_t* strides_bytes, const uint32_t* box);
// Same for a bf16 (f32 = false) or float32 (f32 = true) tensor; box[0] * element size <= 128.
cs_status make_tmap(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                    const uint64_t* strides_bytes, const uint32_t* box, bool f32);
}  // namespace cs
