// lla_tmap.h -- host side of TMA tensor maps: cuTensorMapEncodeTiled, reached through the
// runtime's driver entry point (the library links no driver stub).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace lla {

// Encodes a tiled bf16 tensor map (no interleave; out-of-range elements read as zero; with
// swizzle128 the box's 128-byte rows land in shared memory with the 128-byte swizzle).  dims / strides_bytes / box give rank entries (strides: rank - 1 entries).  Returns
// false when the driver refuses the map.
bool encode_tmap_bf16(CUtensorMap *map, const void *base, int rank, const uint64_t *dims,
                      const uint64_t *strides_bytes, const uint32_t *box, bool swizzle128 = false);

}  // namespace lla
