// TMA tensor maps for the tensor-core kernels (internal).
#pragma once

#include <cuda.h>

#include <cstdint>

namespace mosa {

// True when the driver's tensor-map encoder can be reached.
bool tmap_available();

// A bf16 tensor map with 128-byte swizzle, zero fill outside the tensor and
// 256-byte L2 promotion.  dims / box innermost first; strides in bytes for
// dims 1..rank-1.  The encoded map is a pure function of these arguments, so
// results are cached and reused across calls.  False if encoding fails.
bool tmap_bf16(CUtensorMap *out, const void *base, int rank, const uint64_t *dims,
               const uint64_t *strides, const uint32_t *box);
// The same for fp32 elements (the box's innermost extent then at most 32).
bool tmap_f32(CUtensorMap *out, const void *base, int rank, const uint64_t *dims,
              const uint64_t *strides, const uint32_t *box);

}  // namespace mosa
