// Host-side helpers shared by the libsonic entry points.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "sonic.h"

namespace sonic {

// Encodes a 4-D bf16 TMA tensor map with 128-byte swizzle.
//   dims    : extents, innermost first (elements)
//   strides : byte strides of dims 1..3
//   box     : box extents, innermost first (box[0] * 2 bytes must be <= 128)
// Returns false if the driver rejects the map (bad alignment or extents).
bool make_tmap_bf16_4d(CUtensorMap *map, const void *base, const uint64_t dims[4],
                       const uint64_t strides[3], const uint32_t box[4]);

// The same with 5 dimensions (strides of dims 1..4).
bool make_tmap_bf16_5d(CUtensorMap *map, const void *base, const uint64_t dims[5],
                       const uint64_t strides[4], const uint32_t box[5]);

// Number of SMs of the current device (cached per device).
int device_sm_count();

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace sonic
