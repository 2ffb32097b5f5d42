// Internal helpers shared by the TAPS CUDA sources (not part of the C ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "taps.h"

namespace taps {

// GB300: 152 SMs on two dies. Work splits are planned for this count; the
// result never depends on it.
constexpr int kTargetSms = 152;
constexpr unsigned kFullMask = 0xffffffffu;

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

inline int launch_status() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? TAPS_OK : TAPS_ERR_CUDA;
}

inline bool aligned(const void* p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

// Order-preserving map of a float to uint32 (larger float -> larger uint).
// -0.0 is folded onto +0.0 first so that equal values compare equal.
__device__ __forceinline__ uint32_t f32_to_ordered(float f) {
  uint32_t b = __float_as_uint(f + 0.0f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float ordered_to_f32(uint32_t s) {
  uint32_t b = (s & 0x80000000u) ? (s & 0x7fffffffu) : ~s;
  return __uint_as_float(b);
}

// 64-bit warp maximum built from two 32-bit redux operations.
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t key) {
  uint32_t hi = static_cast<uint32_t>(key >> 32);
  uint32_t lo = static_cast<uint32_t>(key);
  uint32_t mhi = __reduce_max_sync(kFullMask, hi);
  uint32_t mlo = __reduce_max_sync(kFullMask, hi == mhi ? lo : 0u);
  return (static_cast<uint64_t>(mhi) << 32) | mlo;
}

}  // namespace taps
