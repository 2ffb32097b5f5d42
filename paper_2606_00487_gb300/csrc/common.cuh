// Internal helpers shared by the TAPS CUDA sources (not part of the C ABI).
#pragma once

#include <atomic>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <utility>

#include "taps.h"

namespace taps {

// GB300: 152 SMs on two dies. Work splits are planned for this count; the
// result never depends on it.
constexpr int kTargetSms = 152;
constexpr unsigned kFullMask = 0xffffffffu;

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Programmatic dependent launch. Every kernel of the library is launched
// with programmatic stream serialisation, so that its launch and prologue may
// overlap the tail of the kernel before it on the stream. dep_enter() comes
// before every read of an input another kernel may write and before every
// output write (it is the first statement of most kernels; the scorer stages
// its weights ahead of it): it waits until the previous grid has completed and
// its memory is visible, then lets the next kernel on the stream be launched.
__device__ __forceinline__ void dep_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_dep(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Raise the dynamic shared-memory limit of a kernel once per device (atomic
// flags: calls may come from several host threads).
template <typename Kern>
bool smem_limit(Kern kernel, size_t bytes, std::atomic<int>* done) {
  if (bytes <= 48 * 1024) return true;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  // the flag holds the largest size set so far (+1)
  if (done[dev].load(std::memory_order_acquire) > static_cast<int>(bytes)) return true;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(bytes)) != cudaSuccess)
    return false;
  int prev = done[dev].load(std::memory_order_relaxed);
  while (prev <= static_cast<int>(bytes) &&
         !done[dev].compare_exchange_weak(prev, static_cast<int>(bytes) + 1)) {
  }
  return true;
}

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
