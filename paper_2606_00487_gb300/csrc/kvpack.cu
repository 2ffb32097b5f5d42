// Conversion between the logical paged KV cache [num_pages][Hkv][16][D] and
// the TAPS page layout that taps_tree_verify_attn reads: inside each
// (page, head) block of 16 tokens x D dims, token w and dim d sit at byte
//   (w / 8) * (D / 64) * 1024 + (d / 64) * 1024 + (w % 8) * 128
//     + (((d % 64) / 8) XOR (w % 8)) * 16 + (d % 8) * 2,
// i.e. 8-token groups of 128-byte rows with the 128-byte swizzle, the layout
// the tensor core reads, so one contiguous copy per page feeds the MMAs.
#include <algorithm>

#include "common.cuh"

namespace taps {
namespace {

__device__ __forceinline__ int64_t packed_offset(int64_t blk, int w, int q, int D) {
  // q = 16-byte chunk index of the dim (d / 8)
  const int ch = D / 64;
  return blk * (16 * D * 2) + (w >> 3) * (ch * 1024) + (q >> 3) * 1024 + (w & 7) * 128 +
         (((q & 7) ^ (w & 7)) << 4);
}

template <bool kPack>
__global__ void __launch_bounds__(256)
kv_pack_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, int64_t chunks, int D) {
  const int qn = D / 8;                                  // 16-byte chunks per token row
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < chunks;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int q = static_cast<int>(e % qn);
    const int64_t row = e / qn;                          // (block, token)
    const int w = static_cast<int>(row & 15);
    const int64_t blk = row >> 4;
    const int64_t po = packed_offset(blk, w, q, D) / 16;
    if (kPack)
      dst[po] = src[e];
    else
      dst[e] = src[po];
  }
}

int run(bool pack, const void* src, void* dst, int64_t num_pages, int Hkv, int D, void* stream) {
  if (!src || !dst || num_pages <= 0 || Hkv <= 0) return TAPS_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return TAPS_ERR_UNSUPPORTED;
  if (!aligned(src, 16) || !aligned(dst, 16)) return TAPS_ERR_INVALID_ARG;
  const int64_t chunks = num_pages * Hkv * 16 * (D / 8);
  const int blocks = static_cast<int>(std::min<int64_t>((chunks + 255) / 256, 16 * kTargetSms));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (pack)
    kv_pack_kernel<true><<<blocks, 256, 0, s>>>(static_cast<const uint4*>(src),
                                                static_cast<uint4*>(dst), chunks, D);
  else
    kv_pack_kernel<false><<<blocks, 256, 0, s>>>(static_cast<const uint4*>(src),
                                                 static_cast<uint4*>(dst), chunks, D);
  return launch_status();
}

}  // namespace
}  // namespace taps

extern "C" int taps_pack_kv_pages(const void* src, void* dst, int64_t num_pages, int Hkv, int D,
                                  void* stream) {
  return taps::run(true, src, dst, num_pages, Hkv, D, stream);
}

extern "C" int taps_unpack_kv_pages(const void* src, void* dst, int64_t num_pages, int Hkv,
                                    int D, void* stream) {
  return taps::run(false, src, dst, num_pages, Hkv, D, stream);
}
