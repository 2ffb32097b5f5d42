// Stage 4 of a TAPS round: the bit-packed ancestor-or-self mask that tree
// attention applies to the tree part of the keys (Sec. 4.1 stage 3; Sec. 4.3
// requires the verified set to be a connected subtree rooted at the current
// position, so every node's ancestors are in the tree).
//
// One CTA per request; each thread builds one 32-bit word of one row by
// walking the node's parent chain (at most L steps).
#include "common.cuh"

namespace taps {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
mask_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ n_nodes, int n_max,
            int W, uint32_t* __restrict__ mask) {
  dep_enter();
  const int b = blockIdx.x;
  const int n = min(max(n_nodes[b], 0), n_max);
  const int32_t* pb = parent + static_cast<int64_t>(b) * n_max;
  uint32_t* mb = mask + static_cast<int64_t>(b) * n_max * W;
  for (int e = threadIdx.x; e < n_max * W; e += kThreads) {
    const int i = e / W;
    const int w = e % W;
    uint32_t word = 0;
    if (i < n) {
      int j = i;
      // parent[j] < j for a valid tree; stop on anything else
      while (j >= 0) {
        if ((j >> 5) == w) word |= 1u << (j & 31);
        int pj = pb[j];
        if (pj >= j) break;
        j = pj;
      }
    }
    mb[e] = word;
  }
}

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" int taps_build_tree_mask(const int32_t* parent, const int32_t* n_nodes, int B,
                                    int n_max, uint32_t* mask, void* stream) {
  if (!parent || !n_nodes || !mask) return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || n_max <= 0) return TAPS_ERR_INVALID_ARG;
  if (n_max > TAPS_MAX_NODES || B > 65535) return TAPS_ERR_UNSUPPORTED;
  const int W = (n_max + 31) / 32;
  if (launch_dep(mask_kernel, dim3(B), dim3(kThreads), 0, static_cast<cudaStream_t>(stream),
                 parent, n_nodes, n_max, W, mask) != cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}
