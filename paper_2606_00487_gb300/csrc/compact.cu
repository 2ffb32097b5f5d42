// Accepted-path K/V compaction: after acceptance the accepted path becomes
// committed context for the next round of the drafting/verification loop
// (Sec. 4.1), so the K/V of accepted node path[i] moves from logical position
// ctx_len + path[i] (where verification wrote tree node path[i]) to position
// ctx_len + i. The node's key was rotated at position id ctx_len + depth,
// and depth(path[i]) = i, so the moved key needs no re-rotation.
//
// One CTA per (layer, K or V, request, KV head). It loads every moved
// 16-byte chunk of its (head, path) into registers, waits at a barrier, then
// stores them: a destination position may be the source of a later path entry
// (path[j] = i for some j < i), and all reads finish before any write.
// Entries with path[i] == i are already in place and are skipped.
#include "common.cuh"

namespace taps {
namespace {

constexpr int kThreads = 128;
constexpr int kPage = 16;
// (TAPS_MAX_L + 1) tokens x D / 8 chunks (D <= 128) over kThreads threads
constexpr int kPerThread = ((TAPS_MAX_L + 1) * 16 + kThreads - 1) / kThreads;

struct LayerBases {
  uint4* p[2 * TAPS_MAX_LAYERS];   // K of layer l at 2l, V at 2l + 1
};

// 16-byte chunk q (dims 8q .. 8q+7) of row w of a TAPS-layout block, in uint4 units
__device__ __forceinline__ int64_t chunk_index(int64_t blk, int w, int q, int D) {
  const int ch = D / 64;
  return blk * (kPage * D / 8) + (w >> 3) * (ch * 64) + (q >> 3) * 64 + (w & 7) * 8 +
         ((q & 7) ^ (w & 7));
}

__global__ void __launch_bounds__(kThreads)
compact_kernel(LayerBases bases, int B, int Hkv, int D, int64_t num_pages,
               const int32_t* __restrict__ block_table, int max_pages,
               const int32_t* __restrict__ ctx_len, const int32_t* __restrict__ accepted_nodes,
               const int32_t* __restrict__ accept_len, int L, int32_t* status) {
  dep_enter();
  const int lkv = blockIdx.x / B;            // 2 * layer + (0 K, 1 V)
  const int b = blockIdx.x - lkv * B;
  const int h = blockIdx.y;
  uint4* cache = bases.p[lkv];
  const int len = min(max(accept_len[b], 0), L);
  const int ctx = ctx_len[b];
  const int32_t* path = accepted_nodes + static_cast<int64_t>(b) * (L + 1);
  const int32_t* bt = block_table + static_cast<int64_t>(b) * max_pages;
  const int qn = D / 8;
  const int total = (len + 1) * qn;

  // Chunk offset of logical position t of this head, or -1 when its page is
  // outside the block table or the cache.
  auto locate = [&](int64_t t, int q) -> int64_t {
    if (t < 0 || t >= static_cast<int64_t>(max_pages) * kPage) return -1;
    const int page = bt[t / kPage];
    if (page < 0 || page >= num_pages) return -1;
    return chunk_index(static_cast<int64_t>(page) * Hkv + h, static_cast<int>(t % kPage), q, D);
  };

  uint4 buf[kPerThread];
  int64_t dst[kPerThread];
  bool bad = false;
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    dst[r] = -1;
    const int e = threadIdx.x + r * kThreads;
    if (e < total) {
      const int i = e / qn, q = e - (e / qn) * qn;
      const int src_node = path[i];
      if (src_node != i) {
        const int64_t s = locate(static_cast<int64_t>(ctx) + src_node, q);
        const int64_t d = locate(static_cast<int64_t>(ctx) + i, q);
        if (s < 0 || d < 0 || src_node < 0) {
          bad = true;
        } else {
          buf[r] = cache[s];
          dst[r] = d;
        }
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < kPerThread; ++r)
    if (dst[r] >= 0) cache[dst[r]] = buf[r];
  if (bad && status) atomicOr(status, TAPS_DEVFAULT_PAGE);
}

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" int taps_compact_accepted_kv(void* const* k_layers, void* const* v_layers,
                                        int num_layers, int64_t num_pages,
                                        const int32_t* block_table, int max_pages,
                                        const int32_t* ctx_len, const int32_t* accepted_nodes,
                                        const int32_t* accept_len, int B, int L, int Hkv, int D,
                                        int page_size, int32_t* status, void* stream) {
  if (!k_layers || !v_layers || !block_table || !ctx_len || !accepted_nodes || !accept_len)
    return TAPS_ERR_INVALID_ARG;
  if (num_layers <= 0 || num_pages <= 0 || max_pages <= 0 || B <= 0 || L < 0 || Hkv <= 0)
    return TAPS_ERR_INVALID_ARG;
  if (num_layers > TAPS_MAX_LAYERS || L > TAPS_MAX_L || page_size != kPage ||
      (D != 64 && D != 128) || Hkv > 65535 || static_cast<int64_t>(B) * 2 * num_layers > 0x7fffffff)
    return TAPS_ERR_UNSUPPORTED;
  LayerBases bases;
  for (int l = 0; l < num_layers; ++l) {
    if (!k_layers[l] || !v_layers[l] || !aligned(k_layers[l], 16) || !aligned(v_layers[l], 16))
      return TAPS_ERR_INVALID_ARG;
    bases.p[2 * l] = static_cast<uint4*>(k_layers[l]);
    bases.p[2 * l + 1] = static_cast<uint4*>(v_layers[l]);
  }
  const dim3 grid(static_cast<unsigned>(B * 2 * num_layers), static_cast<unsigned>(Hkv));
  if (launch_dep(compact_kernel, grid, dim3(kThreads), 0, static_cast<cudaStream_t>(stream),
                 bases, B, Hkv, D, num_pages, block_table, max_pages, ctx_len, accepted_nodes,
                 accept_len, L, status) != cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}
