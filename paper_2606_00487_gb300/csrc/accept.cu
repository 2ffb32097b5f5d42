// Stage 6 of a TAPS round: lossless greedy acceptance (Sec. 4.1; the
// Limitations section fixes temperature 0, where verification checks each
// draft token against the target's greedy choice).
//
// One CTA per request stages the tree (parent, token, target token) in
// shared memory, finds the matching child of every node in one parallel pass
// and chases the matches from the root, at most L steps.
#include "walk.cuh"

namespace taps {
namespace {

constexpr int kThreads = 128;

__global__ void __launch_bounds__(kThreads)
accept_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ token,
              const int32_t* __restrict__ n_nodes, const int32_t* __restrict__ target_tok,
              int n_max, int L, int32_t* __restrict__ accept_len,
              int32_t* __restrict__ accepted_nodes, int32_t* __restrict__ bonus_tok) {
  dep_enter();
  __shared__ int32_t s_par[TAPS_MAX_NODES], s_tok[TAPS_MAX_NODES], s_tt[TAPS_MAX_NODES];
  __shared__ int32_t s_match[TAPS_MAX_NODES];
  const int b = blockIdx.x;
  const int n = min(max(n_nodes[b], 1), n_max);
  const int64_t o = static_cast<int64_t>(b) * n_max;
  for (int j = threadIdx.x; j < n; j += kThreads) {
    s_par[j] = parent[o + j];
    s_tok[j] = token[o + j];
    s_tt[j] = target_tok[o + j];
  }
  __syncthreads();
  accept_walk(s_par, s_tok, s_tt, s_match, n, L,
              accepted_nodes + static_cast<int64_t>(b) * (L + 1), accept_len + b, bonus_tok + b);
}

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" int taps_accept(const int32_t* parent, const int32_t* token, const int32_t* n_nodes,
                           const int32_t* target_tok, int B, int n_max, int L,
                           int32_t* accept_len, int32_t* accepted_nodes, int32_t* bonus_tok,
                           void* stream) {
  if (!parent || !token || !n_nodes || !target_tok || !accept_len || !accepted_nodes ||
      !bonus_tok)
    return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || n_max <= 0 || L < 0) return TAPS_ERR_INVALID_ARG;
  if (n_max > TAPS_MAX_NODES || L > TAPS_MAX_L || B > 65535) return TAPS_ERR_UNSUPPORTED;
  if (launch_dep(accept_kernel, dim3(B), dim3(kThreads), 0, static_cast<cudaStream_t>(stream),
                 parent, token, n_nodes, target_tok, n_max, L, accept_len, accepted_nodes,
                 bonus_tok) != cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}
