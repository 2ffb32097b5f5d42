// Stage 6 of a TAPS round: lossless greedy acceptance (Sec. 4.1; the
// Limitations section fixes temperature 0, where verification checks each
// draft token against the target's greedy choice).
//
// One warp per request. From the root, the warp scans the nodes after the
// current one for the child whose token equals the target's greedy token at
// the current node (sibling tokens are distinct, so at most one matches) and
// steps into it, at most L times.
#include "common.cuh"

namespace taps {
namespace {

__global__ void __launch_bounds__(32)
accept_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ token,
              const int32_t* __restrict__ n_nodes, const int32_t* __restrict__ target_tok,
              int n_max, int L, int32_t* __restrict__ accept_len,
              int32_t* __restrict__ accepted_nodes, int32_t* __restrict__ bonus_tok) {
  const int b = blockIdx.x;
  const int lane = threadIdx.x;
  const int n = min(max(n_nodes[b], 1), n_max);
  const int64_t o = static_cast<int64_t>(b) * n_max;
  int32_t* path = accepted_nodes + static_cast<int64_t>(b) * (L + 1);
  int v = 0;
  int len = 0;
  if (lane == 0) path[0] = 0;
  for (int step = 0; step < L; ++step) {
    const int want = target_tok[o + v];
    int found = -1;
    for (int c0 = v + 1; c0 < n; c0 += 32) {
      int c = c0 + lane;
      bool hit = c < n && parent[o + c] == v && token[o + c] == want;
      unsigned m = __ballot_sync(kFullMask, hit);
      if (m) {
        found = c0 + __ffs(m) - 1;
        break;
      }
    }
    if (found < 0) break;
    v = found;
    ++len;
    if (lane == 0) path[len] = v;
  }
  for (int i = len + 1 + lane; i <= L; i += 32) path[i] = -1;
  if (lane == 0) {
    accept_len[b] = len;
    bonus_tok[b] = target_tok[o + v];
  }
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
  accept_kernel<<<B, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      parent, token, n_nodes, target_tok, n_max, L, accept_len, accepted_nodes, bonus_tok);
  return launch_status();
}
