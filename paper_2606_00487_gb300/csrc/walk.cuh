// The greedy acceptance walk (Sec. 4.1; temperature 0 per the Limitations
// section), shared by taps_accept and taps_target_greedy_accept.
//
// Instead of scanning the children of the current node at every step, the
// block first finds, in one parallel pass, the matching child of EVERY node:
// match[v] = the lowest c with parent[c] == v and token[c] == target[v]
// (sibling tokens are distinct, so there is at most one). The walk is then a
// chase of at most L pointers in shared memory.
#pragma once

#include <limits.h>

#include "common.cuh"

namespace taps {

// Every thread of the block calls this after s_par, s_tok and s_tt hold the
// first n entries of the request (and a __syncthreads). s_match is scratch of
// n ints. Writes path[0 .. L] (node indices, then -1), *accept_len, *bonus.
__device__ __forceinline__ void accept_walk(const int32_t* s_par, const int32_t* s_tok,
                                            const int32_t* s_tt, int32_t* s_match, int n, int L,
                                            int32_t* path, int32_t* accept_len,
                                            int32_t* bonus) {
  const int tid = threadIdx.x;
  for (int j = tid; j < n; j += blockDim.x) s_match[j] = INT_MAX;
  __syncthreads();
  for (int c = tid + 1; c < n; c += blockDim.x) {
    const int p = s_par[c];
    if (p >= 0 && p < c && s_tok[c] == s_tt[p]) atomicMin(s_match + p, c);
  }
  __syncthreads();
  if (tid >= 32) return;
  const int lane = tid;
  int v = 0, len = 0;
  if (lane == 0) {
    path[0] = 0;
    while (len < L) {
      const int c = s_match[v];
      if (c == INT_MAX) break;
      v = c;
      path[++len] = v;
    }
    *accept_len = len;
    *bonus = s_tt[v];
  }
  len = __shfl_sync(kFullMask, len, 0);
  for (int j = len + 1 + lane; j <= L; j += 32) path[j] = -1;
}

}  // namespace taps
