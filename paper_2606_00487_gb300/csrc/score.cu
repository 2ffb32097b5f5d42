// Stage 2 of a TAPS round (Sec. 4.2, Eq. 1, Algorithm 1): the edge scorer
// and the sibling-wise softmax that turns its logits into q_cond.
//
// One CTA per (position d, request b). The MLP's first layer is linear in
// the concatenated features [E_tok[parent], E_tok[child], E_dep[d+1], logp,
// entropy], so it is split into a per-parent part, a per-child part (which
// also carries the logp column) and a per-position part (depth embedding,
// entropy column and bias); each is computed once and summed per edge.
#include <algorithm>

#include "common.cuh"

namespace taps {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

__global__ void __launch_bounds__(kThreads)
score_kernel(const int32_t* __restrict__ root_tok, const int32_t* __restrict__ ids,
             const float* __restrict__ logp, const float* __restrict__ entropy, int L, int K,
             int kind, int E, int H, int vocab, int max_depth, const float* __restrict__ w,
             float* __restrict__ q_cond) {
  extern __shared__ float sm[];
  const int d = blockIdx.x;
  const int b = blockIdx.y;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int F = 3 * E + 2;
  const int np = d == 0 ? 1 : K;            // parents of position d
  const int64_t row0 = (static_cast<int64_t>(b) * L + d) * K;

  float* s_ell = sm;                         // [K][K]
  float* s_logp = s_ell + K * K;             // [K]
  float* s_P = s_logp + K;                   // [K][H] per-parent pre-activation
  float* s_C = s_P + K * H;                  // [K][H] per-child pre-activation
  float* s_D = s_C + K * H;                  // [H]    per-position pre-activation
  int* s_ptok = reinterpret_cast<int*>(s_D + H);  // [K]
  int* s_ctok = s_ptok + K;                       // [K]
  // MLP operands staged in shared memory (first layer rows padded to an odd
  // stride, so that the threads of a warp, one hidden unit each, read
  // different banks)
  const int FP = F | 1;
  float* s_W1 = reinterpret_cast<float*>(s_ctok + K);   // [H][FP]
  float* s_b1 = s_W1 + H * FP;                          // [H]
  float* s_w2 = s_b1 + H;                               // [H + 1]
  float* s_dep = s_w2 + H + 1;                          // [E] depth embedding of d + 1
  float* s_emb = s_dep + E;                             // [np + K][E] parents', then children's

  const bool mlp = kind == TAPS_SCORER_MLP;
  const float* tok_emb = w;
  const float* dep_emb = tok_emb + static_cast<int64_t>(vocab) * E;
  const float* W1 = dep_emb + static_cast<int64_t>(max_depth) * E;
  const float* b1 = W1 + H * F;
  const float* w2 = b1 + H;
  // The MLP's weights are no output of any kernel of the round: they are
  // staged before the wait for the preceding grid, overlapping its tail
  // (the caller's contract, include/taps.h).
  if (mlp) {
    for (int i = tid; i < H * F; i += kThreads) s_W1[(i / F) * FP + i % F] = W1[i];
    for (int i = tid; i < 2 * H + 1; i += kThreads) s_b1[i] = b1[i];   // b1, then w2 and its logp weight
    const float* drow = dep_emb + static_cast<int64_t>(min(d + 1, max_depth - 1)) * E;
    for (int i = tid; i < E; i += kThreads) s_dep[i] = drow[i];
  }
  dep_enter();
  for (int j = tid; j < K; j += kThreads) {
    s_logp[j] = logp[row0 + j];
    s_ctok[j] = ids[row0 + j];
    s_ptok[j] = d == 0 ? root_tok[b] : ids[row0 - K + j];
  }
  __syncthreads();

  if (!mlp) {
    for (int e = tid; e < np * K; e += kThreads) s_ell[e] = s_logp[e % K];
  } else {
    const float w_lp = s_w2[H];
    const float ent = entropy[static_cast<int64_t>(b) * L + d];
    // the token embedding rows of the parents and the children (0 for an id
    // outside the vocabulary, whose dot product is then skipped)
    for (int i = tid; i < (np + K) * E; i += kThreads) {
      const int rrow = i / E, e = i % E;
      const int tok = rrow < np ? s_ptok[rrow] : s_ctok[rrow - np];
      s_emb[i] = (tok >= 0 && tok < vocab) ? tok_emb[static_cast<int64_t>(tok) * E + e] : 0.f;
    }
    __syncthreads();
    // per-parent, per-child and per-position parts of W1 f + b1
    const int items = (np + K) * H + H;
    for (int it = tid; it < items; it += kThreads) {
      float acc;
      if (it < np * H) {                       // parent part
        const int i = it / H, h = it % H;
        const int tok = s_ptok[i];
        const float* wrow = s_W1 + h * FP;
        const float* emb = s_emb + i * E;
        acc = 0.f;
        if (tok >= 0 && tok < vocab)
          for (int e = 0; e < E; ++e) acc = fmaf(wrow[e], emb[e], acc);
        s_P[i * H + h] = acc;
      } else if (it < (np + K) * H) {          // child part (+ logp column)
        const int r = it - np * H;
        const int j = r / H, h = r % H;
        const int tok = s_ctok[j];
        const float* wrow = s_W1 + h * FP + E;
        const float* emb = s_emb + (np + j) * E;
        acc = 0.f;
        if (tok >= 0 && tok < vocab)
          for (int e = 0; e < E; ++e) acc = fmaf(wrow[e], emb[e], acc);
        acc = fmaf(s_W1[h * FP + 3 * E], s_logp[j], acc);
        s_C[j * H + h] = acc;
      } else {                                 // per-position part
        const int h = it - (np + K) * H;
        const float* wrow = s_W1 + h * FP + 2 * E;
        acc = s_b1[h];
        for (int e = 0; e < E; ++e) acc = fmaf(wrow[e], s_dep[e], acc);
        acc = fmaf(s_W1[h * FP + 3 * E + 1], ent, acc);
        s_D[h] = acc;
      }
    }
    __syncthreads();
    // edge logits: one warp reduction over the hidden units per edge, four
    // edges of a warp at a time so that their reductions overlap
    for (int e0 = warp; e0 < np * K; e0 += 4 * kWarps) {
      float acc[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int e = e0 + u * kWarps;
        acc[u] = 0.f;
        if (e < np * K) {
          const int i = e / K, j = e % K;
          for (int h = lane; h < H; h += 32) {
            const float a = s_P[i * H + h] + s_C[j * H + h] + s_D[h];
            acc[u] = fmaf(s_w2[h], fmaxf(a, 0.f), acc[u]);
          }
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1)
#pragma unroll
        for (int u = 0; u < 4; ++u) acc[u] += __shfl_xor_sync(kFullMask, acc[u], off);
      if (lane == 0)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int e = e0 + u * kWarps;
          if (e < np * K) s_ell[e] = fmaf(w_lp, s_logp[e % K], acc[u]);
        }
    }
  }
  __syncthreads();

  // sibling-wise softmax, one warp per parent row and one lane per child
  // (K <= 32); the marginal-product kind takes each child's marginal
  // probability as it is
  float* out = q_cond + (static_cast<int64_t>(b) * L + d) * K * K;
  const bool in = lane < K;
  for (int i = warp; i < K; i += kWarps) {
    if (i >= np) {
      if (in) out[i * K + lane] = 0.f;
      continue;
    }
    const float x = in ? s_ell[i * K + lane] : -INFINITY;
    if (kind == TAPS_SCORER_MARGINAL_PRODUCT) {
      if (in) out[i * K + lane] = expf(x);
      continue;
    }
    float m = x;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(kFullMask, m, off));
    const float ex = in ? expf(x - m) : 0.f;
    float sum = ex;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(kFullMask, sum, off);
    if (in) out[i * K + lane] = __fdiv_rn(ex, sum);
  }
}

// Eq. 2 for an explicit list of nodes: reach = product of q_cond along the
// path, one IEEE f32 multiply per edge, root to leaf (the operations and order
// of the selection's reach). One thread per (request, path); the slots are
// known up front, so the path's q_cond loads are independent of each other.
__global__ void __launch_bounds__(256)
path_reach_kernel(const float* __restrict__ q_cond, const uint8_t* __restrict__ paths,
                  const int32_t* __restrict__ path_len, int B, int L, int K, int M,
                  float* __restrict__ path_reach) {
  dep_enter();
  const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (e >= static_cast<int64_t>(B) * M) return;
  const int b = static_cast<int>(e / M);
  const int n = path_len[e];
  float r = 0.f;   // not a node of the trie
  if (n >= 0 && n <= L) {
    const uint8_t* p = paths + e * L;
    const float* qb = q_cond + static_cast<int64_t>(b) * L * K * K;
    float qv[TAPS_MAX_L];
    bool ok = true;
    int prev = 0;   // depth-1 children hang off the root, row 0
#pragma unroll
    for (int d = 0; d < TAPS_MAX_L; ++d) {
      if (d < n) {
        const int j = p[d];
        ok = ok && j < K;
        qv[d] = j < K ? qb[(d * K + prev) * K + j] : 0.f;
        prev = j < K ? j : 0;
      }
    }
    if (ok) {
      r = 1.0f;
#pragma unroll
      for (int d = 0; d < TAPS_MAX_L; ++d)
        if (d < n) r = __fmul_rn(r, qv[d]);
    }
  }
  path_reach[e] = r;
}

std::atomic<int> g_score_smem[64];

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" int taps_score_reach(const int32_t* root_tok, const int32_t* topk_ids,
                                const float* topk_logp, const float* entropy, int B, int L, int K,
                                const taps_scorer_params* params, float* q_cond,
                                const uint8_t* paths, const int32_t* path_len, int M,
                                float* path_reach, void* stream) {
  if (!root_tok || !topk_ids || !topk_logp || !q_cond || !params) return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || K <= 0) return TAPS_ERR_INVALID_ARG;
  // the path list is all or nothing
  const bool want_paths = paths || path_len || path_reach;
  if (want_paths && (!paths || !path_len || !path_reach || M <= 0)) return TAPS_ERR_INVALID_ARG;
  if (!want_paths && M != 0) return TAPS_ERR_INVALID_ARG;
  if (want_paths && static_cast<int64_t>(B) * M > (static_cast<int64_t>(1) << 31) - 256)
    return TAPS_ERR_UNSUPPORTED;
  if (K > TAPS_MAX_K || L > TAPS_MAX_L || B > 65535) return TAPS_ERR_UNSUPPORTED;
  int kind = params->kind;
  int E = 0, H = 0;
  if (kind == TAPS_SCORER_MLP) {
    E = params->emb_dim;
    H = params->hidden;
    if (!params->weights || !entropy || E <= 0 || H <= 0 || params->vocab <= 0 ||
        params->max_depth <= L)
      return TAPS_ERR_INVALID_ARG;
    if (E > TAPS_MAX_EMB || H > TAPS_MAX_HIDDEN) return TAPS_ERR_UNSUPPORTED;
  } else if (kind != TAPS_SCORER_MARGINAL && kind != TAPS_SCORER_MARGINAL_PRODUCT) {
    return TAPS_ERR_INVALID_ARG;
  }
  // q/logits, logp, per-parent/child/position parts, token ids, then (MLP) the
  // staged first layer (rows padded to an odd stride), b1, w2, the depth
  // embedding and the parents' and children's token embeddings
  size_t smem = sizeof(float) * (K * K + K + 2 * K * std::max(H, 1) + std::max(H, 1)) +
                sizeof(int) * 2 * K;
  if (kind == TAPS_SCORER_MLP)
    smem += sizeof(float) * (static_cast<size_t>(H) * ((3 * E + 2) | 1) + 2 * H + 1 + E +
                             static_cast<size_t>(2 * K) * E);
  if (!smem_limit(score_kernel, smem, g_score_smem)) return TAPS_ERR_CUDA;
  dim3 grid(L, B);
  if (launch_dep(score_kernel, grid, dim3(kThreads), smem, static_cast<cudaStream_t>(stream),
                 root_tok, topk_ids, topk_logp, entropy, L, K, kind, E, H, params->vocab,
                 params->max_depth, static_cast<const float*>(params->weights), q_cond) !=
      cudaSuccess)
    return TAPS_ERR_CUDA;
  if (want_paths) {
    const int64_t n = static_cast<int64_t>(B) * M;
    if (launch_dep(path_reach_kernel, dim3(static_cast<unsigned>((n + 255) / 256)), dim3(256), 0,
                   static_cast<cudaStream_t>(stream), q_cond, paths, path_len, B, L, K, M,
                   path_reach) != cudaSuccess)
      return TAPS_ERR_CUDA;
  }
  return launch_status();
}
