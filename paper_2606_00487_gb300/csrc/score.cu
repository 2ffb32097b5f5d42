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

__global__ void __launch_bounds__(kThreads)
score_kernel(const int32_t* __restrict__ root_tok, const int32_t* __restrict__ ids,
             const float* __restrict__ logp, const float* __restrict__ entropy, int L, int K,
             int kind, int E, int H, int vocab, int max_depth, const float* __restrict__ w,
             float* __restrict__ q_cond) {
  dep_enter();
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

  for (int j = tid; j < K; j += kThreads) {
    s_logp[j] = logp[row0 + j];
    s_ctok[j] = ids[row0 + j];
    s_ptok[j] = d == 0 ? root_tok[b] : ids[row0 - K + j];
  }
  __syncthreads();

  if (kind != TAPS_SCORER_MLP) {
    for (int e = tid; e < np * K; e += kThreads) s_ell[e] = s_logp[e % K];
  } else {
    const float* tok_emb = w;
    const float* dep_emb = tok_emb + static_cast<int64_t>(vocab) * E;
    const float* W1 = dep_emb + static_cast<int64_t>(max_depth) * E;
    const float* b1 = W1 + H * F;
    const float* w2 = b1 + H;
    const float w_lp = w2[H];
    const float ent = entropy[static_cast<int64_t>(b) * L + d];
    // per-parent, per-child and per-position parts of W1 f + b1
    const int items = (np + K) * H + H;
    for (int it = tid; it < items; it += kThreads) {
      const float* wrow;
      const float* emb;
      float acc;
      int tok;
      if (it < np * H) {                       // parent part
        int i = it / H, h = it % H;
        tok = s_ptok[i];
        wrow = W1 + h * F;
        emb = (tok >= 0 && tok < vocab) ? tok_emb + static_cast<int64_t>(tok) * E : nullptr;
        acc = 0.f;
        if (emb)
          for (int e = 0; e < E; ++e) acc = fmaf(wrow[e], emb[e], acc);
        s_P[i * H + h] = acc;
      } else if (it < (np + K) * H) {          // child part (+ logp column)
        int r = it - np * H;
        int j = r / H, h = r % H;
        tok = s_ctok[j];
        wrow = W1 + h * F + E;
        emb = (tok >= 0 && tok < vocab) ? tok_emb + static_cast<int64_t>(tok) * E : nullptr;
        acc = 0.f;
        if (emb)
          for (int e = 0; e < E; ++e) acc = fmaf(wrow[e], emb[e], acc);
        acc = fmaf(W1[h * F + 3 * E], s_logp[j], acc);
        s_C[j * H + h] = acc;
      } else {                                 // per-position part
        int h = it - (np + K) * H;
        wrow = W1 + h * F + 2 * E;
        emb = dep_emb + static_cast<int64_t>(min(d + 1, max_depth - 1)) * E;
        acc = b1[h];
        for (int e = 0; e < E; ++e) acc = fmaf(wrow[e], emb[e], acc);
        acc = fmaf(W1[h * F + 3 * E + 1], ent, acc);
        s_D[h] = acc;
      }
    }
    __syncthreads();
    // edge logits: one warp reduction over the hidden units per edge
    const int nw = kThreads / 32;
    for (int e = warp; e < np * K; e += nw) {
      int i = e / K, j = e % K;
      float acc = 0.f;
      for (int h = lane; h < H; h += 32) {
        float a = s_P[i * H + h] + s_C[j * H + h] + s_D[h];
        acc = fmaf(w2[h], fmaxf(a, 0.f), acc);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(kFullMask, acc, off);
      if (lane == 0) s_ell[e] = fmaf(w_lp, s_logp[j], acc);
    }
  }
  __syncthreads();

  // sibling-wise softmax, one thread per parent row (the marginal-product
  // kind takes each child's marginal probability as it is)
  float* out = q_cond + (static_cast<int64_t>(b) * L + d) * K * K;
  for (int i = tid; i < K; i += kThreads) {
    if (i < np && kind == TAPS_SCORER_MARGINAL_PRODUCT) {
      for (int j = 0; j < K; ++j) out[i * K + j] = expf(s_ell[i * K + j]);
    } else if (i < np) {
      float m = -INFINITY;
      for (int j = 0; j < K; ++j) m = fmaxf(m, s_ell[i * K + j]);
      float sum = 0.f;
      for (int j = 0; j < K; ++j) sum += expf(s_ell[i * K + j] - m);
      for (int j = 0; j < K; ++j) out[i * K + j] = __fdiv_rn(expf(s_ell[i * K + j] - m), sum);
    } else {
      for (int j = 0; j < K; ++j) out[i * K + j] = 0.f;
    }
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
  size_t smem = sizeof(float) * (K * K + K + 2 * K * std::max(H, 1) + std::max(H, 1)) +
                sizeof(int) * 2 * K;
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
