// Target greedy token of every tree node fused with the acceptance walk.
//
// At temperature 0 (the setting the Limitations section fixes) the target's
// choice after the prefix ending at tree node i is the argmax of its verify
// logits; the acceptance walk of Sec. 4.1 then follows the children whose
// token equals that choice. One launch does both:
//
//  - The rows of one request's live nodes are split into `splits` slices of
//    16-byte vectors; each CTA reads one slice once (streaming loads), keeps a
//    per-thread running maximum with the vector that holds it, and reduces to
//    one 64-bit key: ordered(max) << 32 | (0xffffffff - index), so the largest
//    key is the largest value at the lowest index.
//  - The key is merged into the row's workspace word with atomicMax, then the
//    CTA takes a ticket of its request. The CTA that takes the last ticket
//    decodes every row of its request, writes target_tok, clears the
//    workspace words and the ticket back to zero, and runs the walk.
//
// The pass is HBM-bound: every live row's V logits are read exactly once.
#include <math.h>

#include <algorithm>

#include "walk.cuh"

namespace taps {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kCtasPerSm = 4;                 // 256-thread CTAs resident per SM (<= 64 regs)
constexpr int kBatch = 8;                     // 16-byte loads in flight per thread

struct TargetPlan {
  int splits;        // CTAs per row
  int64_t chunk;     // vectors per CTA
  int64_t nvec;      // full 16-byte vectors per row
};

// Largest element of a 16-byte vector of bf16 or f32 logits.
__device__ __forceinline__ float vec_max(uint4 u, __nv_bfloat16) {
  __nv_bfloat162 a = *reinterpret_cast<__nv_bfloat162*>(&u.x);
  __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&u.y);
  __nv_bfloat162 c = *reinterpret_cast<__nv_bfloat162*>(&u.z);
  __nv_bfloat162 d = *reinterpret_cast<__nv_bfloat162*>(&u.w);
  __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
  return fmaxf(__low2float(m), __high2float(m));
}
__device__ __forceinline__ float vec_max(uint4 u, float) {
  return fmaxf(fmaxf(__uint_as_float(u.x), __uint_as_float(u.y)),
               fmaxf(__uint_as_float(u.z), __uint_as_float(u.w)));
}

// Element e of a 16-byte vector as float.
__device__ __forceinline__ float vec_elem(uint4 u, int e, __nv_bfloat16) {
  const uint32_t w = e < 4 ? (e < 2 ? u.x : u.y) : (e < 6 ? u.z : u.w);
  return __uint_as_float((e & 1) ? (w & 0xffff0000u) : (w << 16));
}
__device__ __forceinline__ float vec_elem(uint4 u, int e, float) {
  const uint32_t w = e < 2 ? (e == 0 ? u.x : u.y) : (e == 2 ? u.z : u.w);
  return __uint_as_float(w);
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T, bool kVec>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
target_greedy_accept_kernel(const T* __restrict__ logits, int64_t row_stride, int n_max, int V,
                            TargetPlan plan, const int32_t* __restrict__ parent,
                            const int32_t* __restrict__ token,
                            const int32_t* __restrict__ n_nodes, int L,
                            int32_t* __restrict__ target_tok, int32_t* __restrict__ accept_len,
                            int32_t* __restrict__ accepted_nodes,
                            int32_t* __restrict__ bonus_tok, unsigned long long* keys,
                            unsigned* tickets) {
  dep_enter();
  constexpr int W = kVec ? static_cast<int>(16 / sizeof(T)) : 1;
  const int row = blockIdx.x / plan.splits;
  const int split = blockIdx.x - row * plan.splits;
  const int b = row / n_max;
  const int i = row - b * n_max;
  const int n = min(max(n_nodes[b], 1), n_max);
  if (i >= n) return;
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  const T* x = logits + static_cast<int64_t>(row) * row_stride;

  // ---- this CTA's slice: vectors [v0, v1), plus the scalar tail on the last split
  const int64_t v0 = split * plan.chunk;
  const int64_t v1 = min(v0 + plan.chunk, plan.nvec);
  float best = -INFINITY;
  int64_t idx = -1;
  if (v0 + tid < v1) {
    if constexpr (kVec) {
      // batches of up to kBatch vectors per thread, all loads in flight before
      // any compare; within a thread vectors are visited in index order
      const uint4* xv = reinterpret_cast<const uint4*>(x);
      int64_t bv = v0 + tid;
      uint4 bu = make_uint4(0, 0, 0, 0);
      for (int64_t base = v0 + tid; base < v1; base += kBatch * kThreads) {
        uint4 u[kBatch];
#pragma unroll
        for (int r = 0; r < kBatch; ++r)
          if (base + r * kThreads < v1) u[r] = __ldcs(xv + base + r * kThreads);
#pragma unroll
        for (int r = 0; r < kBatch; ++r) {
          if (base + r * kThreads < v1) {
            const float m = vec_max(u[r], T());
            if (idx < 0 || m > best) {
              best = m;
              bv = base + r * kThreads;
              bu = u[r];
              idx = 0;
            }
          }
        }
      }
      // lowest element of the winning vector equal to the maximum
      int e = W - 1;
#pragma unroll
      for (int k = W - 2; k >= 0; --k)
        if (vec_elem(bu, k, T()) == best) e = k;
      idx = bv * W + e;
    } else {
      int64_t bv = v0 + tid;
      best = to_f32(x[bv]);
      for (int64_t v = bv + kThreads; v < v1; v += kThreads) {
        const float m = to_f32(x[v]);
        if (m > best) {
          best = m;
          bv = v;
        }
      }
      idx = bv;
    }
  }
  if (kVec && split == plan.splits - 1) {
    // elements past the last full vector; their indices exceed every vector's
    const int64_t t = plan.nvec * W + tid;
    if (t < V) {
      const float m = to_f32(x[t]);
      if (idx < 0 || m > best) {
        best = m;
        idx = t;
      }
    }
  }

  // ---- CTA reduction to one key, merged into the row's word
  __shared__ unsigned long long s_key[kWarps];
  __shared__ int s_last;
  unsigned long long key =
      idx < 0 ? 0ull
              : (static_cast<unsigned long long>(f32_to_ordered(best)) << 32) |
                    (0xffffffffu - static_cast<uint32_t>(idx));
  key = warp_max_u64(key);
  if (lane == 0) s_key[warp] = key;
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < kWarps; ++w) key = max(key, s_key[w]);
    atomicMax(keys + row, key);
    // acq_rel: releases this CTA's key before its ticket, and the CTA that
    // takes the last ticket acquires every earlier CTA's key
    unsigned old;
    asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], 1;"
                 : "=r"(old) : "l"(tickets + b) : "memory");
    s_last = old == static_cast<unsigned>(n) * plan.splits - 1;
  }
  __syncthreads();
  if (!s_last) return;

  // ---- last CTA of request b: decode, reset the workspace, walk
  __shared__ int32_t s_tt[TAPS_MAX_NODES];
  __shared__ int32_t s_par[TAPS_MAX_NODES];
  __shared__ int32_t s_tok[TAPS_MAX_NODES];
  __shared__ int32_t s_match[TAPS_MAX_NODES];
  const int64_t o = static_cast<int64_t>(b) * n_max;
  for (int j = tid; j < n_max; j += kThreads) {
    int32_t t = -1;
    if (j < n) {
      const unsigned long long k = __ldcg(keys + o + j);
      t = static_cast<int32_t>(0xffffffffu - static_cast<uint32_t>(k));
      keys[o + j] = 0ull;
      s_tt[j] = t;
      s_par[j] = parent[o + j];
      s_tok[j] = token[o + j];
    }
    target_tok[o + j] = t;
  }
  if (tid == 0) tickets[b] = 0u;
  __syncthreads();
  accept_walk(s_par, s_tok, s_tt, s_match, n, L,
              accepted_nodes + static_cast<int64_t>(b) * (L + 1), accept_len + b, bonus_tok + b);
}

TargetPlan make_target_plan(int B, int n_max, int V, int W) {
  TargetPlan p;
  p.nvec = V / W;
  const int64_t rows = static_cast<int64_t>(B) * n_max;
  const int64_t want = (static_cast<int64_t>(kTargetSms) * kCtasPerSm + rows - 1) / rows;
  // at least two vectors per thread in every slice
  const int64_t most = std::max<int64_t>(1, p.nvec / (2 * kThreads));
  p.splits = static_cast<int>(std::max<int64_t>(1, std::min(want, most)));
  p.chunk = (p.nvec + p.splits - 1) / p.splits;
  if (p.chunk == 0) p.chunk = 1;
  return p;
}

struct TargetWs {
  size_t keys, tickets, total;
};

TargetWs target_ws(int B, int n_max) {
  TargetWs w;
  w.keys = 0;
  w.tickets = align_up(sizeof(unsigned long long) * static_cast<size_t>(B) * n_max, 256);
  w.total = align_up(w.tickets + sizeof(unsigned) * static_cast<size_t>(B), 256);
  return w;
}

template <typename T, bool kVec>
void launch(const void* logits, int64_t row_stride, int B, int n_max, int V,
            const int32_t* parent, const int32_t* token, const int32_t* n_nodes, int L,
            int32_t* target_tok, int32_t* accept_len, int32_t* accepted_nodes,
            int32_t* bonus_tok, char* ws, cudaStream_t s) {
  constexpr int W = kVec ? static_cast<int>(16 / sizeof(T)) : 1;
  const TargetPlan p = make_target_plan(B, n_max, V, W);
  const TargetWs w = target_ws(B, n_max);
  const int64_t grid = static_cast<int64_t>(B) * n_max * p.splits;
  launch_dep(target_greedy_accept_kernel<T, kVec>, dim3(static_cast<unsigned>(grid)),
             dim3(kThreads), 0, s, static_cast<const T*>(logits), row_stride, n_max, V, p, parent,
             token, n_nodes, L, target_tok, accept_len, accepted_nodes, bonus_tok,
             reinterpret_cast<unsigned long long*>(ws + w.keys),
             reinterpret_cast<unsigned*>(ws + w.tickets));
}

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" size_t taps_target_greedy_accept_workspace_bytes(int B, int n_max) {
  if (B <= 0 || n_max <= 0) return 0;
  return target_ws(B, n_max).total;
}

extern "C" int taps_target_greedy_accept(const void* verify_logits, int dtype,
                                         int64_t row_stride, int B, int n_max, int V,
                                         const int32_t* parent, const int32_t* token,
                                         const int32_t* n_nodes, int L, int32_t* target_tok,
                                         int32_t* accept_len, int32_t* accepted_nodes,
                                         int32_t* bonus_tok, void* ws, size_t ws_bytes,
                                         void* stream) {
  if (!verify_logits || !parent || !token || !n_nodes || !target_tok || !accept_len ||
      !accepted_nodes || !bonus_tok)
    return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || n_max <= 0 || V <= 0 || L < 0 || row_stride < V) return TAPS_ERR_INVALID_ARG;
  if (dtype != TAPS_F32 && dtype != TAPS_BF16) return TAPS_ERR_INVALID_ARG;
  if (n_max > TAPS_MAX_NODES || L > TAPS_MAX_L) return TAPS_ERR_UNSUPPORTED;
  const int64_t rows = static_cast<int64_t>(B) * n_max;
  if (rows * make_target_plan(B, n_max, V, 1).splits > 0x7fffffffLL) return TAPS_ERR_UNSUPPORTED;
  if (!ws || !aligned(ws, 256) || ws_bytes < target_ws(B, n_max).total) return TAPS_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  const size_t esz = dtype == TAPS_F32 ? 4 : 2;
  const bool vec = aligned(verify_logits, 16) && (row_stride * esz) % 16 == 0;
  if (dtype == TAPS_BF16) {
    if (vec)
      launch<__nv_bfloat16, true>(verify_logits, row_stride, B, n_max, V, parent, token, n_nodes,
                                  L, target_tok, accept_len, accepted_nodes, bonus_tok, w, s);
    else
      launch<__nv_bfloat16, false>(verify_logits, row_stride, B, n_max, V, parent, token,
                                   n_nodes, L, target_tok, accept_len, accepted_nodes, bonus_tok,
                                   w, s);
  } else {
    if (vec)
      launch<float, true>(verify_logits, row_stride, B, n_max, V, parent, token, n_nodes, L,
                          target_tok, accept_len, accepted_nodes, bonus_tok, w, s);
    else
      launch<float, false>(verify_logits, row_stride, B, n_max, V, parent, token, n_nodes, L,
                           target_tok, accept_len, accepted_nodes, bonus_tok, w, s);
  }
  return launch_status();
}
