// Device helpers shared by the two stage-1 kernels (topk.cu, topk_cluster.cu):
// running softmax statistics in log2 units, the 64-bit top-K keys, and the
// rank-based selections of a CTA's top-KP. Internal to the library.
#pragma once

#include "common.cuh"

namespace taps {

// Stage 1 for a few rows (topk_cluster.cu): one thread-block cluster per row,
// merged on chip. Returns TAPS_OK or TAPS_ERR_CUDA after launching, or -1
// (nothing launched) when the shape is left to topk_marginals_kernel.
int topk_cluster_try(const void* logits, int dtype, int64_t row_stride, int R, int V, int K,
                     int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s);
// Stage 1 for many rows (topk_stream.cu): one CTA streams one row. Same
// return convention.
int topk_stream_try(const void* logits, int dtype, int64_t row_stride, int R, int V, int K,
                    int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s);

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

int round_kp(int K) {
  int kp = 1;
  while (kp < K) kp <<= 1;
  return kp;
}

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Running softmax statistics in log2 units: m2 = max x*log2(e),
// z = sum 2^(x2 - m2), t2 = sum 2^(x2 - m2) * (x2 - m2).
struct Stats {
  float m2, z, t2;
};

__device__ __forceinline__ void stats_raise(Stats& s, float m2_new) {
  if (m2_new > s.m2) {
    if (s.z > 0.f) {
      float dm = s.m2 - m2_new;
      float sc = ex2f(dm);
      s.t2 = sc * fmaf(s.z, dm, s.t2);
      s.z *= sc;
    }
    s.m2 = m2_new;
  }
}

__device__ __forceinline__ void stats_add(Stats& s, float x2) {
  if (x2 > -INFINITY) {
    float dx = x2 - s.m2;
    float e = ex2f(dx);
    s.z += e;
    s.t2 = fmaf(e, dx, s.t2);
  }
}

__device__ __forceinline__ Stats stats_merge(Stats a, Stats b) {
  float m = fmaxf(a.m2, b.m2);
  Stats r{m, 0.f, 0.f};
  if (a.z > 0.f) {
    float d = a.m2 - m;
    float s = ex2f(d);
    r.z += s * a.z;
    r.t2 += s * fmaf(a.z, d, a.t2);
  }
  if (b.z > 0.f) {
    float d = b.m2 - m;
    float s = ex2f(d);
    r.z += s * b.z;
    r.t2 += s * fmaf(b.z, d, b.t2);
  }
  return r;
}

__device__ __forceinline__ uint64_t make_key(float x, uint32_t id) {
  return (static_cast<uint64_t>(f32_to_ordered(x)) << 32) | static_cast<uint32_t>(~id);
}

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}

// The KP largest of n <= 256 keys in shared memory (unique, 0 = none), by one
// warp: each lane holds eight of them in registers, then KP rounds of a warp
// maximum. Writes out[0, KP) descending (zero-padded).
template <int KP, int R = 8>
__device__ void warp_top(const uint64_t* cand, int n, uint64_t* out, int lane) {
  uint64_t c[R];
#pragma unroll
  for (int i = 0; i < R; ++i) c[i] = lane + 32 * i < n ? cand[lane + 32 * i] : 0ull;
#pragma unroll 1
  for (int r = 0; r < KP; ++r) {
    uint64_t mine = 0;
#pragma unroll
    for (int i = 0; i < R; ++i) mine = c[i] > mine ? c[i] : mine;
    const uint64_t best = warp_max_u64(mine);
    if (lane == 0) out[r] = best;
    if (best != 0 && mine == best) {
#pragma unroll
      for (int i = 0; i < R; ++i) c[i] = c[i] == best ? 0ull : c[i];
    }
  }
}

// Candidate c of cand[0, n) goes to out[rank] when its rank (keys above it,
// equal keys ordered by index; only empty entries, 0, can be equal) is below
// KP. One thread per candidate; the loads are broadcasts.
template <int KP>
__device__ __forceinline__ void rank_into(const uint64_t* cand, int n, int c, uint64_t* out) {
  const uint64_t mine = cand[c];
  int rank = 0;
  int i = 0;
  for (; i + 3 < n; i += 4) {
    const uint64_t a0 = cand[i], a1 = cand[i + 1], a2 = cand[i + 2], a3 = cand[i + 3];
    rank += (a0 > mine || (a0 == mine && i < c)) + (a1 > mine || (a1 == mine && i + 1 < c)) +
            (a2 > mine || (a2 == mine && i + 2 < c)) + (a3 > mine || (a3 == mine && i + 3 < c));
  }
  for (; i < n; ++i) rank += cand[i] > mine || (cand[i] == mine && i < c);
  if (rank < KP) out[rank] = mine;
}

// Top-KP of cand[0, n) into out[0, KP), descending, called by every thread
// of the CTA. thr is a key that at least KP of the candidates reach (0 when
// none is known): a candidate below it has KP candidates above it, so only
// the few at or above it are compacted into comp (one shared atomic per warp)
// and ranked among themselves. *ncomp is 0 on entry and is left at 0. When
// more than cap candidates reach thr, they are ranked with warp maxima.
template <int KP, int NT = kThreads>
__device__ void select_top(const uint64_t* cand, int n, uint64_t thr, uint64_t* comp, int cap,
                           int* ncomp, uint64_t* out, uint64_t* part) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i0 = warp * 32; i0 < n; i0 += NT) {
    const int i = i0 + lane;
    const uint64_t k = i < n ? cand[i] : 0ull;
    const bool keep = i < n && k >= thr;
    const unsigned b = __ballot_sync(kFullMask, keep);
    int base = 0;
    if (lane == 0 && b) base = atomicAdd(ncomp, __popc(b));
    base = __shfl_sync(kFullMask, base, 0);
    const int idx = base + __popc(b & ((1u << lane) - 1u));
    if (keep && idx < cap) comp[idx] = k;
  }
  __syncthreads();
  const int m = *ncomp;
  if (m <= cap) {
    for (int c = tid; c < m; c += NT) rank_into<KP>(comp, m, c, out);
  } else {
    // each warp reduces a slice of at most 32 R keys, then warp 0 the results
    const int slice = (n + NT / 32 - 1) / (NT / 32);
    const int lo = min(n, warp * slice), hi = min(n, lo + slice);
    constexpr int R = NT / 32 > 8 ? NT / 32 : 8;
    warp_top<KP, R>(cand + lo, hi - lo, part + warp * KP, lane);
    __syncthreads();
    if (warp == 0) warp_top<KP, R>(part, (NT / 32) * KP, out, lane);
  }
  __syncthreads();
  if (tid == 0) *ncomp = 0;
}

__device__ __forceinline__ Stats warp_stats(Stats s) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Stats o;
    o.m2 = __shfl_xor_sync(kFullMask, s.m2, off);
    o.z = __shfl_xor_sync(kFullMask, s.z, off);
    o.t2 = __shfl_xor_sync(kFullMask, s.t2, off);
    s = stats_merge(s, o);
  }
  return s;
}

template <int KP>
__device__ void write_row(int row, int K, const uint64_t* top, Stats st, int lane,
                          int32_t* ids, float* logp, float* lse, float* ent) {
  float xmax = ordered_to_f32(static_cast<uint32_t>(top[0] >> 32));
  float lz = logf(st.z);
  float l = xmax + lz;
  if (lane == 0) {
    lse[row] = l;
    ent[row] = lz - (st.t2 * kLn2) / st.z;
  }
  for (int k = lane; k < K; k += 32) {
    uint64_t key = top[k];
    ids[static_cast<int64_t>(row) * K + k] = static_cast<int32_t>(~static_cast<uint32_t>(key));
    logp[static_cast<int64_t>(row) * K + k] =
        ordered_to_f32(static_cast<uint32_t>(key >> 32)) - l;
  }
}

}  // namespace
}  // namespace taps
