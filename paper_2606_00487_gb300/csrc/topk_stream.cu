// Stage 1 of a TAPS round (Sec. 4.1 stage 1, Sec. 4.2 scorer features) for
// many rows (a batched round: 32 requests x 16 positions): one CTA streams one
// whole row.
//
// The row passes through a four-stage ring in shared memory of 8 KB stages
// (each thread copying the two 16-byte vectors it reads with asynchronous
// copies, three stages ahead), four CTAs per SM, so that every row of a
// 512-row batch is in flight at once. Per stage, each thread takes its two
// vectors:
//   - softmax statistics online in log2 units (running max m2, sum of
//     2^(x2-m2), sum of 2^(x2-m2)(x2-m2)), rescaled when the thread's maximum
//     grows, in packed f32x2 pairs;
//   - candidates: the elements whose key (ordered value << 32 | ~token id)
//     reaches the CTA's running threshold key are listed in shared memory
//     with one shared atomic each, a vector being visited only when its
//     maximum reaches the threshold's value.
// The first threshold is the largest over the warps of the KP-th largest lane
// maximum of the first stage (at least KP elements reach it). When the list
// grows past 128 entries it is compacted (ranked by counting): its KP-th
// largest key becomes the threshold and only the KP keys above it stay
// listed, so that the threshold soon follows the row's running top-KP. A
// stage that overflows the list (1,024 entries) is listed again above the
// raised threshold, from the copy still in shared memory; each compaction
// raises the threshold strictly (the listed keys are distinct), so the
// re-listing ends. At the end the list is ranked by counting.
#include <algorithm>
#include <atomic>

#include "common.cuh"
#include "sm100.cuh"
#include "topk_common.cuh"

namespace taps {
namespace {

using sm100::add_f32x2;
using sm100::f32x2;
using sm100::f32x2_split;
using sm100::fma_f32x2;
using sm100::mul_f32x2;

constexpr int kStStages = 4;
constexpr int kStStageVecs = 2 * kThreads;                 // 16-byte vectors per stage (8 KB)
constexpr int kStCap = 1024;                               // listed candidates at most
constexpr int kStCompactAt = 128;                          // compact above this

__device__ __forceinline__ uint32_t word4(const uint4& v, int i) {
  return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}
template <typename T>
__device__ __forceinline__ float elem(const uint4& v, int e);
template <>
__device__ __forceinline__ float elem<float>(const uint4& v, int e) {
  return __uint_as_float(word4(v, e));
}
template <>
__device__ __forceinline__ float elem<__nv_bfloat16>(const uint4& v, int e) {
  const uint32_t w = word4(v, e >> 1);
  return __uint_as_float((e & 1) ? (w & 0xFFFF0000u) : (w << 16));
}
template <typename T>
__device__ __forceinline__ float vmax_of(const uint4& v) {
  if constexpr (sizeof(T) == 4) {
    return fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                 fmaxf(__uint_as_float(v.z), __uint_as_float(v.w)));
  } else {
    const float a = sm100::max3f(elem<T>(v, 0), elem<T>(v, 1), elem<T>(v, 2));
    const float b = sm100::max3f(elem<T>(v, 3), elem<T>(v, 4), elem<T>(v, 5));
    return sm100::max3f(a, b, fmaxf(elem<T>(v, 6), elem<T>(v, 7)));
  }
}

// grid (rows), 256 threads; the row's V / VE whole 16-byte vectors in stages
// of kStStageVecs, then the V mod VE elements after them.
template <int KP, typename T>
__global__ void __launch_bounds__(kThreads, 4)
topk_stream_kernel(const T* __restrict__ logits, int64_t row_stride, int V, int K,
                   int32_t* __restrict__ ids, float* __restrict__ logp, float* __restrict__ lse,
                   float* __restrict__ ent) {
  constexpr int VE = 16 / sizeof(T);
  constexpr int kStageElems = kStStageVecs * VE;
  __shared__ __align__(128) uint4 s_ring[kStStages][kStStageVecs];
  __shared__ uint64_t s_list[kStCap];
  __shared__ uint64_t s_top[KP];
  __shared__ Stats s_wst[kWarps];
  __shared__ unsigned long long s_thr;   // running threshold key
  __shared__ int s_n;                    // listed candidates (runs on past kStCap)

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int row = static_cast<int>(blockIdx.x);
  if (tid == 0) {
    s_thr = 0ull;
    s_n = 0;
  }
  if (tid < KP) s_top[tid] = 0ull;
  __syncthreads();
  dep_enter();

  const T* x = logits + static_cast<int64_t>(row) * row_stride;
  const uint4* xv = reinterpret_cast<const uint4*>(x);
  const int nvec = V / VE;
  const int nst = (nvec + kStStageVecs - 1) / kStStageVecs;
  // Each thread copies the two vectors of a stage it will read itself into
  // its own slots of the ring (16-byte asynchronous copies, L2 only, one
  // commit group per stage), kStStages - 1 stages ahead: no barrier guards the
  // ring, and every thread keeps its own copies in flight.
  auto issue = [&](int s) {
    const int v0 = s * kStStageVecs;
    const int nv = min(kStStageVecs, nvec - v0);
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int i = tid + u * kThreads;
      if (s < nst && i < nv)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                         sm100::smem_u32(&s_ring[s % kStStages][i])),
                     "l"(xv + v0 + i)
                     : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
#pragma unroll
  for (int s = 0; s < kStStages - 1; ++s) issue(s);

  // online statistics relative to the thread's running maximum m2
  float m2 = -INFINITY;
  uint64_t zp = f32x2(0.f, 0.f), tp = f32x2(0.f, 0.f);
  const uint64_t l2e = f32x2(kLog2e, kLog2e);
  auto raise = [&](float m2_new) {
    if (m2_new > m2) {
      if (m2 > -INFINITY) {
        const float dm = m2 - m2_new;
        const float sc = ex2f(dm);
        tp = mul_f32x2(f32x2(sc, sc), fma_f32x2(zp, f32x2(dm, dm), tp));
        zp = mul_f32x2(zp, f32x2(sc, sc));
      }
      m2 = m2_new;
    }
  };
  auto accumulate = [&](const uint4& v) {
    const uint64_t nm2 = f32x2(-m2, -m2);
#pragma unroll
    for (int e = 0; e < VE; e += 2) {
      float d0, d1;
      f32x2_split(fma_f32x2(f32x2(elem<T>(v, e), elem<T>(v, e + 1)), l2e, nm2), d0, d1);
      d0 = fmaxf(d0, -127.f);
      d1 = fmaxf(d1, -127.f);
      const uint64_t ee = f32x2(ex2f(d0), ex2f(d1));
      zp = add_f32x2(zp, ee);
      tp = fma_f32x2(ee, f32x2(d0, d1), tp);
    }
  };
  // list the elements of vector v (token ids from id0) whose key reaches thr
  auto list_vec = [&](const uint4& v, float vm, int id0, uint64_t thr, float tv) {
    if (vm >= tv) {
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const float xe = elem<T>(v, e);
        if (xe >= tv) {
          const uint64_t k = make_key(xe, static_cast<uint32_t>(id0 + e));
          if (k >= thr) {
            const int j = atomicAdd(&s_n, 1);
            if (j < kStCap) s_list[j] = k;
          }
        }
      }
    }
  };
  auto thr_value = [](uint64_t t) {
    return t ? ordered_to_f32(static_cast<uint32_t>(t >> 32)) : -INFINITY;
  };

#pragma unroll 1
  for (int s = 0; s < nst; ++s) {
    const int slot = s % kStStages;
    issue(s + kStStages - 1);   // into the slot stage s - 1 used (read by this thread only)
    asm volatile("cp.async.wait_group %0;" ::"n"(kStStages - 1) : "memory");
    const int v0 = s * kStStageVecs;
    const int nv = min(kStStageVecs, nvec - v0);
    uint4 v[2];
    float vm[2];
    bool live[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int i = tid + u * kThreads;
      live[u] = i < nv;
      v[u] = live[u] ? s_ring[slot][i] : make_uint4(0, 0, 0, 0);
      vm[u] = live[u] ? vmax_of<T>(v[u]) : -INFINITY;
    }
    const float smax = fmaxf(vm[0], vm[1]);
    if (smax > -INFINITY) {
      raise(smax * kLog2e);
#pragma unroll
      for (int u = 0; u < 2; ++u)
        if (live[u]) accumulate(v[u]);
    }
    if (s == 0) {
      // first threshold: per warp the KP-th largest lane maximum counted
      // with multiplicity; the CTA keeps the largest (as a key: every key of
      // that value reaches it)
      uint32_t cur = (live[0] || live[1]) ? f32_to_ordered(smax) : 0u;
      int need = KP;
      uint32_t tw = 0u;
#pragma unroll 1
      while (need > 0) {
        const uint32_t m = __reduce_max_sync(kFullMask, cur);
        if (m == 0u) break;
        need -= __popc(__ballot_sync(kFullMask, cur == m));
        tw = m;
        if (cur == m) cur = 0u;
      }
      if (lane == 0 && need <= 0) atomicMax(&s_thr, static_cast<unsigned long long>(tw) << 32);
      __syncthreads();
    }
    uint64_t thr = *reinterpret_cast<volatile unsigned long long*>(&s_thr);
#pragma unroll
    for (int u = 0; u < 2; ++u)
      if (live[u]) list_vec(v[u], vm[u], (v0 + tid + u * kThreads) * VE, thr, thr_value(thr));
    __syncthreads();   // the stage is read and listed
    int n = s_n;
#pragma unroll 1
    while (n > kStCompactAt) {
      // the KP-th largest listed key becomes the threshold; the KP keys above
      // it stay. If the list overflowed, only this stage can have lost
      // candidates: it is listed again above the new threshold, except for
      // the keys already kept.
      const bool overflow = n > kStCap;
      if (tid < KP) s_top[tid] = 0ull;
      __syncthreads();
      const int nl = min(n, kStCap);
      for (int c = tid; c < nl; c += kThreads) rank_into<KP>(s_list, nl, c, s_top);
      __syncthreads();
      thr = s_top[KP - 1];
      const int lo = v0 * VE, hi = lo + kStageElems;   // this stage's token ids
      __syncthreads();
      if (tid == 0) {
        int m = 0;
        for (int r = 0; r < KP; ++r) {
          const uint64_t k = s_top[r];
          const int id = static_cast<int>(~static_cast<uint32_t>(k));
          if (k != 0ull && !(overflow && id >= lo && id < hi)) s_list[m++] = k;
        }
        s_n = m;
        s_thr = thr;
      }
      __syncthreads();
      if (overflow) {
#pragma unroll
        for (int u = 0; u < 2; ++u)
          if (live[u]) list_vec(v[u], vm[u], (v0 + tid + u * kThreads) * VE, thr, thr_value(thr));
      }
      __syncthreads();
      n = s_n;
    }
  }
  // the elements after the last whole vector
  {
    const int tail_id = nvec * VE + tid;
    if (tail_id < V) {
      const float xt = to_f32<T>(x[tail_id]);
      if (xt > -INFINITY) {
        raise(xt * kLog2e);
        const float d = fmaxf(fmaf(xt, kLog2e, -m2), -127.f);
        const float e = ex2f(d);
        zp = add_f32x2(zp, f32x2(e, 0.f));
        tp = fma_f32x2(f32x2(e, 0.f), f32x2(d, 0.f), tp);
      }
      const uint64_t thr = s_thr;
      const uint64_t k = make_key(xt, static_cast<uint32_t>(tail_id));
      if (k >= thr) {
        const int j = atomicAdd(&s_n, 1);
        if (j < kStCap) s_list[j] = k;
      }
    }
  }
  float z0, z1, t0, t1;
  f32x2_split(zp, z0, z1);
  f32x2_split(tp, t0, t1);
  Stats st{m2, z0 + z1, t0 + t1};
  if (!(st.z > 0.f)) st = Stats{-INFINITY, 0.f, 0.f};
  st = warp_stats(st);
  if (lane == 0) s_wst[warp] = st;
  __syncthreads();
  // the tail can push the list past kStCap only with fewer than VE more keys
  // than a compacted list holds, far below it
  const int n = min(s_n, kStCap);
  if (tid < KP) s_top[tid] = 0ull;
  __syncthreads();
  for (int c = tid; c < n; c += kThreads) rank_into<KP>(s_list, n, c, s_top);
  __syncthreads();
  if (warp == 0) {
    const Stats cs = warp_stats(lane < kWarps ? s_wst[lane] : Stats{-INFINITY, 0.f, 0.f});
    write_row<KP>(row, K, s_top, cs, lane, ids, logp, lse, ent);
  }
}

template <int KP, typename T>
int launch_stream(const void* logits, int64_t row_stride, int R, int V, int K, int32_t* ids,
                  float* logp, float* lse, float* ent, cudaStream_t s) {
  // four CTAs of ~41 KB per SM need the largest shared-memory carveout: ask
  // for it once per device (the flags are atomics: several host threads may
  // call)
  static std::atomic<bool> carveout[64];
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64 &&
      !carveout[dev].load(std::memory_order_acquire)) {
    if (cudaFuncSetAttribute(topk_stream_kernel<KP, T>,
                             cudaFuncAttributePreferredSharedMemoryCarveout,
                             static_cast<int>(cudaSharedmemCarveoutMaxShared)) == cudaSuccess)
      carveout[dev].store(true, std::memory_order_release);
    cudaGetLastError();
  }
  if (launch_dep(topk_stream_kernel<KP, T>, dim3(R), dim3(kThreads), 0, s,
                 static_cast<const T*>(logits), row_stride, V, K, ids, logp, lse, ent) !=
      cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}

template <typename T>
int dispatch_stream(int kp, const void* logits, int64_t row_stride, int R, int V, int K,
                    int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s) {
  switch (kp) {
    case 1: return launch_stream<1, T>(logits, row_stride, R, V, K, ids, logp, lse, ent, s);
    case 2: return launch_stream<2, T>(logits, row_stride, R, V, K, ids, logp, lse, ent, s);
    case 4: return launch_stream<4, T>(logits, row_stride, R, V, K, ids, logp, lse, ent, s);
    case 8: return launch_stream<8, T>(logits, row_stride, R, V, K, ids, logp, lse, ent, s);
    case 16: return launch_stream<16, T>(logits, row_stride, R, V, K, ids, logp, lse, ent, s);
    default: return launch_stream<32, T>(logits, row_stride, R, V, K, ids, logp, lse, ent, s);
  }
}

}  // namespace

int topk_stream_try(const void* logits, int dtype, int64_t row_stride, int R, int V, int K,
                    int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s) {
  const size_t esz = dtype == TAPS_F32 ? 4 : 2;
  if (!aligned(logits, 16) || (row_stride * static_cast<int64_t>(esz)) % 16 != 0) return -1;
  // one CTA per row pays off once the rows alone fill the GPU
  if (R < 2 * kTargetSms) return -1;
  const int kp = round_kp(K);
  return dtype == TAPS_F32
             ? dispatch_stream<float>(kp, logits, row_stride, R, V, K, ids, logp, lse, ent, s)
             : dispatch_stream<__nv_bfloat16>(kp, logits, row_stride, R, V, K, ids, logp, lse,
                                              ent, s);
}

}  // namespace taps
