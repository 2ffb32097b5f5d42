// Stage 1 of a TAPS round (Sec. 4.1 stage 1, Sec. 4.2 scorer features) for a
// few rows at a time (a batch-1 round: L = 16 rows of a 151,936-token
// vocabulary): one thread-block cluster per row, merged on chip.
//
// Each CTA of a row's cluster copies a contiguous slice of the row into shared
// memory (a few bulk copies), and computes:
//   - the slice's softmax statistics in log2 units (max m2, sum of 2^(x2-m2),
//     sum of 2^(x2-m2) (x2-m2)), each thread relative to its own maximum,
//     merged across lanes and warps;
//   - a value threshold: per warp, the KP-th largest of the lanes' maxima
//     counted with multiplicity is a value that at least KP elements reach;
//     the largest over the warps bounds the slice's KP-th largest value from
//     below, so only elements at or above it can be among the slice's top-KP
//     keys (a key is ordered value << 32 | ~token id: larger keys rank first,
//     equal values go to the lower token id);
//   - the slice's top-KP: the elements at or above the threshold are listed in
//     shared memory and ranked by counting.
// Every CTA then writes its top-KP and statistics into the shared memory of the
// cluster's first CTA (distributed shared memory); after one cluster barrier
// one warp of that CTA merges them by rank and writes the row's outputs. No
// partial record goes through global memory, no counter, no workspace. The
// host launches this kernel only when every row's cluster can be resident at
// once; otherwise topk_stream_kernel (topk_stream.cu, from 304 rows) or
// topk_marginals_kernel (topk.cu) runs.
#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "sm100.cuh"
#include "topk_common.cuh"

namespace taps {
namespace {

using sm100::add_f32x2;
using sm100::f32x2;
using sm100::f32x2_split;
using sm100::fma_f32x2;

constexpr int kClThreads = 256;       // 8 warps; two CTAs per SM
constexpr int kClWarps = kClThreads / 32;
constexpr int kClCap = 1024;          // candidates one CTA ranks by counting
constexpr int kClMaxCluster = 16;
constexpr int kClMaxNv = 16;          // 16-byte vectors per thread at most (64 KB a CTA)

__device__ __forceinline__ void st_cluster_u64(uint32_t addr, uint64_t v) {
  asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(addr), "l"(v) : "memory");
}

__device__ __forceinline__ void st_cluster_f32x4(uint32_t addr, float a, float b, float c,
                                                 float d) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b),
               "f"(c), "f"(d)
               : "memory");
}

__device__ __forceinline__ uint32_t word(const uint4& v, int i) {
  return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// Element e of a 16-byte vector as f32 (e is a constant after unrolling).
template <typename T>
__device__ __forceinline__ float vec_elem(const uint4& v, int e);
template <>
__device__ __forceinline__ float vec_elem<float>(const uint4& v, int e) {
  return __uint_as_float(word(v, e));
}
template <>
__device__ __forceinline__ float vec_elem<__nv_bfloat16>(const uint4& v, int e) {
  const uint32_t w = word(v, e >> 1);
  return __uint_as_float((e & 1) ? (w & 0xFFFF0000u) : (w << 16));
}

// Vector maximum as a tree of three-input maxima.
template <typename T>
__device__ __forceinline__ float vec_max(const uint4& v) {
  if constexpr (sizeof(T) == 4) {
    return fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                 fmaxf(__uint_as_float(v.z), __uint_as_float(v.w)));
  } else {
    const float a = sm100::max3f(vec_elem<T>(v, 0), vec_elem<T>(v, 1), vec_elem<T>(v, 2));
    const float b = sm100::max3f(vec_elem<T>(v, 3), vec_elem<T>(v, 4), vec_elem<T>(v, 5));
    return sm100::max3f(a, b, fmaxf(vec_elem<T>(v, 6), vec_elem<T>(v, 7)));
  }
}

// The row's outputs from its top keys (any order; position r of the key in
// descending order given) and statistics: lse = xmax + ln z, entropy =
// ln z - t2 ln(2) / z, logp = logit - lse.
__device__ __forceinline__ void write_entry(int row, int K, int r, uint64_t key, float xmax,
                                            Stats st, int32_t* ids, float* logp) {
  const float l = xmax + logf(st.z);
  ids[static_cast<int64_t>(row) * K + r] = static_cast<int32_t>(~static_cast<uint32_t>(key));
  logp[static_cast<int64_t>(row) * K + r] = ordered_to_f32(static_cast<uint32_t>(key >> 32)) - l;
}

// grid (C, rows), cluster (C, 1, 1): CTA `rank` of row `row` copies the
// vectors [rank * per, rank * per + per) of the row's V / VE whole 16-byte
// vectors into dynamic shared memory (per <= kClMaxNv * kClThreads); the last
// CTA also reads the V mod VE elements after them. Thread t owns the vectors
// t, t + kClThreads, ... of the slice.
template <int KP, typename T>
__global__ void __launch_bounds__(kClThreads, 2)
topk_cluster_kernel(const T* __restrict__ logits, int64_t row_stride, int V, int K, int per,
                    int32_t* __restrict__ ids, float* __restrict__ logp,
                    float* __restrict__ lse, float* __restrict__ ent) {
  constexpr int VE = 16 / sizeof(T);
  extern __shared__ __align__(128) uint4 s_vec[];     // the slice
  __shared__ uint64_t s_list[kClCap];                 // candidates; the first CTA's merge list
  __shared__ uint64_t s_top[KP];                      // this slice's top-KP, descending
  __shared__ uint64_t s_part[kClWarps * KP];
  __shared__ uint64_t s_ckeys[kClMaxCluster * KP];    // [CTA][KP], written by the cluster's CTAs
  __shared__ float4 s_cst[kClMaxCluster];             // [CTA] statistics (m2, z, t2)
  __shared__ float s_vmax[kClMaxNv * kClThreads];     // [vector i][thread] maxima
  __shared__ Stats s_wst[kClWarps];
  __shared__ __align__(8) uint64_t s_bar;             // the slice's copies landed
  __shared__ unsigned s_vthr;   // ordered value that at least KP elements of the slice reach
  __shared__ int s_n;           // listed candidates
  __shared__ int s_nc;          // select_top's compaction counter (zero between calls)

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int C = static_cast<int>(gridDim.x);
  const int rank = static_cast<int>(blockIdx.x);     // == %cluster_ctarank
  const int row = static_cast<int>(blockIdx.y);
  if (tid == 0) {
    s_vthr = 0u;
    s_n = 0;
    s_nc = 0;
    sm100::mbar_init(&s_bar, 1);
    sm100::fence_mbar_init();
  }
  if (tid < KP) s_top[tid] = 0ull;
  // This CTA runs: the cluster barrier's first phase completes once every CTA
  // of the cluster has arrived, and no CTA writes into a peer before that.
  if (C > 1) sm100::cluster_arrive_relaxed();
  __syncthreads();
  dep_enter();

  const T* x = logits + static_cast<int64_t>(row) * row_stride;
  const int nvec = V / VE;
  const int cv0 = min(nvec, rank * per);
  const int span = min(nvec, cv0 + per) - cv0;
  const int nv = span > tid ? (span - tid + kClThreads - 1) / kClThreads : 0;
  if (warp == 0) {
    // the slice in up to eight bulk copies, one per lane (16-byte multiples)
    if (lane == 0) sm100::mbar_arrive_expect_tx(&s_bar, static_cast<uint32_t>(span) * 16u);
    __syncwarp();
    const int piece = (span + 7) / 8;
    const int off = lane * piece;
    const int cnt = lane < 8 ? min(piece, span - off) : 0;
    if (cnt > 0)
      sm100::bulk_load(sm100::smem_u32(s_vec + off), reinterpret_cast<const uint4*>(x) + cv0 + off,
                       static_cast<uint32_t>(cnt) * 16u, &s_bar, sm100::l2_evict_first_policy());
  }
  const int tail_id = nvec * VE + tid;
  const bool has_tail = rank == C - 1 && tail_id < V;
  const float tail_x = has_tail ? to_f32<T>(x[tail_id]) : -INFINITY;
  // token id of element e of the thread's vector i: id0 + i * kIdStep + e
  const int id0 = (cv0 + tid) * VE;
  constexpr int kIdStep = kClThreads * VE;
  sm100::mbar_wait(&s_bar, 0);   // bounded; the copies read memory the caller owns

  // ---- maxima of each of the thread's vectors (kept in shared memory) and of
  // the thread. Rolled loops throughout: the kernel runs once per round, with
  // its code usually evicted from the caches in between, so compact code
  // matters more than loop overhead.
  float tmax = tail_x;
#pragma unroll 1
  for (int i = 0; i < nv; ++i) {
    const float vm = vec_max<T>(s_vec[tid + i * kClThreads]);
    s_vmax[i * kClThreads + tid] = vm;
    tmax = fmaxf(tmax, vm);
  }
  const bool any = nv > 0 || has_tail;

  // ---- value threshold: per warp, the KP-th largest lane maximum counted
  // with multiplicity (at least KP elements of the warp reach it); the CTA
  // keeps the largest over its warps
  {
    uint32_t cur = any ? f32_to_ordered(tmax) : 0u;   // 0 = no element
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
    if (lane == 0 && need <= 0) atomicMax(&s_vthr, tw);
  }

  // ---- statistics relative to the thread's maximum: d = x log2(e) - m2 in
  // one rounding, clamped at -127 so that -inf and values far below the
  // maximum give exactly 0 (ex2 with flush-to-zero) and never 0 * inf; two
  // accumulator pairs
  Stats st{-INFINITY, 0.f, 0.f};
  if (any && tmax > -INFINITY) {
    const float m2 = tmax * kLog2e;
    const uint64_t l2e = f32x2(kLog2e, kLog2e), nm2 = f32x2(-m2, -m2);
    uint64_t zp[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
    uint64_t tp[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
#pragma unroll 2
    for (int i = 0; i < nv; ++i) {
      const uint4 v = s_vec[tid + i * kClThreads];
#pragma unroll
      for (int e = 0; e < VE; e += 2) {
        float d0, d1;
        f32x2_split(fma_f32x2(f32x2(vec_elem<T>(v, e), vec_elem<T>(v, e + 1)), l2e, nm2), d0, d1);
        d0 = fmaxf(d0, -127.f);
        d1 = fmaxf(d1, -127.f);
        const uint64_t ee = f32x2(ex2f(d0), ex2f(d1));
        zp[(e >> 1) & 1] = add_f32x2(zp[(e >> 1) & 1], ee);
        tp[(e >> 1) & 1] = fma_f32x2(ee, f32x2(d0, d1), tp[(e >> 1) & 1]);
      }
    }
    float z0, z1, z2, z3, t0, t1, t2, t3;
    f32x2_split(zp[0], z0, z1);
    f32x2_split(zp[1], z2, z3);
    f32x2_split(tp[0], t0, t1);
    f32x2_split(tp[1], t2, t3);
    st = Stats{m2, (z0 + z1) + (z2 + z3), (t0 + t1) + (t2 + t3)};
    if (has_tail) stats_add(st, tail_x * kLog2e);
  }
  st = warp_stats(st);
  if (lane == 0) s_wst[warp] = st;
  __syncthreads();

  // ---- candidates: the elements whose key reaches the threshold key, listed
  // with one shared atomic each (they are few: only the vectors whose maximum
  // reaches the threshold are visited); the count runs on past the list's
  // capacity
  uint64_t thr = static_cast<uint64_t>(s_vthr) << 32;   // the smallest key of that value
  auto visit = [&](float tv, auto&& fn) {
    if (has_tail && tail_x >= tv) {
      const uint64_t k = make_key(tail_x, static_cast<uint32_t>(tail_id));
      if (k >= thr) fn(k);
    }
    uint32_t m = 0;   // the thread's vectors holding an element at or above tv
#pragma unroll 1
    for (int i = 0; i < nv; ++i) m |= s_vmax[i * kClThreads + tid] >= tv ? (1u << i) : 0u;
#pragma unroll 1
    while (m) {
      const int i = __ffs(m) - 1;
      m &= m - 1;
      const uint4 v = s_vec[tid + i * kClThreads];
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const float xe = vec_elem<T>(v, e);
        const uint64_t k = make_key(xe, static_cast<uint32_t>(id0 + i * kIdStep + e));
        if (xe >= tv && k >= thr) fn(k);
      }
    }
  };
  int n;
#pragma unroll 1
  for (;;) {
    const float tv = thr ? ordered_to_f32(static_cast<uint32_t>(thr >> 32)) : -INFINITY;
    visit(tv, [&](uint64_t k) {
      const int j = atomicAdd(&s_n, 1);
      if (j < kClCap) s_list[j] = k;
    });
    __syncthreads();
    n = s_n;
    if (n <= kClCap) break;
    // More candidates than the list holds (many large values in few lanes):
    // the KP-th largest of the listed keys is a key at least KP elements
    // reach, and above the current threshold; list again above it. Each
    // round drops at least kClCap - KP elements.
    select_top<KP, kClThreads>(s_list, kClCap, 0ull, s_list, 0, &s_nc, s_top, s_part);
    thr = s_top[KP - 1];
    __syncthreads();
    if (tid == 0) s_n = 0;
    if (tid < KP) s_top[tid] = 0ull;
    __syncthreads();
  }
  for (int c = tid; c < n; c += kClThreads) rank_into<KP>(s_list, n, c, s_top);
  __syncthreads();
  Stats cs{-INFINITY, 0.f, 0.f};
  if (warp == 0) cs = warp_stats(lane < kClWarps ? s_wst[lane] : Stats{-INFINITY, 0.f, 0.f});

  if (C == 1) {
    if (warp == 0) write_row<KP>(row, K, s_top, cs, lane, ids, logp, lse, ent);
    return;
  }
  // ---- to the first CTA of the cluster: this slice's top-KP and statistics
  sm100::cluster_wait();   // every CTA of the cluster runs
  if (warp == 0) {
    for (int r = lane; r < KP; r += 32)
      st_cluster_u64(sm100::mapa_shared(sm100::smem_u32(&s_ckeys[rank * KP + r]), 0), s_top[r]);
    if (lane == 0)
      st_cluster_f32x4(sm100::mapa_shared(sm100::smem_u32(&s_cst[rank]), 0), cs.m2, cs.z, cs.t2,
                       0.f);
  }
  sm100::cluster_sync();   // release the writes above / acquire the peers' writes
  if (rank != 0 || warp != 0) return;

  // ---- one warp of the first CTA merges the row. Statistics in one step:
  // M = max m2, z = sum 2^(m2 - M) z_c, t2 = sum 2^(m2 - M) (t2_c + z_c (m2 - M))
  Stats rs{-INFINITY, 0.f, 0.f};
  {
    float mc = -INFINITY, zc = 0.f, tc = 0.f;
    if (lane < C) {
      const float4 p = s_cst[lane];
      mc = p.x;
      zc = p.y;
      tc = p.z;
    }
    float M = mc;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(kFullMask, M, off));
    float zw = 0.f, tw = 0.f;
    if (zc > 0.f) {
      const float d = mc - M;
      const float w = ex2f(d);
      zw = w * zc;
      tw = w * fmaf(zc, d, tc);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      zw += __shfl_xor_sync(kFullMask, zw, off);
      tw += __shfl_xor_sync(kFullMask, tw, off);
    }
    rs = Stats{M, zw, tw};
  }
  // Keys: every slice's list is sorted, so the largest of their KP-th keys
  // is a key that at least KP candidates reach; the ones at or above it are
  // compacted (ballot) and ranked by counting.
  const int nall = C * KP;
  const uint64_t rthr = warp_max_u64(lane < C ? s_ckeys[lane * KP + KP - 1] : 0ull);
  int nc = 0;
  uint64_t kmax = 0ull;
  for (int j0 = 0; j0 < nall; j0 += 32) {
    const int j = j0 + lane;
    const uint64_t k = j < nall ? s_ckeys[j] : 0ull;
    const bool keep = j < nall && k >= rthr;
    const unsigned b = __ballot_sync(kFullMask, keep);
    if (keep) s_list[nc + __popc(b & ((1u << lane) - 1u))] = k;
    nc += __popc(b);
    kmax = k > kmax ? k : kmax;
  }
  kmax = warp_max_u64(kmax);
  __syncwarp();
  const float xmax = ordered_to_f32(static_cast<uint32_t>(kmax >> 32));
  if (lane == 0) {
    const float lz = logf(rs.z);
    lse[row] = xmax + lz;
    ent[row] = lz - (rs.t2 * kLn2) / rs.z;
  }
  for (int c = lane; c < nc; c += 32) {
    const uint64_t mine = s_list[c];
    int r = 0;
    for (int i = 0; i < nc; ++i) {
      const uint64_t o = s_list[i];
      r += (o > mine || (o == mine && i < c)) ? 1 : 0;
    }
    if (r < K) write_entry(row, K, r, mine, xmax, rs, ids, logp);
  }
}

constexpr size_t kClMaxDynSmem = static_cast<size_t>(kClMaxNv) * kClThreads * 16;

// Clusters of c CTAs of one instantiation that the current device can hold at
// once with the largest slice, c = 0..16 (entry 0 unused); queried once per
// device, after raising the kernel's dynamic shared-memory limit.
template <int KP, typename T>
const int* cluster_capacity() {
  static std::mutex mu;
  static int table[64][kClMaxCluster + 1];
  static bool done[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    if (cudaFuncSetAttribute(topk_cluster_kernel<KP, T>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kClMaxDynSmem)) != cudaSuccess ||
        cudaFuncSetAttribute(topk_cluster_kernel<KP, T>,
                             cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    for (int c = 0; c <= kClMaxCluster; ++c) {
      table[dev][c] = 0;
      if (c == 0) continue;
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(c, 1, 1);
      cfg.blockDim = dim3(kClThreads);
      cfg.dynamicSmemBytes = kClMaxDynSmem;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = c;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, topk_cluster_kernel<KP, T>, &cfg) == cudaSuccess)
        table[dev][c] = n;
    }
    cudaGetLastError();
    done[dev] = true;
  }
  return table[dev];
}

template <int KP, typename T>
int launch_cluster(const void* logits, int64_t row_stride, int R, int V, int K, int C, int per,
                   int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s) {
  const int* cap = cluster_capacity<KP, T>();
  if (!cap || cap[C] < R) return -1;   // not all rows at once: the general kernel runs
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = C;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(C, R, 1);
  cfg.blockDim = dim3(kClThreads);
  cfg.dynamicSmemBytes = static_cast<size_t>(per) * 16;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = C > 1 ? 2 : 1;
  if (cudaLaunchKernelEx(&cfg, topk_cluster_kernel<KP, T>, static_cast<const T*>(logits),
                         row_stride, V, K, per, ids, logp, lse, ent) != cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}

template <typename T>
int dispatch_kp(int kp, const void* logits, int64_t row_stride, int R, int V, int K, int C,
                int per, int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s) {
  switch (kp) {
    case 1: return launch_cluster<1, T>(logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s);
    case 2: return launch_cluster<2, T>(logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s);
    case 4: return launch_cluster<4, T>(logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s);
    case 8: return launch_cluster<8, T>(logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s);
    case 16: return launch_cluster<16, T>(logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s);
    default: return launch_cluster<32, T>(logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s);
  }
}

}  // namespace

int topk_cluster_try(const void* logits, int dtype, int64_t row_stride, int R, int V, int K,
                     int32_t* ids, float* logp, float* lse, float* ent, cudaStream_t s) {
  const size_t esz = dtype == TAPS_F32 ? 4 : 2;
  if (!aligned(logits, 16) || (row_stride * static_cast<int64_t>(esz)) % 16 != 0) return -1;
  if (R > kTargetSms) return -1;
  const int VE = static_cast<int>(16 / esz);
  const int nvec = V / VE;
  // one CTA per SM where the rows allow it, at least about one vector per
  // thread, at most kClMaxNv vectors per thread (then up to two CTAs per SM)
  const int by_work = std::max(1, (nvec + kClThreads - 1) / kClThreads);
  int C = std::min(kClMaxCluster, std::min(by_work, std::max(1, kTargetSms / R)));
  int per = (nvec + C - 1) / C;
  if (per > kClMaxNv * kClThreads) {
    C = (nvec + kClMaxNv * kClThreads - 1) / (kClMaxNv * kClThreads);
    if (C > kClMaxCluster || R * C > 2 * kTargetSms) return -1;
    per = (nvec + C - 1) / C;
  }
  const int kp = round_kp(K);
  return dtype == TAPS_F32
             ? dispatch_kp<float>(kp, logits, row_stride, R, V, K, C, per, ids, logp, lse, ent, s)
             : dispatch_kp<__nv_bfloat16>(kp, logits, row_stride, R, V, K, C, per, ids, logp, lse,
                                          ent, s);
}

}  // namespace taps
