// Stage 1 of a TAPS round (Sec. 4.1 stage 1, Sec. 4.2 scorer features):
// per-position full-vocabulary softmax statistics and top-K candidates.
//
// One pass over the logits. Each row (request b, position d) is split into
// `chunks` contiguous slices, one CTA each, so that a batch-1 round still
// spreads over every SM. A CTA reads its slice with 16-byte vector loads,
// keeps per-thread running statistics (max, sum of exponentials, sum of
// exponential-weighted offsets for the entropy) and, per warp, the running
// top-K of 64-bit keys (ordered logit << 32 | ~token id) in registers: each
// tile of two vectors per lane is merged in by K rounds of a warp maximum,
// and skipped when no key beats the current K-th. The CTA's warps merge by
// rank into one partial record. The last CTA of a row (an atomic ticket,
// reset after use) merges the partials by rank and writes the row's outputs.
// No CTA waits on another.
//
// taps_topk_marginals first offers the rows to two specialised kernels: one
// thread-block cluster per row when every row's cluster fits on the GPU at
// once (topk_cluster.cu, batch-1 rounds), one CTA per row from 304 rows
// (topk_stream.cu, batched rounds); this kernel serves the shapes in between
// (e.g. 128 rows) and unaligned logits.
#include <algorithm>
#include <atomic>
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
using sm100::mul_f32x2;

constexpr int kMaxChunks = 64;
constexpr int kRing = 4;                       // tiles per thread in its copy ring
constexpr int kFewKeys = 8;                    // at most this many tile keys: insert one by one
constexpr size_t kRingBytes = static_cast<size_t>(kRing) * 2 * kThreads * 16;

struct Plan {
  int rows, chunks, kp;
};

Plan make_plan(int B, int L, int V, int K) {
  Plan p;
  p.rows = B * L;
  p.kp = round_kp(K);
  // two CTAs per SM (registers and the 64 KB copy ring each allow two), in
  // one wave where the rows are few
  int want = (2 * kTargetSms + p.rows - 1) / p.rows;
  int maxc = std::max(1, V / 2048);
  p.chunks = std::max(1, std::min(want, std::min(maxc, kMaxChunks)));
  return p;
}

struct WsLayout {
  size_t stats, keys, tickets, total;
};

// The per-row tickets always sit in a fixed region at the start of the
// workspace, sized for the largest row count, so that a workspace reused by
// calls of different shapes never finds partial records where a later call
// keeps its counters. Every call leaves its tickets at zero.
constexpr size_t kTicketRegion = sizeof(unsigned) * 65536;

WsLayout ws_layout(const Plan& p) {
  WsLayout w;
  size_t o = 0;
  w.tickets = o;
  o = kTicketRegion;
  w.stats = o;
  o = align_up(o + sizeof(float4) * p.rows * p.chunks, 256);
  w.keys = o;
  o = align_up(o + sizeof(uint64_t) * p.rows * p.chunks * p.kp, 256);
  w.total = o;
  return w;
}


template <int KP, typename T>
__global__ void __launch_bounds__(kThreads)
topk_marginals_kernel(const T* __restrict__ logits, int64_t row_stride, int V, int K, int chunks,
                      int vec_ok, int32_t* __restrict__ ids, float* __restrict__ logp,
                      float* __restrict__ lse, float* __restrict__ ent, float4* ws_stats,
                      uint64_t* ws_keys, unsigned* tickets) {
  dep_enter();
  extern __shared__ __align__(16) unsigned char dyn_smem[];   // copy ring (vector path)
  constexpr int VE = 16 / sizeof(T);
  __shared__ uint64_t s_cand[kMaxChunks * 32];
  __shared__ uint64_t s_top[32];
  __shared__ uint64_t s_part[kWarps * 32];
  __shared__ Stats s_wstats[kWarps];
  __shared__ int s_last;
  // The largest K-th key any warp of this CTA holds: at least KP keys of the
  // row are >= it, so a key below it can be in no top-K (keys are unique, and
  // the key itself sits in the list of the warp that holds it)
  __shared__ unsigned long long s_thr;
  __shared__ int s_ncomp;          // entries in s_part compacted by select_top
  __shared__ unsigned long long s_rthr;
  if (threadIdx.x == 0) {
    s_thr = 0ull;
    s_ncomp = 0;
  }
  __syncthreads();

  const int row = blockIdx.y;
  const int chunk = blockIdx.x;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const T* x = logits + static_cast<int64_t>(row) * row_stride;

  Stats st{-INFINITY, 0.f, 0.f};
  // The warp's running top-KP keys: lane r < KP holds the r-th largest so far;
  // kth is the KP-th largest (0 while fewer than KP elements were seen).
  uint64_t run = 0, kth = 0;
  // Merge one tile (EPT keys per lane, 0 = none) into the running top-KP. A
  // tile with no key above kth changes nothing and is skipped. Otherwise tk =
  // the KP-th largest of the 32 lane maxima: at least KP keys of the tile are
  // >= tk, so its top-KP lies among them. Each lane keeps those (and above kth)
  // in four registers, and KP rounds of a 64-bit warp maximum run over them
  // and the running list; a lane with more than four (heavy ties) sends the
  // tile through the same rounds over all of its keys instead.
  constexpr int EPT = 2 * VE;
  // Insert one key (the same in every lane, above the K-th or the list not
  // full) into the lane-sorted running list: lane r < KP holds the r-th
  // largest; the key goes to position pos = (entries above it) and the entries
  // from pos on shift one lane down. A key that an earlier insertion has
  // already pushed below the K-th (pos == KP) changes nothing.
  auto insert_one = [&](uint64_t key) {
    const int pos = __popc(__ballot_sync(kFullMask, lane < KP && run > key));
    const uint64_t up = __shfl_up_sync(kFullMask, run, 1);
    if (pos < KP) {
      if (lane < KP && lane > pos) run = up;
      if (lane == pos) run = key;
    }
  };
  auto merge_tile = [&](uint64_t (&k)[EPT]) {
    uint64_t lm = 0;
#pragma unroll
    for (int i = 0; i < EPT; ++i) lm = k[i] > lm ? k[i] : lm;
    const uint64_t shared_thr = *reinterpret_cast<volatile unsigned long long*>(&s_thr);
    const uint64_t thr = shared_thr > kth ? shared_thr : kth;
    if (!__any_sync(kFullMask, lm > thr)) return;
    // Insert the candidates c4[0 .. cnt) of every lane into the lane-sorted
    // running list, one key after another. Lane r < KP holds the r-th
    // largest; a new key goes to position pos = (entries above it), and the
    // entries from pos on shift one lane down (the K-th falls off).
    auto insert_all = [&](const uint64_t (&c4)[4], int cnt) {
      unsigned todo = __ballot_sync(kFullMask, cnt > 0);
      while (todo) {
        const int src = __ffs(todo) - 1;
        todo &= todo - 1;
        const int n_src = __shfl_sync(kFullMask, cnt, src);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (j < n_src) {
            insert_one(__shfl_sync(kFullMask, c4[j], src));
          }
        }
      }
      kth = __shfl_sync(kFullMask, run, KP - 1);
      if (lane == 0 && kth > thr) atomicMax(&s_thr, static_cast<unsigned long long>(kth));
    };
    {
      // Few candidates (the usual case once the list has filled): insert the
      // keys above the threshold directly.
      uint64_t c4[4] = {0ull, 0ull, 0ull, 0ull};
      int cnt = 0;
#pragma unroll
      for (int i = 0; i < EPT; ++i) {
        if (k[i] > thr) {
          c4[3] = c4[2];
          c4[2] = c4[1];
          c4[1] = c4[0];
          c4[0] = k[i];
          ++cnt;
        }
      }
      const int total = __reduce_add_sync(kFullMask, static_cast<unsigned>(cnt));
      if (total <= kFewKeys && !__any_sync(kFullMask, cnt > 4)) {
        insert_all(c4, cnt);
        return;
      }
    }
    int rank = 0;   // lane maxima above this lane's (keys are unique, 0 = none)
#pragma unroll
    for (int l = 0; l < 32; ++l) rank += __shfl_sync(kFullMask, lm, l) > lm ? 1 : 0;
    const uint32_t at = __ballot_sync(kFullMask, lm != 0 && rank == KP - 1);
    const uint64_t tk = at ? __shfl_sync(kFullMask, lm, __ffs(at) - 1) : 0ull;
    uint64_t c[4] = {0ull, 0ull, 0ull, 0ull};
    int cnt = 0;
#pragma unroll
    for (int i = 0; i < EPT; ++i) {
      if (k[i] >= tk && k[i] > thr) {
        c[3] = c[2];
        c[2] = c[1];
        c[1] = c[0];
        c[0] = k[i];
        ++cnt;
      }
    }
    const bool wide = __any_sync(kFullMask, cnt > 4);
    // the tile's top-KP lies among these candidates: when they are few, insert
    // them rather than run KP rounds of a warp maximum
    if (!wide && __reduce_add_sync(kFullMask, static_cast<unsigned>(cnt)) <= 2 * kFewKeys) {
      insert_all(c, cnt);
      return;
    }
    uint64_t nrun = 0;
#pragma unroll 1
    for (int r = 0; r < KP; ++r) {
      uint64_t mine = run;
      if (wide) {
#pragma unroll
        for (int i = 0; i < EPT; ++i) mine = k[i] > mine ? k[i] : mine;
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) mine = c[i] > mine ? c[i] : mine;
      }
      const uint64_t best = warp_max_u64(mine);
      if (lane == r) nrun = best;
      if (best != 0 && mine == best) {
        if (run == best) run = 0;
        if (wide) {
#pragma unroll
          for (int i = 0; i < EPT; ++i) k[i] = k[i] == best ? 0ull : k[i];
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i) c[i] = c[i] == best ? 0ull : c[i];
        }
      }
    }
    run = nrun;
    kth = __shfl_sync(kFullMask, nrun, KP - 1);
    if (lane == 0 && kth > thr) atomicMax(&s_thr, static_cast<unsigned long long>(kth));
  };

  if (vec_ok) {
    // two 16-byte vectors per thread and tile
    const int nvec = V / VE;
    const int per = (nvec + chunks - 1) / chunks;
    const int v0 = chunk * per;
    const int v1 = min(nvec, v0 + per);
    const uint4* xv = reinterpret_cast<const uint4*>(x);
    // Each thread streams its own next kRing - 1 tiles into a private ring
    // in shared memory with 16-byte asynchronous copies (one commit group per
    // tile), so that many tiles are in flight without holding registers; it
    // reads back only what it copied itself, so no barrier is needed.
    // Ring layout [slot][vector u][thread]: a warp's reads are contiguous.
    constexpr int kStep = 2 * kThreads;
    // the statistics in packed pairs: two partial sums per thread (kept
    // relative to the thread's running max st.m2), folded into st at the end
    uint64_t zp = f32x2(0.f, 0.f), tp = f32x2(0.f, 0.f);
    const uint64_t l2e = f32x2(kLog2e, kLog2e);
    auto raise = [&](float m2_new) {
      if (m2_new > st.m2) {
        if (st.m2 > -INFINITY) {
          const float dm = st.m2 - m2_new;
          const uint64_t sc = f32x2(ex2f(dm), ex2f(dm));
          tp = mul_f32x2(sc, fma_f32x2(zp, f32x2(dm, dm), tp));
          zp = mul_f32x2(zp, sc);
        }
        st.m2 = m2_new;
      }
    };
    const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(dyn_smem));
    auto slot_addr = [&](int slot, int u) {
      return ring + static_cast<uint32_t>(((slot * 2 + u) * kThreads + tid) * 16);
    };
    auto issue = [&](int slot, int base) {
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int v = base + u * kThreads;
        if (v < v1)
          asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(slot_addr(slot, u)),
                       "l"(xv + v)
                       : "memory");
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    };
#pragma unroll
    for (int a = 0; a < kRing - 1; ++a) issue(a, v0 + tid + a * kStep);
    int slot = 0;
    for (int base = v0 + tid; base - tid < v1; base += kStep) {
      issue((slot + kRing - 1) % kRing, base + (kRing - 1) * kStep);
      asm volatile("cp.async.wait_group %0;" ::"n"(kRing - 1) : "memory");
      uint4 buf[2];
#pragma unroll
      for (int u = 0; u < 2; ++u)
        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(buf[u].x), "=r"(buf[u].y), "=r"(buf[u].z), "=r"(buf[u].w)
                     : "r"(slot_addr(slot, u)));
      slot = slot + 1 == kRing ? 0 : slot + 1;
      float vals[EPT];
      bool live[2];
      float tmax = -INFINITY;
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int v = base + u * kThreads;
        const T* e = reinterpret_cast<const T*>(&buf[u]);
        live[u] = v < v1;
        if (live[u]) {
          float vmax = -INFINITY;
#pragma unroll
          for (int i = 0; i < VE; ++i) {
            vals[u * VE + i] = to_f32<T>(e[i]);
            vmax = fmaxf(vmax, vals[u * VE + i]);
          }
          raise(vmax * kLog2e);
          // per pair: d = x log2(e) - m2 (one rounding), clamped at -127 so
          // that -inf and values far below the max give exactly 0 (ex2 with
          // flush-to-zero) and never 0 * inf
          const uint64_t nm2 = f32x2(-st.m2, -st.m2);
#pragma unroll
          for (int i = 0; i < VE; i += 2) {
            float d0, d1;
            f32x2_split(fma_f32x2(f32x2(vals[u * VE + i], vals[u * VE + i + 1]), l2e, nm2), d0,
                        d1);
            d0 = fmaxf(d0, -127.f);
            d1 = fmaxf(d1, -127.f);
            const uint64_t e = f32x2(ex2f(d0), ex2f(d1));
            zp = add_f32x2(zp, e);
            tp = fma_f32x2(e, f32x2(d0, d1), tp);
          }
          tmax = fmaxf(tmax, vmax);
        }
      }
      // keys are built only for a tile holding a value at or above the current
      // threshold's (a lower value has a lower key whatever its token id)
      const uint64_t shared_thr = *reinterpret_cast<volatile unsigned long long*>(&s_thr);
      const uint64_t thr = shared_thr > kth ? shared_thr : kth;
      float thr_v = thr ? ordered_to_f32(static_cast<uint32_t>(thr >> 32)) : -INFINITY;
      if (__any_sync(kFullMask, (live[0] || live[1]) && (thr == 0 || tmax >= thr_v))) {
        // Warm-up (this warp's list not yet full, no CTA threshold): the
        // KP-th largest lane maximum of the tile, counted with multiplicity,
        // is a value that at least KP of the tile's elements reach, so no
        // element below it can be in the tile's top-KP (nor in the top-KP of
        // the tile and the list). Found by 32-bit warp maxima over the lanes.
        int warm_left = 0;
        if (thr == 0) {
          uint32_t cur = (live[0] || live[1]) ? f32_to_ordered(tmax) : 0u;
          uint32_t t = 0u;
          int need = KP;
          while (need > 0) {
            const uint32_t m = __reduce_max_sync(kFullMask, cur);
            if (m == 0u) break;                    // fewer than KP live lanes
            need -= __popc(__ballot_sync(kFullMask, cur == m));
            t = m;
            if (cur == m) cur = 0u;
          }
          if (need <= 0) thr_v = ordered_to_f32(t);
          warm_left = need;
        }
        // elements whose value reaches the threshold's value: only they can
        // hold a key above it
        uint32_t flag = 0;
#pragma unroll
        for (int i = 0; i < EPT; ++i)
          flag |= (live[i / VE] && vals[i] >= thr_v) ? (1u << i) : 0u;
        const int nflag = __popc(flag);
        const unsigned few = thr != 0 ? kFewKeys : (warm_left <= 0 ? KP + kFewKeys : 0);
        if (__reduce_add_sync(kFullMask, static_cast<unsigned>(nflag)) <= few) {
          // few: visit only the element slots some lane flagged, build those
          // keys, and insert the ones above the threshold
#pragma unroll
          for (int i = 0; i < EPT; ++i) {
            if (__any_sync(kFullMask, (flag >> i) & 1u)) {
              const int v = base + (i / VE) * kThreads;
              const uint64_t key =
                  ((flag >> i) & 1u) ? make_key(vals[i], static_cast<uint32_t>(v * VE + i % VE))
                                     : 0ull;
              unsigned who = __ballot_sync(kFullMask, key > thr);
              while (who) {
                const int src = __ffs(who) - 1;
                who &= who - 1;
                insert_one(__shfl_sync(kFullMask, key, src));
              }
            }
          }
          kth = __shfl_sync(kFullMask, run, KP - 1);
          if (lane == 0 && kth > thr) atomicMax(&s_thr, static_cast<unsigned long long>(kth));
        } else {
          uint64_t k[EPT];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int v = base + u * kThreads;
#pragma unroll
            for (int i = 0; i < VE; ++i)
              k[u * VE + i] =
                  live[u] ? make_key(vals[u * VE + i], static_cast<uint32_t>(v * VE + i)) : 0ull;
          }
          merge_tile(k);
        }
      }
    }
    {
      float z0, z1, t0, t1;
      f32x2_split(zp, z0, z1);
      f32x2_split(tp, t0, t1);
      st.z += z0 + z1;
      st.t2 += t0 + t1;
    }
    // tail elements past the last full vector go to the last chunk
    if (chunk == chunks - 1 && nvec * VE < V) {
      uint64_t k[EPT];
#pragma unroll
      for (int i = 0; i < EPT; ++i) k[i] = 0;
      const int i = nvec * VE + tid;   // fewer than VE tail elements
      if (i < V) {
        const float xv1 = to_f32<T>(x[i]);
        stats_raise(st, xv1 * kLog2e);
        stats_add(st, xv1 * kLog2e);
        k[0] = make_key(xv1, static_cast<uint32_t>(i));
      }
      merge_tile(k);
    }
  } else {
    const int per = (V + chunks - 1) / chunks;
    const int e0 = chunk * per;
    const int e1 = min(V, e0 + per);
    for (int base = e0; base < e1; base += EPT * kThreads) {
      uint64_t k[EPT];
#pragma unroll
      for (int u = 0; u < EPT; ++u) {
        const int i = base + u * kThreads + tid;
        k[u] = 0;
        if (i < e1) {
          const float xv1 = to_f32<T>(x[i]);
          stats_raise(st, xv1 * kLog2e);
          stats_add(st, xv1 * kLog2e);
          k[u] = make_key(xv1, static_cast<uint32_t>(i));
        }
      }
      merge_tile(k);
    }
  }
  if (lane < KP) s_cand[warp * KP + lane] = run;
  st = warp_stats(st);
  if (lane == 0) s_wstats[warp] = st;
  __syncthreads();
  // the CTA's top-KP: only the warp candidates at or above the CTA threshold
  // (the largest K-th key any warp holds) can be in it
  select_top<KP>(s_cand, kWarps * KP, s_thr, s_part, kWarps * 32, &s_ncomp, s_top, s_part);

  if (warp == 0) {
    Stats cs = s_wstats[0];
    for (int w = 1; w < kWarps; ++w) cs = stats_merge(cs, s_wstats[w]);
    if (chunks == 1) {
      __syncwarp();
      write_row<KP>(row, K, s_top, cs, lane, ids, logp, lse, ent);
    } else {
      const int64_t rec = static_cast<int64_t>(row) * chunks + chunk;
      if (lane == 0) ws_stats[rec] = make_float4(cs.m2, cs.z, cs.t2, 0.f);
      __syncwarp();
      for (int r = lane; r < KP; r += 32) ws_keys[rec * KP + r] = s_top[r];
      __threadfence();
      __syncwarp();
      if (lane == 0) s_last = (atomicAdd(&tickets[row], 1u) == static_cast<unsigned>(chunks - 1));
      __syncwarp();
    }
  }
  if (chunks == 1) return;
  __syncthreads();
  if (!s_last) return;

  // ---- last CTA of this row: merge every chunk's partial record. The
  // partial statistics are loaded with the keys, in one round trip.
  __threadfence();
  const int64_t rec0 = static_cast<int64_t>(row) * chunks;
  const int n = chunks * KP;
  for (int i = tid; i < n; i += kThreads) s_cand[i] = __ldcg(ws_keys + rec0 * KP + i);
  Stats cs{-INFINITY, 0.f, 0.f};
  if (warp == 0) {
    // every chunk's list is sorted: the largest of their K-th keys is a key
    // that at least KP candidates reach
    uint64_t kmax = 0ull;
    for (int c = lane; c < chunks; c += 32) {
      float4 p = __ldcg(ws_stats + rec0 + c);
      cs = stats_merge(cs, Stats{p.x, p.y, p.z});
      const uint64_t kk = __ldcg(ws_keys + (rec0 + c) * KP + KP - 1);
      kmax = kk > kmax ? kk : kmax;
    }
    kmax = warp_max_u64(kmax);
    if (lane == 0) s_rthr = kmax;
  }
  __syncthreads();
  select_top<KP>(s_cand, n, s_rthr, s_part, kWarps * 32, &s_ncomp, s_top, s_part);
  if (warp == 0) {
    cs = warp_stats(cs);
    write_row<KP>(row, K, s_top, cs, lane, ids, logp, lse, ent);
    if (lane == 0) tickets[row] = 0u;
  }
}

template <int KP, typename T>
void launch(const void* logits, int64_t row_stride, const Plan& p, int V, int K, int vec_ok,
            int32_t* ids, float* logp, float* lse, float* ent, char* ws, const WsLayout& w,
            cudaStream_t s) {
  dim3 grid(p.chunks, p.rows);
  float4* st = p.chunks > 1 ? reinterpret_cast<float4*>(ws + w.stats) : nullptr;
  uint64_t* keys = p.chunks > 1 ? reinterpret_cast<uint64_t*>(ws + w.keys) : nullptr;
  unsigned* tk = p.chunks > 1 ? reinterpret_cast<unsigned*>(ws + w.tickets) : nullptr;
  // the copy ring exceeds the default 48 KB of dynamic shared memory: raise
  // the limit once per device. The flags are atomics because the entry points
  // may be called from several host threads; two threads setting the same
  // attribute at once is harmless.
  static std::atomic<bool> ring_attr[64];
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64 &&
      !ring_attr[dev].load(std::memory_order_acquire)) {
    if (cudaFuncSetAttribute(topk_marginals_kernel<KP, T>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kRingBytes)) == cudaSuccess)
      ring_attr[dev].store(true, std::memory_order_release);
  }
  launch_dep(topk_marginals_kernel<KP, T>, grid, dim3(kThreads), vec_ok ? kRingBytes : 0, s,
             static_cast<const T*>(logits), row_stride, V, K, p.chunks, vec_ok, ids, logp, lse,
             ent, st, keys, tk);
}

template <typename T>
void dispatch_kp(int kp, const void* logits, int64_t row_stride, const Plan& p, int V, int K,
                 int vec_ok, int32_t* ids, float* logp, float* lse, float* ent, char* ws,
                 const WsLayout& w, cudaStream_t s) {
  switch (kp) {
    case 1: launch<1, T>(logits, row_stride, p, V, K, vec_ok, ids, logp, lse, ent, ws, w, s); break;
    case 2: launch<2, T>(logits, row_stride, p, V, K, vec_ok, ids, logp, lse, ent, ws, w, s); break;
    case 4: launch<4, T>(logits, row_stride, p, V, K, vec_ok, ids, logp, lse, ent, ws, w, s); break;
    case 8: launch<8, T>(logits, row_stride, p, V, K, vec_ok, ids, logp, lse, ent, ws, w, s); break;
    case 16: launch<16, T>(logits, row_stride, p, V, K, vec_ok, ids, logp, lse, ent, ws, w, s); break;
    default: launch<32, T>(logits, row_stride, p, V, K, vec_ok, ids, logp, lse, ent, ws, w, s); break;
  }
}

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" size_t taps_topk_marginals_workspace_bytes(int B, int L, int V, int K) {
  if (B <= 0 || L <= 0 || V <= 0 || K <= 0 || K > TAPS_MAX_K) return 0;
  return ws_layout(make_plan(B, L, V, K)).total;
}

extern "C" int taps_topk_marginals(const void* logits, int dtype, int64_t row_stride, int B,
                                   int L, int V, int K, int32_t* topk_ids, float* topk_logp,
                                   float* lse, float* entropy, void* ws, size_t ws_bytes,
                                   void* stream) {
  if (!logits || !topk_ids || !topk_logp || !lse || !entropy) return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || V <= 0 || K <= 0 || row_stride < V) return TAPS_ERR_INVALID_ARG;
  if (dtype != TAPS_F32 && dtype != TAPS_BF16) return TAPS_ERR_INVALID_ARG;
  if (K > TAPS_MAX_K || K > V || V > TAPS_MAX_V) return TAPS_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(B) * L > 65535) return TAPS_ERR_UNSUPPORTED;
  Plan p = make_plan(B, L, V, K);
  WsLayout w = ws_layout(p);
  if (p.chunks > 1 && (!ws || ws_bytes < w.total || !aligned(ws, 256))) return TAPS_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // a few rows: one cluster per row, merged on chip (no workspace traffic)
  const int rc = topk_cluster_try(logits, dtype, row_stride, B * L, V, K, topk_ids, topk_logp, lse,
                                  entropy, s);
  if (rc != -1) return rc;
  // many rows: one CTA streams each row
  const int rs = topk_stream_try(logits, dtype, row_stride, B * L, V, K, topk_ids, topk_logp, lse,
                                 entropy, s);
  if (rs != -1) return rs;
  const size_t esz = dtype == TAPS_F32 ? 4 : 2;
  const int vec_ok = aligned(logits, 16) && (row_stride * esz) % 16 == 0;
  char* wsc = static_cast<char*>(ws);
  if (dtype == TAPS_F32)
    dispatch_kp<float>(p.kp, logits, row_stride, p, V, K, vec_ok, topk_ids, topk_logp, lse,
                       entropy, wsc, w, s);
  else
    dispatch_kp<__nv_bfloat16>(p.kp, logits, row_stride, p, V, K, vec_ok, topk_ids, topk_logp,
                               lse, entropy, wsc, w, s);
  return launch_status();
}

// ---------------------------------------------------------------------------
// Allocation-free variant of taps_topk_marginals.
//
// Some callers cannot call cudaMalloc: a serving engine that reserved all of
// device memory for its KV cache at start-up, a plugin running inside a host
// framework that owns every device allocation, or a decode loop that cannot
// afford the device-wide synchronisation an allocation may cause. This entry
// point takes inputs and outputs from the caller and keeps its partial records
// in a fixed array in device memory that belongs to this library.
//
// The array below is a file-scope __device__ symbol: every GPU that loads the
// library holds it until the process exits. In host code its name is only a
// host-side stand-in, never a device address, so the host looks the device
// address up with cudaGetSymbolAddress, once per device, with that device
// current, and passes that address to the kernel.
// ---------------------------------------------------------------------------
namespace taps {
namespace {

constexpr size_t kNoAllocTicketBytes = sizeof(unsigned) * TAPS_NOALLOC_MAX_ROWS;

static __device__ __align__(256) unsigned char g_topk_scratch[TAPS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_topk_scratch on the current device (set up on first use).
int scratch_for_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return TAPS_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_topk_scratch) != cudaSuccess || !p) return TAPS_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return TAPS_OK;
}

}  // namespace
}  // namespace taps

extern "C" int taps_topk_marginals_noalloc(const void* logits, int dtype, int64_t row_stride,
                                           int B, int L, int V, int K, int32_t* topk_ids,
                                           float* topk_logp, float* lse, float* entropy,
                                           void* stream) {
  if (!logits || !topk_ids || !topk_logp || !lse || !entropy) return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || V <= 0 || K <= 0 || row_stride < V) return TAPS_ERR_INVALID_ARG;
  if (dtype != TAPS_F32 && dtype != TAPS_BF16) return TAPS_ERR_INVALID_ARG;
  if (K > TAPS_MAX_K || K > V || V > TAPS_MAX_V) return TAPS_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(B) * L > TAPS_NOALLOC_MAX_ROWS) return TAPS_ERR_UNSUPPORTED;
  Plan p = make_plan(B, L, V, K);
  // layout inside the fixed array: tickets, then the partial statistics, then keys
  WsLayout w;
  w.tickets = 0;
  w.stats = kNoAllocTicketBytes;
  w.keys = align_up(w.stats + sizeof(float4) * p.rows * p.chunks, 256);
  w.total = align_up(w.keys + sizeof(uint64_t) * p.rows * p.chunks * p.kp, 256);
  if (w.total > TAPS_NOALLOC_SCRATCH_BYTES) return TAPS_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  int st = scratch_for_current_device(&scratch);
  if (st != TAPS_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the tickets must start at zero; clear the ones this call uses
  if (p.chunks > 1 && cudaMemsetAsync(scratch, 0, sizeof(unsigned) * p.rows, s) != cudaSuccess)
    return TAPS_ERR_CUDA;
  const size_t esz = dtype == TAPS_F32 ? 4 : 2;
  const int vec_ok = aligned(logits, 16) && (row_stride * esz) % 16 == 0;
  char* wsc = static_cast<char*>(scratch);
  if (dtype == TAPS_F32)
    dispatch_kp<float>(p.kp, logits, row_stride, p, V, K, vec_ok, topk_ids, topk_logp, lse,
                       entropy, wsc, w, s);
  else
    dispatch_kp<__nv_bfloat16>(p.kp, logits, row_stride, p, V, K, vec_ok, topk_ids, topk_logp,
                               lse, entropy, wsc, w, s);
  return launch_status();
}
