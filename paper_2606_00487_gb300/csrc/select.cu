// Stage 3 of a TAPS round (Sec. 4.2-4.3, Eq. 2, Eq. 3, Algorithm 1):
// reach, utility and the greedy budgeted prefix-closed selection.
//
// Algorithm 1 adds, one node at a time, the unselected node of largest
// utility. Utility never increases from a parent to a child (q_cond <= 1,
// den(d) non-decreasing, monotone rounding) and ties favour the lower depth,
// so under the total order of the selection key below every child ranks
// strictly after its parent. The greedy loop therefore takes nodes in
// descending key order, and its result is the set of the n_max largest keys
// of the whole candidate tree (those with utility > tau), listed in key
// order; a child's parent index is its parent's position in that list.
//
// One CTA per request computes that set level-synchronously instead of one
// node per step. It keeps T, the best n_max nodes found so far in key order,
// and repeats a pass:
//   1. list the members of T whose children have not been generated yet
//      (in any order; at most 512 / K of them per pass, the rest wait);
//   2. generate their children, one thread per child, and keep the ones
//      that would enter T (utility > tau and, once T is full, a key above
//      T's last key);
//   3. rank T and the kept children together by counting, write the best
//      n_max in order into the other buffer and renumber parent indices.
// It stops when a pass generates every remaining child and keeps none. A
// node that left T never returns (T's last key only rises once T is full),
// and a child that was not kept ranks below every member of T; at the stop
// all members have been expanded, so T is the n_max largest keys. The number
// of passes is about the depth of the selected tree plus one.
//
// Selection key (larger = taken first): utility bits (non-negative floats
// order like their bit patterns) | (31 - depth) | (2^18 - 1 - token) |
// (511 - parent index), i.e. utility desc, depth asc, token asc, parent asc.
// A key is compared only with keys whose parent indices refer to the same T,
// and the relative order of two members of T never changes, so comparing
// indices into the current T is the same as comparing final indices. Equal
// keys (only possible with repeated token ids in a top-K row) are ordered by
// their index in the ranked array, which keeps ranks a permutation.
//
// All reach/utility arithmetic is IEEE f32 round-to-nearest (explicit _rn
// intrinsics, no contraction), root to leaf. q_cond is staged clamped to
// [0, 1] (NaN to 0), which changes nothing for valid input and keeps every
// child after its parent for any input.
#include <algorithm>

#include "common.cuh"

namespace taps {
namespace {

__device__ __forceinline__ uint64_t node_key(float util, int depth, int token, int parent) {
  return (static_cast<uint64_t>(__float_as_uint(util)) << 32) |
         (static_cast<uint64_t>(31 - depth) << 27) |
         (static_cast<uint64_t>((1 << 18) - 1 - token) << 9) |
         static_cast<uint64_t>(511 - parent);
}

constexpr int kThreads = 512;
// children generated per pass (one per thread)
constexpr int kCap = kThreads;
// every pass expands at least one member of T, and a node enters T at most
// once; this bound is never reached and only keeps the loop finite
constexpr int kMaxPasses = 1 << 14;

// One buffer of ranked nodes: T in [0, nT), kept children appended after it.
struct NodeBuf {
  uint64_t* key;
  float* reach;
  float* util;
  int16_t* ppos;          // parent index into the same buffer (-1: root)
  unsigned char* depth;
  unsigned char* slot;    // top-K slot of the node's position
  unsigned char* done;    // children already generated
};

struct SelSmem {
  float* q;          // [L][K][K], clamped to [0, 1]
  int* ids;          // [L][K]
  float* den;        // [32]
  char* buf0;        // two node buffers of n_max + kCap entries
  char* buf1;
  int16_t* newpos;   // [n_max] new index of each member of T (-1: dropped)
  int16_t* list;     // [n_max] members to expand this pass, with their
  float* lreach;     //   reach,
  unsigned char* ldepth;  // depth and q_cond row
  unsigned char* lrow;
  int* cnt;          // [4] listed-member and kept-child counters, two each,
                     //     alternating by pass
};

__host__ __device__ inline size_t sel_round16(size_t x) { return (x + 15) / 16 * 16; }

__host__ __device__ inline size_t node_buf_bytes(size_t C) {
  return sel_round16(8 * C) + 2 * sel_round16(4 * C) + sel_round16(2 * C) + 3 * sel_round16(C);
}

__device__ __forceinline__ NodeBuf node_buf(char* p, size_t C) {
  NodeBuf nb;
  nb.key = reinterpret_cast<uint64_t*>(p);       p += sel_round16(8 * C);
  nb.reach = reinterpret_cast<float*>(p);        p += sel_round16(4 * C);
  nb.util = reinterpret_cast<float*>(p);         p += sel_round16(4 * C);
  nb.ppos = reinterpret_cast<int16_t*>(p);       p += sel_round16(2 * C);
  nb.depth = reinterpret_cast<unsigned char*>(p); p += sel_round16(C);
  nb.slot = reinterpret_cast<unsigned char*>(p); p += sel_round16(C);
  nb.done = reinterpret_cast<unsigned char*>(p);
  return nb;
}

__host__ __device__ inline size_t sel_smem_bytes(int L, int K, int n_max) {
  const size_t C = static_cast<size_t>(n_max) + kCap;
  size_t o = 0;
  o += sel_round16(sizeof(float) * L * K * K);
  o += sel_round16(sizeof(int) * L * K);
  o += sel_round16(sizeof(float) * 32);
  o += 2 * node_buf_bytes(C);
  o += 2 * sel_round16(2 * static_cast<size_t>(n_max)) + sel_round16(4 * static_cast<size_t>(n_max));
  o += 2 * sel_round16(static_cast<size_t>(n_max)) + sel_round16(sizeof(int) * 4);
  return o;
}

__device__ SelSmem carve(char* base, int L, int K, int n_max) {
  const size_t C = static_cast<size_t>(n_max) + kCap;
  char* p = base;
  auto take = [&](size_t bytes) {
    char* r = p;
    p += sel_round16(bytes);
    return r;
  };
  SelSmem s;
  s.q = reinterpret_cast<float*>(take(sizeof(float) * L * K * K));
  s.ids = reinterpret_cast<int*>(take(sizeof(int) * L * K));
  s.den = reinterpret_cast<float*>(take(sizeof(float) * 32));
  s.buf0 = take(node_buf_bytes(C));
  s.buf1 = take(node_buf_bytes(C));
  s.newpos = reinterpret_cast<int16_t*>(take(2 * static_cast<size_t>(n_max)));
  s.list = reinterpret_cast<int16_t*>(take(2 * static_cast<size_t>(n_max)));
  s.lreach = reinterpret_cast<float*>(take(4 * static_cast<size_t>(n_max)));
  s.ldepth = reinterpret_cast<unsigned char*>(take(static_cast<size_t>(n_max)));
  s.lrow = reinterpret_cast<unsigned char*>(take(static_cast<size_t>(n_max)));
  s.cnt = reinterpret_cast<int*>(take(sizeof(int) * 4));
  return s;
}

// Number of keys above k among key[c0], key[c0 + g], ... below index hi;
// eight independent loads in flight.
__device__ __forceinline__ int count_above(const uint64_t* key, int c0, int hi, int g,
                                           uint64_t k) {
  int cnt = 0;
  int c = c0;
  for (; c + 7 * g < hi; c += 8 * g) {
    uint64_t v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = key[c + i * g];
#pragma unroll
    for (int i = 0; i < 8; ++i) cnt += v[i] > k ? 1 : 0;
  }
  for (; c < hi; c += g) cnt += key[c] > k ? 1 : 0;
  return cnt;
}

__global__ void __launch_bounds__(kThreads, 1)
select_kernel(const float* __restrict__ q_cond, const int* __restrict__ ids,
              const int32_t* __restrict__ root_tok, const int32_t* __restrict__ ctx_len, int L,
              int K, float lambda1, float lambda2, float tau, int n_max,
              int32_t* __restrict__ n_nodes_out, int32_t* __restrict__ parent_out,
              int32_t* __restrict__ depth_out, int32_t* __restrict__ token_out,
              int32_t* __restrict__ slot_out, int32_t* __restrict__ pos_out,
              float* __restrict__ reach_out, float* __restrict__ util_out) {
  dep_enter();
  extern __shared__ __align__(16) char smem_raw[];
  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31;
  SelSmem s = carve(smem_raw, L, K, n_max);
  const size_t C = static_cast<size_t>(n_max) + kCap;

  const float* qb = q_cond + static_cast<int64_t>(b) * L * K * K;
  for (int i = tid; i < L * K * K; i += kThreads) {
    const float v = qb[i];
    s.q[i] = v > 0.f ? fminf(v, 1.0f) : 0.f;
  }
  const int32_t* ib = ids + static_cast<int64_t>(b) * L * K;
  for (int i = tid; i < L * K; i += kThreads) s.ids[i] = ib[i];
  if (tid <= L) s.den[tid] = __fadd_rn(lambda1, __fmul_rn(lambda2, static_cast<float>(tid)));
  if (tid == 0) {
    const float den0 = __fadd_rn(lambda1, __fmul_rn(lambda2, 0.0f));
    NodeBuf T = node_buf(s.buf0, C);
    T.key[0] = ~0ull;   // the root ranks first
    T.reach[0] = 1.0f;
    T.util[0] = __fdiv_rn(1.0f, den0);
    T.ppos[0] = -1;
    T.depth[0] = 0;
    T.slot[0] = 0;
    T.done[0] = 0;
    s.cnt[0] = 0;
    s.cnt[2] = 0;
  }
  __syncthreads();

  const int max_expand = kCap / K;
  // this thread's child in step 2: child j_own of listed member li_own
  const int li_own = tid / K;
  const int j_own = tid - li_own * K;
  int cur = 0, nT = 1;
  for (int pass = 0; pass < kMaxPasses; ++pass) {
    const NodeBuf T = node_buf(cur ? s.buf1 : s.buf0, C);
    const NodeBuf Nx = node_buf(cur ? s.buf0 : s.buf1, C);
    int* listed = s.cnt + (pass & 1);
    int* kept = s.cnt + 2 + (pass & 1);

    // 1. list members still to expand (any order); the first max_expand
    //    listed are expanded in this pass, the rest in a later one
    const bool open = tid < nT && !T.done[tid];
    const unsigned bal = __ballot_sync(kFullMask, open);
    int lbase = 0;
    if (lane == 0 && bal) lbase = atomicAdd(listed, __popc(bal));
    lbase = __shfl_sync(kFullMask, lbase, 0);
    if (open) {
      const int idx = lbase + __popc(bal & ((1u << lane) - 1u));
      if (idx < max_expand) {
        const int dp = T.depth[tid];
        s.list[idx] = static_cast<int16_t>(tid);
        s.lreach[idx] = T.reach[tid];
        s.ldepth[idx] = static_cast<unsigned char>(dp);
        s.lrow[idx] = dp == 0 ? 0 : T.slot[tid];
        T.done[tid] = 1;
      }
    }
    __syncthreads();
    // the other pair of counters was last read before this barrier
    if (tid == 0) {
      s.cnt[(pass + 1) & 1] = 0;
      s.cnt[2 + ((pass + 1) & 1)] = 0;
    }
    const int total = *listed;
    const int X = min(total, max_expand);

    // 2. their children; keep those that would enter T
    const uint64_t thr = nT == n_max ? T.key[nT - 1] : 0ull;
    bool keep = false;
    uint64_t key = 0;
    float r = 0.f, u = 0.f;
    int t = 0, dc = 0;
    if (li_own < X) {
      t = s.list[li_own];
      const int dp = s.ldepth[li_own];
      const int row = s.lrow[li_own];
      dc = dp + 1;
      r = __fmul_rn(s.lreach[li_own], s.q[(dp * K + row) * K + j_own]);
      u = __fdiv_rn(r, s.den[dc]);
      key = node_key(u, dc, s.ids[dp * K + j_own], t);
      keep = u > tau && key > thr;
    }
    const unsigned kb = __ballot_sync(kFullMask, keep);
    int base = 0;
    if (lane == 0 && kb) base = atomicAdd(kept, __popc(kb));
    base = __shfl_sync(kFullMask, base, 0);
    if (keep) {
      const int e = nT + base + __popc(kb & ((1u << lane) - 1u));
      T.key[e] = key;
      T.reach[e] = r;
      T.util[e] = u;
      T.ppos[e] = static_cast<int16_t>(t);
      T.depth[e] = static_cast<unsigned char>(dc);
      T.slot[e] = static_cast<unsigned char>(j_own);
      T.done[e] = dc >= L;
    }
    __syncthreads();
    const int m = *kept;
    if (m == 0) {
      if (total == X) break;
      continue;
    }

    // 3. rank T and the kept children: g threads per entry
    const int E = nT + m;
    int lg = 5;
    while (lg > 0 && (E << lg) > kThreads) --lg;
    const int g = 1 << lg;
    const int grp = tid >> lg, sub = tid & (g - 1);
    for (int e0 = 0; e0 < E; e0 += kThreads >> lg) {
      const int e = e0 + grp;
      int cnt = 0;
      uint64_t ke = 0;
      if (e < E) {
        ke = T.key[e];
        // entries ahead of e on this lane's stride, counted over up to three
        // ranges with their thresholds (one loop, so that one copy of the
        // counting code serves every case)
        const uint64_t ke1 = ke - 1;   // kept keys are >= 2^32: "> ke1" is ">= ke"
        const int c0 = nT + sub;
        int lo0 = 0, hi0 = 0, split = c0;
        if (e < nT) {
          // a member: members ahead of it are e; children ahead have a larger key
          if (sub == 0) cnt = e;
        } else {
          // a kept child: members with key >= ke (a prefix of T, whose keys
          // descend), then children with key >= ke before it and > ke after it
          if (nT <= 32 * g) {
            lo0 = sub;
            hi0 = nT;
          } else {
            int lo = 0, hi = sub < nT ? ((nT - 1 - sub) >> lg) + 1 : 0;
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if (T.key[sub + mid * g] > ke1) lo = mid + 1;
              else hi = mid;
            }
            cnt = lo;
          }
          if (e > c0) split = c0 + (((e - c0 + g - 1) >> lg) << lg);
        }
#pragma unroll 1
        for (int rg = 0; rg < 3; ++rg) {
          const int lo = rg == 0 ? lo0 : rg == 1 ? c0 : split;
          const int hi = rg == 0 ? hi0 : rg == 1 ? split : E;
          cnt += count_above(T.key, lo, hi, g, rg == 2 ? ke : ke1);
        }
      }
      for (int o = 1; o < g; o <<= 1) cnt += __shfl_xor_sync(kFullMask, cnt, o);
      if (sub == 0 && e < E) {
        if (e < nT) s.newpos[e] = static_cast<int16_t>(cnt < n_max ? cnt : -1);
        if (cnt < n_max) {
          Nx.key[cnt] = ke;
          Nx.reach[cnt] = T.reach[e];
          Nx.util[cnt] = T.util[e];
          Nx.ppos[cnt] = T.ppos[e];
          Nx.depth[cnt] = T.depth[e];
          Nx.slot[cnt] = T.slot[e];
          Nx.done[cnt] = T.done[e];
        }
      }
    }
    __syncthreads();
    // renumber parents (a parent always ranks before its child, so it stayed)
    nT = min(E, n_max);
    if (tid < nT) {
      const int po = Nx.ppos[tid];
      if (po >= 0) {
        const int pn = s.newpos[po];
        Nx.ppos[tid] = static_cast<int16_t>(pn);
        Nx.key[tid] = (Nx.key[tid] & ~511ull) | static_cast<uint64_t>(511 - pn);
      }
    }
    cur ^= 1;
    // the next pass reads these entries only after its first barrier
  }
  __syncthreads();

  // write the selected nodes in key order, pad the rest
  const NodeBuf T = node_buf(cur ? s.buf1 : s.buf0, C);
  const int64_t o = static_cast<int64_t>(b) * n_max;
  const int c = ctx_len[b];
  for (int i = tid; i < n_max; i += kThreads) {
    if (i < nT) {
      const int d = T.depth[i];
      parent_out[o + i] = T.ppos[i];
      depth_out[o + i] = d;
      slot_out[o + i] = i == 0 ? -1 : T.slot[i];
      token_out[o + i] = i == 0 ? root_tok[b] : s.ids[(d - 1) * K + T.slot[i]];
      pos_out[o + i] = c + d;
      reach_out[o + i] = T.reach[i];
      util_out[o + i] = T.util[i];
    } else {
      parent_out[o + i] = -1;
      depth_out[o + i] = -1;
      slot_out[o + i] = -1;
      token_out[o + i] = -1;
      pos_out[o + i] = -1;
      reach_out[o + i] = 0.f;
      util_out[o + i] = 0.f;
    }
  }
  if (tid == 0) n_nodes_out[b] = nT;
}

int launch_select(const float* q_cond, const int32_t* topk_ids, const int32_t* root_tok,
                  const int32_t* ctx_len, int B, int L, int K, float l1, float l2, float tau,
                  int n_max, int32_t* n_nodes, int32_t* parent, int32_t* depth, int32_t* token,
                  int32_t* slot, int32_t* pos_id, float* reach, float* utility,
                  cudaStream_t stream) {
  const size_t smem = sel_smem_bytes(L, K, n_max);
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return TAPS_ERR_CUDA;
  if (launch_dep(select_kernel, dim3(B), dim3(kThreads), smem, stream, q_cond, topk_ids,
                 root_tok, ctx_len, L, K, l1, l2, tau, n_max, n_nodes, parent, depth, token,
                 slot, pos_id, reach, utility) != cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}

}  // namespace
}  // namespace taps

using namespace taps;

extern "C" int taps_select_subtree(const float* q_cond, const int32_t* topk_ids,
                                   const int32_t* root_tok, const int32_t* ctx_len, int B, int L,
                                   int K, const taps_select_params* params, int32_t* n_nodes,
                                   int32_t* parent, int32_t* depth, int32_t* token, int32_t* slot,
                                   int32_t* pos_id, float* reach, float* utility, void* stream) {
  if (!q_cond || !topk_ids || !root_tok || !ctx_len || !params || !n_nodes || !parent ||
      !depth || !token || !slot || !pos_id || !reach || !utility)
    return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || K <= 0) return TAPS_ERR_INVALID_ARG;
  const float l1 = params->lambda1, l2 = params->lambda2, tau = params->tau;
  const int n_max = params->n_max;
  if (!(l1 > 0.f) || !(l2 >= 0.f) || !(tau >= 0.f) || n_max < 1) return TAPS_ERR_INVALID_ARG;
  if (K > TAPS_MAX_K || L > TAPS_MAX_L || n_max > TAPS_MAX_NODES || B > 65535)
    return TAPS_ERR_UNSUPPORTED;
  return launch_select(q_cond, topk_ids, root_tok, ctx_len, B, L, K, l1, l2, tau, n_max,
                       n_nodes, parent, depth, token, slot, pos_id, reach, utility,
                       static_cast<cudaStream_t>(stream));
}
