// Stage 3 of a TAPS round (Sec. 4.2-4.3, Eq. 2, Eq. 3, Algorithm 1):
// reach, utility and the greedy budgeted prefix-closed selection; and the
// selection fused with the tree mask (stage 4) in one launch per request.
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
// and repeats a pass of two steps, each ending in a CTA barrier:
//   A. generate the children of the members listed for expansion (one thread
//      per child; at most 512 / K members per pass) and append the ones that
//      would enter T (utility > tau and, once T is full, a key above a lower
//      bound of T's last key);
//   B. rank T and the appended children together by counting, write the
//      best n_max in order into the other buffer, and list (in any order)
//      the entries whose children have not been generated, for the next
//      pass; then each thread renumbers the parent index of its own entry.
// It stops when a pass expanded every listed member and appended nothing. A
// node that left T never returns (T's last key only rises once T is full),
// and a child that was not appended ranks below every member of T; at the
// stop all members have been expanded, so T is the n_max largest keys. The
// number of passes is about the depth of the selected tree plus one.
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
#include <atomic>

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
// every pass expands at least one listed member or appends a node, and a
// node enters T at most once; this bound is never reached and only keeps
// the loop finite
constexpr int kMaxPasses = 1 << 14;

// One buffer of ranked nodes: T in [0, nT), appended children after it.
struct NodeBuf {
  uint64_t* key;
  float* reach;
  float* util;
  int16_t* ppos;          // parent index into the same buffer (-1: root)
  unsigned char* depth;
  unsigned char* slot;    // top-K slot of the node's position
  unsigned char* done;    // children generated, or listed for the next pass
};

struct SelSmem {
  float* q;          // [L][K][K], clamped to [0, 1]
  int* ids;          // [L][K]
  float* den;        // [32]
  char* buf0;        // two node buffers of n_max + kCap entries
  char* buf1;
  int16_t* newpos;   // [n_max] new index of each member of T (-1: dropped)
  int16_t* list;     // [kCap] entries listed for expansion in the next pass
  int* cnt;          // [4] appended-child and listed-entry counters, two
                     //     each, alternating by pass
  unsigned long long* thr;   // lower bound of T's last key (0: T not full)
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
  o += sel_round16(2 * static_cast<size_t>(n_max)) + sel_round16(2 * static_cast<size_t>(kCap));
  o += sel_round16(sizeof(int) * 4) + sel_round16(8);
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
  s.list = reinterpret_cast<int16_t*>(take(2 * static_cast<size_t>(kCap)));
  s.cnt = reinterpret_cast<int*>(take(sizeof(int) * 4));
  s.thr = reinterpret_cast<unsigned long long*>(take(8));
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

// The selection passes. On entry s.q, s.ids and s.den hold the request's
// clamped q_cond, top-K ids and utility denominators, and a CTA barrier has
// passed. On return (after a barrier) buffer `cur` holds the nT selected
// nodes in key order.
__device__ void run_selection(const SelSmem& s, int L, int K, float tau, int n_max, int& nT_out,
                              int& cur_out) {
  const int tid = threadIdx.x, lane = tid & 31;
  const size_t C = static_cast<size_t>(n_max) + kCap;
  if (tid == 0) {
    const float den0 = s.den[0];
    NodeBuf T = node_buf(s.buf0, C);
    T.key[0] = ~0ull;   // the root ranks first
    T.reach[0] = 1.0f;
    T.util[0] = __fdiv_rn(1.0f, den0);
    T.ppos[0] = -1;
    T.depth[0] = 0;
    T.slot[0] = 0;
    T.done[0] = 1;      // listed for the first pass
    s.list[0] = 0;
    s.cnt[0] = 0;       // appended children, pass 0
    s.cnt[2] = 1;       // listed entries for pass 0
    *s.thr = n_max == 1 ? ~0ull : 0ull;
  }
  __syncthreads();

  const int max_expand = kCap / K;
  // this thread's child in step A: child j_own of listed member li_own
  const int li_own = tid / K;
  const int j_own = tid - li_own * K;
  int cur = 0, nT = 1;
  for (int pass = 0; pass < kMaxPasses; ++pass) {
    const int ph = pass & 1;
    const NodeBuf T = node_buf(cur ? s.buf1 : s.buf0, C);
    const NodeBuf Nx = node_buf(cur ? s.buf0 : s.buf1, C);
    int* kept = s.cnt + ph;
    int* listed = s.cnt + 2 + ph;

    // A. children of the listed members; append those that would enter T
    const int X = min(*listed, max_expand);
    const uint64_t thr = *s.thr;
    if (tid == 0) {
      // the next pass's counters (last read before the previous barrier)
      s.cnt[ph ^ 1] = 0;
      s.cnt[2 + (ph ^ 1)] = 0;
    }
    bool keep = false;
    uint64_t key = 0;
    float r = 0.f, u = 0.f;
    int t = 0, dc = 0;
    if (li_own < X) {
      t = s.list[li_own];
      const int dp = T.depth[t];
      const int row = dp == 0 ? 0 : T.slot[t];
      dc = dp + 1;
      r = __fmul_rn(T.reach[t], s.q[(dp * K + row) * K + j_own]);
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
    const int listed_now = *listed;
    if (m == 0 && listed_now <= max_expand) break;   // nothing left to expand or add

    // B. rank T and the appended children: g threads per entry. The entry
    //    ranked at n_max - 1 leaves a lower bound of its key (parent field
    //    cleared: renumbering only changes that field) for the next pass
    const int E = nT + m;
    int* listed_next = s.cnt + 2 + (ph ^ 1);
    if (tid == 0 && E < n_max) *s.thr = 0ull;
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
        const uint64_t ke1 = ke - 1;   // appended keys are >= 2^32: "> ke1" is ">= ke"
        const int c0 = nT + sub;
        int lo0 = 0, hi0 = 0, split = c0;
        if (e < nT) {
          // a member: members ahead of it are e; children ahead have a larger key
          if (sub == 0) cnt = e;
        } else {
          // an appended child: members with key >= ke (a prefix of T, whose
          // keys descend), then children with key >= ke before it and > ke
          // after it
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
      // entries that stay and still have children to generate are listed for
      // the next pass: one shared atomic per warp
      const bool open = sub == 0 && e < E && cnt < n_max && !T.done[e];
      const unsigned ob = __ballot_sync(kFullMask, open);
      int obase = 0;
      if (lane == 0 && ob) obase = atomicAdd(listed_next, __popc(ob));
      obase = __shfl_sync(kFullMask, obase, 0);
      if (sub == 0 && e < E) {
        if (e < nT) s.newpos[e] = static_cast<int16_t>(cnt < n_max ? cnt : -1);
        if (cnt < n_max) {
          unsigned char done = T.done[e];
          if (open) {
            const int idx = obase + __popc(ob & ((1u << lane) - 1u));
            if (idx < max_expand) {
              s.list[idx] = static_cast<int16_t>(cnt);
              done = 1;
            }
          }
          Nx.key[cnt] = ke;
          Nx.reach[cnt] = T.reach[e];
          Nx.util[cnt] = T.util[e];
          Nx.ppos[cnt] = T.ppos[e];
          Nx.depth[cnt] = T.depth[e];
          Nx.slot[cnt] = T.slot[e];
          Nx.done[cnt] = done;
          if (cnt == n_max - 1) *s.thr = ke & ~511ull;
        }
      }
    }
    __syncthreads();
    // renumber parents (a parent always ranks before its child, so it stayed);
    // the next pass reads these entries' keys only after its first barrier
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
  }
  __syncthreads();
  nT_out = nT;
  cur_out = cur;
}

// Write the selected nodes in key order, pad the rest.
__device__ void write_selection(const SelSmem& s, int n_max, int K, int nT, int cur, int b,
                                int32_t root_token, int32_t ctx, int32_t* n_nodes_out,
                                int32_t* parent_out, int32_t* depth_out, int32_t* token_out,
                                int32_t* slot_out, int32_t* pos_out, float* reach_out,
                                float* util_out) {
  const size_t C = static_cast<size_t>(n_max) + kCap;
  const NodeBuf T = node_buf(cur ? s.buf1 : s.buf0, C);
  const int64_t o = static_cast<int64_t>(b) * n_max;
  for (int i = threadIdx.x; i < n_max; i += kThreads) {
    if (i < nT) {
      const int d = T.depth[i];
      parent_out[o + i] = T.ppos[i];
      depth_out[o + i] = d;
      slot_out[o + i] = i == 0 ? -1 : T.slot[i];
      token_out[o + i] = i == 0 ? root_token : s.ids[(d - 1) * K + T.slot[i]];
      pos_out[o + i] = ctx + d;
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
  if (threadIdx.x == 0) n_nodes_out[b] = nT;
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
  const int tid = threadIdx.x;
  SelSmem s = carve(smem_raw, L, K, n_max);
  const float* qb = q_cond + static_cast<int64_t>(b) * L * K * K;
  for (int i = tid; i < L * K * K; i += kThreads) {
    const float v = qb[i];
    s.q[i] = v > 0.f ? fminf(v, 1.0f) : 0.f;
  }
  const int32_t* ib = ids + static_cast<int64_t>(b) * L * K;
  for (int i = tid; i < L * K; i += kThreads) s.ids[i] = ib[i];
  if (tid <= L) s.den[tid] = __fadd_rn(lambda1, __fmul_rn(lambda2, static_cast<float>(tid)));
  __syncthreads();
  int nT, cur;
  run_selection(s, L, K, tau, n_max, nT, cur);
  write_selection(s, n_max, K, nT, cur, b, root_tok[b], ctx_len[b], n_nodes_out, parent_out,
                  depth_out, token_out, slot_out, pos_out, reach_out, util_out);
}

// ---------------------------------------------------------------------------
// Selection and the ancestor mask in one launch per request (stages 3-4):
// the same selection as select_kernel, then each mask word built by walking
// the final parent list in shared memory, so the tree never makes a round
// trip through device memory between the two stages.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads, 1)
select_mask_kernel(const float* __restrict__ q_cond, const int* __restrict__ ids,
                   const int32_t* __restrict__ root_tok, const int32_t* __restrict__ ctx_len,
                   int L, int K, float lambda1, float lambda2, float tau, int n_max,
                   int32_t* __restrict__ n_nodes_out, int32_t* __restrict__ parent_out,
                   int32_t* __restrict__ depth_out, int32_t* __restrict__ token_out,
                   int32_t* __restrict__ slot_out, int32_t* __restrict__ pos_out,
                   float* __restrict__ reach_out, float* __restrict__ util_out,
                   uint32_t* __restrict__ mask_out) {
  dep_enter();
  extern __shared__ __align__(16) char smem_raw[];
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  SelSmem s = carve(smem_raw, L, K, n_max);
  const float* qb = q_cond + static_cast<int64_t>(b) * L * K * K;
  for (int i = tid; i < L * K * K; i += kThreads) {
    const float v = qb[i];
    s.q[i] = v > 0.f ? fminf(v, 1.0f) : 0.f;
  }
  const int32_t* ib = ids + static_cast<int64_t>(b) * L * K;
  for (int i = tid; i < L * K; i += kThreads) s.ids[i] = ib[i];
  if (tid <= L) s.den[tid] = __fadd_rn(lambda1, __fmul_rn(lambda2, static_cast<float>(tid)));
  __syncthreads();
  int nT, cur;
  run_selection(s, L, K, tau, n_max, nT, cur);
  write_selection(s, n_max, K, nT, cur, b, root_tok[b], ctx_len[b], n_nodes_out, parent_out,
                  depth_out, token_out, slot_out, pos_out, reach_out, util_out);
  const size_t C = static_cast<size_t>(n_max) + kCap;
  const NodeBuf T = node_buf(cur ? s.buf1 : s.buf0, C);
  const int W = (n_max + 31) / 32;
  uint32_t* mb = mask_out + static_cast<int64_t>(b) * n_max * W;
  for (int e = tid; e < n_max * W; e += kThreads) {
    const int i = e / W, wd = e % W;
    uint32_t word = 0;
    if (i < nT) {
      int j = i;
      while (j >= 0) {
        if ((j >> 5) == wd) word |= 1u << (j & 31);
        j = T.ppos[j];
      }
    }
    mb[e] = word;
  }
}

std::atomic<int> g_select_smem[64];
std::atomic<int> g_select_mask_smem[64];

int launch_select(const float* q_cond, const int32_t* topk_ids, const int32_t* root_tok,
                  const int32_t* ctx_len, int B, int L, int K, float l1, float l2, float tau,
                  int n_max, int32_t* n_nodes, int32_t* parent, int32_t* depth, int32_t* token,
                  int32_t* slot, int32_t* pos_id, float* reach, float* utility,
                  cudaStream_t stream) {
  const size_t smem = sel_smem_bytes(L, K, n_max);
  if (!smem_limit(select_kernel, smem, g_select_smem)) return TAPS_ERR_CUDA;
  if (launch_dep(select_kernel, dim3(B), dim3(kThreads), smem, stream, q_cond, topk_ids,
                 root_tok, ctx_len, L, K, l1, l2, tau, n_max, n_nodes, parent, depth, token,
                 slot, pos_id, reach, utility) != cudaSuccess)
    return TAPS_ERR_CUDA;
  return launch_status();
}

int launch_select_mask(const float* q_cond, const int32_t* topk_ids, const int32_t* root_tok,
                       const int32_t* ctx_len, int B, int L, int K, float l1, float l2, float tau,
                       int n_max, int32_t* n_nodes, int32_t* parent, int32_t* depth,
                       int32_t* token, int32_t* slot, int32_t* pos_id, float* reach,
                       float* utility, uint32_t* mask, cudaStream_t stream) {
  const size_t smem = sel_smem_bytes(L, K, n_max);
  if (!smem_limit(select_mask_kernel, smem, g_select_mask_smem)) return TAPS_ERR_CUDA;
  if (launch_dep(select_mask_kernel, dim3(B), dim3(kThreads), smem, stream, q_cond, topk_ids,
                 root_tok, ctx_len, L, K, l1, l2, tau, n_max, n_nodes, parent, depth, token,
                 slot, pos_id, reach, utility, mask) != cudaSuccess)
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

extern "C" int taps_score_select_mask(const int32_t* root_tok, const int32_t* topk_ids,
                                      const float* topk_logp, const float* entropy,
                                      const int32_t* ctx_len, int B, int L, int K,
                                      const taps_scorer_params* scorer,
                                      const taps_select_params* select, float* q_cond,
                                      int32_t* n_nodes, int32_t* parent, int32_t* depth,
                                      int32_t* token, int32_t* slot, int32_t* pos_id,
                                      float* reach, float* utility, uint32_t* mask,
                                      void* stream) {
  if (!root_tok || !topk_ids || !topk_logp || !ctx_len || !scorer || !select || !q_cond ||
      !n_nodes || !parent || !depth || !token || !slot || !pos_id || !reach || !utility || !mask)
    return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || L <= 0 || K <= 0) return TAPS_ERR_INVALID_ARG;
  const float l1 = select->lambda1, l2 = select->lambda2, tau = select->tau;
  const int n_max = select->n_max;
  if (!(l1 > 0.f) || !(l2 >= 0.f) || !(tau >= 0.f) || n_max < 1) return TAPS_ERR_INVALID_ARG;
  if (K > TAPS_MAX_K || L > TAPS_MAX_L || n_max > TAPS_MAX_NODES || B > 65535)
    return TAPS_ERR_UNSUPPORTED;
  const int kind = scorer->kind;
  int E = 0, H = 0;
  if (kind == TAPS_SCORER_MLP) {
    E = scorer->emb_dim;
    H = scorer->hidden;
    if (!scorer->weights || !entropy || E <= 0 || H <= 0 || scorer->vocab <= 0 ||
        scorer->max_depth <= L)
      return TAPS_ERR_INVALID_ARG;
    if (E > TAPS_MAX_EMB || H > TAPS_MAX_HIDDEN) return TAPS_ERR_UNSUPPORTED;
  } else if (kind != TAPS_SCORER_MARGINAL && kind != TAPS_SCORER_MARGINAL_PRODUCT) {
    return TAPS_ERR_INVALID_ARG;
  }
  // scoring keeps its own launch, one CTA per (position, request), which
  // spreads a batch-1 round over many SMs; selection and mask share one
  const int st = taps_score_reach(root_tok, topk_ids, topk_logp, entropy, B, L, K, scorer, q_cond,
                                  nullptr, nullptr, 0, nullptr, stream);
  if (st != TAPS_OK) return st;
  return launch_select_mask(q_cond, topk_ids, root_tok, ctx_len, B, L, K, l1, l2, tau, n_max,
                            n_nodes, parent, depth, token, slot, pos_id, reach, utility, mask,
                            static_cast<cudaStream_t>(stream));
}
