// Stage 3 of a TAPS round (Sec. 4.2-4.3, Eq. 2, Eq. 3, Algorithm 1):
// reach, utility and the greedy budgeted prefix-closed selection.
//
// One warp per request, everything in shared memory. Algorithm 1 adds, one
// node at a time, the unselected node of largest utility. Utility never
// increases from a parent to a child (q_cond <= 1, den(d) non-decreasing,
// monotone rounding) and ties favour the lower depth, so that node is always
// a child of a selected node, and its ancestors are already selected. Among
// the children of one selected node, they are selected in key order, so the
// frontier only needs, per selected node, its best unselected child: when
// node p's rank-r child is taken, its rank-(r+1) sibling enters the frontier,
// and the new node's rank-0 child enters too. The frontier therefore never
// exceeds n_max + 1 entries; each step is one 64-bit warp maximum.
//
// Frontier key (larger = taken first): utility bits (non-negative floats
// order like their bit patterns) | (31 - depth) | (2^18 - 1 - token) |
// (511 - parent index), i.e. utility desc, depth asc, token asc, parent asc.
//
// All reach/utility arithmetic is IEEE f32 round-to-nearest (explicit _rn
// intrinsics, no contraction), root to leaf.
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

struct SelSmem {
  float* q;          // [L][K][K]
  int* ids;          // [L][K]
  float* den;        // [L + 1]
  int* parent;       // [n_max]
  float* reach;      // [n_max]
  float* util;       // [n_max]
  unsigned char* depth;   // [n_max]
  unsigned char* slot;    // [n_max]
  unsigned char* order;   // [n_max][K]  slot of the rank-r child
  uint64_t* fkey;    // [n_max + 1] frontier keys (0 = empty)
  unsigned* finfo;   // [n_max + 1] parent << 8 | rank
  float* freach;     // [n_max + 1]
};

__host__ __device__ inline size_t sel_smem_bytes(int L, int K, int n_max) {
  size_t o = 0;
  o += sizeof(uint64_t) * (n_max + 1);
  o += sizeof(float) * L * K * K;
  o += sizeof(int) * L * K;
  o += sizeof(float) * 32;
  o += sizeof(int) * n_max + 2 * sizeof(float) * n_max;
  o += sizeof(unsigned) * (n_max + 1) + sizeof(float) * (n_max + 1);
  o += 2 * n_max + static_cast<size_t>(n_max) * K;
  return (o + 15) / 16 * 16;
}

__device__ SelSmem carve(char* base, int L, int K, int n_max) {
  SelSmem s;
  char* p = base;
  s.fkey = reinterpret_cast<uint64_t*>(p);  p += sizeof(uint64_t) * (n_max + 1);
  s.q = reinterpret_cast<float*>(p);        p += sizeof(float) * L * K * K;
  s.ids = reinterpret_cast<int*>(p);        p += sizeof(int) * L * K;
  s.den = reinterpret_cast<float*>(p);      p += sizeof(float) * 32;
  s.parent = reinterpret_cast<int*>(p);     p += sizeof(int) * n_max;
  s.reach = reinterpret_cast<float*>(p);    p += sizeof(float) * n_max;
  s.util = reinterpret_cast<float*>(p);     p += sizeof(float) * n_max;
  s.finfo = reinterpret_cast<unsigned*>(p); p += sizeof(unsigned) * (n_max + 1);
  s.freach = reinterpret_cast<float*>(p);   p += sizeof(float) * (n_max + 1);
  s.depth = reinterpret_cast<unsigned char*>(p); p += n_max;
  s.slot = reinterpret_cast<unsigned char*>(p);  p += n_max;
  s.order = reinterpret_cast<unsigned char*>(p);
  return s;
}

// Lanes j < K compute the keys of node v's children, rank them, record the
// order and return (on every lane) the rank-0 child's key, slot and reach.
__device__ __forceinline__ void expand(const SelSmem& s, int v, int K, int lane,
                                       uint64_t& key0, float& reach0) {
  const int dv = s.depth[v];
  const int row = dv == 0 ? 0 : s.slot[v];
  const float rv = s.reach[v];
  uint64_t key = 0;
  float r = 0.f;
  if (lane < K) {
    r = __fmul_rn(rv, s.q[(dv * K + row) * K + lane]);
    float u = __fdiv_rn(r, s.den[dv + 1]);
    key = node_key(u, dv + 1, s.ids[dv * K + lane], v);
  }
  int rank = 0;
  for (int k = 0; k < K; ++k) {
    uint64_t other = __shfl_sync(kFullMask, key, k);
    rank += (other > key) ? 1 : 0;
  }
  if (lane < K) s.order[v * K + rank] = static_cast<unsigned char>(lane);
  unsigned first = __ballot_sync(kFullMask, lane < K && rank == 0);
  int src = __ffs(first) - 1;
  key0 = __shfl_sync(kFullMask, key, src);
  reach0 = __shfl_sync(kFullMask, r, src);
}

__global__ void __launch_bounds__(32)
select_kernel(const float* __restrict__ q_cond, const int32_t* __restrict__ ids,
              const int32_t* __restrict__ root_tok, const int32_t* __restrict__ ctx_len, int L,
              int K, float lambda1, float lambda2, float tau, int n_max,
              int32_t* __restrict__ n_nodes_out, int32_t* __restrict__ parent_out,
              int32_t* __restrict__ depth_out, int32_t* __restrict__ token_out,
              int32_t* __restrict__ slot_out, int32_t* __restrict__ pos_out,
              float* __restrict__ reach_out, float* __restrict__ util_out) {
  extern __shared__ __align__(16) char smem_raw[];
  const int b = blockIdx.x;
  const int lane = threadIdx.x;
  SelSmem s = carve(smem_raw, L, K, n_max);

  const float* qb = q_cond + static_cast<int64_t>(b) * L * K * K;
  for (int i = lane; i < L * K * K; i += 32) s.q[i] = qb[i];
  const int32_t* ib = ids + static_cast<int64_t>(b) * L * K;
  for (int i = lane; i < L * K; i += 32) s.ids[i] = ib[i];
  if (lane <= L) s.den[lane] = __fadd_rn(lambda1, __fmul_rn(lambda2, static_cast<float>(lane)));
  for (int i = lane; i <= n_max; i += 32) s.fkey[i] = 0;
  __syncwarp();

  // root
  if (lane == 0) {
    s.parent[0] = -1;
    s.depth[0] = 0;
    s.slot[0] = 0;
    s.reach[0] = 1.0f;
    s.util[0] = __fdiv_rn(1.0f, s.den[0]);
  }
  __syncwarp();
  int n = 1;
  int fsize = 0;
  uint64_t my_best = 0;   // best key among the frontier slots this lane owns
  int my_slot = -1;

  if (n < n_max && L > 0) {
    uint64_t k0;
    float r0;
    expand(s, 0, K, lane, k0, r0);
    if (lane == 0) {
      s.fkey[0] = k0;
      s.finfo[0] = 0u;          // parent 0, rank 0
      s.freach[0] = r0;
      my_best = k0;
      my_slot = 0;
    }
    fsize = 1;
    __syncwarp();
  }

  while (n < n_max) {
    uint64_t best = warp_max_u64(my_best);
    if (best == 0) break;
    float bu = __uint_as_float(static_cast<uint32_t>(best >> 32));
    if (!(bu > tau)) break;
    unsigned win = __ballot_sync(kFullMask, my_best == best);
    int wl = __ffs(win) - 1;
    int fslot = __shfl_sync(kFullMask, my_slot, wl);
    unsigned info = s.finfo[fslot];
    float vr = s.freach[fslot];
    int p = static_cast<int>(info >> 8);
    int rank = static_cast<int>(info & 0xffu);
    int dp = s.depth[p];
    int j = s.order[p * K + rank];
    int v = n;
    if (lane == 0) {
      s.parent[v] = p;
      s.depth[v] = static_cast<unsigned char>(dp + 1);
      s.slot[v] = static_cast<unsigned char>(j);
      s.reach[v] = vr;
      s.util[v] = bu;
    }
    __syncwarp();
    n++;
    // candidate 1: next sibling of v (rank + 1 under p)
    uint64_t k_sib = 0;
    float r_sib = 0.f;
    if (rank + 1 < K) {
      int js = s.order[p * K + rank + 1];
      int prow = dp == 0 ? 0 : s.slot[p];
      r_sib = __fmul_rn(s.reach[p], s.q[(dp * K + prow) * K + js]);
      float us = __fdiv_rn(r_sib, s.den[dp + 1]);
      k_sib = node_key(us, dp + 1, s.ids[dp * K + js], p);
    }
    // candidate 2: best child of v
    uint64_t k_ch = 0;
    float r_ch = 0.f;
    if (dp + 1 < L && n < n_max) {
      expand(s, v, K, lane, k_ch, r_ch);
    }
    // the popped slot takes one candidate, a fresh slot the other
    int slot_a = fslot;
    uint64_t ka = k_sib ? k_sib : k_ch;
    unsigned ia = k_sib ? ((static_cast<unsigned>(p) << 8) | (rank + 1))
                        : (static_cast<unsigned>(v) << 8);
    float ra = k_sib ? r_sib : r_ch;
    bool has_b = k_sib && k_ch;
    int slot_b = fsize;
    if (lane == 0) {
      s.fkey[slot_a] = ka;
      s.finfo[slot_a] = ia;
      s.freach[slot_a] = ra;
      if (has_b) {
        s.fkey[slot_b] = k_ch;
        s.finfo[slot_b] = static_cast<unsigned>(v) << 8;
        s.freach[slot_b] = r_ch;
      }
    }
    if (has_b) fsize++;
    __syncwarp();
    // refresh the per-lane maxima of the owners of the touched slots
    if (lane == (slot_a & 31)) {
      my_best = 0;
      my_slot = -1;
      for (int f = lane; f < fsize; f += 32) {
        uint64_t kf = s.fkey[f];
        if (kf > my_best) {
          my_best = kf;
          my_slot = f;
        }
      }
    }
    if (has_b && lane == (slot_b & 31) && lane != (slot_a & 31)) {
      if (k_ch > my_best) {
        my_best = k_ch;
        my_slot = slot_b;
      }
    }
    __syncwarp();
  }

  // write the selected nodes in selection order, pad the rest
  const int64_t o = static_cast<int64_t>(b) * n_max;
  const int c = ctx_len[b];
  for (int i = lane; i < n_max; i += 32) {
    if (i < n) {
      int d = s.depth[i];
      parent_out[o + i] = s.parent[i];
      depth_out[o + i] = d;
      slot_out[o + i] = i == 0 ? -1 : s.slot[i];
      token_out[o + i] = i == 0 ? root_tok[b] : s.ids[(d - 1) * K + s.slot[i]];
      pos_out[o + i] = c + d;
      reach_out[o + i] = s.reach[i];
      util_out[o + i] = s.util[i];
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
  if (lane == 0) n_nodes_out[b] = n;
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
  size_t smem = sel_smem_bytes(L, K, n_max);
  if (smem > 48 * 1024) {
    if (cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess)
      return TAPS_ERR_CUDA;
  }
  select_kernel<<<B, 32, smem, static_cast<cudaStream_t>(stream)>>>(
      q_cond, topk_ids, root_tok, ctx_len, L, K, l1, l2, tau, n_max, n_nodes, parent, depth,
      token, slot, pos_id, reach, utility);
  return launch_status();
}
