// Stage 3 of a TAPS round (Sec. 4.2-4.3, Eq. 2, Eq. 3, Algorithm 1):
// reach, utility and the greedy budgeted prefix-closed selection.
//
// One warp per request, everything in shared memory. Algorithm 1 adds, one
// node at a time, the unselected node of largest utility. Utility never
// increases from a parent to a child (q_cond <= 1, den(d) non-decreasing,
// monotone rounding) and ties favour the lower depth, so that node is always
// a child of a selected node, and its ancestors are already selected. Among
// the children of one selected node, they are selected in key order, so the
// frontier only needs, per selected node, its best unselected child: when a
// child of node p is taken, p's next child in key order (the largest key
// below the taken one) enters the frontier, and the new node's best child
// enters too. The frontier therefore never exceeds n_max + 1 entries. A step
// is one 64-bit warp maximum over the frontier (held in registers), then lane
// k computes child k of the new node and child k of its parent side by side,
// and two more warp maxima pick the two entries.
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
  float* den;        // [32]
  int* parent;       // [n_max]
  float* reach;      // [n_max]
  float* util;       // [n_max]
  unsigned char* depth;   // [n_max]
  unsigned char* slot;    // [n_max]
};

__host__ __device__ inline size_t sel_smem_bytes(int L, int K, int n_max) {
  size_t o = 0;
  o += sizeof(float) * L * K * K;
  o += sizeof(int) * L * K;
  o += sizeof(float) * 32;
  o += sizeof(int) * n_max + 2 * sizeof(float) * n_max;
  o += 2 * n_max;
  return (o + 15) / 16 * 16;
}

__device__ SelSmem carve(char* base, int L, int K, int n_max) {
  SelSmem s;
  char* p = base;
  s.q = reinterpret_cast<float*>(p);        p += sizeof(float) * L * K * K;
  s.ids = reinterpret_cast<int*>(p);        p += sizeof(int) * L * K;
  s.den = reinterpret_cast<float*>(p);      p += sizeof(float) * 32;
  s.parent = reinterpret_cast<int*>(p);     p += sizeof(int) * n_max;
  s.reach = reinterpret_cast<float*>(p);    p += sizeof(float) * n_max;
  s.util = reinterpret_cast<float*>(p);     p += sizeof(float) * n_max;
  s.depth = reinterpret_cast<unsigned char*>(p); p += n_max;
  s.slot = reinterpret_cast<unsigned char*>(p);
  return s;
}

// A frontier entry stands for the best unselected child of a selected node p:
// its key, its reach, p's reach, and packed p (9 bits) | the child's slot (5)
// | p's depth (5) | p's slot (5).
__device__ __forceinline__ uint32_t pack_info(int p, int slot, int dp, int pslot) {
  return (static_cast<uint32_t>(p) << 15) | (static_cast<uint32_t>(slot) << 10) |
         (static_cast<uint32_t>(dp) << 5) | static_cast<uint32_t>(pslot);
}

// Key and reach of the child in slot j of a node at depth dp, row `row` of the
// q_cond table (its own slot; 0 for the root), reach rp, selection index p.
__device__ __forceinline__ uint64_t child_key(const SelSmem& s, int K, int dp, int row, int j,
                                              float rp, int p, float& r) {
  r = __fmul_rn(rp, s.q[(dp * K + row) * K + j]);
  const float u = __fdiv_rn(r, s.den[dp + 1]);
  return node_key(u, dp + 1, s.ids[dp * K + j], p);
}

// Frontier slot f lives in lane f % 32, entry f / 32 of that lane's arrays
// (fully unrolled, so that the arrays stay in registers).
template <int SPL>
__device__ __forceinline__ void set_entry(uint64_t (&fk)[SPL], uint32_t (&fi)[SPL],
                                          float (&fr)[SPL], float (&frp)[SPL], int lane, int f,
                                          uint64_t key, uint32_t info, float r, float rp) {
#pragma unroll
  for (int i = 0; i < SPL; ++i) {
    const bool hit = lane == (f & 31) && i == (f >> 5);
    fk[i] = hit ? key : fk[i];
    fi[i] = hit ? info : fi[i];
    fr[i] = hit ? r : fr[i];
    frp[i] = hit ? rp : frp[i];
  }
}

// SPL: frontier slots per lane.
template <int SPL>
__global__ void __launch_bounds__(32)
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
  const int lane = threadIdx.x;
  SelSmem s = carve(smem_raw, L, K, n_max);

  const float* qb = q_cond + static_cast<int64_t>(b) * L * K * K;
  for (int i = lane; i < L * K * K; i += 32) s.q[i] = qb[i];
  const int32_t* ib = ids + static_cast<int64_t>(b) * L * K;
  for (int i = lane; i < L * K; i += 32) s.ids[i] = ib[i];
  if (lane <= L) s.den[lane] = __fadd_rn(lambda1, __fmul_rn(lambda2, static_cast<float>(lane)));
  if (lane == 0) {
    s.parent[0] = -1;
    s.depth[0] = 0;
    s.slot[0] = 0;
    s.reach[0] = 1.0f;
  }
  __syncwarp();
  if (lane == 0) s.util[0] = __fdiv_rn(1.0f, s.den[0]);

  // the frontier, in registers
  uint64_t fk[SPL];
  uint32_t fi[SPL];
  float fr[SPL], frp[SPL];
#pragma unroll
  for (int i = 0; i < SPL; ++i) {
    fk[i] = 0;
    fi[i] = 0;
    fr[i] = 0.f;
    frp[i] = 0.f;
  }
  uint64_t my_best = 0;
  int n = 1, fsize = 0;

  if (n < n_max && L > 0) {
    float r = 0.f;
    const uint64_t key = lane < K ? child_key(s, K, 0, 0, lane, 1.0f, 0, r) : 0ull;
    const uint64_t k0 = warp_max_u64(key);
    const int src = __ffs(__ballot_sync(kFullMask, key == k0)) - 1;
    set_entry<SPL>(fk, fi, fr, frp, lane, 0, k0, pack_info(0, src, 0, 0),
                   __shfl_sync(kFullMask, r, src), 1.0f);
    fsize = 1;
    my_best = lane == 0 ? fk[0] : 0ull;
  }

  while (n < n_max) {
    const uint64_t best = warp_max_u64(my_best);
    if (best == 0) break;
    const float bu = __uint_as_float(static_cast<uint32_t>(best >> 32));
    if (!(bu > tau)) break;
    // the owner of the winning entry hands it to the warp
    const int wl = __ffs(__ballot_sync(kFullMask, my_best == best)) - 1;
    int wi = 0;
    uint32_t info = 0;
    float r = 0.f, rp = 0.f;
#pragma unroll
    for (int i = 0; i < SPL; ++i)
      if (fk[i] == best) {
        wi = i;
        info = fi[i];
        r = fr[i];
        rp = frp[i];
      }
    const int fslot = (__shfl_sync(kFullMask, wi, wl) << 5) | wl;
    info = __shfl_sync(kFullMask, info, wl);
    r = __shfl_sync(kFullMask, r, wl);
    rp = __shfl_sync(kFullMask, rp, wl);
    const int p = static_cast<int>(info >> 15), j = static_cast<int>((info >> 10) & 31u);
    const int dp = static_cast<int>((info >> 5) & 31u), pslot = static_cast<int>(info & 31u);
    const int v = n, dv = dp + 1;
    if (lane == 0) {
      s.parent[v] = p;
      s.depth[v] = static_cast<unsigned char>(dv);
      s.slot[v] = static_cast<unsigned char>(j);
      s.reach[v] = r;
      s.util[v] = bu;
    }
    n++;
    // child k of v and child k of p, side by side: in lanes k and K + k when
    // 2K lanes suffice (one instruction stream: a divergent branch per node
    // would run the two halves one after the other), else in two passes
    const bool has_child = dv < L && n < n_max;
    float rc = 0.f, rs = 0.f;
    uint64_t kc = 0, ks = 0;
    const int prow = dp == 0 ? 0 : pslot;
    if (2 * K <= 32) {
      const bool of_v = lane < K;
      const int k = of_v ? lane : lane - K;
      float rr = 0.f;
      uint64_t key = 0;
      if ((of_v && has_child) || (!of_v && k < K))
        key = child_key(s, K, of_v ? dv : dp, of_v ? j : prow, k, of_v ? r : rp, of_v ? v : p, rr);
      if (of_v) {
        kc = key;
        rc = rr;
      } else {
        ks = key < best ? key : 0ull;   // p's children taken so far have keys >= the popped one
        rs = rr;
      }
    } else {
      if (lane < K && has_child) kc = child_key(s, K, dv, j, lane, r, v, rc);
      if (lane < K) {
        ks = child_key(s, K, dp, prow, lane, rp, p, rs);
        if (ks >= best) ks = 0;
      }
    }
    const uint64_t k0 = warp_max_u64(kc);
    const uint64_t k1 = warp_max_u64(ks);
    const int c0 = k0 ? __ffs(__ballot_sync(kFullMask, kc == k0)) - 1 : 0;
    const int l1 = k1 ? __ffs(__ballot_sync(kFullMask, ks == k1)) - 1 : 0;
    const int c1 = 2 * K <= 32 && k1 ? l1 - K : l1;   // the child slot of p's entry
    const float r0 = __shfl_sync(kFullMask, rc, c0);
    const float r1 = __shfl_sync(kFullMask, rs, l1);
    // the popped slot takes the sibling (else the child), a fresh slot the child
    const uint32_t child_info = pack_info(v, c0, dv, j);
    if (k1) {
      set_entry<SPL>(fk, fi, fr, frp, lane, fslot, k1, pack_info(p, c1, dp, pslot), r1, rp);
      if (k0) {
        set_entry<SPL>(fk, fi, fr, frp, lane, fsize, k0, child_info, r0, r);
        fsize++;
      }
    } else {
      set_entry<SPL>(fk, fi, fr, frp, lane, fslot, k0, child_info, r0, r);
    }
    my_best = 0;
#pragma unroll
    for (int i = 0; i < SPL; ++i) my_best = fk[i] > my_best ? fk[i] : my_best;
  }
  __syncwarp();

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

template <int SPL>
int launch_select(const float* q_cond, const int32_t* topk_ids, const int32_t* root_tok,
                  const int32_t* ctx_len, int B, int L, int K, float l1, float l2, float tau,
                  int n_max, int32_t* n_nodes, int32_t* parent, int32_t* depth, int32_t* token,
                  int32_t* slot, int32_t* pos_id, float* reach, float* utility,
                  cudaStream_t stream) {
  const size_t smem = sel_smem_bytes(L, K, n_max);
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(select_kernel<SPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return TAPS_ERR_CUDA;
  if (launch_dep(select_kernel<SPL>, dim3(B), dim3(32), smem, stream, q_cond, topk_ids, root_tok,
                 ctx_len, L, K, l1, l2, tau, n_max, n_nodes, parent, depth, token, slot, pos_id,
                 reach, utility) != cudaSuccess)
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
  // the frontier holds at most one entry per selected node (n_max + 1)
  const int fmax = n_max + 1;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
#define TAPS_SELECT_LAUNCH(SPL)                                                               \
  return launch_select<SPL>(q_cond, topk_ids, root_tok, ctx_len, B, L, K, l1, l2, tau, n_max, \
                            n_nodes, parent, depth, token, slot, pos_id, reach, utility, st)
  if (fmax <= 32) TAPS_SELECT_LAUNCH(1);
  if (fmax <= 96) TAPS_SELECT_LAUNCH(3);
  if (fmax <= 288) TAPS_SELECT_LAUNCH(9);
  TAPS_SELECT_LAUNCH(17);
#undef TAPS_SELECT_LAUNCH
}
