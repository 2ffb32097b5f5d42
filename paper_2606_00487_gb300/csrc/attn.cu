// Stage 5 of a TAPS round (Sec. 4.1 stage 3): tree attention of the selected
// nodes against the target's paged bf16 KV cache.
//
// Rows of one KV head are (node, query head in the GQA group) pairs, row
// r = node * group + g, so the whole group shares every K/V tile. The logical
// sequence [0, ctx_len + n_nodes) is split into chunks; one CTA handles one
// (chunk, KV head, 64-row tile, request), runs an online softmax over its
// chunk and either writes the final rows (single chunk) or an unnormalised
// partial that a combine kernel merges with log-sum-exp weights.
#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace taps {
namespace attn {

constexpr int kThreads = 256;
constexpr int kRowTile = 64;
constexpr int kKvTile = 64;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct Plan {
  int group, rows_max, row_tiles, splits, chunk_len;
};

inline Plan make_plan(int B, int n_max, int Hq, int Hkv, int max_ctx) {
  Plan p;
  p.group = Hq / Hkv;
  p.rows_max = n_max * p.group;
  p.row_tiles = (p.rows_max + kRowTile - 1) / kRowTile;
  const int64_t units = static_cast<int64_t>(B) * Hkv * p.row_tiles;
  const int max_total = max_ctx + n_max;
  int want = static_cast<int>((2 * kTargetSms + units - 1) / units);
  int cap = std::max(1, (max_total + 255) / 256);
  int splits = std::max(1, std::min(want, cap));
  int chunk = (max_total + splits - 1) / splits;
  chunk = (chunk + kKvTile - 1) / kKvTile * kKvTile;
  p.chunk_len = chunk;
  p.splits = (max_total + chunk - 1) / chunk;
  return p;
}

struct WsLayout {
  size_t opart, ml, total;
};

inline WsLayout ws_layout(const Plan& p, int B, int Hkv, int D) {
  WsLayout w{0, 0, 0};
  if (p.splits <= 1) return w;
  const size_t slots = static_cast<size_t>(B) * Hkv * p.rows_max * p.splits;
  size_t o = 0;
  w.opart = o;
  o = align_up(o + slots * D * sizeof(float), 256);
  w.ml = o;
  o = align_up(o + slots * sizeof(float2), 256);
  w.total = o;
  return w;
}

struct Args {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k;
  const __nv_bfloat16* v;
  int64_t num_pages;
  const int32_t* block_table;
  int max_pages;
  const int32_t* ctx_len;
  const int32_t* n_nodes;
  const uint32_t* mask;
  int n_max, Hq, Hkv, W;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float* opart;
  float2* ml;
  int32_t* status;
  Plan plan;
};

template <int D>
__global__ void __launch_bounds__(kThreads) attn_chunk_kernel(Args a) {
  constexpr int LD = D + 8;               // padded bf16 row stride of the smem tiles
  constexpr int DPT = D / 4;              // output dims per thread
  extern __shared__ __align__(16) char smem[];
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem);
  __nv_bfloat16* sK = sQ + kRowTile * LD;
  __nv_bfloat16* sV = sK + kKvTile * LD;
  float* sP = reinterpret_cast<float*>(sV + kKvTile * LD);   // [kRowTile][kKvTile + 1]
  __shared__ int s_colok[kKvTile];

  const Plan& pl = a.plan;
  const int b = blockIdx.z;
  const int kv = blockIdx.y / pl.row_tiles;
  const int rt = blockIdx.y % pl.row_tiles;
  const int split = blockIdx.x;
  const int tid = threadIdx.x;
  const int n = min(max(a.n_nodes[b], 0), a.n_max);
  const int C = a.ctx_len[b];
  const int total = C + n;
  const int rows = n * pl.group;
  const int row0 = rt * kRowTile;

  if (row0 >= rows) {
    if (pl.splits == 1 && split == 0) {       // zero the padding rows of this tile
      for (int e = tid; e < kRowTile * D; e += kThreads) {
        int r = row0 + e / D;
        if (r < pl.rows_max) {
          int i = r / pl.group, h = kv * pl.group + r % pl.group;
          a.out[((static_cast<int64_t>(b) * a.n_max + i) * a.Hq + h) * D + e % D] =
              __float2bfloat16(0.f);
          if (a.lse && e % D == 0) a.lse[(static_cast<int64_t>(b) * a.n_max + i) * a.Hq + h] = 0.f;
        }
      }
    }
    return;
  }
  const int pos0 = split * pl.chunk_len;
  const int pos1 = min(pos0 + pl.chunk_len, total);

  // Q tile
  for (int e = tid; e < kRowTile * (D / 8); e += kThreads) {
    int rr = e / (D / 8), c8 = e % (D / 8);
    int r = row0 + rr;
    uint4 val = make_uint4(0, 0, 0, 0);
    if (r < rows) {
      int i = r / pl.group, h = kv * pl.group + r % pl.group;
      val = *reinterpret_cast<const uint4*>(
          a.q + ((static_cast<int64_t>(b) * a.n_max + i) * a.Hq + h) * D + c8 * 8);
    }
    *reinterpret_cast<uint4*>(sQ + rr * LD + c8 * 8) = val;
  }

  const int srow = tid >> 2;              // score row of this thread
  const int cg = tid & 3;                 // columns cg, cg + 4, ... (interleaved)
  const int r_glob = row0 + srow;
  const int node = r_glob / pl.group;
  const uint32_t* mrow = a.mask + (static_cast<int64_t>(b) * a.n_max + min(node, a.n_max - 1)) * a.W;
  float m2 = -INFINITY, l = 0.f;
  float o[DPT];
#pragma unroll
  for (int i = 0; i < DPT; ++i) o[i] = 0.f;

  for (int t0 = pos0; t0 < pos1; t0 += kKvTile) {
    __syncthreads();
    // K/V tile through the block table
    for (int e = tid; e < kKvTile * (D / 8); e += kThreads) {
      int c = e / (D / 8), c8 = e % (D / 8);
      int p = t0 + c;
      uint4 kval = make_uint4(0, 0, 0, 0), vval = make_uint4(0, 0, 0, 0);
      bool ok = false;
      if (p < pos1) {
        int lp = p / 16;
        int page = lp < a.max_pages ? a.block_table[static_cast<int64_t>(b) * a.max_pages + lp] : -1;
        if (page >= 0 && page < a.num_pages) {
          int64_t off = ((static_cast<int64_t>(page) * a.Hkv + kv) * 16 + (p & 15)) * D + c8 * 8;
          kval = *reinterpret_cast<const uint4*>(a.k + off);
          vval = *reinterpret_cast<const uint4*>(a.v + off);
          ok = true;
        } else if (a.status && c8 == 0) {
          atomicOr(a.status, TAPS_DEVFAULT_PAGE);
        }
      }
      *reinterpret_cast<uint4*>(sK + c * LD + c8 * 8) = kval;
      *reinterpret_cast<uint4*>(sV + c * LD + c8 * 8) = vval;
      if (c8 == 0) s_colok[c] = ok;
    }
    __syncthreads();
    // scores for (srow, cg + 4k)
    float s[kKvTile / 4];
    float tmax = -INFINITY;
#pragma unroll
    for (int k = 0; k < kKvTile / 4; ++k) {
      int c = cg + 4 * k;
      float acc = 0.f;
      const __nv_bfloat16* qr = sQ + srow * LD;
      const __nv_bfloat16* kr = sK + c * LD;
#pragma unroll
      for (int d = 0; d < D; d += 8) {
        uint4 qv = *reinterpret_cast<const uint4*>(qr + d);
        uint4 kk = *reinterpret_cast<const uint4*>(kr + d);
        const __nv_bfloat162* q2 = reinterpret_cast<const __nv_bfloat162*>(&qv);
        const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&kk);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          float2 qf = __bfloat1622float2(q2[u]);
          float2 kf = __bfloat1622float2(k2[u]);
          acc = fmaf(qf.x, kf.x, acc);
          acc = fmaf(qf.y, kf.y, acc);
        }
      }
      int p = t0 + c;
      bool vis = s_colok[c] && p < pos1 && r_glob < rows;
      if (vis && p >= C) {
        int j = p - C;
        vis = (mrow[j >> 5] >> (j & 31)) & 1u;
      }
      s[k] = vis ? acc * a.scale_log2 : -INFINITY;
      tmax = fmaxf(tmax, s[k]);
    }
    tmax = fmaxf(tmax, __shfl_xor_sync(kFullMask, tmax, 1));
    tmax = fmaxf(tmax, __shfl_xor_sync(kFullMask, tmax, 2));
    float m_new = fmaxf(m2, tmax);
    float alpha = (m_new == -INFINITY) ? 1.f : exp2f(m2 - m_new);
    float psum = 0.f;
#pragma unroll
    for (int k = 0; k < kKvTile / 4; ++k) {
      float pv = (m_new == -INFINITY) ? 0.f : exp2f(s[k] - m_new);
      psum += pv;
      sP[srow * (kKvTile + 1) + cg + 4 * k] = pv;
    }
    psum += __shfl_xor_sync(kFullMask, psum, 1);
    psum += __shfl_xor_sync(kFullMask, psum, 2);
    l = l * alpha + psum;
    m2 = m_new;
#pragma unroll
    for (int i = 0; i < DPT; ++i) o[i] *= alpha;
    __syncthreads();
    // O += P V for (srow, dims cg*DPT ..)
    const float* prow = sP + srow * (kKvTile + 1);
    for (int c = 0; c < kKvTile; ++c) {
      float pv = prow[c];
      const __nv_bfloat16* vr = sV + c * LD + cg * DPT;
#pragma unroll
      for (int i = 0; i < DPT; i += 8) {
        uint4 vv = *reinterpret_cast<const uint4*>(vr + i);
        const __nv_bfloat162* v2 = reinterpret_cast<const __nv_bfloat162*>(&vv);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          float2 vf = __bfloat1622float2(v2[u]);
          o[i + 2 * u] = fmaf(pv, vf.x, o[i + 2 * u]);
          o[i + 2 * u + 1] = fmaf(pv, vf.y, o[i + 2 * u + 1]);
        }
      }
    }
  }

  if (r_glob >= pl.rows_max) return;
  const int i_node = r_glob / pl.group;
  const int h = kv * pl.group + r_glob % pl.group;
  const int64_t orow = (static_cast<int64_t>(b) * a.n_max + i_node) * a.Hq + h;
  if (pl.splits == 1) {
    const bool valid = r_glob < rows && l > 0.f;
    const float inv = valid ? 1.f / l : 0.f;
#pragma unroll
    for (int i = 0; i < DPT; ++i)
      a.out[orow * D + cg * DPT + i] = __float2bfloat16(valid ? o[i] * inv : 0.f);
    if (a.lse && cg == 0) a.lse[orow] = valid ? (m2 + log2f(l)) * kLn2 : 0.f;
  } else if (r_glob < rows) {
    const int64_t slot =
        ((static_cast<int64_t>(b) * a.Hkv + kv) * pl.rows_max + r_glob) * pl.splits + split;
#pragma unroll
    for (int i = 0; i < DPT; ++i) a.opart[slot * D + cg * DPT + i] = o[i];
    if (cg == 0) a.ml[slot] = make_float2(m2, l);
  }
}

template <int D>
__global__ void __launch_bounds__(256) attn_merge_kernel(Args a, int B) {
  const Plan& pl = a.plan;
  const int64_t wid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t per_b = static_cast<int64_t>(a.Hkv) * pl.rows_max;
  if (wid >= per_b * B) return;
  const int b = static_cast<int>(wid / per_b);
  const int rem = static_cast<int>(wid % per_b);
  const int kv = rem / pl.rows_max;
  const int r = rem % pl.rows_max;
  const int n = min(max(a.n_nodes[b], 0), a.n_max);
  const int rows = n * pl.group;
  const int i_node = r / pl.group;
  const int h = kv * pl.group + r % pl.group;
  const int64_t orow = (static_cast<int64_t>(b) * a.n_max + i_node) * a.Hq + h;
  if (r >= rows) {
    for (int d = lane; d < D; d += 32) a.out[orow * D + d] = __float2bfloat16(0.f);
    if (a.lse && lane == 0) a.lse[orow] = 0.f;
    return;
  }
  const int total = a.ctx_len[b] + n;
  const int active = min(pl.splits, (total + pl.chunk_len - 1) / pl.chunk_len);
  const int64_t slot0 = ((static_cast<int64_t>(b) * a.Hkv + kv) * pl.rows_max + r) * pl.splits;
  float M = -INFINITY;
  for (int s = 0; s < active; ++s) M = fmaxf(M, a.ml[slot0 + s].x);
  float Lsum = 0.f;
  float acc[D / 32];
#pragma unroll
  for (int i = 0; i < D / 32; ++i) acc[i] = 0.f;
  for (int s = 0; s < active; ++s) {
    float2 ml = a.ml[slot0 + s];
    if (!(ml.y > 0.f)) continue;
    float wgt = exp2f(ml.x - M);
    Lsum = fmaf(ml.y, wgt, Lsum);
#pragma unroll
    for (int i = 0; i < D / 32; ++i) acc[i] = fmaf(a.opart[(slot0 + s) * D + lane + 32 * i], wgt, acc[i]);
  }
  const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
#pragma unroll
  for (int i = 0; i < D / 32; ++i) a.out[orow * D + lane + 32 * i] = __float2bfloat16(acc[i] * inv);
  if (a.lse && lane == 0) a.lse[orow] = Lsum > 0.f ? (M + log2f(Lsum)) * kLn2 : 0.f;
}

template <int D>
int launch(Args a, int B, cudaStream_t s) {
  constexpr int LD = D + 8;
  size_t smem = sizeof(__nv_bfloat16) * (kRowTile + 2 * kKvTile) * LD +
                sizeof(float) * kRowTile * (kKvTile + 1);
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(attn_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return TAPS_ERR_CUDA;
  dim3 grid(a.plan.splits, a.Hkv * a.plan.row_tiles, B);
  attn_chunk_kernel<D><<<grid, kThreads, smem, s>>>(a);
  if (a.plan.splits > 1) {
    const int64_t warps = static_cast<int64_t>(B) * a.Hkv * a.plan.rows_max;
    const int blocks = static_cast<int>((warps * 32 + 255) / 256);
    attn_merge_kernel<D><<<blocks, 256, 0, s>>>(a, B);
  }
  return launch_status();
}

}  // namespace attn
}  // namespace taps

using namespace taps;

extern "C" size_t taps_tree_verify_attn_workspace_bytes(int B, int n_max, int Hq, int Hkv, int D,
                                                        int max_ctx) {
  if (B <= 0 || n_max <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || max_ctx < 0) return 0;
  attn::Plan p = attn::make_plan(B, n_max, Hq, Hkv, max_ctx);
  return attn::ws_layout(p, B, Hkv, D).total;
}

extern "C" int taps_tree_verify_attn(const void* q, const void* k_cache, const void* v_cache,
                                     int64_t num_pages, const int32_t* block_table, int max_pages,
                                     const int32_t* ctx_len, const int32_t* n_nodes,
                                     const uint32_t* mask, int B, int n_max, int Hq, int Hkv,
                                     int D, int page_size, float scale, int max_ctx, void* out,
                                     float* lse_out, void* ws, size_t ws_bytes, int32_t* status,
                                     void* stream) {
  if (!q || !k_cache || !v_cache || !block_table || !ctx_len || !n_nodes || !mask || !out)
    return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || n_max <= 0 || Hq <= 0 || Hkv <= 0 || num_pages <= 0 || max_pages <= 0 ||
      max_ctx < 0 || !(scale > 0.f))
    return TAPS_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return TAPS_ERR_INVALID_ARG;
  if ((D != 64 && D != 128) || page_size != 16 || Hq / Hkv > 8 || n_max > TAPS_MAX_NODES ||
      B > 65535)
    return TAPS_ERR_UNSUPPORTED;
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16))
    return TAPS_ERR_INVALID_ARG;
  attn::Plan p = attn::make_plan(B, n_max, Hq, Hkv, max_ctx);
  attn::WsLayout w = attn::ws_layout(p, B, Hkv, D);
  if (p.splits > 1 && (!ws || ws_bytes < w.total || !aligned(ws, 256))) return TAPS_ERR_WORKSPACE;
  attn::Args a;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.k = static_cast<const __nv_bfloat16*>(k_cache);
  a.v = static_cast<const __nv_bfloat16*>(v_cache);
  a.num_pages = num_pages;
  a.block_table = block_table;
  a.max_pages = max_pages;
  a.ctx_len = ctx_len;
  a.n_nodes = n_nodes;
  a.mask = mask;
  a.n_max = n_max;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.W = (n_max + 31) / 32;
  a.scale_log2 = scale * attn::kLog2e;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.lse = lse_out;
  a.opart = p.splits > 1 ? reinterpret_cast<float*>(static_cast<char*>(ws) + w.opart) : nullptr;
  a.ml = p.splits > 1 ? reinterpret_cast<float2*>(static_cast<char*>(ws) + w.ml) : nullptr;
  a.status = status;
  a.plan = p;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return D == 64 ? attn::launch<64>(a, B, s) : attn::launch<128>(a, B, s);
}
