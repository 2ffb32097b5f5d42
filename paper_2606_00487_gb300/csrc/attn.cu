// Stage 5 of a TAPS round (Sec. 4.1 stage 3): tree attention of the selected
// nodes against the target's paged bf16 KV cache, on the 5th-generation
// tensor cores.
//
// Rows of one KV head are (node, query head of its GQA group) pairs, row
// r = node * group + g, so every K/V tile is read once for the whole group.
// One CTA owns up to 256 rows (two 128-row MMA tiles) of one KV head and one
// chunk of the logical sequence [0, ctx_len + n_nodes). When there are fewer
// (request, KV head, row block) units than SMs, the chunks of one unit form a
// thread-block cluster: each CTA stages its normalised rows and (max, sum) in
// shared memory and, after a cluster barrier, reduces a slice of the rows over
// every CTA of the cluster through distributed shared memory, so no partial
// result ever leaves the chip and no second kernel is needed.
//
// Inside a CTA (10 warps):
//   warp 0   TMA producer (one thread): Q rows once (4D box), then per 64-token
//            tile one contiguous bulk copy per page for K and for V into a
//            3-stage ring; the chunk's page ids are first copied to shared
//            memory by the whole warp. The cache uses the TAPS page layout
//            (see taps_pack_kv_pages): a (page, head) block is stored exactly
//            as the tensor core reads it, 8-token groups of 128-byte swizzled
//            rows, so one copy per page feeds the MMAs directly.
//   warp 1   allocates 512 TMEM columns and issues every tcgen05.mma:
//            S = Q K^T (M=128, N=64, K=D) into a double-buffered S region, then
//            O += P V (M=128, N=D, K=64) into the O region.
//   warps 2-9 softmax, one thread per row (TMEM lane): read S, apply the tree
//            mask, online softmax in base 2 with lazy rescaling (O is rescaled
//            in TMEM only when the running max grows by more than 2^8), write
//            P as bf16 into shared memory for the PV MMA; finally normalise O
//            and stage it (swizzled bf16) in the freed Q buffer, from where a
//            TMA tensor store (one chunk) or the cluster reduction writes it.
// Every wait is bounded; a wait that runs out sets TAPS_DEVFAULT_TIMEOUT and
// the CTA winds down (waiting for its own copies and MMAs) before freeing TMEM.
// Launches use programmatic dependent launch: a grid may start its set-up
// while the previous one drains, and waits before touching its inputs.
#include <algorithm>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "sm100.cuh"

namespace taps {
namespace attn {

using namespace sm100;

constexpr int kRowsPerCta = 256;
constexpr int kTile = 64;          // tokens per K/V tile (four 16-token pages)
constexpr int kStages = 3;
constexpr int kThreadsTc = 320;
constexpr uint32_t kTmemCols = 512;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;
constexpr int kMaxCluster = 16;
constexpr int kMaxTokens = 65536;   // ctx_len + n_max per request (page ids kept in shared memory)

struct Plan {
  int group, rows_max, m_blocks, cs, chunk_len;   // cs = chunks per unit = cluster size
};

// max_active[c]: clusters of c CTAs of this kernel the GPU can hold at once.
inline Plan make_plan(int B, int n_max, int Hq, int Hkv, int max_ctx, const int* max_active) {
  Plan p;
  p.group = Hq / Hkv;
  p.rows_max = n_max * p.group;
  p.m_blocks = (p.rows_max + kRowsPerCta - 1) / kRowsPerCta;
  const int64_t units = static_cast<int64_t>(B) * Hkv * p.m_blocks;
  const int max_total = max_ctx + n_max;
  const int want = static_cast<int>(std::min<int64_t>(kMaxCluster, (kTargetSms + units - 1) / units));
  const int cap = std::max(1, (max_total + 2 * kTile - 1) / (2 * kTile));
  int cs = 1;
  for (int c = 2; c <= std::min(want, cap); ++c)
    if (max_active && units <= max_active[c]) cs = c;
  int chunk = (max_total + cs - 1) / cs;
  chunk = (chunk + 15) / 16 * 16;                  // whole pages
  p.chunk_len = chunk;
  p.cs = (max_total + chunk - 1) / chunk;
  return p;
}

struct Args {
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
  int32_t* status;
  Plan plan;
};

struct Maps {
  CUtensorMap q, out;      // [B][n_max][Hq][D], box 64 x group x 128/group x 1
};

// Shared-memory layout (offsets from a 1024-byte aligned base).
template <int D>
struct Smem {
  static constexpr int kChunks = D / 64;                      // 64-dim (128-byte) halves
  static constexpr uint32_t kQ = 0;                           // [2 mt][chunks][128 rows][128 B]
  static constexpr uint32_t kQBytes = 2 * kChunks * 16384;
  static constexpr uint32_t kKV = kQBytes;                    // [stage][K 4 pages | V 4 pages], TAPS page layout
  static constexpr uint32_t kKVStage = 2 * kChunks * 8192;
  static constexpr uint32_t kPageBytes = 16 * D * 2;          // one (page, head) block
  static constexpr uint32_t kGroupStride = kChunks * 1024;    // 8-token groups in a block
  static constexpr uint32_t kP = kKV + kStages * kKVStage;    // [2 mt][128 rows][128 B]
  static constexpr uint32_t kBar = kP + 2 * 16384;
  static constexpr int kNumBars = 2 * kStages + 6;
  static constexpr uint32_t kColMask = kBar + 8 * kNumBars;
  static constexpr uint32_t kTmemSlot = kColMask + 8 * kStages;
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kMl = (kAbort + 4 + 7) / 8 * 8;   // [256] (max, sum) of the rows
  static constexpr uint32_t kPages = kMl + 8 * kRowsPerCta;   // page ids of this CTA's chunk
  static constexpr int kMaxChunkPages = kMaxTokens / 16;
  static constexpr uint32_t kBytes = kPages + 4 * kMaxChunkPages;
  static constexpr uint32_t kAlloc = kBytes + 1024;           // slack for the 1024-byte alignment
};

__device__ __forceinline__ void set_fault(volatile int* abort_flag, int32_t* status, int bit) {
  *abort_flag = 1;
  if (status) atomicOr(status, bit);
}

template <int D>
__global__ void __launch_bounds__(kThreadsTc, 1)
attn_tc_kernel(const __grid_constant__ Maps maps, const Args a) {
  using S = Smem<D>;
  constexpr int CH = S::kChunks;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* kv_full = bars;
  uint64_t* kv_empty = bars + kStages;
  uint64_t* s_full = bars + 2 * kStages;
  uint64_t* p_full = s_full + 2;
  uint64_t* pv_done = p_full + 1;
  uint64_t* q_full = pv_done + 1;
  uint64_t* drain = q_full + 1;
  uint64_t* colmask = reinterpret_cast<uint64_t*>(smem + S::kColMask);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + S::kAbort);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- set-up that reads no input: may overlap the previous grid's tail
  if (threadIdx.x == 0) prefetch_tensormap(&maps.q);
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  pdl_wait();

  const Plan& pl = a.plan;
  const int b = blockIdx.z;
  const int kv = blockIdx.y / pl.m_blocks;
  const int mb = blockIdx.y % pl.m_blocks;
  const int split = blockIdx.x;
  const int n = min(max(a.n_nodes[b], 0), a.n_max);
  const int C = a.ctx_len[b];
  const int total = C + n;
  const int rows = n * pl.group;
  const int row0 = mb * kRowsPerCta;
  const int m_tiles = max(0, min(2, (rows - row0 + 127) / 128));
  const int pos0 = split * pl.chunk_len;
  const int pos1 = min(pos0 + pl.chunk_len, total);
  const int n_tiles = pos1 > pos0 ? (pos1 - pos0 + kTile - 1) / kTile : 0;
  const bool single = pl.cs == 1;

  if (m_tiles == 0) {
    // no row of this block is live (the same for every CTA of a cluster): the
    // first chunk writes the block's padding rows as zeros
    if (split == 0) {
      for (int e = threadIdx.x; e < kRowsPerCta * (D / 8); e += kThreadsTc) {
        int r = row0 + e / (D / 8);
        if (r < pl.rows_max) {
          int i = r / pl.group, h = kv * pl.group + r % pl.group;
          int64_t orow = (static_cast<int64_t>(b) * a.n_max + i) * a.Hq + h;
          reinterpret_cast<uint4*>(a.out + orow * D)[e % (D / 8)] = make_uint4(0, 0, 0, 0);
          if (a.lse && e % (D / 8) == 0) a.lse[orow] = 0.f;
        }
      }
    }
    pdl_launch_dependents();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(*tmem_slot, kTmemCols);
    }
    return;
  }

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    mbar_init(&s_full[0], 1);
    mbar_init(&s_full[1], 1);
    mbar_init(p_full, 128 * m_tiles);
    mbar_init(pv_done, 1);
    mbar_init(q_full, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // TMEM columns: O of M-tile mt at mt * D; S of buffer u, M-tile mt at 256 + u*128 + mt*64
  auto o_col = [](int mt) { return static_cast<uint32_t>(mt * D); };
  auto s_col = [](int u, int mt) { return static_cast<uint32_t>(256 + u * 128 + mt * 64); };

  if (n_tiles == 0) {
    // this chunk is empty for this request: nothing to compute, the epilogue
    // below contributes zero rows with an empty softmax
  } else if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    // page ids of the whole chunk -> shared memory (whole warp, coalesced);
    // -1 marks a logical page missing from the block table
    int32_t* spages = reinterpret_cast<int32_t*>(smem + S::kPages);
    const int32_t* bt = a.block_table + static_cast<int64_t>(b) * a.max_pages;
    const int lp0 = pos0 >> 4;
    const int npg = (pos1 - pos0 + 15) >> 4;
    for (int i = lane; i < npg; i += 32) spages[i] = lp0 + i < a.max_pages ? bt[lp0 + i] : -1;
    __syncwarp();
    if (lane == 0) {
      const uint64_t policy = l2_evict_first_policy();
      int issued = 0;
      for (int j = 0; j < n_tiles; ++j) {
        if (*abort_flag) break;
        const int s = j % kStages;
        if (j >= kStages && !mbar_wait(&kv_empty[s], ((j / kStages) - 1) & 1)) {
          set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          break;
        }
        const int t0 = pos0 + j * kTile;
        int pages[4];
        uint64_t cm = 0;
        uint32_t bytes = 0;
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          pages[p] = -1;
          const int tp = t0 + 16 * p;
          if (tp >= pos1) continue;
          const int pg = spages[j * 4 + p];
          if (pg < 0 || pg >= a.num_pages) {
            if (a.status) atomicOr(a.status, TAPS_DEVFAULT_PAGE);
            continue;
          }
          pages[p] = pg;
          bytes += 2 * CH * 2048;
          const int nv = min(16, pos1 - tp);
          cm |= (nv == 16 ? 0xFFFFull : ((1ull << nv) - 1)) << (16 * p);
        }
        colmask[s] = cm;
        mbar_arrive_expect_tx(&kv_full[s], bytes);
        const uint32_t kbase = sb + S::kKV + s * S::kKVStage;
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          if (pages[p] < 0) continue;
          const int64_t blk = (static_cast<int64_t>(pages[p]) * a.Hkv + kv) * (16 * D);
          bulk_load(kbase + p * S::kPageBytes, a.k + blk, S::kPageBytes, &kv_full[s], policy);
          bulk_load(kbase + 4 * S::kPageBytes + p * S::kPageBytes, a.v + blk, S::kPageBytes,
                    &kv_full[s], policy);
        }
        if (j == 0) {
          // Q rows of this block (issued after the first K/V tile, which comes
          // from DRAM): one box of (64 dims, group heads, 128/group nodes) per
          // M-tile and 64-dim half; nodes past n_max read as zeros
          mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(m_tiles * CH * 16384));
          for (int mt = 0; mt < m_tiles; ++mt)
            for (int c = 0; c < CH; ++c)
              tma_load_4d(sb + S::kQ + (mt * CH + c) * 16384, &maps.q, q_full, c * 64,
                          kv * pl.group, (row0 + mt * 128) / pl.group, b);
        }
        issued = j + 1;
      }
      // never leave the CTA with copies in flight
      if (issued > 0) mbar_wait(q_full, 0);
      for (int j = max(0, issued - kStages); j < issued; ++j)
        mbar_wait(&kv_full[j % kStages], (j / kStages) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_qk = idesc_bf16_f32(128, kTile, false, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, false, true);
    bool ok = __all_sync(kFullMask, mbar_wait(q_full, 0));
    if (!ok && lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
    for (int j = 0; ok && j <= n_tiles; ++j) {
      if (__any_sync(kFullMask, *abort_flag != 0)) break;
      if (j < n_tiles) {
        const int s = j % kStages;
        if (!__all_sync(kFullMask, mbar_wait(&kv_full[s], (j / kStages) & 1))) {
          if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          break;
        }
        const uint64_t cm = colmask[s];
        if (cm != ~0ull) {
          // rows of skipped or out-of-chunk positions: zero V so that P = 0
          // never meets stale (possibly non-finite) data
          uint8_t* vb = smem + S::kKV + s * S::kKVStage + 4 * S::kPageBytes;
          for (int e = lane; e < kTile * 8 * CH; e += 32) {
            const int t = e / (8 * CH), c = (e / 8) % CH, q16 = e % 8;
            const int p = t >> 4, w = t & 15;
            if (!((cm >> t) & 1ull))
              *reinterpret_cast<uint4*>(vb + p * S::kPageBytes + (w >> 3) * S::kGroupStride +
                                        c * 1024 + (w & 7) * 128 + q16 * 16) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) {
          tc_fence_after();
          const uint32_t kb = sb + S::kKV + s * S::kKVStage;
          for (int mt = 0; mt < m_tiles; ++mt) {
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
              const uint64_t ad =
                  sw128_desc(sb + S::kQ + (mt * CH + ks / 4) * 16384 + (ks % 4) * 32, 16, 1024);
              const uint64_t bd =
                  sw128_desc(kb + (ks / 4) * 1024 + (ks % 4) * 32, 16, S::kGroupStride);
              mma_bf16(tmem + s_col(j & 1, mt), ad, bd, idesc_qk, ks > 0 ? 1u : 0u);
            }
          }
          mma_commit(&s_full[j & 1]);
        }
        __syncwarp();
      }
      if (j >= 1) {
        const int jp = j - 1, sp = jp % kStages;
        if (!__all_sync(kFullMask, mbar_wait(p_full, jp & 1))) {
          if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          break;
        }
        if (lane == 0) {
          tc_fence_after();
          const uint32_t vb = sb + S::kKV + sp * S::kKVStage + 4 * S::kPageBytes;
          for (int mt = 0; mt < m_tiles; ++mt) {
#pragma unroll
            for (int ks = 0; ks < kTile / 16; ++ks) {
              const uint64_t ad = sw128_desc(sb + S::kP + mt * 16384 + ks * 32, 16, 1024);
              const uint64_t bd = sw128_desc(vb + ks * S::kPageBytes, 1024, S::kGroupStride);
              mma_bf16(tmem + o_col(mt), ad, bd, idesc_pv, (jp > 0 || ks > 0) ? 1u : 0u);
            }
          }
          mma_commit(pv_done);
          mma_commit(&kv_empty[sp]);
        }
        __syncwarp();
      }
    }
    // every MMA issued by this warp completes before TMEM is released
    if (lane == 0) mma_commit(drain);
    __syncwarp();
    mbar_wait(drain, 0);
  }
  if (warp >= 2) {
    // ------------------------------------------------------------ softmax warps
    const int sw = warp - 2;
    const int mt = sw >> 2;
    const int quarter = warp & 3;                  // TMEM lanes 32*quarter .. +31
    const int r = quarter * 32 + lane;             // row within the M-tile
    const int grow = row0 + mt * 128 + r;
    const bool live = mt < m_tiles;
    const bool valid_row = live && grow < rows;
    const int node = valid_row ? grow / pl.group : 0;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const float scale = a.scale_log2;
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    const bool has_o = live && n_tiles > 0;
    if (has_o) {
      const uint32_t* mrow = a.mask + (static_cast<int64_t>(b) * a.n_max + node) * a.W;
      uint8_t* prow = smem + S::kP + mt * 16384 + r * 128;
      for (int j = 0; j < n_tiles; ++j) {
        if (__any_sync(kFullMask, *abort_flag != 0)) { ok = false; break; }
        const int s = j % kStages;
        // kv_full of this tile completed before its QK MMA: this wait returns at
        // once and makes the producer's column mask visible
        if (!__all_sync(kFullMask, mbar_wait(&s_full[j & 1], (j >> 1) & 1) &&
                                        mbar_wait(&kv_full[s], (j / kStages) & 1))) {
          if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          ok = false;
          break;
        }
        const uint64_t cm = colmask[s];
        tc_fence_after();
        uint32_t sv[64];
        tmem_ld64_sync(lane_base + s_col(j & 1, mt), sv);
        const int t0 = pos0 + j * kTile;
        uint64_t vis = valid_row ? cm : 0ull;
        if (valid_row && t0 + kTile > C) {
          // columns from i0 on are tree nodes jn = t0 + i - C: take a 64-bit
          // window of this row's ancestor mask starting at node jn0
          const int i0 = max(0, C - t0);
          const int jn0 = t0 + i0 - C;
          const int q = jn0 >> 5, o = jn0 & 31;
          const uint32_t w0 = q < a.W ? mrow[q] : 0u;
          const uint32_t w1 = q + 1 < a.W ? mrow[q + 1] : 0u;
          const uint32_t w2 = q + 2 < a.W ? mrow[q + 2] : 0u;
          const uint64_t lo = (static_cast<uint64_t>(w1) << 32) | w0;
          const uint64_t win = o == 0 ? lo : ((lo >> o) | (static_cast<uint64_t>(w2) << (64 - o)));
          const uint64_t ctx_cols = i0 == 0 ? 0ull : ((1ull << i0) - 1);
          vis &= ctx_cols | (win << i0);
        }
        if (vis != ~0ull) {
#pragma unroll
          for (int i = 0; i < 64; ++i)
            if (!((vis >> i) & 1ull)) sv[i] = 0xFF800000u;   // -inf
        }
        float mx[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) mx[k] = __uint_as_float(sv[k]);
#pragma unroll
        for (int i = 8; i < 64; ++i) mx[i & 7] = fmaxf(mx[i & 7], __uint_as_float(sv[i]));
        const float tmax =
            fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                  fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7]))) * scale;
        const float m_new = fmaxf(m_used, tmax);
        const bool grow_max =
            (m_used == -INFINITY) ? (m_new > -INFINITY) : (m_new > m_used + kRescaleThreshold);
        float alpha = 1.f;
        if (grow_max) {
          alpha = (m_used == -INFINITY) ? 0.f : ex2_approx(m_used - m_new);
          m_used = m_new;
        }
        uint32_t pk[32];
        float acc[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] = 0.f;
        if (m_used != -INFINITY) {
          const float nm = -m_used;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float p0 = ex2_approx(fmaf(__uint_as_float(sv[2 * i]), scale, nm));
            const float p1 = ex2_approx(fmaf(__uint_as_float(sv[2 * i + 1]), scale, nm));
            pk[i] = pack_bf16x2(p0, p1);
            acc[i & 7] += p0 + p1;
          }
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) pk[i] = 0u;
        }
        const float psum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) +
                           ((acc[4] + acc[5]) + (acc[6] + acc[7]));
        l = l * alpha + psum;
        // PV of the previous tile must be done before P is overwritten and O touched
        if (j > 0 && !__all_sync(kFullMask, mbar_wait(pv_done, (j - 1) & 1))) {
          if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          ok = false;
          break;
        }
        const bool need_rescale = grow_max && j > 0 && alpha != 1.f;
        if (__any_sync(kFullMask, need_rescale)) {
          tc_fence_after();
          const float f = need_rescale ? alpha : 1.f;
#pragma unroll 1
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            tmem_ld32_sync(lane_base + o_col(mt) + c * 32, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
            tmem_st32(lane_base + o_col(mt) + c * 32, o);
          }
          tmem_wait_st();
        }
#pragma unroll
        for (int j8 = 0; j8 < 8; ++j8)
          *reinterpret_cast<uint4*>(prow + ((j8 ^ (r & 7)) << 4)) =
              make_uint4(pk[4 * j8], pk[4 * j8 + 1], pk[4 * j8 + 2], pk[4 * j8 + 3]);
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(p_full);
      }
      if (ok && !__all_sync(kFullMask, mbar_wait(pv_done, (n_tiles - 1) & 1))) {
        if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
        ok = false;
      }
    }
    if (threadIdx.x == 64) pdl_launch_dependents();
    // ---- epilogue. Once a live warp's last PV is done every MMA has finished,
    // so the Q buffer is free: stage the normalised bf16 rows there in the
    // same swizzled layout, and this row's (max, sum) next to them.
    const bool good = ok && valid_row && l > 0.f;
    const float inv = good ? 1.f / l : 0.f;
    uint8_t* srow = smem + S::kQ + (mt * CH) * 16384 + r * 128;
    if (has_o) {
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < D / 64; ++c) {
        uint32_t o[64];
        tmem_ld64_sync(lane_base + o_col(mt) + c * 64, o);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int j16 = c * 8 + k;                      // 16-byte chunk of the row
          *reinterpret_cast<uint4*>(srow + (j16 >> 3) * 16384 + (((j16 & 7) ^ (r & 7)) << 4)) =
              make_uint4(
                  pack_bf16x2(__uint_as_float(o[8 * k + 0]) * inv, __uint_as_float(o[8 * k + 1]) * inv),
                  pack_bf16x2(__uint_as_float(o[8 * k + 2]) * inv, __uint_as_float(o[8 * k + 3]) * inv),
                  pack_bf16x2(__uint_as_float(o[8 * k + 4]) * inv, __uint_as_float(o[8 * k + 5]) * inv),
                  pack_bf16x2(__uint_as_float(o[8 * k + 6]) * inv, __uint_as_float(o[8 * k + 7]) * inv));
        }
      }
    } else {
#pragma unroll
      for (int j16 = 0; j16 < D / 8; ++j16)
        *reinterpret_cast<uint4*>(srow + (j16 >> 3) * 16384 + (((j16 & 7) ^ (r & 7)) << 4)) =
            make_uint4(0, 0, 0, 0);
    }
    reinterpret_cast<float2*>(smem + S::kMl)[mt * 128 + r] =
        good ? make_float2(m_used, l) : make_float2(-INFINITY, 0.f);
    if (single) {
      if (a.lse && grow < pl.rows_max) {
        const int64_t orow = (static_cast<int64_t>(b) * a.n_max + grow / pl.group) * a.Hq +
                             kv * pl.group + grow % pl.group;
        a.lse[orow] = good ? (m_used + log2f(l)) * kLn2 : 0.f;
      }
      fence_proxy_async_smem();
      named_bar_sync(1, 256);
      if (threadIdx.x == 64) {
        for (int t = 0; t < 2; ++t) {
          if (row0 + t * 128 >= pl.rows_max) break;
          for (int c = 0; c < CH; ++c)
            tma_store_4d(&maps.out, sb + S::kQ + (t * CH + c) * 16384, c * 64, kv * pl.group,
                         (row0 + t * 128) / pl.group, b);
        }
        bulk_commit();
        bulk_wait_read_all();
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  if (single) {
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tmem, kTmemCols);
    }
    return;
  }
  // ---- cluster reduction: CTA `rank` owns a slice of the block's rows and
  // combines them over every CTA (chunk) of the cluster, reading the peers'
  // staged rows and (max, sum) through distributed shared memory.
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (warp >= 2) {
    constexpr int DPL = D / 32;                        // dims per lane
    const int cs = pl.cs;
    const uint32_t rank = cluster_ctarank();
    const int per = (kRowsPerCta + cs - 1) / cs;
    const int rb = static_cast<int>(rank) * per;
    const int re = min(kRowsPerCta, rb + per);
    const int boff = lane * DPL * 2;                   // this lane's bytes of a row
    const int j16 = boff >> 4;
    for (int rr = rb + (warp - 2); rr < re; rr += 8) {
      const int gr = row0 + rr;
      if (gr >= pl.rows_max) break;
      float2 mlv = make_float2(-INFINITY, 0.f);
      if (lane < cs) {
        const uint2 t = ld_cluster_v2(mapa_shared(sb + S::kMl + rr * 8, lane));
        mlv = make_float2(__uint_as_float(t.x), __uint_as_float(t.y));
      }
      float M = mlv.x;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(kFullMask, M, off));
      const float w = mlv.y > 0.f ? mlv.y * ex2_approx(mlv.x - M) : 0.f;
      float Lsum = w;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) Lsum += __shfl_xor_sync(kFullMask, Lsum, off);
      const int rmt = rr >> 7, rrow = rr & 127;
      const uint32_t laddr = sb + S::kQ + (rmt * CH + (j16 >> 3)) * 16384 + rrow * 128 +
                             (((j16 & 7) ^ (rrow & 7)) << 4) + (boff & 15);
      uint32_t v[kMaxCluster][DPL / 2];
#pragma unroll
      for (int q = 0; q < kMaxCluster; ++q) {
        if (q < cs) {
          const uint32_t ra = mapa_shared(laddr, q);
          if (DPL == 4) {
            const uint2 t = ld_cluster_v2(ra);
            v[q][0] = t.x;
            v[q][DPL / 2 - 1] = t.y;
          } else {
            v[q][0] = ld_cluster_u32(ra);
          }
        }
      }
      float acc[DPL];
#pragma unroll
      for (int i = 0; i < DPL; ++i) acc[i] = 0.f;
#pragma unroll
      for (int q = 0; q < kMaxCluster; ++q) {
        const float wq = __shfl_sync(kFullMask, w, q);
        if (q < cs) {
#pragma unroll
          for (int i = 0; i < DPL / 2; ++i) {
            acc[2 * i] = fmaf(wq, __uint_as_float(v[q][i] << 16), acc[2 * i]);
            acc[2 * i + 1] = fmaf(wq, __uint_as_float(v[q][i] & 0xFFFF0000u), acc[2 * i + 1]);
          }
        }
      }
      const bool row_ok = gr < rows && Lsum > 0.f;
      const float linv = row_ok ? 1.f / Lsum : 0.f;
      const int64_t orow = (static_cast<int64_t>(b) * a.n_max + gr / pl.group) * a.Hq +
                           kv * pl.group + gr % pl.group;
      __nv_bfloat16* dst = a.out + orow * D + lane * DPL;
      if (DPL == 4) {
        uint2 o;
        o.x = pack_bf16x2(acc[0] * linv, acc[1] * linv);
        o.y = pack_bf16x2(acc[2] * linv, acc[DPL - 1] * linv);
        *reinterpret_cast<uint2*>(dst) = o;
      } else {
        *reinterpret_cast<uint32_t*>(dst) = pack_bf16x2(acc[0] * linv, acc[1] * linv);
      }
      if (a.lse && lane == 0) a.lse[orow] = row_ok ? (M + log2f(Lsum)) * kLn2 : 0.f;
    }
  }
  // the peers may still be reading this CTA's shared memory
  __syncwarp();
  cluster_sync();
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

bool encode(CUtensorMap* map, const void* base, int rank, const cuuint64_t* dims,
            const cuuint64_t* strides, const cuuint32_t* box) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Clusters of c CTAs of attn_tc_kernel<D> the current device can hold at once,
// c = 0..16 (entry 0 unused); queried once per device.
template <int D>
const int* cluster_capacity() {
  static std::mutex mu;
  static int table[64][kMaxCluster + 1];
  static bool done[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    const int smem = static_cast<int>(Smem<D>::kAlloc);
    if (cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem) != cudaSuccess ||
        cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeNonPortableClusterSizeAllowed,
                             1) != cudaSuccess)
      return nullptr;
    for (int c = 0; c <= kMaxCluster; ++c) {
      table[dev][c] = 0;
      if (c == 0) continue;
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(c, 1, 1);
      cfg.blockDim = dim3(kThreadsTc);
      cfg.dynamicSmemBytes = smem;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = c;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel<D>, &cfg) == cudaSuccess)
        table[dev][c] = n;
    }
    cudaGetLastError();
    done[dev] = true;
  }
  return table[dev];
}

template <int D>
int launch(const void* q, const void* k, const void* v, Args a, int B, cudaStream_t s) {
  const Plan& p = a.plan;
  Maps m;
  // queries / outputs [B][n_max][Hq][D]; the box covers one GQA group for
  // 128/group consecutive nodes of one request
  const cuuint64_t qd[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(a.Hq),
                            static_cast<cuuint64_t>(a.n_max), static_cast<cuuint64_t>(B)};
  const cuuint64_t qs[3] = {static_cast<cuuint64_t>(D) * 2,
                            static_cast<cuuint64_t>(a.Hq) * D * 2,
                            static_cast<cuuint64_t>(a.n_max) * a.Hq * D * 2};
  const cuuint32_t qb[4] = {64, static_cast<cuuint32_t>(p.group),
                            static_cast<cuuint32_t>(128 / p.group), 1};
  if (!encode(&m.q, q, 4, qd, qs, qb) || !encode(&m.out, a.out, 4, qd, qs, qb))
    return TAPS_ERR_CUDA;
  a.k = static_cast<const __nv_bfloat16*>(k);
  a.v = static_cast<const __nv_bfloat16*>(v);
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = p.cs;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.cs, a.Hkv * p.m_blocks, B);
  cfg.blockDim = dim3(kThreadsTc);
  cfg.dynamicSmemBytes = Smem<D>::kAlloc;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = p.cs > 1 ? 2 : 1;
  if (cudaLaunchKernelEx(&cfg, attn_tc_kernel<D>, m, a) != cudaSuccess) return TAPS_ERR_CUDA;
  return launch_status();
}

}  // namespace attn
}  // namespace taps

using namespace taps;

extern "C" size_t taps_tree_verify_attn_workspace_bytes(int B, int n_max, int Hq, int Hkv, int D,
                                                        int max_ctx) {
  // chunks of one unit are reduced on chip (cluster shared memory): no workspace
  (void)B, (void)n_max, (void)Hq, (void)Hkv, (void)D, (void)max_ctx;
  return 0;
}

extern "C" int taps_tree_verify_attn(const void* q, const void* k_cache, const void* v_cache,
                                     int64_t num_pages, const int32_t* block_table, int max_pages,
                                     const int32_t* ctx_len, const int32_t* n_nodes,
                                     const uint32_t* mask, int B, int n_max, int Hq, int Hkv,
                                     int D, int page_size, float scale, int max_ctx, void* out,
                                     float* lse_out, void* ws, size_t ws_bytes, int32_t* status,
                                     void* stream) {
  (void)ws, (void)ws_bytes;
  if (!q || !k_cache || !v_cache || !block_table || !ctx_len || !n_nodes || !mask || !out)
    return TAPS_ERR_INVALID_ARG;
  if (B <= 0 || n_max <= 0 || Hq <= 0 || Hkv <= 0 || num_pages <= 0 || max_pages <= 0 ||
      max_ctx < 0 || !(scale > 0.f))
    return TAPS_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return TAPS_ERR_INVALID_ARG;
  const int group = Hq / Hkv;
  if ((D != 64 && D != 128) || page_size != 16 ||
      (group != 1 && group != 2 && group != 4 && group != 8) || n_max > TAPS_MAX_NODES ||
      B > 65535 || num_pages * Hkv * 16 > 0x7fffffffLL ||
      static_cast<int64_t>(max_ctx) + n_max > attn::kMaxTokens)
    return TAPS_ERR_UNSUPPORTED;
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16))
    return TAPS_ERR_INVALID_ARG;
  const int* cap = D == 64 ? attn::cluster_capacity<64>() : attn::cluster_capacity<128>();
  if (!cap) return TAPS_ERR_CUDA;
  attn::Args a;
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
  a.status = status;
  a.plan = attn::make_plan(B, n_max, Hq, Hkv, max_ctx, cap);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return D == 64 ? attn::launch<64>(q, k_cache, v_cache, a, B, s)
                 : attn::launch<128>(q, k_cache, v_cache, a, B, s);
}
