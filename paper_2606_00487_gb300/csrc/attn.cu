// Stage 5 of a TAPS round (Sec. 4.1 stage 3): tree attention of the selected
// nodes against the target's paged bf16 KV cache, on the 5th-generation
// tensor cores.
//
// Rows of one KV head are (node, query head of its GQA group) pairs, row
// r = node * group + g, so every K/V tile is read once for the whole group.
// One CTA owns 128 rows (one MMA tile) of one KV head and one chunk of the
// logical sequence [0, ctx_len + n_nodes). When there are fewer (request, KV
// head, row block) units than SMs, the chunks of one unit form a thread-block
// cluster: each CTA stages its normalised rows and (max, sum) in shared
// memory and, after a cluster barrier, reduces a slice of the rows over every
// CTA of the cluster through distributed shared memory, so no partial result
// ever leaves the chip and no second kernel is needed.
//
// Inside a CTA (8 warps):
//   warps 0, 2  producers: warp 0 streams the K tiles, warp 2 the V tiles,
//            each into a 2-stage ring, one bulk copy per 16-token page of a
//            128-token tile (lane p copies page p). The cache uses the TAPS
//            page layout (see taps_pack_kv_pages): a (page, head) block is
//            stored exactly as the tensor core reads it, 8-token groups of
//            128-byte swizzled rows, so one copy per page feeds the MMAs.
//   warp 3   copies the chunk's page ids to shared memory, then loads Q (4D
//            tensor-map boxes).
//   warp 1   allocates all 512 TMEM columns and issues every tcgen05.mma.
//            S = Q K^T (M=128, N=128, K=D) goes to one of three S buffers;
//            O += P V (M=128, N=D, K=16 per page) reads P from TMEM. After
//            the softmax of tile j, one burst issues the PV of tile j and the
//            QK of tile j+2 alternately, so consecutive MMAs never chain on
//            one accumulator, while the softmax of tile j+1 already runs.
//   warps 4-7 softmax, one thread per row (TMEM lane): read S, apply the
//            tree mask, online softmax in base 2 with lazy rescaling (O is
//            rescaled in TMEM only when the running max grows by more than
//            2^8), and write P as bf16 over the S columns it came from;
//            finally normalise O and stage it (swizzled bf16) in the freed Q
//            buffer, from where a TMA tensor store (one chunk) or the cluster
//            reduction writes it.
// TMEM columns: O at [0, D), S (fp32) and then P (bf16 pairs) of buffer u at
// [128 + 128 u, 256 + 128 u), u = 0, 1, 2; tile j uses buffer j mod 3.
// With 2 to 32 requests in a launch, block rows take the requests longest
// first, so that long requests do not start in the last wave.
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

constexpr int kRowsPerCta = 128;
constexpr int kTile = 128;             // tokens per K/V tile
constexpr int kTilePages = kTile / 16;  // 16-token pages per tile
constexpr int kKStages = 2;            // K tiles in flight (released after QK)
constexpr int kVStages = 2;            // V tiles in flight (released after PV)
constexpr int kSBufs = 3;              // S / P buffers in TMEM
constexpr int kThreadsTc = 256;
constexpr uint32_t kTmemCols = 512;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;
constexpr int kMaxCluster = 16;
constexpr int kMaxTokens = 65536;   // ctx_len + n_max per request
constexpr int kMaxChunkTokens = 32768;   // page ids of one chunk are kept in shared memory

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
  const int cap = std::max(1, (max_total + kTile - 1) / kTile);
  int cs = 1;
  for (int c = 2; c <= std::min(want, cap); ++c)
    if (max_active && units <= max_active[c]) cs = c;
  cs = std::max(cs, (max_total + kMaxChunkTokens - 1) / kMaxChunkTokens);
  int chunk = (max_total + cs - 1) / cs;
  // whole tiles where the chunk spans more than one, else whole pages: only
  // the chunk holding the end of the sequence then ends inside a tile
  chunk = chunk > kTile ? (chunk + kTile - 1) / kTile * kTile : (chunk + 15) / 16 * 16;
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
  static constexpr uint32_t kPageBytes = 16 * D * 2;          // one (page, head) block
  static constexpr uint32_t kGroupStride = kChunks * 1024;    // 8-token groups in a block
  static constexpr uint32_t kTileBytes = kTilePages * kPageBytes;   // one K or V tile
  static constexpr uint32_t kQ = 0;                           // [chunks][128 rows][128 B]
  static constexpr uint32_t kQBytes = kChunks * 16384;
  static constexpr uint32_t kK = kQBytes;                     // K ring, TAPS page layout
  static constexpr uint32_t kV = kK + kKStages * kTileBytes;  // V ring
  // the peers' partial rows of this CTA's slice (cluster launches):
  // [peer][64-dim half][slice row][128 B], then [peer][slice row] (max, sum);
  // peers x slice rows <= 150 for every cluster size
  static constexpr uint32_t kRecv = kV + kVStages * kTileBytes;
  static constexpr uint32_t kRecvBytes = (152 * (2 * D + 8) + 1023) / 1024 * 1024;
  static constexpr uint32_t kBar = kRecv + kRecvBytes;
  static constexpr int kNumBars = kKStages + 2 * kVStages + 2 * kSBufs + 4;
  static constexpr uint32_t kTmemSlot = kBar + 8 * kNumBars;
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kMl = (kAbort + 4 + 15) / 16 * 16;   // [128] (max, sum) of the rows
  static constexpr uint32_t kStat = kMl + 8 * kRowsPerCta;     // [slice row] (max, sum), cluster-wide
  static constexpr uint32_t kPages = kStat + 8 * kRowsPerCta;  // page ids of this CTA's chunk
  static constexpr int kMaxChunkPages = kMaxChunkTokens / 16;
  static constexpr uint32_t kBytes = kPages + 4 * kMaxChunkPages;
  // at least half of the SM's shared memory, so that two CTAs (which would
  // contend for the 512 TMEM columns) never share an SM
  static constexpr uint32_t kAlloc = std::max<uint32_t>(kBytes + 1024, 120 * 1024);
};

__device__ __forceinline__ void set_fault(volatile int* abort_flag, int32_t* status, int bit) {
  *abort_flag = 1;
  if (status) atomicOr(status, bit);
}

// 64 columns of a row's ancestor mask starting at tree node jn0 (>= 0), from
// the row's W 32-bit words; nodes past the last word are not visible.
__device__ __forceinline__ uint64_t mask_window(const uint32_t* mrow, int W, int jn0) {
  const int q = jn0 >> 5, o = jn0 & 31;
  const uint32_t w0 = q < W ? mrow[q] : 0u;
  const uint32_t w1 = q + 1 < W ? mrow[q + 1] : 0u;
  const uint32_t w2 = q + 2 < W ? mrow[q + 2] : 0u;
  const uint64_t lo = (static_cast<uint64_t>(w1) << 32) | w0;
  return o == 0 ? lo : ((lo >> o) | (static_cast<uint64_t>(w2) << (64 - o)));
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
  uint64_t* k_full = bars;
  uint64_t* v_full = k_full + kKStages;
  // [kVStages] the burst holding PV of a tile done: V slot free, and O holds
  // that tile's product (the softmax waits on it before rescaling O)
  uint64_t* v_empty = v_full + kVStages;
  // [kSBufs] QK of a tile done: S written, and its K slot free (the K
  // producer waits on it too)
  uint64_t* s_full = v_empty + kVStages;
  // [kSBufs] P of a tile written (4 warps arrive). One per buffer: the
  // softmax may finish tile j+1 before the MMA warp has waited for tile j,
  // and a single barrier would then complete two phases in a row
  uint64_t* p_full = s_full + kSBufs;
  uint64_t* o_full = p_full + kSBufs;      // last PV done
  uint64_t* q_full = o_full + 1;
  uint64_t* drain = q_full + 1;
  uint64_t* recv = drain + 1;              // the peers' partial rows of this CTA's slice landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + S::kAbort);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- set-up that reads no input: may overlap the previous grid's tail
  const Plan& pl = a.plan;
  const int kv = blockIdx.y / pl.m_blocks;
  const int mb = blockIdx.y % pl.m_blocks;
  const int split = blockIdx.x;
  const int row0 = mb * kRowsPerCta;
  const int pos0 = split * pl.chunk_len;
  const bool single = pl.cs == 1;
  // cluster exchange geometry: CTA `rank` combines rows [rb, re) of the block
  const int cs = pl.cs;
  const uint32_t rank = single ? 0u : cluster_ctarank();
  const int per = ((kRowsPerCta + cs - 1) / cs + 1) & ~1;   // even: 16-byte (max, sum) pieces
  const int rb = min(kRowsPerCta, static_cast<int>(rank) * per);
  const int re = min(kRowsPerCta, rb + per);
  if (threadIdx.x == 0) {
    prefetch_tensormap(&maps.q);
    for (int s = 0; s < kKStages; ++s) mbar_init(&k_full[s], 1);
    for (int s = 0; s < kVStages; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int u = 0; u < kSBufs; ++u) {
      mbar_init(&s_full[u], 1);
      mbar_init(&p_full[u], 4);
    }
    mbar_init(o_full, 1);
    mbar_init(q_full, 1);
    mbar_init(drain, 1);
    mbar_init(recv, 1);
    *abort_flag = 0;
    fence_mbar_init();
    if (!single) mbar_arrive_expect_tx(recv, static_cast<uint32_t>(cs * (re - rb) * (2 * D + 8)));
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  __syncthreads();   // barriers initialised
  pdl_wait();

  // Requests longest first: blocks start in launch order, the request index
  // (z) slowest, so with 2 to 32 requests block row z takes the request of
  // z-th largest length (ctx_len + n_nodes, ties by index) and the long ones
  // do not end up in the last wave. Every warp ranks the lengths itself.
  int b = blockIdx.z;
  if (gridDim.z > 1 && gridDim.z <= 32) {
    const int B = static_cast<int>(gridDim.z);
    const int len = lane < B ? a.ctx_len[lane] + min(max(a.n_nodes[lane], 0), a.n_max) : -1;
    int rank = 0;
    for (int j = 0; j < B; ++j) {
      const int lj = __shfl_sync(kFullMask, len, j);
      rank += (lj > len || (lj == len && j < lane)) ? 1 : 0;
    }
    b = __ffs(__ballot_sync(kFullMask, lane < B && rank == static_cast<int>(blockIdx.z))) - 1;
  }

  // ---- inputs. The request's lengths and the chunk's page ids are
  // requested together; then Q and each producer's first tile leave at once,
  // before the CTA-wide barrier.
  // page ids of the chunk -> shared memory (warp 3, coalesced; -1 marks a
  // logical page missing from the block table); lane p of the producer warps
  // 0 and 2 reads the id of page p of the first tile for itself
  int32_t* spages = reinterpret_cast<int32_t*>(smem + S::kPages);
  const int32_t* bt = a.block_table + static_cast<int64_t>(b) * a.max_pages;
  const int lp0 = pos0 >> 4;
  int pg0 = -1;
  if (warp == 3) {
    const int npg = (pl.chunk_len + 15) >> 4;   // a full chunk's pages; the unused tail is harmless
    for (int i = lane; i < npg; i += 32) spages[i] = lp0 + i < a.max_pages ? bt[lp0 + i] : -1;
  } else if ((warp == 0 || warp == 2) && lane < kTilePages) {
    pg0 = lp0 + lane < a.max_pages ? bt[lp0 + lane] : -1;
  }
  const int n = min(max(a.n_nodes[b], 0), a.n_max);
  const int C = a.ctx_len[b];
  const int total = C + n;
  const int rows = n * pl.group;
  const int pos1 = min(pos0 + pl.chunk_len, total);
  const int n_tiles = pos1 > pos0 ? (pos1 - pos0 + kTile - 1) / kTile : 0;

  if (row0 >= rows) {
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

  // the first K or V tile: lane p copies page p
  const uint64_t policy = l2_evict_first_policy();
  auto issue_tile = [&](bool is_k, int j, int pg) {
    uint64_t* full = is_k ? k_full : v_full;
    const int s = j % (is_k ? kKStages : kVStages);
    const bool in = lane < kTilePages && pos0 + j * kTile + 16 * lane < pos1;
    const bool valid = in && pg >= 0 && pg < a.num_pages;
    if (is_k && in && !valid && a.status) atomicOr(a.status, TAPS_DEVFAULT_PAGE);
    const uint32_t vm = __ballot_sync(kFullMask, valid);
    if (lane == 0) mbar_arrive_expect_tx(&full[s], __popc(vm) * S::kPageBytes);
    __syncwarp();
    if (valid) {
      const int64_t blk = (static_cast<int64_t>(pg) * a.Hkv + kv) * (16 * D);
      bulk_load(sb + (is_k ? S::kK : S::kV) + s * S::kTileBytes + lane * S::kPageBytes,
                (is_k ? a.k : a.v) + blk, S::kPageBytes, &full[s], policy);
    }
  };
  if (n_tiles > 0 && threadIdx.x == 96) {
    // (warp 3) Q rows of this block: one box of (64 dims, group heads,
    // 128/group nodes) per 64-dim half; nodes past n_max read as zeros. (Not
    // for an empty chunk, whose epilogue stages its zero rows in the Q buffer.)
    mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(CH * 16384));
    for (int c = 0; c < CH; ++c)
      tma_load_4d(sb + S::kQ + c * 16384, &maps.q, q_full, c * 64, kv * pl.group,
                  row0 / pl.group, b);
  }
  if (n_tiles > 0 && (warp == 0 || warp == 2)) issue_tile(warp == 0, 0, pg0);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // peers may push into this CTA only once its barriers exist: waited on
  // before the first push
  if (!single) cluster_arrive_relaxed();
  const uint32_t tmem = *tmem_slot;
  constexpr uint32_t kOCol = 0;
  auto s_col = [](int u) { return static_cast<uint32_t>(128 + u * 128); };

  if (n_tiles == 0) {
    // this chunk is empty for this request: nothing to compute, the epilogue
    // below contributes zero rows with an empty softmax
  } else if (warp == 0 || warp == 2) {
    // ------------------------------------------------------------ TMA producers
    // warp 0 streams the K tiles, warp 2 the V tiles, each into its own ring,
    // so neither producer's wait stalls the other. Lane p handles page p of a
    // tile, with its page id fetched one tile ahead; tile 0 left above.
    const bool is_k = warp == 0;
    const int nst = is_k ? kKStages : kVStages;
    uint64_t* full = is_k ? k_full : v_full;
    auto in_chunk = [&](int j) { return lane < kTilePages && pos0 + j * kTile + 16 * lane < pos1; };
    int pg = n_tiles > 1 && in_chunk(1) ? spages[kTilePages + lane] : -1;
    int issued = 1;
    for (int j = 1; j < n_tiles; ++j) {
      if (__any_sync(kFullMask, *abort_flag != 0)) break;
      const int s = j % nst;
      // slot s last held tile t = j - nst: free once QK (K) or the burst
      // holding PV (V) of tile t is done. Neither barrier can have completed
      // its following phase yet: that needs a tile this warp has not issued.
      const int t = j - nst;
      if (j >= nst && !__all_sync(kFullMask, is_k ? mbar_wait(&s_full[t % kSBufs], (t / kSBufs) & 1)
                                                  : mbar_wait(&v_empty[s], (t / kVStages) & 1))) {
        if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
        break;
      }
      issue_tile(is_k, j, pg);
      issued = j + 1;
      if (j + 1 < n_tiles) pg = in_chunk(j + 1) ? spages[(j + 1) * kTilePages + lane] : -1;
    }
    // never leave the CTA with copies in flight
    if (lane == 0) {
      if (is_k) mbar_wait(q_full, 0);
      for (int j = max(0, issued - nst); j < issued; ++j) mbar_wait(&full[j % nst], (j / nst) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_qk = idesc_bf16_f32(128, kTile, false, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, false, true);
    constexpr int kQkSteps = D / 16;
    auto qk_step = [&](int jj, int ks) {
      const uint32_t kb = sb + S::kK + (jj % kKStages) * S::kTileBytes;
      const uint64_t ad = sw128_desc(sb + S::kQ + (ks / 4) * 16384 + (ks % 4) * 32, 16, 1024);
      const uint64_t bd = sw128_desc(kb + (ks / 4) * 1024 + (ks % 4) * 32, 16, S::kGroupStride);
      mma_bf16(tmem + s_col(jj % kSBufs), ad, bd, idesc_qk, ks > 0 ? 1u : 0u);
    };
    bool ok = __all_sync(kFullMask, mbar_wait(q_full, 0));
    // QK of the first two tiles
    for (int jj = 0; ok && jj < min(2, n_tiles); ++jj) {
      ok = __all_sync(kFullMask, mbar_wait(&k_full[jj % kKStages], (jj / kKStages) & 1));
      if (ok && lane == 0) {
        tc_fence_after();
#pragma unroll
        for (int ks = 0; ks < kQkSteps; ++ks) qk_step(jj, ks);
        mma_commit(&s_full[jj % kSBufs]);
      }
      __syncwarp();
    }
    bool o_started = false;   // O holds a first product
    // Pages holding a valid token, one byte per tile of the chunk (at most
    // kMaxChunkTokens / kTile = 256 tiles): lane l keeps tiles l, l + 32, ...
    // Read once here, while Q and the first tiles load, so that no
    // shared-memory load (queued behind the tensor core's operand reads)
    // sits between two bursts.
    uint64_t live8 = 0;
    for (int t = lane; t < n_tiles; t += 32) {
      uint32_t m = 0;
      for (int p = 0; p < kTilePages; ++p) {
        if (pos0 + t * kTile + 16 * p >= pos1) break;
        const int pg = spages[t * kTilePages + p];
        if (pg >= 0 && pg < a.num_pages) m |= 1u << p;
      }
      live8 |= static_cast<uint64_t>(m) << (8 * (t >> 5));
    }
    // the page cut by the end of the sequence, if any: its rows past the end
    // are zeroed so that P = 0 never meets stale (possibly non-finite) data
    const int cut_tile = (pos1 & 15) ? (pos1 - 1 - pos0) / kTile : -1;
    const int cut_page = (pos1 & 15) ? ((pos1 - 1 - pos0) % kTile) / 16 : 0;
    // burst j: PV of tile j (after its softmax) alternating with QK of tile j+2
    // (no abort-flag poll here: every wait is bounded)
    for (int j = 0; ok && j < n_tiles; ++j) {
      const int jn = j + 2;
      const bool has_qk = jn < n_tiles;
      const int sv = j % kVStages;
      // V tile j, K tile j+2 and P of tile j: the three barriers are tested
      // back to back (their latencies overlap), and only one that has not
      // completed yet is then waited on
      {
        uint64_t* bv = &v_full[sv];
        uint64_t* bk = &k_full[jn % kKStages];
        uint64_t* bp = &p_full[j % kSBufs];
        const uint32_t qv = (j / kVStages) & 1, qk = (jn / kKStages) & 1, qp = (j / kSBufs) & 1;
        bool wv = mbar_try_wait(bv, qv);
        bool wk = !has_qk || mbar_try_wait(bk, qk);
        bool wp = mbar_try_wait(bp, qp);
        if (!wv) wv = mbar_wait(bv, qv);
        if (!wk) wk = mbar_wait(bk, qk);
        if (!wp) wp = mbar_wait(bp, qp);
        if (!__all_sync(kFullMask, wv && wk && wp)) {
          ok = false;
          break;
        }
      }
      const uint32_t page_live =
          static_cast<uint32_t>(__shfl_sync(kFullMask, live8, j & 31) >> (8 * (j >> 5))) & 0xFFu;
      if (j == cut_tile && ((page_live >> cut_page) & 1u)) {
        const int nv = pos1 & 15;
        uint8_t* pb = smem + S::kV + sv * S::kTileBytes + cut_page * S::kPageBytes;
        for (int e = lane; e < 16 * 8 * CH; e += 32) {
          const int w = e / (8 * CH), c = (e / 8) % CH, q16 = e % 8;
          if (w >= nv)
            *reinterpret_cast<uint4*>(pb + (w >> 3) * S::kGroupStride + c * 1024 +
                                      (w & 7) * 128 + q16 * 16) = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
      }
      __syncwarp();
      if (lane == 0) {
        tc_fence_after();
        const uint32_t vb = sb + S::kV + sv * S::kTileBytes;
        const uint32_t pcol = tmem + s_col(j % kSBufs);
#pragma unroll
        for (int ks = 0; ks < kTilePages; ++ks) {
          if ((page_live >> ks) & 1u) {
            const uint64_t bd = sw128_desc(vb + ks * S::kPageBytes, 1024, S::kGroupStride);
            mma_bf16_ts(tmem + kOCol, pcol + ks * 8, bd, idesc_pv, o_started ? 1u : 0u);
            o_started = true;
          }
          if (has_qk && ks < kQkSteps) qk_step(jn, ks);
        }
        // S first: the softmax waits on it; then the V slot / O update
        if (has_qk) mma_commit(&s_full[jn % kSBufs]);
        mma_commit(&v_empty[sv]);
        if (j == n_tiles - 1) mma_commit(o_full);
      }
      __syncwarp();
    }
    if (!ok && lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
    // every MMA issued by this warp completes before TMEM is released
    if (lane == 0) mma_commit(drain);
    __syncwarp();
    mbar_wait(drain, 0);
  }
  if (warp >= 4) {
    // ------------------------------------------------------------ softmax warps
    // (also for an empty chunk: its epilogue stages zero rows for the peers)
    const int quarter = warp & 3;                  // TMEM lanes 32*quarter .. +31
    const int r = quarter * 32 + lane;             // row of the block
    const int grow = row0 + r;
    const bool valid_row = grow < rows;
    const int node = valid_row ? grow / pl.group : 0;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const float scale = a.scale_log2;
    const uint32_t* mrow = a.mask + (static_cast<int64_t>(b) * a.n_max + node) * a.W;
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    // lane p holds the page id of page p of the next tile, fetched one tile
    // ahead: shared-memory loads queue behind the tensor core's operand reads
    auto page_id = [&](int j) {
      return lane < kTilePages && pos0 + j * kTile + 16 * lane < pos1
                 ? spages[j * kTilePages + lane] : -1;
    };
    int pgn = page_id(0);
    for (int j = 0; j < n_tiles; ++j) {
      // visible columns of this row in tile j: on a valid page, inside the
      // chunk, and for tree nodes on the row's ancestor path
      const uint32_t live = __ballot_sync(kFullMask, pgn >= 0 && pgn < a.num_pages);
      if (j + 1 < n_tiles) pgn = page_id(j + 1);
      uint64_t vis[2] = {0ull, 0ull};
      if (valid_row) {
        const int t0 = pos0 + j * kTile;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int th = t0 + 64 * h;
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const int nv = min(16, pos1 - (th + 16 * p));
            if (((live >> (4 * h + p)) & 1u) && nv > 0)
              vis[h] |= (nv == 16 ? 0xFFFFull : ((1ull << nv) - 1)) << (16 * p);
          }
          if (th + 64 > C) {
            // columns from i0 on are tree nodes jn = th + i - C
            const int i0 = max(0, C - th);
            const uint64_t win = mask_window(mrow, a.W, th + i0 - C);
            const uint64_t ctx_cols = i0 == 0 ? 0ull : ((1ull << i0) - 1);
            vis[h] &= ctx_cols | (win << i0);
          }
        }
      }
      // S of tile j. A shared-memory access waits behind the tensor core's
      // operand reads, so the abort flag is read only when S is not ready
      // at the first test (every wait is bounded in any case).
      const int u = j % kSBufs;
      if (!__all_sync(kFullMask, mbar_try_wait(&s_full[u], (j / kSBufs) & 1))) {
        if (__any_sync(kFullMask, *abort_flag != 0)) { ok = false; break; }
        if (!__all_sync(kFullMask, mbar_wait(&s_full[u], (j / kSBufs) & 1))) {
          if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          ok = false;
          break;
        }
      }
      tc_fence_after();
      uint32_t sv[128];
      tmem_ld128_sync(lane_base + s_col(u), sv);
      if ((vis[0] & vis[1]) != ~0ull) {
#pragma unroll
        for (int i = 0; i < 128; ++i)
          if (!((vis[i >> 6] >> (i & 63)) & 1ull)) sv[i] = 0xFF800000u;   // -inf
      }
      // row max: eight chains of three-input maxima
      float mx[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) mx[k] = __uint_as_float(sv[k]);
#pragma unroll
      for (int i = 8; i < 128; i += 2)
        mx[(i >> 1) & 7] = max3f(mx[(i >> 1) & 7], __uint_as_float(sv[i]), __uint_as_float(sv[i + 1]));
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
      // P over the first 64 columns of this S buffer, from each 64-column half
      // of S in turn: x = s * scale - m for two columns per packed FMA, 2^x on
      // the SFU, bf16 pairs, packed row sums
      const float nm = m_used == -INFINITY ? 0.f : -m_used;
      const bool any = m_used != -INFINITY;
      const uint64_t scale2 = f32x2(scale, scale), nm2 = f32x2(nm, nm);
      uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
      // A rolled loop, so that the half's code exists once: the kernel runs
      // measurably faster with this smaller hot loop than with both halves
      // unrolled from the registers that hold the row (and slower again when
      // the row max is taken in slices too). Each half is read again from
      // TMEM and masked again on a partial tile; S columns [64, 128) are
      // intact when the first half's P goes to [0, 32).
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        uint32_t sh[64];
        tmem_ld64_sync(lane_base + s_col(u) + 64 * h, sh);
        const uint64_t vh = h ? vis[1] : vis[0];
        if (vh != ~0ull) {
#pragma unroll
          for (int i = 0; i < 64; ++i)
            if (!((vh >> i) & 1ull)) sh[i] = 0xFF800000u;   // -inf
        }
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const uint64_t x = fma_f32x2(
              f32x2(__uint_as_float(sh[2 * i]), __uint_as_float(sh[2 * i + 1])), scale2, nm2);
          float x0, x1;
          f32x2_split(x, x0, x1);
          const float p0 = any ? ex2_approx(x0) : 0.f;
          const float p1 = any ? ex2_approx(x1) : 0.f;
          pk[i] = pack_bf16x2(p0, p1);
          acc2[i & 3] = add_f32x2(acc2[i & 3], f32x2(p0, p1));
        }
        tmem_st32(lane_base + s_col(u) + 32 * h, pk);
      }
      float a0, a1, a2, a3;
      f32x2_split(add_f32x2(acc2[0], acc2[1]), a0, a1);
      f32x2_split(add_f32x2(acc2[2], acc2[3]), a2, a3);
      const float psum = (a0 + a1) + (a2 + a3);
      l = l * alpha + psum;
      // a grown max rescales O before P of this tile is released; the PV of
      // the previous tile may still be running, so wait for it first
      const bool need_rescale = grow_max && j > 0 && alpha != 1.f;
      if (__any_sync(kFullMask, need_rescale)) {
        if (!__all_sync(kFullMask, mbar_wait(&v_empty[(j - 1) % kVStages],
                                             ((j - 1) / kVStages) & 1))) {
          if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
          ok = false;
          break;
        }
        tc_fence_after();
        const float f = need_rescale ? alpha : 1.f;
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32_sync(lane_base + kOCol + c * 32, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
          tmem_st32(lane_base + kOCol + c * 32, o);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[u]);
    }
    if (ok && n_tiles > 0 && !__all_sync(kFullMask, mbar_wait(o_full, 0))) {
      if (lane == 0) set_fault(abort_flag, a.status, TAPS_DEVFAULT_TIMEOUT);
      ok = false;
    }
    if (threadIdx.x == 128) pdl_launch_dependents();
    // ---- epilogue. Once the last PV is done every MMA reading Q has
    // finished: stage the normalised bf16 rows there in the same swizzled
    // layout, and this row's (max, sum) next to them.
    const bool good = ok && valid_row && l > 0.f;
    const float inv = good ? 1.f / l : 0.f;
    uint8_t* srow = smem + S::kQ + r * 128;
    if (n_tiles > 0 && __any_sync(kFullMask, good)) {
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < D / 64; ++c) {
        uint32_t o[64];
        tmem_ld64_sync(lane_base + kOCol + c * 64, o);
        if (!good) {
#pragma unroll
          for (int k = 0; k < 64; ++k) o[k] = 0u;
        }
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
    reinterpret_cast<float2*>(smem + S::kMl)[r] =
        good ? make_float2(m_used, l) : make_float2(-INFINITY, 0.f);
    // the staged rows and (max, sum) leave through bulk copies (async proxy)
    fence_proxy_async_smem();
    if (single) {
      if (a.lse && grow < pl.rows_max) {
        const int64_t orow = (static_cast<int64_t>(b) * a.n_max + grow / pl.group) * a.Hq +
                             kv * pl.group + grow % pl.group;
        a.lse[orow] = good ? (m_used + log2f(l)) * kLn2 : 0.f;
      }
      named_bar_sync(1, 128);
      if (threadIdx.x == 128) {
        for (int c = 0; c < CH; ++c)
          tma_store_4d(&maps.out, sb + S::kQ + c * 16384, c * 64, kv * pl.group, row0 / pl.group,
                       b);
        bulk_commit();
        bulk_wait_read_all();
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();   // every role is done with TMEM; rows and (max, sum) are staged
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (single) return;
  // ---- cluster reduction. Each CTA pushes every peer that peer's slice of
  // its staged rows and (max, sum) with bulk copies into the peer's receive
  // buffer as soon as its own rows are staged, then combines its own slice
  // over the cluster's chunks from shared memory and writes it out.
  const uint32_t ml_off = static_cast<uint32_t>(cs * CH * per * 128);
  cluster_wait();
  if (warp == 0 && lane < cs) {
    // lane q sends peer q rows [qb, qe) of every 64-dim half and their (max, sum)
    const int qb = min(kRowsPerCta, lane * per), qe = min(kRowsPerCta, qb + per);
    if (qe > qb) {
      const uint32_t dst = mapa_shared(sb + S::kRecv, lane);
      const uint32_t bar = mapa_shared(smem_u32(recv), lane);
      for (int c = 0; c < CH; ++c)
        bulk_copy_to_peer(dst + ((rank * CH + c) * per) * 128, sb + S::kQ + c * 16384 + qb * 128,
                          (qe - qb) * 128, bar);
      bulk_copy_to_peer(dst + ml_off + rank * per * 8, sb + S::kMl + qb * 8, (qe - qb) * 8, bar);
    }
  }
  const bool got = mbar_wait(recv, 0);
  if (!got && threadIdx.x == 0 && a.status) atomicOr(a.status, TAPS_DEVFAULT_TIMEOUT);
  // this CTA's slice has landed, so the peers may release what they sent it
  // (the landing itself was observed on the mbarrier: nothing to release)
  __syncwarp();
  cluster_arrive_relaxed();
  uint8_t* rv = smem + S::kRecv;
  float2* rml = reinterpret_cast<float2*>(rv + ml_off);
  float2* stat = reinterpret_cast<float2*>(smem + S::kStat);
  if (got && threadIdx.x < re - rb) {
    // per row: the cluster-wide max M, each chunk's weight l_q 2^(m_q - M)
    // (in place of m_q) and the total L. Unrolled to the largest cluster, so
    // that every peer's (max, sum) is loaded at once.
    const int i = threadIdx.x;
    float2 ml[kMaxCluster];
#pragma unroll
    for (int q = 0; q < kMaxCluster; ++q)
      ml[q] = q < cs ? rml[q * per + i] : make_float2(-INFINITY, 0.f);
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < kMaxCluster; ++q) M = fmaxf(M, ml[q].x);
    float L = 0.f;
#pragma unroll
    for (int q = 0; q < kMaxCluster; ++q) {
      if (q < cs) {
        const float w = ml[q].y > 0.f ? ml[q].y * ex2_approx(ml[q].x - M) : 0.f;
        rml[q * per + i].x = w;
        L += w;
      }
    }
    stat[i] = make_float2(M, L);
  }
  __syncthreads();
  if (got) {
    // kTpr threads per row, each combining two adjacent 16-byte pieces of it,
    // so that the row's output offset, statistics and reciprocal are worked
    // out once per row rather than once per piece
    constexpr int kTpr = D / 16;
    constexpr int kRowsPerPass = kThreadsTc / kTpr;
    const int qa = 2 * (threadIdx.x % kTpr);        // pieces qa, qa + 1 of the row's D / 8
    for (int i = threadIdx.x / kTpr; i < re - rb; i += kRowsPerPass) {
      const int rr = rb + i, gr = row0 + rr;
      if (gr >= pl.rows_max) continue;
      const float2 st = stat[i];
      const bool row_ok = gr < rows && st.y > 0.f;
      const float linv = row_ok ? 1.f / st.y : 0.f;
      const int64_t orow = (static_cast<int64_t>(b) * a.n_max + gr / pl.group) * a.Hq +
                           kv * pl.group + gr % pl.group;
      const uint8_t* vp = rv + ((qa >> 3) * per + i) * 128;
      const uint32_t oa = ((qa & 7) ^ (rr & 7)) << 4, ob = (((qa + 1) & 7) ^ (rr & 7)) << 4;
      float acc[16];
#pragma unroll
      for (int k = 0; k < 16; ++k) acc[k] = 0.f;
#pragma unroll 4
      for (int q = 0; q < cs; ++q) {
        const float w = rml[q * per + i].x;
        const uint8_t* vq = vp + q * CH * per * 128;
        const uint4 x = *reinterpret_cast<const uint4*>(vq + oa);
        const uint4 y = *reinterpret_cast<const uint4*>(vq + ob);
        const uint32_t u[8] = {x.x, x.y, x.z, x.w, y.x, y.y, y.z, y.w};
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          acc[2 * k] = fmaf(w, __uint_as_float(u[k] << 16), acc[2 * k]);
          acc[2 * k + 1] = fmaf(w, __uint_as_float(u[k] & 0xFFFF0000u), acc[2 * k + 1]);
        }
      }
      uint4* dst = reinterpret_cast<uint4*>(a.out + orow * D + qa * 8);
      dst[0] = make_uint4(
          pack_bf16x2(acc[0] * linv, acc[1] * linv), pack_bf16x2(acc[2] * linv, acc[3] * linv),
          pack_bf16x2(acc[4] * linv, acc[5] * linv), pack_bf16x2(acc[6] * linv, acc[7] * linv));
      dst[1] = make_uint4(
          pack_bf16x2(acc[8] * linv, acc[9] * linv), pack_bf16x2(acc[10] * linv, acc[11] * linv),
          pack_bf16x2(acc[12] * linv, acc[13] * linv),
          pack_bf16x2(acc[14] * linv, acc[15] * linv));
      if (a.lse && qa == 0) a.lse[orow] = row_ok ? (st.x + log2f(st.y)) * kLn2 : 0.f;
    }
  }
  // every peer has received what this CTA sent it before this CTA exits
  __syncwarp();
  cluster_wait();
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
