/*
 * taps.h - C ABI of the TAPS per-round hot path on one GB300 (sm_103a).
 *
 * TAPS (Target-Aware Prefix tree Selection, diffusion-drafted speculative
 * decoding) runs one decoding round in six steps; each has one entry point:
 *
 *   taps_topk_marginals    Sec. 4.1 stage 1 + Sec. 4.2 features
 *   taps_score_reach       Sec. 4.2, Eq. 1, Algorithm 1 (scorer + sibling softmax)
 *   taps_select_subtree    Sec. 4.2-4.3, Eq. 2, Eq. 3, Algorithm 1 (selection)
 *   taps_build_tree_mask   Sec. 4.1 stage 3 / Sec. 4.3 (tree attention needs
 *                          a connected subtree rooted at the current position)
 *   taps_tree_verify_attn  Sec. 4.1 stage 3 (target verifies the subtree with
 *                          tree attention), over a paged bf16 KV cache
 *   taps_accept            Sec. 4.1 and Limitations (greedy, temperature 0,
 *                          lossless acceptance of the longest matching path)
 *
 * taps_score_select_mask runs the second to fourth steps in two launches.
 *
 * and two steps that follow verification in the decoding loop:
 *
 *   taps_target_greedy_accept  Limitations (temperature 0: the target's
 *                          choice is the argmax of its verify logits) fused
 *                          with the acceptance walk of taps_accept
 *   taps_compact_accepted_kv   Sec. 4.1 (drafting and verification
 *                          alternate: the accepted path becomes context)
 *
 * Conventions shared by every call:
 *  - Array arguments are DEVICE pointers owned by the caller. The library never
 *    allocates, frees or synchronises; every call is asynchronous on `stream`
 *    (a cudaStream_t passed as void*, NULL = legacy default stream).
 *  - Parameter structs are HOST pointers, read before the call returns.
 *  - Arrays are dense, row-major, in the shapes given; B = requests,
 *    L = drafted positions (tree depth), V = vocabulary, K = top-K per
 *    position, N = n_max node budget (root included).
 *  - Return value is a taps_status. Host-side argument checks run before any
 *    launch; on any error nothing is launched and outputs are untouched.
 *    TAPS_ERR_CUDA reports a launch failure (cudaGetLastError).
 *  - Device-detected faults (an out-of-range page id) never trap: the kernel
 *    skips the bad access and ORs a TAPS_DEVFAULT_* bit into the caller's
 *    `status` word (nullable), which the caller reads after synchronising.
 *  - Workspaces are caller-allocated device buffers of at least the size the
 *    matching *_workspace_bytes() query returns, 256-byte aligned and
 *    ZERO-FILLED before their first use; every call leaves the counters it
 *    uses back at zero. Calls that share a workspace must not overlap.
 */
#ifndef TAPS_H_
#define TAPS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum taps_status {
  TAPS_OK = 0,
  TAPS_ERR_INVALID_ARG = 1,   /* null pointer, negative size, inconsistent shape */
  TAPS_ERR_UNSUPPORTED = 2,   /* outside the supported limits listed per call   */
  TAPS_ERR_WORKSPACE = 3,     /* workspace missing, too small or misaligned     */
  TAPS_ERR_CUDA = 4,          /* a kernel launch failed                         */
  TAPS_ERR_DEVICE = 5         /* reserved for device-detected faults            */
} taps_status;

enum { TAPS_F32 = 0, TAPS_BF16 = 1 };
enum { TAPS_SCORER_MARGINAL = 0, TAPS_SCORER_MLP = 1, TAPS_SCORER_MARGINAL_PRODUCT = 2 };
enum { TAPS_DEVFAULT_PAGE = 1, TAPS_DEVFAULT_TIMEOUT = 2 };

/* Limits (TAPS_ERR_UNSUPPORTED beyond them). */
#define TAPS_MAX_K 32
#define TAPS_MAX_L 31
#define TAPS_MAX_V 262143      /* token ids must fit in 18 bits */
#define TAPS_MAX_NODES 512
#define TAPS_MAX_EMB 32
#define TAPS_MAX_HIDDEN 64
#define TAPS_MAX_LAYERS 128

const char* taps_status_string(int status);
int taps_version(void);

/* ------------------------------------------------------------------------
 * taps_topk_marginals - Sec. 4.1 stage 1 (the top-K tokens of every drafted
 * position form the candidate tree) and Sec. 4.2 (the scorer reads the child
 * log-probability and the positional entropy).
 *
 * logits     [B, L, V] of dtype TAPS_F32 or TAPS_BF16; row (b, d) starts at
 *            element (b * L + d) * row_stride (row_stride >= V).
 * topk_ids   [B, L, K] int32, out: the K largest logits of each row, ordered
 *            by logit descending, then token id ascending.
 * topk_logp  [B, L, K] f32, out: logit - lse (full-vocabulary log-probability).
 * lse        [B, L] f32, out: log sum_v exp(logit_v).
 * entropy    [B, L] f32, out: -sum_v p_v log p_v in nats, full vocabulary.
 * ws         workspace of taps_topk_marginals_workspace_bytes(B, L, V, K); its
 *            first 256 KiB hold per-row counters that must be zero before the
 *            first call and that every call leaves at zero, so one zero-filled
 *            workspace can serve calls of any shape on one stream.
 * Limits: 1 <= K <= min(32, V), 1 <= V <= 262143. Logits may be -inf
 * (probability 0, no entropy contribution) but not +inf or NaN, and every row
 * needs at least K finite logits for the top-K to be meaningful.
 * Device-side waits: the kernel that serves a few rows waits for the bulk
 * copies of its logits slice with a bound of about 2 s and then carries on
 * either way. There is no status word to report an expired wait: it would
 * need a copy from the caller's memory that never completes.
 * ---------------------------------------------------------------------- */
size_t taps_topk_marginals_workspace_bytes(int B, int L, int V, int K);
int taps_topk_marginals(const void* logits, int dtype, int64_t row_stride,
                        int B, int L, int V, int K,
                        int32_t* topk_ids, float* topk_logp, float* lse, float* entropy,
                        void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * taps_topk_marginals_noalloc - the same computation and outputs as
 * taps_topk_marginals, for callers that cannot allocate device memory. The
 * paper has no counterpart: this is a deployment convenience of this library.
 *
 * Who needs it: a serving engine that reserved all of device memory for its KV
 * cache at start-up, a plugin running inside a host framework that owns every
 * device allocation, or a decode loop that cannot afford the device-wide
 * synchronisation cudaMalloc may cause. The caller still passes inputs and
 * outputs; the partial records live in a fixed array of
 * TAPS_NOALLOC_SCRATCH_BYTES (2 MiB) of device memory inside the library,
 * which every GPU that loads the library holds until the process exits.
 * Nothing is allocated or freed by this call.
 *
 * The first call on each device looks up that array's device address
 * (cudaGetSymbolAddress, with the caller's current device); make that first
 * call before any stream capture. Each call clears the counters it uses before
 * its kernel runs. Every call shares the one array per device, so calls that
 * overlap on the GPU (different streams, or different host threads without
 * ordering) race: serialise them.
 * The library caches per-device state for the life of the process (this
 * array's address, kernel attributes, cluster capacities), so resetting a
 * device (cudaDeviceReset) between calls into the library is not supported.
 * Limits: B * L <= TAPS_NOALLOC_MAX_ROWS (4096); beyond it the call returns
 * TAPS_ERR_UNSUPPORTED and launches nothing. Other limits as above.
 * ---------------------------------------------------------------------- */
#define TAPS_NOALLOC_MAX_ROWS 4096
#define TAPS_NOALLOC_SCRATCH_BYTES (2u * 1024u * 1024u)
int taps_topk_marginals_noalloc(const void* logits, int dtype, int64_t row_stride,
                                int B, int L, int V, int K,
                                int32_t* topk_ids, float* topk_logp, float* lse,
                                float* entropy, void* stream);

/* ------------------------------------------------------------------------
 * taps_score_reach - Sec. 4.2, Eq. 1 and Algorithm 1: for every parent of
 * the candidate trie, q_cond(parent -> child) = softmax over the K siblings
 * of the scorer logit of each edge; optionally Eq. 2, the reach
 * q_reach = product of q_cond along the path, of a caller-given node list.
 *
 * The candidate trie: every node at depth d has the same K children, the
 * top-K tokens of position d; the root (depth 0) carries root_tok[b].
 * q_cond[b, d, i, j] (f32 [B, L, K, K], out) is the conditional acceptance
 * of child slot j of position d given that parent slot i of position d-1 was
 * reached; for d == 0 the parent is the root, row i = 0, and rows i >= 1 are
 * written as 0.
 *
 * Scorer (params->kind):
 *  TAPS_SCORER_MARGINAL  logit = topk_logp[b, d, j] (the paper's ablation that
 *                        ranks by the drafter's marginal confidence, Sec. 5.3).
 *  TAPS_SCORER_MARGINAL_PRODUCT  no softmax: q_cond[b, d, i, j] =
 *                        exp(topk_logp[b, d, j]) for every parent, so reach is
 *                        the product of the path's marginal probabilities, the
 *                        ranking of DDTree-style trees (Sec. 3.1, Limitation 1).
 *                        With lambda2 = 0 and tau = 0 the selection then
 *                        keeps the n_max paths of highest marginal probability.
 *  TAPS_SCORER_MLP       logit = w_lp * logp + w2 . relu(W1 f + b1) with
 *                        f = [E_tok[parent], E_tok[child], E_dep[d+1], logp,
 *                        entropy[b, d]] (Sec. 4.2 feature list). weights is a
 *                        device f32 buffer: tok_emb[vocab][E], dep_emb[max_depth][E],
 *                        W1[H][3E+2], b1[H], w2[H], w_lp[1], packed in that
 *                        order. Token ids must be < vocab; max_depth > L.
 *                        The kernel stages W1, b1, w2, w_lp and the depth
 *                        embeddings before it waits for the kernel launched
 *                        just before it on `stream` (programmatic dependent
 *                        launch), so that kernel must not write them (none
 *                        of this library's kernels does).
 *
 * Reach of an explicit node list (Eq. 2), optional: paths, path_len and
 * path_reach are all NULL with M == 0, or all given with M >= 1.
 *   paths      [B, M, L] uint8: node m of request b is the trie node reached
 *              from the root by top-K slots paths[b, m, 0 .. path_len[b, m]).
 *   path_len   [B, M] int32, its depth (0 = the root).
 *   path_reach [B, M] f32, out: product of q_cond along the path, one IEEE
 *              round-to-nearest multiply per edge, root to leaf: bit-identical
 *              to the reach taps_select_subtree computes for the same node.
 *              A length outside [0, L], or a slot >= K among the first
 *              path_len entries, names no node of the trie: reach 0.
 *   It runs after q_cond is complete, in a second kernel on the same stream.
 * Limits: K <= 32, L <= 31, E <= 32, H <= 64, B * M < 2^31 - 256.
 * ---------------------------------------------------------------------- */
typedef struct taps_scorer_params {
  int kind;
  int emb_dim;     /* E */
  int hidden;      /* H */
  int vocab;       /* rows of tok_emb */
  int max_depth;   /* rows of dep_emb */
  const float* weights;
} taps_scorer_params;

int taps_score_reach(const int32_t* root_tok, const int32_t* topk_ids, const float* topk_logp,
                     const float* entropy, int B, int L, int K,
                     const taps_scorer_params* params, float* q_cond,
                     const uint8_t* paths, const int32_t* path_len, int M,
                     float* path_reach, void* stream);

/* ------------------------------------------------------------------------
 * taps_select_subtree - Eq. 2 (reach = product of q_cond along the path),
 * Eq. 3 (utility = reach / (lambda1 + lambda2 * depth)) and Algorithm 1:
 * starting from S = {root}, repeatedly add the unselected node of largest
 * utility while |S| < n_max and that utility > tau.
 *
 * Arithmetic: reach and utility are f32 with IEEE round-to-nearest multiply
 * and divide, accumulated root to leaf; den(d) = lambda1 + lambda2 * d.
 * Ties: utility descending, then depth ascending, then token id ascending,
 * then the parent's position in the selection order ascending.
 * Outputs ([B, n_max] unless noted), nodes listed in the order the greedy
 * loop adds them (root = node 0, parent[i] < i); entries at i >= n_nodes[b]
 * are -1 (int) or 0 (float):
 *   n_nodes [B], parent, depth, token (root = root_tok[b]), slot (top-K slot
 *   of the node's position, root = -1), pos_id (= ctx_len[b] + depth),
 *   reach, utility.
 * Requires q_cond entries in [0, 1] (as taps_score_reach produces), lambda1 > 0,
 * lambda2 >= 0, tau >= 0, 1 <= n_max <= 512, K <= 32, L <= 31.
 * ---------------------------------------------------------------------- */
typedef struct taps_select_params {
  float lambda1;
  float lambda2;
  float tau;
  int n_max;
} taps_select_params;

int taps_select_subtree(const float* q_cond, const int32_t* topk_ids, const int32_t* root_tok,
                        const int32_t* ctx_len, int B, int L, int K,
                        const taps_select_params* params,
                        int32_t* n_nodes, int32_t* parent, int32_t* depth, int32_t* token,
                        int32_t* slot, int32_t* pos_id, float* reach, float* utility,
                        void* stream);

/* ------------------------------------------------------------------------
 * taps_score_select_mask - stages 2-4 of a round (Sec. 4.2, Eq. 1-3,
 * Algorithm 1, Sec. 4.3) in two launches: exactly the outputs of
 * taps_score_reach (q_cond, no path list), then taps_select_subtree, then
 * taps_build_tree_mask, with the same arguments, limits and errors, bit for
 * bit. The scorer keeps its own launch (one CTA per position and request,
 * which spreads a batch-1 round over many SMs); the selection and the mask
 * share one CTA per request, which builds the mask from the tree in shared
 * memory.
 * q_cond [B, L, K, K], the selection outputs [B] / [B, n_max] and mask
 * [B, n_max, ceil(n_max / 32)] are written as the separate calls write them.
 * ---------------------------------------------------------------------- */
int taps_score_select_mask(const int32_t* root_tok, const int32_t* topk_ids,
                           const float* topk_logp, const float* entropy, const int32_t* ctx_len,
                           int B, int L, int K, const taps_scorer_params* scorer,
                           const taps_select_params* select, float* q_cond, int32_t* n_nodes,
                           int32_t* parent, int32_t* depth, int32_t* token, int32_t* slot,
                           int32_t* pos_id, float* reach, float* utility, uint32_t* mask,
                           void* stream);

/* ------------------------------------------------------------------------
 * taps_build_tree_mask - the ancestor-or-self relation that tree attention
 * needs (Sec. 4.1 stage 3, Sec. 4.3).
 *
 * mask [B, n_max, ceil(n_max / 32)] uint32, out: bit (j % 32) of word j / 32
 * of row i is 1 iff i, j < n_nodes[b] and j is i or an ancestor of i.
 * parent [B, n_max] as written by taps_select_subtree.
 * ---------------------------------------------------------------------- */
int taps_build_tree_mask(const int32_t* parent, const int32_t* n_nodes, int B, int n_max,
                         uint32_t* mask, void* stream);

/* ------------------------------------------------------------------------
 * taps_tree_verify_attn - tree attention of the selected nodes against the
 * target's KV cache (Sec. 4.1 stage 3): for node i and query head h (KV head
 * h / (Hq / Hkv)),
 *   out = softmax(scale * q K^T over visible positions) V,
 * where the visible positions are the whole context [0, ctx_len[b]) and the
 * tree positions ctx_len[b] + j with bit j set in mask row i.
 *
 * q        [B, n_max, Hq, D] bf16 (post-RoPE queries of the tree nodes).
 * k_cache, v_cache [num_pages, Hkv, page_size, D] bf16 blocks in the TAPS page
 *          layout (taps_pack_kv_pages). Logical position t of request b lives
 *          in page block_table[b * max_pages + t / page_size], row t % page_size.
 *          Tree node j's K/V must already sit at logical position ctx_len[b] + j,
 *          so pages must cover ctx_len[b] + n_nodes[b].
 * out      [B, n_max, Hq, D] bf16, out; rows i >= n_nodes[b] are written as 0.
 * lse_out  [B, n_max, Hq] f32, out, nullable: natural-log softmax denominator.
 * max_ctx  host upper bound of ctx_len[b] (sizes the split of the context).
 * ws       unused (the chunks of a long context are combined on chip, inside
 *          a thread-block cluster); taps_tree_verify_attn_workspace_bytes()
 *          returns 0 and ws may be NULL.
 * status   device int32, nullable: TAPS_DEVFAULT_PAGE is ORed in when a page
 *          id is outside [0, num_pages); that page is then skipped.
 *          TAPS_DEVFAULT_TIMEOUT is ORed in if an internal pipeline wait
 *          exceeds its bound (about 2 s); the outputs are then undefined.
 * Limits: D in {64, 128}, page_size == 16, Hq / Hkv in {1, 2, 4, 8},
 *         n_max <= 512, max_ctx + n_max <= 65536.
 * ---------------------------------------------------------------------- */
size_t taps_tree_verify_attn_workspace_bytes(int B, int n_max, int Hq, int Hkv, int D,
                                             int max_ctx);
int taps_tree_verify_attn(const void* q, const void* k_cache, const void* v_cache,
                          int64_t num_pages, const int32_t* block_table, int max_pages,
                          const int32_t* ctx_len, const int32_t* n_nodes, const uint32_t* mask,
                          int B, int n_max, int Hq, int Hkv, int D, int page_size, float scale,
                          int max_ctx, void* out, float* lse_out,
                          void* ws, size_t ws_bytes, int32_t* status, void* stream);

/* ------------------------------------------------------------------------
 * taps_pack_kv_pages / taps_unpack_kv_pages - the paged KV cache layout that
 * taps_tree_verify_attn reads (Sec. 4.1 stage 3 verifies the tree against the
 * target's KV cache; the paper fixes no layout, this one is the library's).
 *
 * The cache is [num_pages][Hkv] blocks of 16 tokens x D bf16 values (D in
 * {64, 128}), 16 * D * 2 bytes each, in the same block order as a logical
 * [num_pages, Hkv, 16, D] cache. Inside a block, token w and dim d sit at byte
 *   (w / 8) * (D / 64) * 1024 + (d / 64) * 1024 + (w % 8) * 128
 *     + (((d % 64) / 8) XOR (w % 8)) * 16 + (d % 8) * 2:
 * 8-token groups of 128-byte rows with the 128-byte swizzle, so one
 * contiguous copy per page lands in shared memory exactly as the tensor core
 * reads it. A model writing its K/V can write this layout directly.
 * pack: src logical -> dst TAPS layout; unpack: the reverse. src and dst are
 * device buffers of num_pages * Hkv * 16 * D bf16, 16-byte aligned, distinct.
 * ---------------------------------------------------------------------- */
int taps_pack_kv_pages(const void* src, void* dst, int64_t num_pages, int Hkv, int D,
                       void* stream);
int taps_unpack_kv_pages(const void* src, void* dst, int64_t num_pages, int Hkv, int D,
                         void* stream);

/* ------------------------------------------------------------------------
 * taps_accept - lossless greedy acceptance (Sec. 4.1, Limitations): from the
 * root, step into the child whose token equals the target's greedy token at
 * the current node, until no child matches.
 *
 * target_tok [B, n_max] int32: the target model's greedy next token after
 *          the prefix ending at node i.
 * accept_len [B] out: accepted draft tokens (depth of the last accepted node).
 * accepted_nodes [B, L + 1] out: node indices root .. last, then -1.
 * bonus_tok [B] out: target_tok at the last accepted node.
 * ---------------------------------------------------------------------- */
int taps_accept(const int32_t* parent, const int32_t* token, const int32_t* n_nodes,
                const int32_t* target_tok, int B, int n_max, int L,
                int32_t* accept_len, int32_t* accepted_nodes, int32_t* bonus_tok, void* stream);

/* ------------------------------------------------------------------------
 * taps_target_greedy_accept - the target's greedy token at every tree node,
 * fused with the acceptance walk. At temperature 0 (Limitations) the target
 * accepts a draft token iff it equals the argmax of the target's logits after
 * the prefix ending at the node's parent; Sec. 4.1 then keeps the longest
 * root path of accepted tokens.
 *
 * verify_logits [B, n_max, V] of dtype TAPS_F32 or TAPS_BF16: the target's
 *          next-token logits after the prefix ending at tree node i; row
 *          (b, i) starts at element (b * n_max + i) * row_stride. Only rows
 *          i < n_nodes[b] are read.
 * parent, token, n_nodes as written by taps_select_subtree.
 * target_tok [B, n_max] int32, out: the lowest vocabulary index attaining the
 *          row's maximum (-0.0 equals +0.0) for i < n_nodes[b], else -1.
 * accept_len, accepted_nodes, bonus_tok: out, exactly as taps_accept computes
 *          them from target_tok.
 * ws       workspace of taps_target_greedy_accept_workspace_bytes(B, n_max),
 *          zero-filled before the first call; every call leaves it at zero.
 * Limits: n_max <= 512, L <= 31, row_stride >= V. Logits must not be NaN.
 * ---------------------------------------------------------------------- */
size_t taps_target_greedy_accept_workspace_bytes(int B, int n_max);
int taps_target_greedy_accept(const void* verify_logits, int dtype, int64_t row_stride,
                              int B, int n_max, int V, const int32_t* parent,
                              const int32_t* token, const int32_t* n_nodes, int L,
                              int32_t* target_tok, int32_t* accept_len, int32_t* accepted_nodes,
                              int32_t* bonus_tok, void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * taps_compact_accepted_kv - commit the accepted path to the KV cache. The
 * decoding loop alternates drafting and verification (Sec. 4.1): after
 * acceptance the accepted tokens are context for the next round, so for
 * i = 0 .. accept_len[b] the K and V at logical position
 * ctx_len[b] + accepted_nodes[b, i] (where verification left tree node
 * accepted_nodes[b, i]) move to position ctx_len[b] + i, in every layer.
 * All reads of a (layer, request, head) finish before its writes; no other
 * position changes. Keys need no re-rotation: the node at path index i has
 * depth i, and its key was rotated at position id ctx_len[b] + i.
 *
 * k_layers, v_layers  HOST arrays of num_layers DEVICE pointers, one K and
 *          one V cache per layer, each [num_pages, Hkv, 16, D] bf16 in the
 *          TAPS page layout (16-byte aligned), updated in place.
 * block_table [B, max_pages], ctx_len [B] as for taps_tree_verify_attn; the
 *          pages holding positions >= ctx_len[b] must belong to request b
 *          alone.
 * accepted_nodes [B, L + 1], accept_len [B] as written by taps_accept.
 * status   device int32, nullable: TAPS_DEVFAULT_PAGE is ORed in when a
 *          position falls outside the block table or a page id outside
 *          [0, num_pages); that move is skipped.
 * Limits: num_layers <= TAPS_MAX_LAYERS, L <= 31, page_size == 16,
 *         D in {64, 128}.
 * ---------------------------------------------------------------------- */
int taps_compact_accepted_kv(void* const* k_layers, void* const* v_layers, int num_layers,
                             int64_t num_pages, const int32_t* block_table, int max_pages,
                             const int32_t* ctx_len, const int32_t* accepted_nodes,
                             const int32_t* accept_len, int B, int L, int Hkv, int D,
                             int page_size, int32_t* status, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* TAPS_H_ */
