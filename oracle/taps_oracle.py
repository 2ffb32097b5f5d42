"""Plain CPU oracle for one TAPS decoding round (test infrastructure only).

TEST INFRASTRUCTURE. Only the tests, ``__graft_entry__.smoke()`` and the CPU
baseline legs of ``bench.py`` may import this module. The library's product
path never calls it, and it shares no code, table or constant with the CUDA
path; it imports nothing from the package.

Every function is written from the paper (TAPS: Target-Aware Prefix Tree
Selection for Diffusion-Drafted Speculative Decoding) in the paper's order and
notation, slowly and plainly:

* ``topk_marginals``   Sec. 4.1 stage 1 and the scorer features of Sec. 4.2.
* ``score_qcond``      Sec. 4.2, Eq. 1 and Algorithm 1 (sibling softmax of
                       the scorer logits).
* ``reach_of_path``    Sec. 4.2, Eq. 2 (product of q_cond along the path).
* ``path_reach``       Eq. 2 for an explicit list of nodes, in the float32
                       arithmetic that decides the tree.
* ``select_subtree``   Sec. 4.3, Eq. 3 and Algorithm 1 (greedy budgeted
                       prefix-closed selection), argmax over the frontier.
* ``select_subtree_literal``  Algorithm 1 over a fully materialised candidate
                       trie (tiny inputs only), argmax over every unselected
                       node and explicit ancestor insertion.
* ``build_tree_mask``  Sec. 4.1 stage 3 / Sec. 4.3: tree attention over a
                       connected subtree rooted at the current position.
* ``tree_verify_attn`` Sec. 4.1 stage 3: the target verifies the subtree with
                       tree attention (textbook masked softmax attention).
* ``accept``           Sec. 4.1 and Limitations: greedy (temperature 0)
                       verification, the longest accepted root path.
* ``target_greedy``    Limitations: at temperature 0 the target's choice at a
                       node is the argmax of its verify logits.
* ``compact_accepted_kv``  Sec. 4.1 (the loop alternates drafting and
                       verification): the accepted path becomes committed
                       context, so its K/V move to consecutive positions.

Precision. Where the paper fixes no precision the oracle computes in float64
(marginal statistics, scorer, attention). Reach and utility decide which nodes
are selected, an integer result, so they are computed in float32 with IEEE
round-to-nearest multiply and divide, in root-to-leaf path order, exactly as
the CUDA path takes the same decision.

Readings of the paper that this oracle encodes (the paper is silent there):

1. The candidate pool is the full implicit trie: every node at depth d-1 has
   the same K children, the top-K tokens of position d.
2. The root is depth 0 (the last committed token) and counts toward N_max.
3. Scorer (trained weights are not published): a random-init two-layer MLP
   over [E_tok[parent], E_tok[child], E_dep[depth], logp(child), H(depth)],
   plus w_lp * logp(child). Kind ``marginal`` is the paper's ablation that
   ranks by the drafter's marginal confidence: logit = logp(child).
   Kind ``marginal_product`` (DDTree-style) uses q = exp(logp(child)) as is.
4. Utility threshold is strict (utility > tau).
5. Total order used by argmax: utility desc, depth asc, token id asc, parent's
   position in the greedy order asc. Top-K ties: logit desc, token id asc.
6. Output nodes are listed in the order Algorithm 1 adds them (root = 0).
7. Attention: scale 1/sqrt(D), contiguous GQA groups, a tree node sees the
   whole context plus its ancestors-or-self; tree node j's K/V sit at logical
   cache position ctx_len + j.
8. Target greedy token: the first (lowest) vocabulary index attaining the
   maximum logit; -0.0 and +0.0 are equal values.
9. After acceptance, the K/V of accepted node path[i] (path[0] = root) moves
   to logical position ctx_len + i; nothing else in the cache changes. The
   node's K was computed at position id ctx_len + depth = ctx_len + i, so no
   re-rotation is needed.
10. Ablation presets (Sec. 5.3): "no target-aware pruning" keeps the scorer
   and selects without the cost term or threshold (lambda2 = 0, tau = 0);
   with lambda2 = 0 the utility is reach / lambda1, so Algorithm 1 fills the
   budget in descending reach. DDTree-style selection is that rule over
   marginal path probabilities.
"""
from __future__ import annotations

import math

import numpy as np

F32 = np.float32


# ---------------------------------------------------------------------------
# Stage 1: per-position marginal statistics and top-K (Sec. 4.1, Sec. 4.2)
# ---------------------------------------------------------------------------

def topk_marginals(logits: np.ndarray, K: int):
    """Top-K candidates of each drafted position, with full-vocab statistics.

    logits: [B, L, V] (exact values; bf16 inputs are passed widened).
    Returns ids [B,L,K] int32 sorted by (logit desc, id asc), logp [B,L,K]
    (= logit - lse, float64), lse [B,L], entropy [B,L] in nats (float64).
    Sec. 4.1 stage 1: the top-K tokens at each position form the candidate
    tree; Sec. 4.2: the scorer reads the child log-probability and the
    positional entropy.
    """
    x = np.asarray(logits, dtype=np.float64)
    B, L, V = x.shape
    m = x.max(axis=-1)
    Z = np.exp(x - m[..., None]).sum(axis=-1)
    lse = m + np.log(Z)
    p = np.exp(x - lse[..., None])
    # tokens of probability 0 (logit -inf) contribute 0 (the 0 log 0 = 0 convention)
    logp_all = np.where(p > 0, x - lse[..., None], 0.0)
    entropy = -(p * logp_all).sum(axis=-1)
    ids = np.empty((B, L, K), np.int32)
    for b in range(B):
        for d in range(L):
            # primary key: logit descending; secondary: token id ascending
            order = np.lexsort((np.arange(V), -x[b, d]))
            ids[b, d] = order[:K]
    logp = np.take_along_axis(x, ids.astype(np.int64), axis=-1) - lse[..., None]
    return ids, logp, lse, entropy


# ---------------------------------------------------------------------------
# Stage 2: edge scorer and sibling softmax (Sec. 4.2, Eq. 1, Algorithm 1)
# ---------------------------------------------------------------------------

def edge_logit_mlp(w: dict, parent_tok: int, child_tok: int, depth: int,
                   logp_child: float, entropy: float) -> float:
    """Scorer logit for one edge (parent -> child at edge depth ``depth``).

    Features (Sec. 4.2): parent token, child token, edge depth, child
    log-probability, positional entropy.
    """
    f = np.concatenate([
        w["tok_emb"][parent_tok].astype(np.float64),
        w["tok_emb"][child_tok].astype(np.float64),
        w["dep_emb"][depth].astype(np.float64),
        np.array([logp_child, entropy], np.float64),
    ])
    h = np.maximum(w["W1"].astype(np.float64) @ f + w["b1"].astype(np.float64), 0.0)
    return float(w["w_lp"][0]) * logp_child + float(w["w2"].astype(np.float64) @ h)


def score_qcond(root_tok, ids, logp, entropy, kind: str = "mlp", weights: dict | None = None):
    """q_cond[b, d, i, j] = Pr(accept child j of position d | reach parent i).

    Parent i is slot i of position d-1, or the root when d == 0 (row i = 0;
    rows i >= 1 at d == 0 are zero). For each parent the scorer logits of its K
    children are normalised with a sibling-wise softmax (Eq. 1, Algorithm 1).
    Kind ``marginal_product`` is the DDTree-style ranking the paper contrasts
    TAPS with (Sec. 3.1, Limitation 1: nodes chosen by the drafter's marginal
    probabilities): no scorer and no renormalisation, q = exp(logp(child)), so
    the reach of a node is the product of its path's marginal probabilities.
    Computed in float64, returned as float32.
    """
    B, L, K = ids.shape
    q = np.zeros((B, L, K, K), np.float64)
    for b in range(B):
        for d in range(L):
            parents = [int(root_tok[b])] if d == 0 else [int(t) for t in ids[b, d - 1]]
            for i, ptok in enumerate(parents):
                ell = np.empty(K, np.float64)
                for j in range(K):
                    if kind in ("marginal", "marginal_product"):
                        ell[j] = float(logp[b, d, j])
                    else:
                        ell[j] = edge_logit_mlp(weights, ptok, int(ids[b, d, j]), d + 1,
                                                float(logp[b, d, j]), float(entropy[b, d]))
                if kind == "marginal_product":
                    q[b, d, i] = np.exp(ell)
                else:
                    e = np.exp(ell - ell.max())
                    q[b, d, i] = e / e.sum()
    return q.astype(F32)


def reach_of_path(q_cond_b: np.ndarray, slots) -> float:
    """Eq. 2: q_reach(v) = product of q_cond along root -> v, in float64."""
    r = 1.0
    parent_slot = 0
    for d, j in enumerate(slots):
        r *= float(q_cond_b[d, parent_slot, j])
        parent_slot = j
    return r


def path_reach(q_cond, paths, path_len):
    """Eq. 2 for an explicit list of trie nodes, in the arithmetic that decides
    the tree: q_reach = product of q_cond along root -> node, float32 with one
    IEEE round-to-nearest multiply per edge, root to leaf (the same operations
    and order as the reach in ``select_subtree``).

    q_cond [B, L, K, K]; paths [B, M, L] top-K slots (a node at depth n is
    named by the slots of its first n edges); path_len [B, M] in [0, L].
    Returns [B, M] float32; a length of 0 is the root (reach 1). A node that
    is not in the trie (length outside [0, L], or a slot >= K among its first
    path_len entries) gets reach 0.
    """
    B, L, K, _ = q_cond.shape
    M = paths.shape[1]
    out = np.zeros((B, M), F32)
    for b in range(B):
        for m in range(M):
            n = int(path_len[b, m])
            slots = [int(j) for j in paths[b, m, :max(n, 0)]]
            if n < 0 or n > L or any(j >= K for j in slots):
                continue
            r = F32(1.0)
            parent_slot = 0                       # depth-1 children hang off the root (row 0)
            for d, j in enumerate(slots):
                r = F32(r * F32(q_cond[b, d, parent_slot, j]))
                parent_slot = j
            out[b, m] = r
    return out


# ---------------------------------------------------------------------------
# Stage 3: utility and greedy budgeted prefix-closed selection (Sec. 4.3)
# ---------------------------------------------------------------------------

def utility_denominators(lambda1: float, lambda2: float, L: int) -> np.ndarray:
    """den[d] = lambda1 + lambda2 * d in float32 (Eq. 3), d = 0..L."""
    l1, l2 = F32(lambda1), F32(lambda2)
    return np.array([F32(l1 + F32(l2 * F32(d))) for d in range(L + 1)], F32)


def _key(node: dict):
    """Total order of Algorithm 1's argmax (larger is better)."""
    return (float(node["utility"]), -node["depth"], -node["token"], -node["parent"])


def select_subtree(q_cond, ids, root_tok, ctx_len, lambda1, lambda2, tau, n_max):
    """Algorithm 1: S = {root}; while |S| < N_max and some v not in S has
    utility(v) > tau, add argmax utility and its ancestors.

    The argmax is taken over the children of S that are not in S. This is the
    same argmax as over every unselected node: utility never increases from a
    parent to its child (q_cond <= 1 and lambda2 >= 0, with monotone rounding),
    and a tie goes to the lower depth, so any unselected node is outranked by
    its highest unselected ancestor, whose parent is in S. For the same reason
    the ancestors of the argmax are already in S.

    Reach and utility are float32 with IEEE rounding, root-to-leaf order.
    Returns a dict of [B, n_max] arrays (padding -1 / 0) and n_nodes [B].
    """
    B, L, K = ids.shape
    den = utility_denominators(lambda1, lambda2, L)
    tau32 = F32(tau)
    out = {k: np.full((B, n_max), -1, np.int32) for k in ("parent", "depth", "token", "slot",
                                                          "pos_id")}
    out["reach"] = np.zeros((B, n_max), F32)
    out["utility"] = np.zeros((B, n_max), F32)
    out["n_nodes"] = np.zeros(B, np.int32)
    for b in range(B):
        root = dict(depth=0, token=int(root_tok[b]), slot=-1, parent=-1, reach=F32(1.0),
                    utility=F32(F32(1.0) / den[0]))
        S = [root]
        chosen = set()            # (parent index, slot) pairs already in S
        while len(S) < n_max:
            best = None
            for u_idx, u in enumerate(S):
                if u["depth"] == L:
                    continue
                d = u["depth"]                    # children sit at position d (depth d+1)
                prow = 0 if d == 0 else u["slot"]
                for j in range(K):
                    if (u_idx, j) in chosen:
                        continue
                    r = F32(u["reach"] * q_cond[b, d, prow, j])
                    c = dict(depth=d + 1, token=int(ids[b, d, j]), slot=j, parent=u_idx,
                             reach=r, utility=F32(r / den[d + 1]))
                    if best is None or _key(c) > _key(best):
                        best = c
            if best is None or not (best["utility"] > tau32):
                break
            chosen.add((best["parent"], best["slot"]))
            S.append(best)
        n = len(S)
        out["n_nodes"][b] = n
        for i, v in enumerate(S):
            out["parent"][b, i] = v["parent"]
            out["depth"][b, i] = v["depth"]
            out["token"][b, i] = v["token"]
            out["slot"][b, i] = v["slot"]
            out["pos_id"][b, i] = int(ctx_len[b]) + v["depth"]
            out["reach"][b, i] = v["reach"]
            out["utility"][b, i] = v["utility"]
    return out


def materialise_trie(q_cond_b, ids_b, root_token, lambda1, lambda2, L, K):
    """Every node of the candidate trie with reach and utility (Algorithm 1,
    depth loop then utility line). Tiny inputs only: K**L nodes at depth L.

    Nodes are keyed by their slot path (tuple); the root is ().
    """
    den = utility_denominators(lambda1, lambda2, L)
    nodes = {(): dict(depth=0, token=int(root_token), reach=F32(1.0),
                      utility=F32(F32(1.0) / den[0]))}
    level = [()]
    for d in range(L):
        nxt = []
        for path in level:
            prow = 0 if d == 0 else path[-1]
            for j in range(K):
                child = path + (j,)
                r = F32(nodes[path]["reach"] * q_cond_b[d, prow, j])
                nodes[child] = dict(depth=d + 1, token=int(ids_b[d, j]), reach=r,
                                    utility=F32(r / den[d + 1]))
                nxt.append(child)
        level = nxt
    return nodes


def select_subtree_literal(q_cond_b, ids_b, root_token, lambda1, lambda2, tau, n_max, L, K):
    """Algorithm 1 as printed, over the materialised trie: the argmax runs over
    every node not in S and each pick brings its ancestors. Returns the list of
    slot paths in the order they join S (ancestors before the pick).
    """
    nodes = materialise_trie(q_cond_b, ids_b, root_token, lambda1, lambda2, L, K)
    tau32 = F32(tau)
    S = [()]
    in_S = {(): 0}
    while len(S) < n_max:
        best, best_key = None, None
        for path, v in nodes.items():
            if path in in_S:
                continue
            parent_pos = in_S.get(path[:-1], 1 << 30)
            key = (float(v["utility"]), -v["depth"], -v["token"], -parent_pos)
            if best is None or key > best_key:
                best, best_key = path, key
        if best is None or not (nodes[best]["utility"] > tau32):
            break
        for k in range(1, len(best) + 1):          # ancestors(v*) then v* itself
            anc = best[:k]
            if anc not in in_S:
                in_S[anc] = len(S)
                S.append(anc)
    return S, nodes


# ---------------------------------------------------------------------------
# Stage 4: tree ancestor mask (Sec. 4.1 stage 3, Sec. 4.3)
# ---------------------------------------------------------------------------

def build_tree_mask(parent, n_nodes, n_max):
    """mask[b, i, w] bit (j % 32) of word j // 32 is set iff node j is node i or
    one of its ancestors, for i, j < n_nodes[b]; every other bit is 0."""
    B = parent.shape[0]
    W = (n_max + 31) // 32
    mask = np.zeros((B, n_max, W), np.uint32)
    for b in range(B):
        for i in range(int(n_nodes[b])):
            j = i
            while j >= 0:
                mask[b, i, j // 32] |= np.uint32(1 << (j % 32))
                j = int(parent[b, j])
    return mask


# ---------------------------------------------------------------------------
# Stage 5: tree-masked verification attention over a paged KV cache
# ---------------------------------------------------------------------------

def tree_verify_attn(q, k_cache, v_cache, block_table, ctx_len, n_nodes, mask, scale=None,
                     only=None):
    """Textbook masked softmax attention of every tree node, in float64.

    q: [B, N, Hq, D]; k_cache, v_cache: [num_pages, Hkv, P, D]; logical
    position t of request b is page block_table[b, t // P], row t % P. Node i
    attends to positions [0, ctx_len) and to ctx_len + j for every j set in
    mask[b, i]. Returns out [B, N, Hq, D] and lse [B, N, Hq] (natural log of
    the softmax denominator of the scaled scores); rows i >= n_nodes are 0.
    ``only``: optional set of (b, i, h) triples; other outputs are left 0 (a
    way to sample single outputs of a large case, same arithmetic).
    """
    q = np.asarray(q, np.float64)
    B, N, Hq, D = q.shape
    _, Hkv, P, _ = k_cache.shape
    group = Hq // Hkv
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    out = np.zeros((B, N, Hq, D), np.float64)
    lse = np.zeros((B, N, Hq), np.float64)
    for b in range(B):
        C, n = int(ctx_len[b]), int(n_nodes[b])
        if only is not None and not any(o[0] == b for o in only):
            continue
        T = C + n
        t = np.arange(T)
        pages = block_table[b, t // P]
        Kb = np.asarray(k_cache[pages, :, t % P, :], np.float64)    # [T, Hkv, D]
        Vb = np.asarray(v_cache[pages, :, t % P, :], np.float64)
        for i in range(n):
            visible = np.zeros(T, bool)
            visible[:C] = True
            for j in range(n):
                if (int(mask[b, i, j // 32]) >> (j % 32)) & 1:
                    visible[C + j] = True
            for h in range(Hq):
                if only is not None and (b, i, h) not in only:
                    continue
                kv = h // group
                s = scale * (Kb[visible, kv, :] @ q[b, i, h])
                m = s.max()
                e = np.exp(s - m)
                out[b, i, h] = (e @ Vb[visible, kv, :]) / e.sum()
                lse[b, i, h] = m + math.log(e.sum())
    return out, lse


# ---------------------------------------------------------------------------
# Stage 6: lossless greedy acceptance (Sec. 4.1, Limitations)
# ---------------------------------------------------------------------------

def accept(parent, token, n_nodes, target_tok, L):
    """Walk from the root: while some child of the current node carries the
    target's greedy token for the current node, step into it.

    Returns accept_len [B] (accepted draft tokens), accepted_nodes [B, L+1]
    (node indices root..last, padded with -1) and bonus_tok [B] (the target's
    token at the last accepted node).
    """
    B = parent.shape[0]
    accept_len = np.zeros(B, np.int32)
    nodes = np.full((B, L + 1), -1, np.int32)
    bonus = np.zeros(B, np.int32)
    for b in range(B):
        n = int(n_nodes[b])
        v = 0
        path = [0]
        while True:
            want = int(target_tok[b, v])
            nxt = [c for c in range(n) if int(parent[b, c]) == v and int(token[b, c]) == want]
            if not nxt:
                break
            v = nxt[0]
            path.append(v)
        accept_len[b] = len(path) - 1
        nodes[b, :len(path)] = path
        bonus[b] = int(target_tok[b, v])
    return accept_len, nodes, bonus


def target_greedy(verify_logits, n_nodes):
    """Target greedy token of every tree node (Limitations: temperature 0).

    verify_logits [B, n_max, V]: the target's next-token logits after the
    prefix ending at node i. Returns target_tok [B, n_max] int32: for i <
    n_nodes[b] the lowest index whose logit equals the row maximum, else -1.
    """
    x = np.asarray(verify_logits, dtype=np.float64)
    B, N, _ = x.shape
    out = np.full((B, N), -1, np.int32)
    for b in range(B):
        for i in range(int(n_nodes[b])):
            row = x[b, i]
            top = row.max()
            out[b, i] = int(np.flatnonzero(row == top)[0])
    return out


def compact_accepted_kv(k_cache, v_cache, block_table, ctx_len, accepted_nodes, accept_len,
                        page=16):
    """Move the accepted path's K/V to consecutive logical positions.

    k_cache, v_cache: logical [num_pages, Hkv, page, D] caches of one layer.
    Logical position t of request b is row t % page of page
    block_table[b, t // page]. For i = 0 .. accept_len[b], the value at
    position ctx_len[b] + accepted_nodes[b, i] (read before any write) is
    written to position ctx_len[b] + i. Returns new arrays; inputs are unchanged.
    """
    k_new = np.array(k_cache, copy=True)
    v_new = np.array(v_cache, copy=True)

    def where(b, t):
        return int(block_table[b, t // page]), t % page

    for b in range(len(ctx_len)):
        c = int(ctx_len[b])
        for i in range(int(accept_len[b]) + 1):
            sp, sr = where(b, c + int(accepted_nodes[b, i]))
            dp, dr = where(b, c + i)
            k_new[dp, :, dr, :] = k_cache[sp, :, sr, :]
            v_new[dp, :, dr, :] = v_cache[sp, :, sr, :]
    return k_new, v_new
