"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks the oracle against something other than itself: closed
forms, a hand-worked example (tests/golden/worked_round.json), brute-force
enumeration on tiny inputs, Algorithm 1 run literally over a materialised
trie, invariants implied by Eq. 1-3, and torch's scaled_dot_product_attention
as an independent route to masked attention.
"""
import itertools
import math

import numpy as np
import pytest

from oracle import taps_oracle as O
import workloads as W

F32 = np.float32


# ---------------------------------------------------------------------------
# Stage 1: marginals and top-K
# ---------------------------------------------------------------------------

def test_marginals_worked_example(golden):
    g = golden["marginals"]
    x = np.log(np.array(g["exp_logits"], np.float64))[None, None, :]
    ids, logp, lse, ent = O.topk_marginals(x, 3)
    assert ids[0, 0].tolist() == g["top3"]
    assert lse[0, 0] == pytest.approx(g["lse"], rel=1e-12)
    assert ent[0, 0] == pytest.approx(g["entropy"], rel=1e-12)
    assert np.exp(logp[0, 0]).tolist() == pytest.approx([g["probs"][i] for i in g["top3"]])


def test_marginals_uniform_closed_form():
    V = 1000
    x = np.full((1, 2, V), 3.25, np.float32)
    ids, logp, lse, ent = O.topk_marginals(x, 5)
    assert ids[0, 0].tolist() == [0, 1, 2, 3, 4]           # all tie: lower id first
    assert lse[0, 0] == pytest.approx(3.25 + math.log(V), rel=1e-13)
    assert ent[0, 1] == pytest.approx(math.log(V), rel=1e-12)
    assert logp[0, 0] == pytest.approx(np.full(5, -math.log(V)), rel=1e-12)


@pytest.mark.parametrize("a,A", [(1, 12.0), (3, 2.5), (7, -1.0)])
def test_marginals_two_level_closed_form(a, A):
    V = 777
    x = np.zeros((1, 1, V), np.float64)
    hot = [5, 100, 300, 301, 450, 600, 700][:a]
    x[0, 0, hot] = A
    ids, logp, lse, ent = O.topk_marginals(x, a + 2)
    Z = a * math.exp(A) + (V - a)
    p_hi, p_lo = math.exp(A) / Z, 1.0 / Z
    H = -a * p_hi * math.log(p_hi) - (V - a) * p_lo * math.log(p_lo)
    assert lse[0, 0] == pytest.approx(math.log(Z), rel=1e-12)
    assert ent[0, 0] == pytest.approx(H, rel=1e-10)
    if A > 0:
        expect = sorted(hot) + [i for i in range(V) if i not in hot][:2]
    else:
        expect = [i for i in range(V) if i not in hot][:a + 2]
    assert ids[0, 0].tolist() == expect


def test_marginals_minus_inf_is_probability_zero():
    """Masked tokens (logit -inf) have probability 0 and add nothing to the
    entropy: the statistics equal those of the row without them."""
    V = 300
    x = np.random.default_rng(8).standard_normal((1, 1, V))
    xm = x.copy()
    xm[0, 0, ::2] = -np.inf
    ids, logp, lse, ent = O.topk_marginals(xm, 4)
    ids2, logp2, lse2, ent2 = O.topk_marginals(x[:, :, 1::2], 4)
    assert lse[0, 0] == pytest.approx(lse2[0, 0], rel=1e-13)
    assert ent[0, 0] == pytest.approx(ent2[0, 0], rel=1e-12)
    assert (ids[0, 0] == 2 * ids2[0, 0] + 1).all()


def test_topk_brute_force_rank_with_ties():
    rng = np.random.default_rng(1)
    x = rng.integers(-3, 4, size=(2, 3, 50)).astype(np.float32)   # many exact ties
    K = 7
    ids, _, _, _ = O.topk_marginals(x, K)
    for b in range(2):
        for d in range(3):
            row = x[b, d]
            for k, t in enumerate(ids[b, d]):
                better = sum(1 for v in range(50) if row[v] > row[t] or (row[v] == row[t] and v < t))
                assert better == k


# ---------------------------------------------------------------------------
# Stage 2: scorer and sibling softmax (Eq. 1)
# ---------------------------------------------------------------------------

def _tiny_inputs(B=2, L=4, K=3, V=50, seed=0):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((B, L, V)) * 2
    ids, logp, lse, ent = O.topk_marginals(x, K)
    root = rng.integers(0, V, size=B).astype(np.int32)
    return x, ids, logp, ent, root


def _weights(V, L, E, H, seed=0, **override):
    rng = np.random.default_rng(seed)
    w = dict(tok_emb=rng.standard_normal((V, E)).astype(F32),
             dep_emb=rng.standard_normal((L + 1, E)).astype(F32),
             W1=rng.standard_normal((H, 3 * E + 2)).astype(F32),
             b1=rng.standard_normal(H).astype(F32),
             w2=rng.standard_normal(H).astype(F32),
             w_lp=np.array([1.0], F32))
    w.update(override)
    return w


def test_marginal_scorer_worked_example(golden):
    g = golden["marginal_scorer"]
    logp = np.log(np.array(g["probs"]))[None, None, :]
    ids = np.array([[[4, 5, 6]]], np.int32)
    q = O.score_qcond(np.array([0]), ids, logp, np.zeros((1, 1)), kind="marginal")
    assert q[0, 0, 0].tolist() == pytest.approx(g["q"], rel=1e-7)
    assert q[0, 0, 1:].sum() == 0.0


def test_marginal_scorer_is_renormalised_topk():
    x, ids, logp, ent, root = _tiny_inputs()
    q = O.score_qcond(root, ids, logp, ent, kind="marginal")
    p = np.exp(logp)
    expect = p / p.sum(-1, keepdims=True)
    for d in range(ids.shape[1]):
        rows = [0] if d == 0 else range(ids.shape[2])
        for i in rows:
            np.testing.assert_allclose(q[:, d, i], expect[:, d], rtol=1e-6)


def test_mlp_rows_sum_to_one():
    x, ids, logp, ent, root = _tiny_inputs()
    w = _weights(50, 4, 4, 5)
    q = O.score_qcond(root, ids, logp, ent, kind="mlp", weights=w)
    sums = q.astype(np.float64).sum(-1)
    np.testing.assert_allclose(sums[:, 1:], 1.0, atol=1e-6)
    np.testing.assert_allclose(sums[:, 0, 0], 1.0, atol=1e-6)
    assert np.all(q[:, 0, 1:] == 0)
    assert np.all(q >= 0) and np.all(q <= 1)


@pytest.mark.parametrize("block", ["parent", "depth", "entropy"])
def test_sibling_constant_features_cancel(block):
    """Features shared by all siblings (parent token, depth, entropy) alone
    shift every sibling's logit equally, so q_cond is the marginal softmax."""
    x, ids, logp, ent, root = _tiny_inputs()
    E, H = 3, 4
    W1 = np.zeros((H, 3 * E + 2), F32)
    rng = np.random.default_rng(5)
    if block == "parent":
        W1[:, 0:E] = rng.standard_normal((H, E))
    elif block == "depth":
        W1[:, 2 * E:3 * E] = rng.standard_normal((H, E))
    else:
        W1[:, 3 * E + 1] = rng.standard_normal(H)
    w = _weights(50, 4, E, H, W1=W1)
    q = O.score_qcond(root, ids, logp, ent, kind="mlp", weights=w)
    qm = O.score_qcond(root, ids, logp, ent, kind="marginal")
    np.testing.assert_allclose(q, qm, rtol=1e-6, atol=1e-7)


def test_logp_feature_closed_form():
    """H=1, only the logp column (weight -1), b1=0: relu(-logp) = -logp, so the
    logit is (w_lp - w2) * logp and q = p**(1-c) renormalised."""
    x, ids, logp, ent, root = _tiny_inputs()
    E, c = 2, 0.4
    W1 = np.zeros((1, 3 * E + 2), F32)
    W1[0, 3 * E] = -1.0
    w = _weights(50, 4, E, 1, W1=W1, b1=np.zeros(1, F32), w2=np.array([c], F32))
    q = O.score_qcond(root, ids, logp, ent, kind="mlp", weights=w)
    p = np.exp(logp) ** (1.0 - c)
    expect = p / p.sum(-1, keepdims=True)
    np.testing.assert_allclose(q[:, 1:, 0], expect[:, 1:], rtol=1e-6)
    np.testing.assert_allclose(q[:, 0, 0], expect[:, 0], rtol=1e-6)


def test_child_feature_independent_of_parent():
    """Only the child-embedding block: every parent row of a position is equal
    and the root token does not matter."""
    x, ids, logp, ent, root = _tiny_inputs()
    E, H = 3, 4
    W1 = np.zeros((H, 3 * E + 2), F32)
    W1[:, E:2 * E] = np.random.default_rng(2).standard_normal((H, E))
    w = _weights(50, 4, E, H, W1=W1)
    q = O.score_qcond(root, ids, logp, ent, kind="mlp", weights=w)
    for d in range(1, 4):
        for i in range(1, 3):
            np.testing.assert_array_equal(q[:, d, i], q[:, d, 0])
    q2 = O.score_qcond((root + 1) % 50, ids, logp, ent, kind="mlp", weights=w)
    np.testing.assert_array_equal(q, q2)
    qm = O.score_qcond(root, ids, logp, ent, kind="marginal")
    assert np.abs(q - qm).max() > 1e-3          # the child feature does change q


def test_depth_embedding_index_is_edge_depth():
    """E=1, H=1: relu(E_dep[depth] + E_tok[child]) is active only at one
    chosen edge depth; only that position departs from the marginal softmax."""
    x, ids, logp, ent, root = _tiny_inputs(L=4)
    E, delta = 1, 3                                  # edge depth 3 = position index 2
    dep = np.full((5, 1), -100.0, F32)
    dep[delta, 0] = 0.0
    tok = np.random.default_rng(3).uniform(0.5, 3.0, size=(50, 1)).astype(F32)
    W1 = np.zeros((1, 3 * E + 2), F32)
    W1[0, E] = 1.0          # child embedding
    W1[0, 2 * E] = 1.0      # depth embedding
    w = _weights(50, 4, E, 1, tok_emb=tok, dep_emb=dep, W1=W1, b1=np.zeros(1, F32),
                 w2=np.array([1.0], F32))
    q = O.score_qcond(root, ids, logp, ent, kind="mlp", weights=w)
    qm = O.score_qcond(root, ids, logp, ent, kind="marginal")
    for d in range(4):
        diff = np.abs(q[:, d] - qm[:, d]).max()
        if d == delta - 1:
            assert diff > 1e-3
        else:
            assert diff < 1e-6


def test_entropy_feature_is_the_child_position():
    """E=1, H=1: relu(E_tok[child] + H) with a different entropy H at each
    position. Position d's rows are then softmax(relu(e_child + H[d])) over
    the siblings, a closed form that fixes which position's entropy enters."""
    L = 3
    ids = np.array([[[0, 1, 2]] * L], np.int32)
    e = np.array([0.0, -1.0, -2.0])
    tok = np.zeros((50, 1), F32)
    tok[:3, 0] = e
    ent = np.array([[0.0, 1.5, 3.0]])
    W1 = np.zeros((1, 3 * 1 + 2), F32)
    W1[0, 1] = 1.0          # child embedding
    W1[0, 4] = 1.0          # positional entropy
    w = _weights(50, L, 1, 1, tok_emb=tok, W1=W1, b1=np.zeros(1, F32),
                 w2=np.array([1.0], F32), w_lp=np.array([0.0], F32))
    q = O.score_qcond(np.array([7]), ids, np.zeros((1, L, 3)), ent, kind="mlp", weights=w)
    for d in range(L):
        h = np.maximum(e + ent[0, d], 0.0)
        expect = np.exp(h) / np.exp(h).sum()
        rows = [0] if d == 0 else range(3)
        for i in rows:
            np.testing.assert_allclose(q[0, d, i], expect, rtol=1e-6)
    assert np.abs(q[0, 1, 0] - q[0, 2, 0]).max() > 1e-2     # the positions do differ


def test_parent_token_enters_through_interaction():
    """E=1, H=1: relu(E_tok[parent] + E_tok[child] - 5) is non-zero only under
    one chosen parent token; rows of other parents equal the marginal."""
    x, ids, logp, ent, root = _tiny_inputs(B=1, L=3, K=3)
    special = int(ids[0, 0, 1])                      # slot 1 of position 0
    tok = np.zeros((50, 1), F32)
    tok[special, 0] = 5.0
    tok[:, 0] += np.random.default_rng(4).uniform(0.1, 1.0, size=50).astype(F32)
    tok[special, 0] = 5.0
    W1 = np.zeros((1, 3 * 1 + 2), F32)
    W1[0, 0] = 1.0
    W1[0, 1] = 1.0
    w = _weights(50, 3, 1, 1, tok_emb=tok, W1=W1, b1=np.array([-5.0], F32),
                 w2=np.array([1.0], F32))
    if int(root[0]) == special:
        root = (root + 1) % 50
    q = O.score_qcond(root, ids, logp, ent, kind="mlp", weights=w)
    qm = O.score_qcond(root, ids, logp, ent, kind="marginal")
    assert np.abs(q[0, 1, 1] - qm[0, 1, 1]).max() > 1e-3   # parent = special token
    np.testing.assert_allclose(q[0, 1, 0], qm[0, 1, 0], rtol=1e-6)
    np.testing.assert_allclose(q[0, 1, 2], qm[0, 1, 2], rtol=1e-6)


# ---------------------------------------------------------------------------
# Stage 3: reach, utility and greedy selection (Eq. 2, Eq. 3, Algorithm 1)
# ---------------------------------------------------------------------------

def _golden_select(golden, n_max):
    q = np.array(golden["q_cond"], F32)[None]
    ids = np.array(golden["ids"], np.int32)[None]
    return O.select_subtree(q, ids, np.array([golden["root_tok"]]), np.array([golden["ctx_len"]]),
                            golden["lambda1"], golden["lambda2"], golden["tau"], n_max)


@pytest.mark.parametrize("case", [0, 1])
def test_select_worked_example(golden, case):
    c = golden["cases"][case]
    s = _golden_select(golden, c["n_max"])
    n = c["n_nodes"]
    assert s["n_nodes"][0] == n
    for k in ("parent", "depth", "token", "slot", "pos_id"):
        assert s[k][0, :n].tolist() == c[k], k
        assert np.all(s[k][0, n:] == -1)
    np.testing.assert_allclose(s["reach"][0, :n], c["reach"], rtol=1e-7)
    np.testing.assert_allclose(s["utility"][0, :n], c["utility"], rtol=1e-7)


def test_mask_and_accept_worked_example(golden):
    c = golden["cases"][1]
    s = _golden_select(golden, c["n_max"])
    mask = O.build_tree_mask(s["parent"], s["n_nodes"], c["n_max"])
    assert mask[0, :c["n_nodes"], 0].tolist() == c["mask_rows"]
    assert np.all(mask[0, c["n_nodes"]:] == 0)
    y = np.array([c["target_seq"]], np.int32)
    tt = W.target_tokens_for_tree(y, s["depth"], s["n_nodes"])
    alen, nodes, bonus = O.accept(s["parent"], s["token"], s["n_nodes"], tt, golden["L"])
    assert alen[0] == c["accept_len"]
    assert nodes[0, :alen[0] + 1].tolist() == c["accepted_nodes"]
    assert bonus[0] == c["bonus_tok"]


def _random_qcond(rng, L, K, ties=False):
    if ties:
        # few distinct probabilities -> many exact utility ties
        raw = rng.choice([1.0, 2.0, 4.0], size=(L, K, K))
    else:
        raw = rng.random((L, K, K)) + 0.05
    q = (raw / raw.sum(-1, keepdims=True)).astype(F32)
    q[0, 1:] = 0
    return q


def _check_tree_invariants(s, b, ids, root_tok, ctx_len, n_max, L):
    n = int(s["n_nodes"][b])
    assert 1 <= n <= n_max
    assert s["parent"][b, 0] == -1 and s["depth"][b, 0] == 0 and s["token"][b, 0] == root_tok
    seen = set()
    for i in range(1, n):
        p = int(s["parent"][b, i])
        assert 0 <= p < i
        d = int(s["depth"][b, i])
        assert d == s["depth"][b, p] + 1 and d <= L
        j = int(s["slot"][b, i])
        assert s["token"][b, i] == ids[b, d - 1, j]
        assert (p, j) not in seen
        seen.add((p, j))
        assert s["pos_id"][b, i] == ctx_len + d
    # greedy order: keys never increase
    util = s["utility"][b, :n]
    assert np.all(util[1:] <= util[:-1])


@pytest.mark.parametrize("seed", range(12))
def test_frontier_equals_literal_algorithm1(seed):
    rng = np.random.default_rng(100 + seed)
    L, K = [(3, 2), (2, 3), (4, 2), (3, 3)][seed % 4]
    ties = seed % 2 == 1
    q = _random_qcond(rng, L, K, ties)[None]
    ids = np.stack([rng.permutation(20)[:K] for _ in range(L)]).astype(np.int32)[None]
    trie_size = sum(K ** d for d in range(L + 1))
    lam2 = [0.0, 0.3][seed % 2]
    for n_max in (1, 2, 5, trie_size // 2, trie_size, trie_size + 3):
        for tau in (0.0, 0.05):
            s = O.select_subtree(q, ids, np.array([3]), np.array([10]), 1.0, lam2, tau, n_max)
            lit, _ = O.select_subtree_literal(q[0], ids[0], 3, 1.0, lam2, tau, n_max, L, K)
            n = int(s["n_nodes"][0])
            assert n == len(lit)
            # rebuild slot paths of the frontier result
            paths = [()]
            for i in range(1, n):
                paths.append(paths[int(s["parent"][0, i])] + (int(s["slot"][0, i]),))
            assert paths == lit
            _check_tree_invariants(s, 0, ids, 3, 10, n_max, L)


@pytest.mark.parametrize("seed", range(12))
def test_algorithm1_is_the_top_n_of_the_trie(seed):
    """Algorithm 1 adds nodes in descending key order, so its result is the
    n_max largest nodes of the whole trie (utility > tau) under the key order
    utility desc, depth asc, token asc, then the parents' own order (Eq. 3 and
    the argmax of Algorithm 1): a plain sort of the materialised trie must give
    the same nodes in the same order. Half the cases carry exact utility ties."""
    import functools
    rng = np.random.default_rng(300 + seed)
    L, K = [(3, 2), (2, 3), (4, 2), (3, 3)][seed % 4]
    ties = seed % 2 == 1
    q = _random_qcond(rng, L, K, ties)[None]
    ids = np.stack([rng.permutation(20)[:K] for _ in range(L)]).astype(np.int32)[None]
    lam2 = [0.0, 0.3, 0.1][seed % 3]
    nodes = O.materialise_trie(q[0], ids[0], 3, 1.0, lam2, L, K)

    def cmp(a, b):
        if a == b:
            return 0
        ua, ub = float(nodes[a]["utility"]), float(nodes[b]["utility"])
        if ua != ub:
            return -1 if ua > ub else 1
        if len(a) != len(b):
            return -1 if len(a) < len(b) else 1
        ta, tb = nodes[a]["token"], nodes[b]["token"]
        if ta != tb:
            return -1 if ta < tb else 1
        return cmp(a[:-1], b[:-1])

    for tau in (0.0, 0.05):
        alive = [p for p in nodes if p == () or nodes[p]["utility"] > np.float32(tau)]
        ranked = sorted(alive, key=functools.cmp_to_key(cmp))
        for n_max in (1, 3, len(nodes) // 3, len(nodes)):
            s = O.select_subtree(q, ids, np.array([3]), np.array([10]), 1.0, lam2, tau, n_max)
            n = int(s["n_nodes"][0])
            paths = [()]
            for i in range(1, n):
                paths.append(paths[int(s["parent"][0, i])] + (int(s["slot"][0, i]),))
            assert paths == ranked[:n_max]


def _prefix_closed_subsets(all_paths, size):
    nonroot = [p for p in all_paths if p != ()]
    for combo in itertools.combinations(nonroot, size - 1):
        sset = set(combo) | {()}
        if all(p[:-1] in sset for p in combo):
            yield sset


@pytest.mark.parametrize("seed", range(6))
def test_brute_force_subtree_enumeration(seed):
    """Among all prefix-closed subtrees of the same size, the selected one has
    the largest total utility and the lexicographically largest sorted
    utility vector."""
    rng = np.random.default_rng(200 + seed)
    L, K = [(3, 2), (2, 3)][seed % 2]
    q = _random_qcond(rng, L, K, ties=seed >= 4)[None]
    ids = np.stack([rng.permutation(20)[:K] for _ in range(L)]).astype(np.int32)[None]
    nodes = O.materialise_trie(q[0], ids[0], 3, 1.0, 0.25, L, K)
    for n_max in range(2, 8):
        s = O.select_subtree(q, ids, np.array([3]), np.array([0]), 1.0, 0.25, 0.0, n_max)
        n = int(s["n_nodes"][0])
        paths = [()]
        for i in range(1, n):
            paths.append(paths[int(s["parent"][0, i])] + (int(s["slot"][0, i]),))
        sel_util = sorted((float(nodes[p]["utility"]) for p in paths), reverse=True)
        best_total = -1.0
        best_vec = None
        for sset in _prefix_closed_subsets(list(nodes), n):
            u = sorted((float(nodes[p]["utility"]) for p in sset), reverse=True)
            best_total = max(best_total, math.fsum(u))
            best_vec = u if best_vec is None or u > best_vec else best_vec
        assert math.fsum(sel_util) == pytest.approx(best_total, rel=1e-12)
        assert sel_util == best_vec


@pytest.mark.parametrize("seed", range(4))
def test_reach_is_product_of_qcond(seed):
    rng = np.random.default_rng(300 + seed)
    L, K = 6, 4
    q = _random_qcond(rng, L, K)[None]
    ids = np.stack([rng.permutation(100)[:K] for _ in range(L)]).astype(np.int32)[None]
    s = O.select_subtree(q, ids, np.array([1]), np.array([0]), 1.0, 0.1, 0.0, 200)
    n = int(s["n_nodes"][0])
    paths = [()]
    for i in range(1, n):
        paths.append(paths[int(s["parent"][0, i])] + (int(s["slot"][0, i]),))
        exact = O.reach_of_path(q[0].astype(np.float64), paths[-1])
        assert s["reach"][0, i] == pytest.approx(exact, rel=1e-6)
        den = 1.0 + 0.1 * len(paths[-1])
        assert s["utility"][0, i] == pytest.approx(exact / den, rel=1e-6)


def test_path_reach_hand_worked():
    """Eq. 2 on a two-level trie whose q_cond values are exact in float32:
    every product is exact, and a wrong parent row or a transposed q_cond
    index changes the (1, 0) and (0, 1) entries."""
    q = np.zeros((1, 2, 2, 2), F32)
    q[0, 0, 0] = [0.75, 0.25]           # depth-1 children of the root (row 0)
    q[0, 1, 0] = [0.5, 0.5]             # children of slot 0
    q[0, 1, 1] = [0.125, 0.875]         # children of slot 1
    cases = {(): 1.0, (0,): 0.75, (1,): 0.25, (0, 0): 0.375, (0, 1): 0.375,
             (1, 0): 0.03125, (1, 1): 0.21875}
    paths = np.zeros((1, len(cases) + 3, 2), np.uint8)
    plen = np.zeros((1, len(cases) + 3), np.int32)
    for m, path in enumerate(cases):
        paths[0, m, :len(path)] = path
        plen[0, m] = len(path)
    m0 = len(cases)
    paths[0, m0] = [2, 0]; plen[0, m0] = 1            # slot 2 >= K: not a node
    paths[0, m0 + 1] = [0, 0]; plen[0, m0 + 1] = 3    # deeper than L: not a node
    paths[0, m0 + 2] = [1, 2]; plen[0, m0 + 2] = 1    # the bad slot lies past the length
    r = O.path_reach(q, paths, plen)
    assert r.dtype == F32
    assert r[0, :m0].tolist() == list(cases.values())
    assert r[0, m0:].tolist() == [0.0, 0.0, 0.25]


@pytest.mark.parametrize("seed", range(3))
def test_path_reach_within_rounding_of_exact_product(seed):
    """float32, one rounding per edge: within L * 2^-24 (relative) of the
    float64 product of the same q_cond values."""
    rng = np.random.default_rng(500 + seed)
    B, L, K, M = 2, 12, 5, 40
    q = np.stack([_random_qcond(rng, L, K) for _ in range(B)])
    paths = rng.integers(0, K, size=(B, M, L)).astype(np.uint8)
    plen = rng.integers(0, L + 1, size=(B, M)).astype(np.int32)
    r = O.path_reach(q, paths, plen)
    for b in range(B):
        for m in range(M):
            exact = O.reach_of_path(q[b].astype(np.float64), paths[b, m, :plen[b, m]].tolist())
            assert abs(float(r[b, m]) - exact) <= L * 2.0 ** -24 * exact * 1.0001


def test_path_reach_equals_the_selected_tree_reach():
    """The reach that decides the tree (select_subtree, built parent to child)
    and path_reach of each selected node's slot path are the same float32
    operations in the same order: bit-identical."""
    rng = np.random.default_rng(77)
    B, L, K = 2, 7, 4
    q = np.stack([_random_qcond(rng, L, K) for _ in range(B)])
    ids = np.stack([np.stack([rng.permutation(100)[:K] for _ in range(L)])
                    for _ in range(B)]).astype(np.int32)
    s = O.select_subtree(q, ids, np.array([1, 2]), np.array([0, 0]), 1.0, 0.1, 0.0, 90)
    paths = np.zeros((B, 90, L), np.uint8)
    plen = np.zeros((B, 90), np.int32)
    for b in range(B):
        walk = [()]
        for i in range(1, int(s["n_nodes"][b])):
            walk.append(walk[int(s["parent"][b, i])] + (int(s["slot"][b, i]),))
            paths[b, i, :len(walk[-1])] = walk[-1]
            plen[b, i] = len(walk[-1])
    r = O.path_reach(q, paths, plen)
    for b in range(B):
        n = int(s["n_nodes"][b])
        assert r[b, :n].view(np.uint32).tolist() == s["reach"][b, :n].view(np.uint32).tolist()


def test_children_reach_sums_to_parent_reach():
    rng = np.random.default_rng(7)
    L, K = 3, 3
    q = _random_qcond(rng, L, K)[None]
    ids = np.stack([rng.permutation(100)[:K] for _ in range(L)]).astype(np.int32)[None]
    full = sum(K ** d for d in range(L + 1))
    s = O.select_subtree(q, ids, np.array([1]), np.array([0]), 1.0, 0.1, 0.0, full)
    assert s["n_nodes"][0] == full                      # tau = 0: the whole trie
    n = full
    for v in range(n):
        kids = [c for c in range(n) if s["parent"][0, c] == v]
        if kids:
            assert len(kids) == K
            tot = math.fsum(float(s["reach"][0, c]) for c in kids)
            assert tot == pytest.approx(float(s["reach"][0, v]), rel=1e-6)


def test_chain_when_k_is_one():
    """K = 1 is single-path verification (DFlash): a chain of min(L, N-1) nodes."""
    L = 6
    q = np.ones((1, L, 1, 1), F32)
    ids = np.arange(L, dtype=np.int32).reshape(1, L, 1) + 10
    for n_max in (1, 3, 7, 12):
        s = O.select_subtree(q, ids, np.array([0]), np.array([5]), 1.0, 0.2, 0.0, n_max)
        n = int(s["n_nodes"][0])
        assert n == min(L, n_max - 1) + 1
        assert s["parent"][0, :n].tolist() == [-1] + list(range(n - 1))
        assert s["token"][0, 1:n].tolist() == list(range(10, 10 + n - 1))


@pytest.mark.parametrize("c", [2.0, 0.25])
def test_utility_scales_with_the_cost_weights(c):
    """Eq. 3 is homogeneous: multiplying lambda1 and lambda2 by c divides every
    utility by c, so with tau divided by c the same tree is selected. For c a
    power of two every IEEE operation scales exactly, so the scaled run is
    bit-identical up to the factor; the root's utility is 1 / lambda1."""
    rng = np.random.default_rng(21)
    L, K = 5, 3
    q = _random_qcond(rng, L, K)[None]
    ids = np.stack([rng.permutation(30)[:K] for _ in range(L)]).astype(np.int32)[None]
    root, ctx = np.array([2]), np.array([50])
    a = O.select_subtree(q, ids, root, ctx, 1.0, 0.1, 0.05, 40)
    b = O.select_subtree(q, ids, root, ctx, 1.0 * c, 0.1 * c, 0.05 / c, 40)
    for k in ("n_nodes", "parent", "depth", "token", "slot", "pos_id", "reach"):
        np.testing.assert_array_equal(a[k], b[k])
    n = int(a["n_nodes"][0])
    assert 1 < n < 40
    np.testing.assert_array_equal(b["utility"][0, :n], (a["utility"][0, :n] / F32(c)).astype(F32))
    assert b["utility"][0, 0] == F32(1.0 / c)


def test_threshold_stops_selection():
    rng = np.random.default_rng(9)
    q = _random_qcond(rng, 4, 3)[None]
    ids = np.stack([rng.permutation(30)[:3] for _ in range(4)]).astype(np.int32)[None]
    s = O.select_subtree(q, ids, np.array([0]), np.array([0]), 2.0, 0.1, 0.5, 50)
    assert s["n_nodes"][0] == 1                           # every child utility <= 1/2.1 < 0.5
    s = O.select_subtree(q, ids, np.array([0]), np.array([0]), 1.0, 0.1, 0.02, 100)
    n = int(s["n_nodes"][0])
    assert np.all(s["utility"][0, 1:n] > F32(0.02))
    nodes = O.materialise_trie(q[0], ids[0], 0, 1.0, 0.1, 4, 3)
    passing = sum(1 for p, v in nodes.items() if p != () and v["utility"] > F32(0.02))
    assert n == 1 + passing                               # adaptive tree size


# ---------------------------------------------------------------------------
# Stage 4: mask
# ---------------------------------------------------------------------------

def test_mask_invariants():
    rng = np.random.default_rng(11)
    q = _random_qcond(rng, 5, 3)[None]
    ids = np.stack([rng.permutation(30)[:3] for _ in range(5)]).astype(np.int32)[None]
    n_max = 70
    s = O.select_subtree(q, ids, np.array([0]), np.array([0]), 1.0, 0.1, 0.0, n_max)
    m = O.build_tree_mask(s["parent"], s["n_nodes"], n_max)
    n = int(s["n_nodes"][0])
    for i in range(n):
        bits = [(int(m[0, i, j // 32]) >> (j % 32)) & 1 for j in range(n_max)]
        assert sum(bits) == s["depth"][0, i] + 1
        assert bits[i] == 1 and not any(bits[i + 1:])
        if i:
            p = int(s["parent"][0, i])
            pb = [(int(m[0, p, j // 32]) >> (j % 32)) & 1 for j in range(n_max)]
            assert [a | (k == i) for k, a in enumerate(pb)] == bits


# ---------------------------------------------------------------------------
# Stage 5: attention
# ---------------------------------------------------------------------------

def _attn_case(seed, n, Hq=4, Hkv=2, D=16, C=37, P=16, parents=None, zero_q=False):
    rng = np.random.default_rng(seed)
    n_max = n + 2
    need = (C + n_max + P - 1) // P
    num_pages = need + 2
    bt = rng.permutation(num_pages)[:need].astype(np.int32)[None]
    k = rng.standard_normal((num_pages, Hkv, P, D))
    v = rng.standard_normal((num_pages, Hkv, P, D))
    q = np.zeros((1, n_max, Hq, D)) if zero_q else rng.standard_normal((1, n_max, Hq, D))
    if parents is None:
        parents = [-1] + [int(rng.integers(0, i)) for i in range(1, n)]
    parent = np.full((1, n_max), -1, np.int32)
    parent[0, :n] = parents
    nn = np.array([n], np.int32)
    mask = O.build_tree_mask(parent, nn, n_max)
    return q, k, v, bt, np.array([C], np.int32), nn, mask


def _sdpa_reference(q, k, v, bt, ctx, nn, mask):
    torch = pytest.importorskip("torch")
    B, N, Hq, D = q.shape
    _, Hkv, P, _ = k.shape
    C, n = int(ctx[0]), int(nn[0])
    t = np.arange(C + n)
    Kb = torch.from_numpy(k[bt[0, t // P], :, t % P, :]).permute(1, 0, 2)   # [Hkv, T, D]
    Vb = torch.from_numpy(v[bt[0, t // P], :, t % P, :]).permute(1, 0, 2)
    Kb = Kb.repeat_interleave(Hq // Hkv, 0)
    Vb = Vb.repeat_interleave(Hq // Hkv, 0)
    allowed = torch.zeros(n, C + n, dtype=torch.bool)
    allowed[:, :C] = True
    for i in range(n):
        for j in range(n):
            allowed[i, C + j] = bool((int(mask[0, i, j // 32]) >> (j % 32)) & 1)
    Q = torch.from_numpy(q[0, :n]).permute(1, 0, 2)                         # [Hq, n, D]
    out = torch.nn.functional.scaled_dot_product_attention(Q, Kb, Vb, attn_mask=allowed)
    return out.permute(1, 0, 2).numpy()


@pytest.mark.parametrize("seed,n,parents", [(0, 1, [-1]), (1, 6, [-1, 0, 1, 2, 3, 4]),
                                            (2, 9, None), (3, 20, None)])
def test_attention_matches_sdpa(seed, n, parents):
    q, k, v, bt, ctx, nn, mask = _attn_case(seed, n, parents=parents)
    out, lse = O.tree_verify_attn(q, k, v, bt, ctx, nn, mask)
    ref = _sdpa_reference(q, k, v, bt, ctx, nn, mask)
    np.testing.assert_allclose(out[0, :n], ref, rtol=1e-10, atol=1e-12)
    assert np.all(out[0, n:] == 0)


def test_attention_zero_query_is_mean_of_visible_values():
    q, k, v, bt, ctx, nn, mask = _attn_case(4, 5, zero_q=True, parents=[-1, 0, 0, 1, 3])
    out, lse = O.tree_verify_attn(q, k, v, bt, ctx, nn, mask)
    C, P = int(ctx[0]), k.shape[2]
    anc = {0: [0], 1: [0, 1], 2: [0, 2], 3: [0, 1, 3], 4: [0, 1, 3, 4]}
    for i, a in anc.items():
        pos = list(range(C)) + [C + j for j in a]
        for h in range(4):
            rows = np.stack([v[bt[0, t // P], h // 2, t % P] for t in pos])
            np.testing.assert_allclose(out[0, i, h], rows.mean(0), rtol=1e-12)
            assert lse[0, i, h] == pytest.approx(math.log(len(pos)), rel=1e-12)


def test_attention_identical_keys_closed_form():
    """Every key of a KV head is the same vector k_h: all visible scores of a
    query equal s = q.k_h / sqrt(D), so the softmax is uniform (the output is
    the mean of the visible values) and lse = s + log(number visible)."""
    q, k, v, bt, ctx, nn, mask = _attn_case(6, 5, parents=[-1, 0, 0, 1, 3])
    rng = np.random.default_rng(60)
    kvec = rng.standard_normal((k.shape[1], k.shape[3]))
    k = np.broadcast_to(kvec[None, :, None, :], k.shape).copy()
    q = 3.0 * q
    out, lse = O.tree_verify_attn(q, k, v, bt, ctx, nn, mask)
    C, P, D = int(ctx[0]), k.shape[2], k.shape[3]
    anc = {0: [0], 1: [0, 1], 2: [0, 2], 3: [0, 1, 3], 4: [0, 1, 3, 4]}
    for i, a in anc.items():
        pos = list(range(C)) + [C + j for j in a]
        for h in range(4):
            s = float(q[0, i, h] @ kvec[h // 2]) / math.sqrt(D)
            assert abs(s) > 0.1
            assert lse[0, i, h] == pytest.approx(s + math.log(len(pos)), rel=1e-12, abs=1e-12)
            rows = np.stack([v[bt[0, t // P], h // 2, t % P] for t in pos])
            np.testing.assert_allclose(out[0, i, h], rows.mean(0), rtol=1e-10, atol=1e-12)


def test_attention_page_placement_invariance():
    q, k, v, bt, ctx, nn, mask = _attn_case(5, 7)
    out1, _ = O.tree_verify_attn(q, k, v, bt, ctx, nn, mask)
    perm = np.random.default_rng(0).permutation(k.shape[0])
    inv = np.argsort(perm)
    out2, _ = O.tree_verify_attn(q, k[perm], v[perm], inv[bt].astype(np.int32), ctx, nn, mask)
    np.testing.assert_allclose(out1, out2, rtol=1e-13)


# ---------------------------------------------------------------------------
# Stage 6: acceptance walk
# ---------------------------------------------------------------------------

def _brute_force_accept(parent, token, n, target_tok):
    best = 0
    for v in range(n):
        ok, a = True, v
        while a > 0:
            if token[a] != target_tok[parent[a]]:
                ok = False
                break
            a = parent[a]
        if ok and (best == 0 or _depth(parent, v) > _depth(parent, best)):
            best = v
    return best


def _depth(parent, v):
    d = 0
    while parent[v] >= 0:
        v, d = parent[v], d + 1
    return d


@pytest.mark.parametrize("seed", range(8))
def test_accept_brute_force(seed):
    rng = np.random.default_rng(400 + seed)
    L, K = 5, 3
    q = _random_qcond(rng, L, K)[None]
    ids = np.stack([rng.permutation(6)[:K] for _ in range(L)]).astype(np.int32)[None]
    s = O.select_subtree(q, ids, np.array([0]), np.array([0]), 1.0, 0.1, 0.0, 40)
    n = int(s["n_nodes"][0])
    y = rng.integers(0, 6, size=(1, L + 1)).astype(np.int32)
    tt = W.target_tokens_for_tree(y, s["depth"], s["n_nodes"])
    alen, nodes, bonus = O.accept(s["parent"], s["token"], s["n_nodes"], tt, L)
    last = _brute_force_accept(s["parent"][0], s["token"][0], n, tt[0])
    assert nodes[0, alen[0]] == last
    assert alen[0] == _depth(s["parent"][0], last)
    # accepted draft tokens + bonus = the target's greedy continuation
    toks = [int(s["token"][0, v]) for v in nodes[0, 1:alen[0] + 1]] + [int(bonus[0])]
    assert toks == y[0, :alen[0] + 1].tolist()


@pytest.mark.parametrize("seed", range(8))
def test_accept_brute_force_per_node_targets(seed):
    """The target's greedy token at a node depends on the node's whole prefix,
    so two nodes of the same depth can want different tokens: random target
    tokens per node, checked against brute force over root paths."""
    rng = np.random.default_rng(450 + seed)
    L, K, A, n_max = 5, 3, 4, 40
    q = _random_qcond(rng, L, K)[None]
    ids = np.stack([rng.permutation(A)[:K] for _ in range(L)]).astype(np.int32)[None]
    s = O.select_subtree(q, ids, np.array([0]), np.array([0]), 1.0, 0.1, 0.0, n_max)
    n = int(s["n_nodes"][0])
    tt = np.full((1, n_max), -1, np.int32)
    tt[0, :n] = rng.integers(0, A, size=n)
    alen, nodes, bonus = O.accept(s["parent"], s["token"], s["n_nodes"], tt, L)
    last = _brute_force_accept(s["parent"][0], s["token"][0], n, tt[0])
    chain = [last]
    while chain[-1] != 0:
        chain.append(int(s["parent"][0, chain[-1]]))
    assert alen[0] == len(chain) - 1
    assert nodes[0, :len(chain)].tolist() == chain[::-1]
    assert np.all(nodes[0, len(chain):] == -1)
    assert bonus[0] == tt[0, last]


def test_accept_chain_is_longest_prefix_match():
    L = 6
    parent = np.array([[-1, 0, 1, 2, 3, 4, 5]], np.int32)
    token = np.array([[9, 1, 2, 3, 4, 5, 6]], np.int32)
    for y, expect in (([1, 2, 3, 7, 0, 0, 0], 3), ([5, 0, 0, 0, 0, 0, 0], 0),
                      ([1, 2, 3, 4, 5, 6, 8], 6)):
        y = np.array([y], np.int32)
        depth = np.arange(7, dtype=np.int32)[None]
        tt = W.target_tokens_for_tree(y, depth, np.array([7]))
        alen, nodes, bonus = O.accept(parent, token, np.array([7]), tt, L)
        assert alen[0] == expect
        assert bonus[0] == y[0, expect]


# ---------------------------------------------------------------------------
# Target greedy token (temperature 0) and the accepted path's K/V compaction
# ---------------------------------------------------------------------------

def _first_max_python(row):
    best = 0
    for i in range(1, len(row)):
        if float(row[i]) > float(row[best]):
            best = i
    return best


@pytest.mark.parametrize("seed", range(4))
def test_target_greedy_brute_force_with_ties(seed):
    rng = np.random.default_rng(700 + seed)
    B, N, V = 2, 5, 40
    # few distinct values, so most rows have tied maxima
    x = rng.integers(-3, 3, size=(B, N, V)).astype(np.float32)
    x[0, 1] = -np.inf
    x[0, 1, 17] = -0.0
    x[0, 1, 23] = 0.0                      # -0.0 == +0.0: index 17 wins
    x[1, 2] = -np.inf                      # all -inf: index 0
    n_nodes = np.array([5, 3], np.int32)
    t = O.target_greedy(x, n_nodes)
    for b in range(B):
        for i in range(N):
            want = _first_max_python(x[b, i]) if i < n_nodes[b] else -1
            assert t[b, i] == want, (b, i)
    assert t[0, 1] == 17 and t[1, 2] == 0


def test_target_greedy_planted_spike_gives_target_tokens():
    """Verify logits whose row i peaks at y[depth(i)] reproduce the tree's target tokens."""
    rng = np.random.default_rng(11)
    L, K, V = 5, 3, 64
    q = _random_qcond(rng, L, K)[None]
    ids = np.stack([rng.permutation(V)[:K] for _ in range(L)]).astype(np.int32)[None]
    s = O.select_subtree(q, ids, np.array([0]), np.array([0]), 1.0, 0.1, 0.0, 24)
    y = rng.integers(0, V, size=(1, L + 1)).astype(np.int32)
    tt = W.target_tokens_for_tree(y, s["depth"], s["n_nodes"])
    x = rng.standard_normal((1, 24, V)).astype(np.float32)
    n = int(s["n_nodes"][0])
    for i in range(n):
        x[0, i, tt[0, i]] = 50.0
    got = O.target_greedy(x, s["n_nodes"])
    assert (got[0, :n] == tt[0, :n]).all() and (got[0, n:] == -1).all()


def _labelled_cache(num_pages, Hkv=2, D=4, page=16):
    """Cache whose entry at (page p, head h, row r, dim d) encodes all four."""
    p, h, r, d = np.meshgrid(np.arange(num_pages), np.arange(Hkv), np.arange(page),
                             np.arange(D), indexing="ij")
    return (p * 100000 + h * 10000 + r * 100 + d).astype(np.float64)


def test_compact_chain_path_is_identity():
    bt = np.array([[3, 0, 2, 1]], np.int32)
    k = _labelled_cache(4)
    v = -k
    path = np.array([[0, 1, 2, 3, 4, 5]], np.int32)
    kn, vn = O.compact_accepted_kv(k, v, bt, np.array([20]), path, np.array([5]))
    assert (kn == k).all() and (vn == v).all()


@pytest.mark.parametrize("seed", range(4))
def test_compact_moves_each_accepted_row_and_nothing_else(seed):
    rng = np.random.default_rng(900 + seed)
    B, L, page = 3, 6, 16
    ctx = np.array([5, 30, 16], np.int32)
    n_tree = 40
    need = (ctx + n_tree + page - 1) // page
    perm = rng.permutation(int(need.sum()) + 2).astype(np.int32)
    bt = np.full((B, int(need.max())), -1, np.int32)
    o = 0
    for b in range(B):
        bt[b, :need[b]] = perm[o:o + need[b]]
        o += int(need[b])
    k = _labelled_cache(len(perm))
    v = k + 0.5
    alen = rng.integers(0, L + 1, size=B).astype(np.int32)
    path = np.full((B, L + 1), -1, np.int32)
    for b in range(B):
        steps = np.sort(rng.choice(np.arange(1, n_tree), size=alen[b], replace=False))
        path[b, :alen[b] + 1] = np.concatenate([[0], steps])
    kn, vn = O.compact_accepted_kv(k, v, bt, ctx, path, alen)

    def at(c, b, t):
        return c[bt[b, t // page], :, t % page, :]

    touched = set()
    for b in range(B):
        for i in range(alen[b] + 1):
            dst, src = ctx[b] + i, ctx[b] + path[b, i]
            assert (at(kn, b, dst) == at(k, b, src)).all()
            assert (at(vn, b, dst) == at(v, b, src)).all()
            touched.add((int(bt[b, dst // page]), dst % page))
    for p in range(len(perm)):
        for r in range(page):
            if (p, r) not in touched:
                assert (kn[p, :, r] == k[p, :, r]).all() and (vn[p, :, r] == v[p, :, r]).all()


# ---------------------------------------------------------------------------
# Ablation presets (Sec. 5.3) and the DDTree-style marginal ranking (Sec. 3.1)
# ---------------------------------------------------------------------------

def _all_slot_paths(L, K):
    paths = [()]
    for d in range(L):
        paths += [p + (j,) for p in paths if len(p) == d for j in range(K)]
    return paths


def _selected_slot_paths(s, b=0):
    n = int(s["n_nodes"][b])
    paths = {0: ()}
    for i in range(1, n):
        paths[i] = paths[int(s["parent"][b, i])] + (int(s["slot"][b, i]),)
    return set(paths.values())


def _top_n(paths, score, n):
    ranked = sorted(paths, key=lambda p: -score(p))
    # the cut must not fall on a near-tie, or float32 rounding could decide it
    if len(ranked) > n:
        a, b = score(ranked[n - 1]), score(ranked[n])
        assert a > b * (1 + 1e-4), "seed gives a near-tie at the budget cut"
    return set(ranked[:n])


@pytest.mark.parametrize("seed", range(6))
def test_budget_fill_is_top_n_by_reach(seed):
    """lambda2 = 0, tau = 0: the selected set is the n_max trie nodes of
    largest reach (reach only falls along a path, so that set is prefix-closed)."""
    rng = np.random.default_rng(1100 + seed)
    L, K, n_max = 4, 3, 15
    q = _random_qcond(rng, L, K)
    ids = np.stack([rng.permutation(20)[:K] for _ in range(L)]).astype(np.int32)
    s = O.select_subtree(q[None], ids[None], np.array([0]), np.array([0]), 1.0, 0.0, 0.0, n_max)
    assert int(s["n_nodes"][0]) == n_max                       # the budget is filled

    def reach(p):                                               # float64 product along p
        r = 1.0
        for d, j in enumerate(p):
            r *= float(q[d, 0 if d == 0 else p[d - 1], j])
        return r

    assert _selected_slot_paths(s) == _top_n(_all_slot_paths(L, K), reach, n_max)


@pytest.mark.parametrize("seed", range(6))
def test_ddtree_mode_is_top_n_by_marginal_path_probability(seed):
    B, L, K, V = 1, 4, 3, 30
    x, ids, logp, ent, root = _tiny_inputs(B=B, L=L, K=K, V=V, seed=1200 + seed)
    q = O.score_qcond(root, ids, logp, ent, "marginal_product")
    # closed form: each parent's row is the children's full-vocabulary marginals
    z = np.asarray(x, np.float64)
    p_full = np.exp(z - z.max(-1, keepdims=True))
    p_full /= p_full.sum(-1, keepdims=True)
    marg = np.take_along_axis(p_full[0], ids[0].astype(np.int64), axis=-1)     # [L, K]
    for d in range(L):
        for i in range(1 if d == 0 else K):
            np.testing.assert_allclose(q[0, d, i], marg[d], rtol=1e-6)
        assert q[0, d, 0].sum() <= 1.0 + 1e-6
    n_max = 12
    s = O.select_subtree(q, ids, root, np.array([0]), 1.0, 0.0, 0.0, n_max)

    def path_prob(p):
        r = 1.0
        for d, j in enumerate(p):
            r *= marg[d, j]
        return r

    assert _selected_slot_paths(s) == _top_n(_all_slot_paths(L, K), path_prob, n_max)
