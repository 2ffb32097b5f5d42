"""Mutation check of the oracle's pins.

Each case plants one plausible mistake into a copy of the CPU oracle (a
dropped term, a wrong sign, a wrong or off-by-one index, a transposed operand,
a tie broken the other way) and runs the pin suite, tests/test_oracle_pins.py,
against that copy in a separate process. Some pin must fail for every case:
a mistake that no pin notices would make a parity result against the oracle
worthless. The unchanged copy must pass, so that a failure means the planted
mistake was seen and not that the copy is broken.

The mistakes are planted only in the copies, on the CPU; the oracle in the
tree, the CUDA path and the library are not touched. Every case changes what
the function computes on some input (no equivalent rewrites).
"""
import concurrent.futures as cf
import os
import re
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE = os.path.join(ROOT, "oracle", "taps_oracle.py")

# (function, what the mistake is, exact text in the oracle, replacement)
MUTANTS = [
    # Stage 1: marginals, entropy, top-K (Sec. 4.1 stage 1, Sec. 4.2 features)
    ("topk_marginals", "log-sum-exp without the maximum",
     "lse = m + np.log(Z)", "lse = np.log(Z)"),
    ("topk_marginals", "entropy with the wrong sign",
     "entropy = -(p * logp_all).sum(axis=-1)", "entropy = (p * logp_all).sum(axis=-1)"),
    ("topk_marginals", "entropy's log-probability taken against the maximum, not lse",
     "logp_all = np.where(p > 0, x - lse[..., None], 0.0)",
     "logp_all = np.where(p > 0, x - m[..., None], 0.0)"),
    ("topk_marginals", "equal logits ranked by descending token id",
     "order = np.lexsort((np.arange(V), -x[b, d]))",
     "order = np.lexsort((-np.arange(V), -x[b, d]))"),
    ("topk_marginals", "the 0 log 0 = 0 convention dropped (-inf logits)",
     "logp_all = np.where(p > 0, x - lse[..., None], 0.0)", "logp_all = x - lse[..., None]"),
    ("topk_marginals", "child log-probability taken against the maximum, not lse",
     "logp = np.take_along_axis(x, ids.astype(np.int64), axis=-1) - lse[..., None]",
     "logp = np.take_along_axis(x, ids.astype(np.int64), axis=-1) - m[..., None]"),
    ("topk_marginals", "entropy weighted by unnormalised probabilities",
     "p = np.exp(x - lse[..., None])", "p = np.exp(x - m[..., None])"),
    ("topk_marginals", "top-K list starting one rank down",
     "ids[b, d] = order[:K]", "ids[b, d] = order[1:K + 1]"),
    # Stage 2: scorer and sibling softmax (Sec. 4.2, Eq. 1)
    ("edge_logit_mlp", "parent and child embeddings swapped",
     'w["tok_emb"][parent_tok].astype(np.float64),\n        w["tok_emb"][child_tok]',
     'w["tok_emb"][child_tok].astype(np.float64),\n        w["tok_emb"][parent_tok]'),
    ("edge_logit_mlp", "scalar features in the wrong order",
     "np.array([logp_child, entropy], np.float64)", "np.array([entropy, logp_child], np.float64)"),
    ("edge_logit_mlp", "hidden layer without the ReLU",
     'h = np.maximum(w["W1"].astype(np.float64) @ f + w["b1"].astype(np.float64), 0.0)',
     'h = w["W1"].astype(np.float64) @ f + w["b1"].astype(np.float64)'),
    ("edge_logit_mlp", "hidden layer without its bias",
     'h = np.maximum(w["W1"].astype(np.float64) @ f + w["b1"].astype(np.float64), 0.0)',
     'h = np.maximum(w["W1"].astype(np.float64) @ f, 0.0)'),
    ("edge_logit_mlp", "direct log-probability term dropped",
     'return float(w["w_lp"][0]) * logp_child + float(w["w2"].astype(np.float64) @ h)',
     'return float(w["w2"].astype(np.float64) @ h)'),
    ("edge_logit_mlp", "depth embedding of the parent's depth",
     'w["dep_emb"][depth].astype(np.float64)', 'w["dep_emb"][depth - 1].astype(np.float64)'),
    ("edge_logit_mlp", "direct term multiplies the entropy",
     'return float(w["w_lp"][0]) * logp_child +', 'return float(w["w_lp"][0]) * entropy +'),
    ("score_qcond", "edge depth off by one (position index used)",
     "edge_logit_mlp(weights, ptok, int(ids[b, d, j]), d + 1,",
     "edge_logit_mlp(weights, ptok, int(ids[b, d, j]), d,"),
    ("score_qcond", "parents taken from the same position as the children",
     "else [int(t) for t in ids[b, d - 1]]", "else [int(t) for t in ids[b, d]]"),
    ("score_qcond", "entropy of the parent's position, not the child's",
     "float(logp[b, d, j]), float(entropy[b, d]))",
     "float(logp[b, d, j]), float(entropy[b, max(d - 1, 0)]))"),
    ("score_qcond", "every parent row of the first position filled from the root",
     "parents = [int(root_tok[b])] if d == 0", "parents = [int(root_tok[b])] * K if d == 0"),
    ("score_qcond", "sibling logits not normalised",
     "q[b, d, i] = e / e.sum()", "q[b, d, i] = e"),
    ("score_qcond", "marginal-product scores renormalised to the best sibling",
     "q[b, d, i] = np.exp(ell)", "q[b, d, i] = np.exp(ell - ell.max())"),
    ("score_qcond", "marginal scorer's softmax taken over probabilities, not log-probabilities",
     "ell[j] = float(logp[b, d, j])", "ell[j] = float(np.exp(logp[b, d, j]))"),
    # Eq. 2: reach
    ("reach_of_path", "q_cond indexed [child, parent]",
     "r *= float(q_cond_b[d, parent_slot, j])", "r *= float(q_cond_b[d, j, parent_slot])"),
    ("reach_of_path", "q_cond summed instead of multiplied",
     "r *= float(q_cond_b[d, parent_slot, j])", "r += float(q_cond_b[d, parent_slot, j])"),
    ("reach_of_path", "every edge read from the root's row",
     "        r *= float(q_cond_b[d, parent_slot, j])\n        parent_slot = j",
     "        r *= float(q_cond_b[d, parent_slot, j])\n        parent_slot = 0"),
    ("path_reach", "q_cond indexed [child, parent]",
     "r = F32(r * F32(q_cond[b, d, parent_slot, j]))",
     "r = F32(r * F32(q_cond[b, d, j, parent_slot]))"),
    ("path_reach", "every edge read from the root's row",
     "            r = F32(r * F32(q_cond[b, d, parent_slot, j]))\n                parent_slot = j",
     "            r = F32(r * F32(q_cond[b, d, parent_slot, j]))\n                parent_slot = 0"),
    ("path_reach", "full-length paths treated as outside the trie",
     "if n < 0 or n > L or any(j >= K for j in slots):", "if n < 0 or n >= L or any(j >= K for j in slots):"),
    ("path_reach", "the root treated as outside the trie",
     "if n < 0 or n > L or any(j >= K for j in slots):", "if n <= 0 or n > L or any(j >= K for j in slots):"),
    ("path_reach", "edge depths counted from 1",
     "for d, j in enumerate(slots):\n                r = F32(", "for d, j in enumerate(slots, 1):\n                r = F32("),
    # Eq. 3 and Algorithm 1
    ("utility_denominators", "cost term counted one level deeper",
     "F32(l1 + F32(l2 * F32(d)))", "F32(l1 + F32(l2 * F32(d + 1)))"),
    ("utility_denominators", "cost multiplied in instead of added",
     "F32(l1 + F32(l2 * F32(d)))", "F32(l1 * F32(l2 * F32(d)))"),
    ("_key", "utility ties go to the deeper node",
     '-node["depth"], -node["token"]', 'node["depth"], -node["token"]'),
    ("_key", "utility ties go to the larger token id",
     '-node["depth"], -node["token"]', '-node["depth"], node["token"]'),
    ("_key", "full ties go to the parent added later",
     '-node["token"], -node["parent"])', '-node["token"], node["parent"])'),
    ("select_subtree", "every child read from the root's q_cond row",
     'prow = 0 if d == 0 else u["slot"]', "prow = 0"),
    ("select_subtree", "q_cond indexed [child, parent]",
     'r = F32(u["reach"] * q_cond[b, d, prow, j])', 'r = F32(u["reach"] * q_cond[b, d, j, prow])'),
    ("select_subtree", "utility divided by the parent's depth cost",
     'reach=r, utility=F32(r / den[d + 1]))', 'reach=r, utility=F32(r / den[d]))'),
    ("select_subtree", "threshold not strict (utility >= tau)",
     'if best is None or not (best["utility"] > tau32):',
     'if best is None or not (best["utility"] >= tau32):'),
    ("select_subtree", "position id of node i taken as ctx_len + i",
     'out["pos_id"][b, i] = int(ctx_len[b]) + v["depth"]', 'out["pos_id"][b, i] = int(ctx_len[b]) + i'),
    ("select_subtree", "nodes at depth L - 1 not expanded",
     'if u["depth"] == L:\n                    continue', 'if u["depth"] == L - 1:\n                    continue'),
    ("select_subtree", "budget counted without the root",
     "        while len(S) < n_max:\n            best = None", "        while len(S) < n_max - 1:\n            best = None"),
    ("select_subtree", "root utility without its denominator",
     "reach=F32(1.0),\n                    utility=F32(F32(1.0) / den[0]))\n        S = [root]",
     "reach=F32(1.0),\n                    utility=F32(1.0))\n        S = [root]"),
    ("select_subtree", "reach carried in double precision (a different rounding)",
     'r = F32(u["reach"] * q_cond[b, d, prow, j])', 'r = float(u["reach"]) * float(q_cond[b, d, prow, j])'),
    ("select_subtree", "slot output holds the token",
     'out["slot"][b, i] = v["slot"]', 'out["slot"][b, i] = v["token"]'),
    ("materialise_trie", "every child read from the root's q_cond row",
     "prow = 0 if d == 0 else path[-1]", "prow = 0"),
    # Stage 4: ancestor mask
    ("build_tree_mask", "mask transposed (descendants instead of ancestors)",
     "mask[b, i, j // 32] |= np.uint32(1 << (j % 32))", "mask[b, j, i // 32] |= np.uint32(1 << (i % 32))"),
    ("build_tree_mask", "a node does not see itself",
     "            j = i\n            while j >= 0:",
     "            j = int(parent[b, i])\n            while j >= 0:"),
    ("build_tree_mask", "rows past n_nodes filled in",
     "for i in range(int(n_nodes[b])):\n            j = i", "for i in range(n_max):\n            j = i"),
    # Stage 5: verification attention
    ("tree_verify_attn", "scores scaled by 1/D instead of 1/sqrt(D)",
     "scale = 1.0 / math.sqrt(D) if scale is None else scale",
     "scale = 1.0 / D if scale is None else scale"),
    ("tree_verify_attn", "query heads mapped to KV heads interleaved",
     "kv = h // group", "kv = h % Hkv"),
    ("tree_verify_attn", "query read with the KV head's index",
     "s = scale * (Kb[visible, kv, :] @ q[b, i, h])", "s = scale * (Kb[visible, kv, :] @ q[b, i, kv])"),
    ("tree_verify_attn", "block table ignored (pages taken in logical order)",
     "pages = block_table[b, t // P]", "pages = t // P"),
    ("tree_verify_attn", "tree mask read transposed",
     "if (int(mask[b, i, j // 32]) >> (j % 32)) & 1:", "if (int(mask[b, j, i // 32]) >> (i % 32)) & 1:"),
    ("tree_verify_attn", "last context position hidden",
     "visible[:C] = True", "visible[:max(C - 1, 0)] = True"),
    ("tree_verify_attn", "lse without the maximum",
     "lse[b, i, h] = m + math.log(e.sum())", "lse[b, i, h] = math.log(e.sum())"),
    ("tree_verify_attn", "values read from the key cache",
     "out[b, i, h] = (e @ Vb[visible, kv, :]) / e.sum()", "out[b, i, h] = (e @ Kb[visible, kv, :]) / e.sum()"),
    ("tree_verify_attn", "output not normalised",
     "out[b, i, h] = (e @ Vb[visible, kv, :]) / e.sum()", "out[b, i, h] = e @ Vb[visible, kv, :]"),
    ("tree_verify_attn", "tree positions not offset by the context length",
     "visible[C + j] = True", "visible[j] = True"),
    # Stage 6: acceptance and the target's greedy tokens
    ("accept", "target token looked up by depth instead of by node",
     "want = int(target_tok[b, v])", "want = int(target_tok[b, len(path) - 1])"),
    ("accept", "bonus token taken from the draft instead of the target",
     "bonus[b] = int(target_tok[b, v])", "bonus[b] = int(token[b, v])"),
    ("accept", "the root counted as an accepted token",
     "accept_len[b] = len(path) - 1", "accept_len[b] = len(path)"),
    ("accept", "a matching token anywhere in the tree accepted, not only among the children",
     "if int(parent[b, c]) == v and int(token[b, c]) == want]",
     "if c > v and int(token[b, c]) == want]"),
    ("target_greedy", "tied maxima go to the highest index",
     "out[b, i] = int(np.flatnonzero(row == top)[0])", "out[b, i] = int(np.flatnonzero(row == top)[-1])"),
    ("target_greedy", "rows past n_nodes filled in",
     "for i in range(int(n_nodes[b])):\n            row = x[b, i]",
     "for i in range(N):\n            row = x[b, i]"),
    ("compact_accepted_kv", "the last accepted row is not moved",
     "for i in range(int(accept_len[b]) + 1):\n            sp, sr",
     "for i in range(int(accept_len[b])):\n            sp, sr"),
    ("compact_accepted_kv", "V rows copied from the K cache",
     "v_new[dp, :, dr, :] = v_cache[sp, :, sr, :]", "v_new[dp, :, dr, :] = k_cache[sp, :, sr, :]"),
    ("compact_accepted_kv", "page and row of a position swapped",
     "return int(block_table[b, t // page]), t % page", "return int(block_table[b, t % page]), t // page"),
    ("compact_accepted_kv", "source position without the context offset",
     "sp, sr = where(b, c + int(accepted_nodes[b, i]))", "sp, sr = where(b, int(accepted_nodes[b, i]))"),
    ("compact_accepted_kv", "destination one position late",
     "dp, dr = where(b, c + i)", "dp, dr = where(b, c + i + 1)"),
]


def _ids():
    return [f"{fn}:{i}" for i, (fn, _, _, _) in enumerate(MUTANTS)]


def _copy_tree(dst, source_text):
    """The files the pin suite needs, with the oracle's source replaced."""
    os.makedirs(os.path.join(dst, "oracle"))
    os.makedirs(os.path.join(dst, "tests"))
    shutil.copy(os.path.join(ROOT, "oracle", "__init__.py"), os.path.join(dst, "oracle"))
    with open(os.path.join(dst, "oracle", "taps_oracle.py"), "w") as f:
        f.write(source_text)
    shutil.copy(os.path.join(ROOT, "workloads.py"), dst)
    for name in ("conftest.py", "test_oracle_pins.py"):
        shutil.copy(os.path.join(ROOT, "tests", name), os.path.join(dst, "tests"))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(dst, "tests", "golden"))


def _run_pins(dst):
    env = dict(os.environ, PYTHONDONTWRITEBYTECODE="1")
    p = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        "-m", "not gpu", os.path.join("tests", "test_oracle_pins.py")],
                       cwd=dst, env=env, capture_output=True, text=True, timeout=600)
    caught = re.findall(r"^FAILED (\S+)", p.stdout, re.M)
    return p.returncode, caught, p.stdout[-3000:]


@pytest.fixture(scope="module")
def outcomes(tmp_path_factory):
    """Run the pin suite against the unchanged copy and every mutant, in parallel."""
    with open(ORACLE) as f:
        src = f.read()
    jobs = {"unchanged": src}
    for key, (fn, what, old, new) in zip(_ids(), MUTANTS):
        assert src.count(old) == 1, f"{key} ({what}): the text to replace must occur once"
        jobs[key] = src.replace(old, new)
    base = tmp_path_factory.mktemp("oracle_mutants")
    dirs = {}
    for i, (key, text) in enumerate(jobs.items()):
        dirs[key] = str(base / f"m{i}")
        _copy_tree(dirs[key], text)
    workers = max(1, min(len(jobs), len(os.sched_getaffinity(0))))
    with cf.ThreadPoolExecutor(workers) as pool:
        futs = {key: pool.submit(_run_pins, d) for key, d in dirs.items()}
        return {key: f.result() for key, f in futs.items()}


def test_unchanged_copy_passes(outcomes):
    rc, caught, tail = outcomes["unchanged"]
    assert rc == 0, tail


@pytest.mark.parametrize("key", _ids())
def test_planted_mistake_is_caught(outcomes, key):
    fn, what, _, _ = MUTANTS[int(key.split(":")[1])]
    rc, caught, tail = outcomes[key]
    # 1 = some test failed; 2 or more would be a collection or usage error
    assert rc == 1 and caught, f"{fn}: '{what}' passed every pin (rc {rc})\n{tail}"
