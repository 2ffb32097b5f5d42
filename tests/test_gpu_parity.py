"""Parity of every CUDA stage (through the C ABI) with the CPU oracle.

Tolerances (each follows from the arithmetic of its stage):
* integer results (top-K ids, tree topology, mask, acceptance) bit-exact;
* lse, entropy: 1e-5 relative; logp = logit - lse: 1e-5 of max(|logp|, |lse|);
* q_cond (same inputs on both sides): 1e-5 relative, 1e-7 absolute floor;
* reach and utility from the same q_cond: bit-exact (same f32 IEEE operations);
* attention outputs (bf16): 2e-2 absolute against the float64 oracle.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import workloads as W  # noqa: E402
from oracle import taps_oracle as O  # noqa: E402

ATTN_ATOL = 2e-2


@pytest.fixture(scope="module")
def taps():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00487_gb300 as t
    return t


DEV = "cuda:0"


def dt(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def bf(a):
    return dt(np.asarray(a, np.float32)).to(torch.bfloat16)


def host(t):
    return t.cpu().numpy()


# ---------------------------------------------------------------------------
# Stage 1
# ---------------------------------------------------------------------------

def _check_topk(taps, x, K, dtype=torch.float32, x_dev=None):
    xd = x_dev if x_dev is not None else dt(x.astype(np.float32)).to(dtype)
    ids, logp, lse, ent = taps.taps_topk_marginals(xd, K)
    torch.cuda.synchronize()
    r_ids, r_logp, r_lse, r_ent = O.topk_marginals(x, K)
    np.testing.assert_array_equal(host(ids), r_ids)
    np.testing.assert_allclose(host(lse), r_lse, rtol=1e-5)
    np.testing.assert_allclose(host(ent), r_ent, rtol=1e-5, atol=1e-6)
    scale = np.maximum(np.abs(r_logp), np.abs(r_lse)[..., None])
    assert np.all(np.abs(host(logp) - r_logp) <= 1e-5 * scale)


@pytest.mark.parametrize("name", ["tiny", "qwen3_4b", "qwen3_8b", "long", "llama31_8b"])
def test_topk_configs(taps, name):
    cfg = W.CONFIGS[name]
    B = min(cfg.B, 2)
    x = W.make_logits(cfg, B=B)
    _check_topk(taps, x, cfg.K, torch.float32 if cfg.logits_dtype == "f32" else torch.bfloat16)


@pytest.mark.slow
def test_topk_batched_full(taps):
    cfg = W.CONFIGS["batched"]
    x = W.make_logits(cfg)
    _check_topk(taps, x, cfg.K, torch.bfloat16)


@pytest.mark.parametrize("V,K,B,L", [(1, 1, 1, 1), (7, 7, 1, 3), (2047, 5, 2, 2), (4099, 32, 1, 2),
                                     (151937, 8, 1, 2), (100003, 16, 3, 5), (262143, 3, 1, 1)])
def test_topk_ragged_sizes(taps, V, K, B, L):
    rng = np.random.default_rng(V)
    x = (rng.standard_normal((B, L, V)) * 4).astype(np.float32)
    _check_topk(taps, x, K)
    _check_topk(taps, W.round_to_bf16(x), K, torch.bfloat16)


def test_topk_ties_and_minus_inf(taps):
    rng = np.random.default_rng(3)
    x = rng.integers(-4, 3, size=(2, 3, 30011)).astype(np.float32)     # heavy exact ties
    x[0, 0, ::3] = -np.inf
    x[1, 2, :] = 0.0
    x[1, 2, 17] = -0.0
    _check_topk(taps, x, 32)
    _check_topk(taps, x, 1)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_topk_value_ties_at_the_threshold(taps, dtype):
    """Long rows whose largest values repeat (quantised to a coarse grid), so
    that the running threshold's value is shared by many elements and the
    token-id tie-break decides membership: exercises the value pre-filter and
    the insertion merges over many tiles and across the CTA's warps."""
    rng = np.random.default_rng(17)
    B, L, V = 4, 16, 151936
    x = np.round(rng.standard_normal((B, L, V)) * 2.0 * 4) / 4        # steps of 0.25
    for b in range(B):
        for d in range(L):
            top = rng.choice(V, size=20, replace=False)              # 20 tied maxima
            x[b, d, top] = x[b, d].max() + 0.25
    x = x.astype(np.float32)
    _check_topk(taps, x, 8, dtype)
    _check_topk(taps, x, 16, dtype)


def _padded(x, dtype, mult=8):
    """x on the device in a row buffer padded to a multiple of `mult`
    elements, so that rows start on 16-byte boundaries whatever V is (the
    vector paths, including the one-cluster-per-row kernel for few rows)."""
    B, L, V = x.shape
    Vp = -(-V // mult) * mult
    full = np.zeros((B, L, Vp), np.float32)
    full[:, :, :V] = x
    return dt(full).to(dtype)[:, :, :V]


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V,K,B,L", [(1, 1, 1, 1), (7, 7, 1, 3), (2047, 5, 2, 2), (4099, 32, 1, 2),
                                     (32000, 4, 1, 8), (100003, 16, 1, 5), (128256, 8, 1, 10),
                                     (151936, 8, 1, 16), (151937, 1, 1, 16), (262143, 3, 1, 1),
                                     (151936, 2, 4, 24)])
def test_topk_few_rows_aligned(taps, V, K, B, L, dtype):
    """Rows on 16-byte boundaries with few rows: the one-cluster-per-row path
    (partial vectors at the end of the row, rows shorter than a CTA's slice,
    every K from 1 to 32, and a shape with too many rows for it)."""
    rng = np.random.default_rng(V + K)
    x = (rng.standard_normal((B, L, V)) * 4).astype(np.float32)
    if dtype == torch.bfloat16:
        x = W.round_to_bf16(x)
    _check_topk(taps, x, K, dtype, x_dev=_padded(x, dtype))


def test_topk_few_rows_ties_and_minus_inf(taps):
    rng = np.random.default_rng(5)
    x = rng.integers(-4, 3, size=(1, 16, 30011)).astype(np.float32)   # heavy exact ties
    x[0, 0, ::3] = -np.inf
    x[0, 1, :] = 0.0
    x[0, 1, 17] = -0.0
    x[0, 2, :] = -np.inf                                               # 40 finite logits
    x[0, 2, rng.choice(30011, size=40, replace=False)] = rng.integers(-2, 2, size=40)
    x[0, 3, 32:] = -np.inf                                             # exactly K finite
    for dtype in (torch.float32, torch.bfloat16):
        _check_topk(taps, x, 32, dtype, x_dev=_padded(x, dtype))
        _check_topk(taps, x, 1, dtype, x_dev=_padded(x, dtype))


@pytest.mark.parametrize("K", [16, 32])
def test_topk_few_rows_many_candidates(taps, K):
    """Every 256-th 16-byte vector repeats (value falling with the vector index
    modulo 256): the lanes holding the largest values hold many copies of them,
    so far more elements than one CTA lists reach the first key threshold and
    the threshold is raised until they fit. Exact ties everywhere, decided by
    token id."""
    V = 151936
    vec = np.arange(V) // 8
    x = (-(vec % 256) * 0.125).astype(np.float32)[None, None, :].repeat(16, axis=1)
    x[0, 1] = x[0, 1][::-1]
    x[0, 2, ::2] -= 0.0625
    for dtype in (torch.bfloat16, torch.float32):
        xd = W.round_to_bf16(x) if dtype == torch.bfloat16 else x
        _check_topk(taps, xd, K, dtype, x_dev=_padded(xd, dtype))


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V,K", [(30011, 8), (65539, 32), (4093, 1), (151936, 16)])
def test_topk_many_rows(taps, V, K, dtype):
    """320 rows (20 requests x 16 positions): one CTA streams each row
    (partial last stage, the elements after the last whole vector, K from 1
    to 32)."""
    rng = np.random.default_rng(V + 7 * K)
    x = (rng.standard_normal((20, 16, V)) * 3).astype(np.float32)
    if dtype == torch.bfloat16:
        x = W.round_to_bf16(x)
    _check_topk(taps, x, K, dtype, x_dev=_padded(x, dtype))


def test_topk_many_rows_ties_and_special_rows(taps):
    """320 rows of heavy exact ties (small integers), so the first threshold's
    value is shared by thousands of elements and a stage overflows the
    candidate list; plus rows of one value, rows mostly -inf, and rows whose
    16-byte vectors repeat every 256 vectors."""
    rng = np.random.default_rng(11)
    V = 20011
    x = rng.integers(-3, 3, size=(20, 16, V)).astype(np.float32)
    x[0, 0, :] = 1.5                                                   # one value
    x[0, 1, :] = -np.inf
    x[0, 1, rng.choice(V, size=40, replace=False)] = rng.integers(-2, 2, size=40)
    x[0, 2, ::2] = -np.inf
    vec = np.arange(V) // 8
    x[1, 0] = -(vec % 256) * 0.125                                     # periodic vectors
    x[1, 1] = x[1, 0][::-1]
    for dtype in (torch.float32, torch.bfloat16):
        for K in (32, 8, 1):
            _check_topk(taps, x, K, dtype, x_dev=_padded(x, dtype))


def test_topk_strided_rows(taps):
    """Rows with a stride that is not a multiple of 16 bytes take the scalar path."""
    rng = np.random.default_rng(4)
    V, pad = 5003, 3
    full = (rng.standard_normal((2, 4, V + pad)) * 2).astype(np.float32)
    xd = dt(full)[:, :, :V]
    _check_topk(taps, full[:, :, :V], 8, x_dev=xd)


# ---------------------------------------------------------------------------
# Stage 2 (same inputs on both sides: the oracle's stage-1 results in f32)
# ---------------------------------------------------------------------------

_STAGE1 = {}


def _oracle_stage1(cfg, B=None):
    """Logits and the oracle's stage-1 results (ids, logp, lse, entropy), cached:
    the full batch-32 workload takes tens of seconds to draw and rank on the CPU."""
    B = cfg.B if B is None else B
    key = (cfg, B)
    if key not in _STAGE1:
        x = W.make_logits(cfg, B=B)
        _STAGE1[key] = (x,) + tuple(O.topk_marginals(x, cfg.K))
    return _STAGE1[key]


def _stage1_inputs(cfg, B=None):
    """Stage-2 inputs as the GPU stages take them (f32)."""
    x, ids, logp, lse, ent = _oracle_stage1(cfg, B)
    root = W.make_root_tokens(cfg, B=x.shape[0])
    return x, ids, logp.astype(np.float32), ent.astype(np.float32), root


@pytest.mark.parametrize("name,kind", [("tiny", "mlp"), ("tiny", "marginal"),
                                       ("qwen3_8b", "mlp"), ("long", "mlp"),
                                       ("qwen3_8b", "marginal"), ("llama31_8b", "mlp"),
                                       ("tiny", "marginal_product"),
                                       ("qwen3_8b", "marginal_product"),
                                       ("long", "marginal_product"),
                                       ("qwen3_4b", "mlp"), ("qwen3_4b", "marginal"),
                                       ("batched", "mlp")])
def test_score_parity(taps, name, kind):
    """Every request of the batch-32 workload (per-request indexing), two of the others."""
    cfg = W.CONFIGS[name]
    x, ids, logp, ent, root = _stage1_inputs(cfg, B=cfg.B if name == "batched" else min(cfg.B, 2))
    w = W.make_scorer_weights(cfg)
    if kind == "mlp":
        sp = taps.scorer_params("mlp", dt(w["packed"]), w["E"], w["H"], w["V"], w["max_depth"])
    else:
        sp = taps.scorer_params(kind)
    q = taps.taps_score_reach(dt(root), dt(ids), dt(logp), dt(ent), sp)
    torch.cuda.synchronize()
    ref = O.score_qcond(root, ids, logp, ent, kind, w)
    np.testing.assert_allclose(host(q), ref, rtol=1e-5, atol=1e-7)


@pytest.mark.parametrize("name", ["tiny", "qwen3_8b", "long", "llama31_8b"])
def test_score_path_reach(taps, name):
    """Eq. 2 reach of an explicit node list: bit-exact against the oracle's
    float32 path product on the GPU's own q_cond, nodes outside the trie give
    0, and every selected node's reach equals the selection's reach."""
    cfg = W.CONFIGS[name]
    x, ids, logp, ent, root = _stage1_inputs(cfg, B=min(cfg.B, 2))
    B = x.shape[0]
    w = W.make_scorer_weights(cfg)
    sp = taps.scorer_params("mlp", dt(w["packed"]), w["E"], w["H"], w["V"], w["max_depth"])
    rng = np.random.default_rng(41)
    M = 333
    paths = rng.integers(0, cfg.K, size=(B, M, cfg.L)).astype(np.uint8)
    plen = rng.integers(0, cfg.L + 1, size=(B, M)).astype(np.int32)
    plen[0, :4] = [cfg.L + 1, -1, 1, 0]
    paths[0, 2, 0] = cfg.K                      # a slot past the top-K
    q, pr = taps.taps_score_reach(dt(root), dt(ids), dt(logp), dt(ent), sp,
                                  paths=dt(paths), path_len=dt(plen))
    torch.cuda.synchronize()
    ref = O.path_reach(host(q), paths, plen)
    np.testing.assert_array_equal(host(pr).view(np.uint32), ref.view(np.uint32))
    assert host(pr)[0, :4].tolist() == [0.0, 0.0, 0.0, 1.0]
    # the selection's own reach of each selected node, bit for bit
    ctx = W.make_ctx_lens(cfg, B=B)
    sel = taps.taps_select_subtree(q, dt(ids), dt(root), dt(ctx), cfg.lambda1, cfg.lambda2,
                                   0.0, cfg.n_max)
    torch.cuda.synchronize()
    s = {k: host(v) for k, v in sel.items()}
    tp = np.zeros((B, cfg.n_max, cfg.L), np.uint8)
    tl = np.zeros((B, cfg.n_max), np.int32)
    for b in range(B):
        walk = [()]
        for i in range(1, int(s["n_nodes"][b])):
            walk.append(walk[int(s["parent"][b, i])] + (int(s["slot"][b, i]),))
            tp[b, i, :len(walk[-1])] = walk[-1]
            tl[b, i] = len(walk[-1])
    _, pr2 = taps.taps_score_reach(dt(root), dt(ids), dt(logp), dt(ent), sp,
                                   paths=dt(tp), path_len=dt(tl))
    torch.cuda.synchronize()
    for b in range(B):
        n = int(s["n_nodes"][b])
        np.testing.assert_array_equal(host(pr2)[b, :n].view(np.uint32),
                                      s["reach"][b, :n].view(np.uint32))


# ---------------------------------------------------------------------------
# Stage 3 (same q_cond on both sides: bit-exact)
# ---------------------------------------------------------------------------

SEL_KEYS = ("n_nodes", "parent", "depth", "token", "slot", "pos_id", "reach", "utility")


def _check_select(taps, q, ids, root, ctx, l1, l2, tau, n_max):
    out = taps.taps_select_subtree(dt(q), dt(ids), dt(root), dt(ctx), l1, l2, tau, n_max)
    torch.cuda.synchronize()
    ref = O.select_subtree(q, ids, root, ctx, l1, l2, tau, n_max)
    for k in SEL_KEYS:
        np.testing.assert_array_equal(host(out[k]), ref[k], err_msg=k)
    return ref


@pytest.mark.parametrize("name,n_max", [("tiny", 16), ("qwen3_8b", 32), ("qwen3_8b", 64),
                                        ("qwen3_8b", 128), ("qwen3_8b", 256), ("long", 256),
                                        ("llama31_8b", 64),
                                        ("qwen3_4b", 512)])
def test_select_parity(taps, name, n_max):
    cfg = W.CONFIGS[name]
    x, ids, logp, ent, root = _stage1_inputs(cfg, B=min(cfg.B, 2))
    w = W.make_scorer_weights(cfg)
    q = O.score_qcond(root, ids, logp, ent, "mlp", w)
    ctx = W.make_ctx_lens(cfg, B=x.shape[0])
    _check_select(taps, q, ids, root, ctx, cfg.lambda1, cfg.lambda2, 0.0, n_max)


@pytest.mark.parametrize("mode,name,n_max", [("budget_fill", "qwen3_8b", 64),
                                             ("budget_fill", "long", 256),
                                             ("no_scorer", "qwen3_8b", 64),
                                             ("ddtree", "qwen3_8b", 64),
                                             ("ddtree", "qwen3_8b", 512),
                                             ("ddtree", "llama31_8b", 512)])
def test_select_ablation_modes(taps, mode, name, n_max):
    """Selection presets (Sec. 5.3 ablations, DDTree-style ranking of Sec. 3.1)
    on the scorer output of that mode; budget-filling modes fill n_max."""
    from paper_2606_00487_gb300.round import MODES
    preset = MODES[mode]
    cfg = W.CONFIGS[name]
    x, ids, logp, ent, root = _stage1_inputs(cfg, B=min(cfg.B, 2))
    w = W.make_scorer_weights(cfg)
    q = O.score_qcond(root, ids, logp, ent, preset["scorer_kind"], w)
    ctx = W.make_ctx_lens(cfg, B=x.shape[0])
    l2 = preset.get("lambda2", cfg.lambda2)
    tau = preset.get("tau", cfg.tau)
    ref = _check_select(taps, q, ids, root, ctx, cfg.lambda1, l2, tau, n_max)
    if l2 == 0.0 and tau == 0.0:
        assert (ref["n_nodes"] == n_max).all()


def test_select_batched_requests(taps):
    cfg = W.CONFIGS["batched"]
    rng = np.random.default_rng(11)
    B, L, K = 32, 16, 8
    raw = rng.random((B, L, K, K)) ** 3 + 1e-3
    q = (raw / raw.sum(-1, keepdims=True)).astype(np.float32)
    q[:, 0, 1:] = 0
    ids = np.stack([np.stack([rng.permutation(151936)[:K] for _ in range(L)]) for _ in range(B)])
    ids = ids.astype(np.int32)
    root = rng.integers(0, 151936, size=B).astype(np.int32)
    ctx = W.make_ctx_lens(cfg)
    _check_select(taps, q, ids, root, ctx, 1.0, 0.1, 0.0, 64)


@pytest.mark.parametrize("tau", [1e-3, 2e-2, 0.3, 5.0])
def test_select_adaptive_threshold(taps, tau):
    cfg = W.CONFIGS["qwen3_8b"]
    x, ids, logp, ent, root = _stage1_inputs(cfg, B=1)
    q = O.score_qcond(root, ids, logp, ent, "marginal")
    ref = _check_select(taps, q, ids, root, np.array([7], np.int32), 1.0, 0.1, tau, 256)
    assert ref["n_nodes"][0] < 256 or tau < 1e-2


def test_select_ties_chain_and_limits(taps):
    rng = np.random.default_rng(5)
    # exact ties everywhere: few distinct probabilities
    L, K = 31, 32
    raw = rng.choice([1.0, 2.0, 4.0], size=(1, L, K, K))
    q = (raw / raw.sum(-1, keepdims=True)).astype(np.float32)
    q[:, 0, 1:] = 0
    ids = np.stack([rng.permutation(262143)[:K] for _ in range(L)])[None].astype(np.int32)
    _check_select(taps, q, ids, np.array([5], np.int32), np.array([0], np.int32),
                  1.0, 0.0, 0.0, 512)
    _check_select(taps, q, ids, np.array([5], np.int32), np.array([0], np.int32),
                  0.5, 0.25, 0.0, 300)
    # K = 1: a chain (single-path verification)
    q1 = np.ones((1, 12, 1, 1), np.float32)
    ids1 = np.arange(12, dtype=np.int32).reshape(1, 12, 1)
    ref = _check_select(taps, q1, ids1, np.array([3], np.int32), np.array([9], np.int32),
                        1.0, 0.1, 0.0, 8)
    assert ref["n_nodes"][0] == 8
    # budget 1: the root only
    ref = _check_select(taps, q1, ids1, np.array([3], np.int32), np.array([9], np.int32),
                        1.0, 0.1, 0.0, 1)
    assert ref["n_nodes"][0] == 1


def test_select_underflowing_reach(taps):
    """Tiny q_cond values make deep reach underflow to subnormals and zero."""
    L, K = 20, 4
    q = np.zeros((1, L, K, K), np.float32)
    q[0, :, :, :] = np.array([1 - 3e-8, 1e-8, 1e-8, 1e-8], np.float32)
    q[0, 0, 1:] = 0
    q[0, 5:, :, 1:] = np.float32(1e-30)
    ids = np.tile(np.arange(K, dtype=np.int32), (1, L, 1)) + 100
    _check_select(taps, q, ids, np.array([1], np.int32), np.array([0], np.int32),
                  1.0, 0.1, 0.0, 200)


# ---------------------------------------------------------------------------
# Stages 2-4 through taps_score_select_mask (selection and mask in one launch)
# ---------------------------------------------------------------------------

def _scorer(taps, kind, cfg):
    if kind != "mlp":
        return taps.scorer_params(kind), None
    w = W.make_scorer_weights(cfg)
    return taps.scorer_params("mlp", dt(w["packed"]), w["E"], w["H"], w["V"], w["max_depth"]), w


def _check_fused(taps, ids, logp, ent, root, ctx, sp, l1, l2, tau, n_max):
    """The fused launch equals the three separate calls bit for bit, and its
    selection and mask equal the oracle's on its own q_cond."""
    args = (dt(root), dt(ids), dt(logp), dt(ent))
    q1 = taps.taps_score_reach(*args, sp)
    s1 = taps.taps_select_subtree(q1, dt(ids), dt(root), dt(ctx), l1, l2, tau, n_max)
    m1 = taps.taps_build_tree_mask(s1["parent"], s1["n_nodes"])
    q2, s2, m2 = taps.taps_score_select_mask(dt(root), dt(ids), dt(logp), dt(ent), dt(ctx), sp,
                                              l1, l2, tau, n_max)
    torch.cuda.synchronize()
    assert torch.equal(q1.view(torch.int32), q2.view(torch.int32))
    for k in SEL_KEYS:
        assert torch.equal(s1[k], s2[k]), k
    assert torch.equal(m1, m2)
    ref = O.select_subtree(host(q2), ids, root, ctx, l1, l2, tau, n_max)
    for k in SEL_KEYS:
        np.testing.assert_array_equal(host(s2[k]), ref[k], err_msg=k)
    np.testing.assert_array_equal(host(m2).view(np.uint32),
                                  O.build_tree_mask(ref["parent"], ref["n_nodes"], n_max))
    return q2, ref


@pytest.mark.parametrize("name,n_max,kind,tau", [("tiny", 16, "mlp", 0.0),
                                                 ("qwen3_8b", 64, "mlp", 0.0),
                                                 ("qwen3_8b", 256, "mlp", 0.0),
                                                 ("qwen3_8b", 256, "mlp", 2e-2),
                                                 ("qwen3_4b", 512, "marginal", 0.0),
                                                 ("qwen3_8b", 64, "marginal_product", 0.0),
                                                 ("long", 256, "mlp", 0.0),
                                                 ("llama31_8b", 64, "mlp", 0.0),
                                                 ("batched", 64, "mlp", 0.0)])
def test_fused_score_select_mask(taps, name, n_max, kind, tau):
    cfg = W.CONFIGS[name]
    x, ids, logp, ent, root = _stage1_inputs(cfg, B=cfg.B if name == "batched" else min(cfg.B, 2))
    sp, w = _scorer(taps, kind, cfg)
    ctx = W.make_ctx_lens(cfg, B=x.shape[0])
    l2 = 0.0 if kind == "marginal_product" else cfg.lambda2
    q, ref = _check_fused(taps, ids, logp, ent, root, ctx, sp, cfg.lambda1, l2, tau, n_max)
    np.testing.assert_allclose(host(q), O.score_qcond(root, ids, logp, ent, kind, w),
                               rtol=1e-5, atol=1e-7)
    if tau > 0:
        assert (ref["n_nodes"] < n_max).any()


def test_fused_large_shape(taps):
    """The largest tables the limits allow in practice: L = 24, K = 32,
    n_max = 512 (ranking passes over 512 + appended entries)."""
    rng = np.random.default_rng(23)
    B, L, K = 2, 24, 32
    ids = np.stack([np.stack([rng.permutation(100000)[:K] for _ in range(L)])
                    for _ in range(B)]).astype(np.int32)
    logp = -np.sort(rng.exponential(3.0, size=(B, L, K)), axis=-1).astype(np.float32)
    ent = rng.random((B, L)).astype(np.float32) * 5
    root = rng.integers(0, 100000, size=B).astype(np.int32)
    ctx = np.array([10, 2000], np.int32)
    _check_fused(taps, ids, logp, ent, root, ctx, taps.scorer_params("marginal"), 1.0, 0.05,
                 0.0, 512)


# ---------------------------------------------------------------------------
# Stage 4
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n_max", [1, 16, 33, 64, 256, 512])
def test_mask_parity(taps, n_max):
    rng = np.random.default_rng(n_max)
    B = 3
    parent = np.full((B, n_max), -1, np.int32)
    n_nodes = np.array([n_max, max(1, n_max // 2), 1], np.int32)
    for b in range(B):
        for i in range(1, n_nodes[b]):
            parent[b, i] = rng.integers(max(0, i - 20), i)
    m = taps.taps_build_tree_mask(dt(parent), dt(n_nodes))
    torch.cuda.synchronize()
    ref = O.build_tree_mask(parent, n_nodes, n_max)
    np.testing.assert_array_equal(host(m).view(np.uint32), ref)


# ---------------------------------------------------------------------------
# Stage 5
# ---------------------------------------------------------------------------

def _tree(rng, n_max, n, L=16):
    parent = np.full((1, n_max), -1, np.int32)
    depth = np.zeros(n, int)
    for i in range(1, n):
        cands = [j for j in range(i) if depth[j] < L]
        parent[0, i] = rng.choice(cands)
        depth[i] = depth[parent[0, i]] + 1
    return parent


def _attn_inputs(cfg, B, n_nodes, ctx, n_max, device_kv=False, seed=0):
    rng = np.random.default_rng(seed)
    parent = np.concatenate([_tree(rng, n_max, int(n)) for n in n_nodes])
    mask = O.build_tree_mask(parent, n_nodes, n_max)
    bt, num_pages = W.make_block_table(cfg, ctx, n_max)
    if device_kv:
        kc, vc = W.make_kv_torch(cfg, num_pages, 0, DEV)
        q = W.make_q_torch(cfg, B, n_max, 0, DEV)
    else:
        kn, vn = W.make_kv_numpy(cfg, num_pages)
        kc, vc = bf(kn), bf(vn)
        q = bf(W.make_q_numpy(cfg, B, n_max))
    return q, kc, vc, bt, mask


def _run_attn(taps, q, kc, vc, bt, ctx, n_nodes, mask, status=None):
    """kc, vc: logical [num_pages, Hkv, 16, D] caches, packed here. Without a
    caller-supplied status word, the device status must stay 0 (no page
    fault, no wait that ran out)."""
    kc = taps.taps_pack_kv_pages(kc)
    vc = taps.taps_pack_kv_pages(vc)
    own = status is None
    if own:
        status = torch.zeros(1, dtype=torch.int32, device=q.device)
    out, lse = taps.taps_tree_verify_attn(q, kc, vc, dt(bt), dt(ctx), dt(n_nodes),
                                          dt(mask.view(np.int32)), int(ctx.max()),
                                          want_lse=True, status=status)
    torch.cuda.synchronize()
    if own:
        assert int(status.item()) == 0, int(status.item())
    return out, lse


def _f32(t):
    return t.float().cpu().numpy()


@pytest.mark.parametrize("name,n,ctx", [("tiny", 16, 512), ("tiny", 1, 512), ("tiny", 5, 0),
                                        ("tiny", 13, 37), ("qwen3_8b", 64, 300),
                                        ("qwen3_8b", 33, 1000)])
def test_attention_parity_small(taps, name, n, ctx):
    cfg = W.CONFIGS[name]
    n_max = max(16, n)
    ctx_a = np.array([ctx], np.int32)
    nn = np.array([n], np.int32)
    q, kc, vc, bt, mask = _attn_inputs(cfg, 1, nn, ctx_a, n_max)
    out, lse = _run_attn(taps, q, kc, vc, bt, ctx_a, nn, mask)
    ref, ref_lse = O.tree_verify_attn(_f32(q), _f32(kc), _f32(vc), bt, ctx_a, nn, mask)
    assert np.abs(_f32(out) - ref).max() <= ATTN_ATOL
    np.testing.assert_allclose(host(lse)[0, :n], ref_lse[0, :n], rtol=1e-4, atol=1e-4)
    assert np.all(_f32(out)[0, n:] == 0)


def _sampled_check(q, kc, vc, bt, ctx, nn, mask, out, rng, per_req=6):
    """Oracle on sampled (request, node, head) rows, gathering the request's pages."""
    B, n_max, Hq, D = q.shape
    qh, kh, vh = _f32(q), None, None
    o = _f32(out)
    worst = 0.0
    for b in range(B):
        n = int(nn[b])
        pages = bt[b][bt[b] >= 0]
        kb = kc[torch.from_numpy(pages.astype(np.int64)).to(kc.device)].float().cpu().numpy()
        vb = vc[torch.from_numpy(pages.astype(np.int64)).to(vc.device)].float().cpu().numpy()
        bt_b = np.arange(len(pages), dtype=np.int32)[None]
        rows = {(0, int(rng.integers(0, n)), int(rng.integers(0, Hq))) for _ in range(per_req)}
        rows |= {(0, n - 1, Hq - 1), (0, 0, 0)}
        ref, _ = O.tree_verify_attn(qh[b:b + 1], kb, vb, bt_b, ctx[b:b + 1], nn[b:b + 1],
                                    mask[b:b + 1], only=rows)
        for (_, i, h) in rows:
            worst = max(worst, float(np.abs(o[b, i, h] - ref[0, i, h]).max()))
        assert np.all(o[b, n:] == 0)
    assert worst <= ATTN_ATOL, worst
    return worst


def test_attention_parity_many_tiles(taps):
    """Every output row against the oracle where each CTA streams several
    128-token tiles (ctx 4000, 64 nodes: chunks of 4-6 tiles, a ragged last
    page), so the S/P buffers and the K and V rings wrap around (the lazy
    rescale has its own test below)."""
    cfg = W.CONFIGS["qwen3_8b"]
    ctx_a = np.array([4000], np.int32)
    nn = np.array([64], np.int32)
    q, kc, vc, bt, mask = _attn_inputs(cfg, 1, nn, ctx_a, 64)
    out, lse = _run_attn(taps, q, kc, vc, bt, ctx_a, nn, mask)
    ref, ref_lse = O.tree_verify_attn(_f32(q), _f32(kc), _f32(vc), bt, ctx_a, nn, mask)
    assert np.abs(_f32(out) - ref).max() <= ATTN_ATOL
    np.testing.assert_allclose(host(lse)[0, :64], ref_lse[0, :64], rtol=1e-4, atol=1e-4)


def test_attention_lazy_rescale(taps):
    """Keys of every third 128-token tile scaled by 4, so that within a chunk
    a row's running maximum jumps by more than 8 (base 2) from one tile to the
    next and the output accumulator is rescaled in TMEM (the lazy-rescale
    path, which unscaled synthetic keys never reach); every row against the
    oracle."""
    cfg = W.CONFIGS["qwen3_8b"]
    ctx_a = np.array([4000], np.int32)
    nn = np.array([64], np.int32)
    rng = np.random.default_rng(0)
    parent = _tree(rng, 64, 64)
    mask = O.build_tree_mask(parent, nn, 64)
    bt, num_pages = W.make_block_table(cfg, ctx_a, 64)
    kn, vn = W.make_kv_numpy(cfg, num_pages)
    pos = np.arange(int(ctx_a[0]))
    spike = (pos // 128) % 3 == 2
    kn = kn.copy()
    kn[bt[0][pos[spike] // 16], :, pos[spike] % 16, :] *= 4
    q, kc, vc = bf(W.make_q_numpy(cfg, 1, 64)), bf(kn), bf(vn)
    # the premise: a spike tile's maximum exceeds the tile before it by more
    # than 8 (base 2) in most rows of KV head 0
    group = cfg.Hq // cfg.Hkv
    rows = _f32(q)[0, :, :group, :].reshape(-1, cfg.D)
    k0 = _f32(kc)[bt[0][pos // 16], 0, pos % 16, :]
    s2 = rows @ k0.T * (np.log2(np.e) / np.sqrt(cfg.D))
    tmax = np.stack([s2[:, t:t + 128].max(axis=1) for t in range(0, 3840, 128)], axis=1)
    jumps = tmax[:, 2::3] > tmax[:, 1::3][:, :tmax[:, 2::3].shape[1]] + 8
    assert jumps.any(axis=1).mean() > 0.5
    out, lse = _run_attn(taps, q, kc, vc, bt, ctx_a, nn, mask)
    ref, ref_lse = O.tree_verify_attn(_f32(q), _f32(kc), _f32(vc), bt, ctx_a, nn, mask)
    assert np.abs(_f32(out) - ref).max() <= ATTN_ATOL
    np.testing.assert_allclose(host(lse)[0, :64], ref_lse[0, :64], rtol=1e-4, atol=1e-4)


def test_attention_ragged_batch_sampled(taps):
    """Requests of very different lengths in one launch (one of them a single
    node on a one-token context), so chunks end inside tiles and some chunks
    of a cluster are empty."""
    cfg = W.CONFIGS["qwen3_8b"]
    ctx = np.array([4000, 1700, 1, 129], np.int32)
    nn = np.array([64, 17, 1, 40], np.int32)
    q, kc, vc, bt, mask = _attn_inputs(cfg, 4, nn, ctx, 64, device_kv=True)
    out, _ = _run_attn(taps, q, kc, vc, bt, ctx, nn, mask)
    _sampled_check(q, kc, vc, bt, ctx, nn, mask, out, np.random.default_rng(3), per_req=8)


@pytest.mark.parametrize("name,n", [("qwen3_8b", 64), ("qwen3_8b", 256), ("qwen3_4b", 64),
                                    ("llama31_8b", 64)])
def test_attention_full_size_sampled(taps, name, n):
    cfg = W.CONFIGS[name]
    ctx = W.make_ctx_lens(cfg)
    nn = np.array([n], np.int32)
    q, kc, vc, bt, mask = _attn_inputs(cfg, 1, nn, ctx, n, device_kv=True)
    out, _ = _run_attn(taps, q, kc, vc, bt, ctx, nn, mask)
    _sampled_check(q, kc, vc, bt, ctx, nn, mask, out, np.random.default_rng(1))


@pytest.mark.slow
@pytest.mark.parametrize("name", ["batched", "long"])
def test_attention_batched_and_long_sampled(taps, name):
    cfg = W.CONFIGS[name]
    ctx = W.make_ctx_lens(cfg)
    rng = np.random.default_rng(2)
    nn = rng.integers(1, cfg.n_max + 1, size=cfg.B).astype(np.int32)
    nn[0] = cfg.n_max
    q, kc, vc, bt, mask = _attn_inputs(cfg, cfg.B, nn, ctx, cfg.n_max, device_kv=True)
    out, _ = _run_attn(taps, q, kc, vc, bt, ctx, nn, mask)
    _sampled_check(q, kc, vc, bt, ctx, nn, mask, out, rng, per_req=3)


def test_attention_bad_page_sets_status(taps):
    cfg = W.CONFIGS["tiny"]
    ctx = np.array([200], np.int32)
    nn = np.array([4], np.int32)
    q, kc, vc, bt, mask = _attn_inputs(cfg, 1, nn, ctx, 16)
    bt = bt.copy()
    bt[0, 3] = kc.shape[0] + 5            # out of range: skipped and reported
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    out, _ = _run_attn(taps, q, kc, vc, bt, ctx, nn, mask, status=status)
    assert int(status.item()) & taps.TAPS_DEVFAULT_PAGE
    assert np.all(np.isfinite(_f32(out)))
    status.zero_()
    bt[0, 3] = 0
    _run_attn(taps, q, kc, vc, bt, ctx, nn, mask, status=status)
    assert int(status.item()) == 0


@pytest.mark.parametrize("D", [64, 128])
def test_kv_pack_layout(taps, D):
    """The packed cache puts token w, dim d of each (page, head) block at the
    byte offset the header documents; unpack inverts pack."""
    rng = np.random.default_rng(D)
    num_pages, Hkv = 5, 3
    x = rng.standard_normal((num_pages, Hkv, 16, D)).astype(np.float32)
    xd = bf(x)
    packed = taps.taps_pack_kv_pages(xd)
    back = taps.taps_unpack_kv_pages(packed)
    torch.cuda.synchronize()
    assert torch.equal(back, xd)
    raw = packed.view(torch.int16).cpu().numpy().reshape(num_pages * Hkv, -1)
    src = xd.view(torch.int16).cpu().numpy().reshape(num_pages * Hkv, 16, D)
    ch = D // 64
    for blk in range(num_pages * Hkv):
        for w in range(16):
            for d in range(D):
                off = ((w // 8) * ch * 1024 + (d // 64) * 1024 + (w % 8) * 128
                       + ((((d % 64) // 8) ^ (w % 8)) * 16) + (d % 8) * 2)
                assert raw[blk, off // 2] == src[blk, w, d]


# ---------------------------------------------------------------------------
# Stage 6
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("per_node", [False, True])
@pytest.mark.parametrize("seed", range(6))
def test_accept_parity(taps, seed, per_node):
    """Target tokens either follow one target sequence (a function of depth)
    or are drawn per node (nodes of one depth want different tokens, as their
    prefixes differ)."""
    rng = np.random.default_rng(seed)
    B, L, K, n_max = 4, 16, 4, 96
    raw = rng.random((B, L, K, K)) + 0.05
    q = (raw / raw.sum(-1, keepdims=True)).astype(np.float32)
    q[:, 0, 1:] = 0
    ids = rng.integers(0, 5, size=(B, L, K)).astype(np.int32)
    for b in range(B):
        for d in range(L):
            ids[b, d] = rng.permutation(6)[:K]
    sel = O.select_subtree(q, ids, np.zeros(B, np.int32), np.zeros(B, np.int32), 1.0, 0.1, 0.0,
                           n_max)
    y = rng.integers(0, 6, size=(B, L + 1)).astype(np.int32)
    tt = W.target_tokens_for_tree(y, sel["depth"], sel["n_nodes"])
    if per_node:
        for b in range(B):
            n = int(sel["n_nodes"][b])
            tt[b, :n] = rng.integers(0, 6, size=n)
    alen, nodes, bonus = taps.taps_accept(dt(sel["parent"]), dt(sel["token"]),
                                          dt(sel["n_nodes"]), dt(tt), L)
    torch.cuda.synchronize()
    r = O.accept(sel["parent"], sel["token"], sel["n_nodes"], tt, L)
    np.testing.assert_array_equal(host(alen), r[0])
    np.testing.assert_array_equal(host(nodes), r[1])
    np.testing.assert_array_equal(host(bonus), r[2])


# ---------------------------------------------------------------------------
# End to end through TapsRound
# ---------------------------------------------------------------------------

def _near_tie_valid(tree, q_ref, ids, L, K, lambda1, lambda2, rtol=1e-5):
    """The GPU's tree is a valid greedy result under the oracle's q_cond, up to
    a relative utility tolerance: no unselected child of the tree beats a
    selected node by more than rtol."""
    n = int(tree["n_nodes"])
    paths = [()]
    for i in range(1, n):
        paths.append(paths[int(tree["parent"][i])] + (int(tree["slot"][i]),))
    pset = set(paths)

    def util(p):
        return O.reach_of_path(q_ref.astype(np.float64), p) / (lambda1 + lambda2 * len(p))
    sel_min = min(util(p) for p in paths[1:]) if n > 1 else np.inf
    front_max = 0.0
    for p in paths:
        if len(p) < L:
            for j in range(K):
                c = p + (j,)
                if c not in pset:
                    front_max = max(front_max, util(c))
    return front_max <= sel_min * (1 + rtol)


@pytest.mark.parametrize("name,n_max,mode", [("tiny", 16, "taps"), ("qwen3_8b", 64, "taps"),
                                             ("qwen3_8b", 256, "taps"), ("llama31_8b", 64, "taps"),
                                             ("qwen3_8b", 64, "ddtree"),
                                             ("qwen3_8b", 64, "budget_fill"),
                                             ("tiny", 16, "no_scorer"),
                                             ("qwen3_4b", 64, "taps"),
                                             pytest.param("batched", 64, "taps",
                                                          marks=pytest.mark.slow),
                                             pytest.param("long", 256, "taps",
                                                          marks=pytest.mark.slow)])
def test_round_end_to_end(taps, name, n_max, mode):
    """A whole round through TapsRound on one workload, every stage against the
    oracle. The batch-32 (ragged contexts) and long-context (B=8, K=16,
    N=256) cases check every request, so per-request indexing through the
    whole round is covered; their attention is checked on sampled rows of
    every request."""
    from paper_2606_00487_gb300.round import MODES
    preset = MODES[mode]
    kind = preset["scorer_kind"]
    cfg = W.CONFIGS[name].with_(lambda2=preset.get("lambda2", W.CONFIGS[name].lambda2),
                                tau=preset.get("tau", W.CONFIGS[name].tau))
    x, ids, logp, lse, ent = _oracle_stage1(W.CONFIGS[name])
    root, ctx = W.make_root_tokens(cfg), W.make_ctx_lens(cfg)
    w = W.make_scorer_weights(cfg)
    bt, num_pages = W.make_block_table(cfg, ctx, n_max)
    r = taps.TapsRound(B=cfg.B, L=cfg.L, V=cfg.V, K=cfg.K, n_max=n_max, Hq=cfg.Hq, Hkv=cfg.Hkv,
                       D=cfg.D, max_ctx=int(ctx.max()), device=DEV,
                       scorer_weights=dt(w["packed"]), emb_dim=w["E"], hidden=w["H"],
                       lambda1=cfg.lambda1, mode=mode)
    assert (r.lambda2, r.tau) == (cfg.lambda2, cfg.tau)
    xd = dt(x).to(torch.float32 if cfg.logits_dtype == "f32" else torch.bfloat16)
    r.select(xd, dt(root), dt(ctx))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(r.ids), ids)
    q_ref = O.score_qcond(root, ids, logp, ent, kind, w)
    np.testing.assert_allclose(host(r.q_cond), q_ref, rtol=1e-4, atol=1e-6)
    # topology: bit-exact given the GPU's own q_cond, near-tie valid under the oracle's
    gq = host(r.q_cond)
    ref = O.select_subtree(gq, ids, root, ctx, cfg.lambda1, cfg.lambda2, cfg.tau, n_max)
    sel = {k: host(v) for k, v in r.sel.items()}
    for k in SEL_KEYS:
        np.testing.assert_array_equal(sel[k], ref[k], err_msg=k)
    for b in range(cfg.B):
        tree_b = {k: v[b] for k, v in sel.items()}
        assert _near_tie_valid(tree_b, q_ref[b], ids[b], cfg.L, cfg.K, cfg.lambda1, cfg.lambda2)
    mask = O.build_tree_mask(sel["parent"], sel["n_nodes"], n_max)
    np.testing.assert_array_equal(host(r.mask).view(np.uint32), mask)
    # one verification layer
    if cfg.B > 1:
        kc, vc = W.make_kv_torch(cfg, num_pages, 0, DEV)
        qd = W.make_q_torch(cfg, cfg.B, n_max, 0, DEV)
        out = torch.empty_like(qd)
        r.verify_layer(qd, taps.taps_pack_kv_pages(kc), taps.taps_pack_kv_pages(vc), dt(bt),
                       dt(ctx), out)
        torch.cuda.synchronize()
        assert int(r.status.item()) == 0
        _sampled_check(qd, kc, vc, bt, ctx, sel["n_nodes"], mask, out,
                       np.random.default_rng(5), per_req=3)
        del kc, vc, qd, out
    elif cfg.D * cfg.Hq * n_max <= 128 * 32 * 256:
        kn, vn = W.make_kv_numpy(cfg, num_pages)
        qn = W.make_q_numpy(cfg, cfg.B, n_max)
        out = torch.empty((cfg.B, n_max, cfg.Hq, cfg.D), dtype=torch.bfloat16, device=DEV)
        r.verify_layer(bf(qn), taps.taps_pack_kv_pages(bf(kn)), taps.taps_pack_kv_pages(bf(vn)),
                       dt(bt), dt(ctx), out)
        torch.cuda.synchronize()
        rows = {(0, i, h) for i in range(0, int(sel["n_nodes"][0]), 7) for h in (0, cfg.Hq - 1)}
        o_ref, _ = O.tree_verify_attn(qn, kn, vn, bt, ctx, sel["n_nodes"], mask, only=rows)
        o = _f32(out)
        for (_, i, h) in rows:
            assert np.abs(o[0, i, h] - o_ref[0, i, h]).max() <= ATTN_ATOL
    y = W.make_target_sequence(cfg, x)
    tt = W.target_tokens_for_tree(y, sel["depth"], sel["n_nodes"])
    r.accept(dt(tt))
    torch.cuda.synchronize()
    a = O.accept(sel["parent"], sel["token"], sel["n_nodes"], tt, cfg.L)
    np.testing.assert_array_equal(host(r.accept_len), a[0])
    np.testing.assert_array_equal(host(r.accepted_nodes), a[1])
    np.testing.assert_array_equal(host(r.bonus_tok), a[2])
    # the same acceptance from verify logits whose greedy tokens are the targets
    r.accept_len.fill_(-7)
    r.accept_greedy(W.make_verify_logits_torch(cfg, dt(tt), DEV))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(r.target_tok), tt)
    np.testing.assert_array_equal(host(r.accept_len), a[0])
    np.testing.assert_array_equal(host(r.accepted_nodes), a[1])
    np.testing.assert_array_equal(host(r.bonus_tok), a[2])
