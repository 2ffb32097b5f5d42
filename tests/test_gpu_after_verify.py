"""Parity of the steps that follow verification with the CPU oracle:
the target's greedy token per tree node fused with acceptance, and the
accepted path's K/V compaction. All results are integers or moved bytes,
so every comparison is bit-exact."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import workloads as W  # noqa: E402
from oracle import taps_oracle as O  # noqa: E402

DEV = "cuda:0"


@pytest.fixture(scope="module")
def taps():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00487_gb300 as t
    return t


def dt(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    return t.cpu().numpy()


def _random_tree(rng, n_max, n, L, V):
    """Prefix-closed tree in selection order (parent index < child index),
    distinct sibling tokens, depth <= L. Stops early when no node can take
    another child; returns (parent, token, depth, nodes built)."""
    parent = np.full(n_max, -1, np.int32)
    token = np.full(n_max, -1, np.int32)
    depth = np.zeros(n_max, np.int32)
    token[0] = rng.integers(0, V)
    used = [set()]
    for i in range(1, n):
        cands = [p for p in range(i) if depth[p] < L and len(used[p]) < V]
        if not cands:
            return parent, token, depth, i
        p = int(rng.choice(cands))
        free = [t for t in range(V) if t not in used[p]] if V <= 64 else None
        if free is not None:
            t = int(rng.choice(free))
        else:
            t = int(rng.integers(0, V))
            while t in used[p]:
                t = int(rng.integers(0, V))
        used[p].add(t)
        used.append(set())
        parent[i], token[i], depth[i] = p, t, depth[p] + 1
    return parent, token, depth, n


def _verify_case(rng, B, n_max, V, L, n_nodes, follow=0.7):
    """Random verify logits; at most nodes the row's maximum is planted on the
    token of one of its children, so acceptance walks several levels.
    n_nodes is updated in place where a tree cannot hold that many nodes."""
    parent = np.full((B, n_max), -1, np.int32)
    token = np.full((B, n_max), -1, np.int32)
    x = rng.standard_normal((B, n_max, V)).astype(np.float32) * 2.0
    for b in range(B):
        parent[b], token[b], _, built = _random_tree(rng, n_max, int(n_nodes[b]), L, V)
        n_nodes[b] = built
        for i in range(built):
            kids = [c for c in range(built) if parent[b, c] == i]
            if kids and rng.random() < follow:
                x[b, i, token[b, rng.choice(kids)]] = 9.0
    return x, parent, token


def _check(taps, x_dev, x_ref, parent, token, n_nodes, L):
    tt, alen, nodes, bonus = taps.taps_target_greedy_accept(x_dev, dt(parent), dt(token),
                                                            dt(n_nodes), L)
    torch.cuda.synchronize()
    r_tt = O.target_greedy(x_ref, n_nodes)
    np.testing.assert_array_equal(host(tt), r_tt)
    r = O.accept(parent, token, n_nodes, r_tt, L)
    np.testing.assert_array_equal(host(alen), r[0])
    np.testing.assert_array_equal(host(nodes), r[1])
    np.testing.assert_array_equal(host(bonus), r[2])
    return r


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V", [1, 7, 4099, 32000])
def test_target_greedy_accept_parity(taps, dtype, V):
    rng = np.random.default_rng(V)
    B, n_max, L = 3, 48, 8
    n_nodes = np.array([48, 17, 1], np.int32)
    x, parent, token = _verify_case(rng, B, n_max, V, L, n_nodes)
    xd = dt(x).to(dtype)
    x_ref = host(xd.float())
    _check(taps, xd, x_ref, parent, token, n_nodes, L)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_target_greedy_ties_zeros_and_minus_inf(taps, dtype):
    rng = np.random.default_rng(5)
    B, n_max, V, L = 2, 32, 9000, 6
    n_nodes = np.array([32, 30], np.int32)
    x, parent, token = _verify_case(rng, B, n_max, V, L, n_nodes)
    x[0, 0, 123] = x[0, 0, 8000] = 40.0            # tie across CTAs: lower index wins
    x[0, 1, 4000] = x[0, 1, 4001] = 40.0           # tie inside one 16-byte vector
    x[0, 2, 8999] = x[0, 2, 8998] = 40.0           # tie in the tail
    x[0, 3] = -np.inf                              # all -inf: index 0
    x[0, 4] = -np.inf
    x[0, 4, 7000] = 0.0
    x[0, 4, 50] = -0.0                             # -0.0 == +0.0: index 50
    x[1, 5] = 3.0                                  # a constant row: index 0
    xd = dt(x).to(dtype)
    r = _check(taps, xd, host(xd.float()), parent, token, n_nodes, L)
    assert r is not None


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_target_greedy_strided_rows(taps, dtype):
    """Rows that are not 16-byte aligned take the scalar path."""
    rng = np.random.default_rng(9)
    B, n_max, V, L = 2, 20, 3001, 5
    n_nodes = np.array([20, 11], np.int32)
    x, parent, token = _verify_case(rng, B, n_max, V, L, n_nodes)
    big = torch.zeros((B, n_max, V + 3), dtype=dtype, device=DEV)
    big[..., 1:V + 1] = dt(x).to(dtype)
    xd = big[..., 1:V + 1]
    _check(taps, xd, host(xd.float()), parent, token, n_nodes, L)


@pytest.mark.parametrize("B,n_max", [(1, 64), (1, 256), (8, 64)])
def test_target_greedy_full_vocab(taps, B, n_max):
    """Qwen3 vocabulary (151936) in bf16, at the launch shapes of the round."""
    rng = np.random.default_rng(B * 1000 + n_max)
    V, L = 151936, 16
    n_nodes = rng.integers(1, n_max + 1, size=B).astype(np.int32)
    n_nodes[0] = n_max
    x, parent, token = _verify_case(rng, B, n_max, V, L, n_nodes)
    xd = dt(x).to(torch.bfloat16)
    _check(taps, xd, host(xd.float()), parent, token, n_nodes, L)


def test_target_greedy_workspace_reuse(taps):
    """The workspace is left at zero: repeated calls with different shapes agree."""
    rng = np.random.default_rng(3)
    for B, n_max, V in ((2, 16, 5000), (1, 64, 20000), (4, 8, 100), (2, 16, 5000)):
        n_nodes = rng.integers(1, n_max + 1, size=B).astype(np.int32)
        x, parent, token = _verify_case(rng, B, n_max, V, 6, n_nodes)
        xd = dt(x).to(torch.bfloat16)
        _check(taps, xd, host(xd.float()), parent, token, n_nodes, 6)


# ---------------------------------------------------------------------------
# Accepted-path K/V compaction
# ---------------------------------------------------------------------------

def _compact_case(rng, cfg, B, L, n_tree, layers, alens=None):
    ctx = rng.integers(0, 300, size=B).astype(np.int32)
    bt, num_pages = W.make_block_table(cfg, ctx, n_tree)
    alen = (rng.integers(0, L + 1, size=B) if alens is None else np.array(alens)).astype(np.int32)
    path = np.full((B, L + 1), -1, np.int32)
    for b in range(B):
        steps = np.sort(rng.choice(np.arange(1, n_tree), size=alen[b], replace=False))
        path[b, :alen[b] + 1] = np.concatenate([[0], steps])
    ks, vs = [], []
    for layer in range(layers):
        k, v = W.make_kv_numpy(cfg, num_pages, layer)
        ks.append(k)
        vs.append(v)
    return ctx, bt, num_pages, alen, path, ks, vs


@pytest.mark.parametrize("D,Hkv,layers", [(128, 8, 3), (64, 2, 2)])
def test_compact_parity(taps, D, Hkv, layers):
    cfg = W.CONFIGS["qwen3_8b"].with_(D=D, Hkv=Hkv, Hq=Hkv * 4, config_id=7)
    rng = np.random.default_rng(D + Hkv)
    B, L, n_tree = 4, 16, 64
    ctx, bt, num_pages, alen, path, ks, vs = _compact_case(rng, cfg, B, L, n_tree, layers,
                                                           alens=[16, 0, 5, 1])
    kd = [taps.taps_pack_kv_pages(dt(k).to(torch.bfloat16)) for k in ks]
    vd = [taps.taps_pack_kv_pages(dt(v).to(torch.bfloat16)) for v in vs]
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    taps.taps_compact_accepted_kv(kd, vd, dt(bt), dt(ctx), dt(path), dt(alen), status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for layer in range(layers):
        rk, rv = O.compact_accepted_kv(ks[layer], vs[layer], bt, ctx, path, alen)
        gk = host(taps.taps_unpack_kv_pages(kd[layer]).float())
        gv = host(taps.taps_unpack_kv_pages(vd[layer]).float())
        np.testing.assert_array_equal(gk, rk)
        np.testing.assert_array_equal(gv, rv)


def test_compact_after_greedy_accept_round_trip(taps):
    """Fused greedy acceptance feeds compaction directly (device to device)."""
    cfg = W.CONFIGS["qwen3_8b"].with_(config_id=8)
    rng = np.random.default_rng(21)
    B, n_max, V, L = 2, 40, 5000, 16
    n_nodes = np.array([40, 25], np.int32)
    x, parent, token = _verify_case(rng, B, n_max, V, L, n_nodes, follow=0.95)
    ctx = np.array([37, 130], np.int32)
    bt, num_pages = W.make_block_table(cfg, ctx, n_max)
    k, v = W.make_kv_numpy(cfg, num_pages, 0)
    kd = [taps.taps_pack_kv_pages(dt(k).to(torch.bfloat16))]
    vd = [taps.taps_pack_kv_pages(dt(v).to(torch.bfloat16))]
    xd = dt(x).to(torch.bfloat16)
    _, alen, nodes, _ = taps.taps_target_greedy_accept(xd, dt(parent), dt(token), dt(n_nodes), L)
    taps.taps_compact_accepted_kv(kd, vd, dt(bt), dt(ctx), nodes, alen)
    torch.cuda.synchronize()
    r_tt = O.target_greedy(host(xd.float()), n_nodes)
    r_alen, r_nodes, _ = O.accept(parent, token, n_nodes, r_tt, L)
    assert r_alen.max() >= 2
    rk, rv = O.compact_accepted_kv(k, v, bt, ctx, r_nodes, r_alen)
    np.testing.assert_array_equal(host(taps.taps_unpack_kv_pages(kd[0]).float()), rk)
    np.testing.assert_array_equal(host(taps.taps_unpack_kv_pages(vd[0]).float()), rv)


def test_compact_bad_page_sets_status(taps):
    cfg = W.CONFIGS["tiny"].with_(config_id=9)
    rng = np.random.default_rng(2)
    B, L, n_tree = 1, 8, 16
    ctx, bt, num_pages, alen, path, ks, vs = _compact_case(rng, cfg, B, L, n_tree, 1, alens=[3])
    bt = bt.copy()
    bt[0, (int(ctx[0]) + int(path[0, 3])) // 16] = num_pages + 5     # a source page out of range
    kd = [taps.taps_pack_kv_pages(dt(ks[0]).to(torch.bfloat16))]
    vd = [taps.taps_pack_kv_pages(dt(vs[0]).to(torch.bfloat16))]
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    taps.taps_compact_accepted_kv(kd, vd, dt(bt), dt(ctx), dt(path), dt(alen), status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & taps.TAPS_DEVFAULT_PAGE


def test_round_inputs_single_upload_and_results_download(taps):
    """Inputs staged in one pinned buffer reach the device views in one copy;
    a round run on those views matches the oracle, and its results come back
    in one copy in the documented order."""
    cfg = W.CONFIGS["tiny"]
    B, n_max = 1, 16
    x = W.make_logits(cfg)
    root, ctx = W.make_root_tokens(cfg), W.make_ctx_lens(cfg)
    inp = taps.RoundInputs(B=B, L=cfg.L, V=cfg.V, n_max=n_max, Hq=cfg.Hq, D=cfg.D, layers=2,
                           logits_dtype=torch.float32, device=DEV)
    inp.host["logits"].copy_(torch.from_numpy(x))
    inp.host["root_tok"].copy_(torch.from_numpy(root))
    inp.host["target_tok"].fill_(-1)
    inp.upload()
    torch.cuda.synchronize()
    assert torch.equal(inp.dev["logits"].cpu(), torch.from_numpy(x))
    r = taps.TapsRound(B=B, L=cfg.L, V=cfg.V, K=cfg.K, n_max=n_max, Hq=cfg.Hq, Hkv=cfg.Hkv,
                       D=cfg.D, max_ctx=int(ctx.max()), device=DEV, mode="no_scorer")
    r.select(inp.dev["logits"], inp.dev["root_tok"], dt(ctx))
    torch.cuda.synchronize()
    ids, logp, _, ent = O.topk_marginals(x, cfg.K)
    q = O.score_qcond(root, ids, logp, ent, "marginal")
    sel = O.select_subtree(host(r.q_cond), ids, root, ctx, cfg.lambda1, cfg.lambda2, cfg.tau,
                           n_max)
    y = W.make_target_sequence(cfg, x)
    tt = W.target_tokens_for_tree(y, sel["depth"], sel["n_nodes"])
    inp.host["target_tok"].copy_(torch.from_numpy(tt))
    inp.upload()
    r.accept(inp.dev["target_tok"])
    res = torch.empty(r.results.shape, dtype=torch.int32, pin_memory=True)
    r.download(res)
    torch.cuda.synchronize()
    a_len, nodes, bonus = O.accept(sel["parent"], sel["token"], sel["n_nodes"], tt, cfg.L)
    res = res.numpy()
    np.testing.assert_allclose(host(r.q_cond), q, rtol=1e-5, atol=1e-7)
    assert res[0] == sel["n_nodes"][0] and res[1] == a_len[0] and res[2] == bonus[0]
    np.testing.assert_array_equal(res[3:].reshape(B, cfg.L + 1), nodes)
