"""Host-side arithmetic of bench.py (no GPU): the roofline numerator and the
workload/mode presets that name what a bench line measured."""
import itertools

import numpy as np

import bench
import workloads as W
from oracle import taps_oracle as O


def test_attention_bytes_at_the_qwen3_8b_shape():
    """One verification layer reads K and V of the context and the tree
    (2 tensors x 2 bytes x Hkv x D per position) and Q, writes O (2 bytes x Hq
    x D per node each): (4096 + 64) * 8 * 128 * 4 + 64 * 32 * 128 * 4 bytes."""
    cfg = W.CONFIGS["qwen3_8b"]
    depth = np.zeros((1, 64), np.int64)
    byt, _ = bench.attn_bytes_flops(cfg, np.array([4096]), np.array([64]), depth)
    assert byt == 4160 * 8 * 128 * 4 + 64 * 32 * 128 * 4 == 18_087_936


def test_attention_flops_count_the_visible_pairs():
    """Flops are 4 * Hq * D per visible (query node, key) pair: every node sees
    the whole context and its ancestors-or-self, counted here by brute force
    over a random tree's ancestor mask."""
    cfg = W.CONFIGS["tiny"]
    rng = np.random.default_rng(3)
    n_max = 16
    B = 2
    parent = np.full((B, n_max), -1, np.int32)
    depth = np.full((B, n_max), -1, np.int64)
    n_nodes = np.array([16, 9], np.int32)
    for b in range(B):
        depth[b, 0] = 0
        for i in range(1, n_nodes[b]):
            parent[b, i] = rng.integers(0, i)
            depth[b, i] = depth[b, parent[b, i]] + 1
    ctx = np.array([100, 37])
    mask = O.build_tree_mask(parent, n_nodes, n_max)
    pairs = 0
    for b in range(B):
        for i in range(n_nodes[b]):
            visible_tree = sum(int(mask[b, i, j // 32]) >> (j % 32) & 1 for j in range(n_max))
            pairs += int(ctx[b]) + visible_tree
    _, fl = bench.attn_bytes_flops(cfg, ctx, n_nodes, depth)
    assert fl == 4 * cfg.Hq * cfg.D * pairs


def test_mode_presets_and_metric_names():
    for mode, (kind, over) in bench.MODE_PARAMS.items():
        cfg = bench.workload_config("qwen3_8b", mode=mode)
        if over is None:
            assert (cfg.lambda2, cfg.tau) == (W.CONFIGS["qwen3_8b"].lambda2,
                                              W.CONFIGS["qwen3_8b"].tau)
        else:
            assert (cfg.lambda2, cfg.tau) == over
    for name, n_max, layers in itertools.product(["qwen3_8b", "llama31_8b"], [None, 32],
                                                 [None, 2]):
        cfg = bench.workload_config(name, n_max=n_max, layers=layers)
        assert cfg.n_max == (W.CONFIGS[name].n_max if n_max is None else n_max)
        assert cfg.layers == (W.CONFIGS[name].layers if layers is None else layers)
    assert "Qwen3-8B" in bench.metric_name("qwen3_8b")
    assert "LLaMA-3.1-8B" in bench.metric_name("llama31_8b")


def test_all_cores_oracle_split_covers_every_row_once():
    """The all-cores CPU baseline splits stage 5 by (request, head) over worker
    processes; the workers' outputs, summed, equal the serial oracle's."""
    cfg = W.CONFIGS["tiny"].with_(B=2)
    bench._attn_worker_init(cfg)
    inp = bench._W["inp"]
    rng = np.random.default_rng(8)
    n_nodes = np.array([16, 7], np.int32)
    parent = np.full((2, 16), -1, np.int32)
    for b in range(2):
        for i in range(1, n_nodes[b]):
            parent[b, i] = rng.integers(0, i)
    mask = O.build_tree_mask(parent, n_nodes, 16)
    ref, _ = O.tree_verify_attn(inp["q"], inp["k"], inp["v"], inp["bt"], inp["ctx"], n_nodes, mask)
    pairs = [(b, h) for b in range(cfg.B) for h in range(cfg.Hq)]
    n_w = 3
    parts = [bench._attn_worker_rows((pairs[i::n_w], n_nodes, mask)) for i in range(n_w)]
    assert np.array_equal(sum(parts), ref)
    bench._W.clear()


def test_roofline_names_the_binding_bound():
    """N = 64 at the Qwen3-8B shape is HBM-bound (its byte floor is the higher
    one), N = 256 tensor-bound (4 flops per byte per node: intensity ~ 4 n)."""
    peaks = (6704.5, 1911.0, 1736.0, "measured")
    for n, bound in ((64, "hbm"), (256, "tensor")):
        cfg = W.CONFIGS["qwen3_8b"].with_(n_max=n)
        rs = bench.RoundSetup.__new__(bench.RoundSetup)
        rs.cfg = cfg
        rs.ctx_h = np.array([4096])
        depth = np.full((1, n), 4, np.int64)
        depth[0, 0] = 0
        rs.sel_h = {"n_nodes": np.array([n]), "depth": depth}
        rl = rs.roofline(36 * 0.010, peaks)          # 10 us per layer
        assert rl["bound"] == bound
        assert rl["avg_launch_us"] == 10.0
        assert abs(rl["hbm_frac"] - rl["algorithmic_bytes_per_launch"] / 10e-6 / 1e9 / 6704.5) < 1e-4


def test_reference_arm_sample_size():
    """The reference arm times a whole layer of stage 5 per step while the run is
    short, otherwise a share of a layer's (request, head) pairs that keeps the run
    to about the same number of layers, never below the floor of pairs."""
    cfg = W.CONFIGS["qwen3_8b"]
    total = cfg.B * cfg.Hq
    assert bench.reference_attn_pairs(cfg, 20, 5) == 0
    assert bench.reference_attn_pairs(cfg, bench.REF_LAYER_BUDGET - 3, 3) == 0
    for steps in (40, 100, 200, 5000):
        n = bench.reference_attn_pairs(cfg, steps, 5)
        assert bench.REF_MIN_PAIRS <= n < total
        assert n == max(bench.REF_MIN_PAIRS, total * bench.REF_LAYER_BUDGET // (steps + 5))
    assert "4 of the 32" in bench.sample_desc(cfg, 1, 4)
    assert "1 of 36 layers" in bench.sample_desc(cfg, 1, 0)


def test_oracle_step_pair_sample_covers_the_sampled_rows():
    """A stage-5 sample of some (request, head) pairs computes exactly those pairs'
    rows of the layer (the same values as the whole layer there, zeros elsewhere)."""
    cfg = W.CONFIGS["tiny"].with_(B=2)
    inp = bench.oracle_attn_inputs(cfg)
    rng = np.random.default_rng(9)
    n_nodes = np.array([16, 5], np.int32)
    parent = np.full((2, 16), -1, np.int32)
    for b in range(2):
        for i in range(1, n_nodes[b]):
            parent[b, i] = rng.integers(0, i)
    mask = O.build_tree_mask(parent, n_nodes, 16)
    ref, _ = O.tree_verify_attn(inp["q"], inp["k"], inp["v"], inp["bt"], inp["ctx"], n_nodes, mask)
    pairs = [(0, 3), (1, 0), (1, 5)]
    only = {(b, i, h) for (b, h) in pairs for i in range(int(n_nodes[b]))}
    got, _ = O.tree_verify_attn(inp["q"], inp["k"], inp["v"], inp["bt"], inp["ctx"], n_nodes, mask,
                                only=only)
    keep = np.zeros(ref.shape, bool)
    for b, h in pairs:
        keep[b, :, h] = True
    assert np.array_equal(got[keep], ref[keep])
    assert not got[~keep].any()
    # and the timed step runs with such a sample (time scaled to whole layers)
    full = bench.oracle_inputs(cfg)
    scaled, wall = bench.oracle_step(cfg, full, 1, "mlp", None, pairs)
    assert scaled > 0 and wall > 0
