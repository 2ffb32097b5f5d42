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
