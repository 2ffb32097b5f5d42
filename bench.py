"""Benchmark: TAPS rounds per second (select + tree verify) on one GB300.

One step = one full TAPS round over one batch of synthetic input, all stages
of Sec. 4.1 on the GPU: top-K marginals, scoring, selection, mask, tree
verification attention for every layer of the target, acceptance. The round
is captured as three CUDA graphs (stages 1-4, the per-layer attention calls,
stage 6) and replayed; CUDA events between the graphs time the attention
stage live for the roofline figure. The end-to-end figure (``e2e``) replays the
whole round with its uploads from pinned host memory and the read of its
results as one graph per round, waiting for the results before the next round.

Workload (default): Qwen3-8B shape, batch 1, draft block L=16, vocab 151936,
bf16 drafter logits (Zipf s=1.1 with position temperature 0.6 -> 1.4), top-K 8,
node budget 64, 36 layers x (32 q heads, 8 KV heads, head dim 128), context
4096, paged bf16 KV cache with 16-token pages, a distinct cache per layer.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

``--impl reference`` times the plain CPU oracle (the method written from the
paper) on the host cores on a bounded sample of the same workload.
Multi-GPU: the round does not shard (replicas only); under torchrun every
rank runs its own replica and rank 0 reports the aggregate.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
# the end-to-end round uploads the tree queries in this many groups of layers,
# each group of verification layers waiting only for its own
E2E_QUERY_GROUPS = 4


def attn_source_sha256():
    """Hash of the attention kernel's sources (the kernel and its PTX helpers)."""
    import hashlib
    h = hashlib.sha256()
    for f in ("attn.cu", "sm100.cuh"):
        with open(os.path.join(ROOT, "paper_2606_00487_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def load_peaks():
    """(HBM GB/s, bf16 TF/s burst, bf16 TF/s sustained, source). The attention
    kernel runs inside a long step, so its tensor rate is compared with the
    sustained figure."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        burst = float(d["bf16_tflops"])
        return (float(d["hbm_gbs"]), burst, float(d.get("bf16_tflops_sustained", burst)),
                "measured")
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


# scorer kind and (lambda2, tau) overrides of each selection preset; the
# library's TapsRound takes the same presets by name
MODE_PARAMS = {"taps": ("mlp", None), "no_scorer": ("marginal", None),
               "budget_fill": ("mlp", (0.0, 0.0)), "ddtree": ("marginal_product", (0.0, 0.0))}


def workload_config(name, n_max=None, layers=None, mode="taps"):
    import workloads as W
    cfg = W.CONFIGS[name]
    cfg = cfg.with_(n_max=cfg.n_max if n_max is None else n_max,
                    layers=cfg.layers if layers is None else layers)
    over = MODE_PARAMS[mode][1]
    return cfg if over is None else cfg.with_(lambda2=over[0], tau=over[1])


SHAPE_NAMES = {"qwen3_8b": "Qwen3-8B", "qwen3_4b": "Qwen3-4B", "llama31_8b": "LLaMA-3.1-8B",
               "batched": "Qwen3-8B batch-32", "long": "Qwen3-8B long-context", "tiny": "tiny"}


def metric_name(workload):
    return (f"TAPS rounds/sec (select+tree verify) at {SHAPE_NAMES.get(workload, workload)} "
            "shape, 1 GB300; % HBM roofline")


def attn_bytes_flops(cfg, ctx, n_nodes, depth):
    """Algorithmic bytes and flops of one attention layer (every request):
    K and V of the visible context plus the tree nodes, Q read and O write;
    flops count QK^T and PV over the context and the ancestor-or-self pairs."""
    byt, fl = 0, 0
    for b in range(len(ctx)):
        C, n = int(ctx[b]), int(n_nodes[b])
        byt += (C + n) * cfg.Hkv * cfg.D * 2 * 2 + 2 * n * cfg.Hq * cfg.D * 2
        pairs = n * C + int(sum(int(d) + 1 for d in depth[b][:n]))
        fl += 4 * cfg.Hq * cfg.D * pairs
    return byt, fl


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU baseline: the oracle as it stands, on a bounded sample of the workload
# ---------------------------------------------------------------------------

def oracle_step(cfg, inp, sample_layers, kind="mlp", pool=None, pairs=None):
    """One oracle round: stages 1-4 and 6 on the whole batch, stage 5 on
    ``sample_layers`` of the cfg.layers layers; returns seconds scaled to the
    full round. With ``pool`` (worker processes holding the same inputs), each
    sampled layer's stage 5 is split over the workers by (request, head).
    With ``pairs`` (a list of (request, query head)), each sampled layer's
    stage 5 computes only those pairs' rows, and its time is scaled by the
    number of pairs in a layer over the number sampled."""
    from oracle import taps_oracle as O
    t0 = time.perf_counter()
    ids, logp, lse, ent = O.topk_marginals(inp["logits"], cfg.K)
    q = O.score_qcond(inp["root"], ids, logp, ent, kind, inp["w"])
    sel = O.select_subtree(q, ids, inp["root"], inp["ctx"], cfg.lambda1, cfg.lambda2, cfg.tau,
                           cfg.n_max)
    mask = O.build_tree_mask(sel["parent"], sel["n_nodes"], cfg.n_max)
    import workloads as W
    tt = W.target_tokens_for_tree(inp["y"], sel["depth"], sel["n_nodes"])
    O.accept(sel["parent"], sel["token"], sel["n_nodes"], tt, cfg.L)
    t1 = time.perf_counter()
    if pool is not None:
        # each task: a group of (request, head) pairs and this round's tree
        n_w = pool._processes
        pairs = [(b, h) for b in range(cfg.B) for h in range(cfg.Hq)]
        tasks = [(pairs[i::n_w], sel["n_nodes"], mask) for i in range(n_w)]
        for _ in range(sample_layers):
            # the workers' outputs cover disjoint rows: their sum is the layer's output
            sum(pool.map(_attn_worker_rows, tasks, chunksize=1))
        t2 = time.perf_counter()
    else:
        only = None
        if pairs is not None:
            only = {(b, i, h) for (b, h) in pairs for i in range(int(sel["n_nodes"][b]))}
        for _ in range(sample_layers):
            O.tree_verify_attn(inp["q"], inp["k"], inp["v"], inp["bt"], inp["ctx"],
                               sel["n_nodes"], mask, only=only)
        t2 = time.perf_counter()
    per_layer = (t2 - t1) / max(sample_layers, 1)
    if pairs is not None and pool is None:
        per_layer *= cfg.B * cfg.Hq / len(pairs)
    return (t1 - t0) + cfg.layers * per_layer, t2 - t0


def oracle_inputs(cfg):
    import workloads as W
    logits = W.make_logits(cfg)
    inp = oracle_attn_inputs(cfg)
    inp.update(logits=logits, root=W.make_root_tokens(cfg), w=W.make_scorer_weights(cfg),
               y=W.make_target_sequence(cfg, logits))
    return inp


def oracle_attn_inputs(cfg):
    import workloads as W
    ctx = W.make_ctx_lens(cfg)
    bt, num_pages = W.make_block_table(cfg, ctx)
    k, v = W.make_kv_numpy(cfg, num_pages)
    return dict(ctx=ctx, bt=bt, k=k, v=v, q=W.make_q_numpy(cfg, cfg.B, cfg.n_max))


# worker-process state of the all-cores oracle (spawned processes, no CUDA)
_W = {}


def _attn_worker_init(cfg):
    # one BLAS thread per worker process (numpy is first imported below)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[v] = "1"
    _W["cfg"] = cfg
    _W["inp"] = oracle_attn_inputs(cfg)


def _attn_worker_ready(_):
    return "inp" in _W


def _attn_worker_rows(task):
    """Stage 5 of the oracle for the given (request, head) pairs, every node."""
    from oracle import taps_oracle as O
    pairs, nn, mask = task
    inp = _W["inp"]
    only = {(b, i, h) for (b, h) in pairs for i in range(int(nn[b]))}
    out, _ = O.tree_verify_attn(inp["q"], inp["k"], inp["v"], inp["bt"], inp["ctx"], nn, mask,
                                only=only)
    return out


def cpu_child(args):
    """Runs in a fresh process without CUDA: prints the oracle timing JSON."""
    cfg = workload_config(args.workload, args.n_max, args.layers, args.mode)
    kind = MODE_PARAMS[args.mode][0]
    inp = oracle_inputs(cfg)
    pool = None
    if args.cpu_cores > 1:
        import multiprocessing as mp
        pool = mp.get_context("spawn").Pool(args.cpu_cores, initializer=_attn_worker_init,
                                            initargs=(cfg,))
        assert all(pool.map(_attn_worker_ready, range(4 * args.cpu_cores), chunksize=1))
    steps, warm = args.steps, args.warmup
    # with --attn-pairs n, step t samples n (request, head) pairs of a layer,
    # taken in turn from the list of all pairs so that the steps cover them evenly
    all_pairs = [(b, h) for b in range(cfg.B) for h in range(cfg.Hq)]

    def pairs_of(t):
        n = args.attn_pairs
        if n <= 0 or n >= len(all_pairs):
            return None
        return [all_pairs[(t * n + k) % len(all_pairs)] for k in range(n)]

    for t in range(warm):
        oracle_step(cfg, inp, args.sample_layers, kind, pool, pairs_of(t))
    scaled, wall = [], []
    for t in range(steps):
        s, w = oracle_step(cfg, inp, args.sample_layers, kind, pool, pairs_of(warm + t))
        scaled.append(s)
        wall.append(w)
    if pool is not None:
        pool.close()
        pool.join()
    print(json.dumps({"scaled_s": scaled, "wall_s": wall, "cores": args.cpu_cores}))


def run_cpu_baseline(args, steps, warmup, sample_layers, cores=1, attn_pairs=0):
    cfg = workload_config(args.workload, args.n_max, args.layers, args.mode)
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, os.path.abspath(__file__), "--cpu-child", "--workload", args.workload,
           "--mode", args.mode,
           "--n-max", str(cfg.n_max), "--layers", str(cfg.layers), "--steps", str(steps),
           "--warmup", str(warmup), "--sample-layers", str(sample_layers),
           "--cpu-cores", str(cores), "--attn-pairs", str(attn_pairs)]
    r = subprocess.run(cmd, env=env, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"cpu baseline child failed:\n{r.stderr[-2000:]}")
    return json.loads(r.stdout.strip().splitlines()[-1])


def sample_desc(cfg, sample_layers, attn_pairs=0):
    if 0 < attn_pairs < cfg.B * cfg.Hq:
        return (f"oracle stages 1-4 and 6 on the whole round, stage 5 on {attn_pairs} of the "
                f"{cfg.B * cfg.Hq} (request, query head) pairs of one layer, taken in turn "
                f"(timed, then scaled to {cfg.layers} whole layers)")
    return (f"oracle stages 1-4 and 6 on the whole round, stage 5 on {sample_layers} of "
            f"{cfg.layers} layers (timed, then scaled to {cfg.layers} layers)")


# the reference arm's stage-5 sample: a whole layer per step while the run has at
# most this many steps (warm-up included), otherwise a share of a layer's pairs
# sized to keep the run to about as many layers in all; never fewer than 4 pairs
# (below that, the per-request gathers of K and V outweigh the sampled rows and
# the scaled time overstates a layer)
REF_LAYER_BUDGET = 30
REF_MIN_PAIRS = 4


def reference_attn_pairs(cfg, steps, warmup):
    total = cfg.B * cfg.Hq
    n = steps + warmup
    if n <= REF_LAYER_BUDGET:
        return 0
    return min(total, max(REF_MIN_PAIRS, total * REF_LAYER_BUDGET // n))


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def dist_setup(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def max_over_ranks(x: float, world: int, device=None) -> float:
    """Largest value of x over all ranks (the job's wall time is the slowest rank's)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


L2_BYTES = 129 * 1024 * 1024


def after_verify(taps, W, cfg, r, layers, bt, ctx, target, sel_h, s, stream, reps, dev):
    """Time the target greedy + acceptance kernel and the K/V compaction."""
    import torch
    nbytes = cfg.B * cfg.n_max * cfg.V * 2
    nbuf = max(2, -(-2 * L2_BYTES // nbytes))
    bufs = [W.make_verify_logits_torch(cfg, target, dev, seed_offset=i) for i in range(nbuf)]
    outs = (torch.empty((cfg.B, cfg.n_max), dtype=torch.int32, device=dev),
            torch.empty(cfg.B, dtype=torch.int32, device=dev),
            torch.empty((cfg.B, cfg.L + 1), dtype=torch.int32, device=dev),
            torch.empty(cfg.B, dtype=torch.int32, device=dev))
    ws = torch.zeros(max(taps.target_greedy_accept_workspace_bytes(cfg.B, cfg.n_max), 1),
                     dtype=torch.uint8, device=dev)
    sel = r.sel

    def k7(x):
        taps.taps_target_greedy_accept(x, sel["parent"], sel["token"], sel["n_nodes"], cfg.L,
                                       out=outs, ws=ws)

    k7(bufs[0])
    r.accept(target)
    torch.cuda.synchronize()
    # the planted logits reproduce the stand-in target's tokens and its acceptance
    assert torch.equal(outs[0], target), "greedy tokens differ from the planted targets"
    assert torch.equal(outs[1], r.accept_len) and torch.equal(outs[2], r.accepted_nodes)

    def timed(fn, n_inner):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            fn()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps / n_inner * 1e3

    k7_us = timed(lambda: [k7(x) for x in bufs], len(bufs))
    ks = [kc for (_, kc, _, _) in layers]
    vs = [vc for (_, _, vc, _) in layers]
    k8_us = timed(lambda: taps.taps_compact_accepted_kv(ks, vs, bt, ctx, r.accepted_nodes,
                                                        r.accept_len, status=r.status), 1)
    torch.cuda.synchronize()
    assert int(r.status.item()) == 0, "device fault status after compaction"
    live = int(sel_h["n_nodes"].sum())
    k7_bytes = live * cfg.V * 2
    hbm = load_peaks()[0]
    gbs = k7_bytes / (k7_us * 1e-6) / 1e9
    moved = int(r.accept_len.sum().item()) + cfg.B
    del bufs
    return {
        "stage_us": {"s7_target_greedy_accept": round(k7_us, 2),
                     "s8_compact_kv_all_layers": round(k8_us, 2)},
        "target_greedy_accept": {
            "bytes_per_launch": k7_bytes, "us": round(k7_us, 2), "achieved_gbs": round(gbs, 1),
            "frac_of_measured_hbm": round(gbs / hbm, 3),
            "l2": f"{nbuf} rotating verify-logit buffers ({nbuf * nbytes / 1e6:.0f} MB)"},
        "compact_kv": {"layers": cfg.layers, "accepted_positions": moved, "us": round(k8_us, 2)},
    }


class RoundSetup:
    """Every device buffer of one workload's round (seeded synthetic inputs,
    KV caches and queries drawn on the device), the TapsRound and its three
    CUDA graphs (stages 1-4, the per-layer attention calls, stage 6)."""

    def __init__(self, taps, W, cfg, mode, dev):
        import torch
        self.cfg = cfg
        self.logits_h = W.make_logits(cfg)
        root_h, self.ctx_h = W.make_root_tokens(cfg), W.make_ctx_lens(cfg)
        w = W.make_scorer_weights(cfg)
        self.bt_h, num_pages = W.make_block_table(cfg, self.ctx_h)
        self.y = W.make_target_sequence(cfg, self.logits_h)
        ldt = torch.bfloat16 if cfg.logits_dtype == "bf16" else torch.float32
        # the round's per-step inputs live in one staging buffer (one upload per round)
        self.inp = inp = taps.RoundInputs(B=cfg.B, L=cfg.L, V=cfg.V, n_max=cfg.n_max, Hq=cfg.Hq,
                                          D=cfg.D, layers=cfg.layers, logits_dtype=ldt,
                                          device=dev)
        self.logits = inp.dev["logits"]
        self.logits.copy_(torch.from_numpy(self.logits_h).to(dev).to(ldt))
        self.root = inp.dev["root_tok"]
        self.root.copy_(torch.from_numpy(root_h).to(dev))
        self.ctx = torch.from_numpy(self.ctx_h).to(dev)
        self.bt = torch.from_numpy(self.bt_h).to(dev)
        self.layers = []
        for layer in range(cfg.layers):
            kc, vc = W.make_kv_torch(cfg, num_pages, layer, dev)
            kc, vc = taps.taps_pack_kv_pages(kc), taps.taps_pack_kv_pages(vc)   # TAPS page layout
            q = inp.dev["q"][layer]
            q.copy_(W.make_q_torch(cfg, cfg.B, cfg.n_max, layer, dev))
            self.layers.append((q, kc, vc, self.bt))
        self.outs = [torch.empty_like(self.layers[0][0]) for _ in range(cfg.layers)]
        self.r = r = taps.TapsRound(
            B=cfg.B, L=cfg.L, V=cfg.V, K=cfg.K, n_max=cfg.n_max, Hq=cfg.Hq, Hkv=cfg.Hkv,
            D=cfg.D, max_ctx=int(self.ctx_h.max()), device=dev,
            scorer_weights=torch.from_numpy(w["packed"]).to(dev), emb_dim=w["E"], hidden=w["H"],
            lambda1=cfg.lambda1, lambda2=cfg.lambda2, tau=cfg.tau,
            mode=None if mode == "taps" else mode)
        assert (r.lambda2, r.tau) == (cfg.lambda2, cfg.tau)
        # the stand-in target model's greedy tokens depend on the (deterministic) tree
        r.select(self.logits, self.root, self.ctx)
        torch.cuda.synchronize()
        self.sel_h = {k: v.cpu().numpy() for k, v in r.sel.items()}
        tt_h = W.target_tokens_for_tree(self.y, self.sel_h["depth"], self.sel_h["n_nodes"])
        self.target = inp.dev["target_tok"]
        self.target.copy_(torch.from_numpy(tt_h).to(dev))
        self.kv_bytes = sum(kc.numel() * kc.element_size() + vc.numel() * vc.element_size()
                            for (_, kc, vc, _) in self.layers)

        # ---- capture the round as three graphs
        self.s = s = torch.cuda.Stream(device=dev)
        s.wait_stream(torch.cuda.current_stream(dev))
        with torch.cuda.stream(s):
            for _ in range(2):
                r.run(self.logits, self.root, self.ctx, self.layers, self.outs, self.target)
        torch.cuda.current_stream(dev).wait_stream(s)
        torch.cuda.synchronize()
        self.g_pre, self.g_attn, self.g_post = (torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(),
                                                torch.cuda.CUDAGraph())
        with torch.cuda.graph(self.g_pre, stream=s):
            r.select(self.logits, self.root, self.ctx)
        with torch.cuda.graph(self.g_attn, stream=s):
            for (q, kc, vc, b_t), o in zip(self.layers, self.outs):
                r.verify_layer(q, kc, vc, b_t, self.ctx, o)
        with torch.cuda.graph(self.g_post, stream=s):
            r.accept(self.target)
        torch.cuda.synchronize()
        self.stream = torch.cuda.current_stream(dev)

    def capture_e2e(self, res_pin, groups):
        """One round with its host copies as one CUDA graph, through
        TapsRound.capture_round_graph: the head upload, the queries in
        ``groups`` groups of layers on a copy stream, the round, and the read
        of its results into ``res_pin``."""
        import torch
        g = self.r.capture_round_graph(self.inp, self.ctx, self.layers, self.outs, res_pin,
                                       groups, stream=self.s)
        torch.cuda.synchronize()
        return g

    def step(self, ev_a=None, ev_b=None):
        self.g_pre.replay()
        if ev_a is not None:
            ev_a.record(self.stream)
        self.g_attn.replay()
        if ev_b is not None:
            ev_b.record(self.stream)
        self.g_post.replay()

    def time_steps(self, steps, warmup, world=1, clocks=None):
        """W untimed rounds, then exactly ``steps`` rounds between a barrier and
        a synchronize on each side. Returns (elapsed ms of the whole region,
        per-round ms, per-round attention ms), each round's and its attention
        stage's span taken with CUDA events on the launching stream."""
        import torch
        for _ in range(warmup):
            self.step()
        torch.cuda.synchronize()
        if clocks is not None:
            clocks.start()
            time.sleep(0.3)
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier(world)
        torch.cuda.synchronize()
        e0.record(self.stream)
        for k in range(steps):
            ev[k][0].record(self.stream)
            self.step(ev[k][1], ev[k][2])
        e1.record(self.stream)
        torch.cuda.synchronize()
        barrier(world)
        elapsed_ms = e0.elapsed_time(e1)
        rounds = [ev[k][0].elapsed_time(ev[k + 1][0]) for k in range(steps - 1)]
        rounds.append(ev[-1][0].elapsed_time(e1))
        attn = [a.elapsed_time(b) for (_, a, b) in ev]
        return elapsed_ms, rounds, attn

    def roofline(self, attn_ms_per_round, peaks):
        """Attention (the dominant kernel): algorithmic bytes and flops of one
        layer over its average launch time, against the measured HBM copy rate
        and the sustained bf16 tensor rate; ``bound`` is the roofline whose
        floor is higher for this workload."""
        hbm, _, bf16_sus, src = peaks
        byt, fl = attn_bytes_flops(self.cfg, self.ctx_h, self.sel_h["n_nodes"],
                                   self.sel_h["depth"])
        per_launch_s = attn_ms_per_round / self.cfg.layers / 1e3
        gbs = byt / per_launch_s / 1e9
        tf = fl / per_launch_s / 1e12
        t_hbm, t_tc = byt / (hbm * 1e9), fl / (bf16_sus * 1e12)
        return {"bound": "hbm" if t_hbm >= t_tc else "tensor",
                "achieved_gbs": round(gbs, 1), "hbm_frac": round(gbs / hbm, 4),
                "tensor_tflops": round(tf, 1), "tensor_frac": round(tf / bf16_sus, 4),
                "floor_us": round(max(t_hbm, t_tc) * 1e6, 2),
                "avg_launch_us": round(per_launch_s * 1e6, 2),
                "algorithmic_bytes_per_launch": byt, "algorithmic_flops_per_launch": fl,
                "peak_source": src}


# The other configurations of the benchmark suite: the node-budget sweep at
# the Qwen3-8B shape, the Qwen3-4B shape, the batch-32 serving round and the
# long-context stress round (workload name, node budget).
SWEEP = [("qwen3_8b", 32), ("qwen3_8b", 128), ("qwen3_8b", 256), ("qwen3_4b", 64),
         ("batched", 64), ("long", 256)]


def run_sweep(taps, W, args, dev, peaks):
    import torch
    out = {}
    steps, warmup = max(5, min(args.steps, 20)), 3
    for name, n in SWEEP:
        cfg = workload_config(name, n, None, args.mode)
        rs = RoundSetup(taps, W, cfg, args.mode, dev)
        elapsed_ms, rounds, attn = rs.time_steps(steps, warmup)
        status = int(rs.r.status.item())
        rl = rs.roofline(statistics.median(attn), peaks)
        out[f"{name}_n{n}"] = {
            "rounds_per_s": round(steps / (elapsed_ms / 1e3), 2),
            "ms_per_round_median": round(statistics.median(rounds), 4),
            "B": cfg.B, "n_max": n, "layers": cfg.layers,
            "n_nodes_total": int(rs.sel_h["n_nodes"].sum()),
            "attention": rl, "steps": steps, "device_status": status}
        assert status == 0, f"device fault status {status} on {name}"
        del rs
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
    return out


def run_ours(args):
    import torch

    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00487_gb300 as taps
    import workloads as W

    world, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    cfg = workload_config(args.workload, args.n_max, args.layers, args.mode)
    peaks = load_peaks()

    rs = RoundSetup(taps, W, cfg, args.mode, dev)
    r, s, stream = rs.r, rs.s, rs.stream
    logits, root, ctx, target = rs.logits, rs.root, rs.ctx, rs.target
    layers, outs, sel_h = rs.layers, rs.outs, rs.sel_h

    clocks = ClockSampler(local)
    elapsed_ms, rounds_ms, attn_list = rs.time_steps(args.steps, args.warmup, world, clocks)
    attn_ms = sum(attn_list) / args.steps
    clk = clocks.stop()
    elapsed_ms = max_over_ranks(elapsed_ms, world, dev)
    status = int(r.status.item())
    assert status == 0, f"device fault status {status}"

    # ---- select + one-layer round (stages 1-4, one attention layer, stage 6)
    g_one = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_one, stream=s):
        r.select(logits, root, ctx)
        q0, k0, v0, b0 = layers[0]
        r.verify_layer(q0, k0, v0, b0, ctx, outs[0])
        r.accept(target)
    for _ in range(3):
        g_one.replay()
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(min(args.steps, 200), 20)
    f0.record(stream)
    for _ in range(reps):
        g_one.replay()
    f1.record(stream)
    torch.cuda.synchronize()
    one_layer_us = f0.elapsed_time(f1) / reps * 1e3

    # ---- per-stage time: each stage alone as a graph, replayed back to back
    q0, k0, v0, b0 = layers[0]
    stage_fns = {
        "s1_topk": lambda: taps.taps_topk_marginals(
            logits, cfg.K, out=(r.ids, r.logp, r.lse, r.entropy), ws=r.ws_topk),
        "s2_score": lambda: taps.taps_score_reach(root, r.ids, r.logp, r.entropy, r.scorer,
                                                  out=r.q_cond),
        "s3_select": lambda: taps.taps_select_subtree(r.q_cond, r.ids, root, ctx, r.lambda1,
                                                      r.lambda2, r.tau, r.n_max, out=r.sel),
        "s4_mask": lambda: taps.taps_build_tree_mask(r.sel["parent"], r.sel["n_nodes"],
                                                     out=r.mask),
        "s2_s3_s4_fused": lambda: taps.taps_score_select_mask(
            root, r.ids, r.logp, r.entropy, ctx, r.scorer, r.lambda1, r.lambda2, r.tau, r.n_max,
            out=(r.q_cond, r.sel, r.mask)),
        "s5_attention_one_layer": lambda: r.verify_layer(q0, k0, v0, b0, ctx, outs[0]),
        "s6_accept": lambda: r.accept(target),
    }
    # the latency-bound stages back to back in one graph (what a round spends
    # outside top-K and verification): as the round runs them (scoring,
    # selection and mask in one launch, then acceptance), and one launch per stage
    stage_fns["s2_s3_s4_s6_in_one_graph"] = lambda: [stage_fns[k]() for k in (
        "s2_s3_s4_fused", "s6_accept")]
    stage_fns["s2_s3_s4_s6_one_launch_per_stage"] = lambda: [stage_fns[k]() for k in (
        "s2_score", "s3_select", "s4_mask", "s6_accept")]
    stage_us = {}
    for name, fn in stage_fns.items():
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            fn()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        f0.record(stream)
        for _ in range(reps):
            g.replay()
        f1.record(stream)
        torch.cuda.synchronize()
        stage_us[name] = round(f0.elapsed_time(f1) / reps * 1e3, 2)

    # ---- steps after verification (not part of the round above): the target's
    # greedy token per node fused with acceptance, and the accepted path's K/V
    # commit over all layers. The verify logits rotate over enough buffers to
    # exceed L2, so every launch reads its logits from HBM.
    after = after_verify(taps, W, cfg, r, layers, rs.bt, ctx, target, sel_h, s, stream, reps,
                         dev)
    stage_us.update(after.pop("stage_us"))

    # ---- end to end through the public API with host buffers
    e2e = None
    inp = rs.inp
    if not args.no_e2e:
        # The host staging buffer holds every input of a round (logits, root
        # tokens, the 36 layers' tree queries, target tokens). Each round, as
        # one CUDA graph: the head (logits, root and target tokens) uploads on
        # the compute stream; the queries upload on a copy stream in
        # E2E_QUERY_GROUPS groups of layers while the selection stages run, and
        # each group of verification layers waits only for its own queries;
        # then acceptance and one read of the round's results. The host waits
        # for that read before the next round starts, as a decoding loop must.
        torch.cuda.synchronize()
        inp.host_buf.copy_(inp.device_buf)
        res_pin = torch.empty(r.results.shape, dtype=r.results.dtype, pin_memory=True)
        h2d = inp.nbytes
        d2h = res_pin.numel() * res_pin.element_size()
        g_e2e = rs.capture_e2e(res_pin, E2E_QUERY_GROUPS)

        def e2e_step():
            g_e2e.replay()
            stream.synchronize()

        for _ in range(args.warmup):
            e2e_step()
        barrier(world)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            e2e_step()
        t_e2e = max_over_ranks(time.perf_counter() - t0, world, dev)
        e2e = {"value": round(world * args.steps / t_e2e, 2), "unit": "rounds/s",
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)}

    # ---- roofline of the attention stage (dominant kernel)
    hbm, bf16_burst, bf16_sus, src = peaks
    rl = rs.roofline(attn_ms, peaks)
    traffic = None
    tp = os.path.join(ROOT, "profiles", "attn_traffic.json")
    if os.path.exists(tp):
        try:
            t = json.load(open(tp))
            # counters taken on another version of the kernel do not count
            if (t.get("workload") == cfg.name and t.get("n_max") == cfg.n_max
                    and t.get("source_sha256") == attn_source_sha256()):
                traffic = t.get("bytes_per_launch")
        except Exception:
            traffic = None
    roofline = {"bound": "hbm", "achieved": rl["achieved_gbs"], "peak": hbm, "unit": "GB/s",
                "frac": rl["hbm_frac"], "traffic": traffic,
                "peak_source": src, "kernel": "taps_tree_verify_attn (one layer)",
                "algorithmic_bytes_per_launch": rl["algorithmic_bytes_per_launch"],
                "avg_launch_us": rl["avg_launch_us"],
                "tensor_tflops": rl["tensor_tflops"], "tensor_frac": rl["tensor_frac"],
                "tensor_peak": bf16_sus,
                "tensor_peak_note": "sustained bf16 (the kernel runs inside a long step)",
                "binding_roofline": rl["bound"], "floor_us": rl["floor_us"]}

    sweep = None
    if not args.no_sweep and args.workload == "qwen3_8b" and args.n_max in (None, 64):
        sweep = run_sweep(taps, W, args, dev, peaks)

    launches = args.steps * (r.launches_per_select + cfg.layers * r.launches_per_layer + 1)
    line = {
        "metric": metric_name(args.workload),
        "value": round(world * args.steps / (elapsed_ms / 1e3), 2),
        "unit": "rounds/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(elapsed_ms / args.steps, 4),
        "ms_per_step_median": round(statistics.median(rounds_ms), 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": f"synthetic (seeded; shapes of the {SHAPE_NAMES.get(args.workload, args.workload)} "
                "round, no weights or datasets)",
        "config": {"workload": f"{cfg.name}: B={cfg.B} L={cfg.L} V={cfg.V} K={cfg.K} "
                               f"n_max={cfg.n_max} layers={cfg.layers} Hq={cfg.Hq} Hkv={cfg.Hkv} "
                               f"D={cfg.D} ctx={cfg.ctx} page={cfg.page}",
                   "global_batch": cfg.B, "seq_len": int(rs.ctx_h.max()),
                   "parallelism": "replicas",
                   "l2": f"inputs larger than L2: {cfg.layers} distinct KV layers, "
                         f"{rs.kv_bytes / 1e9:.1f} GB per step",
                   "n_nodes": int(sel_h["n_nodes"][0]),
                   "mode": args.mode,
                   "select_plus_one_layer_round_us": round(one_layer_us, 2),
                   "attention_stage_us_per_round": round(attn_ms * 1e3, 2)},
        "roofline": roofline,
        "stage_us": stage_us,
        "after_verify": after,
        "e2e": e2e,
        "gpu_launches": launches,
        "clocks": clk,
    }
    if sweep is not None:
        line["sweep"] = sweep
    if rank == 0 and not args.no_cpu_baseline:
        cb = run_cpu_baseline(args, steps=1, warmup=0, sample_layers=args.sample_layers)
        line["cpu_baseline"] = {"value": round(1.0 / cb["scaled_s"][0], 4), "unit": "rounds/s",
                                "cores": 1, "kind": "oracle",
                                "sample": sample_desc(cfg, args.sample_layers)
                                + f"; wall {cb['wall_s'][0]:.1f} s"}
        cores = os.cpu_count() or 1
        if cores > 1:
            cb = run_cpu_baseline(args, steps=1, warmup=0, sample_layers=args.sample_layers,
                                  cores=cores)
            line["cpu_baseline_all_cores"] = {
                "value": round(1.0 / cb["scaled_s"][0], 4), "unit": "rounds/s", "cores": cores,
                "kind": "oracle",
                "sample": sample_desc(cfg, args.sample_layers)
                + f"; stage 5 spread over {cores} processes by (request, head); "
                  f"wall {cb['wall_s'][0]:.1f} s"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_only_topk(args):
    """Stage 1 alone on the workload's logits (for profiling it at a given batch
    without allocating the KV caches): prints microseconds per call, as one call
    per CUDA graph replay (graph launch included, as in stage_us) and as 20 calls
    back to back in one graph (each launch overlapping the previous one's tail,
    as in the round)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00487_gb300 as taps
    import workloads as W
    cfg = workload_config(args.workload, args.n_max, args.layers, args.mode)
    ldt = torch.bfloat16 if cfg.logits_dtype == "bf16" else torch.float32
    x = torch.from_numpy(W.make_logits(cfg)).to("cuda").to(ldt)
    B, L = x.shape[0], x.shape[1]
    outs = (torch.empty((B, L, cfg.K), dtype=torch.int32, device="cuda"),
            torch.empty((B, L, cfg.K), dtype=torch.float32, device="cuda"),
            torch.empty((B, L), dtype=torch.float32, device="cuda"),
            torch.empty((B, L), dtype=torch.float32, device="cuda"))
    ws = torch.zeros(taps.topk_marginals_workspace_bytes(B, L, cfg.V, cfg.K), dtype=torch.uint8,
                     device="cuda")
    s = torch.cuda.Stream()
    res = {}
    with torch.cuda.stream(s):   # the graphs are replayed, and timed, on s
        for name, calls in (("us_per_call_one_per_graph", 1), ("us_per_call_back_to_back", 20)):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                for _ in range(calls):
                    taps.taps_topk_marginals(x, cfg.K, out=outs, ws=ws)
            for _ in range(args.warmup):
                g.replay()
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s)
            for _ in range(args.steps):
                g.replay()
            b.record(s)
            torch.cuda.synchronize()
            res[name] = round(a.elapsed_time(b) / (args.steps * calls) * 1e3, 2)
    nbytes = x.numel() * x.element_size()
    print(json.dumps({"stage": "topk_marginals", "workload": cfg.name, **res, "bytes": nbytes,
                      "gbs_back_to_back": round(nbytes / res["us_per_call_back_to_back"] / 1e3, 1)}),
          flush=True)


def run_reference(args):
    """The oracle arm: rank 0 times the CPU oracle; other ranks exit."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    cfg = workload_config(args.workload, args.n_max, args.layers, args.mode)
    pairs = reference_attn_pairs(cfg, args.steps, args.warmup)
    cb = run_cpu_baseline(args, steps=args.steps, warmup=args.warmup, sample_layers=1,
                          attn_pairs=pairs)
    total = sum(cb["scaled_s"])
    value = args.steps / total
    line = {
        "impl": "reference",
        "metric": metric_name(args.workload),
        "value": round(value, 5), "unit": "rounds/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 2),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": f"synthetic (seeded; shapes of the {SHAPE_NAMES.get(args.workload, args.workload)} "
                "round, no weights or datasets)",
        "config": {"workload": f"{cfg.name}: B={cfg.B} L={cfg.L} V={cfg.V} K={cfg.K} "
                               f"n_max={cfg.n_max} layers={cfg.layers} Hq={cfg.Hq} Hkv={cfg.Hkv} "
                               f"D={cfg.D} ctx={cfg.ctx} page={cfg.page}",
                   "global_batch": cfg.B, "seq_len": cfg.ctx if isinstance(cfg.ctx, int) else None,
                   "parallelism": "none (host CPU)"},
        "cpu_baseline": {"value": round(value, 5), "unit": "rounds/s", "cores": 1,
                         "kind": "oracle", "sample": sample_desc(cfg, 1, pairs) + " per step"},
        "e2e": {"value": round(value, 5), "unit": "rounds/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="qwen3_8b")
    ap.add_argument("--n-max", type=int, default=None, help="node budget (default: workload's)")
    ap.add_argument("--layers", type=int, default=None, help="layers (default: workload's)")
    ap.add_argument("--sample-layers", type=int, default=3)
    ap.add_argument("--mode", default="taps",
                    choices=["taps", "no_scorer", "budget_fill", "ddtree"],
                    help="selection preset: TAPS, or one of its ablations")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the other configurations (budget sweep, Qwen3-4B, batch 32, long)")
    ap.add_argument("--cpu-cores", type=int, default=1, help=argparse.SUPPRESS)
    ap.add_argument("--attn-pairs", type=int, default=0, help=argparse.SUPPRESS)
    ap.add_argument("--only-topk", action="store_true",
                    help="time stage 1 alone on the workload's logits (profiling aid)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-child", action="store_true", help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.warmup < 3 and not args.cpu_child:
        args.warmup = 3
    if args.cpu_child:
        cpu_child(args)
    elif args.only_topk:
        run_only_topk(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
