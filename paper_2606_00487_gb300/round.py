"""One TAPS decoding round over preallocated device buffers.

Sequencing only: the six stages run in the order of Sec. 4.1 (top-K
marginals -> scoring -> selection -> mask -> per-layer tree verification ->
acceptance) as calls into libtaps.so on the caller's stream; scoring,
selection and the mask are one call (taps_score_select_mask, whose selection
and mask share one launch). With
the target's verify logits at hand, acceptance can instead take the greedy
token of every node from them (accept_greedy), and commit_kv moves the
accepted path's K/V into place for the next round. All
outputs and workspaces are allocated once here, so a round can be captured
in a CUDA graph and replayed.
"""
from __future__ import annotations

import torch

from . import _binding as tb


# Selection presets. "taps" is the method; "no_scorer" and "budget_fill" are
# the two ablations of Sec. 5.3 (marginal confidence instead of the scorer;
# the scorer without cost-aware pruning, lambda2 = 0 and tau = 0); "ddtree"
# ranks paths by the product of the drafter's marginal probabilities and fills
# the budget, the DDTree-style tree of Sec. 3.1.
MODES = {
    "taps": {"scorer_kind": "mlp"},
    "no_scorer": {"scorer_kind": "marginal"},
    "budget_fill": {"scorer_kind": "mlp", "lambda2": 0.0, "tau": 0.0},
    "ddtree": {"scorer_kind": "marginal_product", "lambda2": 0.0, "tau": 0.0},
}


class TapsRound:
    def __init__(self, *, B, L, V, K, n_max, Hq, Hkv, D, max_ctx, device, scorer_kind="mlp",
                 scorer_weights=None, emb_dim=16, hidden=32, max_depth=None, lambda1=1.0,
                 lambda2=0.1, tau=0.0, mode=None):
        if mode is not None:
            preset = MODES[mode]
            scorer_kind = preset["scorer_kind"]
            lambda2 = preset.get("lambda2", lambda2)
            tau = preset.get("tau", tau)
        self.mode = mode or "taps"
        dev = torch.device(device)
        self.B, self.L, self.V, self.K, self.n_max = B, L, V, K, n_max
        self.Hq, self.Hkv, self.D, self.max_ctx = Hq, Hkv, D, max_ctx
        self.lambda1, self.lambda2, self.tau = lambda1, lambda2, tau
        self.device = dev
        i32, f32 = torch.int32, torch.float32
        self.ids = torch.empty((B, L, K), dtype=i32, device=dev)
        self.logp = torch.empty((B, L, K), dtype=f32, device=dev)
        self.lse = torch.empty((B, L), dtype=f32, device=dev)
        self.entropy = torch.empty((B, L), dtype=f32, device=dev)
        self.q_cond = torch.empty((B, L, K, K), dtype=f32, device=dev)
        # the round's results (n_nodes, accept_len, bonus_tok, accepted_nodes)
        # live in one int32 buffer, so that the host reads them in one copy
        self.results = torch.empty(3 * B + B * (L + 1), dtype=i32, device=dev)
        self.sel = {"n_nodes": self.results[0:B]}
        for k in ("parent", "depth", "token", "slot", "pos_id"):
            self.sel[k] = torch.empty((B, n_max), dtype=i32, device=dev)
        for k in ("reach", "utility"):
            self.sel[k] = torch.empty((B, n_max), dtype=f32, device=dev)
        self.mask = torch.empty((B, n_max, (n_max + 31) // 32), dtype=i32, device=dev)
        self.accept_len = self.results[B:2 * B]
        self.accepted_nodes = self.results[3 * B:].view(B, L + 1)
        self.bonus_tok = self.results[2 * B:3 * B]
        self.status = torch.zeros(1, dtype=i32, device=dev)
        self.target_tok = torch.empty((B, n_max), dtype=i32, device=dev)
        nb = tb.target_greedy_accept_workspace_bytes(B, n_max)
        self.ws_target = torch.zeros(max(nb, 1), dtype=torch.uint8, device=dev)
        nb = tb.topk_marginals_workspace_bytes(B, L, V, K)
        self.ws_topk = torch.zeros(max(nb, 1), dtype=torch.uint8, device=dev)
        nb = tb.tree_verify_attn_workspace_bytes(B, n_max, Hq, Hkv, D, max_ctx)
        self.ws_attn = torch.zeros(max(nb, 1), dtype=torch.uint8, device=dev)
        if scorer_kind in ("marginal", "marginal_product"):
            self.scorer = tb.scorer_params(scorer_kind)
        else:
            self.scorer_weights = scorer_weights
            self.scorer = tb.scorer_params("mlp", scorer_weights, emb_dim, hidden, V,
                                           max_depth if max_depth is not None else L + 1)
        self.launches_per_select = 3
        self.launches_per_layer = 1 + (1 if tb.lib.taps_tree_verify_attn_workspace_bytes(
            B, n_max, Hq, Hkv, D, max_ctx) > 0 else 0)

    def select(self, logits, root_tok, ctx_len, stream=None):
        """Stage 1, scoring, then selection and mask in one launch."""
        tb.taps_topk_marginals(logits, self.K, out=(self.ids, self.logp, self.lse, self.entropy),
                               ws=self.ws_topk, stream=stream)
        tb.taps_score_select_mask(root_tok, self.ids, self.logp, self.entropy, ctx_len,
                                  self.scorer, self.lambda1, self.lambda2, self.tau, self.n_max,
                                  out=(self.q_cond, self.sel, self.mask), stream=stream)

    def select_staged(self, logits, root_tok, ctx_len, stream=None):
        """The same results with one launch per stage (stages 1-4)."""
        tb.taps_topk_marginals(logits, self.K, out=(self.ids, self.logp, self.lse, self.entropy),
                               ws=self.ws_topk, stream=stream)
        tb.taps_score_reach(root_tok, self.ids, self.logp, self.entropy, self.scorer,
                            out=self.q_cond, stream=stream)
        tb.taps_select_subtree(self.q_cond, self.ids, root_tok, ctx_len, self.lambda1,
                               self.lambda2, self.tau, self.n_max, out=self.sel, stream=stream)
        tb.taps_build_tree_mask(self.sel["parent"], self.sel["n_nodes"], out=self.mask,
                                stream=stream)

    def verify_layer(self, q, k_cache, v_cache, block_table, ctx_len, out, stream=None):
        tb.taps_tree_verify_attn(q, k_cache, v_cache, block_table, ctx_len, self.sel["n_nodes"],
                                 self.mask, self.max_ctx, out=out, status=self.status,
                                 ws=self.ws_attn, stream=stream)

    def accept(self, target_tok, stream=None):
        tb.taps_accept(self.sel["parent"], self.sel["token"], self.sel["n_nodes"], target_tok,
                       self.L, out=(self.accept_len, self.accepted_nodes, self.bonus_tok),
                       stream=stream)

    def accept_greedy(self, verify_logits, stream=None):
        """Target greedy token of every node (argmax of its verify logits
        [B, n_max, V]) fused with acceptance; fills target_tok as well."""
        tb.taps_target_greedy_accept(verify_logits, self.sel["parent"], self.sel["token"],
                                     self.sel["n_nodes"], self.L,
                                     out=(self.target_tok, self.accept_len, self.accepted_nodes,
                                          self.bonus_tok),
                                     ws=self.ws_target, stream=stream)

    def commit_kv(self, k_layers, v_layers, block_table, ctx_len, stream=None):
        """Move the accepted path's K/V to positions ctx_len .. ctx_len +
        accept_len in every layer; the caller then advances ctx_len by
        accept_len + 1."""
        tb.taps_compact_accepted_kv(k_layers, v_layers, block_table, ctx_len,
                                    self.accepted_nodes, self.accept_len, status=self.status,
                                    stream=stream)

    def download(self, host_results, stream=None):
        """Copy the round's results (n_nodes, accept_len, bonus_tok, then
        accepted_nodes row by row, int32) into a pinned host tensor of
        results.numel() elements: one device-to-host copy."""
        with torch.cuda.stream(stream or torch.cuda.current_stream(self.device)):
            host_results.copy_(self.results, non_blocking=True)

    def run(self, logits, root_tok, ctx_len, layers, outs, target_tok, stream=None):
        """layers: list of (q, k_cache, v_cache, block_table); outs: one output per layer."""
        self.select(logits, root_tok, ctx_len, stream)
        for (q, kc, vc, bt), o in zip(layers, outs):
            self.verify_layer(q, kc, vc, bt, ctx_len, o, stream)
        self.accept(target_tok, stream)

    def capture_round_graph(self, inputs, ctx_len, layers, outs, host_results, groups=4,
                            stream=None):
        """Capture one whole round with its host copies as one CUDA graph and
        return it; each ``replay()`` then runs a round from what the host
        buffer of ``inputs`` (a RoundInputs) holds at that moment.

        In the graph: the head (logits, root and target tokens) uploads on the
        capture stream; the queries upload on a second stream in ``groups``
        groups of layers while stages 1-4 run, and each group of verification
        layers waits only for its own queries; then acceptance and one
        device-to-host copy of ``results`` into ``host_results`` (pinned,
        results.numel() int32). ``layers`` is a list of (q, k_cache, v_cache,
        block_table) whose q must be the device views ``inputs.dev["q"][i]``,
        so that the graph's uploads feed them; ``outs`` holds one output per
        layer. ``stream`` is the capture stream (a fresh one by default; it
        must not be the legacy default stream). The caller synchronizes the
        stream it replays on before reading ``host_results``."""
        if len(layers) != inputs.layers or len(outs) != inputs.layers:
            raise ValueError("one (q, k_cache, v_cache, block_table) and one output per layer")
        for li, (q, _, _, _) in enumerate(layers):
            if q.data_ptr() != inputs.dev["q"][li].data_ptr():
                raise ValueError(f"layer {li}: q is not the upload buffer's view of that layer")
        if host_results.numel() != self.results.numel() or not host_results.is_pinned():
            raise ValueError("host_results must be pinned with results.numel() elements")
        groups = max(1, min(int(groups), inputs.layers))
        per = (inputs.layers + groups - 1) // groups
        spans = [(a, min(inputs.layers, a + per)) for a in range(0, inputs.layers, per)]
        s = stream or torch.cuda.Stream(device=self.device)
        cs = torch.cuda.Stream(device=self.device)
        evs = [torch.cuda.Event() for _ in spans]
        logits, root, target = inputs.dev["logits"], inputs.dev["root_tok"], inputs.dev["target_tok"]
        s.wait_stream(torch.cuda.current_stream(self.device))
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            cs.wait_stream(s)
            inputs.upload_head(s)
            for (a, b), e in zip(spans, evs):
                inputs.upload_queries(cs, a, b)
                e.record(cs)
            self.select(logits, root, ctx_len, s)
            for (a, b), e in zip(spans, evs):
                s.wait_event(e)
                for li in range(a, b):
                    q, kc, vc, bt = layers[li]
                    self.verify_layer(q, kc, vc, bt, ctx_len, outs[li], s)
            self.accept(target, s)
            s.wait_stream(cs)
            self.download(host_results, s)
        torch.cuda.current_stream(self.device).wait_stream(s)
        return g


class RoundInputs:
    """A round's inputs in one device buffer mirrored by one pinned host
    buffer: the drafter's logits [B, L, V], the root tokens [B], the target's
    greedy tokens [B, n_max] (the head, needed from the first stage on), then
    every layer's tree-node queries [layers, B, n_max, Hq, D] bf16 (needed
    only by verification). ``dev[name]`` and ``host[name]`` are views of the
    two buffers. upload() copies everything at once; upload_head() and
    upload_queries() copy the two parts, so that the queries can travel on
    another stream while the selection stages run."""

    def __init__(self, *, B, L, V, n_max, Hq, D, layers, logits_dtype, device):
        parts = [("logits", (B, L, V), logits_dtype),
                 ("root_tok", (B,), torch.int32),
                 ("target_tok", (B, n_max), torch.int32),
                 ("q", (layers, B, n_max, Hq, D), torch.bfloat16)]
        offs, o = {}, 0
        for name, shape, dt in parts:
            n = 1
            for x in shape:
                n *= x
            nbytes = n * torch.empty((), dtype=dt).element_size()
            offs[name] = (o, nbytes, shape, dt)
            o += (nbytes + 255) // 256 * 256
        self.nbytes = o
        self.payload_bytes = sum(v[1] for v in offs.values())
        self.device_buf = torch.empty(o, dtype=torch.uint8, device=device)
        self.host_buf = torch.empty(o, dtype=torch.uint8, pin_memory=True)

        def views(buf):
            return {name: buf[a:a + nb].view(dt).view(shape)
                    for name, (a, nb, shape, dt) in offs.items()}

        self.dev = views(self.device_buf)
        self.host = views(self.host_buf)
        self.head_bytes = offs["q"][0]
        self.layers = layers
        self.layer_bytes = offs["q"][1] // layers

    def _copy(self, a, b, stream):
        with torch.cuda.stream(stream or torch.cuda.current_stream(self.device_buf.device)):
            self.device_buf[a:b].copy_(self.host_buf[a:b], non_blocking=True)

    def upload(self, stream=None):
        """Host buffer -> device buffer, asynchronously on ``stream``."""
        self._copy(0, self.nbytes, stream)

    def upload_head(self, stream=None):
        """Logits, root tokens and target tokens only."""
        self._copy(0, self.head_bytes, stream)

    def upload_queries(self, stream=None, first=0, last=None):
        """The tree-node queries of layers [first, last) only (default: all)."""
        last = self.layers if last is None else last
        a = self.head_bytes + first * self.layer_bytes
        b = self.nbytes if last == self.layers else self.head_bytes + last * self.layer_bytes
        self._copy(a, b, stream)
