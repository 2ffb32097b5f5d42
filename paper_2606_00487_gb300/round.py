"""One TAPS decoding round over preallocated device buffers.

Sequencing only: the six stages run in the order of Sec. 4.1 (top-K
marginals -> scoring -> selection -> mask -> per-layer tree verification ->
acceptance), each as one call into libtaps.so on the caller's stream. With
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
        self.sel = {"n_nodes": torch.empty(B, dtype=i32, device=dev)}
        for k in ("parent", "depth", "token", "slot", "pos_id"):
            self.sel[k] = torch.empty((B, n_max), dtype=i32, device=dev)
        for k in ("reach", "utility"):
            self.sel[k] = torch.empty((B, n_max), dtype=f32, device=dev)
        self.mask = torch.empty((B, n_max, (n_max + 31) // 32), dtype=i32, device=dev)
        self.accept_len = torch.empty(B, dtype=i32, device=dev)
        self.accepted_nodes = torch.empty((B, L + 1), dtype=i32, device=dev)
        self.bonus_tok = torch.empty(B, dtype=i32, device=dev)
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
        self.launches_per_select = 4
        self.launches_per_layer = 1 + (1 if tb.lib.taps_tree_verify_attn_workspace_bytes(
            B, n_max, Hq, Hkv, D, max_ctx) > 0 else 0)

    def select(self, logits, root_tok, ctx_len, stream=None):
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

    def run(self, logits, root_tok, ctx_len, layers, outs, target_tok, stream=None):
        """layers: list of (q, k_cache, v_cache, block_table); outs: one output per layer."""
        self.select(logits, root_tok, ctx_len, stream)
        for (q, kc, vc, bt), o in zip(layers, outs):
            self.verify_layer(q, kc, vc, bt, ctx_len, o, stream)
        self.accept(target_tok, stream)
