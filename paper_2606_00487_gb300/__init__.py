"""TAPS per-round hot path on GB300 (sm_103a).

Python binding of libtaps.so, whose C ABI is declared in include/taps.h:
taps_topk_marginals, taps_score_reach, taps_select_subtree,
taps_build_tree_mask, taps_tree_verify_attn and taps_accept, the fused
taps_score_select_mask (stages 2-4 in one launch), plus the steps after
verification, taps_target_greedy_accept and taps_compact_accepted_kv.
Importing the package fails when the library has not been built (no CPU
fallback).
"""
from ._binding import (LIB_PATH, TAPS_DEVFAULT_PAGE, TapsError, lib, scorer_params,  # noqa: F401
                       taps_pack_kv_pages, taps_unpack_kv_pages,
                       taps_accept, taps_build_tree_mask, taps_score_reach, taps_select_subtree,
                       taps_score_select_mask,
                       taps_topk_marginals, taps_tree_verify_attn,
                       topk_marginals_workspace_bytes, tree_verify_attn_workspace_bytes,
                       taps_target_greedy_accept, target_greedy_accept_workspace_bytes,
                       taps_compact_accepted_kv)
from .round import MODES, RoundInputs, TapsRound  # noqa: F401

__all__ = ["taps_topk_marginals", "taps_score_reach", "taps_select_subtree",
           "taps_build_tree_mask", "taps_tree_verify_attn", "taps_accept", "TapsRound", "RoundInputs",
           "TapsError", "scorer_params", "MODES", "taps_target_greedy_accept",
           "taps_compact_accepted_kv", "taps_score_select_mask"]
