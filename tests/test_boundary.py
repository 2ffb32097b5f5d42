"""The C ABI: the library builds, loads without a GPU, exports every entry
point include/taps.h declares, and rejects bad arguments on the host before
any launch (no GPU needed for any of these)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "taps.h")


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    path = __graft_entry__._build_module().build()
    return ctypes.CDLL(path)


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(taps_\w+)\s*\(", src)))


def test_header_declares_the_six_stages():
    names = declared_functions()
    for f in ("taps_topk_marginals", "taps_score_reach", "taps_select_subtree",
              "taps_build_tree_mask", "taps_tree_verify_attn", "taps_accept"):
        assert f in names


def test_library_exports_every_declared_symbol(lib):
    missing = [f for f in declared_functions() if not hasattr(lib, f)]
    assert not missing, f"not exported: {missing}"


def test_status_strings(lib):
    lib.taps_status_string.restype = ctypes.c_char_p
    assert lib.taps_status_string(0) == b"ok"
    assert b"invalid" in lib.taps_status_string(1)
    assert lib.taps_version() >= 1


def _b():
    import paper_2606_00487_gb300._binding as tb
    return tb


def test_workspace_queries_are_host_only(lib):
    tb = _b()
    assert tb.topk_marginals_workspace_bytes(1, 16, 151936, 8) > 0
    assert tb.topk_marginals_workspace_bytes(1, 16, 151936, 33) == 0      # K > 32
    # attention combines context chunks on chip: never a workspace
    assert tb.tree_verify_attn_workspace_bytes(1, 64, 32, 8, 128, 4096) == 0
    assert tb.tree_verify_attn_workspace_bytes(32, 64, 32, 8, 128, 8192) == 0


FAKE = ctypes.c_void_p(0x1000)   # never dereferenced: every call below fails host checks


def test_topk_rejects_bad_arguments(lib):
    tb = _b()
    f = tb.lib.taps_topk_marginals
    ok = dict(B=1, L=2, V=100, K=4)
    def call(logits=FAKE, dtype=0, stride=100, B=1, L=2, V=100, K=4, ws=None, wsb=0):
        return f(logits, dtype, stride, B, L, V, K, FAKE, FAKE, FAKE, FAKE, ws, wsb, None)
    assert call(logits=None) == 1
    assert call(B=0) == 1
    assert call(stride=99) == 1
    assert call(dtype=7) == 1
    assert call(K=33) == 2
    assert call(K=101) == 2
    assert call(V=300000, stride=300000) == 2
    # a large row needs a workspace
    assert call(L=1, V=151936, stride=151936, ws=None) == 3


def test_score_select_mask_accept_reject_bad_arguments(lib):
    tb = _b()
    score = tb.lib.taps_score_reach
    nopath = (None, None, 0, None)
    sp = tb.ScorerParams(tb.TAPS_SCORER_MLP, 16, 32, 100, 3, None)
    assert score(FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), FAKE, *nopath,
                 None) == 1                                          # no weights
    sp = tb.ScorerParams(tb.TAPS_SCORER_MLP, 64, 32, 100, 3, FAKE)
    assert score(FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), FAKE, *nopath,
                 None) == 2                                          # E > 32
    sp = tb.ScorerParams(tb.TAPS_SCORER_MLP, 16, 32, 100, 2, FAKE)
    assert score(FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), FAKE, *nopath,
                 None) == 1                                          # max_depth <= L
    # the path list (Eq. 2 reach of given nodes) is all or nothing
    sp = tb.ScorerParams(tb.TAPS_SCORER_MARGINAL, 0, 0, 0, 0, None)
    assert score(FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), FAKE, FAKE, None, 3,
                 FAKE, None) == 1                                    # path_len missing
    assert score(FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), FAKE, FAKE, FAKE, 0,
                 FAKE, None) == 1                                    # M = 0 with paths
    assert score(FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), FAKE, None, None, 5,
                 None, None) == 1                                    # M without paths
    assert score(FAKE, FAKE, FAKE, FAKE, 2, 2, 4, ctypes.byref(sp), FAKE, FAKE, FAKE,
                 2 ** 30, FAKE, None) == 2                           # B * M too large
    sel = tb.lib.taps_select_subtree
    args = [FAKE] * 8
    for (l1, l2, tau, n), code in (((0.0, 0.1, 0.0, 8), 1), ((1.0, -0.1, 0.0, 8), 1),
                                   ((1.0, 0.1, -1.0, 8), 1), ((1.0, 0.1, 0.0, 0), 1),
                                   ((1.0, 0.1, 0.0, 513), 2)):
        p = tb.SelectParams(l1, l2, tau, n)
        assert sel(FAKE, FAKE, FAKE, FAKE, 1, 4, 4, ctypes.byref(p), *args, None) == code
    p = tb.SelectParams(1.0, 0.1, 0.0, 8)
    assert sel(FAKE, FAKE, FAKE, FAKE, 1, 32, 4, ctypes.byref(p), *args, None) == 2   # L > 31
    assert tb.lib.taps_build_tree_mask(FAKE, FAKE, 1, 600, FAKE, None) == 2
    # stages 2-4 in one launch: the same checks as the separate calls
    fused = tb.lib.taps_score_select_mask
    outs = [FAKE] * 10
    sp = tb.ScorerParams(tb.TAPS_SCORER_MARGINAL, 0, 0, 0, 0, None)
    for (l1, l2, tau, n), code in (((0.0, 0.1, 0.0, 8), 1), ((1.0, -0.1, 0.0, 8), 1),
                                   ((1.0, 0.1, 0.0, 0), 1), ((1.0, 0.1, 0.0, 513), 2)):
        p = tb.SelectParams(l1, l2, tau, n)
        assert fused(FAKE, FAKE, FAKE, FAKE, FAKE, 1, 4, 4, ctypes.byref(sp), ctypes.byref(p),
                     *outs, None) == code
    p = tb.SelectParams(1.0, 0.1, 0.0, 8)
    assert fused(FAKE, FAKE, FAKE, FAKE, FAKE, 1, 32, 4, ctypes.byref(sp), ctypes.byref(p),
                 *outs, None) == 2                                    # L > 31
    sp = tb.ScorerParams(tb.TAPS_SCORER_MLP, 16, 32, 100, 3, None)
    assert fused(FAKE, FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), ctypes.byref(p),
                 *outs, None) == 1                                    # no weights
    sp = tb.ScorerParams(7, 0, 0, 0, 0, None)
    assert fused(FAKE, FAKE, FAKE, FAKE, FAKE, 1, 2, 4, ctypes.byref(sp), ctypes.byref(p),
                 *outs, None) == 1                                    # unknown scorer
    assert fused(FAKE, FAKE, FAKE, FAKE, None, 1, 2, 4, ctypes.byref(sp), ctypes.byref(p),
                 *outs, None) == 1                                    # no ctx_len
    assert tb.lib.taps_build_tree_mask(None, FAKE, 1, 8, FAKE, None) == 1
    assert tb.lib.taps_accept(FAKE, FAKE, FAKE, FAKE, 1, 8, 40, FAKE, FAKE, FAKE, None) == 2
    assert tb.lib.taps_accept(FAKE, FAKE, None, FAKE, 1, 8, 4, FAKE, FAKE, FAKE, None) == 1


def test_attention_rejects_bad_arguments(lib):
    tb = _b()
    f = tb.lib.taps_tree_verify_attn
    def call(D=128, P=16, Hq=32, Hkv=8, scale=0.1, ws=None, wsb=0, q=FAKE, B=1, n=64, ctx=4096):
        return f(q, FAKE, FAKE, 100, FAKE, 10, FAKE, FAKE, FAKE, B, n, Hq, Hkv, D, P, scale,
                 ctx, FAKE, None, ws, wsb, None, None)
    assert call(q=None) == 1
    assert call(scale=0.0) == 1
    assert call(Hq=30) == 1
    assert call(D=96) == 2
    assert call(P=32) == 2
    assert call(Hq=80, Hkv=8) == 2                                   # group 10 > 8
    assert call(Hq=24, Hkv=8) == 2                                   # group 3
    assert call(ctx=65536 - 63) == 2                                 # ctx + n_max > 65536


def test_target_greedy_accept_rejects_bad_arguments(lib):
    tb = _b()
    f = tb.lib.taps_target_greedy_accept
    WS = ctypes.c_void_p(0x10000)      # 256-byte aligned, never dereferenced
    nb = tb.target_greedy_accept_workspace_bytes(2, 64)
    assert nb >= 2 * 64 * 8 and tb.target_greedy_accept_workspace_bytes(0, 64) == 0

    def call(x=FAKE, dtype=1, stride=1000, B=2, n=64, V=1000, L=16, ws=WS, wsb=nb):
        return f(x, dtype, stride, B, n, V, FAKE, FAKE, FAKE, L, FAKE, FAKE, FAKE, FAKE, ws, wsb,
                 None)
    assert call(x=None) == 1
    assert call(dtype=7) == 1
    assert call(stride=999) == 1
    assert call(V=0) == 1
    assert call(n=600) == 2
    assert call(L=32) == 2
    assert call(ws=None) == 3
    assert call(wsb=nb - 1) == 3
    assert call(ws=ctypes.c_void_p(0x10010)) == 3                     # not 256-byte aligned


def test_compact_accepted_kv_rejects_bad_arguments(lib):
    tb = _b()
    f = tb.lib.taps_compact_accepted_kv
    ptrs = (ctypes.c_void_p * 2)(0x1000, 0x2000)

    def call(k=ptrs, v=ptrs, layers=2, pages=10, L=16, Hkv=8, D=128, P=16, bt=FAKE):
        return f(k, v, layers, pages, bt, 4, FAKE, FAKE, FAKE, 1, L, Hkv, D, P, None, None)
    assert call(k=None) == 1
    assert call(bt=None) == 1
    assert call(layers=0) == 1
    assert call(pages=0) == 1
    assert call(layers=129) == 2
    assert call(L=32) == 2
    assert call(D=96) == 2
    assert call(P=32) == 2
    bad = (ctypes.c_void_p * 2)(0x1000, 0x2008)                        # not 16-byte aligned
    assert call(v=bad) == 1
