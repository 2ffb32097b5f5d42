"""ctypes binding of libtaps.so (C ABI declared in include/taps.h).

Argument marshalling only: every function checks shapes and dtypes of the
torch tensors it is given, allocates outputs (torch is used for device
memory and streams), and passes raw device pointers plus the current CUDA
stream to the library. All computation happens in the library's kernels.
There is no CPU fallback: importing this module fails loudly when the
library has not been built.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libtaps.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is not built; run paper_2606_00487_gb300.build.build() "
                      "(or __graft_entry__.build()) first")

lib = ctypes.CDLL(LIB_PATH)

TAPS_OK = 0
TAPS_F32, TAPS_BF16 = 0, 1
TAPS_SCORER_MARGINAL, TAPS_SCORER_MLP, TAPS_SCORER_MARGINAL_PRODUCT = 0, 1, 2
TAPS_DEVFAULT_PAGE = 1
STATUS_NAMES = {0: "TAPS_OK", 1: "TAPS_ERR_INVALID_ARG", 2: "TAPS_ERR_UNSUPPORTED",
                3: "TAPS_ERR_WORKSPACE", 4: "TAPS_ERR_CUDA", 5: "TAPS_ERR_DEVICE"}


class TapsError(RuntimeError):
    def __init__(self, fn: str, status: int):
        msg = lib.taps_status_string(status).decode()
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)} ({msg})")
        self.status = status


class ScorerParams(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("emb_dim", ctypes.c_int), ("hidden", ctypes.c_int),
                ("vocab", ctypes.c_int), ("max_depth", ctypes.c_int),
                ("weights", ctypes.c_void_p)]


class SelectParams(ctypes.Structure):
    _fields_ = [("lambda1", ctypes.c_float), ("lambda2", ctypes.c_float),
                ("tau", ctypes.c_float), ("n_max", ctypes.c_int)]


_P, _I, _I64, _F, _SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t

lib.taps_status_string.argtypes = [_I]
lib.taps_status_string.restype = ctypes.c_char_p
lib.taps_version.restype = _I
lib.taps_topk_marginals_workspace_bytes.argtypes = [_I, _I, _I, _I]
lib.taps_topk_marginals_workspace_bytes.restype = _SZ
lib.taps_topk_marginals.argtypes = [_P, _I, _I64, _I, _I, _I, _I, _P, _P, _P, _P, _P, _SZ, _P]
lib.taps_topk_marginals.restype = _I
lib.taps_score_reach.argtypes = [_P, _P, _P, _P, _I, _I, _I, ctypes.POINTER(ScorerParams), _P,
                                 _P, _P, _I, _P, _P]
lib.taps_score_reach.restype = _I
lib.taps_select_subtree.argtypes = [_P, _P, _P, _P, _I, _I, _I, ctypes.POINTER(SelectParams),
                                    _P, _P, _P, _P, _P, _P, _P, _P, _P]
lib.taps_select_subtree.restype = _I
lib.taps_build_tree_mask.argtypes = [_P, _P, _I, _I, _P, _P]
lib.taps_build_tree_mask.restype = _I
lib.taps_tree_verify_attn_workspace_bytes.argtypes = [_I, _I, _I, _I, _I, _I]
lib.taps_tree_verify_attn_workspace_bytes.restype = _SZ
lib.taps_tree_verify_attn.argtypes = [_P, _P, _P, _I64, _P, _I, _P, _P, _P, _I, _I, _I, _I, _I,
                                      _I, _F, _I, _P, _P, _P, _SZ, _P, _P]
lib.taps_tree_verify_attn.restype = _I
lib.taps_accept.argtypes = [_P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P]
lib.taps_accept.restype = _I


def _check(fn: str, status: int):
    if status != TAPS_OK:
        raise TapsError(fn, status)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None, device=None):
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t, dtype, shape=None, name="tensor"):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


_WS = {}


def workspace(nbytes: int, device, tag: str, stream=None) -> torch.Tensor | None:
    """Zero-filled workspace cached per (device, stream, tag); grown on demand.

    The kernels leave the counters they use back at zero, so a cached
    workspace stays valid between calls on the same stream.
    """
    if nbytes == 0:
        return None
    dev = torch.device(device)
    sid = (stream or torch.cuda.current_stream(dev)).cuda_stream
    key = (dev.index, sid, tag)
    buf = _WS.get(key)
    if buf is None or buf.numel() < nbytes:
        buf = torch.zeros(nbytes + 256, dtype=torch.uint8, device=dev)
        _WS[key] = buf
    off = (-buf.data_ptr()) % 256
    return buf[off:off + nbytes]


# ---------------------------------------------------------------------------
# the six entry points
# ---------------------------------------------------------------------------

def topk_marginals_workspace_bytes(B, L, V, K) -> int:
    return int(lib.taps_topk_marginals_workspace_bytes(B, L, V, K))


def taps_topk_marginals(logits: torch.Tensor, K: int, out=None, ws=None, stream=None):
    """Stage 1: (ids [B,L,K] i32, logp [B,L,K] f32, lse [B,L] f32, entropy [B,L] f32)."""
    if logits.dtype not in (torch.float32, torch.bfloat16) or not logits.is_cuda:
        raise TypeError("logits must be a CUDA float32 or bfloat16 tensor")
    B, L, V = logits.shape
    if logits.stride(2) != 1 or logits.stride(0) != L * logits.stride(1):
        raise ValueError("logits rows must be unit-stride with a uniform row stride")
    dev = logits.device
    if out is None:
        out = (torch.empty((B, L, K), dtype=torch.int32, device=dev),
               torch.empty((B, L, K), dtype=torch.float32, device=dev),
               torch.empty((B, L), dtype=torch.float32, device=dev),
               torch.empty((B, L), dtype=torch.float32, device=dev))
    ids, logp, lse, ent = out
    nbytes = topk_marginals_workspace_bytes(B, L, V, K)
    if ws is None:
        ws = workspace(nbytes, dev, "topk", stream)
    dtype = TAPS_F32 if logits.dtype == torch.float32 else TAPS_BF16
    st = lib.taps_topk_marginals(_ptr(logits), dtype, logits.stride(1), B, L, V, K, _ptr(ids),
                                 _ptr(logp), _ptr(lse), _ptr(ent), _ptr(ws),
                                 0 if ws is None else ws.numel(), _stream(stream, dev))
    _check("taps_topk_marginals", st)
    return ids, logp, lse, ent


def scorer_params(kind: str, weights: torch.Tensor | None = None, emb_dim=0, hidden=0, vocab=0,
                  max_depth=0) -> ScorerParams:
    if kind == "marginal":
        return ScorerParams(TAPS_SCORER_MARGINAL, 0, 0, 0, 0, None)
    if kind == "marginal_product":
        return ScorerParams(TAPS_SCORER_MARGINAL_PRODUCT, 0, 0, 0, 0, None)
    if kind != "mlp":
        raise ValueError(f"unknown scorer kind {kind!r}")
    _need(weights, torch.float32, name="scorer weights")
    F = 3 * emb_dim + 2
    expect = vocab * emb_dim + max_depth * emb_dim + hidden * F + 2 * hidden + 1
    if weights.numel() != expect:
        raise ValueError(f"scorer weights must hold {expect} floats, got {weights.numel()}")
    return ScorerParams(TAPS_SCORER_MLP, emb_dim, hidden, vocab, max_depth, weights.data_ptr())


def taps_score_reach(root_tok, topk_ids, topk_logp, entropy, params: ScorerParams, out=None,
                     paths=None, path_len=None, path_reach=None, stream=None):
    """Stage 2: q_cond [B, L, K, K] f32. With ``paths`` [B, M, L] uint8 slots and
    ``path_len`` [B, M] int32, also the reach of those nodes (Eq. 2), returned as
    (q_cond, path_reach [B, M] f32)."""
    B, L, K = topk_ids.shape
    _need(root_tok, torch.int32, (B,), "root_tok")
    _need(topk_ids, torch.int32, (B, L, K), "topk_ids")
    _need(topk_logp, torch.float32, (B, L, K), "topk_logp")
    _need(entropy, torch.float32, (B, L), "entropy")
    dev = topk_ids.device
    q = out if out is not None else torch.empty((B, L, K, K), dtype=torch.float32, device=dev)
    M = 0
    if paths is not None:
        M = paths.shape[1] if paths.dim() == 3 else -1
        _need(paths, torch.uint8, (B, M, L), "paths")
        _need(path_len, torch.int32, (B, M), "path_len")
        if path_reach is None:
            path_reach = torch.empty((B, M), dtype=torch.float32, device=dev)
        _need(path_reach, torch.float32, (B, M), "path_reach")
    st = lib.taps_score_reach(_ptr(root_tok), _ptr(topk_ids), _ptr(topk_logp), _ptr(entropy),
                              B, L, K, ctypes.byref(params), _ptr(q), _ptr(paths),
                              _ptr(path_len), M, _ptr(path_reach) if paths is not None else None,
                              _stream(stream, dev))
    _check("taps_score_reach", st)
    return (q, path_reach) if paths is not None else q


def taps_select_subtree(q_cond, topk_ids, root_tok, ctx_len, lambda1, lambda2, tau, n_max,
                        out=None, stream=None):
    """Stage 3: dict of n_nodes [B] and [B, n_max] parent/depth/token/slot/pos_id/reach/utility."""
    B, L, K = topk_ids.shape
    _need(q_cond, torch.float32, (B, L, K, K), "q_cond")
    _need(topk_ids, torch.int32, (B, L, K), "topk_ids")
    _need(root_tok, torch.int32, (B,), "root_tok")
    _need(ctx_len, torch.int32, (B,), "ctx_len")
    dev = topk_ids.device
    if out is None:
        out = {"n_nodes": torch.empty(B, dtype=torch.int32, device=dev)}
        for k in ("parent", "depth", "token", "slot", "pos_id"):
            out[k] = torch.empty((B, n_max), dtype=torch.int32, device=dev)
        for k in ("reach", "utility"):
            out[k] = torch.empty((B, n_max), dtype=torch.float32, device=dev)
    p = SelectParams(float(lambda1), float(lambda2), float(tau), int(n_max))
    st = lib.taps_select_subtree(_ptr(q_cond), _ptr(topk_ids), _ptr(root_tok), _ptr(ctx_len),
                                 B, L, K, ctypes.byref(p), _ptr(out["n_nodes"]),
                                 _ptr(out["parent"]), _ptr(out["depth"]), _ptr(out["token"]),
                                 _ptr(out["slot"]), _ptr(out["pos_id"]), _ptr(out["reach"]),
                                 _ptr(out["utility"]), _stream(stream, dev))
    _check("taps_select_subtree", st)
    return out


lib.taps_score_select_mask.argtypes = [_P, _P, _P, _P, _P, _I, _I, _I,
                                       ctypes.POINTER(ScorerParams), ctypes.POINTER(SelectParams),
                                       _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P]
lib.taps_score_select_mask.restype = _I


def taps_score_select_mask(root_tok, topk_ids, topk_logp, entropy, ctx_len, params: ScorerParams,
                           lambda1, lambda2, tau, n_max, out=None, stream=None):
    """Stages 2-4 (scoring, then selection and mask in one launch): returns (q_cond [B, L, K, K],
    selection dict as taps_select_subtree, mask [B, n_max, ceil(n_max/32)]).
    ``out`` = (q_cond, sel, mask) preallocated, or None."""
    B, L, K = topk_ids.shape
    _need(root_tok, torch.int32, (B,), "root_tok")
    _need(topk_ids, torch.int32, (B, L, K), "topk_ids")
    _need(topk_logp, torch.float32, (B, L, K), "topk_logp")
    _need(entropy, torch.float32, (B, L), "entropy")
    _need(ctx_len, torch.int32, (B,), "ctx_len")
    dev = topk_ids.device
    W = (n_max + 31) // 32
    if out is None:
        sel = {"n_nodes": torch.empty(B, dtype=torch.int32, device=dev)}
        for k in ("parent", "depth", "token", "slot", "pos_id"):
            sel[k] = torch.empty((B, n_max), dtype=torch.int32, device=dev)
        for k in ("reach", "utility"):
            sel[k] = torch.empty((B, n_max), dtype=torch.float32, device=dev)
        out = (torch.empty((B, L, K, K), dtype=torch.float32, device=dev), sel,
               torch.empty((B, n_max, W), dtype=torch.int32, device=dev))
    q, sel, mask = out
    _need(q, torch.float32, (B, L, K, K), "q_cond")
    _need(mask, torch.int32, (B, n_max, W), "mask")
    p = SelectParams(float(lambda1), float(lambda2), float(tau), int(n_max))
    st = lib.taps_score_select_mask(_ptr(root_tok), _ptr(topk_ids), _ptr(topk_logp),
                                    _ptr(entropy), _ptr(ctx_len), B, L, K, ctypes.byref(params),
                                    ctypes.byref(p), _ptr(q), _ptr(sel["n_nodes"]),
                                    _ptr(sel["parent"]), _ptr(sel["depth"]), _ptr(sel["token"]),
                                    _ptr(sel["slot"]), _ptr(sel["pos_id"]), _ptr(sel["reach"]),
                                    _ptr(sel["utility"]), _ptr(mask), _stream(stream, dev))
    _check("taps_score_select_mask", st)
    return q, sel, mask


def taps_build_tree_mask(parent, n_nodes, out=None, stream=None):
    """Stage 4: mask [B, n_max, ceil(n_max/32)] uint32 (returned as int32 storage)."""
    B, n_max = parent.shape
    _need(parent, torch.int32, (B, n_max), "parent")
    _need(n_nodes, torch.int32, (B,), "n_nodes")
    W = (n_max + 31) // 32
    mask = out if out is not None else torch.empty((B, n_max, W), dtype=torch.int32,
                                                    device=parent.device)
    st = lib.taps_build_tree_mask(_ptr(parent), _ptr(n_nodes), B, n_max, _ptr(mask),
                                  _stream(stream, parent.device))
    _check("taps_build_tree_mask", st)
    return mask


def tree_verify_attn_workspace_bytes(B, n_max, Hq, Hkv, D, max_ctx) -> int:
    return int(lib.taps_tree_verify_attn_workspace_bytes(B, n_max, Hq, Hkv, D, max_ctx))


def taps_tree_verify_attn(q, k_cache, v_cache, block_table, ctx_len, n_nodes, mask, max_ctx,
                          scale=None, out=None, lse_out=None, want_lse=False, status=None,
                          ws=None, stream=None):
    """Stage 5: out [B, n_max, Hq, D] bf16 (and lse [B, n_max, Hq] f32 if requested)."""
    B, n_max, Hq, D = q.shape
    num_pages, Hkv, P, Dk = k_cache.shape
    _need(q, torch.bfloat16, None, "q")
    _need(k_cache, torch.bfloat16, None, "k_cache")
    _need(v_cache, torch.bfloat16, tuple(k_cache.shape), "v_cache")
    if Dk != D:
        raise ValueError("q and k_cache head dims differ")
    _need(block_table, torch.int32, None, "block_table")
    if block_table.dim() != 2 or block_table.shape[0] != B:
        raise ValueError("block_table must be [B, max_pages]")
    _need(ctx_len, torch.int32, (B,), "ctx_len")
    _need(n_nodes, torch.int32, (B,), "n_nodes")
    _need(mask, torch.int32, (B, n_max, (n_max + 31) // 32), "mask")
    dev = q.device
    if out is None:
        out = torch.empty_like(q)
    if want_lse and lse_out is None:
        lse_out = torch.empty((B, n_max, Hq), dtype=torch.float32, device=dev)
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    nbytes = tree_verify_attn_workspace_bytes(B, n_max, Hq, Hkv, D, int(max_ctx))
    if ws is None:
        ws = workspace(nbytes, dev, "attn", stream)
    st = lib.taps_tree_verify_attn(_ptr(q), _ptr(k_cache), _ptr(v_cache), num_pages,
                                   _ptr(block_table), block_table.shape[1], _ptr(ctx_len),
                                   _ptr(n_nodes), _ptr(mask), B, n_max, Hq, Hkv, D, P,
                                   float(scale), int(max_ctx), _ptr(out), _ptr(lse_out),
                                   _ptr(ws), 0 if ws is None else ws.numel(), _ptr(status),
                                   _stream(stream, dev))
    _check("taps_tree_verify_attn", st)
    return (out, lse_out) if want_lse or lse_out is not None else out


def taps_accept(parent, token, n_nodes, target_tok, L, out=None, stream=None):
    """Stage 6: (accept_len [B], accepted_nodes [B, L+1], bonus_tok [B]) int32."""
    B, n_max = parent.shape
    for t, nm in ((parent, "parent"), (token, "token"), (target_tok, "target_tok")):
        _need(t, torch.int32, (B, n_max), nm)
    _need(n_nodes, torch.int32, (B,), "n_nodes")
    dev = parent.device
    if out is None:
        out = (torch.empty(B, dtype=torch.int32, device=dev),
               torch.empty((B, L + 1), dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev))
    alen, nodes, bonus = out
    st = lib.taps_accept(_ptr(parent), _ptr(token), _ptr(n_nodes), _ptr(target_tok), B, n_max,
                         L, _ptr(alen), _ptr(nodes), _ptr(bonus), _stream(stream, dev))
    _check("taps_accept", st)
    return alen, nodes, bonus


# ---------------------------------------------------------------------------
# allocation-free variant of stage 1 (no counterpart in the paper)
# ---------------------------------------------------------------------------

lib.taps_topk_marginals_noalloc.argtypes = [_P, _I, _I64, _I, _I, _I, _I, _P, _P, _P, _P, _P]
lib.taps_topk_marginals_noalloc.restype = _I


def taps_topk_marginals_noalloc(logits: torch.Tensor, K: int, out, stream=None):
    """Stage 1 for callers that cannot allocate device memory: the library
    keeps its partial records in a fixed 2 MiB device array instead of a
    workspace. ``out`` = (ids, logp, lse, entropy) must be preallocated by the
    caller. Calls that overlap on the GPU share that array and race."""
    if logits.dtype not in (torch.float32, torch.bfloat16) or not logits.is_cuda:
        raise TypeError("logits must be a CUDA float32 or bfloat16 tensor")
    B, L, V = logits.shape
    if logits.stride(2) != 1 or logits.stride(0) != L * logits.stride(1):
        raise ValueError("logits rows must be unit-stride with a uniform row stride")
    ids, logp, lse, ent = out
    _need(ids, torch.int32, (B, L, K), "ids")
    _need(logp, torch.float32, (B, L, K), "logp")
    _need(lse, torch.float32, (B, L), "lse")
    _need(ent, torch.float32, (B, L), "entropy")
    dtype = TAPS_F32 if logits.dtype == torch.float32 else TAPS_BF16
    st = lib.taps_topk_marginals_noalloc(_ptr(logits), dtype, logits.stride(1), B, L, V, K,
                                         _ptr(ids), _ptr(logp), _ptr(lse), _ptr(ent),
                                         _stream(stream, logits.device))
    _check("taps_topk_marginals_noalloc", st)
    return ids, logp, lse, ent


# ---------------------------------------------------------------------------
# KV cache layout conversion
# ---------------------------------------------------------------------------

lib.taps_pack_kv_pages.argtypes = [_P, _P, _I64, _I, _I, _P]
lib.taps_pack_kv_pages.restype = _I
lib.taps_unpack_kv_pages.argtypes = [_P, _P, _I64, _I, _I, _P]
lib.taps_unpack_kv_pages.restype = _I


def taps_pack_kv_pages(cache: torch.Tensor, out: torch.Tensor | None = None, stream=None):
    """Logical [num_pages, Hkv, 16, D] bf16 cache -> the TAPS page layout
    (same shape and size; element order inside each (page, head) block)."""
    _need(cache, torch.bfloat16, None, "cache")
    num_pages, Hkv, P, D = cache.shape
    if P != 16:
        raise ValueError("pages hold 16 tokens")
    out = torch.empty_like(cache) if out is None else out
    st = lib.taps_pack_kv_pages(_ptr(cache), _ptr(out), num_pages, Hkv, D,
                                _stream(stream, cache.device))
    _check("taps_pack_kv_pages", st)
    return out


def taps_unpack_kv_pages(cache: torch.Tensor, out: torch.Tensor | None = None, stream=None):
    """The TAPS page layout -> logical [num_pages, Hkv, 16, D]."""
    _need(cache, torch.bfloat16, None, "cache")
    num_pages, Hkv, P, D = cache.shape
    out = torch.empty_like(cache) if out is None else out
    st = lib.taps_unpack_kv_pages(_ptr(cache), _ptr(out), num_pages, Hkv, D,
                                  _stream(stream, cache.device))
    _check("taps_unpack_kv_pages", st)
    return out


# ---------------------------------------------------------------------------
# steps after verification: target greedy tokens + acceptance, K/V commit
# ---------------------------------------------------------------------------

lib.taps_target_greedy_accept_workspace_bytes.argtypes = [_I, _I]
lib.taps_target_greedy_accept_workspace_bytes.restype = _SZ
lib.taps_target_greedy_accept.argtypes = [_P, _I, _I64, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P,
                                          _P, _P, _SZ, _P]
lib.taps_target_greedy_accept.restype = _I
lib.taps_compact_accepted_kv.argtypes = [ctypes.POINTER(_P), ctypes.POINTER(_P), _I, _I64, _P,
                                         _I, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P]
lib.taps_compact_accepted_kv.restype = _I


def target_greedy_accept_workspace_bytes(B, n_max) -> int:
    return int(lib.taps_target_greedy_accept_workspace_bytes(B, n_max))


def taps_target_greedy_accept(verify_logits: torch.Tensor, parent, token, n_nodes, L,
                              out=None, ws=None, stream=None):
    """Target greedy token per tree node fused with acceptance: returns
    (target_tok [B, n_max], accept_len [B], accepted_nodes [B, L+1], bonus_tok [B])."""
    if verify_logits.dtype not in (torch.float32, torch.bfloat16) or not verify_logits.is_cuda:
        raise TypeError("verify_logits must be a CUDA float32 or bfloat16 tensor")
    B, n_max, V = verify_logits.shape
    if verify_logits.stride(2) != 1 or verify_logits.stride(0) != n_max * verify_logits.stride(1):
        raise ValueError("verify_logits rows must be unit-stride with a uniform row stride")
    _need(parent, torch.int32, (B, n_max), "parent")
    _need(token, torch.int32, (B, n_max), "token")
    _need(n_nodes, torch.int32, (B,), "n_nodes")
    dev = verify_logits.device
    if out is None:
        out = (torch.empty((B, n_max), dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev),
               torch.empty((B, L + 1), dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev))
    tt, alen, nodes, bonus = out
    _need(tt, torch.int32, (B, n_max), "target_tok")
    _need(alen, torch.int32, (B,), "accept_len")
    _need(nodes, torch.int32, (B, L + 1), "accepted_nodes")
    _need(bonus, torch.int32, (B,), "bonus_tok")
    nb = target_greedy_accept_workspace_bytes(B, n_max)
    if ws is None:
        ws = workspace(nb, dev, "target", stream)
    dtype = TAPS_F32 if verify_logits.dtype == torch.float32 else TAPS_BF16
    st = lib.taps_target_greedy_accept(_ptr(verify_logits), dtype, verify_logits.stride(1), B,
                                       n_max, V, _ptr(parent), _ptr(token), _ptr(n_nodes), L,
                                       _ptr(tt), _ptr(alen), _ptr(nodes), _ptr(bonus), _ptr(ws),
                                       nb, _stream(stream, dev))
    _check("taps_target_greedy_accept", st)
    return tt, alen, nodes, bonus


def taps_compact_accepted_kv(k_layers, v_layers, block_table, ctx_len, accepted_nodes,
                             accept_len, status=None, stream=None):
    """Move each layer's accepted-path K/V to consecutive positions after
    ctx_len (in place). k_layers / v_layers: lists of TAPS-layout caches."""
    if len(k_layers) != len(v_layers) or not k_layers:
        raise ValueError("need one K and one V cache per layer")
    num_pages, Hkv, P, D = k_layers[0].shape
    for t in list(k_layers) + list(v_layers):
        _need(t, torch.bfloat16, (num_pages, Hkv, P, D), "cache")
    B, max_pages = block_table.shape
    _need(block_table, torch.int32, (B, max_pages), "block_table")
    _need(ctx_len, torch.int32, (B,), "ctx_len")
    L = accepted_nodes.shape[1] - 1
    _need(accepted_nodes, torch.int32, (B, L + 1), "accepted_nodes")
    _need(accept_len, torch.int32, (B,), "accept_len")
    n = len(k_layers)
    kp = (_P * n)(*[t.data_ptr() for t in k_layers])
    vp = (_P * n)(*[t.data_ptr() for t in v_layers])
    dev = k_layers[0].device
    st = lib.taps_compact_accepted_kv(kp, vp, n, num_pages, _ptr(block_table), max_pages,
                                      _ptr(ctx_len), _ptr(accepted_nodes), _ptr(accept_len), B,
                                      L, Hkv, D, P, _ptr(status), _stream(stream, dev))
    _check("taps_compact_accepted_kv", st)
