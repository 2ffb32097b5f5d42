"""The allocation-free top-K entry point against the regular one.

taps_topk_marginals_noalloc serves callers that cannot call cudaMalloc (a
serving engine that reserved all device memory up front, a plugin inside a
framework that owns every allocation, a decode loop that cannot afford an
allocation's device-wide synchronisation). It keeps its partial records in a
fixed device array inside the library. This file is collected last so that a
run stopping at the first failure has already run every other test; it also
passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import workloads as W  # noqa: E402


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00487_gb300 as taps
    return taps


def _call_noalloc(lib, x, K):
    """Straight through the C ABI with caller-owned outputs."""
    B, L, V = x.shape
    dev = x.device
    ids = torch.full((B, L, K), -7, dtype=torch.int32, device=dev)
    logp = torch.full((B, L, K), float("nan"), dtype=torch.float32, device=dev)
    lse = torch.full((B, L), float("nan"), dtype=torch.float32, device=dev)
    ent = torch.full((B, L), float("nan"), dtype=torch.float32, device=dev)
    dtype = 0 if x.dtype == torch.float32 else 1
    st = lib.lib.taps_topk_marginals_noalloc(
        ctypes.c_void_p(x.data_ptr()), dtype, x.stride(1), B, L, V, K,
        ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(logp.data_ptr()),
        ctypes.c_void_p(lse.data_ptr()), ctypes.c_void_p(ent.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, lib.lib.taps_status_string(st)
    return ids, logp, lse, ent


def _compare(a, b):
    np.testing.assert_array_equal(a[0].cpu().numpy(), b[0].cpu().numpy())
    for x, y in zip(a[1:], b[1:]):
        np.testing.assert_allclose(x.cpu().numpy(), y.cpu().numpy(), rtol=1e-5, atol=1e-6)


def test_noalloc_matches_regular_entry_point_twice(lib):
    dev = torch.device("cuda:0")
    cfg = W.CONFIGS["qwen3_8b"]
    x1 = torch.from_numpy(W.make_logits(cfg)).to(dev).to(torch.bfloat16)
    cfg_t = W.CONFIGS["tiny"]
    x2 = torch.from_numpy(W.make_logits(cfg_t)).to(dev)
    for x, K in ((x1, cfg.K), (x2, cfg_t.K)):          # two calls in a row, different shapes
        got = _call_noalloc(lib, x, K)
        torch.cuda.synchronize()
        ref = lib.taps_topk_marginals(x, K)
        torch.cuda.synchronize()
        _compare(got, ref)
    # and the same call again: the shared array keeps the last call's contents
    got = _call_noalloc(lib, x1, cfg.K)
    torch.cuda.synchronize()
    _compare(got, lib.taps_topk_marginals(x1, cfg.K))


def test_noalloc_rejects_sizes_beyond_its_array(lib):
    x = torch.zeros((1, 4097, 8), dtype=torch.float32, device="cuda:0")
    outs = (torch.empty((1, 4097, 4), dtype=torch.int32, device="cuda:0"),
            torch.empty((1, 4097, 4), dtype=torch.float32, device="cuda:0"),
            torch.empty((1, 4097), dtype=torch.float32, device="cuda:0"),
            torch.empty((1, 4097), dtype=torch.float32, device="cuda:0"))
    with pytest.raises(lib.TapsError) as e:
        lib._binding.taps_topk_marginals_noalloc(x, 4, outs)
    assert e.value.status == 2
