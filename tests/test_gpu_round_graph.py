"""The whole round with its host uploads and the read of its results captured
as one CUDA graph by TapsRound.capture_round_graph (the form bench.py's
end-to-end figure replays: the head on the compute stream, the queries in
groups of layers on a copy stream, each group of verification layers waiting
only for its own), against the same round run stage by stage from inputs
already on the device. The device copy of the inputs is cleared first, so the
graph's own uploads must supply them; the results must match bit for bit."""
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import workloads as W  # noqa: E402


@pytest.fixture(scope="module")
def taps():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00487_gb300 as t
    return t


@pytest.mark.parametrize("name,layers,groups", [("tiny", None, 1), ("qwen3_8b", 6, 4),
                                                ("batched", 3, 2)])
def test_round_graph_with_uploads_matches_stagewise(taps, name, layers, groups):
    import bench
    cfg = bench.workload_config(name, layers=layers)
    dev = torch.device("cuda:0")
    rs = bench.RoundSetup(taps, W, cfg, "taps", dev)
    r, inp = rs.r, rs.inp
    torch.cuda.synchronize()
    inp.host_buf.copy_(inp.device_buf)
    # stage by stage, from the inputs already on the device
    expected = torch.empty(r.results.shape, dtype=r.results.dtype, pin_memory=True)
    rs.step()
    r.download(expected, rs.stream)
    rs.stream.synchronize()
    # one graph: uploads, the round, the read of its results
    got = torch.full(r.results.shape, -7, dtype=r.results.dtype, pin_memory=True)
    g = rs.capture_e2e(got, groups)
    inp.device_buf.zero_()
    r.results.zero_()
    torch.cuda.synchronize()
    g.replay()
    rs.stream.synchronize()
    assert torch.equal(got, expected)
    # and again, from the state the first replay left
    got.fill_(-7)
    g.replay()
    rs.stream.synchronize()
    assert torch.equal(got, expected)


def test_round_graph_rejects_unfed_queries(taps):
    """capture_round_graph refuses a layer whose q is not the upload buffer's
    view of that layer (the graph's uploads would never reach it) and a result
    buffer that is not pinned or has the wrong size."""
    import bench
    cfg = bench.workload_config("tiny")
    dev = torch.device("cuda:0")
    rs = bench.RoundSetup(taps, W, cfg, "taps", dev)
    r = rs.r
    res = torch.empty(r.results.shape, dtype=r.results.dtype, pin_memory=True)
    layers = list(rs.layers)
    q, kc, vc, bt = layers[0]
    layers[0] = (q.clone(), kc, vc, bt)
    with pytest.raises(ValueError):
        r.capture_round_graph(rs.inp, rs.ctx, layers, rs.outs, res)
    with pytest.raises(ValueError):
        r.capture_round_graph(rs.inp, rs.ctx, rs.layers, rs.outs,
                              torch.empty(r.results.shape, dtype=r.results.dtype))
    with pytest.raises(ValueError):
        r.capture_round_graph(rs.inp, rs.ctx, rs.layers[:-1], rs.outs[:-1], res)
