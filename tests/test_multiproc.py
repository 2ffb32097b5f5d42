"""The N > 1 path of bench.py on CPU: two gloo ranks (no GPU).

bench.py runs one replica per rank (rounds are independent: no data-path
collective), takes the slowest rank's timed region as the job's time, and
reports value = N x steps / that time. These tests check the rank-side
helpers that implement it (barrier, max over ranks) and the aggregation."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        # each rank's "elapsed" time differs; the job's is the slowest
        elapsed = 10.0 + 5.0 * rank
        worst = bench.max_over_ranks(elapsed, world)
        steps = 20
        value = world * steps / (worst / 1e3)
        out[rank] = (worst, value)
        bench.barrier(world)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_replicas_max_over_ranks_gloo(world):
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    worst = 10.0 + 5.0 * (world - 1)
    for r in range(world):
        assert out[r][0] == pytest.approx(worst)
        # whole-job throughput: all ranks' rounds over the slowest rank's time
        assert out[r][1] == pytest.approx(world * 20 / (worst / 1e3))


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(3.25, 1) == 3.25
    bench.barrier(1)
