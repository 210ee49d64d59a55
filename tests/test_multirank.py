"""Multi-rank host logic of bench.py on CPU (gloo, world size 2).

The path shards by request with no data-path collective: every rank runs its
own requests and only the timing is reduced (max over ranks) and the
throughput aggregated over ranks.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ws, r, local = bench.dist_env()
    assert (ws, r, local) == (world, rank, rank)
    bench.barrier(ws)
    t = bench.max_over_ranks(1.0 + rank, ws)            # rank 1 is the slow one
    v = bench.aggregate_value(2880, 10, ws, t)
    out[rank] = (t, v)
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_rank_max_time_and_weak_scaling_aggregate():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(90)
        assert p.exitcode == 0
    assert out[0] == out[1]
    t, v = out[0]
    assert t == 2.0                                      # max over ranks
    assert v == pytest.approx(2880 * 10 * 2 / 2.0)       # both ranks' tokens over the slowest time


def test_single_rank_helpers_are_identity():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.aggregate_value(100, 2, 1, 4.0) == 50.0
