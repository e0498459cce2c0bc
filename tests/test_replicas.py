"""The N > 1 bookkeeping of bench.py (replicas only: no data-path
collective) on two gloo CPU processes: rendezvous, barrier, the slowest
rank's time and the whole-job rate."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    import torch.distributed as dist
    w, r, _ = bench.dist_setup(None, backend="gloo")
    assert (w, r) == (world, rank)
    bench.barrier(w)
    slowest = bench.max_over_ranks(10.0 + rank, w)  # rank r took 10 + r ms
    out[rank] = (slowest, bench.job_throughput(100.0, w, 4, slowest))
    dist.destroy_process_group()


def test_two_replicas_gloo():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for r in range(world):
        slowest, rate = out[r]
        assert slowest == 11.0                                   # every rank sees the slowest time
        assert rate == pytest.approx(100.0 * 2 * 4 / 11e-3)      # all ranks' units over that time
