"""Replica timing of bench.py across ranks (world size 2, gloo, CPU).

The path does not shard: with N GPUs the benchmark runs N independent
replicas of the store, and the job's time is the slowest rank's.  This
checks that reduction and the whole-job throughput on two CPU ranks."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, e2e = bench.max_over_ranks([10.0 + rank, 20.0 - rank])
    out[rank] = (ms, e2e, bench.job_throughput(256 * 20, world, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_throughput():
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(2):
        ms, e2e, thr = out[r]
        assert ms == 11.0 and e2e == 20.0
        assert thr == pytest.approx(256 * 20 * 2 / 0.011)


def test_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([3.0, 4.0]) == [3.0, 4.0]
    assert bench.job_throughput(100, 1, 1000.0) == pytest.approx(100.0)
