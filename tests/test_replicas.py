"""The multi-GPU mode of the benchmark is independent replicas (the path has no
exchange step): one process per GPU, a barrier around the timed region, the
slowest rank's time, and the whole-job rate summed over ranks.  These tests run
that host logic as two gloo ranks on the CPU."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist

    r, w, _ = bench.dist_init()
    assert dist.get_backend() == "gloo"
    # Each rank times a different step; every rank must end with the slowest.
    slowest = bench.dist_max(1.0 + 0.5 * r)
    bench.dist_barrier()
    q.put((r, w, slowest, bench.replica_value(w, 4, slowest)))
    dist.destroy_process_group()


def test_two_replicas_share_the_slowest_time():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    assert [g[0] for g in got] == [0, 1]
    for r, w, slowest, value in got:
        assert w == 2 and slowest == 1.5
        # Whole-job tokens/s: 2 replicas x batch 4 per slowest step of 1.5 ms.
        assert value == pytest.approx(2 * 4 / 1.5e-3)


def test_single_process_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.dist_max(2.5) == 2.5
    bench.dist_barrier()
    assert bench.replica_value(1, 1, 0.25) == pytest.approx(4000.0)
