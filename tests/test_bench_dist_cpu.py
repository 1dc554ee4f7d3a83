"""Host logic of bench.py's multi-rank mode on CPU (gloo, world size 2): ranks are
independent replicas; the reported time is the max over ranks and the value counts the
tokens of every rank."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update({"RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    r, w = bench.init_dist("gloo")
    t = 0.010 * (r + 1)                     # rank 1 is the slow one
    bench.barrier(w)
    tmax = bench.max_over_ranks(t, w)
    q.put((r, w, tmax, bench.aggregate_value(32, w, tmax)))
    dist.destroy_process_group()


def test_two_rank_aggregation():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for r, w, tmax, val in res:
        assert w == 2
        assert tmax == pytest.approx(0.020)
        assert val == pytest.approx(64 / 0.020)


def test_single_rank_helpers_are_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(1.5, 1) == 1.5
    assert bench.aggregate_value(8, 1, 0.5) == 16.0
