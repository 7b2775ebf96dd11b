"""The multi-GPU path of bench.py is replicas with no data-path collective:
check its rank plumbing (barrier, max and sum over ranks, per-rank seeds)
with two gloo processes on the CPU."""

import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update({"RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    import bench
    r = bench.Ranks("gloo")
    r.barrier()
    mx = r.max(10.0 + rank)
    sm = r.sum(1.5 * (rank + 1))
    seed = bench.replica_seed(7001, rank)
    r.barrier()
    q.put((rank, mx, sm, seed))
    r.dist.destroy_process_group()


def test_two_rank_gloo_reductions():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(rk, world, port, q)) for rk in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [x[1] for x in res] == [11.0, 11.0]      # max over ranks
    assert [x[2] for x in res] == [4.5, 4.5]        # sum over ranks
    assert res[0][3] != res[1][3]                   # replicas draw different inputs


def test_single_rank_needs_no_process_group(monkeypatch):
    import sys
    sys.path.insert(0, ROOT)
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    import bench
    r = bench.Ranks("gloo")
    assert r.world == 1 and r.max(3.0) == 3.0 and r.sum(2.0) == 2.0
