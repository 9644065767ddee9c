"""The multi-rank host logic of the bench on CPU: two gloo ranks, each a weak-
scaling replica with its own batch seed; they meet only for a barrier and the
max-over-ranks timing reduction."""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2608_29291_gb300 import runtime


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    info = runtime.rank_info()
    dist = runtime.init_group(info, "gloo")
    try:
        runtime.barrier(dist)
        slow = runtime.max_over_ranks(dist, 1.0 + rank)          # rank r "took" 1 + r ms
        total = runtime.sum_over_ranks(dist, 10.0 * (rank + 1))
        out.put((rank, info.world, info.is_root, runtime.replica_seed(0, rank), slow, total))
    finally:
        dist.destroy_process_group()


def test_two_rank_gloo_timing_reduction():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[0] for r in res] == [0, 1]
    assert all(r[1] == 2 for r in res)
    assert [r[2] for r in res] == [True, False]
    assert res[0][3] != res[1][3]                  # each replica draws its own batch
    assert all(r[4] == 2.0 for r in res)           # the slowest rank's time, on every rank
    assert all(r[5] == 30.0 for r in res)


def test_single_rank_needs_no_group(monkeypatch):
    for v in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(v, raising=False)
    info = runtime.rank_info()
    assert (info.rank, info.world, info.is_root) == (0, 1, True)
    dist = runtime.init_group(info, "gloo")
    assert dist is None
    assert runtime.max_over_ranks(dist, 3.5) == 3.5
