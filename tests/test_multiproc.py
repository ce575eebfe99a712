"""Host logic of the multi-process bench path on CPU: two gloo ranks (world size 2).

The layer shards by token rows with no collective on the data path; the only cross-rank steps
are the barrier around the timed region and the max-over-ranks of the elapsed time, which sets
the whole-job throughput.  These run here on CPU exactly as bench.py calls them.
"""
from __future__ import annotations

import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank: int, world: int, port: int, q):
    try:
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                          WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
        sys.path.insert(0, ROOT)
        import bench
        r, w, local = bench.dist_env()
        dist = bench.init_dist(w, "gloo")
        bench.barrier(w)
        # each rank reports a different elapsed time; every rank must see the slowest
        elapsed = [3.5, 7.25][rank]
        slowest = bench.max_over_ranks(elapsed, w)
        value = bench.aggregate_value(flops_per_step=2.0e9, steps=10, world=w, total_ms=slowest)
        bench.barrier(w)
        dist.destroy_process_group()
        q.put((r, w, local, slowest, value))
    except Exception as e:  # surface the failure to the parent
        q.put(("error", repr(e)))


def test_two_gloo_ranks_max_and_aggregate():
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    q = mp.Queue()
    port = _free_port()
    procs = [mp.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert all(o[0] != "error" for o in out), out
    out.sort()
    assert [o[0] for o in out] == [0, 1]
    for r, w, local, slowest, value in out:
        assert w == 2 and local == r
        assert slowest == 7.25
        # whole-job value: both ranks' work over the slowest rank's time
        assert value == pytest.approx(2.0e9 * 10 * 2 / (7.25e-3) / 1e12)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(1.5, 1) == 1.5
    bench.barrier(1)
    assert bench.aggregate_value(2.0e12, 3, 1, 1000.0) == pytest.approx(6.0)
