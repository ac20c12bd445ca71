"""The N > 1 path of bench.py on CPU: two gloo ranks (world size 2) run the
host logic the GPU replicas use -- max-over-ranks timing, the whole-job
value, the barrier -- and the reference arm runs on rank 0 only."""
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    try:
        w, r, _ = bench.dist_env()
        dist = bench.init_dist(w, r, backend="gloo")
        t = bench.max_over_ranks(dist, 1.0 + 0.5 * rank)     # rank 1 is the slower
        bench.barrier(dist)
        value = bench.replica_value(w, 64, t)
        # the reference arm: rank 0 alone runs the oracle; the others return at once
        out = io.StringIO()
        rc = None
        if rank != 0:
            class A:
                config, layers, warmup, steps, ref_seconds = "stack", 96, 0, 1, 1.0
            with redirect_stdout(out):
                rc = bench.run_reference(A)
        dist.destroy_process_group()
        q.put((rank, t, value, rc, out.getvalue()))
    except Exception as e:  # reported to the parent
        q.put((rank, "error", repr(e), None, ""))


def test_two_gloo_ranks_share_the_slowest_time_and_the_job_value():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, t, value, rc, out in res:
        assert t != "error", value
        assert t == pytest.approx(1.5)                 # max over ranks, on every rank
        assert value == pytest.approx(2 * 64 / 1.5)    # units of both replicas / slowest time
        if rank == 1:
            assert rc == 0 and out == ""               # only rank 0 prints a line


def test_replica_value_is_weak_scaling():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.replica_value(1, 64, 16.0) == pytest.approx(4.0)
    assert bench.replica_value(8, 64, 16.0) == pytest.approx(32.0)
