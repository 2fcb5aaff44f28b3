"""The benchmark's multi-rank path on CPU (gloo, world size 2): each rank gets its own instance pool
and window, the step time is the maximum over ranks, and the job rate counts every rank's work.
The data path has no collective; only the timing is reduced."""
import os
import socket

import numpy as np
import pytest

import bench
import workload as W


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        seed = bench.rank_seed(0, rank)
        wl = W.generate(0, seed=seed)
        ms = 10.0 + 5.0 * rank  # this rank's step time
        got = bench.max_over_ranks(ms, "cpu")
        q.put((rank, seed, got, int(wl.window.chain_hash[:8].sum() % (1 << 62)), wl.window.R))
    finally:
        dist.destroy_process_group()


def test_two_ranks_independent_pools_and_max_time():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=240)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(2))
    (r0, s0, t0, h0, R0), (r1, s1, t1, h1, R1) = res
    assert (r0, r1) == (0, 1)
    assert s1 == s0 + 1                 # distinct seeds: independent problems
    assert h0 != h1                     # and different windows
    assert t0 == t1 == 15.0             # both ranks report the slowest rank's step time
    assert bench.job_rate(2, R0 * 8, 15.0) == pytest.approx(2 * R0 * 8 / 0.015)


def test_single_process_max_is_identity():
    assert bench.max_over_ranks(3.5, "cpu") == 3.5
    assert bench.job_rate(1, 100, 10.0) == pytest.approx(10000.0)
