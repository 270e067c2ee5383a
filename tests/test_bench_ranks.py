"""The multi-process side of bench.py on CPU: two gloo ranks aggregate their
figures as the benchmark does (max of times, sum of tokens), and the
reference arm does no work on ranks other than 0."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r: timed region 10 + r ms, 100 * (r + 1) tokens, e2e 0.5 + r s for 50 + r tokens
        res = bench.aggregate_ranks(10.0 + rank, 100.0 * (rank + 1), 0.5 + rank, 50.0 + rank, "cpu")
        out.put((rank, res, bench.dist_env()))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_max_time_and_total_tokens():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, res, env in sorted(got):
        assert res == (11.0, 300.0, 1.5, 101.0)  # slowest rank's times, all ranks' tokens
        assert env == (rank, 2, rank)


def test_single_process_keeps_its_own_figures():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_ranks(3.0, 7.0, 1.0, 2.0, "cpu") == (3.0, 7.0, 1.0, 2.0)


def test_reference_arm_idles_on_other_ranks(monkeypatch):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    ns = type("A", (), dict(workload="4b-b1", tau=None, steps=1, warmup=1, cpu_seconds=1.0, force=0))()
    assert bench.run_reference(ns) is None  # returns before loading weights or the oracle
