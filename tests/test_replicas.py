"""The multi-GPU path of bench.py is independent replicas (every layer,
sequence and KV head is independent; there is no exchange step): each rank
runs the whole workload, the job's time is the slowest rank's, and the value
is all ranks' tokens over that time. Checked here with two gloo ranks on the
CPU; no GPU is involved."""
import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        mine = [10.0 + rank, 5.0 - rank, 7.0 * (rank + 1)]
        got = bench.max_over_ranks(dist, mine, "cpu")
        rate = bench.job_rate(world, 3, 1000, got[0])
        q.put((rank, got, rate))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_rate_with_two_gloo_ranks():
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
    for rank, got, rate in res:
        assert got == [11.0, 5.0, 14.0]          # element-wise maximum over both ranks
        assert rate == pytest.approx(2 * 3 * 1000 / 0.011)  # both ranks' tokens over the slowest time


def test_single_process_needs_no_process_group():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(None, [1.5, 2.5], "cpu") == [1.5, 2.5]
    assert bench.job_rate(1, 2, 500, 1000.0) == pytest.approx(1000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    # rank 1 returns before building or timing anything
    assert bench.main() == 0
