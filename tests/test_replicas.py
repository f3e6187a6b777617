"""The N > 1 path of bench.py on CPU: world size 2 over gloo (127.0.0.1).

Each rank runs an independent replica of the step (no data-path exchange);
the only collective is the max-over-ranks reduction of the step time, and the
whole-job figure is world x the per-rank ops over that slowest time."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(WORLD_SIZE=str(world), RANK=str(rank), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        assert bench.dist_env() == (world, rank, rank)
        ms_local = 2.0 + 3.0 * rank  # rank 1 is the slow one
        ms = bench.max_over_ranks(torch, dist, ms_local, "cpu")
        out.put((rank, ms, bench.job_tops(1e12, world, ms)))
    finally:
        dist.destroy_process_group()


def test_two_rank_replicas_take_the_slowest_rank():
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, ms, tops in got:
        assert ms == 5.0                               # max over ranks, on every rank
        assert tops == pytest.approx(2 * 1e12 / 5e-3 / 1e12)  # 2 replicas x ops / slowest time


def test_single_process_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(None, None, 3.5, "cpu") == 3.5
    assert bench.job_tops(4.31e12, 1, 5.52) == pytest.approx(4.31e12 / 5.52e-3 / 1e12)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    # a non-zero rank returns at once (exit 0), before touching the oracle
    assert bench.run_reference(None) == 0
