"""The N > 1 path of bench.py on the CPU: one replica per rank (no data-path
collective), timed by the slowest rank, value = the tokens of all ranks over
that time; rank 0 alone runs the reference arm.  Two gloo ranks stand in for
two GPUs."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        # rank r took 100 + 50 r ms for 10 steps of 2048 tokens
        ms, value = bench.job_throughput(100.0 + 50.0 * rank, 10, 2048, dist, "cpu")
        q.put((r, w, local, ms, value))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_replicas_are_timed_by_the_slowest_rank():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        got = sorted(q.get(timeout=120) for _ in range(2))
    finally:
        for p in procs:
            p.join(timeout=60)
    assert [p.exitcode for p in procs] == [0, 0]
    for rank, (r, w, local, ms, value) in enumerate(got):
        assert (r, w, local) == (rank, 2, rank)
        assert ms == pytest.approx(15.0)                       # max(100, 150) ms / 10 steps
        assert value == pytest.approx(2 * 2048 / 15.0e-3)      # both ranks' tokens over the slowest time


def test_single_process_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    ms, value = bench.job_throughput(30.0, 3, 512)
    assert ms == pytest.approx(10.0) and value == pytest.approx(512 / 10.0e-3)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    assert bench.run_reference(None) is None   # returns before parsing its arguments or doing work
    assert capsys.readouterr().out == ""
