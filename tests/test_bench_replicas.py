"""The bench's multi-GPU path is replicas only: every rank runs the whole path
on its own copy of the trace, with no collective on the data path.  What is
shared is the host logic around it, tested here on the CPU with two gloo
ranks: the slowest rank's time (an all-reduce MAX), the whole-job rate over
all replicas, and the reference arm running on rank 0 alone."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # rank r took (r + 1) * 10 ms: the job lasts as long as the slowest replica
        total_ms = bench.max_over_ranks(10.0 * (rank + 1), world, "cpu")
        out.put((rank, total_ms, bench.whole_job_rate(1000, 5, world, total_ms)))
    finally:
        dist.destroy_process_group()


def test_slowest_rank_and_whole_job_rate_two_gloo_ranks():
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    world, port = 2, _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, total_ms, rate in got:
        assert total_ms == 20.0  # the max over both ranks, seen by each
        # 2 replicas x 1000 units x 5 steps in 20 ms
        assert rate == pytest.approx(2 * 1000 * 5 / 0.020)


def test_one_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.whole_job_rate(100, 4, 1, 2.0) == pytest.approx(100 * 4 / 0.002)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0"])
    args = bench.parse_args()
    bench.run_reference(args, 2, 1)  # rank 1 of 2: no work, no output
    assert capsys.readouterr().out == ""


def test_dist_env_reads_torchrun_variables(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "4")
    monkeypatch.setenv("RANK", "3")
    monkeypatch.setenv("LOCAL_RANK", "1")
    assert bench.dist_env() == (4, 3, 1)
