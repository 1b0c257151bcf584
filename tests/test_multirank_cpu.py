"""The N > 1 path of bench.py on CPU: world-size-2 gloo ranks (no GPU).

Each GPU runs its own replica of the step (no data-path collective), so the
host logic to check is the job's clock (the slowest rank's time, by an
all-reduce MAX), the whole-job rate (units of every rank over that time) and
the reference arm, which only rank 0 runs and prints.
"""
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


def _rank_main(rank, world, port, results):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        local_ms = [30.0, 45.0][rank]            # the second rank is slower
        total = bench.max_over_ranks(local_ms, world, "cpu")
        rate = bench.job_rate(128, 5, world, total)
        alone = bench.max_over_ranks(local_ms, 1, "cpu")
        results[rank] = (total, rate, alone)
    finally:
        dist.destroy_process_group()


def test_job_clock_is_the_slowest_rank_and_rate_counts_every_rank():
    world = 2
    results = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, _free_port(), results), nprocs=world, join=True)
    for rank in range(world):
        total, rate, alone = results[rank]
        assert total == 45.0                       # MAX over ranks, the same on every rank
        assert rate == pytest.approx(128 * 5 * 2 / 0.045)
        assert alone == [30.0, 45.0][rank]         # world 1: no collective


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    called = []
    monkeypatch.setattr(bench, "main_reference", lambda args: called.append(args) or {})
    assert bench.main(["--impl", "reference", "--gpus", "2"]) == 0
    assert called == [] and capsys.readouterr().out == ""
    monkeypatch.setenv("RANK", "0")
    assert bench.main(["--impl", "reference", "--gpus", "2"]) == 0
    assert len(called) == 1 and capsys.readouterr().out.strip() == "{}"
