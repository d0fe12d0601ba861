"""Replicas-only multi-GPU path of bench.py, on CPU with the gloo backend
(world size 2): the timed region is the max over ranks, the job time per
step counts the steps of every replica, and the reference arm runs on rank
0 only."""
import os
import socket

import pytest

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, local_ms, out_path):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        job_ms = bench.max_over_ranks(local_ms[rank], world)
        us = bench.job_us_per_step(job_ms, steps_per_rank=10, world=world)
        with open(f"{out_path}.{rank}", "w") as f:
            f.write(f"{job_ms!r} {us!r}\n")
    finally:
        dist.destroy_process_group()


def test_max_over_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp
    local = [12.5, 20.0]          # ms of the timed region on each rank
    out = str(tmp_path / "res")
    mp.spawn(_worker, args=(2, _free_port(), local, out), nprocs=2, join=True)
    for rank in range(2):
        job_ms, us = map(float, open(f"{out}.{rank}").read().split())
        assert job_ms == 20.0                      # every rank sees the slowest
        assert us == pytest.approx(20.0 * 1000 / (10 * 2))


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(7.25, 1) == 7.25
    assert bench.job_us_per_step(7.25, 5, 1) == pytest.approx(1450.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class Args:
        workload, seed, steps, warmup, gamma, tau = "tiny_f32", 0, 1, 0, 0.1, 1.0
    assert bench.run_reference(Args()) is None
    assert capsys.readouterr().out == ""
