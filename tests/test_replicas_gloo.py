"""The N > 1 path of the benchmark on CPU: two gloo ranks, no GPU.

bench.py runs one independent replica of the optimizer step per GPU ("replicas
only": one AGS step has no exchange once the K replica gradients sit in one
GPU's memory), so its only cross-rank logic is the timing: every rank reports
its elapsed time, the job takes the slowest rank's, and the throughput counts
the parameters of every rank.  These tests drive that logic with gloo ranks of
different speeds, and check that the reference arm does its work on rank 0
only.
"""
import json
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, times, out_path):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        t_max = bench.max_over_ranks(times[rank], device="cpu")
        value = bench.job_throughput(1000, 10, world, t_max)
        with open(f"{out_path}.{rank}", "w") as f:
            json.dump({"t_max": t_max, "value": value}, f)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("times", [(5.0, 8.0), (9.5, 2.0)])
def test_job_time_is_the_slowest_rank(tmp_path, times):
    out = str(tmp_path / "r")
    mp.start_processes(_rank_main, args=(2, _free_port(), times, out), nprocs=2,
                       start_method="spawn", join=True)
    res = [json.load(open(f"{out}.{r}")) for r in range(2)]
    slowest = max(times)
    for r in res:
        assert r["t_max"] == slowest
        # 2 ranks x 1000 params x 10 steps in the slowest rank's time
        assert r["value"] == pytest.approx(2 * 1000 * 10 / (slowest / 1e3))


def test_single_process_keeps_its_own_time():
    assert not dist.is_initialized()
    assert bench.max_over_ranks(3.25, device="cpu") == 3.25
    assert bench.job_throughput(500, 4, 1, 2.0) == pytest.approx(500 * 4 / 2e-3)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")
    from paper_2603_18112_gb300 import workloads as W
    wl = W.workload("resnet20")

    class Args:
        steps, warmup = 3, 3

    bench.run_reference(Args, wl)  # rank 1: no work, no output
    assert capsys.readouterr().out == ""
