"""Host logic of bench.py's multi-GPU path, run as two gloo ranks on CPU.

Under torchrun every rank scores its own replica (independent trajectories,
no collective on the data path); the job's time is the max over ranks, and
rank 0 alone reports the whole-job throughput."""

import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    import bench as b
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # per-rank step times: the job time is the slowest rank's
        ms = b.reduce_max(10.0 + 2.5 * rank, world)
        e2e = b.reduce_max(20.0 - rank, world)
        dist.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{ms} {e2e}\n")
    finally:
        dist.destroy_process_group()


def test_reduce_max_over_two_gloo_ranks(tmp_path):
    port = _free_port()
    mp.start_processes(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn", join=True)
    for r in range(2):
        ms, e2e = map(float, (tmp_path / f"rank{r}.txt").read_text().split())
        assert ms == 12.5          # max(10.0, 12.5)
        assert e2e == 20.0         # max(20.0, 19.0)


def test_reduce_max_world_one_is_identity():
    assert bench.reduce_max(3.25, 1) == 3.25


def test_job_value_counts_every_rank():
    # 1000 scored tokens per rank, 2 ranks, 4 ms for the job -> 500k tokens/s
    assert bench.job_value(1000, 2, 4.0) == pytest.approx(500000.0)
    assert bench.job_value(1000, 1, 4.0) == pytest.approx(250000.0)


def test_replicas_are_distinct_per_rank():
    seeds = {bench.replica_seed(cfg, r) for cfg in (2, 3, 4, 5) for r in range(8)}
    assert len(seeds) == 4 * 8


def test_reference_arm_rank1_does_no_work(monkeypatch, capsys):
    def boom(*a, **k):
        raise AssertionError("rank 1 must not build a workload")
    monkeypatch.setattr(bench, "make_workload", boom)

    class A:
        config, K, f, n_traj, warmup, steps, cpu_seconds = 2, 8, 0.6, None, 1, 1, 1.0
    bench.run_reference(A(), rank=1, world=2)
    assert capsys.readouterr().out == ""


def test_reference_arm_reports_whole_job_throughput(monkeypatch, capsys):
    """The reference line's value is all timed steps' sampled tokens over
    their total time (warm-up steps excluded), like the bench's own CPU
    baseline, not a median of per-step rates."""
    import json
    samples = iter([(8, 99.0), (8, 1.0), (8, 3.0), (16, 4.0)])   # (tokens, seconds); the first is warm-up

    def fake_sample(w, budget_s, seed, detail=False):
        assert detail
        done, dt = next(samples)
        return done, dt, 16, ["oracle"]
    monkeypatch.setattr(bench, "cpu_sample", fake_sample)
    monkeypatch.setattr(bench, "make_workload", lambda *a, **k: {"rows": bench_rows(10)})
    monkeypatch.setattr(bench, "describe", lambda w: {"workload": "test"})

    class A:
        config, K, f, n_traj, warmup, steps, cpu_seconds, rope, events = 4, 8, 0.6, None, 1, 3, 3.0, None, None
    bench.run_reference(A(), rank=0, world=1)
    line = json.loads(capsys.readouterr().out)
    assert line["impl"] == "reference"
    assert line["value"] == pytest.approx(32 / 8.0)
    assert line["cpu_baseline"]["value"] == line["value"] == line["e2e"]["value"]
    assert "32 sampled scored tokens over 3 steps" in line["cpu_baseline"]["sample"]


def bench_rows(n):
    import torch
    return torch.arange(n, dtype=torch.int32)
