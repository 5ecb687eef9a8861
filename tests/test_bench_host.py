"""Host-side pieces of bench.py that need no GPU: the workload description,
the rotary option and the inputs the end-to-end leg uploads every step."""

import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_e2e_uploads_step_inputs_but_not_the_weight():
    w = {"cfg": 4, "W": torch.zeros(4, 2), "Q": torch.zeros(3, 1, 2), "rows": torch.zeros(2, dtype=torch.int32),
         "heads": (1, 1, 2), "record": object()}
    device_keys = {"W", "Q", "rows", "noise"}
    up = bench.e2e_inputs(w, device_keys)
    assert set(up) == {"Q", "rows"}
    assert "W" in bench.RESIDENT


def test_rotary_option_is_recorded_in_the_workload():
    w = bench.make_workload(2, pin=False, rope=1e6, n_traj=1)
    assert w["rope"] == 1e6
    d = bench.describe(w)
    assert d["rope_theta"] == 1e6 and d["trajectories"] == 1
    # the LM-head-only workload has no attention, so no rotary setting
    assert "rope" not in bench.make_workload(3, pin=False, rope=1e6)


def test_clip_range_is_the_papers_asymmetric_one():
    assert (bench.EPS_LO, bench.EPS_HI) == (0.2, 0.28)


def test_events_option_builds_an_offload_retrieve_workload():
    """--events P turns the record into offload / retrieve events whose
    views the oracle validates; the description says so."""
    from oracle import nonmonotone as N
    w = bench.make_workload(2, pin=False, events=0.5, n_traj=2)
    assert w["events_p"] == 0.5 and len(w["events"]) == 2
    for T, e in zip(w["record"].seqlens, w["events"]):
        N.validate_events(T, e)
    d = bench.describe(w)
    assert "offload / retrieve" in d["views"] and d["retrieved_spans"] > 0


def test_bench_rejects_option_combinations_before_any_gpu_work():
    import subprocess
    for args, word in ((["--config", "3", "--events", "0.3"], "--events"),
                       (["--config", "4", "--packed"], "--packed"),
                       (["--config", "2", "--events", "1.5"], "--events"),
                       (["--sdcc", "--config", "2"], "--sdcc")):
        r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], capture_output=True, text=True,
                           timeout=120)
        assert r.returncode == 2 and word in r.stderr, (args, r.stderr[-500:])
