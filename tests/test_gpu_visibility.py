"""GPU visibility builder vs the oracle, bit for bit (every array)."""

import json
import os

import numpy as np
import pytest

import synth
from oracle import visibility as OV

pytestmark = pytest.mark.gpu


def _gpu(seqlens, edits):
    import torch
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    torch.cuda.synchronize()
    vis.check_status()
    return vis.arrays()


def _compare(seqlens, edits):
    return _check_arrays(_gpu(seqlens, edits), seqlens, edits)


def _check_arrays(got, seqlens, edits):
    want = OV.build(seqlens, edits)
    for key in ("omega", "seg", "qtile_traj", "fwd_ptr", "fwd_idx", "bwd_ptr", "bwd_idx", "pairs", "keymask",
                "seg_len", "cpos"):
        np.testing.assert_array_equal(got[key], want[key], err_msg=key)
    defined = want["csrc"] != -2          # the compact maps past a segment's last tile are unspecified
    np.testing.assert_array_equal(got["csrc"][defined], want["csrc"][defined], err_msg="csrc")
    assert got["pairs_total"] == want["pairs_total"]
    assert len(got["cls"]) == len(want["cls"])
    for a, b in zip(got["cls"], want["cls"]):
        np.testing.assert_array_equal(np.tril(a), np.tril(b), err_msg="cls")
    return got


def test_running_example():
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "running_example.json")))
    edits = [(J, [tuple(s) for s in sp]) for J, sp in g["edits"]]
    got = _compare([14], [edits])
    assert list(got["omega"][[5, 8, 11]]) == [7, 10, 12]


def _rand_record(rng, n_traj):
    seqlens, edits = [], []
    for _ in range(n_traj):
        T = int(rng.choice([1, 2, 127, 128, 129, 300, 777, 1024, 1500]))
        K = int(rng.integers(0, min(6, T - 1) + 1)) if T > 1 else 0
        Js = sorted(rng.choice(np.arange(1, T), size=K, replace=False).tolist()) if K else []
        e = []
        for J in Js:
            sp = []
            for _ in range(int(rng.integers(0, 5))):
                a = int(rng.integers(0, J))
                sp.append((a, int(rng.integers(a + 1, J + 1))))
            e.append((J, sp))
        seqlens.append(T)
        edits.append(e)
    return seqlens, edits


@pytest.mark.parametrize("seed", range(10))
def test_random_records(seed):
    rng = np.random.default_rng(seed)
    _compare(*_rand_record(rng, int(rng.integers(1, 6))))


def test_empty_trajectory_inside_record():
    _compare([300, 0, 129], [[(100, [(0, 50)])], [], [(5, [(1, 3)])]])


def test_empty_record():
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility([], [])
    assert vis.layout.n_tiles == 0 and vis.pairs_total == 0


@pytest.mark.parametrize("cfg", [1, 2, 4])
def test_config_records(cfg):
    r = synth.config_record(cfg)
    _compare(r.seqlens, r.edits)


@pytest.mark.parametrize("K", synth.CONFIGS[5]["sweep_K"])
@pytest.mark.parametrize("f", synth.CONFIGS[5]["sweep_f"])
def test_sweep_records(K, f):
    r = synth.config_record(5, K=K, f=f)
    _compare(r.seqlens, r.edits)


def test_bad_record_raises():
    import paper_2609_00865_gb300 as mw
    with pytest.raises(mw.MWError) as e:
        mw.build_visibility([50], [[(10, [(5, 12)])]])
    assert e.value.status == 2


def test_many_tiles_and_long_trajectory():
    """More tiles than one scan block (1,024) and a trajectory longer than
    one shared-memory chunk of k-tile statistics (2,048 tiles): the
    multi-block list-pointer scan, the chunked class pass and several
    256-tile compact-map chunks per segment, against the oracle."""
    c = synth.CONFIGS[5]
    r = synth.record(4, [300_000, 70_000, 0, 140_000], 6, 0.6, c["summary"], c["prompt"], c["Lp"], c["Lo"], 7700)
    assert sum((T + 127) // 128 for T in r.seqlens) > 3 * 1024
    _compare(r.seqlens, r.edits)


def _mask_case(seqlens, edits):
    import torch
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    for b, (T, e) in enumerate(zip(seqlens, edits)):
        got = mw.export_dense_mask(vis, seqlens, b)
        torch.cuda.synchronize()
        want = OV.dense_mask(T, e)
        np.testing.assert_array_equal(got.cpu().numpy(), want, err_msg=f"trajectory {b}")


def test_dense_mask_export_running_example_and_random():
    """mw_export_dense_mask against the oracle's literal dense mask (list
    membership of each row's live view, causal), bit for bit."""
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "running_example.json")))
    _mask_case([14], [[(J, [tuple(s) for s in sp]) for J, sp in g["edits"]]])
    rng = np.random.default_rng(11)
    for _ in range(4):
        _mask_case(*_rand_record(rng, int(rng.integers(1, 5))))
    _mask_case([300, 0, 129], [[(100, [(0, 50)])], [], [(5, [(1, 3)])]])


def test_dense_mask_export_config2_trajectory():
    """One 16,384-token trajectory of the attention workload (32 MB of bits)."""
    r = synth.config_record(2)
    _mask_case(r.seqlens[:1], r.edits[:1])


def test_builds_back_to_back_without_synchronising():
    """Records of different sizes built one after another with no
    synchronisation in between, on one stream and then alternating two: the
    builder's two page-locked staging buffers are reused (and grown) while
    earlier builds may still be in flight. Every build equals the oracle's."""
    import torch
    import paper_2609_00865_gb300 as mw
    rng = np.random.default_rng(77)
    recs = [_rand_record(rng, int(rng.integers(1, 6))) for _ in range(6)]
    big = synth.config_record(2)
    recs.insert(3, (big.seqlens, big.edits))          # grows the staging buffers mid-run
    streams = [torch.cuda.current_stream(), torch.cuda.Stream()]
    built = []
    for i, r in enumerate(recs + recs):
        s = streams[0] if i < len(recs) else streams[i % 2]
        built.append((r, mw.build_visibility(*r, stream=s)))
    torch.cuda.synchronize()
    for r, vis in built:
        vis.check_status()
        _check_arrays(vis.arrays(), *r)


def test_build_beside_a_large_upload():
    """A build issued while a 1 GiB upload from page-locked memory runs on
    another stream (a training loop prefetching its next batch) is correct;
    its record goes up by a kernel, not behind that copy."""
    import torch
    import paper_2609_00865_gb300 as mw
    h = torch.empty(1 << 30, dtype=torch.uint8).pin_memory()
    d = torch.empty(1 << 30, dtype=torch.uint8, device="cuda")
    copy = torch.cuda.Stream()
    rec = synth.config_record(2)
    with torch.cuda.stream(copy):
        d.copy_(h, non_blocking=True)
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    torch.cuda.synchronize()
    vis.check_status()
    _check_arrays(vis.arrays(), rec.seqlens, rec.edits)

