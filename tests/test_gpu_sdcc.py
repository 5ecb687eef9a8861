"""GPU diverging rows of SDCC (§5; App. B Def. "trajectory tree") vs the
oracle, bit for bit."""

import json
import os

import numpy as np
import pytest
import torch

from oracle import sdcc as OS

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(__file__)


def _check(seqlens, edits):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    got = mw.diverging_rows(vis)
    torch.cuda.synchronize()
    want = np.concatenate([OS.diverging_rows(T, e) for T, e in zip(seqlens, edits)]).astype(np.uint8)
    np.testing.assert_array_equal(got.cpu().numpy()[: want.size], want)
    return want


def test_running_example():
    with open(os.path.join(HERE, "golden", "running_example.json")) as f:
        g = json.load(f)
    edits = [(J, [tuple(s) for s in spans]) for J, spans in g["edits"]]
    want = _check([len(g["tokens"])], [edits])
    assert want.sum() == 5   # y6, y7, y9, y10, y12


def test_packed_ragged_record_with_overlaps():
    """Several trajectories (an empty one, one longer than a 1024-row scan
    chunk), overlapping spans evicted twice."""
    seqlens = [1, 0, 300, 2500, 129]
    edits = [[], [], [(150, [(20, 140)]), (280, [(150, 260), (20, 40)])],
             [(1100, [(10, 900)]), (2000, [(1000, 1900), (5, 8)]), (2400, [(2001, 2300)])],
             [(128, [(5, 127)])]]
    _check(seqlens, edits)
