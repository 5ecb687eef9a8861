"""The debug library (libmw_debug.so: the kernels with index checks) on the
GPU. ``debug_workload.py`` runs every kernel family that indexes through
memory on the debug library in a child process; each run's status check must
stay clean (no index out of range anywhere), and its results must equal the
release library's on the same inputs: the checks change no arithmetic."""

import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_debug_library_clean_and_equal_to_release(tmp_path):
    import paper_2609_00865_gb300 as mw  # noqa: F401  (release library in this process)
    from paper_2609_00865_gb300 import _lib
    debug_so = os.path.join(ROOT, "paper_2609_00865_gb300", "libmw_debug.so")
    if not os.path.exists(debug_so):
        from paper_2609_00865_gb300 import build as B
        B.build(debug=True)
    assert _lib.build_flags() == 0
    out = tmp_path / "debug.pt"
    env = dict(os.environ, MW_DEBUG="1")
    r = subprocess.run([sys.executable, os.path.join(HERE, "debug_workload.py"), str(out)], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "status checks clean" in r.stdout

    import debug_workload as D
    want = D.run_all()
    got = torch.load(out)
    assert set(got) == set(want)
    for case in want:
        assert set(got[case]) == set(want[case]), case
        for k, w in want[case].items():
            g = got[case][k]
            assert g.dtype == w.dtype and g.shape == w.shape, (case, k)
            assert torch.equal(g, w), (case, k, (g.double() - w.double()).abs().max().item())
