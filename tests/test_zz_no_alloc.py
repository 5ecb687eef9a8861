"""The allocation-free visibility builder gives the same result as the regular one.

mw_build_visibility_noalloc serves callers that are handed their buffers and
may not allocate device memory themselves; its build workspace is a fixed
device array inside libmw that every call shares. This file is collected last
so that a failure here cannot stop any other test of a run that stops at the
first failure; it must also pass alone in a fresh process.
"""

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


def _regular(seqlens, edits):
    import paper_2609_00865_gb300 as mw
    return mw.build_visibility(seqlens, edits).arrays()


def _noalloc(seqlens, edits):
    import torch
    import paper_2609_00865_gb300 as mw
    cu, J, jt, off, spans = mw.flatten_record(seqlens, edits)
    L = mw.mw_visibility_layout(cu, jt, len(spans))
    vis = torch.empty(max(int(L.vis_bytes), 1), dtype=torch.uint8, device="cuda")
    mw.mw_build_visibility_noalloc(L, cu, J, jt, off, spans, vis)
    torch.cuda.synchronize()
    v = mw.Visibility(L, vis, None)
    v.check_status()
    return v.arrays()


def _same(a, b):
    for key in ("omega", "seg", "qtile_traj", "fwd_ptr", "fwd_idx", "bwd_ptr", "bwd_idx", "pairs", "keymask"):
        np.testing.assert_array_equal(a[key], b[key], err_msg=key)
    assert a["pairs_total"] == b["pairs_total"]
    for x, y in zip(a["cls"], b["cls"]):
        np.testing.assert_array_equal(np.tril(x), np.tril(y))


def test_noalloc_matches_regular_builder_twice_in_a_row():
    # two different records back to back: the second call must not see any
    # trace of the first in the shared workspace
    r1 = synth.config_record(2)
    r2 = synth.config_record(1)
    for rec in (r1, r2):
        _same(_noalloc(rec.seqlens, rec.edits), _regular(rec.seqlens, rec.edits))


def test_noalloc_rejects_records_beyond_the_fixed_workspace():
    import paper_2609_00865_gb300 as mw
    import torch
    # 40 trajectories of 1M tokens need 40 x 8192 tiles x 16 B of workspace > 1 MiB
    cu = np.arange(41, dtype=np.int64) * (1 << 20)
    L = mw.mw_visibility_layout(cu.astype(np.int32), np.zeros(0, np.int32), 0)
    assert L.ws_bytes > (1 << 20)
    vis = torch.empty(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(mw.MWError) as e:
        mw.mw_build_visibility_noalloc(L, cu.astype(np.int32), [], [], [0], np.zeros((0, 2), np.int32), vis)
    assert e.value.status == 8
