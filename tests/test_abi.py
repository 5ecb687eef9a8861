"""C-ABI checks that need no GPU: the library loads, exports every symbol the
header declares, and rejects malformed calls on the host before any launch."""

import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _lib():
    mw = pytest.importorskip("paper_2609_00865_gb300")
    from paper_2609_00865_gb300 import _lib as L
    if not os.path.exists(L.LIB_PATH):
        from paper_2609_00865_gb300 import build as B
        B.build()
    return L, L._lib()


def _declared():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            names |= set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(mw_\w+)\s*\(", src, re.M))
    return names


def test_header_symbols_exported():
    L, h = _lib()
    declared = _declared()
    assert {"mw_build_visibility", "mw_masked_attn_fwd", "mw_masked_attn_bwd",
            "mw_logprob_loss_fwd", "mw_logprob_loss_bwd"} <= declared
    for name in declared:
        assert hasattr(h, name), name
    assert declared <= set(L.exported_names())


def test_debug_library_exports_the_same_symbols():
    """libmw_debug.so (-DMW_DEBUG: index checks in the kernels) carries the
    same ABI as libmw.so and says which it is through mw_build_flags."""
    L, h = _lib()
    from paper_2609_00865_gb300 import build as B
    if not os.path.exists(B.LIB_DEBUG):
        B.build(debug=True)
    d = ctypes.CDLL(B.LIB_DEBUG)
    for name in _declared():
        assert hasattr(d, name), name
    assert (h.mw_build_flags(), d.mw_build_flags()) == (0, 1)
    assert d.mw_abi_version() == h.mw_abi_version()


def test_status_strings_and_version():
    L, h = _lib()
    assert h.mw_status_str(0) == b"ok"
    assert b"junction" in h.mw_status_str(2)
    assert h.mw_abi_version() >= 1


def test_layout_is_host_only_and_consistent():
    L, h = _lib()
    cu = np.array([0, 300, 300, 1000], np.int32)   # includes an empty trajectory
    lay = L.mw_visibility_layout(cu, np.array([0, 2, 2], np.int32), 5)
    assert lay.n_traj == 3 and lay.total_tokens == 1000
    assert lay.n_tiles == 3 + 0 + 6
    assert lay.n_tri == 6 + 0 + 21
    assert lay.n_keymask == 2 * 3 + 1 * 0 + 3 * 6
    assert lay.max_segs == 3
    offs = sorted(getattr(lay, f) for f, _ in L.VisLayout._fields_ if f.startswith("off_"))
    assert all(o % 256 == 0 for o in offs) and offs == sorted(set(offs))
    assert lay.vis_bytes >= offs[-1]


@pytest.mark.parametrize("cu,jt,err", [
    ([5, 10], [], 2),          # cu_seqlens must start at 0
    ([0, 10, 5], [], 2),       # decreasing offsets
    ([0, 10], [1], 2),         # junction names a missing trajectory
    ([0, 10, 20], [1, 0], 2),  # junctions not grouped by trajectory
])
def test_layout_rejects_bad_shapes(cu, jt, err):
    L, h = _lib()
    with pytest.raises(L.MWError) as e:
        L.mw_visibility_layout(np.array(cu, np.int32), np.array(jt, np.int32), 0)
    assert e.value.status == err


@pytest.mark.parametrize("J,spans,off", [
    ([0], [], [0, 0]),              # junction at 0
    ([10], [], [0, 0]),             # junction at T
    ([5, 5], [], [0, 0, 0]),        # not ascending
    ([5], [[2, 7]], [0, 1]),        # span past J
    ([5], [[3, 3]], [0, 1]),        # empty span
    ([5], [[-1, 2]], [0, 1]),       # negative start
])
def test_build_rejects_bad_records_before_launch(J, spans, off):
    """Validation runs on the host; with null device buffers nothing could
    be launched, so an MW_EEDITS here proves the check precedes any launch."""
    L, h = _lib()
    cu = np.array([0, 10], np.int32)
    jt = np.zeros(len(J), np.int32)
    lay = L.mw_visibility_layout(cu, jt, len(spans))
    sp = np.array(spans, np.int32).reshape(-1)
    st = h.mw_build_visibility(ctypes.byref(lay), cu.ctypes.data_as(L._IP), len(J),
                               np.array(J, np.int32).ctypes.data_as(L._IP), jt.ctypes.data_as(L._IP),
                               np.array(off, np.int32).ctypes.data_as(L._IP),
                               sp.ctypes.data_as(L._IP) if sp.size else None,
                               ctypes.c_void_p(256), ctypes.c_void_p(256), None)
    assert st == 2


def test_build_rejects_unaligned_buffers_before_launch():
    """`vis` and `ws` must be 256-byte aligned (the layout's arrays sit at
    256-byte offsets): a valid record with an unaligned buffer is MW_EINVAL,
    found on the host before anything could be launched."""
    L, h = _lib()
    cu = np.array([0, 10], np.int32)
    J, jt, off = np.array([5], np.int32), np.zeros(1, np.int32), np.array([0, 1], np.int32)
    sp = np.array([2, 4], np.int32)
    lay = L.mw_visibility_layout(cu, jt, 1)
    for vis, ws in ((16, 256), (256, 16)):
        st = h.mw_build_visibility(ctypes.byref(lay), cu.ctypes.data_as(L._IP), 1, J.ctypes.data_as(L._IP),
                                   jt.ctypes.data_as(L._IP), off.ctypes.data_as(L._IP), sp.ctypes.data_as(L._IP),
                                   ctypes.c_void_p(ws), ctypes.c_void_p(vis), None)
        assert st == 1


def test_attention_and_lmhead_reject_bad_args_on_host():
    L, h = _lib()
    lay = L.mw_visibility_layout(np.array([0, 10], np.int32), np.zeros(0, np.int32), 0)
    P = ctypes.c_void_p(16)
    # Hq not a multiple of Hkv
    assert h.mw_masked_attn_fwd(ctypes.byref(lay), P, P, P, P, P, P, 6, 4, 128, 1, 0.1, P, None) == 3
    # bad dtype, bad head dim, bad scale
    assert h.mw_masked_attn_fwd(ctypes.byref(lay), P, P, P, P, P, P, 4, 4, 128, 7, 0.1, P, None) == 4
    assert h.mw_masked_attn_fwd(ctypes.byref(lay), P, P, P, P, P, P, 4, 4, 96, 1, 0.1, P, None) == 3
    assert h.mw_masked_attn_fwd(ctypes.byref(lay), P, P, P, P, P, P, 4, 4, 128, 1, -1.0, P, None) == 1
    # log-prob: M > N, bad eps, null loss
    n = ctypes.c_size_t()
    assert h.mw_logprob_ws(10, 11, 128, 100, 0, ctypes.byref(n)) == 3
    assert h.mw_logprob_loss_fwd(P, P, P, P, 4, P, P, 1.5, 0.2, 10, 128, 100, 0, P, P, P, P, P, None) == 1
    assert h.mw_logprob_loss_fwd(P, P, P, P, 4, P, P, 0.2, 0.2, 10, 128, 100, 0, P, P, P, None, P, None) == 1
    # KL term: negative or non-finite beta; beta > 0 without lp_ref
    assert h.mw_logprob_loss_fwd_kl(P, P, P, P, 4, P, P, 0.2, 0.2, P, -1.0, 10, 128, 100, 0, P, P, P, P, P, None) == 1
    assert h.mw_logprob_loss_fwd_kl(P, P, P, P, 4, P, P, 0.2, 0.2, P, float("nan"), 10, 128, 100, 0, P, P, P, P, P,
                                    None) == 1
    assert h.mw_logprob_loss_fwd_kl(P, P, P, P, 4, P, P, 0.2, 0.28, None, 1e-3, 10, 128, 100, 0, P, P, P, P, P,
                                    None) == 1


def test_rope_entry_points_reject_bad_args_on_host():
    L, h = _lib()
    lay = L.mw_visibility_layout(np.array([0, 10], np.int32), np.zeros(0, np.int32), 0)
    P = ctypes.c_void_p(16)
    # table: negative length, odd head dim, bad theta
    assert h.mw_rope_table(-1, 128, 1e4, P, None) == 3
    assert h.mw_rope_table(10, 127, 1e4, P, None) == 3
    assert h.mw_rope_table(10, 128, 0.0, P, None) == 1
    assert h.mw_rope_table(10, 128, float("inf"), P, None) == 1
    assert h.mw_rope_table(10, 128, 1e4, None, None) == 1
    # rows: table shorter than 128 * max_tiles, bad dtype, no heads, null pos
    assert h.mw_rope_rows(ctypes.byref(lay), P, P, P, 64, P, P, 2, 128, 1, 0, None) == 3
    assert h.mw_rope_rows(ctypes.byref(lay), P, P, P, 128, P, P, 2, 128, 7, 0, None) == 4
    assert h.mw_rope_rows(ctypes.byref(lay), P, P, P, 128, P, P, 0, 128, 1, 0, None) == 3
    assert h.mw_rope_rows(ctypes.byref(lay), P, None, P, 128, P, P, 2, 128, 1, 0, None) == 1
    assert h.mw_logical_positions(ctypes.byref(lay), P, None, None) == 1
    # attention: short table, missing workspace, GQA shape
    args = (P, P, P, P, P, 4, 2, 128, 1, 0.1)   # Q K V O LSE Hq Hkv Dh dtype scale
    assert h.mw_masked_attn_rope_fwd(ctypes.byref(lay), P, P, P, 64, *args, P, None) == 3
    assert h.mw_masked_attn_rope_fwd(ctypes.byref(lay), P, P, P, 128, *args, None, None) == 1
    assert h.mw_masked_attn_rope_fwd(ctypes.byref(lay), P, P, P, 128, P, P, P, P, P, 6, 4, 128, 1, 0.1, P,
                                     None) == 3
    assert h.mw_masked_attn_rope_bwd(ctypes.byref(lay), P, P, P, 64, P, P, P, P, P, P, P, P, P, 4, 2, 128, 1, 0.1,
                                     P, None) == 3


def test_rope_workspace_holds_rotated_queries_and_keys():
    L, h = _lib()
    cu = np.array([0, 300, 1000], np.int32)
    lay = L.mw_visibility_layout(cu, np.array([0, 1, 1], np.int32), 4)
    Hq, Hkv, Dh = 4, 2, 128
    krows = lay.n_keymask * 128
    for dtype, esz in ((0, 4), (1, 2)):
        f, b = L.mw_masked_attn_rope_ws(L.Visibility(lay, None, None), Hq, Hkv, Dh, dtype)
        # rotated queries, then (CUDA cores) the segment key rows or (tensor
        # cores) the compact K and V, both krows rows
        need = esz * lay.total_tokens * Hq * Dh + (esz if dtype == 0 else 2 * esz) * krows * Hkv * Dh
        assert need <= f < need + 1024
        if dtype == 0:
            # CUDA-core backward: Delta per (head, row) and the float32 segment-key gradient
            need_b = f + 4 * lay.total_tokens * Hq + 4 * krows * Hkv * Dh
        else:
            # tensor-core backward: the (-LSE log2 e, Delta) pair array over whole
            # tiles, and float32 dK and dV partials per compact row
            need_b = f + 8 * lay.n_tiles * 128 * Hq + 2 * 4 * krows * Hkv * Dh
        assert need_b <= b < need_b + 1536


def test_diverging_rows_rejects_null_output():
    L, h = _lib()
    lay = L.mw_visibility_layout(np.array([0, 10], np.int32), np.zeros(0, np.int32), 0)
    assert h.mw_diverging_rows(ctypes.byref(lay), ctypes.c_void_p(16), None, None) == 1
    assert h.mw_diverging_rows(None, ctypes.c_void_p(16), ctypes.c_void_p(16), None) == 1


def test_forward_kl_rejects_bad_args_on_host():
    L, h = _lib()
    P = ctypes.c_void_p(16)
    n = ctypes.c_size_t()
    assert h.mw_forward_kl_ws(4, 512, 100, 0, ctypes.byref(n)) == 3          # d above the CUDA-core limit
    assert h.mw_forward_kl_ws(4, 64, 100, 9, ctypes.byref(n)) == 4           # dtype
    assert h.mw_forward_kl_ws(4, 64, 100, 0, ctypes.byref(n)) == 0 and n.value >= 2 * 4 * 4
    # more pairs than (distinct) student rows, no teacher rows, negative lambda, null loss
    assert h.mw_forward_kl_fwd(P, P, P, P, 5, P, 8, 4, 64, 100, 0, 0.1, P, P, P, None) == 3
    assert h.mw_forward_kl_fwd(P, P, P, P, 4, P, 0, 8, 64, 100, 0, 0.1, P, P, P, None) == 3
    assert h.mw_forward_kl_fwd(P, P, P, P, 4, P, 4, 8, 64, 100, 0, -0.1, P, P, P, None) == 1
    assert h.mw_forward_kl_fwd(P, P, P, P, 4, P, 4, 8, 64, 100, 0, 0.1, P, None, P, None) == 1
    assert h.mw_forward_kl_bwd(P, P, P, P, 4, P, 4, 8, 64, 100, 0, 0.1, float("nan"), 0, P, P, P, None) == 1
    assert h.mw_forward_kl_bwd(P, P, P, P, 4, P, 4, 8, 64, 100, 0, 0.1, 1.0, 0, P, P, None, None) == 1


def test_logdiff_rejects_bad_args_on_host():
    L, h = _lib()
    P = ctypes.c_void_p(16)
    assert h.mw_logdiff(P, P, -1, P, None) == 3
    assert h.mw_logdiff(P, P, 4, None, None) == 1
    assert h.mw_logdiff(None, P, 4, P, None) == 1


def test_final_walk_rejects_null_outputs():
    L, h = _lib()
    lay = L.mw_visibility_layout(np.array([0, 10], np.int32), np.zeros(0, np.int32), 0)
    P = ctypes.c_void_p(16)
    assert h.mw_final_walk(ctypes.byref(lay), P, P, P, None, None) == 1
    assert h.mw_final_walk(ctypes.byref(lay), P, None, P, P, None) == 1
    assert h.mw_final_walk(None, P, P, P, P, None) == 1


_C_PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "mw.h"
int main(void) {
    int32_t cu[3] = {0, 300, 1000};
    int32_t jt[2] = {1, 1};
    mw_vis_layout L;
    if (mw_visibility_layout(2, cu, 2, jt, 3, &L) != MW_OK) return 2;
    if (L.n_tiles != 3 + 6 || L.max_segs != 3 || L.vis_bytes <= 0) return 3;
    if (mw_visibility_layout(2, cu, 2, jt, -1, &L) == MW_OK) return 4;   /* negative span count */
    if (strcmp(mw_status_str(MW_OK), "ok") != 0) return 5;
    printf("%d %lld\n", mw_abi_version(), (long long)L.n_keymask);
    return 0;
}
"""


def test_c_program_links_and_calls_the_abi(tmp_path):
    """The boundary is a C ABI: a C99 program includes the header, links
    libmw.so and calls its host-only entry points (no GPU needed)."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    L, _ = _lib()
    src = tmp_path / "abi.c"
    src.write_text(_C_PROGRAM)
    exe = tmp_path / "abi"
    libdir = os.path.dirname(L.LIB_PATH)
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-pedantic", "-I", os.path.join(ROOT, "include"),
                        str(src), "-L", libdir, "-lmw", "-Wl,-rpath," + libdir, "-o", str(exe)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    env = dict(os.environ)
    env["LD_LIBRARY_PATH"] = ":".join(p for p in (libdir, "/usr/local/cuda/lib64", env.get("LD_LIBRARY_PATH", ""))
                                      if p)
    run = subprocess.run([str(exe)], capture_output=True, text=True, env=env)
    assert run.returncode == 0, (run.returncode, run.stderr)
    ver, n_keymask = map(int, run.stdout.split())
    assert ver >= 4 and n_keymask == (1 + 0) * 3 + (1 + 2) * 6


def test_dense_mask_export_rejects_bad_args_on_host():
    L, h = _lib()
    cu = np.array([0, 10, 70000], np.int32)
    lay = L.mw_visibility_layout(cu, np.zeros(0, np.int32), 0)
    P = ctypes.c_void_p(256)
    cup = cu.ctypes.data_as(L._IP)
    assert h.mw_export_dense_mask(ctypes.byref(lay), P, cup, 1, P, None) == 3      # T > MW_DENSE_MASK_MAX_T
    assert h.mw_export_dense_mask(ctypes.byref(lay), P, cup, -1, P, None) == 1     # no such trajectory
    assert h.mw_export_dense_mask(ctypes.byref(lay), P, cup, 2, P, None) == 1
    assert h.mw_export_dense_mask(ctypes.byref(lay), P, None, 0, P, None) == 1     # offsets missing
    assert h.mw_export_dense_mask(ctypes.byref(lay), P, cup, 0, None, None) == 1   # mask missing
    bad = np.array([0, 10, 60000], np.int32)                                       # offsets of another record
    assert h.mw_export_dense_mask(ctypes.byref(lay), P, bad.ctypes.data_as(L._IP), 0, P, None) == 1
