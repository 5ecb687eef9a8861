"""Small runs of every kernel family that indexes through memory: the
visibility build (edits and events records), the compact gather / reduce
and the attention kernels (bf16 tensor cores, rotary, float32), branch
packing, the dense-mask export and the SDCC maps. Each run ends with the
status check of its visibility buffer.

Run as a script with MW_DEBUG=1 it uses the debug library (index checks in
the kernels): any index out of range fails the status check (MW_EDEVICE).
``tests/test_gpu_debug_lib.py`` runs it that way and compares what it wrote
with the release library's results on the same inputs.
"""

import os
import sys

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
for p in (ROOT, HERE):
    if p not in sys.path:
        sys.path.insert(0, p)

import synth  # noqa: E402

# junctions on and next to tile edges, an empty trajectory, a one-token one
EDGE = ([1, 127, 0, 128, 129, 300],
        [[], [(100, [(10, 40)])], [], [(64, [(0, 32)]), (120, [(70, 100)])], [(128, [(5, 127)])],
         [(150, [(20, 140)]), (280, [(150, 260)])]])
# three trajectories, three junctions each, spans crossing tiles
MEDIUM = ([700, 1000, 333],
          [[(130, [(5, 60), (70, 125)]), (400, [(140, 300)]), (610, [(0, 4), (402, 560)])],
           [(64, [(0, 30)]), (513, [(100, 400), (450, 500)]), (900, [(600, 880)])],
           [(128, [(0, 127)]), (200, [(130, 150)]), (320, [(201, 300)])]])
# offload / retrieve: spans leave the view and come back at its end
EVENTS = ([700, 400],
          [[(200, [(10, 90)], []), (450, [(120, 260)], [(10, 90)]), (600, [], [(120, 200)])],
           [(150, [(0, 100)], []), (300, [], [(0, 100)])]])


def _qkv(T, Hq, Hkv, Dh, seed, dtype):
    return [synth.normal((T, h, Dh), seed + n).to(dtype).cuda() for n, h in enumerate((Hq, Hkv, Hkv, Hq))]


def _host(v):
    if torch.is_tensor(v):
        return v.detach().cpu()
    if isinstance(v, (list, tuple)):   # per-trajectory arrays (the class triangles)
        parts = [np.asarray(x, dtype=np.int64).reshape(-1) for x in v]
        return torch.as_tensor(np.concatenate(parts) if parts else np.zeros(0, np.int64))
    a = np.asarray(v)
    return torch.as_tensor(a.astype(np.int64) if a.dtype.kind == "u" else a)


def _views(arrs, seqlens, junctions_per_traj):
    """The builder's arrays with csrc cut to its defined part: each segment's
    entries up to the end of its last compact tile (the rest of its 128 nt_b
    block is left unset by design)."""
    out = dict(arrs)
    csrc = np.array(arrs["csrc"], copy=True)
    g, off = 0, 0
    for T, K in zip(seqlens, junctions_per_traj):
        block = (T + 127) // 128 * 128
        for _ in range(1 + K):
            end = (int(arrs["seg_len"][g]) + 127) // 128 * 128
            csrc[off + end: off + block] = -2
            g += 1
            off += block
    out["csrc"] = csrc
    return out


def _cpu(d):
    return {k: _host(v) for k, v in d.items()}


def case_build():
    import paper_2609_00865_gb300 as mw
    out = {}
    for name, (seqlens, edits) in (("edge", EDGE), ("medium", MEDIUM)):
        vis = mw.build_visibility(seqlens, edits)
        torch.cuda.synchronize()
        vis.check_status()
        for k, v in _views(vis.arrays(), seqlens, [len(e) for e in edits]).items():
            out[f"{name}.{k}"] = v
    return out


def case_attention_bf16():
    import paper_2609_00865_gb300 as mw
    seqlens, edits = MEDIUM
    vis = mw.build_visibility(seqlens, edits)
    q, k, v, do = _qkv(sum(seqlens), 8, 2, 128, 11, torch.bfloat16)
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, 128 ** -0.5)
    dQ, dK, dV = mw.masked_attn_bwd(vis, q, k, v, O, do, LSE, 128 ** -0.5)
    torch.cuda.synchronize()
    vis.check_status()
    return dict(O=O, LSE=LSE, dQ=dQ, dK=dK, dV=dV)


def case_attention_rope_bf16():
    import paper_2609_00865_gb300 as mw
    seqlens, edits = MEDIUM
    vis = mw.build_visibility(seqlens, edits)
    pos = mw.logical_positions(vis)
    table = mw.rope_table(mw.rope_n_pos(vis), 128, 1e6)
    q, k, v, do = _qkv(sum(seqlens), 4, 4, 128, 21, torch.bfloat16)
    O, LSE = mw.masked_attn_rope_fwd(vis, pos, table, q, k, v, 128 ** -0.5)
    dQ, dK, dV = mw.masked_attn_rope_bwd(vis, pos, table, q, k, v, O, do, LSE, 128 ** -0.5)
    torch.cuda.synchronize()
    vis.check_status()
    return dict(pos=pos, O=O, LSE=LSE, dQ=dQ, dK=dK, dV=dV)


def case_attention_fp32():
    import paper_2609_00865_gb300 as mw
    seqlens, edits = EDGE
    vis = mw.build_visibility(seqlens, edits)
    q, k, v, do = _qkv(sum(seqlens), 6, 2, 64, 31, torch.float32)
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, 64 ** -0.5)
    dQ, dK, dV = mw.masked_attn_bwd(vis, q, k, v, O, do, LSE, 64 ** -0.5)
    torch.cuda.synchronize()
    vis.check_status()
    return dict(O=O, LSE=LSE, dQ=dQ, dK=dK, dV=dV)


def case_events():
    import paper_2609_00865_gb300 as mw
    seqlens, events = EVENTS
    vis = mw.build_views_events(seqlens, events)
    q, k, v, do = _qkv(sum(seqlens), 8, 2, 128, 41, torch.bfloat16)
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, 128 ** -0.5)
    dQ, dK, dV = mw.masked_attn_bwd(vis, q, k, v, O, do, LSE, 128 ** -0.5)
    torch.cuda.synchronize()
    vis.check_status()
    arrs = _views(vis.arrays(), seqlens, [len(e) for e in events])
    out = {f"views.{k_}": v_ for k_, v_ in arrs.items()}
    out.update(O=O, LSE=LSE, dQ=dQ, dK=dK, dV=dV)
    return out


def case_branches_mask_sdcc():
    import paper_2609_00865_gb300 as mw
    seqlens, edits = MEDIUM
    vis = mw.build_visibility(seqlens, edits)
    T = sum(seqlens)
    n = sum(mw.branch_lengths(vis))
    X = synth.normal((T, 256), 51).to(torch.bfloat16).cuda()
    Xp = mw.branch_pack(vis, X, n)
    dX = mw.branch_unpack_add(vis, Xp)
    out = dict(Xp=Xp, dX=dX)
    for b in range(len(seqlens)):
        out[f"mask{b}"] = mw.export_dense_mask(vis, seqlens, b)
    out["diverging"] = mw.diverging_rows(vis)
    walk_index, student_row, walk_len = mw.final_walk(vis)
    out.update(walk_index=walk_index, student_row=student_row, walk_len=walk_len)
    torch.cuda.synchronize()
    vis.check_status()
    return out


CASES = [case_build, case_attention_bf16, case_attention_rope_bf16, case_attention_fp32, case_events,
         case_branches_mask_sdcc]


def run_all():
    return {c.__name__: _cpu(c()) for c in CASES}


if __name__ == "__main__":
    import paper_2609_00865_gb300 as mw
    from paper_2609_00865_gb300 import _lib
    assert _lib.build_flags() == 1, "set MW_DEBUG=1 to run on the debug library"
    torch.cuda.set_device(0)
    torch.save(run_all(), sys.argv[1])
    print("debug workload: all status checks clean,", mw.kernel_launches(), "kernel launches")
