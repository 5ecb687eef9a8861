"""ctypes binding of libmw (include/mw.h): argument marshalling only.

Every step of the path runs inside libmw's CUDA kernels; this module converts
torch tensors to pointers, allocates outputs with torch (device memory and
streams are torch's), and raises ``MWError`` on a non-OK status. It fails
loudly when libmw.so is missing: there is no CPU fallback.
"""

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
# MW_DEBUG=1 in the environment selects the debug library (index checks in
# the kernels; build.build(debug=True) makes it)
DEBUG = os.environ.get("MW_DEBUG") == "1"
LIB_PATH = os.path.join(HERE, "libmw_debug.so" if DEBUG else "libmw.so")

MW_F32, MW_BF16 = 0, 1
TILE = 128
STATUS = ["MW_OK", "MW_EINVAL", "MW_EEDITS", "MW_ESHAPE", "MW_EDTYPE", "MW_ECUDA",
          "MW_ETIMEOUT", "MW_EDEVICE", "MW_ENOSPACE"]


class MWError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        name = STATUS[status] if 0 <= status < len(STATUS) else str(status)
        super().__init__(f"{where}: {name} ({_lib().mw_status_str(status).decode()})")


class VisLayout(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("n_traj", "n_junc", "n_spans", "max_tiles")] + \
               [(n, ctypes.c_int64) for n in (
                   "total_tokens", "n_tiles", "n_tri", "n_segs", "n_keymask",
                   "off_omega", "off_seg", "off_traj_tok", "off_traj_tile", "off_traj_seg",
                   "off_traj_tri", "off_traj_km", "off_seg_start", "off_tile_traj", "off_cls",
                   "off_fwd_ptr", "off_fwd_idx", "off_bwd_ptr", "off_bwd_idx", "off_pairs",
                   "off_keymask", "off_status", "vis_bytes",
                   "ws_off_spans", "ws_off_tstat", "ws_off_cnt", "ws_bytes", "max_segs",
                   "off_seg_len", "off_cpos", "off_csrc", "kind")]


_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_LP = ctypes.POINTER(VisLayout)
_IP = ctypes.POINTER(ctypes.c_int32)

_SIGS = {
    "mw_status_str": (ctypes.c_char_p, [_I]),
    "mw_last_cuda_error": (_I, []),
    "mw_abi_version": (_I, []),
    "mw_build_flags": (_I, []),
    "mw_kernel_launches": (ctypes.c_uint64, []),
    "mw_visibility_layout": (_I, [_I, _IP, _I, _IP, _I, _LP]),
    "mw_build_visibility": (_I, [_LP, _IP, _I, _IP, _IP, _IP, _IP, _P, _P, _P]),
    "mw_build_visibility_noalloc": (_I, [_LP, _IP, _I, _IP, _IP, _IP, _IP, _P, _P]),
    "mw_events_layout": (_I, [_I, _IP, _I, _IP, _I, _LP]),
    "mw_branch_pack": (_I, [_LP, _P, _P, _P, _I, _I, _P]),
    "mw_branch_unpack_add": (_I, [_LP, _P, _P, _P, _I, _I, _P]),
    "mw_build_views_events": (_I, [_LP, _IP, _I, _IP, _IP, _IP, _IP, _IP, _P, _P, _P]),
    "mw_masked_attn_fwd_ws": (_I, [_LP, _I, _I, _I, ctypes.POINTER(ctypes.c_size_t)]),
    "mw_masked_attn_fwd": (_I, [_LP, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _F, _P, _P]),
    "mw_masked_attn_bwd_ws": (_I, [_LP, _I, _I, _I, _I, ctypes.POINTER(ctypes.c_size_t)]),
    "mw_masked_attn_bwd": (_I, [_LP, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _F, _P, _P]),
    "mw_logprob_ws": (_I, [_I, _I, _I, _I, _I, ctypes.POINTER(ctypes.c_size_t)]),
    "mw_logprob_loss_fwd": (_I, [_P, _P, _P, _P, _I, _P, _P, _F, _F, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P]),
    "mw_logprob_loss_fwd_kl": (_I, [_P, _P, _P, _P, _I, _P, _P, _F, _F, _P, _F, _I, _I, _I, _I, _P, _P, _P, _P, _P,
                                    _P]),
    "mw_logprob_loss_bwd": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _F, _P, _P, _P]),
    "mw_logical_positions": (_I, [_LP, _P, _P, _P]),
    "mw_diverging_rows": (_I, [_LP, _P, _P, _P]),
    "mw_final_walk": (_I, [_LP, _P, _P, _P, _P, _P]),
    "mw_logdiff": (_I, [_P, _P, _I, _P, _P]),
    "mw_forward_kl_ws": (_I, [_I, _I, _I, _I, ctypes.POINTER(ctypes.c_size_t)]),
    "mw_forward_kl_fwd": (_I, [_P, _P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P]),
    "mw_forward_kl_bwd": (_I, [_P, _P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _F, _F, _I, _P, _P, _P, _P]),
    "mw_forward_kl_check_status": (_I, [_I, _I, _I, _I, _P, _P]),
    "mw_rope_table": (_I, [_I, _I, ctypes.c_double, _P, _P]),
    "mw_rope_rows": (_I, [_LP, _P, _P, _P, _I, _P, _P, _I, _I, _I, _I, _P]),
    "mw_masked_attn_rope_ws": (_I, [_LP, _I, _I, _I, _I, ctypes.POINTER(ctypes.c_size_t),
                                    ctypes.POINTER(ctypes.c_size_t)]),
    "mw_masked_attn_rope_fwd": (_I, [_LP, _P, _P, _P, _I, _P, _P, _P, _P, _P, _I, _I, _I, _I, _F, _P, _P]),
    "mw_masked_attn_rope_bwd": (_I, [_LP, _P, _P, _P, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _F,
                                     _P, _P]),
    "mw_check_status": (_I, [_LP, _P, _P]),
    "mw_export_dense_mask": (_I, [_LP, _P, _IP, _I, _P, _P]),
    "mw_logprob_check_status": (_I, [_I, _I, _I, _I, _I, _P, _P]),
    "mw_selftest_wait_timeout": (_I, [ctypes.c_int64, _P, _P]),
}

_handle = None


def _lib():
    global _handle
    if _handle is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{os.path.basename(LIB_PATH)} not built at {LIB_PATH}; run __graft_entry__.build()")
        h = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(h, name)
            fn.restype = res
            fn.argtypes = args
        _handle = h
    return _handle


def kernel_launches():
    """Kernels libmw has launched in this process so far."""
    return int(_lib().mw_kernel_launches())


def build_flags():
    """mw_build_flags(): 1 (MW_BUILD_DEBUG) for the debug library."""
    return int(_lib().mw_build_flags())


def exported_names():
    return list(_SIGS)


def _check(st, where):
    if st != 0:
        raise MWError(st, where)


def _i32(a):
    a = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return a, a.ctypes.data_as(_IP)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _dtype_code(t):
    import torch
    if t.dtype == torch.float32:
        return MW_F32
    if t.dtype == torch.bfloat16:
        return MW_BF16
    raise MWError(4, f"dtype {t.dtype}")


def _need(t, name, dtype=None, device=None):
    import torch
    if not t.is_cuda or not t.is_contiguous():
        raise MWError(1, f"{name} must be a contiguous CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise MWError(4, f"{name} dtype {t.dtype}")
    return t


# --- records ------------------------------------------------------------------

def flatten_record(seqlens, edits_per_traj):
    """Record -> (cu_seqlens, junctions, junc_traj, junc_span_off, spans) arrays."""
    cu = np.zeros(len(seqlens) + 1, dtype=np.int32)
    cu[1:] = np.cumsum(seqlens)
    J, jt, off, spans = [], [], [0], []
    for b, edits in enumerate(edits_per_traj):
        for j, sp in edits:
            J.append(j)
            jt.append(b)
            for a, e in sp:
                spans.append((a, e))
            off.append(len(spans))
    return (cu, np.asarray(J, np.int32), np.asarray(jt, np.int32), np.asarray(off, np.int32),
            np.asarray(spans, np.int32).reshape(-1, 2))


def mw_visibility_layout(cu_seqlens, junc_traj, n_spans):
    L = VisLayout()
    cu, cup = _i32(cu_seqlens)
    jt, jtp = _i32(junc_traj)
    _check(_lib().mw_visibility_layout(len(cu) - 1, cup, len(jt), jtp, int(n_spans), ctypes.byref(L)),
           "mw_visibility_layout")
    return L


def mw_build_visibility(layout, cu_seqlens, junctions, junc_traj, junc_span_off, spans, ws, vis, stream=None):
    cu, cup = _i32(cu_seqlens)
    J, Jp = _i32(junctions)
    jt, jtp = _i32(junc_traj)
    off, offp = _i32(junc_span_off)
    sp, spp = _i32(np.asarray(spans).reshape(-1))
    _check(_lib().mw_build_visibility(ctypes.byref(layout), cup, len(J), Jp, jtp, offp, spp,
                                      _ptr(ws), _ptr(vis), _stream(stream)), "mw_build_visibility")


def mw_build_visibility_noalloc(layout, cu_seqlens, junctions, junc_traj, junc_span_off, spans, vis, stream=None):
    """Allocation-free build: the workspace is libmw's fixed device array
    (for callers that may not allocate; see include/mw.h)."""
    cu, cup = _i32(cu_seqlens)
    J, Jp = _i32(junctions)
    jt, jtp = _i32(junc_traj)
    off, offp = _i32(junc_span_off)
    sp, spp = _i32(np.asarray(spans).reshape(-1))
    _check(_lib().mw_build_visibility_noalloc(ctypes.byref(layout), cup, len(J), Jp, jtp, offp, spp,
                                              _ptr(vis), _stream(stream)), "mw_build_visibility_noalloc")


def flatten_events(seqlens, events_per_traj):
    """Events record -> (cu_seqlens, junctions, junc_traj, out_off, in_off,
    spans): the out-spans of every event in event order, then the in-spans,
    in one span table; out_off / in_off are the CSR offsets of each event's
    ranges in it."""
    cu = np.zeros(len(seqlens) + 1, dtype=np.int32)
    cu[1:] = np.cumsum(seqlens)
    J, jt, outs, ins, out_off, in_off = [], [], [], [], [0], [0]
    for b, events in enumerate(events_per_traj):
        for j, sp_out, sp_in in events:
            J.append(j)
            jt.append(b)
            outs.extend((a, e) for a, e in sp_out)
            ins.extend((a, e) for a, e in sp_in)
            out_off.append(len(outs))
            in_off.append(len(ins))
    spans = np.asarray(outs + ins, np.int32).reshape(-1, 2)
    return (cu, np.asarray(J, np.int32), np.asarray(jt, np.int32), np.asarray(out_off, np.int32),
            np.asarray(in_off, np.int32) + len(outs), spans)


def mw_events_layout(cu_seqlens, junc_traj, n_spans):
    L = VisLayout()
    cu, cup = _i32(cu_seqlens)
    jt, jtp = _i32(junc_traj)
    _check(_lib().mw_events_layout(len(cu) - 1, cup, len(jt), jtp, int(n_spans), ctypes.byref(L)),
           "mw_events_layout")
    return L


def mw_build_views_events(layout, cu_seqlens, junctions, junc_traj, out_off, in_off, spans, ws, vis, stream=None):
    cu, cup = _i32(cu_seqlens)
    J, Jp = _i32(junctions)
    jt, jtp = _i32(junc_traj)
    oo, oop = _i32(out_off)
    io, iop = _i32(in_off)
    sp, spp = _i32(np.asarray(spans).reshape(-1))
    _check(_lib().mw_build_views_events(ctypes.byref(layout), cup, len(J), Jp, jtp, oop, iop, spp, _ptr(ws),
                                        _ptr(vis), _stream(stream)), "mw_build_views_events")


def build_views_events(seqlens, events_per_traj, device="cuda", stream=None):
    """Views of an events (offload / retrieve) record: flatten, allocate with
    torch, run the builder. ``events_per_traj[b]`` lists (J, out_spans,
    in_spans) per event."""
    import torch
    cu, J, jt, oo, io, spans = flatten_events(seqlens, events_per_traj)
    L = mw_events_layout(cu, jt, len(spans))
    vis = torch.empty(max(int(L.vis_bytes), 1), dtype=torch.uint8, device=device)
    ws = torch.empty(max(int(L.ws_bytes), 1), dtype=torch.uint8, device=device)
    mw_build_views_events(L, cu, J, jt, oo, io, spans, ws, vis, stream)
    return Visibility(L, vis, ws)


class Visibility:
    """Device visibility buffer of one packed record plus its layout."""

    def __init__(self, layout, vis, ws):
        self.layout = layout
        self.vis = vis
        self.ws = ws

    def _arr(self, off, count, dtype):
        import torch
        nbytes = int(count) * np.dtype(dtype).itemsize
        t = self.vis[off: off + nbytes].cpu().numpy()
        return t.view(dtype).copy()

    def arrays(self):
        """Copy every artefact to the host in the oracle's ``build`` format."""
        L = self.layout
        n = L.n_tiles
        fwd_ptr = self._arr(L.off_fwd_ptr, n + 1, np.int32)   # all zero for an events record
        bwd_ptr = self._arr(L.off_bwd_ptr, n + 1, np.int32)
        tok = self._arr(L.off_traj_tok, L.n_traj + 1, np.int32)
        tile = self._arr(L.off_traj_tile, L.n_traj + 1, np.int32)
        tri = self._arr(L.off_traj_tri, L.n_traj + 1, np.int64)
        cls_flat = self._arr(L.off_cls, L.n_tri, np.uint8)
        classes = []
        for b in range(L.n_traj):
            nt = int(tile[b + 1] - tile[b])
            c = np.zeros((nt, nt), dtype=np.int32)
            base = int(tri[b])
            for q in range(nt):
                c[q, : q + 1] = cls_flat[base + q * (q + 1) // 2: base + q * (q + 1) // 2 + q + 1]
            classes.append(c)
        pairs = self._arr(L.off_pairs, L.n_traj + 1, np.int64)
        return {
            "omega": self._arr(L.off_omega, L.total_tokens, np.int32),
            "seg": self._arr(L.off_seg, L.total_tokens, np.int32),
            "qtile_traj": self._arr(L.off_tile_traj, n, np.int32),
            "cls": classes,
            "fwd_ptr": fwd_ptr,
            "fwd_idx": self._arr(L.off_fwd_idx, int(fwd_ptr[-1]), np.int32),
            "bwd_ptr": bwd_ptr,
            "bwd_idx": self._arr(L.off_bwd_idx, int(bwd_ptr[-1]), np.int32),
            "pairs": pairs[:-1],
            "pairs_total": int(pairs[-1]),
            "keymask": self._arr(L.off_keymask, L.n_keymask * 4, np.uint32).reshape(-1, 4),
            "traj_tok": tok,
            "seg_len": self._arr(L.off_seg_len, L.n_segs, np.int32),
            "cpos": self._arr(L.off_cpos, L.n_keymask * TILE, np.int32),
            "csrc": self._arr(L.off_csrc, L.n_keymask * TILE, np.int32),
        }

    @property
    def seg_len(self):
        """Length of every segment's live view, in global segment order (host copy)."""
        L = self.layout
        return self._arr(L.off_seg_len, L.n_segs, np.int32)

    @property
    def pairs_total(self):
        L = self.layout
        return int(self._arr(L.off_pairs + 8 * L.n_traj, 1, np.int64)[0])

    def check_status(self, stream=None):
        _check(_lib().mw_check_status(ctypes.byref(self.layout), _ptr(self.vis), _stream(stream)),
               "mw_check_status")


def build_visibility(seqlens, edits_per_traj, device="cuda", stream=None):
    """Flatten a record, allocate its buffers with torch, run the builder."""
    import torch
    cu, J, jt, off, spans = flatten_record(seqlens, edits_per_traj)
    L = mw_visibility_layout(cu, jt, len(spans))
    vis = torch.empty(max(int(L.vis_bytes), 1), dtype=torch.uint8, device=device)
    ws = torch.empty(max(int(L.ws_bytes), 1), dtype=torch.uint8, device=device)
    mw_build_visibility(L, cu, J, jt, off, spans, ws, vis, stream)
    return Visibility(L, vis, ws)


def mw_export_dense_mask(vis, cu_seqlens, traj, mask, stream=None):
    cu, cup = _i32(cu_seqlens)
    _check(_lib().mw_export_dense_mask(ctypes.byref(vis.layout), _ptr(vis.vis), cup, int(traj), _ptr(mask),
                                       _stream(stream)), "mw_export_dense_mask")


def export_dense_mask(vis, seqlens, traj, stream=None):
    """Trajectory ``traj``'s dense visibility as a bool tensor [T, T] on the
    device (mw_export_dense_mask, bit-packed words unpacked here). Row i sees
    key j iff j is in the live view of i's segment at or before i's own place
    in it; for small trajectories only."""
    import torch
    cu = np.zeros(len(seqlens) + 1, dtype=np.int32)
    cu[1:] = np.cumsum(seqlens)
    T = int(seqlens[traj])
    words = (T + 31) // 32
    mask = torch.zeros(max(T * words, 1), dtype=torch.int32, device=vis.vis.device)
    mw_export_dense_mask(vis, cu, traj, mask, stream)
    bits = torch.arange(32, dtype=torch.int32, device=mask.device)
    dense = ((mask[: T * words].view(T, words, 1) >> bits) & 1).bool().view(T, words * 32)
    return dense[:, :T]


# --- branch-replicated packing (stacked layers) --------------------------------

def branch_lengths(vis):
    """Host list of every segment's compact-sequence length (|view_s|, read
    back from the build; the packed branches' record)."""
    return [int(x) for x in vis._arr(vis.layout.off_seg_len, vis.layout.n_segs, np.int32)]


def mw_branch_pack(vis, X, Xp, stream=None):
    row = int(np.prod(X.shape[1:]))
    _check(_lib().mw_branch_pack(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(X), _ptr(Xp), row, _dtype_code(X),
                                 _stream(stream)), "mw_branch_pack")


def mw_branch_unpack_add(vis, dXp, dX, stream=None):
    row = int(np.prod(dXp.shape[1:]))
    _check(_lib().mw_branch_unpack_add(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(dXp), _ptr(dX), row,
                                       _dtype_code(dXp), _stream(stream)), "mw_branch_unpack_add")


def branch_pack(vis, X, n_packed, stream=None):
    """Packed branch copies [n_packed, ...] of the per-token rows of X
    (mw_branch_pack)."""
    import torch
    Xp = torch.empty((n_packed,) + tuple(X.shape[1:]), dtype=X.dtype, device=X.device)
    mw_branch_pack(vis, X, Xp, stream)
    return Xp


def branch_unpack_add(vis, dXp, stream=None):
    """Per-token sums [total_tokens, ...] of the packed copies' rows
    (mw_branch_unpack_add)."""
    import torch
    dX = torch.empty((int(vis.layout.total_tokens),) + tuple(dXp.shape[1:]), dtype=dXp.dtype, device=dXp.device)
    mw_branch_unpack_add(vis, dXp, dX, stream)
    return dX


# --- attention ----------------------------------------------------------------

def mw_masked_attn_fwd_ws(vis, Hkv, Dh, dtype):
    n = ctypes.c_size_t()
    _check(_lib().mw_masked_attn_fwd_ws(ctypes.byref(vis.layout), Hkv, Dh, dtype, ctypes.byref(n)),
           "mw_masked_attn_fwd_ws")
    return int(n.value)


def mw_masked_attn_fwd(vis, Q, K, V, O, LSE, scale, ws, stream=None):
    Hq, Dh = Q.shape[1], Q.shape[2]
    Hkv = K.shape[1]
    _check(_lib().mw_masked_attn_fwd(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(Q), _ptr(K), _ptr(V),
                                     _ptr(O), _ptr(LSE), Hq, Hkv, Dh, _dtype_code(Q), float(scale),
                                     _ptr(ws), _stream(stream)), "mw_masked_attn_fwd")


def masked_attn_fwd(vis, Q, K, V, scale=None, ws=None, stream=None):
    """Allocate O [T, Hq, Dh] and LSE [Hq, T] (and the workspace) and run the
    forward."""
    import torch
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _need(t, n, dtype=Q.dtype)
    scale = float(Q.shape[2]) ** -0.5 if scale is None else scale
    if ws is None:
        nbytes = mw_masked_attn_fwd_ws(vis, K.shape[1], Q.shape[2], _dtype_code(Q))
        ws = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=Q.device)
    O = torch.empty_like(Q)
    LSE = torch.empty(Q.shape[1], Q.shape[0], dtype=torch.float32, device=Q.device)
    mw_masked_attn_fwd(vis, Q, K, V, O, LSE, scale, ws, stream)
    return O, LSE


def mw_masked_attn_bwd_ws(vis, Hq, Hkv, Dh, dtype):
    n = ctypes.c_size_t()
    _check(_lib().mw_masked_attn_bwd_ws(ctypes.byref(vis.layout), Hq, Hkv, Dh, dtype, ctypes.byref(n)),
           "mw_masked_attn_bwd_ws")
    return int(n.value)


def mw_masked_attn_bwd(vis, Q, K, V, O, dO, LSE, dQ, dK, dV, scale, ws, stream=None):
    Hq, Dh = Q.shape[1], Q.shape[2]
    Hkv = K.shape[1]
    _check(_lib().mw_masked_attn_bwd(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(Q), _ptr(K), _ptr(V), _ptr(O),
                                     _ptr(dO), _ptr(LSE), _ptr(dQ), _ptr(dK), _ptr(dV), Hq, Hkv, Dh,
                                     _dtype_code(Q), float(scale), _ptr(ws), _stream(stream)),
           "mw_masked_attn_bwd")


def masked_attn_bwd(vis, Q, K, V, O, dO, LSE, scale=None, ws=None, stream=None):
    """Allocate dQ, dK, dV (and the workspace) and run the backward."""
    import torch
    for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O"), (dO, "dO")):
        _need(t, n, dtype=Q.dtype)
    _need(LSE, "LSE", dtype=torch.float32)
    scale = float(Q.shape[2]) ** -0.5 if scale is None else scale
    if ws is None:
        nbytes = mw_masked_attn_bwd_ws(vis, Q.shape[1], K.shape[1], Q.shape[2], _dtype_code(Q))
        ws = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=Q.device)
    dQ, dK, dV = torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V)
    mw_masked_attn_bwd(vis, Q, K, V, O, dO, LSE, dQ, dK, dV, scale, ws, stream)
    return dQ, dK, dV


# --- row-wise logical positions and rotary attention ---------------------------

def diverging_rows(vis, stream=None):
    """uint8 [total_tokens]: 1 on the rows SDCC's KL term applies to
    (mw_diverging_rows)."""
    import torch
    out = torch.empty(max(int(vis.layout.total_tokens), 1), dtype=torch.uint8, device=vis.vis.device)
    _check(_lib().mw_diverging_rows(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(out), _stream(stream)),
           "mw_diverging_rows")
    return out


def final_walk(vis, stream=None):
    """(walk_index [T], student_row [T], walk_len [n_traj]) int32 device
    tensors of the final compressed walk (mw_final_walk).

    ``student_row`` is given for every row; an SDCC caller keeps loss row r
    only where ``walk_index[r + 1] >= 0`` (leaf y_(r+1) survives on the walk,
    inside the same trajectory), since an evicted token has no student score."""
    import torch
    L = vis.layout
    dev = vis.vis.device
    wi = torch.empty(max(int(L.total_tokens), 1), dtype=torch.int32, device=dev)
    sr = torch.empty_like(wi)
    wl = torch.empty(max(int(L.n_traj), 1), dtype=torch.int32, device=dev)
    _check(_lib().mw_final_walk(ctypes.byref(L), _ptr(vis.vis), _ptr(wi), _ptr(sr), _ptr(wl), _stream(stream)),
           "mw_final_walk")
    return wi, sr, wl


def logdiff(lp_train, lp_rollout, stream=None):
    """Eq. "logdiff": mean |lp_train - lp_rollout| as a one-element float32
    device tensor (mw_logdiff)."""
    import torch
    _need(lp_train, "lp_train", dtype=torch.float32)
    _need(lp_rollout, "lp_rollout", dtype=torch.float32)
    out = torch.empty(1, dtype=torch.float32, device=lp_train.device)
    _check(_lib().mw_logdiff(_ptr(lp_train), _ptr(lp_rollout), int(lp_train.numel()), _ptr(out), _stream(stream)),
           "mw_logdiff")
    return out


def mw_forward_kl_ws(M, d, Vocab, dtype):
    n = ctypes.c_size_t()
    _check(_lib().mw_forward_kl_ws(int(M), int(d), int(Vocab), int(dtype), ctypes.byref(n)), "mw_forward_kl_ws")
    return int(n.value)


def mw_forward_kl_fwd(HT, rows_T, HS, rows_S, W, kl, loss, ws, lam=1.0, stream=None):
    M, d, V = int(rows_T.numel()), HT.shape[1], W.shape[0]
    _check(_lib().mw_forward_kl_fwd(_ptr(HT), _ptr(rows_T), _ptr(HS), _ptr(rows_S), M, _ptr(W), HT.shape[0],
                                    HS.shape[0], d, V, _dtype_code(HT), float(lam), _ptr(kl), _ptr(loss), _ptr(ws),
                                    _stream(stream)), "mw_forward_kl_fwd")


def forward_kl_fwd(HT, rows_T, HS, rows_S, W, lam=1.0, stream=None):
    """SDCC consistency term: kl [M], loss (lam * sum kl) and the workspace
    the backward needs (mw_forward_kl_fwd)."""
    import torch
    _need(HT, "HT")
    _need(HS, "HS", dtype=HT.dtype)
    _need(W, "W", dtype=HT.dtype)
    M, d, V = int(rows_T.numel()), HT.shape[1], W.shape[0]
    ws = torch.empty(max(mw_forward_kl_ws(M, d, V, _dtype_code(HT)), 1), dtype=torch.uint8, device=HT.device)
    kl = torch.empty(max(M, 1), dtype=torch.float32, device=HT.device)
    loss = torch.empty(1, dtype=torch.float32, device=HT.device)
    mw_forward_kl_fwd(HT, rows_T, HS, rows_S, W, kl, loss, ws, lam, stream)
    return kl[:M], loss, ws


def forward_kl_check_status(rows_T, HT, W, ws, stream=None):
    """Synchronise and raise MWError if a bounded device wait of the
    tensor-core KL passes gave up (MW_ETIMEOUT) or a pair's row index was out
    of range (MW_EDEVICE) (mw_forward_kl_check_status)."""
    _check(_lib().mw_forward_kl_check_status(int(rows_T.numel()), HT.shape[1], W.shape[0], _dtype_code(HT),
                                             _ptr(ws), _stream(stream)), "mw_forward_kl_check_status")


def mw_forward_kl_bwd(HT, rows_T, HS, rows_S, W, ws, dHS, dW, lam=1.0, dloss=1.0, accumulate=False, stream=None):
    M, d, V = int(rows_T.numel()), HT.shape[1], W.shape[0]
    _check(_lib().mw_forward_kl_bwd(_ptr(HT), _ptr(rows_T), _ptr(HS), _ptr(rows_S), M, _ptr(W), HT.shape[0],
                                    HS.shape[0], d, V, _dtype_code(HT), float(lam), float(dloss), int(accumulate),
                                    _ptr(ws), _ptr(dHS), _ptr(dW), _stream(stream)), "mw_forward_kl_bwd")


def forward_kl_bwd(HT, rows_T, HS, rows_S, W, ws, lam=1.0, dloss=1.0, stream=None):
    """Student gradients of the SDCC term: dHS (like HS), dW (float32)."""
    import torch
    d, V = HT.shape[1], W.shape[0]
    dHS = torch.empty_like(HS)
    dW = torch.empty(V, d, dtype=torch.float32, device=HT.device)
    mw_forward_kl_bwd(HT, rows_T, HS, rows_S, W, ws, dHS, dW, lam, dloss, False, stream)
    return dHS, dW


def mw_logical_positions(vis, pos, stream=None):
    _check(_lib().mw_logical_positions(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(pos), _stream(stream)),
           "mw_logical_positions")


def logical_positions(vis, stream=None):
    """int32 [n_keymask * 128]: rank of key j in segment s's live view at
    (traj_km[b] + s nt_b) 128 + j, -1 for non-members (mw_logical_positions)."""
    import torch
    L = vis.layout
    pos = torch.empty(max(int(L.n_keymask) * TILE, 1), dtype=torch.int32, device=vis.vis.device)
    mw_logical_positions(vis, pos, stream)
    return pos


def rope_table(n_pos, Dh, theta, device="cuda", stream=None):
    """float32 [n_pos, Dh/2, 2] (cos, sin) table (mw_rope_table)."""
    import torch
    t = torch.empty(max(int(n_pos), 1), Dh // 2, 2, dtype=torch.float32, device=device)
    _check(_lib().mw_rope_table(int(n_pos), int(Dh), float(theta), _ptr(t), _stream(stream)), "mw_rope_table")
    return t


def rope_n_pos(vis):
    """Smallest table length the rotary entry points accept for this record."""
    return TILE * int(vis.layout.max_tiles)


def rope_rows(vis, pos, table, X, inverse=False, out=None, stream=None):
    """Rotate every row of X [T, H, Dh] by its own logical position."""
    import torch
    _need(X, "X")
    Y = torch.empty_like(X) if out is None else out
    _check(_lib().mw_rope_rows(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(pos), _ptr(table), table.shape[0],
                               _ptr(X), _ptr(Y), X.shape[1], X.shape[2], _dtype_code(X), int(bool(inverse)),
                               _stream(stream)), "mw_rope_rows")
    return Y


def mw_masked_attn_rope_ws(vis, Hq, Hkv, Dh, dtype):
    f, b = ctypes.c_size_t(), ctypes.c_size_t()
    _check(_lib().mw_masked_attn_rope_ws(ctypes.byref(vis.layout), Hq, Hkv, Dh, dtype, ctypes.byref(f),
                                         ctypes.byref(b)), "mw_masked_attn_rope_ws")
    return int(f.value), int(b.value)


def mw_masked_attn_rope_fwd(vis, pos, table, Q, K, V, O, LSE, scale, ws, stream=None):
    Hq, Dh, Hkv = Q.shape[1], Q.shape[2], K.shape[1]
    _check(_lib().mw_masked_attn_rope_fwd(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(pos), _ptr(table),
                                          table.shape[0], _ptr(Q), _ptr(K), _ptr(V), _ptr(O), _ptr(LSE), Hq, Hkv,
                                          Dh, _dtype_code(Q), float(scale), _ptr(ws), _stream(stream)),
           "mw_masked_attn_rope_fwd")


def mw_masked_attn_rope_bwd(vis, pos, table, Q, K, V, O, dO, LSE, dQ, dK, dV, scale, ws, stream=None):
    Hq, Dh, Hkv = Q.shape[1], Q.shape[2], K.shape[1]
    _check(_lib().mw_masked_attn_rope_bwd(ctypes.byref(vis.layout), _ptr(vis.vis), _ptr(pos), _ptr(table),
                                          table.shape[0], _ptr(Q), _ptr(K), _ptr(V), _ptr(O), _ptr(dO), _ptr(LSE),
                                          _ptr(dQ), _ptr(dK), _ptr(dV), Hq, Hkv, Dh, _dtype_code(Q), float(scale),
                                          _ptr(ws), _stream(stream)), "mw_masked_attn_rope_bwd")


def masked_attn_rope_fwd(vis, pos, table, Q, K, V, scale=None, ws=None, stream=None):
    """Masked attention with per-row logical rotary positions; returns O, LSE."""
    import torch
    for t, n in ((Q, "Q"), (K, "K"), (V, "V")):
        _need(t, n, dtype=Q.dtype)
    Hq, Dh, Hkv = Q.shape[1], Q.shape[2], K.shape[1]
    scale = float(Dh) ** -0.5 if scale is None else scale
    if ws is None:
        nbytes = mw_masked_attn_rope_ws(vis, Hq, Hkv, Dh, _dtype_code(Q))[0]
        ws = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=Q.device)
    O = torch.empty_like(Q)
    LSE = torch.empty(Hq, Q.shape[0], dtype=torch.float32, device=Q.device)
    mw_masked_attn_rope_fwd(vis, pos, table, Q, K, V, O, LSE, scale, ws, stream)
    return O, LSE


def masked_attn_rope_bwd(vis, pos, table, Q, K, V, O, dO, LSE, scale=None, ws=None, stream=None):
    """Backward of masked_attn_rope_fwd; returns dQ, dK, dV."""
    import torch
    for t, n in ((Q, "Q"), (K, "K"), (V, "V"), (O, "O"), (dO, "dO")):
        _need(t, n, dtype=Q.dtype)
    _need(LSE, "LSE", dtype=torch.float32)
    Hq, Dh, Hkv = Q.shape[1], Q.shape[2], K.shape[1]
    scale = float(Dh) ** -0.5 if scale is None else scale
    if ws is None:
        nbytes = mw_masked_attn_rope_ws(vis, Hq, Hkv, Dh, _dtype_code(Q))[1]
        ws = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=Q.device)
    dQ, dK, dV = torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V)
    mw_masked_attn_rope_bwd(vis, pos, table, Q, K, V, O, dO, LSE, dQ, dK, dV, scale, ws, stream)
    return dQ, dK, dV


# --- LM head ------------------------------------------------------------------

def mw_logprob_ws(N, M, d, Vocab, dtype):
    n = ctypes.c_size_t()
    _check(_lib().mw_logprob_ws(N, M, d, Vocab, dtype, ctypes.byref(n)), "mw_logprob_ws")
    return int(n.value)


def mw_logprob_loss_fwd(H, W, targets, rows, lp_old, adv, eps_lo, eps_hi, lp, ratio, lse, loss, ws, stream=None):
    N, d = H.shape
    _check(_lib().mw_logprob_loss_fwd(_ptr(H), _ptr(W), _ptr(targets), _ptr(rows), int(rows.numel()),
                                      _ptr(lp_old), _ptr(adv), float(eps_lo), float(eps_hi), N, d, W.shape[0],
                                      _dtype_code(H), _ptr(lp), _ptr(ratio), _ptr(lse), _ptr(loss), _ptr(ws),
                                      _stream(stream)), "mw_logprob_loss_fwd")


def mw_logprob_loss_fwd_kl(H, W, targets, rows, lp_old, adv, eps_lo, eps_hi, lp_ref, beta, lp, ratio, lse, loss,
                           ws, stream=None):
    N, d = H.shape
    _check(_lib().mw_logprob_loss_fwd_kl(_ptr(H), _ptr(W), _ptr(targets), _ptr(rows), int(rows.numel()),
                                         _ptr(lp_old), _ptr(adv), float(eps_lo), float(eps_hi), _ptr(lp_ref),
                                         float(beta), N, d, W.shape[0], _dtype_code(H), _ptr(lp), _ptr(ratio),
                                         _ptr(lse), _ptr(loss), _ptr(ws), _stream(stream)), "mw_logprob_loss_fwd_kl")


def logprob_loss_fwd(H, W, targets, rows, lp_old, adv, eps_lo=0.2, eps_hi=0.28, stream=None, lp_ref=None, beta=0.0):
    """Allocate outputs + workspace; returns dict(lp, ratio, lse, loss, ws).
    With ``lp_ref`` (float32 [M]) and ``beta`` > 0 the loss includes the KL
    term of ``mw_logprob_loss_fwd_kl``."""
    import torch
    _need(H, "H")
    _need(W, "W", dtype=H.dtype)
    _need(targets, "targets", dtype=torch.int32)
    _need(rows, "rows", dtype=torch.int32)
    _need(lp_old, "lp_old", dtype=torch.float32)
    _need(adv, "adv", dtype=torch.float32)
    M = rows.numel()
    dev = H.device
    ws = torch.empty(max(mw_logprob_ws(H.shape[0], M, H.shape[1], W.shape[0], _dtype_code(H)), 1),
                     dtype=torch.uint8, device=dev)
    out = {k: torch.empty(M, dtype=torch.float32, device=dev) for k in ("lp", "ratio", "lse")}
    out["loss"] = torch.empty(1, dtype=torch.float32, device=dev)
    if lp_ref is not None or beta != 0.0:
        if lp_ref is not None:
            _need(lp_ref, "lp_ref", dtype=torch.float32)
        mw_logprob_loss_fwd_kl(H, W, targets, rows, lp_old, adv, eps_lo, eps_hi, lp_ref, beta, out["lp"],
                               out["ratio"], out["lse"], out["loss"], ws, stream)
    else:
        mw_logprob_loss_fwd(H, W, targets, rows, lp_old, adv, eps_lo, eps_hi, out["lp"], out["ratio"], out["lse"],
                            out["loss"], ws, stream)
    out["ws"] = ws
    return out


def mw_logprob_loss_bwd(H, W, targets, rows, lse, ws, dloss, dH, dW, stream=None):
    N, d = H.shape
    _check(_lib().mw_logprob_loss_bwd(_ptr(H), _ptr(W), _ptr(targets), _ptr(rows), int(rows.numel()), N, d,
                                      W.shape[0], _dtype_code(H), _ptr(lse), _ptr(ws), float(dloss), _ptr(dH),
                                      _ptr(dW), _stream(stream)), "mw_logprob_loss_bwd")


def mw_logprob_check_status(H, W, rows, ws, stream=None):
    """Raise MWError if an LM-head kernel that last ran on ``ws`` gave up a
    bounded wait (MW_ETIMEOUT) or met a loss row or target out of range
    (MW_EDEVICE); synchronises the stream."""
    N, d = H.shape
    _check(_lib().mw_logprob_check_status(N, int(rows.numel()), d, W.shape[0], _dtype_code(H), _ptr(ws),
                                          _stream(stream)), "mw_logprob_check_status")


def mw_selftest_wait_timeout(limit_ns, status, stream=None):
    """Run the bounded-wait self-test; returns the raw status code
    (MW_ETIMEOUT = 6 is the expected outcome). ``status``: device int32[8]."""
    return int(_lib().mw_selftest_wait_timeout(int(limit_ns), _ptr(status), _stream(stream)))


def logprob_loss_bwd(H, W, targets, rows, lse, ws, dloss=1.0, stream=None):
    """Allocate dH (H's dtype) and dW (float32) and run the backward."""
    import torch
    dH = torch.empty_like(H)
    dW = torch.empty(W.shape, dtype=torch.float32, device=W.device)
    mw_logprob_loss_bwd(H, W, targets, rows, lse, ws, dloss, dH, dW, stream)
    return dH, dW
