"""Oracle: per-segment compact attention, forward and backward, in float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

This is the LogitTree formulation (§4.1; App. E.2 "The five methods"): split
the rollout at its junctions, materialise each segment's live view as its own
compact sequence, and run ordinary causal softmax attention on it alone. The
segment's rows are the tail of that compact sequence, so each row attends to
the compact prefix up to and including itself. Theorem "materialization
equivalence" (§4.3, proof in App. C.3) states that the packed 4D-masked
computation gives the same outputs and gradients; the CUDA path is checked
against this file.

Layouts (token-major, trajectories packed back to back):
``Q, O``: ``[T_total, Hq, Dh]``; ``K, V``: ``[T_total, Hkv, Dh]``;
``LSE``: ``[Hq, T_total]`` (natural log). Query head ``h`` reads KV head
``h // (Hq // Hkv)`` (contiguous GQA groups).

Rotary positions (optional, ``rope_theta``): §4.2 gives every row position
ids under which its visible keys form a gap-free sequence. On the compact
sequence of a segment that is simply the compact index, so queries and keys
are rotated by their index in ``view_s`` before the scores are taken, and the
gradients are rotated back.

Arithmetic: float64 CPU tensors (torch), so that the library's matrix
products and element-wise passes use every host core; inputs and outputs are
numpy arrays. Each formula below is the textbook one, evaluated as written.
"""

import numpy as np
import torch

from .visibility import live_views

_ROW_CHUNK = 512


def _t(x):
    """float64 CPU tensor view of an array (copies only when it must)."""
    return torch.from_numpy(np.ascontiguousarray(np.asarray(x, dtype=np.float64)))


def _ix(x):
    return torch.from_numpy(np.asarray(x, dtype=np.int64))


def _segments(seqlens, edits_per_traj, views=None):
    """Yield ``(global_rows, global_view_positions, n_before)`` per segment.

    ``views`` maps ``(T, edits)`` to the ``[(row_lo, row_hi, view)]`` lists of
    each segment (default: ``visibility.live_views``; ``nonmonotone.live_views``
    for records whose events also bring spans back). The compact sequence is
    the view list in its own order."""
    views = live_views if views is None else views
    base = 0
    for T, edits in zip(seqlens, edits_per_traj):
        for lo, hi, view in views(T, edits):
            idx = np.asarray(view, dtype=np.int64) + base
            yield np.arange(lo, hi, dtype=np.int64) + base, idx, len(view) - (hi - lo)
        base += T


def _rope_t(x, pos, theta, inverse=False):
    """Rotary position embedding (RoFormer, Su et al. 2021) in the
    rotate-half pairing on a float64 tensor: feature f (f < Dh/2) is paired
    with f + Dh/2 and the pair is turned by the angle
    ``pos * theta ** (-2 f / Dh)``. ``x`` is ``[n, ..., Dh]`` with one
    position per leading index; ``inverse`` turns by the opposite angle (the
    transpose of the rotation)."""
    half = x.shape[-1] // 2
    w = float(theta) ** (-2.0 * torch.arange(half, dtype=torch.float64) / x.shape[-1])
    ang = torch.as_tensor(np.asarray(pos, dtype=np.float64))[:, None] * w[None, :]
    if inverse:
        ang = -ang
    ang = ang.reshape((ang.shape[0],) + (1,) * (x.ndim - 2) + (half,))
    c, s = torch.cos(ang), torch.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return torch.cat([a * c - b * s, b * c + a * s], dim=-1)


def rope(x, pos, theta, inverse=False):
    """``_rope_t`` on numpy arrays (float64 in, float64 out)."""
    return _rope_t(_t(x), pos, theta, inverse).numpy()


def _probs(q, k, scale, compact_rows):
    """Row softmax of the scaled scores of compact rows against the compact
    keys, causal: ``compact_rows[r]`` is the compact index of row r of ``q``,
    which sees compact keys ``0 .. compact_rows[r]`` and nothing after.
    Masked entries are excluded exactly (their exponential is 0). Returns
    ``(P, row max, row sum)``."""
    s = (q @ k.T) * scale
    c = torch.arange(k.shape[0])[None, :]
    s.masked_fill_(c > _ix(compact_rows)[:, None], float("-inf"))
    m = s.amax(dim=1, keepdim=True)
    p = torch.exp(s - m)
    l = p.sum(dim=1, keepdim=True)
    return p, m, l


def attn_fwd(seqlens, edits_per_traj, Q, K, V, scale, rows=None, heads=None, rope_theta=None, views=None):
    """Masked GQA attention forward via per-segment compact sequences.

    Returns ``(O_sel, LSE_sel)`` for the selected global rows (default: all)
    and query heads (default: all): ``O_sel[r, h_i, :]``, ``LSE_sel[h_i, r]``.
    Softmax over each row's visible keys exactly (no large-negative fill).
    With ``rope_theta`` queries and keys are rotated by their compact index.
    """
    Q, K, V = _t(Q), _t(K), _t(V)
    Ttot, Hq, Dh = Q.shape
    Hkv = K.shape[1]
    grp = Hq // Hkv
    heads = list(range(Hq)) if heads is None else list(heads)
    rows = np.arange(Ttot) if rows is None else np.asarray(rows, dtype=np.int64)
    pos_of = np.full(Ttot, -1, dtype=np.int64)
    pos_of[rows] = np.arange(rows.size)
    O = torch.full((len(rows), len(heads), Dh), float("nan"), dtype=torch.float64)
    L = torch.full((len(heads), len(rows)), float("nan"), dtype=torch.float64)
    want = np.zeros(Ttot, dtype=bool)
    want[rows] = True
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj, views):
        sel = np.nonzero(want[seg_rows])[0]
        if sel.size == 0:
            continue
        ti = _ix(idx)
        for g in sorted({h // grp for h in heads}):
            # the segment's compact key / value sequence of KV head g
            k = K[ti, g]
            v = V[ti, g]
            if rope_theta is not None:
                k = _rope_t(k, np.arange(idx.size), rope_theta)
            for c0 in range(0, sel.size, _ROW_CHUNK):
                part = sel[c0 : c0 + _ROW_CHUNK]
                # compact index of each selected row = n_before + local offset
                grows = _ix(seg_rows[part])
                out_pos = _ix(pos_of[seg_rows[part]])
                for hi, h in enumerate(heads):
                    if h // grp != g:
                        continue
                    q = Q[grows, h]
                    if rope_theta is not None:
                        q = _rope_t(q, n_before + part, rope_theta)
                    p, m, l = _probs(q, k, scale, n_before + part)
                    O[out_pos, hi] = (p @ v) / l
                    L[hi, out_pos] = (m + torch.log(l))[:, 0]
    return O.numpy(), L.numpy()


def attn_bwd(seqlens, edits_per_traj, Q, K, V, dO, scale, groups=None, rope_theta=None, views=None):
    """Textbook softmax-attention backward on every segment's compact sequence.

    For one segment and head (compact rows r, compact keys c):
    ``P = softmax(S)``, ``dP = dO V^T``, ``dS = P * (dP - rowsum(P * dP))``,
    ``dQ = scale dS K``, ``dK += scale dS^T Q``, ``dV += P^T dO``; dK and dV
    are scatter-added to the physical key rows across every segment and every
    query head of the KV group.

    ``groups`` restricts the computation to some KV groups (all their query
    heads); returns full-size ``(dQ, dK, dV)`` with NaN outside the selection.
    With ``rope_theta`` the scores use rotated q and k (compact index) and
    dQ, dK are the rotated-space gradients turned back by the same angles.
    """
    Q, K, V, dO = _t(Q), _t(K), _t(V), _t(dO)
    Ttot, Hq, Dh = Q.shape
    Hkv = K.shape[1]
    grp = Hq // Hkv
    groups = list(range(Hkv)) if groups is None else list(groups)
    dQ = torch.full_like(Q, float("nan"))
    dK = torch.full_like(K, float("nan"))
    dV = torch.full_like(V, float("nan"))
    for g in groups:
        dQ[:, g * grp : (g + 1) * grp] = 0.0
        dK[:, g] = 0.0
        dV[:, g] = 0.0
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj, views):
        ti = _ix(idx)
        for g in groups:
            k = K[ti, g]
            v = V[ti, g]
            if rope_theta is not None:
                k = _rope_t(k, np.arange(idx.size), rope_theta)
            dk = torch.zeros_like(k)
            dv = torch.zeros_like(v)
            for c0 in range(0, seg_rows.size, _ROW_CHUNK):
                grows = _ix(seg_rows[c0 : c0 + _ROW_CHUNK])
                crow = n_before + c0 + np.arange(grows.numel())
                for h in range(g * grp, (g + 1) * grp):
                    q = Q[grows, h]
                    if rope_theta is not None:
                        q = _rope_t(q, crow, rope_theta)
                    do = dO[grows, h]
                    p, _, l = _probs(q, k, scale, crow)
                    p = p / l
                    dp = do @ v.T
                    ds = p * (dp - (p * dp).sum(dim=1, keepdim=True))
                    dq = scale * (ds @ k)
                    if rope_theta is not None:
                        dq = _rope_t(dq, crow, rope_theta, inverse=True)
                    dQ[grows, h] = dq
                    dk += scale * (ds.T @ q)
                    dv += p.T @ do
            if rope_theta is not None:
                dk = _rope_t(dk, np.arange(idx.size), rope_theta, inverse=True)
            dK[:, g].index_add_(0, ti, dk)
            dV[:, g].index_add_(0, ti, dv)
    return dQ.numpy(), dK.numpy(), dV.numpy()


def attn_bwd_rows(seqlens, edits_per_traj, Q, K, V, dO, scale, rows, heads, rope_theta=None, with_kv=False, views=None):
    """dQ of a few physical rows and query heads (same formulas as
    ``attn_bwd``, rotary positions included; a row's dQ needs only its own
    segment's compact view and its own dO row). Returns ``dQ_sel[r, h_i, :]``.

    With ``with_kv`` also returns those rows' contributions to dK and dV
    (``scale dS^T q`` and ``P^T dO`` of the selected rows and heads,
    scatter-added to the physical key rows, float64 ``[T_total, Hkv, Dh]``):
    summed over every row and head they are ``attn_bwd``'s dK and dV."""
    Q, K, V, dO = _t(Q), _t(K), _t(V), _t(dO)
    Hq = Q.shape[1]
    grp = Hq // K.shape[1]
    rows = np.asarray(rows, dtype=np.int64)
    pos_of = np.full(Q.shape[0], -1, dtype=np.int64)
    pos_of[rows] = np.arange(rows.size)
    out = torch.full((rows.size, len(heads), Q.shape[2]), float("nan"), dtype=torch.float64)
    dK = torch.zeros_like(K) if with_kv else None
    dV = torch.zeros_like(V) if with_kv else None
    want = np.zeros(Q.shape[0], dtype=bool)
    want[rows] = True
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj, views):
        part = np.nonzero(want[seg_rows])[0]
        if part.size == 0:
            continue
        ti = _ix(idx)
        grows = _ix(seg_rows[part])
        outp = _ix(pos_of[seg_rows[part]])
        kv = {}
        for hi, h in enumerate(heads):
            if h // grp not in kv:
                k = K[ti, h // grp]
                if rope_theta is not None:
                    k = _rope_t(k, np.arange(idx.size), rope_theta)
                kv = {h // grp: (k, V[ti, h // grp])}
            k, v = kv[h // grp]
            q = Q[grows, h]
            if rope_theta is not None:
                q = _rope_t(q, n_before + part, rope_theta)
            p, _, l = _probs(q, k, scale, n_before + part)
            p = p / l
            dp = dO[grows, h] @ v.T
            ds = p * (dp - (p * dp).sum(dim=1, keepdim=True))
            dq = scale * (ds @ k)
            if rope_theta is not None:
                dq = _rope_t(dq, n_before + part, rope_theta, inverse=True)
            out[outp, hi] = dq
            if with_kv:
                q = Q[grows, h] if rope_theta is None else _rope_t(Q[grows, h], n_before + part, rope_theta)
                dk = scale * (ds.T @ q)
                if rope_theta is not None:
                    dk = _rope_t(dk, np.arange(idx.size), rope_theta, inverse=True)
                dK[:, h // grp].index_add_(0, ti, dk)
                dV[:, h // grp].index_add_(0, ti, p.T @ dO[grows, h])
    if with_kv:
        return out.numpy(), dK.numpy(), dV.numpy()
    return out.numpy()


def attn_bwd_keys(seqlens, edits_per_traj, Q, K, V, dO, scale, g, keys, rope_theta=None, views=None):
    """dK, dV of KV group ``g`` for a few physical key rows only.

    Same textbook formulas as ``attn_bwd`` (rotary positions included: a key's
    contribution from a segment is turned back by its angle in that segment);
    only the columns of the selected keys of each segment's ``dS`` and ``P``
    are accumulated, but every row's softmax is still normalised over its full
    live view. A row before a key never sees it (the compact sequence is
    causal), so each segment's rows are taken from the first one at or after
    its earliest selected key. Used for sampled checks on workloads too large
    for the full backward.
    """
    Q, K, V, dO = _t(Q), _t(K), _t(V), _t(dO)
    Hq = Q.shape[1]
    grp = Hq // K.shape[1]
    keys = np.asarray(keys, dtype=np.int64)
    dk_out = torch.zeros((keys.size, K.shape[2]), dtype=torch.float64)
    dv_out = torch.zeros((keys.size, K.shape[2]), dtype=torch.float64)
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj, views):
        where = {int(p): c for c, p in enumerate(idx)}
        cols = [(n, where[int(kk)]) for n, kk in enumerate(keys) if int(kk) in where]
        if not cols:
            continue
        kn = _ix([a for a, _ in cols])
        kc_np = np.asarray([b for _, b in cols])
        kc = _ix(kc_np)
        ti = _ix(idx)
        k = K[ti, g]
        v = V[ti, g]
        if rope_theta is not None:
            k = _rope_t(k, np.arange(idx.size), rope_theta)
        # compact row c sees compact key c' only if c' <= c
        first = max(0, int(kc_np.min()) - n_before)
        for c0 in range(first, seg_rows.size, _ROW_CHUNK):
            grows = _ix(seg_rows[c0 : c0 + _ROW_CHUNK])
            crow = n_before + c0 + np.arange(grows.numel())
            for h in range(g * grp, (g + 1) * grp):
                q = Q[grows, h]
                if rope_theta is not None:
                    q = _rope_t(q, crow, rope_theta)
                do = dO[grows, h]
                p, _, l = _probs(q, k, scale, crow)
                p = p / l
                dp = do @ v.T
                ds = p * (dp - (p * dp).sum(dim=1, keepdim=True))
                dk = scale * (ds[:, kc].T @ q)
                if rope_theta is not None:
                    dk = _rope_t(dk, kc_np, rope_theta, inverse=True)
                dk_out.index_add_(0, kn, dk)
                dv_out.index_add_(0, kn, p[:, kc].T @ do)
    return dk_out.numpy(), dv_out.numpy()
