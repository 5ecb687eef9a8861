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
"""

import numpy as np

from .visibility import live_views

_ROW_CHUNK = 512


def _segments(seqlens, edits_per_traj):
    """Yield ``(global_rows, global_view_positions, n_before)`` per segment."""
    base = 0
    for T, edits in zip(seqlens, edits_per_traj):
        for lo, hi, view in live_views(T, edits):
            idx = np.asarray(view, dtype=np.int64) + base
            yield np.arange(lo, hi, dtype=np.int64) + base, idx, len(view) - (hi - lo)
        base += T


def rope(x, pos, theta, inverse=False):
    """Rotary position embedding (RoFormer, Su et al. 2021) in the
    rotate-half pairing: feature f (f < Dh/2) is paired with f + Dh/2 and the
    pair is turned by the angle ``pos * theta ** (-2 f / Dh)``. ``x`` is
    ``[n, ..., Dh]`` with one position per leading index; ``inverse`` turns by
    the opposite angle (the transpose of the rotation).
    """
    x = np.asarray(x, dtype=np.float64)
    half = x.shape[-1] // 2
    w = float(theta) ** (-2.0 * np.arange(half, dtype=np.float64) / x.shape[-1])
    ang = np.asarray(pos, dtype=np.float64)[:, None] * w[None, :]
    if inverse:
        ang = -ang
    ang = ang.reshape((ang.shape[0],) + (1,) * (x.ndim - 2) + (half,))
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def _scores(q, k, scale, compact_rows):
    """Scaled scores of compact rows against the compact keys, causal.

    ``compact_rows[r]`` is the compact index of row r of ``q``; that row may
    see compact keys ``0 .. compact_rows[r]`` and nothing after.
    """
    s = (q @ k.T) * scale
    c = np.arange(k.shape[0])[None, :]
    s[c > np.asarray(compact_rows)[:, None]] = -np.inf
    return s


def attn_fwd(seqlens, edits_per_traj, Q, K, V, scale, rows=None, heads=None, rope_theta=None):
    """Masked GQA attention forward via per-segment compact sequences.

    Returns ``(O_sel, LSE_sel)`` for the selected global rows (default: all)
    and query heads (default: all): ``O_sel[r, h_i, :]``, ``LSE_sel[h_i, r]``.
    Softmax over each row's visible keys exactly (no large-negative fill).
    With ``rope_theta`` queries and keys are rotated by their compact index.
    """
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Ttot, Hq, Dh = Q.shape
    Hkv = K.shape[1]
    grp = Hq // Hkv
    heads = list(range(Hq)) if heads is None else list(heads)
    rows = np.arange(Ttot) if rows is None else np.asarray(rows, dtype=np.int64)
    pos_of = {int(r): n for n, r in enumerate(rows)}
    O = np.full((len(rows), len(heads), Dh), np.nan)
    L = np.full((len(heads), len(rows)), np.nan)
    want = np.zeros(Ttot, dtype=bool)
    want[rows] = True
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj):
        sel = np.nonzero(want[seg_rows])[0]
        if sel.size == 0:
            continue
        for c0 in range(0, sel.size, _ROW_CHUNK):
            part = sel[c0 : c0 + _ROW_CHUNK]
            # compact index of each selected row = n_before + local offset
            grows = seg_rows[part]
            out_pos = [pos_of[int(r)] for r in grows]
            for hi, h in enumerate(heads):
                g = h // grp
                k = K[idx, g]
                v = V[idx, g]
                q = Q[grows, h]
                if rope_theta is not None:
                    k = rope(k, np.arange(idx.size), rope_theta)
                    q = rope(q, n_before + part, rope_theta)
                s = _scores(q, k, scale, n_before + part)
                m = s.max(axis=1, keepdims=True)
                p = np.exp(s - m)
                l = p.sum(axis=1, keepdims=True)
                O[out_pos, hi] = (p @ v) / l
                L[hi, out_pos] = (m + np.log(l))[:, 0]
    return O, L


def attn_bwd(seqlens, edits_per_traj, Q, K, V, dO, scale, groups=None, rope_theta=None):
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
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    dO = np.asarray(dO, dtype=np.float64)
    Ttot, Hq, Dh = Q.shape
    Hkv = K.shape[1]
    grp = Hq // Hkv
    groups = list(range(Hkv)) if groups is None else list(groups)
    dQ = np.full_like(Q, np.nan)
    dK = np.full_like(K, np.nan)
    dV = np.full_like(V, np.nan)
    for g in groups:
        dQ[:, g * grp : (g + 1) * grp] = 0.0
        dK[:, g] = 0.0
        dV[:, g] = 0.0
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj):
        for c0 in range(0, seg_rows.size, _ROW_CHUNK):
            grows = seg_rows[c0 : c0 + _ROW_CHUNK]
            crow = n_before + c0 + np.arange(grows.size)
            for g in groups:
                k = K[idx, g]
                v = V[idx, g]
                if rope_theta is not None:
                    k = rope(k, np.arange(idx.size), rope_theta)
                dk = np.zeros_like(k)
                dv = np.zeros_like(v)
                for h in range(g * grp, (g + 1) * grp):
                    q = Q[grows, h]
                    if rope_theta is not None:
                        q = rope(q, crow, rope_theta)
                    do = dO[grows, h]
                    s = _scores(q, k, scale, crow)
                    m = s.max(axis=1, keepdims=True)
                    p = np.exp(s - m)
                    p /= p.sum(axis=1, keepdims=True)
                    dp = do @ v.T
                    ds = p * (dp - (p * dp).sum(axis=1, keepdims=True))
                    dq = scale * (ds @ k)
                    if rope_theta is not None:
                        dq = rope(dq, crow, rope_theta, inverse=True)
                    dQ[grows, h] = dq
                    dk += scale * (ds.T @ q)
                    dv += p.T @ do
                if rope_theta is not None:
                    dk = rope(dk, np.arange(idx.size), rope_theta, inverse=True)
                np.add.at(dK[:, g], idx, dk)
                np.add.at(dV[:, g], idx, dv)
    return dQ, dK, dV


def attn_bwd_rows(seqlens, edits_per_traj, Q, K, V, dO, scale, rows, heads, rope_theta=None):
    """dQ of a few physical rows and query heads (same formulas as
    ``attn_bwd``, rotary positions included; a row's dQ needs only its own
    segment's compact view). Returns ``dQ_sel[r, h_i, :]``."""
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    dO = np.asarray(dO, dtype=np.float64)
    Hq = Q.shape[1]
    grp = Hq // K.shape[1]
    rows = np.asarray(rows, dtype=np.int64)
    pos_of = {int(r): n for n, r in enumerate(rows)}
    out = np.full((rows.size, len(heads), Q.shape[2]), np.nan)
    want = np.zeros(Q.shape[0], dtype=bool)
    want[rows] = True
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj):
        part = np.nonzero(want[seg_rows])[0]
        if part.size == 0:
            continue
        grows = seg_rows[part]
        outp = [pos_of[int(r)] for r in grows]
        for hi, h in enumerate(heads):
            k = K[idx, h // grp]
            v = V[idx, h // grp]
            q = Q[grows, h]
            if rope_theta is not None:
                k = rope(k, np.arange(idx.size), rope_theta)
                q = rope(q, n_before + part, rope_theta)
            s = _scores(q, k, scale, n_before + part)
            m = s.max(axis=1, keepdims=True)
            p = np.exp(s - m)
            p /= p.sum(axis=1, keepdims=True)
            dp = dO[grows, h] @ v.T
            ds = p * (dp - (p * dp).sum(axis=1, keepdims=True))
            dq = scale * (ds @ k)
            if rope_theta is not None:
                dq = rope(dq, n_before + part, rope_theta, inverse=True)
            out[outp, hi] = dq
    return out


def attn_bwd_keys(seqlens, edits_per_traj, Q, K, V, dO, scale, g, keys, rope_theta=None):
    """dK, dV of KV group ``g`` for a few physical key rows only.

    Same textbook formulas as ``attn_bwd`` (rotary positions included: a key's
    contribution from a segment is turned back by its angle in that segment);
    only the columns of the selected keys of each segment's ``dS`` and ``P``
    are accumulated, but every row's softmax is still normalised over its full
    live view. Used for sampled checks on workloads too large for the full
    backward.
    """
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    dO = np.asarray(dO, dtype=np.float64)
    Hq = Q.shape[1]
    grp = Hq // K.shape[1]
    keys = np.asarray(keys, dtype=np.int64)
    dk_out = np.zeros((keys.size, K.shape[2]))
    dv_out = np.zeros((keys.size, K.shape[2]))
    for seg_rows, idx, n_before in _segments(seqlens, edits_per_traj):
        where = {int(p): c for c, p in enumerate(idx)}
        cols = [(n, where[int(kk)]) for n, kk in enumerate(keys) if int(kk) in where]
        if not cols:
            continue
        kn = np.asarray([a for a, _ in cols])
        kc = np.asarray([b for _, b in cols])
        k = K[idx, g]
        v = V[idx, g]
        if rope_theta is not None:
            k = rope(k, np.arange(idx.size), rope_theta)
        for c0 in range(0, seg_rows.size, _ROW_CHUNK):
            grows = seg_rows[c0 : c0 + _ROW_CHUNK]
            crow = n_before + c0 + np.arange(grows.size)
            for h in range(g * grp, (g + 1) * grp):
                q = Q[grows, h]
                if rope_theta is not None:
                    q = rope(q, crow, rope_theta)
                do = dO[grows, h]
                s = _scores(q, k, scale, crow)
                m = s.max(axis=1, keepdims=True)
                p = np.exp(s - m)
                p /= p.sum(axis=1, keepdims=True)
                dp = do @ v.T
                ds = p * (dp - (p * dp).sum(axis=1, keepdims=True))
                dk = scale * (ds[:, kc].T @ q)
                if rope_theta is not None:
                    dk = rope(dk, kc, rope_theta, inverse=True)
                np.add.at(dk_out, kn, dk)
                np.add.at(dv_out, kn, p[:, kc].T @ do)
    return dk_out, dv_out
