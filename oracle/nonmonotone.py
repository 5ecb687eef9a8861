"""Oracle: live views of records whose edits also bring spans back (non-monotone
lifetimes: MemexRL's offload / retrieve).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``). Float64, lists, literal.

The paper's MemexRL harness (App. F harness notes) offloads a named span and
later retrieves it, so a token can leave the live view and re-enter it; the
harness figure's MemexRL panel (e) draws the retrieved span re-entering after
the tokens that were decoded meanwhile. Reading taken (the paper gives no
formula): an event ``(J, out_spans, in_spans)`` fires at junction J like a
compression (rows i >= J see the post-event view); ``out_spans`` leave the
view, then the positions of ``in_spans`` (which must be out of the view at J)
re-enter at its end in their original order, before the segment's own rows.
A view is therefore an ordered list that need not follow physical order; a
row's keys are the members of its segment's list up to and including itself,
and its rotary positions are list indices.

``build`` gives the artefacts the GPU builder of such records produces (the
segments, each segment's compact sequence and its ranks, the view bits and
the visible pairs), straight from the lists; the attention oracle runs on the
same lists (``oracle.attention`` with ``views=live_views``).
"""

import numpy as np

from .visibility import RecordError


def validate_events(T, events):
    """Junctions strictly ascending inside [1, T-1]; spans inside [0, J); a
    retrieved position must be out of the view when its event fires."""
    if T < 0:
        raise RecordError("negative trajectory length")
    prev = 0
    out = set()
    for J, spans_out, spans_in in events:
        if not (1 <= J <= T - 1):
            raise RecordError(f"junction {J} outside [1, T-1] for T={T}")
        if J <= prev:
            raise RecordError("junctions must be strictly ascending")
        prev = J
        for a, b in list(spans_out) + list(spans_in):
            if not (0 <= a < b <= J):
                raise RecordError(f"span [{a},{b}) not inside [0,{J})")
        for a, b in spans_out:
            out.update(range(a, b))
        for a, b in spans_in:
            if not all(j in out for j in range(a, b)):
                raise RecordError(f"retrieved span [{a},{b}) is not out of the view at {J}")
            out.difference_update(range(a, b))


def live_views(T, events):
    """Each segment's live view as an ordered list (see the module reading).

    Returns ``[(row_lo, row_hi, view)]``; the segment's own rows are the last
    ``row_hi - row_lo`` entries of ``view``.
    """
    validate_events(T, events)
    bounds = [0] + [J for J, _, _ in events] + [T]
    view, res = [], []
    for s in range(len(bounds) - 1):
        lo, hi = bounds[s], bounds[s + 1]
        if s >= 1:
            _, spans_out, spans_in = events[s - 1]
            gone = set()
            for a, b in spans_out:
                gone.update(range(a, b))
            view = [j for j in view if j not in gone]
            for a, b in spans_in:
                view.extend(range(a, b))
        view = view + list(range(lo, hi))
        res.append((lo, hi, list(view)))
    return res


def dense_mask(T, events):
    """Row i sees key j iff j is in its segment's view at or before i's own
    entry (the compact sequence is causal in view order)."""
    vis = np.zeros((T, T), dtype=bool)
    for lo, hi, view in live_views(T, events):
        for i in range(lo, hi):
            upto = view[: view.index(i) + 1]
            vis[i, upto] = True
    return vis


def replay_mask(T, events):
    """Second formulation: replay each key's in/out state through the events
    (a key exists from its own row on; an event's out-spans switch it off and
    its in-spans back on for every row from the event's junction); row i sees
    j iff j <= i and j is on at i. Order within the view does not enter."""
    validate_events(T, events)
    state = np.ones((T, T), dtype=bool)           # state[i, j]: key j on at row i
    for J, spans_out, spans_in in events:
        for a, b in spans_out:
            state[J:, a:b] = False
        for a, b in spans_in:
            state[J:, a:b] = True
    causal = np.tril(np.ones((T, T), dtype=bool))
    return state & causal


def logical_positions(T, events):
    """Rank of every key in every segment's ordered view, -1 off the view."""
    views = live_views(T, events)
    pos = np.full((len(views), T), -1, dtype=np.int64)
    for s, (_, _, view) in enumerate(views):
        for n, j in enumerate(view):
            pos[s, j] = n
    return pos


def attn_fwd(T, events, Q, K, V, scale, rope_theta=None):
    """Softmax attention of every row over its segment's compact sequence (one
    trajectory; ``Q`` [T, Hq, Dh], ``K``, ``V`` [T, Hkv, Dh]); with
    ``rope_theta`` queries and keys are rotated by their view index."""
    from .attention import rope
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    Hq, Hkv = Q.shape[1], K.shape[1]
    grp = Hq // Hkv
    O = np.zeros_like(Q)
    for lo, hi, view in live_views(T, events):
        idx = np.asarray(view, dtype=np.int64)
        n0 = len(view) - (hi - lo)
        for h in range(Hq):
            k = K[idx, h // grp]
            q = Q[lo:hi, h]
            if rope_theta is not None:
                k = rope(k, np.arange(idx.size), rope_theta)
                q = rope(q, n0 + np.arange(hi - lo), rope_theta)
            s = (q @ k.T) * scale
            c = np.arange(idx.size)[None, :]
            s[c > (n0 + np.arange(hi - lo))[:, None]] = -np.inf
            p = np.exp(s - s.max(axis=1, keepdims=True))
            O[lo:hi, h] = (p / p.sum(axis=1, keepdims=True)) @ V[idx, h // grp]
    return O


def build(seqlens, events_per_traj, tile=128):
    """Per packed record (trajectories back to back), in the GPU layout:
    ``seg`` int32 [T_total] segment of each row; ``seg_len`` int32 [n_segs]
    length of each view list; ``cpos`` / ``csrc`` int32 (entry
    ``(km_b + s nt_b) tile + j``, km_b the trajectory's first (segment, tile)
    entry): the index of key j in view_s (-1 if absent) and the key at index
    c (-1 from the list's end to the end of its last tile, -2 after, left
    unspecified); ``keymask`` uint32 [entries][tile / 32] view membership
    bits; ``pairs`` int64 [n_traj] visible pairs (a row at list index c sees
    c + 1 keys) and ``pairs_total``."""
    seg, seg_len, cpos, csrc, keymask, pairs = [], [], [], [], [], []
    for T, events in zip(seqlens, events_per_traj):
        nt = -(-T // tile)
        sg = np.zeros(T, dtype=np.int32)
        npairs = 0
        for s, (lo, hi, view) in enumerate(live_views(T, events)):
            sg[lo:hi] = s
            seg_len.append(len(view))
            pos = np.full(nt * tile, -1, dtype=np.int64)
            pos[np.asarray(view, dtype=np.int64)] = np.arange(len(view))
            cpos.append(pos)
            src = np.full(nt * tile, -2, dtype=np.int64)
            src[: -(-len(view) // tile) * tile] = -1
            src[: len(view)] = view
            csrc.append(src)
            bits = (pos >= 0).reshape(nt, tile // 32, 32).astype(np.uint64)
            keymask.append((bits << np.arange(32, dtype=np.uint64)).sum(-1).astype(np.uint32))
            npairs += sum(view.index(i) + 1 for i in range(lo, hi))
        seg.append(sg)
        pairs.append(npairs)
    cat = lambda xs, dt: np.concatenate(xs).astype(dt) if xs else np.zeros(0, dt)   # noqa: E731
    return {
        "seg": cat(seg, np.int32),
        "seg_len": np.asarray(seg_len, dtype=np.int32),
        "cpos": cat(cpos, np.int32),
        "csrc": cat(csrc, np.int32),
        "keymask": np.concatenate(keymask) if keymask else np.zeros((0, tile // 32), np.uint32),
        "pairs": np.asarray(pairs, dtype=np.int64),
        "pairs_total": int(sum(pairs)),
    }
