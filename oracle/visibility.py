"""Oracle: live views, visibility mask, tile classes and tile lists.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``). Plain Python lists and
numpy; nothing here is shared with, or imported by, the CUDA path.

Conventions (readings of the paper, pinned by the running example of §3.2 and
Table "running-prefixes" in App. B.4):

* Physical positions are 0-based; the prompt token is position 0, so the
  paper's ``s, y1 .. y12, y_ans`` are positions 0 .. 13.
* A trajectory's record is a list of edits ``(J_k, spans_k)`` with
  ``J_1 < J_2 < ...``. ``J_k`` is the physical index of the last token that
  existed before the k-th edit fired; every row ``i >= J_k`` is computed under
  the post-edit view. Row ``i`` predicts token ``i + 1``.
* ``spans_k`` is a list of half-open ``[a, b)`` ranges, the evicted set
  ``E_k`` (App. B Def. "trajectory tree": ``E_k`` lies before ``J_k``). The
  build requires ``0 <= a < b <= J_k``.
* Segment ``s`` is the row range ``[J_s, J_{s+1})`` with ``J_0 = 0`` and
  ``J_{K+1} = T``.

Tile conventions used by the GPU structures (not from the paper, which gives
no kernel): 128x128 tiles, trajectory-local, the last tile ragged. A tile is
EMPTY (0) when no in-range pair is visible, FULL (2) when every in-range pair
is visible, else PARTIAL (1). A PARTIAL off-diagonal tile also carries DEAD_LO
(4) / DEAD_HI (8) when none of its pairs with the k-tile's first / second half
of keys is visible. Tile-list entries are ``(tile << 4) | code``, code = class
plus those bits.
"""

import numpy as np

TILE = 128
EMPTY, PARTIAL, FULL = 0, 1, 2
DEAD_LO, DEAD_HI = 4, 8
NEVER = np.iinfo(np.int32).max  # lifetime end of a key that is never evicted


class RecordError(ValueError):
    pass


def validate_edits(T, edits):
    """Reject records that the conventions above do not admit.

    App. B Def. "trajectory tree": compressions fire at increasing physical
    positions and each evicts positions before its junction.
    """
    if T < 0:
        raise RecordError("negative trajectory length")
    prev = 0
    for J, spans in edits:
        if not (1 <= J <= T - 1):
            raise RecordError(f"junction {J} outside [1, T-1] for T={T}")
        if J <= prev:
            raise RecordError("junctions must be strictly ascending")
        prev = J
        for a, b in spans:
            if not (0 <= a < b <= J):
                raise RecordError(f"span [{a},{b}) not inside [0,{J})")


def live_views(T, edits):
    """Materialise each segment's live view as a list, literally.

    §3.2 (live view equation): the policy at step t conditions on the physical
    history with exactly the edits fired by step t applied. Segment 0 sees
    ``[0, J_1)``; at each junction the evicted positions are removed from the
    running list and the segment's own rows are appended.

    Returns a list of ``(row_lo, row_hi, view)`` where ``view`` is the ordered
    list of physical positions of segment ``[row_lo, row_hi)``'s compact
    sequence; the segment's rows are the last ``row_hi - row_lo`` entries.
    """
    validate_edits(T, edits)
    bounds = [0] + [J for J, _ in edits] + [T]
    view = []
    out = []
    for s in range(len(bounds) - 1):
        lo, hi = bounds[s], bounds[s + 1]
        if s >= 1:
            _, spans = edits[s - 1]
            gone = set()
            for a, b in spans:
                gone.update(range(a, b))
            view = [j for j in view if j not in gone]
        view = view + list(range(lo, hi))
        out.append((lo, hi, list(view)))
    return out


def segment_ids(T, edits):
    """Segment id of every row: the number of junctions ``J_k <= i``.

    App. B.1: rows decoded within ``[J_{k-1}, J_k)`` form one branch layer.
    """
    seg = np.zeros(T, dtype=np.int32)
    for s, (lo, hi, _) in enumerate(live_views(T, edits)):
        seg[lo:hi] = s
    return seg


def membership(T, view):
    """Boolean vector over ``[0, T)``: position is in the given view list."""
    m = np.zeros(T, dtype=bool)
    m[np.asarray(view, dtype=np.int64)] = True
    return m


def dense_mask(T, edits):
    """Dense ``[T, T]`` visibility from list membership (small T only).

    Row i sees key j iff j is in its segment's live view and ``j <= i``
    (the compact sequence is causal: the row attends to the view's prefix up
    to and including itself).
    """
    vis = np.zeros((T, T), dtype=bool)
    for lo, hi, view in live_views(T, edits):
        m = membership(T, view)
        for i in range(lo, hi):
            vis[i, : i + 1] = m[: i + 1]
    return vis


def lifetimes(T, edits):
    """Lifetime end ``omega(j) = min{J_k : j in E_k}`` (NEVER if never evicted).

    §4.2, 4D-mask equation: key j is visible to row i iff
    ``tau(j) <= i < omega(j)`` with ``tau(j) = j`` on the physical union.
    This is the second, independent formulation used only to cross-check
    ``dense_mask`` in the oracle's own tests.
    """
    validate_edits(T, edits)
    om = np.full(T, NEVER, dtype=np.int64)
    for J, spans in edits:
        for a, b in spans:
            om[a:b] = np.minimum(om[a:b], J)
    return om


def lifetime_mask(T, edits):
    """Dense mask from lifetimes: ``j <= i < omega(j)`` (§4.2)."""
    om = lifetimes(T, edits)
    i = np.arange(T)[:, None]
    j = np.arange(T)[None, :]
    return (j <= i) & (i < om[None, :])


def tile_counts(T, edits, tile=TILE):
    """Visible-pair count of every (q-tile, k-tile) of one trajectory.

    For a row i of segment s the visible keys are the members of ``view_s``
    at positions ``<= i``; the count inside k-tile ``[k0, k1)`` is read off a
    prefix sum of the membership vector. Returns an int64 array
    ``[nt, nt]`` (upper triangle zero) and the in-range area of each tile.
    """
    nt = (T + tile - 1) // tile
    counts = np.zeros((nt, nt), dtype=np.int64)
    kt_lo = np.arange(nt) * tile
    kt_hi = np.minimum(kt_lo + tile, T)
    views = live_views(T, edits)
    seg = np.zeros(T, dtype=np.int64)
    prefix = []
    for s, (lo, hi, view) in enumerate(views):
        seg[lo:hi] = s
        prefix.append(np.concatenate([[0], np.cumsum(membership(T, view), dtype=np.int64)]))
    for qt in range(nt):
        rows = np.arange(kt_lo[qt], kt_hi[qt])
        for s in np.unique(seg[rows]):
            r = rows[seg[rows] == s]
            cs = prefix[s]
            upto = np.minimum(kt_hi[None, :], r[:, None] + 1)
            c = np.where(upto > kt_lo[None, :], cs[upto] - cs[kt_lo][None, :], 0)
            counts[qt] += c.sum(axis=0)
    area = (kt_hi - kt_lo)[:, None] * (kt_hi - kt_lo)[None, :]
    return counts, area


def tile_classes(T, edits, tile=TILE):
    """EMPTY / PARTIAL / FULL for every tile pair ``kt <= qt``."""
    counts, area = tile_counts(T, edits, tile)
    cls = np.where(counts == 0, EMPTY, np.where(counts == area, FULL, PARTIAL))
    nt = counts.shape[0]
    cls[np.triu_indices(nt, 1)] = EMPTY
    return cls.astype(np.int32), counts


def dead_halves(T, edits, cls, tile=TILE):
    """DEAD_LO / DEAD_HI bits of every PARTIAL off-diagonal tile.

    Key half h of tile (qt, kt) holds keys ``[kt*tile + h*tile/2, ... +
    tile/2)``; it is dead when none of its pairs with the q-tile's rows is
    visible. The counts come from the same per-segment view prefix sums as
    the tile classes, at half-tile granularity: the q-tile's two half-row
    tiles against the half-key tile. Halves past the trajectory's end are dead.
    """
    h = tile // 2
    c, _ = tile_counts(T, edits, h)
    nt = cls.shape[0]
    c_pad = np.zeros((2 * nt + 2, 2 * nt + 2), dtype=np.int64)
    c_pad[:c.shape[0], :c.shape[1]] = c
    q = np.arange(nt)
    partial_off = (cls == PARTIAL) & (q[:, None] > q[None, :])
    out = np.zeros_like(cls)
    for hh, bit in ((0, DEAD_LO), (1, DEAD_HI)):
        kh = 2 * q + hh
        cnt = c_pad[2 * q][:, kh] + c_pad[2 * q + 1][:, kh]
        out |= np.where(partial_off & (cnt == 0), bit, 0).astype(cls.dtype)
    return out


def logical_positions(T, edits):
    """Row-wise logical position of every key in every segment's live view.

    §4.2 reassigns position ids so that the keys a row sees form a gap-free
    sequence (condition (ii) of the 4D-mask equivalence proposition, App. C):
    in segment s the key at physical position j takes the position it has in
    the compact list ``view_s``, i.e. its index there. Returns int64
    ``[S, T]``, -1 where j is not a member of ``view_s``. A row i of segment s
    is a member of its own view, so ``out[s, i]`` is the row's own position.
    """
    views = live_views(T, edits)
    out = np.full((len(views), T), -1, dtype=np.int64)
    for s, (_, _, view) in enumerate(views):
        for n, j in enumerate(view):
            out[s, j] = n
    return out


def segment_keymask(T, edits, tile=TILE):
    """Per (segment, k-tile) 128-bit membership of the segment's live view.

    Bit c of word w of entry ``[s, kt]`` is set iff position
    ``kt*tile + 32*w + c`` is in ``view_s``. Returns uint32 ``[S, nt, 4]``.
    """
    views = live_views(T, edits)
    nt = (T + tile - 1) // tile
    out = np.zeros((len(views), nt, tile // 32), dtype=np.uint32)
    for s, (_, _, view) in enumerate(views):
        m = np.zeros(nt * tile, dtype=bool)
        m[np.asarray(view, dtype=np.int64)] = True
        bits = m.reshape(nt, tile // 32, 32).astype(np.uint64)
        out[s] = (bits << np.arange(32, dtype=np.uint64)).sum(-1).astype(np.uint32)
    return out


def build(seqlens, edits_per_traj, tile=TILE):
    """All visibility artefacts of a packed multi-trajectory record.

    Trajectories are packed back to back; tiles are trajectory-local and
    numbered globally in trajectory order. Returns a dict of numpy arrays in
    the exact layout the GPU builder produces, so tests compare bit for bit:

    ``omega`` int32 [T_total]  lifetime end (trajectory-local, NEVER = int32 max)
    ``seg``   int32 [T_total]  segment id of each row
    ``qtile_traj`` int32 [n_tiles]
    ``cls``   list of per-trajectory [nt, nt] tile codes (class | DEAD bits)
    ``fwd_ptr``/``fwd_idx``  per global q-tile, ascending non-empty k-tiles
    ``bwd_ptr``/``bwd_idx``  per global k-tile, ascending non-empty q-tiles
    ``pairs`` int64 [n_traj], ``pairs_total`` int
    ``keymask`` uint32 [sum_b S_b * nt_b, 4] (per trajectory: segment-major)
    ``seg_len`` int32 [n_segs]  length of each segment's live view (its compact sequence)
    ``cpos``  int32 [sum_b S_b * nt_b * 128] rank of key j in view_s (``logical_positions``,
              -1 if absent), entry ``(km_b + s nt_b) 128 + j`` with km_b the trajectory's
              first keymask entry
    ``csrc``  int32, same indexing by rank c: the key at index c of the list view_s,
              -1 from ``len(view_s)`` to the end of its last 128-entry tile, -2 after
              (left unspecified)
    """
    omega, seg, qtraj, classes = [], [], [], []
    fwd_ptr, fwd_idx, bwd_ptr, bwd_idx = [0], [], [0], []
    pairs, keymask = [], []
    seg_len, cpos, csrc = [], [], []
    for b, (T, edits) in enumerate(zip(seqlens, edits_per_traj)):
        cls, counts = tile_classes(T, edits, tile)
        cls = cls | dead_halves(T, edits, cls, tile)
        nt = cls.shape[0]
        om = lifetimes(T, edits)
        # The dense-mask path is the definition; lifetimes are stored as the
        # GPU's compact encoding and must agree with the views (tested).
        omega.append(np.where(om == NEVER, NEVER, om).astype(np.int32))
        seg.append(segment_ids(T, edits))
        qtraj.append(np.full(nt, b, dtype=np.int32))
        classes.append(cls)
        # fwd list of q-tile qt: its non-EMPTY k-tiles in ascending order
        # (row-major scan of the class matrix); bwd list of k-tile kt: its
        # non-EMPTY q-tiles in ascending order (scan of the transpose).
        q_nz, k_nz = np.nonzero(cls != EMPTY)
        fwd_idx.extend(((k_nz << 4) | cls[q_nz, k_nz]).tolist())
        fwd_ptr.extend((fwd_ptr[-1] + np.cumsum(np.bincount(q_nz, minlength=nt))).tolist())
        k_nz2, q_nz2 = np.nonzero(cls.T != EMPTY)
        bwd_idx.extend(((q_nz2 << 4) | cls[q_nz2, k_nz2]).tolist())
        bwd_ptr.extend((bwd_ptr[-1] + np.cumsum(np.bincount(k_nz2, minlength=nt))).tolist())
        pairs.append(int(counts.sum()))
        keymask.append(segment_keymask(T, edits, tile).reshape(-1, tile // 32))
        lp = logical_positions(T, edits)
        for s, (_, _, view) in enumerate(live_views(T, edits)):
            seg_len.append(len(view))
            pos = np.full(nt * tile, -1, dtype=np.int64)
            pos[:T] = lp[s]
            cpos.append(pos)
            src = np.full(nt * tile, -2, dtype=np.int64)
            src[: -(-len(view) // tile) * tile] = -1
            src[: len(view)] = view
            csrc.append(src)
    cat = (lambda xs: np.concatenate(xs).astype(np.int32)) if cpos else (lambda xs: np.zeros(0, np.int32))
    return {
        "omega": np.concatenate(omega),
        "seg": np.concatenate(seg),
        "qtile_traj": np.concatenate(qtraj),
        "cls": classes,
        "fwd_ptr": np.asarray(fwd_ptr, dtype=np.int32),
        "fwd_idx": np.asarray(fwd_idx, dtype=np.int32),
        "bwd_ptr": np.asarray(bwd_ptr, dtype=np.int32),
        "bwd_idx": np.asarray(bwd_idx, dtype=np.int32),
        "pairs": np.asarray(pairs, dtype=np.int64),
        "pairs_total": int(sum(pairs)),
        "keymask": np.concatenate(keymask) if keymask else np.zeros((0, tile // 32), np.uint32),
        "seg_len": np.asarray(seg_len, dtype=np.int32),
        "cpos": cat(cpos),
        "csrc": cat(csrc),
    }
