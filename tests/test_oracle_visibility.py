"""Pins for the visibility oracle (CPU only).

The oracle is checked against values printed in the paper (golden fixtures),
against a second formulation of the same mask (lifetimes, §4.2), and against
brute force on small records.
"""

import json
import os

import numpy as np
import pytest

import synth
from oracle import visibility as V

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _edits(raw):
    return [(J, [tuple(s) for s in spans]) for J, spans in raw]


def test_running_example_live_views():
    g = _load("running_example.json")
    tok = g["tokens"]
    pos = {t: n for n, t in enumerate(tok)}
    edits = _edits(g["edits"])
    T = len(tok)
    mask = V.dense_mask(T, edits)
    for leaf, prefix in g["live_view_prefix"].items():
        row = pos[leaf] - 1
        want = {0} | {pos[t] for t in prefix}
        assert set(np.nonzero(mask[row])[0].tolist()) == want, leaf


def test_running_example_final_walk_and_divergence():
    g = _load("running_example.json")
    tok = g["tokens"]
    pos = {t: n for n, t in enumerate(tok)}
    edits = _edits(g["edits"])
    final_view = V.live_views(len(tok), edits)[-1][2]
    mask = V.dense_mask(len(tok), edits)
    for leaf, prefix in g["final_walk_prefix"].items():
        cut = pos[leaf]
        got = {j for j in final_view if j < cut}
        assert got == {0} | {pos[t] for t in prefix}, leaf
        live = set(np.nonzero(mask[cut - 1])[0].tolist())
        assert live - got == {pos[t] for t in g["diverges_by"][leaf]}, leaf


def test_running_example_pins_the_junction_convention():
    """The alternative reading 'an edit takes effect one row after J_k' fails
    the table's y_ans row, so the golden file discriminates the two."""
    g = _load("running_example.json")
    pos = {t: n for n, t in enumerate(g["tokens"])}
    shifted = [(J + 1, spans) for J, spans in _edits(g["edits"])]
    mask = V.dense_mask(len(g["tokens"]), shifted)
    row = pos["y_ans"] - 1
    want = {0} | {pos[t] for t in g["live_view_prefix"]["y_ans"]}
    assert set(np.nonzero(mask[row])[0].tolist()) != want


def test_blackbox_grid():
    g = _load("blackbox_grid.json")
    tok = g["tokens"]
    pos = {t: n for n, t in enumerate(tok)}
    mask = V.dense_mask(len(tok), _edits(g["edits"]))
    for decoded, ctx in g["decoded_under"].items():
        row = pos[decoded] - 1
        assert set(np.nonzero(mask[row])[0].tolist()) == {pos[t] for t in ctx}, decoded


def test_running_example_lifetimes():
    g = _load("running_example.json")
    om = V.lifetimes(14, _edits(g["edits"]))
    assert om[5] == 7 and om[8] == 10 and om[11] == 12
    assert (np.delete(om, [5, 8, 11]) == V.NEVER).all()


def _random_edits(T, rng, K):
    Js = sorted(rng.choice(np.arange(1, T), size=min(K, T - 1), replace=False).tolist())
    edits = []
    for J in Js:
        spans = []
        for _ in range(rng.integers(0, 4)):
            a = int(rng.integers(0, J))
            b = int(rng.integers(a + 1, J + 1))
            spans.append((a, b))
        edits.append((J, spans))
    return edits


@pytest.mark.parametrize("seed", range(12))
def test_views_equal_lifetime_mask(seed):
    """Two formulations: literal per-segment lists vs j <= i < omega(j)."""
    rng = np.random.default_rng(seed)
    T = int(rng.integers(2, 300))
    edits = _random_edits(T, rng, int(rng.integers(0, 8)))
    assert (V.dense_mask(T, edits) == V.lifetime_mask(T, edits)).all()


def test_no_edits_is_causal():
    T = 77
    assert (V.dense_mask(T, []) == np.tril(np.ones((T, T), dtype=bool))).all()
    cls, counts = V.tile_classes(T, [], tile=16)
    nt = cls.shape[0]
    for q in range(nt):
        for k in range(nt):
            if k < q:
                assert cls[q, k] == V.FULL
            elif k == q:
                assert cls[q, k] == (V.FULL if min(16, T - 16 * q) == 1 else V.PARTIAL)
    assert counts.sum() == T * (T + 1) // 2


@pytest.mark.parametrize("seed", range(8))
def test_tile_classes_brute_force(seed):
    """Tile classes and counts from the prefix-sum path equal any/all over
    the dense mask, including a ragged last tile."""
    rng = np.random.default_rng(100 + seed)
    tile = 16
    T = int(rng.integers(17, 200))
    edits = _random_edits(T, rng, int(rng.integers(1, 6)))
    mask = V.dense_mask(T, edits)
    cls, counts = V.tile_classes(T, edits, tile=tile)
    nt = (T + tile - 1) // tile
    for q in range(nt):
        for k in range(q + 1):
            blk = mask[q * tile : (q + 1) * tile, k * tile : (k + 1) * tile]
            assert counts[q, k] == blk.sum()
            want = V.EMPTY if not blk.any() else (V.FULL if blk.all() else V.PARTIAL)
            assert cls[q, k] == want


@pytest.mark.parametrize("seed", range(8))
def test_dead_halves_brute_force(seed):
    """A key half of a PARTIAL off-diagonal tile is flagged dead exactly when
    the dense mask has no visible pair between the q-tile's rows and that
    half's keys (keys past the end count as dead); never both halves, never
    on FULL or diagonal tiles."""
    rng = np.random.default_rng(300 + seed)
    tile = 16
    T = int(rng.integers(40, 260))
    edits = _random_edits(T, rng, int(rng.integers(1, 7)))
    mask = V.dense_mask(T, edits)
    cls, _ = V.tile_classes(T, edits, tile=tile)
    dead = V.dead_halves(T, edits, cls, tile=tile)
    nt = (T + tile - 1) // tile
    h = tile // 2
    seen = 0
    for q in range(nt):
        for k in range(q + 1):
            if cls[q, k] != V.PARTIAL or k == q:
                assert dead[q, k] == 0
                continue
            rows = mask[q * tile:(q + 1) * tile]
            want = 0
            for hh, bit in ((0, V.DEAD_LO), (1, V.DEAD_HI)):
                blk = rows[:, k * tile + hh * h:k * tile + (hh + 1) * h]
                if not blk.any():
                    want |= bit
            assert dead[q, k] == want, (q, k)
            assert want != V.DEAD_LO | V.DEAD_HI
            seen += want != 0
    assert seen > 0 or seed > 3   # the generator's evictions leave dead halves in most records


def test_build_lists_and_pairs():
    r = synth.config_record(1)
    out = V.build(r.seqlens, r.edits, tile=V.TILE)
    T = r.seqlens[0]
    mask = V.dense_mask(T, r.edits[0])
    assert out["pairs_total"] == int(mask.sum())
    # fwd and bwd lists name the same tiles with the same classes
    fwd = {(q, e >> 4, e & 15) for q in range(len(out["fwd_ptr"]) - 1)
           for e in out["fwd_idx"][out["fwd_ptr"][q]:out["fwd_ptr"][q + 1]]}
    bwd = {(e >> 4, k, e & 15) for k in range(len(out["bwd_ptr"]) - 1)
           for e in out["bwd_idx"][out["bwd_ptr"][k]:out["bwd_ptr"][k + 1]]}
    assert fwd == bwd
    # every visible pair lies in a listed tile
    for (q, k, c) in fwd:
        assert c & 3 in (V.PARTIAL, V.FULL)
    nt = (T + 127) // 128
    listed = np.zeros((nt, nt), dtype=bool)
    for (q, k, _) in fwd:
        listed[q, k] = True
    for i, j in zip(*np.nonzero(mask)):
        assert listed[i // 128, j // 128]


def test_keymask_matches_views():
    r = synth.config_record(1)
    T, edits = r.seqlens[0], r.edits[0]
    km = V.segment_keymask(T, edits)
    for s, (_, _, view) in enumerate(V.live_views(T, edits)):
        bits = np.zeros(km.shape[1] * 128, dtype=bool)
        for j in range(bits.size):
            bits[j] = (km[s, j // 128, (j % 128) // 32] >> (j % 32)) & 1
        assert set(np.nonzero(bits)[0].tolist()) == set(view)


def test_conditioning_invariant_on_views():
    """Adding an edit at J leaves every row before J unchanged (§3.3 Def.
    conditioning consistency: only edits fired through step t matter)."""
    rng = np.random.default_rng(7)
    T = 150
    edits = _random_edits(T, rng, 3)
    J_new = edits[-1][0] + 5 if edits and edits[-1][0] + 5 < T else T - 1
    more = edits + [(J_new, [(J_new - 1, J_new)])]  # never evicted before
    a, b = V.dense_mask(T, edits), V.dense_mask(T, more)
    assert (a[:J_new] == b[:J_new]).all()
    assert not (a[J_new:] == b[J_new:]).all()


@pytest.mark.parametrize("bad", [
    [(0, [])],                       # junction at 0
    [(5, []), (5, [])],              # not strictly ascending
    [(5, [(3, 6)])],                 # span reaches past J
    [(5, [(4, 4)])],                 # empty span
    [(200, [])],                     # junction beyond T-1
])
def test_invalid_records_rejected(bad):
    with pytest.raises(V.RecordError):
        V.live_views(100, bad)


def test_compact_maps_running_example():
    """Each segment's compact sequence (``csrc``) read up to a row's own index
    is exactly the prefix Table "running-prefixes" prints for the leaf that
    row predicts; ``cpos`` is its inverse and ``seg_len`` its length."""
    g = _load("running_example.json")
    tok = g["tokens"]
    pos = {t: n for n, t in enumerate(tok)}
    edits = _edits(g["edits"])
    T = len(tok)
    out = V.build([T], [edits])
    nt = -(-T // V.TILE)
    seg = V.segment_ids(T, edits)
    for leaf, prefix in g["live_view_prefix"].items():
        row = pos[leaf] - 1
        s = int(seg[row])
        base = s * nt * V.TILE
        c_row = int(out["cpos"][base + row])
        assert c_row >= 0
        got = out["csrc"][base: base + c_row + 1].tolist()
        assert got == sorted({0} | {pos[t] for t in prefix}), leaf
    assert out["seg_len"].tolist() == [7, 9, 10, 11]


@pytest.mark.parametrize("seed", range(5))
def test_compact_maps_inverse(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(130, 600))
    Js = sorted(rng.choice(np.arange(2, T), size=4, replace=False).tolist())
    edits = [(J, [(int(a), int(min(J, a + rng.integers(1, 40))))
                  for a in rng.integers(0, J - 1, 3)]) for J in Js]
    out = V.build([T], [edits])
    nt = -(-T // V.TILE)
    for s, (lo, hi, view) in enumerate(V.live_views(T, edits)):
        base = s * nt * V.TILE
        src = out["csrc"][base: base + nt * V.TILE]
        pos = out["cpos"][base: base + nt * V.TILE]
        L = int(out["seg_len"][s])
        assert L == len(view)
        assert all(pos[src[c]] == c for c in range(L))
        assert int((pos[:T] >= 0).sum()) == L
        assert (src[L: -(-L // V.TILE) * V.TILE] == -1).all()
        assert src[L - (hi - lo): L].tolist() == list(range(lo, hi))   # the segment's rows are the tail


def test_on_policy_summary_rows_see_the_folded_prefix():
    """On-policy summaries (AgentFold: the policy summarises the foldable
    prefix, the summary is trained, then the prefix is replaced by it): the
    fold's junction is the summary's last token, so the rows that decode the
    summary see the folded spans, and every later row sees the summary but
    not the folded spans."""
    r = synth.record(1, 700, 2, 0.6, 40, 32, 40, 30, 5, on_policy_summary=True)
    t = r.trajs[0]
    mask = V.dense_mask(t.T, t.edits)
    for J, spans in t.edits:
        gone = [j for a, b in spans for j in range(a, b)]
        assert gone
        summary = range(J - 39, J + 1)
        for i in range(J - 40, J):                  # rows predicting summary tokens
            assert mask[i, gone].all()
        for i in range(J, min(t.T, J + 30)):
            assert not mask[i, gone].any()
            assert mask[i, list(summary)].all()
