"""Pins of the non-monotone (offload / retrieve) view oracle: the harness
figure's MemexRL panel, a second formulation by per-key replay, reduction to
the monotone oracle, the conditioning invariant, rotary positions in view
order, and masked attention equal to the compact per-segment computation."""

import json
import os

import numpy as np
import pytest
import torch

from oracle import attention as A
from oracle import nonmonotone as N
from oracle import visibility as V

HERE = os.path.dirname(__file__)


def _panel():
    with open(os.path.join(HERE, "golden", "memexrl_panel.json")) as f:
        g = json.load(f)
    events = [(J, [tuple(s) for s in o], [tuple(s) for s in i]) for J, o, i in g["events"]]
    return g, g["tokens"], events


def test_memexrl_panel_rows():
    g, tok, events = _panel()
    T = len(tok)
    views = N.live_views(T, events)
    slots = {tok.index(x) for x in g["slots"]}
    for name, want in g["rows"].items():
        r = tok.index(want["row"])
        view = next(v for lo, hi, v in views if lo <= r < hi)
        upto = view[: view.index(r) + 1]
        assert [tok[j] for j in upto if j not in slots] == want["view"], name


def _random_events(rng, T):
    events, out = [], set()
    Js = np.sort(rng.choice(np.arange(3, T - 1), size=int(rng.integers(2, 6)), replace=False))
    for J in Js:
        J = int(J)
        spans_in = []
        if out and rng.random() < 0.6:
            # bring back one maximal run of currently-out positions
            run = sorted(out)
            a = run[int(rng.integers(0, len(run)))]
            b = a
            while b in out:
                b += 1
            spans_in.append((a, b))
            out.difference_update(range(a, b))
        spans_out = []
        cand = [j for j in range(J) if j not in out and all(not (a <= j < b) for a, b in spans_in)]
        if cand and rng.random() < 0.8:
            a = int(rng.choice(cand))
            b = a + 1
            while b < J and b in cand and b - a < 8:
                b += 1
            spans_out.append((a, b))
            out.update(range(a, b))
        events.append((J, spans_out, spans_in))
    return events


@pytest.mark.parametrize("seed", range(8))
def test_views_equal_per_key_replay(seed):
    rng = np.random.default_rng(800 + seed)
    T = int(rng.integers(30, 120))
    events = _random_events(rng, T)
    np.testing.assert_array_equal(N.dense_mask(T, events), N.replay_mask(T, events))


@pytest.mark.parametrize("seed", range(4))
def test_without_retrievals_equals_the_monotone_oracle(seed):
    rng = np.random.default_rng(900 + seed)
    T = 80
    Js = sorted(rng.choice(np.arange(5, T - 1), size=3, replace=False).tolist())
    edits = [(int(J), [(int(a), int(min(J, a + 5)))]) for J, a in zip(Js, rng.integers(0, 4, 3))]
    events = [(J, s, []) for J, s in edits]
    assert N.live_views(T, events) == V.live_views(T, edits)
    np.testing.assert_array_equal(N.logical_positions(T, events), V.logical_positions(T, edits))


def test_later_event_leaves_earlier_views_unchanged():
    rng = np.random.default_rng(11)
    T = 90
    events = _random_events(rng, T)
    more = events + [(T - 1, [(0, 2)], [])]    # after every junction of the record
    a, b = N.live_views(T, events), N.live_views(T, more)
    assert a[:-1] == b[:-2]
    assert a[-1][2][: a[-1][2].index(T - 2) + 1] == b[-2][2]   # the split segment's rows before T - 1


def test_reentered_tokens_take_positions_after_later_tokens():
    """Rotary positions follow the view's order: in the panel's last segment
    y1..y3 come after y4 (and the offload call), not at their physical places."""
    _, tok, events = _panel()
    pos = N.logical_positions(len(tok), events)
    last = pos[-1]
    assert last[tok.index("y4")] < last[tok.index("y1")] < last[tok.index("y2")] < last[tok.index("y3")]
    assert last[tok.index("y1")] == 3          # s, offload, y4, then y1


@pytest.mark.parametrize("seed", range(3))
def test_masked_attention_equals_compact_views(seed):
    """Without positions the order inside a view does not matter: the compact
    computation equals SDPA over the physical history with the replay mask."""
    rng = np.random.default_rng(950 + seed)
    T = 70
    events = _random_events(rng, T)
    Q, K, Vx = (rng.standard_normal((T, 2, 8)) for _ in range(3))
    O = N.attn_fwd(T, events, Q, K, Vx, 0.35)
    mask = torch.from_numpy(N.replay_mask(T, events))
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(Q).transpose(0, 1), torch.from_numpy(K).transpose(0, 1),
        torch.from_numpy(Vx).transpose(0, 1), attn_mask=mask, scale=0.35).transpose(0, 1)
    np.testing.assert_allclose(O, ref.numpy(), rtol=1e-10, atol=1e-12)


def test_rotary_attention_uses_view_order():
    """With rotary positions, a row whose view holds re-entered keys differs
    from the same keys taken in physical order (so the reading matters), and
    a record without retrievals matches the monotone oracle."""
    _, tok, events = _panel()
    T = len(tok)
    rng = np.random.default_rng(3)
    Q, K, Vx = (rng.standard_normal((T, 1, 8)) for _ in range(3))
    O = N.attn_fwd(T, events, Q, K, Vx, 0.35, rope_theta=100.0)
    phys = [(J, o, i) for J, o, i in events]
    # physical-order variant of the last segment: sort its view
    last_lo = events[-1][0]
    view = N.live_views(T, phys)[-1][2]
    srt = sorted(view)
    q = A.rope(Q[last_lo:, 0], [srt.index(r) for r in range(last_lo, T)], 100.0)
    k = A.rope(K[srt, 0], np.arange(len(srt)), 100.0)
    s = (q @ k.T) * 0.35
    s[np.arange(len(srt))[None, :] > np.array([srt.index(r) for r in range(last_lo, T)])[:, None]] = -np.inf
    p = np.exp(s - s.max(axis=1, keepdims=True))
    O_phys = (p / p.sum(axis=1, keepdims=True)) @ Vx[srt, 0]
    assert np.abs(O[last_lo:, 0] - O_phys).max() > 1e-6
    edits = [(4, [(1, 4)])]
    np.testing.assert_allclose(N.attn_fwd(T, [(4, [(1, 4)], [])], Q, K, Vx, 0.35, rope_theta=100.0),
                               A.attn_fwd([T], [edits], Q, K, Vx, 0.35, rope_theta=100.0)[0], rtol=1e-12)


@pytest.mark.parametrize("seed", range(4))
def test_build_matches_replay_and_lists(seed):
    """``build``'s artefacts against the replay formulation and the lists:
    the visible pairs are the replay mask's, a row's compact index is the
    number of keys it sees minus one, each segment's membership bits are its
    view's keys, and csrc / cpos invert each other."""
    rng = np.random.default_rng(970 + seed)
    seqlens = [int(rng.integers(130, 300)), int(rng.integers(60, 140))]
    events = [_random_events(rng, T) for T in seqlens]
    out = N.build(seqlens, events)
    assert out["pairs_total"] == sum(int(N.replay_mask(T, e).sum()) for T, e in zip(seqlens, events))
    base_t, km = 0, 0
    for T, e in zip(seqlens, events):
        nt = -(-T // 128)
        rep = N.replay_mask(T, e)
        for s, (lo, hi, view) in enumerate(N.live_views(T, e)):
            base = (km + s * nt) * 128
            pos = out["cpos"][base: base + nt * 128]
            src = out["csrc"][base: base + nt * 128]
            for i in range(lo, hi):
                assert pos[i] == rep[i].sum() - 1              # row i's index = keys it sees - 1
            members = np.nonzero(pos >= 0)[0]
            assert sorted(members.tolist()) == sorted(view)
            assert all(pos[src[c]] == c for c in range(len(view)))
            bits = out["keymask"][km + s * nt: km + (s + 1) * nt]
            got = [128 * t + 32 * w + c for t in range(nt) for w in range(4) for c in range(32)
                   if (int(bits[t, w]) >> c) & 1]
            assert got == sorted(view)
            assert (out["seg"][base_t + lo: base_t + hi] == s).all()
        base_t += T
        km += (1 + len(e)) * nt


def test_build_memexrl_panel():
    """The panel's last row sees its prefix list in view order (retrieved
    y1..y3 after y4) as csrc's first entries."""
    g, tok, events = _panel()
    T = len(tok)
    out = N.build([T], [events])
    nt = 1
    S = 1 + len(events)
    base = (S - 1) * nt * 128
    view = N.live_views(T, events)[-1][2]
    assert out["csrc"][base: base + len(view)].tolist() == view
    assert out["seg_len"][-1] == len(view)


@pytest.mark.parametrize("seed", range(3))
def test_attention_oracle_on_event_views(seed):
    """``oracle.attention`` run on event views equals SDPA with the replay
    mask (forward) and autograd through it (backward): its compact-sequence
    formulas need no single-interval lifetimes."""
    rng = np.random.default_rng(990 + seed)
    T = 90
    events = _random_events(rng, T)
    Q, K, Vx, dO = (rng.standard_normal((T, h, 8)) for h in (4, 2, 2, 4))
    O, _ = A.attn_fwd([T], [events], Q, K, Vx, 0.35, views=N.live_views)
    np.testing.assert_allclose(O[:, :, :], N.attn_fwd(T, events, Q, K, Vx, 0.35), rtol=1e-10, atol=1e-12)
    mask = torch.from_numpy(N.replay_mask(T, events))
    q, k, v = (torch.tensor(x, requires_grad=True) for x in (Q, K, Vx))
    kk = k.repeat_interleave(2, dim=1)
    vv = v.repeat_interleave(2, dim=1)
    ref = torch.nn.functional.scaled_dot_product_attention(
        q.transpose(0, 1), kk.transpose(0, 1), vv.transpose(0, 1), attn_mask=mask, scale=0.35).transpose(0, 1)
    np.testing.assert_allclose(O, ref.detach().numpy(), rtol=1e-10, atol=1e-12)
    ref.backward(torch.from_numpy(dO))
    dQ, dK, dV = A.attn_bwd([T], [events], Q, K, Vx, dO, 0.35, views=N.live_views)
    np.testing.assert_allclose(dQ, q.grad.numpy(), rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dK, k.grad.numpy(), rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dV, v.grad.numpy(), rtol=1e-9, atol=1e-11)
