"""Pins of the oracle's row-wise logical positions and rotary attention.

§4.2 reassigns position ids so that the keys each row sees form a gap-free
sequence; the 4D-mask equivalence proposition (App. C, conditions (i) and
(ii)) states that the masked computation on the physical history, with those
per-row positions, equals the forward on each branch's compact sequence. The
oracle computes the compact side; these tests pin it to the paper's running
example, to an independent derivation from the lifetimes, to a dense masked
computation with a per-(row, key) position table, and to the algebra of the
rotation itself.
"""

import json
import os

import numpy as np
import pytest
import torch

from oracle import attention as A
from oracle import visibility as V

HERE = os.path.dirname(__file__)


def _rng(seed):
    return np.random.default_rng(seed)


# --------------------------------------------------------------------------
# the rotation


def test_rope_is_orthogonal_and_composes():
    rng = _rng(0)
    x = rng.standard_normal((7, 3, 16))
    p = np.array([0, 1, 5, 17, 100, 4095, 65535])
    y = A.rope(x, p, 10000.0)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-12)
    np.testing.assert_allclose(A.rope(x, np.zeros(7), 10000.0), x, atol=0)
    np.testing.assert_allclose(A.rope(y, p, 10000.0, inverse=True), x, atol=1e-12)
    q = np.array([3, 8, 1, 0, 9, 2, 7])
    np.testing.assert_allclose(A.rope(A.rope(x, p, 10000.0), q, 10000.0), A.rope(x, p + q, 10000.0),
                               atol=1e-9)


def test_rope_scores_depend_on_offset_only():
    rng = _rng(1)
    q = rng.standard_normal((1, 64))
    k = rng.standard_normal((1, 64))
    ref = (A.rope(q, [40], 1e6) * A.rope(k, [13], 1e6)).sum()
    for c in (-13, 1, 250, 30000):
        got = (A.rope(q, [40 + c], 1e6) * A.rope(k, [13 + c], 1e6)).sum()
        assert abs(got - ref) < 1e-9
    # and the offset does matter
    assert abs((A.rope(q, [41], 1e6) * A.rope(k, [13], 1e6)).sum() - ref) > 1e-3


def test_rope_two_dims_is_complex_rotation():
    # Dh = 2: one pair with frequency theta^0 = 1, i.e. multiplication of
    # x0 + i x1 by exp(i p).
    x = np.array([[0.3, -1.7]])
    for p in (0, 1, 2, 7, 1000):
        z = complex(0.3, -1.7) * np.exp(1j * p)
        np.testing.assert_allclose(A.rope(x, [p], 10000.0)[0], [z.real, z.imag], atol=1e-12)


def test_rope_pairs_feature_f_with_f_plus_half():
    # The pair (f, f + Dh/2) turns at theta^(-2f/Dh) radians per position; the
    # angle is read back with atan2 from a unit vector in feature f.
    Dh, theta = 8, 10000.0
    for f in range(Dh // 2):
        e = np.zeros((1, Dh))
        e[0, f] = 1.0
        y = A.rope(e, [1], theta)[0]
        assert np.count_nonzero(np.abs(y) > 1e-15) <= 2
        ang = np.arctan2(y[f + Dh // 2], y[f])
        assert abs(ang - theta ** (-2.0 * f / Dh)) < 1e-12


# --------------------------------------------------------------------------
# logical positions


def test_logical_positions_running_example():
    """App. B.4 Table "running-prefixes": the row that scores leaf y_t is the
    row of y_(t-1); the prompt s is position 0 and the table's prefix tokens
    (which end with the row's own token) take positions 1, 2, ... in order."""
    with open(os.path.join(HERE, "golden", "running_example.json")) as f:
        g = json.load(f)
    tok = g["tokens"]
    edits = [(J, [tuple(s) for s in spans]) for J, spans in g["edits"]]
    T = len(tok)
    pos = V.logical_positions(T, edits)
    seg = V.segment_ids(T, edits)
    for leaf, prefix in g["live_view_prefix"].items():
        row = tok.index(leaf) - 1
        s = seg[row]
        assert pos[s, 0] == 0
        for n, name in enumerate(prefix):
            assert pos[s, tok.index(name)] == n + 1, (leaf, name)
        assert pos[s, row] == len(prefix)
        evicted = set(range(row)) - {0} - {tok.index(n) for n in prefix}
        for j in evicted:
            assert pos[s, j] == -1


@pytest.mark.parametrize("seed", range(4))
def test_logical_positions_equal_lifetime_counts(seed):
    """Second formulation from the lifetimes (§4.2): key j is a member of
    segment s's view iff omega(j) > J_s and j < J_(s+1); its position is the
    number of members before it."""
    rng = _rng(100 + seed)
    T = int(rng.integers(40, 200))
    edits = _random_edits(rng, T)
    om = V.lifetimes(T, edits)
    bounds = [0] + [J for J, _ in edits] + [T]
    pos = V.logical_positions(T, edits)
    for s in range(len(bounds) - 1):
        member = (om > bounds[s]) & (np.arange(T) < bounds[s + 1])
        want = np.where(member, np.cumsum(member) - 1, -1)
        np.testing.assert_array_equal(pos[s], want)


def _random_edits(rng, T):
    n_j = int(rng.integers(1, 5))
    Js = np.sort(rng.choice(np.arange(2, T - 1), size=n_j, replace=False))
    edits = []
    for J in Js:
        spans = []
        a = int(rng.integers(0, J))
        while a < J and len(spans) < 3:
            b = int(min(J, a + rng.integers(1, 12)))
            spans.append((a, b))
            a = b + int(rng.integers(1, 15))
        edits.append((int(J), spans))
    return edits


# --------------------------------------------------------------------------
# the equivalence of §4.2 / App. C with row-wise positions


def _dense_rope_masked(T, edits, Q, K, Vv, scale, theta, positions):
    """Attention on the physical history under the lifetime mask, one row at a
    time, with a per-(row, key) position table: row i's query is rotated by
    positions[i, i], key j by positions[i, j] (float64 torch, autograd)."""
    mask = torch.from_numpy(V.lifetime_mask(T, edits))
    Dh = Q.shape[-1]
    half = Dh // 2
    w = theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / Dh)

    def rot(x, p):
        ang = p.to(torch.float64)[:, None] * w[None, :]
        c, s = torch.cos(ang), torch.sin(ang)
        return torch.cat([x[:, :half] * c - x[:, half:] * s, x[:, half:] * c + x[:, :half] * s], dim=-1)

    outs = []
    for i in range(T):
        js = torch.nonzero(mask[i]).flatten()
        qi = rot(Q[i : i + 1], positions[i, i : i + 1])
        kj = rot(K[js], positions[i, js])
        p = torch.softmax((qi @ kj.T)[0] * scale, dim=0)
        outs.append(p @ Vv[js])
    return torch.stack(outs)


def _row_positions(T, edits):
    """Gap-free positions per row from the lifetime mask: key j's position in
    row i is the number of keys before j that row i sees."""
    m = V.lifetime_mask(T, edits)
    return torch.from_numpy(np.cumsum(m, axis=1) - 1)


@pytest.mark.parametrize("seed", range(3))
def test_rowwise_positions_masked_equals_compact(seed):
    rng = _rng(200 + seed)
    T, Dh = 60, 16
    edits = _random_edits(rng, T)
    Q = rng.standard_normal((T, 1, Dh))
    K = rng.standard_normal((T, 1, Dh))
    Vv = rng.standard_normal((T, 1, Dh))
    scale = Dh ** -0.5
    O, _ = A.attn_fwd([T], [edits], Q, K, Vv, scale, rope_theta=10000.0)
    pos = _row_positions(T, edits)
    ref = _dense_rope_masked(T, edits, torch.from_numpy(Q[:, 0]), torch.from_numpy(K[:, 0]),
                             torch.from_numpy(Vv[:, 0]), scale, 10000.0, pos)
    np.testing.assert_allclose(O[:, 0], ref.numpy(), rtol=1e-10, atol=1e-12)
    # Without the reassignment (physical positions) the masked result is a
    # different function as soon as an evicted key lies inside a row's view.
    phys = torch.arange(T)[None, :].expand(T, T)
    bad = _dense_rope_masked(T, edits, torch.from_numpy(Q[:, 0]), torch.from_numpy(K[:, 0]),
                             torch.from_numpy(Vv[:, 0]), scale, 10000.0, phys)
    assert np.abs(O[:, 0] - bad.numpy()).max() > 1e-3


def test_rowwise_positions_equal_oracle_positions():
    rng = _rng(7)
    T = 90
    edits = _random_edits(rng, T)
    pos = V.logical_positions(T, edits)
    seg = V.segment_ids(T, edits)
    rowpos = _row_positions(T, edits).numpy()
    m = V.lifetime_mask(T, edits)
    for i in range(T):
        js = np.nonzero(m[i])[0]
        np.testing.assert_array_equal(rowpos[i, js], pos[seg[i], js])


@pytest.mark.parametrize("seed", range(2))
def test_rope_backward_equals_autograd(seed):
    rng = _rng(300 + seed)
    T, Hq, Hkv, Dh = 48, 2, 1, 8
    edits = _random_edits(rng, T)
    Q = rng.standard_normal((T, Hq, Dh))
    K = rng.standard_normal((T, Hkv, Dh))
    Vv = rng.standard_normal((T, Hkv, Dh))
    dO = rng.standard_normal((T, Hq, Dh))
    scale = 0.4
    dQ, dK, dV = A.attn_bwd([T], [edits], Q, K, Vv, dO, scale, rope_theta=500.0)
    q = torch.from_numpy(Q).requires_grad_()
    k = torch.from_numpy(K).requires_grad_()
    v = torch.from_numpy(Vv).requires_grad_()
    pos = _row_positions(T, edits)
    out = torch.stack([_dense_rope_masked(T, edits, q[:, h], k[:, 0], v[:, 0], scale, 500.0, pos)
                       for h in range(Hq)], dim=1)
    out.backward(torch.from_numpy(dO))
    np.testing.assert_allclose(dQ, q.grad.numpy(), rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dK, k.grad.numpy(), rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dV, v.grad.numpy(), rtol=1e-9, atol=1e-11)


def test_rope_without_edits_is_plain_causal_rope():
    rng = _rng(9)
    T, Dh = 30, 8
    Q = rng.standard_normal((T, 1, Dh))
    K = rng.standard_normal((T, 1, Dh))
    Vv = rng.standard_normal((T, 1, Dh))
    O, L = A.attn_fwd([T], [[]], Q, K, Vv, 0.5, rope_theta=100.0)
    q = torch.from_numpy(A.rope(Q, np.arange(T), 100.0)[:, 0])
    k = torch.from_numpy(A.rope(K, np.arange(T), 100.0)[:, 0])
    ref = torch.nn.functional.scaled_dot_product_attention(q[None], k[None], torch.from_numpy(Vv[:, 0])[None],
                                                           is_causal=True, scale=0.5)[0]
    np.testing.assert_allclose(O[:, 0], ref.numpy(), rtol=1e-10, atol=1e-12)


def test_rope_row_sampled_dq_matches_full():
    """The sampled-row dQ (used to time the oracle on large workloads) equals
    the full backward's rows with rotary positions too."""
    rng = _rng(11)
    seqlens = [70, 90]
    edits = [_random_edits(rng, 70), _random_edits(rng, 90)]
    T = sum(seqlens)
    Q = rng.standard_normal((T, 4, 8))
    K = rng.standard_normal((T, 2, 8))
    Vv = rng.standard_normal((T, 2, 8))
    dO = rng.standard_normal((T, 4, 8))
    dQ, _, _ = A.attn_bwd(seqlens, edits, Q, K, Vv, dO, 0.3, rope_theta=300.0)
    rows = np.array([0, 5, 69, 70, 111, 159])
    got = A.attn_bwd_rows(seqlens, edits, Q, K, Vv, dO, 0.3, rows, [1, 3], rope_theta=300.0)
    np.testing.assert_allclose(got, dQ[rows][:, [1, 3]], rtol=1e-12, atol=1e-12)


def test_rope_key_sampled_dk_dv_match_full():
    """The sampled-key dK / dV (keys whose positions differ between segments)
    equal the full backward's rows with rotary positions."""
    rng = _rng(12)
    T = 120
    edits = _random_edits(rng, T)
    Q = rng.standard_normal((T, 4, 8))
    K = rng.standard_normal((T, 2, 8))
    Vv = rng.standard_normal((T, 2, 8))
    dO = rng.standard_normal((T, 4, 8))
    _, dK, dV = A.attn_bwd([T], [edits], Q, K, Vv, dO, 0.3, rope_theta=300.0)
    keys = np.array([0, 3, 17, 40, 77, 119])
    dk, dv = A.attn_bwd_keys([T], [edits], Q, K, Vv, dO, 0.3, 1, keys, rope_theta=300.0)
    np.testing.assert_allclose(dk, dK[keys, 1], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dv, dV[keys, 1], rtol=1e-12, atol=1e-12)


def test_rope_row_sampled_kv_contributions_sum_to_full():
    """Per-row dK / dV contributions with rotary positions (each turned back by
    the key's angle in the row's segment) add up to the full backward."""
    rng = _rng(13)
    seqlens = [70, 90]
    edits = [_random_edits(rng, 70), _random_edits(rng, 90)]
    T = sum(seqlens)
    Q = rng.standard_normal((T, 4, 8))
    K = rng.standard_normal((T, 2, 8))
    Vv = rng.standard_normal((T, 2, 8))
    dO = rng.standard_normal((T, 4, 8))
    _, dK, dV = A.attn_bwd(seqlens, edits, Q, K, Vv, dO, 0.3, rope_theta=300.0)
    sk, sv = np.zeros_like(dK), np.zeros_like(dV)
    for rows in (np.arange(0, T, 2), np.arange(1, T, 2)):
        _, dk, dv = A.attn_bwd_rows(seqlens, edits, Q, K, Vv, dO, 0.3, rows, [0, 1, 2, 3],
                                    rope_theta=300.0, with_kv=True)
        sk += dk
        sv += dv
    np.testing.assert_allclose(sk, dK, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(sv, dV, rtol=1e-10, atol=1e-12)
