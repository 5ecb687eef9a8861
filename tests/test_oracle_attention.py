"""Pins for the attention oracle (CPU only, float64).

The per-segment compact computation is checked against library routines on
the physical union (torch scaled_dot_product_attention with the causal flag,
or with the lifetime mask of §4.2 -- a formulation the oracle does not use),
against autograd and finite differences, and against the conditioning
invariant (§3.3).
"""

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import attention as A
from oracle import visibility as V


def _inputs(T, Hq, Hkv, Dh, seed):
    g = np.random.default_rng(seed)
    return (g.standard_normal((T, Hq, Dh)), g.standard_normal((T, Hkv, Dh)),
            g.standard_normal((T, Hkv, Dh)), g.standard_normal((T, Hq, Dh)))


def _edits(T, seed, K):
    rng = np.random.default_rng(seed)
    Js = sorted(rng.choice(np.arange(1, T), size=K, replace=False).tolist())
    return [(J, [(a, min(a + int(rng.integers(1, 6)), J))
                 for a in sorted(rng.choice(J, size=min(2, J), replace=False).tolist())])
            for J in Js]


def _sdpa(Q, K, V_, mask, scale, Hq, Hkv):
    """Library reference on the packed union, one trajectory."""
    q = torch.tensor(Q).permute(1, 0, 2)
    k = torch.tensor(K).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)
    v = torch.tensor(V_).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)
    if mask is None:
        o = F.scaled_dot_product_attention(q, k, v, is_causal=True, scale=scale)
    else:
        o = F.scaled_dot_product_attention(q, k, v, attn_mask=torch.tensor(mask), scale=scale)
    return o.permute(1, 0, 2).numpy()


def test_no_edits_equals_causal_sdpa():
    T, Hq, Hkv, Dh = 70, 4, 2, 16
    Q, K, V_, _ = _inputs(T, Hq, Hkv, Dh, 0)
    O, L = A.attn_fwd([T], [[]], Q, K, V_, 0.25)
    ref = _sdpa(Q, K, V_, None, 0.25, Hq, Hkv)
    np.testing.assert_allclose(O, ref, rtol=1e-12, atol=1e-12)
    # LSE against a direct log-sum-exp of the causal scores
    s = np.einsum("ihd,jhd->hij", Q, np.repeat(K, 2, axis=1)) * 0.25
    s = np.where(np.tril(np.ones((T, T), bool))[None], s, -np.inf)
    np.testing.assert_allclose(L, np.log(np.exp(s).sum(-1)), rtol=1e-12)


@pytest.mark.parametrize("seed", range(4))
def test_edits_equal_masked_sdpa(seed):
    """Theorem 'materialization equivalence' (§4.3): per-segment compact
    forwards equal one packed forward under the 4D lifetime mask."""
    T, Hq, Hkv, Dh = 90, 4, 1, 8
    edits = _edits(T, seed, 3)
    Q, K, V_, _ = _inputs(T, Hq, Hkv, Dh, seed)
    O, _ = A.attn_fwd([T], [edits], Q, K, V_, 0.3)
    ref = _sdpa(Q, K, V_, V.lifetime_mask(T, edits), 0.3, Hq, Hkv)
    np.testing.assert_allclose(O, ref, rtol=1e-11, atol=1e-12)


def test_rows_and_heads_subset_match_full():
    T, Hq, Hkv, Dh = 60, 4, 2, 8
    edits = _edits(T, 9, 2)
    Q, K, V_, _ = _inputs(T, Hq, Hkv, Dh, 9)
    O, L = A.attn_fwd([T], [edits], Q, K, V_, 0.5)
    rows = [3, 59, 17, 40]
    Os, Ls = A.attn_fwd([T], [edits], Q, K, V_, 0.5, rows=rows, heads=[1, 3])
    # equal up to BLAS rounding order (different row blocking)
    np.testing.assert_allclose(Os, O[rows][:, [1, 3]], rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(Ls, L[[1, 3]][:, rows], rtol=1e-13, atol=1e-14)


def test_packed_trajectories_are_independent():
    Ts = [40, 33]
    e = [_edits(40, 1, 2), _edits(33, 2, 1)]
    Q, K, V_, _ = _inputs(sum(Ts), 2, 1, 8, 3)
    O, _ = A.attn_fwd(Ts, e, Q, K, V_, 0.4)
    O0, _ = A.attn_fwd([40], [e[0]], Q[:40], K[:40], V_[:40], 0.4)
    O1, _ = A.attn_fwd([33], [e[1]], Q[40:], K[40:], V_[40:], 0.4)
    np.testing.assert_allclose(O, np.concatenate([O0, O1]), rtol=1e-13, atol=1e-14)


def test_conditioning_invariant_forward():
    """A row's output is unchanged by edits after it (§3.3), up to BLAS
    rounding order (the segment holding the row is split into two chunks)."""
    T = 80
    edits = _edits(T, 4, 2)
    Q, K, V_, _ = _inputs(T, 2, 2, 8, 4)
    J_new = edits[-1][0] + 3
    more = edits + [(J_new, [(0, 5), (J_new - 2, J_new)])]
    a, _ = A.attn_fwd([T], [edits], Q, K, V_, 0.5)
    b, _ = A.attn_fwd([T], [more], Q, K, V_, 0.5)
    np.testing.assert_allclose(a[:J_new], b[:J_new], rtol=1e-13, atol=1e-14)
    assert np.abs(a[J_new:] - b[J_new:]).max() > 1e-6


@pytest.mark.parametrize("seed", range(3))
def test_backward_equals_autograd(seed):
    T, Hq, Hkv, Dh = 50, 4, 2, 8
    edits = _edits(T, 20 + seed, 3)
    Q, K, V_, dO = _inputs(T, Hq, Hkv, Dh, 20 + seed)
    dQ, dK, dV = A.attn_bwd([T], [edits], Q, K, V_, dO, 0.35)
    q = torch.tensor(Q, requires_grad=True)
    k = torch.tensor(K, requires_grad=True)
    v = torch.tensor(V_, requires_grad=True)
    mask = torch.tensor(V.lifetime_mask(T, edits))
    o = F.scaled_dot_product_attention(
        q.permute(1, 0, 2), k.permute(1, 0, 2).repeat_interleave(2, 0),
        v.permute(1, 0, 2).repeat_interleave(2, 0), attn_mask=mask, scale=0.35)
    (o.permute(1, 0, 2) * torch.tensor(dO)).sum().backward()
    np.testing.assert_allclose(dQ, q.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dK, k.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dV, v.grad.numpy(), rtol=1e-10, atol=1e-12)
    # key-sampled variant agrees with the full backward
    keys = [0, 7, 31, 49]
    dk, dv = A.attn_bwd_keys([T], [edits], Q, K, V_, dO, 0.35, 1, keys)
    np.testing.assert_allclose(dk, dK[keys, 1], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(dv, dV[keys, 1], rtol=1e-11, atol=1e-13)


def test_backward_finite_differences():
    T, Dh = 24, 4
    edits = [(9, [(2, 4)]), (17, [(10, 12), (0, 1)])]
    Q, K, V_, dO = _inputs(T, 2, 1, Dh, 5)
    dQ, dK, dV = A.attn_bwd([T], [edits], Q, K, V_, dO, 0.5)

    def f(Q_, K_, V__):
        O, _ = A.attn_fwd([T], [edits], Q_, K_, V__, 0.5)
        return float((O * dO).sum())

    eps = 1e-6
    for arr, grad, idx in [(Q, dQ, (13, 1, 2)), (K, dK, (5, 0, 1)), (V_, dV, (16, 0, 3)),
                           (K, dK, (11, 0, 0))]:
        a1, a2 = arr.copy(), arr.copy()
        a1[idx] += eps
        a2[idx] -= eps
        args1 = [a1 if arr is x else x for x in (Q, K, V_)]
        args2 = [a2 if arr is x else x for x in (Q, K, V_)]
        fd = (f(*args1) - f(*args2)) / (2 * eps)
        assert abs(fd - grad[idx]) < 1e-6 * max(1.0, abs(fd))


def test_row_sampled_dq_matches_full():
    T, Hq, Hkv, Dh = 64, 4, 2, 8
    edits = _edits(T, 30, 3)
    Q, K, V_, dO = _inputs(T, Hq, Hkv, Dh, 30)
    dQ, _, _ = A.attn_bwd([T], [edits], Q, K, V_, dO, 0.4)
    rows = [0, 63, 20, 41]
    got = A.attn_bwd_rows([T], [edits], Q, K, V_, dO, 0.4, rows, [0, 3])
    np.testing.assert_allclose(got, dQ[rows][:, [0, 3]], rtol=1e-11, atol=1e-13)


def test_row_sampled_kv_contributions_sum_to_full():
    """The per-row dK / dV contributions (``with_kv``, which the CPU baseline
    times per sampled row) add up over a partition of the rows and all heads
    to the full backward's dK / dV, and their dQ is unchanged."""
    T, Hq, Hkv, Dh = 64, 4, 2, 8
    edits = _edits(T, 31, 3)
    Q, K, V_, dO = _inputs(T, Hq, Hkv, Dh, 31)
    dQ, dK, dV = A.attn_bwd([T], [edits], Q, K, V_, dO, 0.4)
    parts = [np.arange(0, T, 3), np.arange(1, T, 3), np.arange(2, T, 3)]
    sk, sv = np.zeros_like(dK), np.zeros_like(dV)
    for rows in parts:
        dq, dk, dv = A.attn_bwd_rows([T], [edits], Q, K, V_, dO, 0.4, rows, list(range(Hq)), with_kv=True)
        np.testing.assert_allclose(dq, dQ[rows], rtol=1e-11, atol=1e-13)
        sk += dk
        sv += dv
    np.testing.assert_allclose(sk, dK, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(sv, dV, rtol=1e-10, atol=1e-12)
