"""Pins of the SDCC oracle (§5; App. B Def. "trajectory tree"; App. F.1).

Diverging rows and final-walk prefixes against the paper's running example
(App. B.4 Table "running-prefixes"), two independent formulations of
divergence, the teacher-prefix reconstruction against the live views, the
forward KL against a closed form and autograd, and the schedule of lambda.
"""

import json
import os

import numpy as np
import pytest
import torch

from oracle import sdcc as S
from oracle import visibility as V

HERE = os.path.dirname(__file__)


def _golden():
    with open(os.path.join(HERE, "golden", "running_example.json")) as f:
        g = json.load(f)
    edits = [(J, [tuple(s) for s in spans]) for J, spans in g["edits"]]
    return g, g["tokens"], edits


def _random_edits(rng, T, overlap=False):
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
        if overlap and edits:
            spans.append(edits[-1][1][0])   # evict an earlier edit's span again
        edits.append((int(J), spans))
    return edits


def test_running_example_final_walk_prefixes():
    g, tok, edits = _golden()
    T = len(tok)
    for leaf, names in g["final_walk_prefix"].items():
        row = tok.index(leaf) - 1
        assert S.walk_prefix(T, edits, row) == [0] + [tok.index(n) for n in names], leaf


def test_running_example_diverging_rows():
    """The table's divergence column: y6, y7 by y5; y9, y10 by y8; y12 by y11;
    y_ans re-converges after the last junction."""
    g, tok, edits = _golden()
    T = len(tok)
    div = S.diverging_rows(T, edits)
    for leaf, by in g["diverges_by"].items():
        row = tok.index(leaf) - 1
        assert div[row] == bool(by), leaf
        extra = set(S.live_prefix(T, edits, row)) - set(S.walk_prefix(T, edits, row))
        assert extra == {tok.index(n) for n in by}, leaf
    # rows whose prefixes precede every evicted span, and rows at or after the
    # last junction, never diverge (App. B)
    first_evicted = min(a for _, spans in edits for a, _ in spans)
    assert not div[:first_evicted].any()
    assert not div[edits[-1][0]:].any()


@pytest.mark.parametrize("seed", range(6))
def test_diverging_rows_two_formulations(seed):
    rng = np.random.default_rng(400 + seed)
    T = int(rng.integers(30, 150))
    edits = _random_edits(rng, T, overlap=seed % 2 == 1)
    np.testing.assert_array_equal(S.diverging_rows(T, edits), S.diverging_rows_from_lifetimes(T, edits))


@pytest.mark.parametrize("seed", range(6))
def test_teacher_reconstruction_equals_live_prefix(seed):
    """Eq. "teacher-reconstruction" rebuilds exactly the prefix the token was
    decoded from (overlapping spans included for odd seeds)."""
    rng = np.random.default_rng(500 + seed)
    T = int(rng.integers(30, 150))
    edits = _random_edits(rng, T, overlap=seed % 2 == 1)
    for r in range(T):
        assert S.teacher_prefix(T, edits, r) == S.live_prefix(T, edits, r), r


def test_running_example_teacher_prefix_single_span():
    """The common case of Eq. "teacher-reconstruction" for y6: trunk
    [s, y1..y4] + re-inserted span [y5] + empty suffix."""
    _, tok, edits = _golden()
    row = tok.index("y6") - 1
    assert S.teacher_prefix(len(tok), edits, row) == [tok.index(n) for n in ("s", "y1", "y2", "y3", "y4", "y5")]


def test_forward_kl_two_classes_closed_form():
    """V = 2 with logits (0, x): the distributions are Bernoulli(sigmoid(x)),
    whose KL is p log(p/q) + (1-p) log((1-p)/(1-q))."""
    W = np.array([[0.0], [1.0]])
    xt = np.array([[0.7], [-2.0], [3.0]])
    xs = np.array([[-0.4], [-2.0], [0.5]])
    kl, _, _ = S.forward_kl(xt, xs, W)
    p = 1.0 / (1.0 + np.exp(-xt[:, 0]))
    q = 1.0 / (1.0 + np.exp(-xs[:, 0]))
    want = p * np.log(p / q) + (1 - p) * np.log((1 - p) / (1 - q))
    np.testing.assert_allclose(kl, want, rtol=1e-12, atol=1e-15)


def test_forward_kl_nonnegative_and_zero_on_equal_rows():
    rng = np.random.default_rng(6)
    W = rng.standard_normal((50, 8))
    H = rng.standard_normal((5, 8))
    kl, dh, dW = S.forward_kl(H, H, W)
    np.testing.assert_allclose(kl, 0.0, atol=1e-12)
    np.testing.assert_allclose(dh, 0.0, atol=1e-12)
    np.testing.assert_allclose(dW, 0.0, atol=1e-12)
    kl2, _, _ = S.forward_kl(H, rng.standard_normal((5, 8)), W)
    assert (kl2 > 0).all()
    # forward, not reverse: swapping teacher and student changes the value
    kl3, _, _ = S.forward_kl(rng.standard_normal((5, 8)), H, W)
    kl4, _, _ = S.forward_kl(H, rng.standard_normal((5, 8)), W)
    assert not np.allclose(kl3, kl4)


def test_forward_kl_gradients_equal_autograd_with_stopped_teacher():
    rng = np.random.default_rng(7)
    M, d, Vv = 6, 5, 40
    HT = rng.standard_normal((M, d))
    HS = rng.standard_normal((M, d))
    W = rng.standard_normal((Vv, d)) * 0.5
    kl, dHS, dW = S.forward_kl(HT, HS, W)
    hs = torch.from_numpy(HS).requires_grad_()
    w = torch.from_numpy(W).requires_grad_()
    lt = torch.log_softmax(torch.from_numpy(HT) @ w.detach().T, dim=1)   # teacher: stop-gradient
    ls = torch.log_softmax(hs @ w.T, dim=1)
    loss = (lt.exp() * (lt - ls)).sum()
    loss.backward()
    np.testing.assert_allclose(kl.sum(), loss.item(), rtol=1e-12)
    np.testing.assert_allclose(dHS, hs.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dW, w.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_sdcc_penalty_is_leaf_gated():
    rng = np.random.default_rng(8)
    T, d, Vv = 20, 4, 30
    HT, HS, W = rng.standard_normal((T, d)), rng.standard_normal((T, d)), rng.standard_normal((Vv, d))
    none = np.zeros(T, dtype=bool)
    pen, dHS, dW = S.sdcc_penalty(HT, HS, W, none, 0.1)
    assert pen == 0.0 and not dHS.any() and not dW.any()
    some = np.zeros(T, dtype=bool)
    some[[3, 7, 8]] = True
    pen0, _, _ = S.sdcc_penalty(HT, HS, W, some, 0.0)
    assert pen0 == 0.0
    pen, dHS, dW = S.sdcc_penalty(HT, HS, W, some, 0.1)
    kl, _, _ = S.forward_kl(HT[[3, 7, 8]], HS[[3, 7, 8]], W)
    assert abs(pen - 0.1 * kl.sum()) < 1e-12
    assert not dHS[~some].any() and dHS[some].any()


def test_lambda_ramp_schedule():
    """App. F.1: linear from 0 to 0.1 over the first 20% of steps, then flat."""
    assert S.lambda_ramp(0, 1000) == 0.0
    assert abs(S.lambda_ramp(100, 1000) - 0.05) < 1e-15
    assert abs(S.lambda_ramp(200, 1000) - 0.1) < 1e-15
    assert S.lambda_ramp(900, 1000) == 0.1
    assert S.lambda_ramp(10, 0) == 0.1


@pytest.mark.parametrize("seed", range(3))
def test_walk_scoring_drifts_exactly_on_diverging_rows(seed):
    """Eq. "logdiff" between scoring on the final compressed walk
    (Naive-Compressed) and scoring under the live views (the exact methods),
    one attention layer + LM head: a row's log-prob moves iff the row
    diverges, since a non-diverging row attends to the same set of keys in
    both (no positional encoding)."""
    from oracle import attention as A
    from oracle import logprob as LP
    rng = np.random.default_rng(600 + seed)
    T, Dh, Vv = 90, 8, 50
    edits = _random_edits(rng, T)
    Q = rng.standard_normal((T, 1, Dh))
    K = rng.standard_normal((T, 1, Dh))
    Vx = rng.standard_normal((T, 1, Dh))
    W = rng.standard_normal((Vv, Dh))
    targets = rng.integers(0, Vv, T)
    live, _ = A.attn_fwd([T], [edits], Q, K, Vx, 0.4)
    walk = S.final_walk(T, edits)
    wo, _ = A.attn_fwd([len(walk)], [[]], Q[walk], K[walk], Vx[walk], 0.4)
    where = {j: n for n, j in enumerate(walk)}
    # the student predicts y_(r+1) from the walk row of the last survivor <= r
    rows = [r for r in range(T) if S.walk_prefix(T, edits, r)]
    stud = np.stack([wo[where[S.walk_prefix(T, edits, r)[-1]], 0] for r in rows])
    lp_live, _ = LP.logprob(live[:, 0], W, targets, np.array(rows))
    lp_walk, _ = LP.logprob(stud, W, np.asarray(targets)[rows], np.arange(len(rows)))
    div = S.diverging_rows(T, edits)[rows]
    drift = np.abs(lp_live - lp_walk)
    assert (drift[~div] < 1e-12).all()
    assert (drift[div] > 1e-9).all()
    assert abs(LP.logdiff(lp_live, lp_walk) - drift.mean()) < 1e-15
    assert LP.logdiff([], []) == 0.0


def _torch_objective(T, edits, Q, K, Vx, W, targets, loss_rows, lp_old, adv, lam, scale):
    """The same objective through torch: the teacher from dense attention
    under the lifetime mask, the student from causal SDPA over the surviving
    positions, torch log-softmax and KL."""
    q, k, v, w = (torch.from_numpy(np.asarray(x, dtype=np.float64)) for x in (Q, K, Vx, W))
    walk = S.final_walk(T, edits)
    mask = torch.from_numpy(V.lifetime_mask(T, edits))
    st = torch.nn.functional.scaled_dot_product_attention(
        q[walk].transpose(0, 1), k[walk].transpose(0, 1), v[walk].transpose(0, 1), is_causal=True,
        scale=scale).transpose(0, 1).reshape(len(walk), -1)
    te = torch.nn.functional.scaled_dot_product_attention(
        q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1), attn_mask=mask, scale=scale
    ).transpose(0, 1).reshape(T, -1)
    where = {j: n for n, j in enumerate(walk)}
    rows = [r for r in loss_rows if r + 1 < T and (r + 1) in where]      # surviving leaves
    pred = [where[r + 1] - 1 for r in rows]                              # the walk row before each
    sel = [list(loss_rows).index(r) for r in rows]
    ls = torch.log_softmax(st @ w.T, dim=1)
    lp = ls[pred, torch.from_numpy(np.asarray(targets)[rows])]
    ratio = torch.exp(lp - torch.from_numpy(np.asarray(lp_old)[sel]))
    a = torch.from_numpy(np.asarray(adv)[sel])
    task = -torch.minimum(ratio * a, ratio.clamp(0.8, 1.28) * a).mean()
    pen = torch.zeros((), dtype=torch.float64)
    div = S.diverging_rows(T, edits)
    for r, pr in zip(rows, pred):
        if div[r]:
            lt = torch.log_softmax(te[r] @ w.T, dim=0)
            pen = pen + (lt.exp() * (lt - ls[pr])).sum()
    return float(task + lam * pen), float(task), float(lam * pen)


@pytest.mark.parametrize("seed", range(3))
def test_sdcc_objective_matches_an_independent_composition(seed):
    rng = np.random.default_rng(700 + seed)
    T, H, Dh, Vv = 70, 2, 4, 40
    edits = _random_edits(rng, T)
    Q, K, Vx = (rng.standard_normal((T, H, Dh)) for _ in range(3))
    W = rng.standard_normal((Vv, H * Dh)) * 0.5
    targets = rng.integers(0, Vv, T)
    loss_rows = np.sort(rng.choice(T, 40, replace=False))
    lp_old = rng.standard_normal(40) * 0.1 - 3.5
    adv = rng.standard_normal(40)
    got = S.sdcc_objective(T, edits, Q, K, Vx, W, targets, loss_rows, lp_old, adv, 0.1, 0.5)
    want = _torch_objective(T, edits, Q, K, Vx, W, targets, loss_rows, lp_old, adv, 0.1, 0.5)
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)
    assert got[2] > 0
    # lambda = 0 is Naive-Compressed exactly
    z = S.sdcc_objective(T, edits, Q, K, Vx, W, targets, loss_rows, lp_old, adv, 0.0, 0.5)
    assert z[0] == z[1] == got[1] and z[2] == 0.0


def test_sdcc_objective_without_edits_is_the_task_loss():
    rng = np.random.default_rng(710)
    T = 30
    Q, K, Vx = (rng.standard_normal((T, 1, 4)) for _ in range(3))
    W = rng.standard_normal((20, 4))
    rows = np.arange(T)
    obj, task, pen = S.sdcc_objective(T, [], Q, K, Vx, W, rng.integers(0, 20, T), rows,
                                      np.full(T, -3.0), rng.standard_normal(T), 0.1, 0.5)
    assert pen == 0.0 and obj == task


def test_forward_kl_dw_vocab_matches_full():
    """The sampled-vocabulary dW equals the full dW's rows."""
    rng = np.random.default_rng(31)
    HT, HS, W = rng.standard_normal((7, 16)), rng.standard_normal((7, 16)), 0.4 * rng.standard_normal((50, 16))
    _, _, dW = S.forward_kl(HT, HS, W)
    vocab = np.array([0, 3, 17, 49])
    np.testing.assert_allclose(S.forward_kl_dw_vocab(HT, HS, W, vocab), dW[vocab], rtol=1e-12, atol=1e-14)
