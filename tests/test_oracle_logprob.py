"""Pins for the LM-head log-prob / clipped-loss oracle (CPU only, float64)."""

import numpy as np
import pytest
import torch

from oracle import logprob as LP


def _case(N, d, V, M, seed, wstd=0.5):
    g = np.random.default_rng(seed)
    H = g.standard_normal((N, d))
    W = g.standard_normal((V, d)) * wstd
    targets = g.integers(0, V, N)
    rows = np.sort(g.permutation(N)[:M])
    return H, W, targets, rows


def test_logprob_equals_log_softmax():
    H, W, t, rows = _case(40, 16, 300, 25, 0)
    lp, lse = LP.logprob(H, W, t, rows)
    z = torch.tensor(H[rows]) @ torch.tensor(W).T
    ref = torch.log_softmax(z, dim=-1)
    np.testing.assert_allclose(lp, ref[torch.arange(25), torch.tensor(t[rows])].numpy(), rtol=1e-12)
    np.testing.assert_allclose(lse, torch.logsumexp(z, -1).numpy(), rtol=1e-13)


def test_zero_weights_give_uniform():
    H, W, t, rows = _case(10, 8, 1000, 10, 1)
    lp, lse = LP.logprob(H, np.zeros_like(W), t, rows)
    np.testing.assert_allclose(lp, -np.log(1000.0), rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse, np.log(1000.0), rtol=0, atol=1e-14)


def test_ratio_one_closed_form():
    g = np.random.default_rng(2)
    lp = g.standard_normal(50)
    adv = g.standard_normal(50)
    ratio, per, loss, grad = LP.policy_loss(lp, lp, adv, 0.2, 0.28)
    np.testing.assert_array_equal(ratio, 1.0)
    assert loss == pytest.approx(-adv.mean(), rel=1e-14)
    np.testing.assert_allclose(grad, -adv / 50, rtol=1e-14)


def test_clipped_region_has_zero_gradient():
    lp_old = np.zeros(4)
    lp = np.log(np.array([1.5, 1.5, 0.5, 0.5]))   # far outside [0.8, 1.2]
    adv = np.array([1.0, -1.0, 1.0, -1.0])
    ratio, per, loss, g = LP.policy_loss(lp, lp_old, adv, 0.2, 0.2)
    # A>0, rho>1+eps and A<0, rho<1-eps are flat; the other two are not
    np.testing.assert_allclose(g, [0.0, 1.5 / 4, -0.5 / 4, 0.0], rtol=1e-14)
    np.testing.assert_allclose(per, [-1.2, 1.5, -0.5, 0.8], rtol=1e-14)


def test_policy_loss_gradient_equals_autograd():
    g = np.random.default_rng(3)
    lp = g.standard_normal(200) * 0.3
    lp_old = lp + g.standard_normal(200) * 0.3
    adv = g.standard_normal(200)
    _, _, loss, grad = LP.policy_loss(lp, lp_old, adv, 0.2, 0.28, dloss=1.7)
    x = torch.tensor(lp, requires_grad=True)
    r = torch.exp(x - torch.tensor(lp_old))
    a = torch.tensor(adv)
    L = -torch.minimum(r * a, torch.clamp(r, 0.8, 1.28) * a).mean()
    (1.7 * L).backward()
    assert loss == pytest.approx(L.item(), rel=1e-14)
    np.testing.assert_allclose(grad, x.grad.numpy(), rtol=1e-12, atol=1e-15)


def test_kl_k3_is_unbiased_for_the_exact_kl():
    """Averaged under pi_theta, the per-token estimate equals KL(pi_theta ||
    pi_ref) computed directly from the two distributions; it is zero when
    the policies agree and ~d^2 / 2 for a small log-ratio d."""
    rng = np.random.default_rng(11)
    for _ in range(5):
        V = int(rng.integers(2, 40))
        lp = np.log(rng.dirichlet(np.ones(V)))
        lp_ref = np.log(rng.dirichlet(np.ones(V)))
        k3, _ = LP.kl_k3(lp, lp_ref)
        p = np.exp(lp)
        exact_kl = float(np.sum(p * (lp - lp_ref)))
        assert float(np.sum(p * k3)) == pytest.approx(exact_kl, rel=1e-12, abs=1e-14)
    k3, dk3 = LP.kl_k3(np.array([-1.5, -0.2]), np.array([-1.5, -0.2]))
    assert (k3 == 0).all() and (dk3 == 0).all()
    d = 1e-4
    k3, _ = LP.kl_k3(np.array([0.0]), np.array([d]))
    assert k3[0] == pytest.approx(d * d / 2, rel=1e-3)


def test_policy_loss_with_kl_gradient_equals_autograd():
    g = np.random.default_rng(5)
    lp = g.standard_normal(150) * 0.3 - 2.0
    lp_old = lp + g.standard_normal(150) * 0.3
    lp_ref = lp + g.standard_normal(150) * 0.5
    adv = g.standard_normal(150)
    _, _, loss, grad = LP.policy_loss(lp, lp_old, adv, 0.2, 0.28, dloss=0.9, lp_ref=lp_ref, beta=0.3)
    x = torch.tensor(lp, requires_grad=True)
    r = torch.exp(x - torch.tensor(lp_old))
    a = torch.tensor(adv)
    ratio_ref = torch.exp(torch.tensor(lp_ref) - x)          # pi_ref / pi_theta
    kl = ratio_ref - torch.log(ratio_ref) - 1.0
    L = (-torch.minimum(r * a, torch.clamp(r, 0.8, 1.28) * a) + 0.3 * kl).mean()
    (0.9 * L).backward()
    assert loss == pytest.approx(L.item(), rel=1e-13)
    np.testing.assert_allclose(grad, x.grad.numpy(), rtol=1e-12, atol=1e-15)
    # beta = 0 or no reference: the plain clipped loss
    _, _, l0, g0 = LP.policy_loss(lp, lp_old, adv, 0.2, 0.28, lp_ref=lp_ref, beta=0.0)
    _, _, l1, g1 = LP.policy_loss(lp, lp_old, adv, 0.2, 0.28)
    assert l0 == l1 and (g0 == g1).all()


def test_backward_equals_autograd():
    N, d, V, M = 30, 12, 200, 17
    H, W, t, rows = _case(N, d, V, M, 4)
    g = np.random.default_rng(5)
    lp_old = g.standard_normal(M) * 0.05
    adv = g.standard_normal(M)
    lp, lse = LP.logprob(H, W, t, rows)
    lp_old = lp + lp_old
    _, _, loss, grad = LP.policy_loss(lp, lp_old, adv, 0.2, 0.2)
    dH, dW = LP.logprob_loss_bwd(H, W, t, rows, lse, grad)

    h = torch.tensor(H, requires_grad=True)
    w = torch.tensor(W, requires_grad=True)
    z = h[torch.tensor(rows)] @ w.T
    lpt = torch.log_softmax(z, -1)[torch.arange(M), torch.tensor(t[rows])]
    r = torch.exp(lpt - torch.tensor(lp_old))
    a = torch.tensor(adv)
    L = -torch.minimum(r * a, torch.clamp(r, 0.8, 1.2) * a).mean()
    L.backward()
    assert loss == pytest.approx(L.item(), rel=1e-13)
    np.testing.assert_allclose(dH, h.grad.numpy(), rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(dW, w.grad.numpy(), rtol=1e-10, atol=1e-14)
    notloss = np.setdiff1d(np.arange(N), rows)
    assert (dH[notloss] == 0).all()
    vocab = [0, 5, 199, int(t[rows[0]])]
    np.testing.assert_allclose(LP.logprob_loss_bwd_vocab(H, W, t, rows, lse, grad, vocab),
                               dW[vocab], rtol=1e-11, atol=1e-15)


def test_finite_difference_through_whole_head():
    N, d, V, M = 8, 5, 40, 6
    H, W, t, rows = _case(N, d, V, M, 6)
    g = np.random.default_rng(7)
    adv = g.standard_normal(M)
    lp0, _ = LP.logprob(H, W, t, rows)
    lp_old = lp0 + 0.05 * g.standard_normal(M)

    def L(H_, W_):
        lp, _ = LP.logprob(H_, W_, t, rows)
        return LP.policy_loss(lp, lp_old, adv, 0.2, 0.2)[2]

    lp, lse = LP.logprob(H, W, t, rows)
    grad = LP.policy_loss(lp, lp_old, adv, 0.2, 0.2)[3]
    dH, dW = LP.logprob_loss_bwd(H, W, t, rows, lse, grad)
    eps = 1e-6
    for arr, gr, idx in [(H, dH, (rows[2], 3)), (W, dW, (int(t[rows[1]]), 1)), (W, dW, (7, 4))]:
        a1, a2 = arr.copy(), arr.copy()
        a1[idx] += eps
        a2[idx] -= eps
        if arr is H:
            fd = (L(a1, W) - L(a2, W)) / (2 * eps)
        else:
            fd = (L(H, a1) - L(H, a2)) / (2 * eps)
        assert abs(fd - gr[idx]) < 1e-7
