"""Oracle: LM-head log-probabilities and the clipped policy loss, in float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

The importance ratio of App. B.4 ("Pitfall A, RL view") is
``rho_t = pi_theta(a_t | view) / pi_old(a_t | view)``, both under the live
view; the paper trains with GRPO/PPO clipping (§6.1 "Optimization"; App. F.1:
clip range 0.2 low / 0.28 high). The per-token surrogate is PPO's
``-min(rho A, clip(rho, 1-eps_lo, 1+eps_hi) A)``, averaged over the M
loss-carrying tokens (the logdiff average of Eq. 1 runs over the same set).

Layouts: ``H [N, d]`` hidden rows, ``W [V, d]`` LM-head weight (torch Linear
layout), ``targets [N]`` next-token ids by physical row, ``rows [M]`` the
physical rows that carry loss (distinct), ``lp_old, adv [M]``.

Arithmetic: the logit products and the softmax passes run on float64 CPU
tensors (torch, every host core); inputs and outputs are numpy arrays.
"""

import numpy as np
import torch

_ROW_CHUNK = 256


def _t(x):
    """float64 CPU tensor view of an array (copies only when it must)."""
    return torch.from_numpy(np.ascontiguousarray(np.asarray(x, dtype=np.float64)))


def _ix(x):
    return torch.from_numpy(np.asarray(x, dtype=np.int64))


def logits(H, W, rows):
    """``z[m, v] = sum_d H[rows[m], d] W[v, d]`` (small problems only)."""
    return (_t(H)[_ix(rows)] @ _t(W).T).numpy()


def logprob(H, W, targets, rows):
    """Per loss row: ``lse = log sum_v exp(z_v)``, ``lp = z_target - lse``.

    Rows are processed in chunks; each row is independent.
    """
    H, W = _t(H), _t(W)
    rows = np.asarray(rows, dtype=np.int64)
    tgt = _ix(np.asarray(targets, dtype=np.int64)[rows])
    lse = torch.empty(rows.size, dtype=torch.float64)
    lp = torch.empty(rows.size, dtype=torch.float64)
    for c0 in range(0, rows.size, _ROW_CHUNK):
        r = _ix(rows[c0 : c0 + _ROW_CHUNK])
        z = H[r] @ W.T
        m = z.amax(dim=1, keepdim=True)
        l = m[:, 0] + torch.log(torch.exp(z - m).sum(dim=1))
        lse[c0 : c0 + r.numel()] = l
        lp[c0 : c0 + r.numel()] = z[torch.arange(r.numel()), tgt[c0 : c0 + r.numel()]] - l
    return lp.numpy(), lse.numpy()


def kl_k3(lp, lp_ref):
    """Low-variance estimate of KL(pi_theta || pi_ref) per token (App. F.1 trains
    with a KL coefficient and "the low-variance estimator"; the paper gives no
    formula, and this is the standard one, k3): with ``d = lp_ref - lp``,
    ``k3 = exp(d) - d - 1`` (>= 0, zero iff d = 0) and ``dk3/dlp = 1 - exp(d)``.
    Returns ``(k3, dk3/dlp)``."""
    d = np.asarray(lp_ref, dtype=np.float64) - np.asarray(lp, dtype=np.float64)
    return np.expm1(d) - d, -np.expm1(d)


def policy_loss(lp, lp_old, adv, eps_lo, eps_hi, dloss=1.0, lp_ref=None, beta=0.0):
    """Ratio, clipped surrogate, mean loss and ``g_t = dL/dlp_t``.

    ``rho = exp(lp - lp_old)``; ``l_t = -min(rho A, clip(rho) A)``;
    ``L = mean_t l_t``. Differentiating the min case by case: the unclipped
    term is selected (gradient ``-A rho / M``) unless the clipped term is
    strictly smaller, which happens exactly when ``A > 0, rho > 1 + eps_hi``
    or ``A < 0, rho < 1 - eps_lo``; there the surrogate is flat in lp and the
    gradient is 0. At equality both terms coincide and the unclipped branch
    is used. ``dloss`` scales the gradient (upstream dL). With ``lp_ref`` and
    ``beta`` each token adds ``beta * k3`` (``kl_k3``) to its loss term and
    ``beta * dk3/dlp / M`` to ``g``.
    """
    lp = np.asarray(lp, dtype=np.float64)
    lp_old = np.asarray(lp_old, dtype=np.float64)
    adv = np.asarray(adv, dtype=np.float64)
    M = lp.size
    ratio = np.exp(lp - lp_old)
    unclipped = ratio * adv
    clipped = np.clip(ratio, 1.0 - eps_lo, 1.0 + eps_hi) * adv
    per_tok = -np.minimum(unclipped, clipped)
    loss = per_tok.mean() if M else 0.0
    flat = clipped < unclipped
    g = np.where(flat, 0.0, -adv * ratio) / max(M, 1) * dloss
    if lp_ref is not None and beta:
        k3, dk3 = kl_k3(lp, lp_ref)
        per_tok = per_tok + beta * k3
        loss = per_tok.mean() if M else 0.0
        g = g + beta * dk3 / max(M, 1) * dloss
    return ratio, per_tok, loss, g


def logprob_loss_bwd(H, W, targets, rows, lse, g, dh_rows=None):
    """Gradients of ``L`` with respect to ``H`` and ``W``.

    With ``lp_t = z_{t,tgt} - lse_t``, ``dlp_t/dz_{t,v} = 1[v = tgt] - p_{t,v}``
    where ``p = softmax(z_t)``, so ``dz_{t,v} = g_t (1[v = tgt] - p_{t,v})``;
    ``dH_t = sum_v dz_{t,v} W_v`` (zero on rows outside the loss) and
    ``dW_v = sum_t dz_{t,v} H_t``.

    ``dh_rows`` (optional, a subset of ``rows``) computes only those rows' dH
    and skips dW (returned as None): sampled checks on big heads.
    """
    H, W = _t(H), _t(W)
    rows = np.asarray(rows, dtype=np.int64)
    tgt_all = np.asarray(targets, dtype=np.int64)[rows]
    lse_all = np.asarray(lse, dtype=np.float64)
    g_all = np.asarray(g, dtype=np.float64)
    sel = np.arange(rows.size)
    if dh_rows is not None:
        sel = np.nonzero(np.isin(rows, np.asarray(dh_rows, dtype=np.int64)))[0]
    dH = torch.zeros_like(H)
    dW = None if dh_rows is not None else torch.zeros_like(W)
    for c0 in range(0, sel.size, _ROW_CHUNK):
        s = sel[c0 : c0 + _ROW_CHUNK]
        r = _ix(rows[s])
        z = H[r] @ W.T
        p = torch.exp(z - _t(lse_all[s])[:, None])
        onehot = torch.zeros_like(p)
        onehot[torch.arange(s.size), _ix(tgt_all[s])] = 1.0
        dz = _t(g_all[s])[:, None] * (onehot - p)
        dH[r] = dz @ W
        if dW is not None:
            dW += dz.T @ H[r]
    return dH.numpy(), (None if dW is None else dW.numpy())


def logprob_loss_bwd_vocab(H, W, targets, rows, lse, g, vocab):
    """``dW`` for a few vocabulary rows only (sampled checks on big heads)."""
    H = _t(H)
    Wv = _t(W)[_ix(vocab)]
    rows = np.asarray(rows, dtype=np.int64)
    tgt = np.asarray(targets, dtype=np.int64)[rows]
    vocab = np.asarray(vocab, dtype=np.int64)
    Hr = H[_ix(rows)]
    z = Hr @ Wv.T
    p = torch.exp(z - _t(lse)[:, None])
    onehot = _t((tgt[:, None] == vocab[None, :]).astype(np.float64))
    dz = _t(g)[:, None] * (onehot - p)
    return (dz.T @ Hr).numpy()


def logdiff(lp_train, lp_rollout):
    """Eq. "logdiff" (§3): the train-inference logits drift, the mean over
    the loss-carrying tokens of |log p(y_t | c_train) - log p(y_t | c_rollout)|
    under one set of weights. Returns 0 for no tokens."""
    a = np.asarray(lp_train, dtype=np.float64)
    b = np.asarray(lp_rollout, dtype=np.float64)
    if a.size == 0:
        return 0.0
    return float(np.abs(a - b).mean())

