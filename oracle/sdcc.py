"""Oracle: SDCC (self-distillation for conditioning consistency), float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

§5 (SDCC): the student is the policy on the final compressed walk (every
edit applied), the teacher the same policy, gradients stopped, on the live
prefix a token was decoded from; at every *diverging* leaf (its live prefix
differs from its final-walk prefix, App. B Def. "trajectory tree") the loss
adds lambda times the forward KL(teacher || student) of the next-token
distributions (Eq. "soft_loss"); lambda ramps linearly (App. F.1).

Conventions as in ``oracle.visibility``: 0-based physical positions, row r
predicts token r + 1, so the leaf y_(r+1) is scored by row r, and row r's
live prefix is its segment's view up to and including r.
"""

import numpy as np

from .visibility import NEVER, lifetimes, live_views, validate_edits


def final_walk(T, edits):
    """The final compressed walk: the positions no edit ever evicts, in order
    (§5: the replay trajectory that remains after all edits)."""
    validate_edits(T, edits)
    gone = set()
    for _, spans in edits:
        for a, b in spans:
            gone.update(range(a, b))
    return [j for j in range(T) if j not in gone]


def live_prefix(T, edits, r):
    """Row r's live prefix: the members of its segment's view up to r."""
    for lo, hi, view in live_views(T, edits):
        if lo <= r < hi:
            return [j for j in view if j <= r]
    raise IndexError(r)


def walk_prefix(T, edits, r):
    """Row r's prefix on the final compressed walk: the surviving positions
    up to r (the row's own token included only if it survives)."""
    return [j for j in final_walk(T, edits) if j <= r]


def diverging_rows(T, edits):
    """Rows whose live prefix differs from their final-walk prefix, read off
    the two lists literally (App. B Def. "trajectory tree": a node is
    diverging iff its leg and spine colourings disagree)."""
    return np.array([live_prefix(T, edits, r) != walk_prefix(T, edits, r) for r in range(T)], dtype=bool)


def diverging_rows_from_lifetimes(T, edits):
    """Second formulation: row r diverges iff some key it saw is evicted
    later, i.e. there is j <= r with r < omega(j) < NEVER (an eviction that
    fires after r reaches back into r's prefix)."""
    om = lifetimes(T, edits)
    out = np.zeros(T, dtype=bool)
    for r in range(T):
        js = om[: r + 1]
        out[r] = bool(np.any((js > r) & (js < NEVER)))
    return out


def teacher_prefix(T, edits, r):
    """Eq. "teacher-reconstruction": the final walk's prefix with every span
    active at r put back at its original slot. A position is active when an
    edit that fires after r evicts it and no edit at or before r already had
    (overlapping spans); positions past r are not part of the prefix. The
    physical order is the original insertion order."""
    walk = final_walk(T, edits)
    before, after = set(), set()
    for J, spans in edits:
        for a, b in spans:
            (after if J > r else before).update(j for j in range(a, b) if j <= r)
    return sorted(set(j for j in walk if j <= r) | (after - before))


def lambda_ramp(step, total_steps, lam_max=0.1, warm_frac=0.2):
    """App. F.1: lambda rises linearly from 0 to ``lam_max`` over the first
    ``warm_frac`` of the update steps and stays there."""
    warm = warm_frac * total_steps
    if warm <= 0:
        return lam_max
    return lam_max * min(1.0, step / warm)


def _log_softmax(z):
    m = z.max(axis=1, keepdims=True)
    return z - m - np.log(np.exp(z - m).sum(axis=1, keepdims=True))


def forward_kl(HT, HS, W):
    """Forward KL(teacher || student) per row over the vocabulary, and its
    gradients with respect to the student (the teacher is stop-gradient).

    ``HT``, ``HS`` [M, d] teacher / student hidden rows, ``W`` [V, d]:
    z = h W^T, p = softmax(z), KL_m = sum_v pT (log pT - log pS).
    dKL_m / dzS = pS - pT, so dHS_m = (pS - pT)_m W and dW = (pS - pT)^T HS.
    Returns (kl [M], dHS [M, d], dW [V, d]) for the loss sum_m KL_m.
    """
    HT = np.asarray(HT, dtype=np.float64)
    HS = np.asarray(HS, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    lt = _log_softmax(HT @ W.T)
    ls = _log_softmax(HS @ W.T)
    pt = np.exp(lt)
    kl = (pt * (lt - ls)).sum(axis=1)
    dz = np.exp(ls) - pt
    return kl, dz @ W, dz.T @ HS


def forward_kl_dw_vocab(HT, HS, W, vocab):
    """``forward_kl``'s dW for a few vocabulary rows only (sampled checks on
    big heads): each row's full softmax of both sides, then
    ``dW[v] = sum_m (pS - pT)_{m,v} HS_m`` for the selected v."""
    HT = np.asarray(HT, dtype=np.float64)
    HS = np.asarray(HS, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    vocab = np.asarray(vocab, dtype=np.int64)
    lt = _log_softmax(HT @ W.T)[:, vocab]
    ls = _log_softmax(HS @ W.T)[:, vocab]
    return (np.exp(ls) - np.exp(lt)).T @ HS


def sdcc_penalty(HT, HS, W, diverging, lam):
    """The SDCC term of Eq. "soft_loss" for one trajectory: ``lam`` times the
    sum of the forward KLs over the diverging rows (leaf-gated: rows that do
    not diverge contribute nothing). ``HT`` / ``HS`` hold one teacher /
    student row per physical row. Returns (penalty, dHS, dW)."""
    HT = np.asarray(HT, dtype=np.float64)
    HS = np.asarray(HS, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    idx = np.nonzero(np.asarray(diverging, dtype=bool))[0]
    dHS = np.zeros_like(HS)
    if idx.size == 0 or lam == 0.0:
        return 0.0, dHS, np.zeros_like(W)
    kl, dh, dW = forward_kl(HT[idx], HS[idx], W)
    dHS[idx] = lam * dh
    return lam * float(kl.sum()), dHS, lam * dW


def student_rows(T, edits):
    """For every row r with a non-empty final-walk prefix, the walk index of
    the last surviving position <= r. When the leaf y_(r+1) survives on the
    walk this is the walk row just before it, whose output is the student's
    prediction of it (§5: f(H_comp) at the leaf's place). Returns
    {r: walk index}."""
    walk = final_walk(T, edits)
    where = {j: n for n, j in enumerate(walk)}
    out = {}
    for r in range(T):
        pre = walk_prefix(T, edits, r)
        if pre:
            out[r] = where[pre[-1]]
    return out


def sdcc_objective(T, edits, Q, K, V, W, targets, loss_rows, lp_old, adv, lam, scale, eps_lo=0.2, eps_hi=0.28):
    """Eq. "soft_loss" for one trajectory and one attention layer feeding the
    LM head (hidden row = attention output, heads concatenated):

      student  attention over the final compressed walk (causal, no edits);
               a leaf y_(r+1) (loss row r) is a token of the walk only if it
               survives every edit, and the walk row before it predicts it
               (``student_rows``); task loss = the clipped surrogate over those
               leaves (Naive-Compressed);
      teacher  attention under each row's live view (the exact 4D mask),
               gradients stopped;
      penalty  lam * sum over the diverging ones of those leaves of
               KL(teacher || student) (§5: the set C of diverging leaves).

    Returns (objective, task, penalty). Plain composition of the oracle's own
    attention, log-prob and KL functions, in their definitions' order.
    """
    from .attention import attn_fwd
    from .logprob import logprob, policy_loss
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    walk = final_walk(T, edits)
    where = {j: n for n, j in enumerate(walk)}
    Os, _ = attn_fwd([len(walk)], [[]], Q[walk], K[walk], V[walk], scale)
    Hs = Os.reshape(len(walk), -1)
    Ot, _ = attn_fwd([T], [edits], Q, K, V, scale)
    Ht = Ot.reshape(T, -1)
    srow = student_rows(T, edits)
    leaves = [r for r in loss_rows if r + 1 < T and (r + 1) in where]
    # the walk row before leaf y_(r+1) predicts it; its target is y_(r+1)'s id
    tg = np.zeros(len(walk), dtype=np.int64)
    for r in leaves:
        tg[srow[r]] = np.asarray(targets)[r]
    lp, _ = logprob(Hs, W, tg, np.array([srow[r] for r in leaves], dtype=np.int64))
    sel = [list(loss_rows).index(r) for r in leaves]
    _, _, task, _ = policy_loss(lp, np.asarray(lp_old)[sel], np.asarray(adv)[sel], eps_lo, eps_hi)
    div = diverging_rows(T, edits)
    pairs = [(r, srow[r]) for r in leaves if div[r]]
    penalty = 0.0
    if pairs and lam != 0.0:
        kl, _, _ = forward_kl(Ht[[a for a, _ in pairs]], Hs[[b for _, b in pairs]], W)
        penalty = lam * float(kl.sum())
    return task + penalty, task, penalty
