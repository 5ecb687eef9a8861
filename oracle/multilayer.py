"""Oracle: stacked attention layers under compressed views (reading of
App. G "branch-replicated packing"), float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

A test model of L attention layers with identity projections and residuals:
h_0 = X, and layer l computes h_l = h_{l-1} + attn(q = k = v = h_{l-1}) (one
head group, Hq = Hkv). Two ways to run it on an edited rollout:

* ``per_branch`` -- LogitTree (§4.1): every segment's live view is its own
  compact sequence, and *every* token of it (the trunk included) is
  recomputed through all L layers inside that branch; a segment's rows are
  scored from their branch. This is what the policy computed at rollout
  time (the live context is re-read after each edit).
* ``physical_union`` -- each physical token computed once, at every layer,
  under its own segment's view (the single-copy 4D mask applied layer by
  layer).

At one layer they agree exactly (Theorem "materialization equivalence",
§4.3: the keys are the given inputs). From the second layer on, a trunk
token's layer-1 state inside branch s sees only the keys that survived to s,
while its single physical copy saw the keys of its own segment; wherever an
edit evicted a key before it, they differ. The exact multi-layer step is
therefore the per-branch one, which ``packed_branches`` computes a third
way: all branches' compact sequences concatenated into one sequence under a
block-diagonal causal mask (the paper's branch-replicated packing).
"""

import numpy as np

from .visibility import dense_mask, live_views


def _softmax_attn(h, mask, scale):
    """attn(q = k = v = h) with boolean mask [rows, keys] (row sees key)."""
    s = np.einsum("ihd,jhd->hij", h, h) * scale
    s = np.where(mask[None], s, -np.inf)
    m = s.max(axis=2, keepdims=True)
    p = np.exp(s - m)
    p /= p.sum(axis=2, keepdims=True)
    return np.einsum("hij,jhd->ihd", p, h)


def per_branch(T, edits, X, scale, layers):
    """Output of the last layer for every physical row, each row taken from
    its own segment's branch (the branch's compact sequence run through all
    layers). ``X`` [T, H, Dh]."""
    X = np.asarray(X, dtype=np.float64)
    out = np.zeros_like(X)
    for lo, hi, view in live_views(T, edits):
        h = X[np.asarray(view)]
        causal = np.tril(np.ones((len(view), len(view)), dtype=bool))
        for _ in range(layers):
            h = h + _softmax_attn(h, causal, scale)
        out[lo:hi] = h[len(view) - (hi - lo):]
    return out


def physical_union(T, edits, X, scale, layers):
    """Every physical token once per layer, under its own segment's view."""
    h = np.asarray(X, dtype=np.float64)
    mask = dense_mask(T, edits)
    for _ in range(layers):
        h = h + _softmax_attn(h, mask, scale)
    return h


def packed_branches(T, edits, X, scale, layers):
    """``per_branch`` as one packed sequence: the branches' compact
    sequences back to back under a block-diagonal causal mask."""
    X = np.asarray(X, dtype=np.float64)
    views = live_views(T, edits)
    idx = np.concatenate([np.asarray(v) for _, _, v in views])
    n = idx.size
    block = np.zeros((n, n), dtype=bool)
    o = 0
    for _, _, v in views:
        block[o: o + len(v), o: o + len(v)] = np.tril(np.ones((len(v), len(v)), dtype=bool))
        o += len(v)
    h = X[idx]
    for _ in range(layers):
        h = h + _softmax_attn(h, block, scale)
    out = np.zeros_like(X)
    o = 0
    for lo, hi, v in views:
        out[lo:hi] = h[o + len(v) - (hi - lo): o + len(v)]
        o += len(v)
    return out
