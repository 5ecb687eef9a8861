"""Reading of stacked layers (App. G branch-replicated packing): where a
single physical copy per token stops being exact, and the packed
per-branch computation that stays exact."""

import numpy as np
import pytest
import torch

from oracle import multilayer as ML
from oracle import visibility as V

EDITS = [(20, [(3, 9)]), (35, [(12, 18), (22, 25)]), (50, [(1, 3), (30, 40)])]
T = 64


def _x(seed, T=T):
    return np.random.default_rng(seed).standard_normal((T, 2, 8))


def test_one_layer_single_copy_is_exact():
    """One layer: the physical-union mask equals the per-branch computation
    (§4.3 Theorem "materialization equivalence")."""
    X = _x(1)
    np.testing.assert_allclose(ML.physical_union(T, EDITS, X, 0.3, 1), ML.per_branch(T, EDITS, X, 0.3, 1),
                               rtol=1e-11, atol=1e-12)


def test_two_layers_single_copy_differs_after_an_eviction():
    """Two layers: rows of the first segment and rows whose branch keeps every
    earlier key agree; rows whose branch holds trunk tokens that saw a
    since-evicted key differ."""
    X = _x(2)
    a = ML.physical_union(T, EDITS, X, 0.3, 2)
    b = ML.per_branch(T, EDITS, X, 0.3, 2)
    J1 = EDITS[0][0]
    np.testing.assert_allclose(a[:J1], b[:J1], rtol=1e-11, atol=1e-12)
    diff = np.abs(a - b).max(axis=(1, 2))
    assert (diff[J1:] > 1e-6).all()


def test_two_layers_without_edits_agree():
    X = _x(3)
    np.testing.assert_allclose(ML.physical_union(T, [], X, 0.3, 2), ML.per_branch(T, [], X, 0.3, 2),
                               rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("layers", [1, 2, 3])
def test_packed_branches_equal_per_branch(layers):
    X = _x(4)
    np.testing.assert_allclose(ML.packed_branches(T, EDITS, X, 0.3, layers), ML.per_branch(T, EDITS, X, 0.3, layers),
                               rtol=1e-11, atol=1e-12)


def test_per_branch_two_layers_against_sdpa():
    """The per-branch stack through torch's SDPA on each compact sequence
    (causal, float64), layer by layer."""
    X = _x(5)
    got = ML.per_branch(T, EDITS, X, 0.3, 2)
    for lo, hi, view in V.live_views(T, EDITS):
        h = torch.from_numpy(X[np.asarray(view)]).transpose(0, 1)
        for _ in range(2):
            h = h + torch.nn.functional.scaled_dot_product_attention(h, h, h, is_causal=True, scale=0.3)
        np.testing.assert_allclose(got[lo:hi], h.transpose(0, 1)[len(view) - (hi - lo):].numpy(),
                                   rtol=1e-11, atol=1e-12)
