"""A two-layer step over branch-replicated packing (App. G), from one
visibility build of the record: pack each segment's live view (the compact
maps), run both layers' masked attention over the packed branches (one build
of the packed record, reused by both layers), score each segment's rows from
its own branch, and sum the packed copies' gradients per token. Checked
against the per-branch (LogitTree) stack computed by torch's float64 SDPA with
autograd on the CPU, equal to ``oracle.multilayer.per_branch`` (pinned in
``test_oracle_multilayer``)."""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, assert_rel, np64
from oracle.visibility import live_views

pytestmark = pytest.mark.gpu


def _reference(seqlens, edits, X, G, scale, layers=2):
    """Per-branch stack (h_l = h_{l-1} + attn(q = k = v = h_{l-1}), causal
    over each branch's compact sequence), the segments' rows taken from their
    own branch; returns (out [T], dX [T]) for the loss sum(out * G)."""
    x = X.detach().double().clone().requires_grad_(True)
    outs = torch.zeros_like(x)
    base = 0
    for T, e in zip(seqlens, edits):
        for lo, hi, view in live_views(T, e):
            h = x[torch.tensor(view, dtype=torch.int64) + base].transpose(0, 1)
            for _ in range(layers):
                h = h + torch.nn.functional.scaled_dot_product_attention(h, h, h, is_causal=True, scale=scale)
            outs[base + lo: base + hi] = h.transpose(0, 1)[len(view) - (hi - lo):]
        base += T
    (outs * G.double()).sum().backward()
    return outs.detach().numpy(), x.grad.numpy()


def _gpu_two_layers(seqlens, edits, X, G, scale):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    lens = mw.branch_lengths(vis)
    vis_p = mw.build_visibility(lens, [[] for _ in lens])        # the packed branches: one build, both layers
    n = sum(lens)
    h0 = mw.branch_pack(vis, X.cuda(), n)
    O1, L1 = mw.masked_attn_fwd(vis_p, h0, h0, h0, scale)
    h1 = h0 + O1
    O2, L2 = mw.masked_attn_fwd(vis_p, h1, h1, h1, scale)
    h2 = h1 + O2
    # each segment's rows are the tail of its branch
    tails, rows, o, base, s = [], [], 0, 0, 0
    for T, e in zip(seqlens, edits):
        bounds = [0] + [J for J, _ in e] + [T]
        for lo, hi in zip(bounds[:-1], bounds[1:]):
            tails.extend(range(o + lens[s] - (hi - lo), o + lens[s]))
            rows.extend(range(base + lo, base + hi))
            o += lens[s]
            s += 1
        base += T
    tails = torch.tensor(tails, dtype=torch.int64, device="cuda")
    rows = torch.tensor(rows, dtype=torch.int64, device="cuda")
    out = torch.empty_like(X.cuda())
    out[rows] = h2[tails]
    # backward: the upstream gradient sits on the tails; q = k = v = h, so a
    # layer passes on dh + dQ + dK + dV
    g2 = torch.zeros_like(h2)
    g2[tails] = G.cuda().to(h2.dtype)[rows]
    dQ, dK, dV = mw.masked_attn_bwd(vis_p, h1, h1, h1, O2, g2, L2, scale)
    g1 = g2 + dQ + dK + dV
    dQ, dK, dV = mw.masked_attn_bwd(vis_p, h0, h0, h0, O1, g1, L1, scale)
    g0 = g1 + dQ + dK + dV
    dX = mw.branch_unpack_add(vis, g0)
    torch.cuda.synchronize()
    vis_p.check_status()
    return out, dX


def _record(seed):
    rng = np.random.default_rng(seed)
    seqlens = [500, 340]
    edits = []
    for T in seqlens:
        Js = sorted(rng.choice(np.arange(40, T), size=3, replace=False).tolist())
        e = []
        for J in Js:
            a = int(rng.integers(0, J - 1))
            e.append((J, [(a, min(J, a + int(rng.integers(5, 90))))]))
        edits.append(e)
    return seqlens, edits


def test_two_layers_fp32():
    seqlens, edits = _record(1)
    T = sum(seqlens)
    X = 0.5 * synth.normal((T, 2, 64), 501)
    G = synth.normal((T, 2, 64), 502)
    out, dX = _gpu_two_layers(seqlens, edits, X, G, 0.125)
    out_r, dX_r = _reference(seqlens, edits, X, G, 0.125)
    assert_rel(np64(out), out_r, 1e-4, "out")
    assert_rel(np64(dX), dX_r, 1e-4, "dX")


def test_two_layers_bf16_tensor_cores():
    seqlens, edits = _record(2)
    T = sum(seqlens)
    X = (0.5 * synth.normal((T, 4, 128), 511)).to(torch.bfloat16)
    G = synth.normal((T, 4, 128), 512).to(torch.bfloat16)
    out, dX = _gpu_two_layers(seqlens, edits, X, G, 128 ** -0.5)
    out_r, dX_r = _reference(seqlens, edits, X, G, 128 ** -0.5)
    assert_maxabs(np64(out), out_r, 5e-2, "out")     # two bf16 layers and residuals
    assert_grad_bf16(np64(dX), dX_r, "dX")


def test_pack_and_unpack_are_adjoint():
    """unpack_add sums exactly the copies pack made: <pack(X), Y> = <X, unpack_add(Y)>."""
    import paper_2609_00865_gb300 as mw
    seqlens, edits = _record(3)
    vis = mw.build_visibility(seqlens, edits)
    n = sum(mw.branch_lengths(vis))
    X = synth.normal((sum(seqlens), 8), 521).cuda()
    Y = synth.normal((n, 8), 522).cuda()
    lhs = float((mw.branch_pack(vis, X, n).double() * Y.double()).sum())
    rhs = float((X.double() * mw.branch_unpack_add(vis, Y).double()).sum())
    assert abs(lhs - rhs) <= 1e-5 * max(1.0, abs(lhs))      # float32 sums of up to a few copies
