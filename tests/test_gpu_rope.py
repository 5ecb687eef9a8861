"""GPU row-wise logical positions and rotary masked attention vs the oracle.

§4.2 reassigns position ids per row so that the keys a row sees form a
gap-free sequence. The oracle computes that on each segment's compact
sequence (position = compact index); the CUDA path computes positions from
the view bits and reads keys rotated per segment.
"""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, assert_rel, np64
from oracle import attention as OA
from oracle import visibility as OV

pytestmark = pytest.mark.gpu

_TILE_EDGE = (
    [1, 127, 0, 128, 129, 300],
    [[], [(100, [(10, 40)])], [], [(64, [(0, 32)]), (120, [(70, 100)])], [(128, [(5, 127)])],
     [(150, [(20, 140)]), (280, [(150, 260)])]],
)


def _medium_record(seed):
    rng = np.random.default_rng(seed)
    seqlens = [700, 1000, 333]
    edits = []
    for T in seqlens:
        Js = sorted(rng.choice(np.arange(64, T), size=3, replace=False).tolist())
        e = []
        for J in Js:
            sp = []
            for _ in range(3):
                a = int(rng.integers(0, J - 1))
                sp.append((a, min(J, a + int(rng.integers(1, 120)))))
            e.append((J, sp))
        edits.append(e)
    return seqlens, edits


def _expected_positions(seqlens, edits):
    """Oracle positions in the library's layout: per trajectory, segment-major
    rows of 128 nt_b entries, -1 for non-members and the ragged tail."""
    out = []
    for T, e in zip(seqlens, edits):
        nt = (T + 127) // 128
        lp = OV.logical_positions(T, e)
        arr = np.full((lp.shape[0], nt * 128), -1, dtype=np.int64)
        arr[:, :T] = lp
        out.append(arr.reshape(-1))
    return np.concatenate(out) if out else np.zeros(0, np.int64)


def _tensors(T, Hq, Hkv, Dh, seed, dtype):
    Q = synth.normal((T, Hq, Dh), seed).to(dtype)
    K = synth.normal((T, Hkv, Dh), seed + 1).to(dtype)
    V = synth.normal((T, Hkv, Dh), seed + 2).to(dtype)
    dO = synth.normal((T, Hq, Dh), seed + 3).to(dtype)
    return Q, K, V, dO


@pytest.mark.parametrize("rec", ["edge", "medium"])
def test_logical_positions_bit_exact(rec):
    import paper_2609_00865_gb300 as mw
    seqlens, edits = _TILE_EDGE if rec == "edge" else _medium_record(3)
    vis = mw.build_visibility(seqlens, edits)
    pos = mw.logical_positions(vis)
    torch.cuda.synchronize()
    want = _expected_positions(seqlens, edits)
    got = pos.cpu().numpy()[: want.size]
    np.testing.assert_array_equal(got, want)


def test_rope_table_matches_float64():
    import paper_2609_00865_gb300 as mw
    n_pos, Dh, theta = 4096, 128, 1e6
    t = mw.rope_table(n_pos, Dh, theta).cpu().numpy().astype(np.float64)
    ang = np.arange(n_pos)[:, None] * theta ** (-2.0 * np.arange(Dh // 2) / Dh)[None, :]
    assert_maxabs(t[..., 0], np.cos(ang), 1e-7, "cos")
    assert_maxabs(t[..., 1], np.sin(ang), 1e-7, "sin")


# Dh 64: 16-byte vector kernel for both dtypes; 40: vectors for float32 only
# (half a bf16 row is 40 bytes); 36: element kernel for both
@pytest.mark.parametrize("Dh", [64, 40, 36])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_rope_rows_rotate_by_own_logical_position(dtype, Dh):
    import paper_2609_00865_gb300 as mw
    seqlens, edits = _medium_record(4)
    vis = mw.build_visibility(seqlens, edits)
    pos = mw.logical_positions(vis)
    table = mw.rope_table(mw.rope_n_pos(vis), Dh, 1e4)
    X = synth.normal((sum(seqlens), 3, Dh), 77).to(dtype)
    x = X.cuda()
    Y = mw.rope_rows(vis, pos, table, x)
    # own position of every row, from the oracle's views
    own = []
    for T, e in zip(seqlens, edits):
        lp = OV.logical_positions(T, e)
        seg = OV.segment_ids(T, e)
        own.append(lp[seg, np.arange(T)])
    own = np.concatenate(own)
    assert (own >= 0).all()
    ref = OA.rope(np64(X), own, 1e4)
    if dtype == torch.float32:
        assert_rel(np64(Y), ref, 1e-5, "Y")
    else:
        assert_maxabs(np64(Y), ref, 2e-2, "Y")
    # inverse, in place, undoes it
    mw.rope_rows(vis, pos, table, Y, inverse=True, out=Y)
    torch.cuda.synchronize()
    tol = 1e-5 if dtype == torch.float32 else 3e-2
    assert_maxabs(np64(Y), np64(X), tol * 8, "round trip")


def _run(seqlens, edits, Q, K, V, dO, scale, theta):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    pos = mw.logical_positions(vis)
    table = mw.rope_table(mw.rope_n_pos(vis), Q.shape[2], theta)
    q, k, v, do = (t.cuda() for t in (Q, K, V, dO))
    O, LSE = mw.masked_attn_rope_fwd(vis, pos, table, q, k, v, scale)
    dQ, dK, dV = mw.masked_attn_rope_bwd(vis, pos, table, q, k, v, O, do, LSE, scale)
    torch.cuda.synchronize()
    vis.check_status()
    return O, LSE, dQ, dK, dV


@pytest.mark.parametrize("Dh", [64, 128])
def test_rope_attention_fp32(Dh):
    seqlens, edits = _medium_record(5)
    Q, K, V, dO = _tensors(sum(seqlens), 8, 2, Dh, 121, torch.float32)
    scale, theta = Dh ** -0.5, 1e4
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale, theta)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale, rope_theta=theta)
    assert_rel(np64(O), Or, 1e-4, "O")
    assert_rel(np64(LSE), Lr, 1e-4, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale, rope_theta=theta)
    assert_rel(np64(dQ), dQr, 1e-4, "dQ")
    assert_rel(np64(dK), dKr, 1e-4, "dK")
    assert_rel(np64(dV), dVr, 1e-4, "dV")


def test_rope_attention_bf16_tile_edges():
    seqlens, edits = _TILE_EDGE
    Q, K, V, dO = _tensors(sum(seqlens), 6, 2, 128, 131, torch.bfloat16)
    scale, theta = 128 ** -0.5, 1e6
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale, theta)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale, rope_theta=theta)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale, rope_theta=theta)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


@pytest.mark.parametrize("Hq,Hkv", [(8, 2), (4, 4)])
def test_rope_attention_bf16_tensor_cores(Hq, Hkv):
    """bf16 with Dh 128 runs on the tensor-core kernels with segment key rows:
    junctions inside q-tiles (one CTA per segment of such a tile) and keys
    whose position differs between segments."""
    seqlens, edits = _medium_record(8)
    Q, K, V, dO = _tensors(sum(seqlens), Hq, Hkv, 128, 151 + Hq, torch.bfloat16)
    scale, theta = 128 ** -0.5, 1e6
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale, theta)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale, rope_theta=theta)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale, rope_theta=theta)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


def test_rope_attention_bf16_junctions_on_tile_edges():
    """Junctions at a tile's first row (128) and two and four rows into that
    tile (130, 132): three segments inside one q-tile."""
    seqlens = [700]
    edits = [[(128, [(0, 100)]), (130, [(101, 120)]), (132, [(5, 7)]), (300, [(129, 250)])]]
    Q, K, V, dO = _tensors(700, 4, 2, 128, 161, torch.bfloat16)
    scale, theta = 128 ** -0.5, 1e4
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale, theta)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale, rope_theta=theta)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale, rope_theta=theta)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


def test_rope_attention_bf16_head_dim_64():
    """bf16 with Dh 64 takes the CUDA-core kernels."""
    seqlens, edits = _medium_record(9)
    Q, K, V, dO = _tensors(sum(seqlens), 4, 2, 64, 171, torch.bfloat16)
    scale, theta = 64 ** -0.5, 1e4
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale, theta)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale, rope_theta=theta)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale, rope_theta=theta)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


def test_rope_later_edit_leaves_earlier_rows_unchanged():
    """Conditioning invariant (§3.3) with rotary positions: a junction added at
    row 600 changes neither the positions nor the outputs of rows before it."""
    T = 900
    base = [(200, [(20, 90)]), (400, [(210, 300)])]
    more = base + [(600, [(100, 399)])]
    Q, K, V, dO = _tensors(T, 4, 2, 64, 141, torch.float32)
    O1, L1, *_ = _run([T], [base], Q, K, V, dO, 0.125, 1e4)
    O2, L2, *_ = _run([T], [more], Q, K, V, dO, 0.125, 1e4)
    assert torch.equal(O1[:600], O2[:600])
    assert torch.equal(L1[:, :600], L2[:, :600])
    assert not torch.equal(O1[600:], O2[600:])

