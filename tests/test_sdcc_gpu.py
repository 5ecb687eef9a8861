"""GPU diverging rows of SDCC (§5; App. B Def. "trajectory tree") vs the
oracle, bit for bit."""

import json
import os

import numpy as np
import pytest
import torch

from helpers import assert_grad_bf16, assert_maxabs, assert_rel, np64
from oracle import sdcc as OS

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(__file__)


def _check(seqlens, edits):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    got = mw.diverging_rows(vis)
    torch.cuda.synchronize()
    want = np.concatenate([OS.diverging_rows(T, e) for T, e in zip(seqlens, edits)]).astype(np.uint8)
    np.testing.assert_array_equal(got.cpu().numpy()[: want.size], want)
    return want


def test_running_example():
    with open(os.path.join(HERE, "golden", "running_example.json")) as f:
        g = json.load(f)
    edits = [(J, [tuple(s) for s in spans]) for J, spans in g["edits"]]
    want = _check([len(g["tokens"])], [edits])
    assert want.sum() == 5   # y6, y7, y9, y10, y12


def test_packed_ragged_record_with_overlaps():
    """Several trajectories (an empty one, one longer than a 1024-row scan
    chunk), overlapping spans evicted twice."""
    seqlens = [1, 0, 300, 2500, 129]
    edits = [[], [], [(150, [(20, 140)]), (280, [(150, 260), (20, 40)])],
             [(1100, [(10, 900)]), (2000, [(1000, 1900), (5, 8)]), (2400, [(2001, 2300)])],
             [(128, [(5, 127)])]]
    _check(seqlens, edits)


def _check_walk(seqlens, edits):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    wi, sr, wl = mw.final_walk(vis)
    torch.cuda.synchronize()
    want_wi, want_sr, want_wl = [], [], []
    for T, e in zip(seqlens, edits):
        walk = OS.final_walk(T, e) if T else []
        w = np.full(T, -1)
        w[walk] = np.arange(len(walk))
        srow = OS.student_rows(T, e) if T else {}
        want_wi.append(w)
        want_sr.append([srow.get(r, -1) for r in range(T)])
        want_wl.append(len(walk))
    n = sum(seqlens)
    np.testing.assert_array_equal(wi.cpu().numpy()[:n], np.concatenate(want_wi))
    np.testing.assert_array_equal(sr.cpu().numpy()[:n], np.concatenate([np.asarray(x, dtype=np.int64)
                                                                         for x in want_sr]))
    np.testing.assert_array_equal(wl.cpu().numpy()[: len(seqlens)], want_wl)


def test_final_walk_running_example_and_ragged_record():
    """Walk indices, student rows and walk lengths, bit for bit (§5)."""
    with open(os.path.join(HERE, "golden", "running_example.json")) as f:
        g = json.load(f)
    edits = [(J, [tuple(s) for s in spans]) for J, spans in g["edits"]]
    _check_walk([len(g["tokens"])], [edits])
    _check_walk([1, 0, 300, 2500, 129],
                [[], [], [(150, [(20, 140)]), (280, [(150, 260), (20, 40)])],
                 [(1100, [(10, 900)]), (2000, [(1000, 1900), (5, 8)]), (2400, [(2001, 2300)])],
                 [(128, [(5, 127)])]])


def _kl_case(M, N_T, N_S, d, V, seed, dtype):
    rng = np.random.default_rng(seed)
    HT = torch.from_numpy(rng.standard_normal((N_T, d))).to(dtype)
    HS = torch.from_numpy(rng.standard_normal((N_S, d))).to(dtype)
    W = torch.from_numpy(0.3 * rng.standard_normal((V, d))).to(dtype)
    rows_T = torch.from_numpy(rng.integers(0, N_T, M).astype(np.int32))
    rows_S = torch.from_numpy(rng.permutation(N_S)[:M].astype(np.int32))   # distinct
    return HT, HS, W, rows_T, rows_S


def _kl_run(HT, HS, W, rows_T, rows_S, lam, dloss):
    import paper_2609_00865_gb300 as mw
    dev = [t.cuda() for t in (HT, rows_T, HS, rows_S, W)]
    kl, loss, ws = mw.forward_kl_fwd(*dev, lam=lam)
    dHS, dW = mw.forward_kl_bwd(*dev, ws, lam=lam, dloss=dloss)
    torch.cuda.synchronize()
    return kl, loss, dHS, dW


def _assert_kl_bf16(kl, HT, HS, W, rows_T, rows_S):
    """The tensor-core KL takes E_pT[z_S] = h_S . sum_v pT_v W_v with the
    weights pT rounded to bf16 (relative error <= 2^-9 each), so per pair
    |dKL| <= 2^-9 sum_v pT_v |zT_v - zS_v| plus float32 rounding; the bar is
    twice that bound plus 1e-3, with the logits from a plain float64 product."""
    from oracle import sdcc as OSd
    rt, rs = rows_T.numpy().astype(np.int64), rows_S.numpy().astype(np.int64)
    klr, _, _ = OSd.forward_kl(np64(HT)[rt], np64(HS)[rs], np64(W))
    zt, zs = np64(HT)[rt] @ np64(W).T, np64(HS)[rs] @ np64(W).T
    pt = np.exp(zt - zt.max(axis=1, keepdims=True))
    pt /= pt.sum(axis=1, keepdims=True)
    bound = 2.0 ** -8 * (pt * np.abs(zt - zs)).sum(axis=1) + 1e-3
    err = np.abs(np64(kl) - klr)
    assert (err <= bound).all(), f"kl: worst err / bound {float((err / bound).max()):.3g}"


def _kl_ref(HT, HS, W, rows_T, rows_S, lam, dloss):
    from oracle import sdcc as OSd
    rt, rs = rows_T.numpy().astype(np.int64), rows_S.numpy().astype(np.int64)
    kl, dh, dW = OSd.forward_kl(np64(HT)[rt], np64(HS)[rs], np64(W))
    dHS = np.zeros(tuple(HS.shape))
    dHS[rs] = lam * dloss * dh
    return kl, lam * kl.sum(), dHS, lam * dloss * dW


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_forward_kl_matches_oracle(dtype):
    """Forward KL(teacher || student) over a 3,001-column vocabulary (a ragged
    last tile of 256 columns), 37 pairs (ragged blocks of 8, 16 and 32),
    teacher rows drawn with repeats, student rows distinct; both gradients
    of the student."""
    d = 64 if dtype == torch.float32 else 128
    case = _kl_case(37, 50, 45, d, 3001, 7, dtype)
    kl, loss, dHS, dW = _kl_run(*case, lam=0.1, dloss=1.3)
    klr, lossr, dHSr, dWr = _kl_ref(*case, lam=0.1, dloss=1.3)
    if dtype == torch.float32:      # CUDA cores, float32 throughout
        assert_rel(np64(kl), klr, 1e-4, "kl")
        assert_rel(np64(loss), [lossr], 1e-4, "loss")
        assert_rel(np64(dHS), dHSr, 1e-4, "dHS")
        assert_rel(np64(dW), dWr, 1e-4, "dW")
    else:                           # tensor cores: bf16 softmax weights in E
        _assert_kl_bf16(kl, *case)
        assert abs(float(loss.item()) - lossr) <= 1e-3 * abs(lossr)
        assert_grad_bf16(np64(dHS), dHSr, "dHS")
        assert_grad_bf16(np64(dW), dWr, "dW")
    untouched = np.setdiff1d(np.arange(case[1].shape[0]), case[4].numpy())
    assert not np64(dHS)[untouched].any()


def test_forward_kl_of_equal_rows_is_zero():
    HT, _, W, _, _ = _kl_case(10, 10, 10, 32, 500, 9, torch.float32)
    rows = torch.arange(10, dtype=torch.int32)
    kl, loss, dHS, dW = _kl_run(HT, HT, W, rows, rows, 1.0, 1.0)
    assert_maxabs(np64(kl), np.zeros(10), 1e-5, "kl")
    assert_maxabs(np64(dHS), np.zeros(tuple(HT.shape)), 1e-6, "dHS")
    assert_maxabs(np64(dW), np.zeros(tuple(W.shape)), 1e-6, "dW")


def test_forward_kl_tc_equal_rows_is_exactly_zero():
    """Tensor-core path: a student equal to its teacher gives KL 0, dHS 0 and
    dW 0 bit for bit (both passes form the same numbers; the two dW passes
    cancel exactly)."""
    HT, _, W, _, _ = _kl_case(40, 40, 40, 128, 1000, 19, torch.bfloat16)
    rows = torch.arange(40, dtype=torch.int32)
    kl, loss, dHS, dW = _kl_run(HT, HT, W, rows, rows, 0.5, 1.0)
    assert not np64(kl).any() and not np64(dHS).any() and not np64(dW).any()


@pytest.mark.parametrize("d,V", [(1536, 151936), (3584, 152064)])
def test_forward_kl_tc_workload_sizes(d, V):
    """The hidden sizes and vocabularies of the log-prob and 7B-shaped
    workloads (W ~ N(0, 0.02^2), rows ~ N(0, 1)), 512 pairs with repeated
    teacher rows: kl per pair and the loss, dHS on every student row, dW on
    sampled vocabulary rows."""
    from oracle import sdcc as OSd
    M = 512
    g = torch.Generator().manual_seed(d)
    HT = torch.randn(600, d, generator=g).to(torch.bfloat16)
    HS = torch.randn(700, d, generator=g).to(torch.bfloat16)
    W = (0.02 * torch.randn(V, d, generator=g)).to(torch.bfloat16)
    rng = np.random.default_rng(d)
    rows_T = torch.from_numpy(rng.integers(0, 600, M).astype(np.int32))
    rows_S = torch.from_numpy(rng.permutation(700)[:M].astype(np.int32))
    kl, loss, dHS, dW = _kl_run(HT, HS, W, rows_T, rows_S, 0.1, 1.0)
    rt, rs = rows_T.numpy().astype(np.int64), rows_S.numpy().astype(np.int64)
    klr, dhr, _ = OSd.forward_kl(np64(HT)[rt], np64(HS)[rs], np64(W))
    _assert_kl_bf16(kl, HT, HS, W, rows_T, rows_S)
    lossr = 0.1 * klr.sum()
    assert abs(float(loss.item()) - lossr) <= 1e-3 * abs(lossr)
    assert_grad_bf16(np64(dHS)[rs], 0.1 * dhr, "dHS")
    vocab = np.unique(np.concatenate([[0, V - 1], rng.integers(0, V, 62)]))
    dWr = OSd.forward_kl_dw_vocab(np64(HT)[rt], np64(HS)[rs], np64(W), vocab)
    assert_grad_bf16(np64(dW)[vocab], 0.1 * dWr, "dW (sampled vocabulary rows)")


def test_forward_kl_without_pairs():
    HT, HS, W, _, _ = _kl_case(0, 5, 6, 32, 300, 10, torch.float32)
    empty = torch.zeros(0, dtype=torch.int32)
    kl, loss, dHS, dW = _kl_run(HT, HS, W, empty, empty, 0.1, 1.0)
    assert float(loss.item()) == 0.0
    assert not dHS.any() and not dW.any()


@pytest.mark.parametrize("M", [0, 1, 1000, 70001])
def test_logdiff_matches_oracle(M):
    """Eq. "logdiff" over M tokens (one block of 1,024 threads: 69 strides
    each at M = 70,001)."""
    import paper_2609_00865_gb300 as mw
    from oracle import logprob as OL
    rng = np.random.default_rng(M)
    a = torch.from_numpy(rng.standard_normal(M).astype(np.float32))
    b = torch.from_numpy((rng.standard_normal(M) * 0.1).astype(np.float32)) + a
    got = mw.logdiff(a.cuda(), b.cuda())
    torch.cuda.synchronize()
    want = OL.logdiff(np64(a), np64(b))
    assert abs(float(got.item()) - want) <= 1e-5 * want   # exact 0 without tokens


def test_sdcc_objective_end_to_end():
    """SDCC's objective for one layer (Eq. "soft_loss") assembled from the GPU
    entry points: masked attention under the live views (teacher), the final
    walk and causal attention over it (student), the clipped task loss on the
    leaves that survive on the walk, the diverging rows and the forward KL;
    equal to oracle.sdcc.sdcc_objective in float32."""
    import paper_2609_00865_gb300 as mw
    rng = np.random.default_rng(77)
    T, H, Dh, Vv = 300, 2, 64, 500
    edits = [(90, [(10, 40)]), (150, [(50, 80), (100, 120)]), (230, [(5, 9), (160, 200)])]
    Q, K, Vx = (torch.from_numpy(rng.standard_normal((T, H, Dh)).astype(np.float32)) for _ in range(3))
    W = torch.from_numpy((0.05 * rng.standard_normal((Vv, H * Dh))).astype(np.float32))
    targets = rng.integers(0, Vv, T).astype(np.int32)
    loss_rows = np.sort(rng.choice(T - 1, 150, replace=False))
    lp_old = rng.standard_normal(150) * 0.1 - 6.0
    adv = rng.standard_normal(150)
    lam, scale = 0.1, Dh ** -0.5
    vis = mw.build_visibility([T], [edits])
    Ot, _ = mw.masked_attn_fwd(vis, Q.cuda(), K.cuda(), Vx.cuda(), scale)            # teacher
    wi, sr, wl = mw.final_walk(vis)
    div = mw.diverging_rows(vis)
    torch.cuda.synchronize()
    wi, sr, div, n = wi.cpu().numpy()[:T], sr.cpu().numpy()[:T], div.cpu().numpy()[:T] > 0, int(wl.cpu()[0])
    walk = np.argsort(np.where(wi >= 0, wi, T + np.arange(T)))[:n]                    # walk order
    vis_w = mw.build_visibility([n], [[]])
    Os, _ = mw.masked_attn_fwd(vis_w, Q[walk].cuda(), K[walk].cuda(), Vx[walk].cuda(), scale)   # student
    leaves = [i for i, r in enumerate(loss_rows) if wi[r + 1] >= 0]
    srows = np.array([sr[loss_rows[i]] for i in leaves], dtype=np.int32)
    tg = np.zeros(n, dtype=np.int32)
    tg[srows] = targets[loss_rows[leaves]]
    out = mw.logprob_loss_fwd(Os.reshape(n, -1).contiguous(), W.cuda(), torch.from_numpy(tg).cuda(),
                              torch.from_numpy(srows).cuda(),
                              torch.from_numpy(lp_old[leaves].astype(np.float32)).cuda(),
                              torch.from_numpy(adv[leaves].astype(np.float32)).cuda(), 0.2, 0.28)
    pairs = [(loss_rows[i], sr[loss_rows[i]]) for i in leaves if div[loss_rows[i]]]
    assert pairs
    rt = torch.tensor([a for a, _ in pairs], dtype=torch.int32).cuda()
    rs = torch.tensor([b for _, b in pairs], dtype=torch.int32).cuda()
    _, pen, _ = mw.forward_kl_fwd(Ot.reshape(T, -1).contiguous(), rt, Os.reshape(n, -1).contiguous(), rs,
                                  W.cuda(), lam=lam)
    torch.cuda.synchronize()
    _, task, penalty = OS.sdcc_objective(T, edits, np64(Q), np64(K), np64(Vx), np64(W), targets, loss_rows,
                                         lp_old, adv, lam, scale)
    assert abs(float(out["loss"].item()) - task) <= 1e-4 * abs(task) + 1e-6
    assert abs(float(pen.item()) - penalty) <= 1e-4 * abs(penalty)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_forward_kl_bwd_accumulates(dtype):
    """accumulate = 1 adds the KL's gradients to dHS / dW (the task loss's
    buffers in an SDCC step) and leaves rows without a pair alone: a second
    call doubles the first call's result."""
    import paper_2609_00865_gb300 as mw
    d = 64 if dtype == torch.float32 else 128
    HT, HS, W, rows_T, rows_S = (t.cuda() for t in _kl_case(21, 30, 28, d, 700, 23, dtype))
    kl, loss, ws = mw.forward_kl_fwd(HT, rows_T, HS, rows_S, W, lam=0.3)
    dHS = torch.full_like(HS, 0.0)
    dW = torch.zeros(W.shape[0], d, dtype=torch.float32, device="cuda")
    mw.mw_forward_kl_bwd(HT, rows_T, HS, rows_S, W, ws, dHS, dW, 0.3, 1.0, False)
    first = (dHS.float().clone(), dW.clone())
    mw.mw_forward_kl_bwd(HT, rows_T, HS, rows_S, W, ws, dHS, dW, 0.3, 1.0, True)
    torch.cuda.synchronize()
    if dtype == torch.float32:
        assert torch.allclose(dHS, 2 * first[0], rtol=1e-6, atol=0)
    else:
        assert torch.allclose(dHS.float(), 2 * first[0], rtol=8e-3, atol=0)   # one more bf16 rounding
    # tensor cores: dW is the sum of two nearly cancelling passes, added in
    # another order the second time, so it doubles up to rounding of the parts
    tol = 1e-6 if dtype == torch.float32 else 1e-3
    assert torch.allclose(dW, 2 * first[1], rtol=tol, atol=tol * float(first[1].abs().max()))
    untouched = np.setdiff1d(np.arange(HS.shape[0]), rows_S.cpu().numpy())
    assert not dHS[torch.from_numpy(untouched).cuda()].float().any()
