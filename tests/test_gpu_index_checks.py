"""Device-side checks of the index arrays no host check sees.

The loss rows, their targets and SDCC's pair rows are device arrays. A row
outside [0, N) or a target outside [0, Vocab) must not be followed: the
kernels skip it, the status check reports MW_EDEVICE, and the rows that are
in range keep their results. Every access these cases make is guarded in the
kernels (the gathers and the dH writes read each index once through a range
check), so the cases run no out-of-range access.
"""

import numpy as np
import pytest
import torch

import synth
from oracle import logprob as OL

pytestmark = pytest.mark.gpu

MW_EDEVICE = 7


def _lm_case(N, d, V, dtype, seed):
    H = synth.normal((N, d), seed).to(dtype).cuda()
    W = synth.normal((V, d), seed + 1, std=0.02).to(dtype).cuda()
    targets = synth.uniform_int(N, V, seed + 2).cuda()
    rows = np.arange(1, N, 3, dtype=np.int32)
    M = len(rows)
    adv = synth.normal((M,), seed + 3).cuda()
    lp_old = torch.full((M,), -8.0, dtype=torch.float32).cuda()
    return H, W, targets, rows, adv, lp_old


def _fwd_bwd(H, W, targets, rows, adv, lp_old):
    import paper_2609_00865_gb300 as mw
    r = torch.tensor(rows, dtype=torch.int32).cuda()
    out = mw.logprob_loss_fwd(H, W, targets, r, lp_old, adv, 0.2, 0.28)
    st_fwd = _status(lambda: mw.mw_logprob_check_status(H, W, r, out["ws"]))
    dH, dW = mw.logprob_loss_bwd(H, W, targets, r, out["lse"], out["ws"])
    st_bwd = _status(lambda: mw.mw_logprob_check_status(H, W, r, out["ws"]))
    return out, dH, st_fwd, st_bwd


def _status(call):
    import paper_2609_00865_gb300 as mw
    try:
        call()
        return 0
    except mw.MWError as e:
        return e.status


# (N, d, V, dtype): the tensor-core path (bf16, d a multiple of 64) and the
# CUDA-core path (float32)
LM_CASES = [(600, 256, 3001, torch.bfloat16), (300, 64, 1000, torch.float32)]


@pytest.mark.parametrize("N,d,V,dtype", LM_CASES)
@pytest.mark.parametrize("bad", ["row_past_end", "row_negative", "target_past_end", "target_negative"])
def test_logprob_index_out_of_range_is_reported_and_skipped(N, d, V, dtype, bad):
    H, W, targets, rows, adv, lp_old = _lm_case(N, d, V, dtype, 91)
    clean, dH_clean, st0, st1 = _fwd_bwd(H, W, targets, rows, adv, lp_old)
    assert (st0, st1) == (0, 0)

    k = 5   # the loss row that goes bad
    rows_bad, targets_bad = rows.copy(), targets.clone()
    if bad == "row_past_end":
        rows_bad[k] = N
    elif bad == "row_negative":
        rows_bad[k] = -7
    elif bad == "target_past_end":
        targets_bad[rows[k]] = V
    else:
        targets_bad[rows[k]] = -2
    out, dH, st_fwd, st_bwd = _fwd_bwd(H, W, targets_bad, rows_bad, adv, lp_old)
    assert st_fwd == MW_EDEVICE and st_bwd == MW_EDEVICE

    keep = np.ones(len(rows), bool)
    keep[k] = False
    keep_t = torch.tensor(keep).cuda()
    # every other row's log-prob is unchanged: rows are computed independently
    assert torch.allclose(out["lp"][keep_t], clean["lp"][keep_t], rtol=0, atol=1e-5)
    assert torch.allclose(out["lse"][keep_t], clean["lse"][keep_t], rtol=0, atol=1e-5)
    # the skipped row's dH row is not written (stays 0); rows outside the loss stay 0
    if bad.startswith("row"):
        other = np.setdiff1d(np.arange(N), rows_bad[keep])
    else:
        other = np.setdiff1d(np.arange(N), rows[keep])
    assert torch.all(dH[torch.tensor(other).cuda()].float() == 0)
    torch.cuda.synchronize()

    # the context is intact and the status word resets with the next call
    again, _, st2, st3 = _fwd_bwd(H, W, targets, rows, adv, lp_old)
    assert (st2, st3) == (0, 0)
    assert torch.allclose(again["lp"], clean["lp"], rtol=0, atol=1e-6)


def test_logprob_oracle_agrees_on_rows_in_range():
    """The in-range rows of a call with one bad row match the oracle."""
    N, d, V = 600, 256, 3001
    H, W, targets, rows, adv, lp_old = _lm_case(N, d, V, torch.bfloat16, 93)
    rows_bad = rows.copy()
    rows_bad[3] = N + 100
    out, _, st_fwd, _ = _fwd_bwd(H, W, targets, rows_bad, adv, lp_old)
    assert st_fwd == MW_EDEVICE
    keep = np.ones(len(rows), bool)
    keep[3] = False
    f64 = lambda t: t.detach().to("cpu", torch.float64).numpy()
    lp_r, _ = OL.logprob(f64(H), f64(W), targets.cpu().numpy(), rows[keep])
    assert np.abs(f64(out["lp"])[keep] - lp_r).max() <= 1e-2


@pytest.mark.parametrize("d,dtype", [(256, torch.bfloat16), (64, torch.float32)])
@pytest.mark.parametrize("side", ["teacher", "student"])
def test_forward_kl_row_out_of_range_is_reported(d, dtype, side):
    import paper_2609_00865_gb300 as mw
    N_T, N_S, V, M = 300, 200, 1500, 40
    HT = synth.normal((N_T, d), 95).to(dtype).cuda()
    HS = synth.normal((N_S, d), 96).to(dtype).cuda()
    W = synth.normal((V, d), 97, std=0.05).to(dtype).cuda()
    rT = torch.tensor(np.arange(0, 2 * M, 2), dtype=torch.int32).cuda()
    rS = torch.tensor(np.arange(3, 3 + M), dtype=torch.int32).cuda()
    kl0, _, ws0 = mw.forward_kl_fwd(HT, rT, HS, rS, W)
    assert _status(lambda: mw.forward_kl_check_status(rT, HT, W, ws0)) == 0

    bT, bS = rT.clone(), rS.clone()
    if side == "teacher":
        bT[7] = N_T
    else:
        bS[7] = -1
    kl, _, ws = mw.forward_kl_fwd(HT, bT, HS, bS, W)
    assert _status(lambda: mw.forward_kl_check_status(bT, HT, W, ws)) == MW_EDEVICE
    keep = torch.ones(M, dtype=torch.bool).cuda()
    keep[7] = False
    assert torch.allclose(kl[keep], kl0[keep], rtol=0, atol=1e-5)
    dHS, _ = mw.forward_kl_bwd(HT, bT, HS, bS, W, ws)
    # the status words hold the forward's report through the backward
    assert _status(lambda: mw.forward_kl_check_status(bT, HT, W, ws)) == MW_EDEVICE
    # student rows outside the pairs (and a student index out of range) get no gradient
    b = bS.cpu().numpy()
    untouched = np.setdiff1d(np.arange(N_S), b[(b >= 0) & (b < N_S)])
    assert torch.all(dHS[torch.tensor(untouched).cuda()].float() == 0)
