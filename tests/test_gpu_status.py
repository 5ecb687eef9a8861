"""Failure detection on the GPU without a GPU fault: a bounded device-side
wait that runs out is reported as MW_ETIMEOUT through a status word, the
context stays usable, and the LM-head status check is clean after real work."""

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

MW_OK, MW_ETIMEOUT = 0, 6


def test_wait_timeout_is_reported_and_context_survives():
    import paper_2609_00865_gb300 as mw
    status = torch.zeros(8, dtype=torch.int32, device="cuda")
    # a wait on a barrier nothing arrives on, given up after 20 ms
    st = mw.mw_selftest_wait_timeout(20_000_000, status)
    assert st == MW_ETIMEOUT
    s = status.cpu().numpy()
    assert s[1] == 1 and s[2] == 999
    # the context is still usable: a real visibility build and a status check
    rec = synth.config_record(1)
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    torch.cuda.synchronize()
    vis.check_status()
    # and the self-test is repeatable
    assert mw.mw_selftest_wait_timeout(1_000_000, status) == MW_ETIMEOUT


def test_selftest_rejects_bad_limits():
    import paper_2609_00865_gb300 as mw
    status = torch.zeros(8, dtype=torch.int32, device="cuda")
    assert mw.mw_selftest_wait_timeout(0, status) == 1          # MW_EINVAL
    assert mw.mw_selftest_wait_timeout(2_000_000_000, status) == 1


@pytest.mark.parametrize("d", [512, 1536])
def test_logprob_status_clean_after_fwd_bwd(d):
    import paper_2609_00865_gb300 as mw
    N, V = 640, 4096
    g = torch.Generator(device="cuda").manual_seed(d)
    H = torch.randn(N, d, device="cuda", generator=g).to(torch.bfloat16)
    W = (0.02 * torch.randn(V, d, device="cuda", generator=g)).to(torch.bfloat16)
    tg = torch.randint(0, V, (N,), device="cuda", generator=g, dtype=torch.int32)
    rows = torch.tensor(np.arange(0, N, 2), dtype=torch.int32, device="cuda")
    M = rows.numel()
    lp_old = torch.full((M,), -8.0, device="cuda")
    adv = torch.randn(M, device="cuda", generator=g)
    out = mw.logprob_loss_fwd(H, W, tg, rows, lp_old, adv, 0.2, 0.2)
    mw.mw_logprob_check_status(H, W, rows, out["ws"])
    dH, dW = mw.logprob_loss_bwd(H, W, tg, rows, out["lse"], out["ws"])
    mw.mw_logprob_check_status(H, W, rows, out["ws"])
    assert torch.isfinite(dH.float()).all() and torch.isfinite(dW).all()
