"""The whole path chained as the step bench.py times: visibility -> masked
attention fwd -> H = O -> fused LM-head log-prob + clipped loss fwd/bwd ->
attention bwd with dO = dH. Checked against the oracle run on the same chain."""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, assert_rel, np64
from oracle import attention as OA
from oracle import logprob as OL

pytestmark = pytest.mark.gpu


def _gpu_chain(rec, Q, K, V, W, tg, rows, lp_old, adv, eps):
    import paper_2609_00865_gb300 as mw
    T, Hq, Dh = Q.shape
    scale = Dh ** -0.5
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    O, LSE = mw.masked_attn_fwd(vis, Q, K, V, scale)
    H = O.view(T, Hq * Dh)
    out = mw.logprob_loss_fwd(H, W, tg, rows, lp_old, adv, eps, eps)
    dH, dW = mw.logprob_loss_bwd(H, W, tg, rows, out["lse"], out["ws"])
    dQ, dK, dV = mw.masked_attn_bwd(vis, Q, K, V, O, dH.view(T, Hq, Dh), LSE, scale)
    torch.cuda.synchronize()
    vis.check_status()
    return O, out, dH, dW, dQ, dK, dV


def test_config1_chained_fp32():
    c = synth.CONFIGS[1]
    rec = synth.config_record(1)
    T, Hq, Hkv, Dh, V = rec.total, c["Hq"], c["Hkv"], c["Dh"], c["V"]
    Q = synth.normal((T, Hq, Dh), 81)
    K = synth.normal((T, Hkv, Dh), 82)
    Vv = synth.normal((T, Hkv, Dh), 83)
    W = synth.normal((V, Hq * Dh), 84, std=0.02)
    tg = synth.uniform_int(T, V, 85)
    rows = rec.loss_rows()
    M = len(rows)
    adv = synth.normal((M,), 86)
    scale = Dh ** -0.5
    # oracle chain
    Or, _ = OA.attn_fwd(rec.seqlens, rec.edits, np64(Q), np64(K), np64(Vv), scale)
    Hr = Or.reshape(T, Hq * Dh)
    lp_r, lse_r = OL.logprob(Hr, np64(W), tg.numpy(), rows)
    lp_old = torch.tensor(lp_r + np64(synth.normal((M,), 87, std=0.05)), dtype=torch.float32)
    ratio_r, _, loss_r, g_r = OL.policy_loss(lp_r, np64(lp_old), np64(adv), 0.2, 0.2)
    dHr, dWr = OL.logprob_loss_bwd(Hr, np64(W), tg.numpy(), rows, lse_r, g_r)
    dQr, dKr, dVr = OA.attn_bwd(rec.seqlens, rec.edits, np64(Q), np64(K), np64(Vv),
                                dHr.reshape(T, Hq, Dh), scale)
    dev = lambda t: t.cuda()
    O, out, dH, dW, dQ, dK, dV = _gpu_chain(rec, dev(Q), dev(K), dev(Vv), dev(W), dev(tg),
                                            torch.tensor(rows, dtype=torch.int32).cuda(), dev(lp_old),
                                            dev(adv), 0.2)
    assert_rel(np64(O), Or, 1e-4, "O")
    assert_rel(np64(out["lp"]), lp_r, 1e-4, "lp")
    assert abs(out["loss"].item() - loss_r) <= 1e-4 * max(abs(loss_r), 1e-6)
    assert_rel(np64(dH), dHr, 1e-4, "dH")
    assert_rel(np64(dW), dWr, 1e-4, "dW")
    assert_rel(np64(dQ), dQr, 1e-4, "dQ")
    assert_rel(np64(dK), dKr, 1e-4, "dK")
    assert_rel(np64(dV), dVr, 1e-4, "dV")


def test_config4_chained_sampled():
    """Full-size 7B-shaped layer step. For sampled loss rows the oracle chains
    its own attention output into its own LM head: lp, lse, and the dH row
    (which the GPU feeds back as dO)."""
    c = synth.CONFIGS[4]
    rec = synth.config_record(4)
    T, Hq, Hkv, Dh, V = rec.total, c["Hq"], c["Hkv"], c["Dh"], c["V"]
    d = Hq * Dh
    g = torch.Generator(device="cuda").manual_seed(404)
    Q = torch.randn(T, Hq, Dh, device="cuda", generator=g).to(torch.bfloat16)
    K = torch.randn(T, Hkv, Dh, device="cuda", generator=g).to(torch.bfloat16)
    Vv = torch.randn(T, Hkv, Dh, device="cuda", generator=g).to(torch.bfloat16)
    W = (0.02 * torch.randn(V, d, device="cuda", generator=g)).to(torch.bfloat16)
    tg = torch.randint(0, V, (T,), device="cuda", generator=g, dtype=torch.int32)
    rows = rec.loss_rows()
    M = len(rows)
    adv = torch.randn(M, device="cuda", generator=g)
    rng = np.random.default_rng(44)
    pick = np.sort(rng.choice(M, 24, replace=False))
    srow = rows[pick]
    scale = Dh ** -0.5
    Q64, K64, V64, W64, t_np = np64(Q), np64(K), np64(Vv), np64(W), tg.cpu().numpy()
    Os, _ = OA.attn_fwd(rec.seqlens, rec.edits, Q64, K64, V64, scale, rows=srow)
    Hs = np.zeros((T, d))
    Hs[srow] = Os.reshape(len(srow), d)
    lp_s, lse_s = OL.logprob(Hs, W64, t_np, srow)
    # lp_old: the oracle's lp + noise on the sampled rows; a fixed value elsewhere
    lp_old = np.full(M, -np.log(V))
    lp_old[pick] = lp_s + 0.05 * rng.standard_normal(len(pick))
    lp_old_t = torch.tensor(lp_old, dtype=torch.float32, device="cuda")
    O, out, dH, dW, dQ, dK, dV = _gpu_chain(rec, Q, K, Vv, W, tg, torch.tensor(rows, dtype=torch.int32).cuda(),
                                            lp_old_t, adv, 0.2)
    assert_maxabs(np64(O[srow]), Os, 2e-2, "O (sampled rows)")
    assert_maxabs(np64(out["lp"])[pick], lp_s, 1e-2, "lp (sampled rows)")
    _, _, _, g_s = OL.policy_loss(lp_s, lp_old[pick], np64(adv)[pick], 0.2, 0.2)
    g_s = g_s * len(pick) / M        # g carries 1/M over all loss rows
    dHr, _ = OL.logprob_loss_bwd(Hs, W64, t_np, srow, lse_s, g_s)
    assert_grad_bf16(np64(dH)[srow], dHr[srow], "dH (sampled rows)")
    for t in (dW, dQ, dK, dV):
        assert torch.isfinite(t.float()).all()
