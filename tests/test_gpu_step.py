"""The whole path chained as the step bench.py times: visibility -> masked
attention fwd -> H = O -> fused LM-head log-prob + clipped loss fwd/bwd ->
attention bwd with dO = dH. Checked against the oracle run on the same chain."""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, assert_rel, lifetime_keys, np64
from oracle import attention as OA
from oracle import logprob as OL
from oracle.visibility import lifetimes

pytestmark = pytest.mark.gpu


def _gpu_chain(rec, Q, K, V, W, tg, rows, lp_old, adv, eps, eps_hi=None):
    import paper_2609_00865_gb300 as mw
    T, Hq, Dh = Q.shape
    scale = Dh ** -0.5
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    O, LSE = mw.masked_attn_fwd(vis, Q, K, V, scale)
    H = O.view(T, Hq * Dh)
    out = mw.logprob_loss_fwd(H, W, tg, rows, lp_old, adv, eps, eps if eps_hi is None else eps_hi)
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


def test_on_policy_summaries_chained_fp32():
    """AgentFold-style record (the policy writes each fold's summary under the
    pre-fold view; the summary rows carry loss): the whole chain in fp32
    against the oracle at 1e-4, on every loss row, summary rows included."""
    rec = synth.record(2, 700, 3, 0.6, 40, 32, 40, 30, 123, on_policy_summary=True)
    T, Hq, Hkv, Dh, V = rec.total, 2, 2, 64, 1024
    Q = synth.normal((T, Hq, Dh), 131)
    K = synth.normal((T, Hkv, Dh), 132)
    Vv = synth.normal((T, Hkv, Dh), 133)
    W = synth.normal((V, Hq * Dh), 134, std=0.02)
    tg = synth.uniform_int(T, V, 135)
    rows = rec.loss_rows()
    M = len(rows)
    adv = synth.normal((M,), 136)
    scale = Dh ** -0.5
    Or, _ = OA.attn_fwd(rec.seqlens, rec.edits, np64(Q), np64(K), np64(Vv), scale)
    Hr = Or.reshape(T, Hq * Dh)
    lp_r, lse_r = OL.logprob(Hr, np64(W), tg.numpy(), rows)
    lp_old = torch.tensor(lp_r + np64(synth.normal((M,), 137, std=0.05)), dtype=torch.float32)
    ratio_r, _, loss_r, g_r = OL.policy_loss(lp_r, np64(lp_old), np64(adv), 0.2, 0.28)
    dHr, dWr = OL.logprob_loss_bwd(Hr, np64(W), tg.numpy(), rows, lse_r, g_r)
    dQr, dKr, dVr = OA.attn_bwd(rec.seqlens, rec.edits, np64(Q), np64(K), np64(Vv), dHr.reshape(T, Hq, Dh), scale)
    dev = lambda t: t.cuda()
    O, out, dH, dW, dQ, dK, dV = _gpu_chain(rec, dev(Q), dev(K), dev(Vv), dev(W), dev(tg),
                                            torch.tensor(rows, dtype=torch.int32).cuda(), dev(lp_old),
                                            dev(adv), 0.2, 0.28)
    summary_rows = [i for b, t in enumerate(rec.trajs) for J, _ in t.edits
                    for i in range(sum(rec.seqlens[:b]) + J - 40, sum(rec.seqlens[:b]) + J)]
    assert set(summary_rows) <= set(rows.tolist())
    assert_rel(np64(O), Or, 1e-4, "O")
    assert_rel(np64(out["lp"]), lp_r, 1e-4, "lp")
    assert abs(out["loss"].item() - loss_r) <= 1e-4 * max(abs(loss_r), 1e-6)
    for got, ref, what in ((dH, dHr, "dH"), (dW, dWr, "dW"), (dQ, dQr, "dQ"), (dK, dKr, "dK"), (dV, dVr, "dV")):
        assert_rel(np64(got), ref, 1e-4, what)


EPS_LO, EPS_HI = 0.2, 0.28       # App. F.1's clip range, as the bench runs the step


@pytest.mark.slow
def test_config4_chained_full():
    """The full-size 7B-shaped layer step exactly as bench.py runs it (bf16,
    clip 0.2 / 0.28), against the oracle's own chain (§4.3 Theorem
    "materialization equivalence"): attention at every loss row, the LM head
    over the whole vocabulary at every loss row, ratio, clipped loss and g
    (lp_old = the oracle's lp + N(0, 0.05^2)). Compared: O and lp at every
    loss row, the mean loss (1e-3 relative), and the chained backward at
    sampled places -- dH rows, dW vocabulary rows, dQ rows, and dK / dV of
    keys whose lifetimes end at the first two junctions or never end (their
    rows' dO is the oracle's own dH; keys ending at every junction are checked
    with a random dO in ``test_gpu_attention``)."""
    c = synth.CONFIGS[4]
    rec = synth.config_record(4)
    T, Hq, Hkv, Dh, V = rec.total, c["Hq"], c["Hkv"], c["Dh"], c["V"]
    d = Hq * Dh
    scale = Dh ** -0.5
    g = torch.Generator(device="cuda").manual_seed(404)
    Q = torch.randn(T, Hq, Dh, device="cuda", generator=g).to(torch.bfloat16)
    K = torch.randn(T, Hkv, Dh, device="cuda", generator=g).to(torch.bfloat16)
    Vv = torch.randn(T, Hkv, Dh, device="cuda", generator=g).to(torch.bfloat16)
    W = (0.02 * torch.randn(V, d, device="cuda", generator=g)).to(torch.bfloat16)
    tg = torch.randint(0, V, (T,), device="cuda", generator=g, dtype=torch.int32)
    rows = rec.loss_rows()
    M = len(rows)
    adv = torch.randn(M, device="cuda", generator=g)
    Q64, K64, V64, W64, t_np, adv64 = np64(Q), np64(K), np64(Vv), np64(W), tg.cpu().numpy(), np64(adv)

    # oracle forward chain over every loss row
    Or, _ = OA.attn_fwd(rec.seqlens, rec.edits, Q64, K64, V64, scale, rows=rows)
    Hr = np.zeros((T, d))
    Hr[rows] = Or.reshape(M, d)
    lp_r, lse_r = OL.logprob(Hr, W64, t_np, rows)
    rng = np.random.default_rng(44)
    lp_old = lp_r + 0.05 * rng.standard_normal(M)
    ratio_r, _, loss_r, g_r = OL.policy_loss(lp_r, lp_old, adv64, EPS_LO, EPS_HI)
    # no ratio may sit where fp32 and fp64 could pick different clip branches
    assert np.min(np.abs(ratio_r - (1 - EPS_LO))) > 1e-3 and np.min(np.abs(ratio_r - (1 + EPS_HI))) > 1e-3

    lp_old_t = torch.tensor(lp_old, dtype=torch.float32, device="cuda")
    O, out, dH, dW, dQ, dK, dV = _gpu_chain(rec, Q, K, Vv, W, tg, torch.tensor(rows, dtype=torch.int32).cuda(),
                                            lp_old_t, adv, EPS_LO, EPS_HI)
    assert_maxabs(np64(O[rows]), Or, 2e-2, "O (every loss row)")
    assert_maxabs(np64(out["lp"]), lp_r, 1e-2, "lp (every loss row)")
    loss = float(out["loss"].item())
    assert abs(loss - loss_r) <= 1e-3 * max(abs(loss_r), np.mean(np.abs(ratio_r * adv64))), (loss, loss_r)

    # chained backward at sampled places
    t0 = rec.trajs[0]
    om = lifetimes(t0.T, t0.edits)
    J2, J_last = t0.edits[1][0], t0.edits[-1][0]
    # keys whose lifetimes end at the first two junctions (one of them visible
    # across a whole segment) and never-evicted keys of the last segment: the
    # oracle's dH is needed at every loss row that sees them
    keys = np.array([j for j in lifetime_keys(t0.T, t0.edits, seed=4) if om[j] <= J2 or j >= J_last])
    in_loss = np.zeros(T, dtype=bool)
    in_loss[rows] = True
    need = np.zeros(T, dtype=bool)          # rows whose dO the sampled keys read
    for j in keys:
        need[j : min(int(om[j]), t0.T)] = True
    pick = np.sort(rng.choice(M, 24, replace=False))
    qrows = rows[pick]
    need[qrows] = True
    dh_rows = np.nonzero(need & in_loss)[0]
    dHr, _ = OL.logprob_loss_bwd(Hr, W64, t_np, rows, lse_r, g_r, dh_rows=dh_rows)
    assert_grad_bf16(np64(dH[dh_rows]), dHr[dh_rows], "dH (sampled rows)")
    assert float(dH[~torch.from_numpy(in_loss).cuda()].abs().max()) == 0.0, "dH off the loss rows"

    vocab = np.unique(np.concatenate([[0, V - 1], t_np[qrows[:8]], rng.integers(0, V, 48)]))
    dWr = OL.logprob_loss_bwd_vocab(Hr, W64, t_np, rows, lse_r, g_r, vocab)
    assert_grad_bf16(np64(dW[torch.from_numpy(vocab).cuda()]), dWr, "dW (sampled vocabulary rows)")

    dO64 = dHr.reshape(T, Hq, Dh)
    heads = [0, 13, Hq - 1]
    dQr = OA.attn_bwd_rows(rec.seqlens, rec.edits, Q64, K64, V64, dO64, scale, qrows, heads)
    assert_grad_bf16(np64(dQ[qrows][:, heads]), dQr, "dQ (sampled rows)")
    grp = 1
    dkr, dvr = OA.attn_bwd_keys(rec.seqlens[:1], rec.edits[:1], Q64[: t0.T], K64[: t0.T], V64[: t0.T],
                                dO64[: t0.T], scale, grp, keys)
    assert_grad_bf16(np64(dK[keys, grp]), dkr, "dK (keys by lifetime)")
    assert_grad_bf16(np64(dV[keys, grp]), dvr, "dV (keys by lifetime)")


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
