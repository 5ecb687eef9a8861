"""GPU fused LM-head log-prob + clipped loss (fwd + bwd) vs the oracle."""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, assert_rel, np64
from oracle import logprob as OL

pytestmark = pytest.mark.gpu


def _case(N, d, V, rows, seed, dtype, eps=0.2):
    H = synth.normal((N, d), seed).to(dtype)
    W = synth.normal((V, d), seed + 1, std=0.02).to(dtype)
    targets = synth.uniform_int(N, V, seed + 2)
    M = len(rows)
    adv = synth.normal((M,), seed + 3)
    noise = synth.normal((M,), seed + 4, std=0.05)
    lp_ref, lse_ref = OL.logprob(np64(H), np64(W), targets.numpy(), rows)
    lp_old = torch.tensor(lp_ref + noise.double().numpy(), dtype=torch.float32)
    return H, W, targets, torch.tensor(rows, dtype=torch.int32), lp_old, adv, lp_ref, lse_ref


def _run(H, W, targets, rows, lp_old, adv, eps_lo, eps_hi, dloss=1.0):
    import paper_2609_00865_gb300 as mw
    dev = [t.cuda() for t in (H, W, targets, rows, lp_old, adv)]
    out = mw.logprob_loss_fwd(*dev, eps_lo=eps_lo, eps_hi=eps_hi)
    dH, dW = mw.logprob_loss_bwd(dev[0], dev[1], dev[2], dev[3], out["lse"], out["ws"], dloss)
    torch.cuda.synchronize()
    return out, dH, dW


def _check(H, W, targets, rows, lp_old, adv, lp_ref, lse_ref, out, dH, dW, eps_lo, eps_hi, fp32, dloss=1.0):
    ratio_r, per_r, loss_r, g_r = OL.policy_loss(lp_ref, np64(lp_old), np64(adv), eps_lo, eps_hi, dloss)
    # tokens whose oracle ratio sits within 1e-3 of a clip edge may flip side;
    # there are none in these cases (asserted) so every token is compared
    edge = np.minimum(np.abs(ratio_r - (1 - eps_lo)), np.abs(ratio_r - (1 + eps_hi))) < 1e-3
    assert edge.sum() == 0
    if fp32:
        assert_rel(np64(out["lp"]), lp_ref, 1e-4, "lp")
        assert_rel(np64(out["lse"]), lse_ref, 1e-4, "lse")
    else:
        assert_maxabs(np64(out["lp"]), lp_ref, 1e-2, "lp")
    assert_rel(np64(out["ratio"]), ratio_r, 1e-4 if fp32 else 2e-2, "ratio")
    loss = float(out["loss"].item())
    assert abs(loss - loss_r) <= 1e-3 * max(abs(loss_r), np.mean(np.abs(ratio_r * np64(adv)))), (loss, loss_r)
    dHr, dWr = OL.logprob_loss_bwd(np64(H), np64(W), targets.numpy(), rows.numpy(), lse_ref, g_r)
    if fp32:
        assert_rel(np64(dH), dHr, 1e-4, "dH")
        assert_rel(np64(dW), dWr, 1e-4, "dW")
    else:
        assert_grad_bf16(np64(dH), dHr, "dH")
        assert_grad_bf16(np64(dW), dWr, "dW")


def test_config1_fp32_full():
    c = synth.CONFIGS[1]
    r = synth.config_record(1)
    rows = r.loss_rows()
    args = _case(r.total, c["d"], c["V"], rows, 51, torch.float32)
    out, dH, dW = _run(*args[:6], 0.2, 0.2)
    _check(*args, out, dH, dW, 0.2, 0.2, fp32=True)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_medium(dtype):
    N, d, V = 1000, 256, 5000
    rows = synth.loss_rows_fraction(N, 0.7, 61)
    args = _case(N, d, V, rows, 62, dtype)
    out, dH, dW = _run(*args[:6], 0.2, 0.28, dloss=1.3)
    _check(*args, out, dH, dW, 0.2, 0.28, fp32=dtype == torch.float32, dloss=1.3)


def test_zero_weights_uniform():
    N, d, V = 200, 128, 3000
    rows = np.arange(0, N, 3)
    H = synth.normal((N, d), 71)
    W = torch.zeros(V, d)
    t = synth.uniform_int(N, V, 72)
    M = len(rows)
    out, dH, dW = _run(H, W, t, torch.tensor(rows, dtype=torch.int32), torch.zeros(M), torch.ones(M), 0.2, 0.2)
    np.testing.assert_allclose(np64(out["lp"]), -np.log(V), rtol=1e-6)


@pytest.mark.parametrize("N,M,d,V", [
    # the backward splits d over a group of C CTAs, each owning a d-slice of at
    # most 256 columns (the fewest CTAs per group)
    (300, 200, 256, 4097),      # one CTA per group (C = 1)
    (700, 450, 512, 3001),      # ragged vocab tail (C = 2)
    (500, 260, 960, 5003),      # C = 5, d-slice 192
    (600, 300, 1536, 2999),     # the config-3 hidden size (C = 6)
    (1200, 700, 3584, 152064),  # the config-4 hidden size and vocabulary (C = 14)
    (200, 130, 64, 100),        # the smallest hidden size, a vocabulary below one 256-wide tile
])
def test_tensor_core_shapes(N, M, d, V):
    rows = np.sort(np.random.default_rng(N).permutation(N)[:M])
    args = _case(N, d, V, rows, 70 + d, torch.bfloat16)
    out, dH, dW = _run(*args[:6], 0.2, 0.28, dloss=0.7)
    _check(*args, out, dH, dW, 0.2, 0.28, fp32=False, dloss=0.7)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_no_loss_rows(dtype):
    """M = 0: the loss is 0 and dH, dW are written as zeros (the outputs start
    uninitialised)."""
    import paper_2609_00865_gb300 as mw
    N, d, V = 300, 128, 1000
    H = synth.normal((N, d), 81).to(dtype).cuda()
    W = synth.normal((V, d), 82, std=0.02).to(dtype).cuda()
    t = synth.uniform_int(N, V, 83).cuda()
    rows = torch.zeros(0, dtype=torch.int32, device="cuda")
    empty = torch.zeros(0, dtype=torch.float32, device="cuda")
    out = mw.logprob_loss_fwd(H, W, t, rows, empty, empty, 0.2, 0.28)
    dH, dW = mw.logprob_loss_bwd(H, W, t, rows, out["lse"], out["ws"], 1.0)
    torch.cuda.synchronize()
    assert out["lp"].numel() == 0
    assert float(out["loss"].item()) == 0.0
    assert (dH == 0).all() and (dW == 0).all()


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_kl_to_reference(dtype):
    """The KL-to-reference term (App. F.1, low-variance k3 estimate) in the loss
    and, through g, in dH and dW; asymmetric clip 0.2 / 0.28."""
    import paper_2609_00865_gb300 as mw
    N, d, V = 400, 128, 3000
    rows = np.sort(np.random.default_rng(91).permutation(N)[:250])
    H, W, targets, rows_t, lp_old, adv, lp_o, lse_o = _case(N, d, V, rows, 91, dtype)
    M = len(rows)
    lp_refpol = torch.tensor(lp_o + 0.2 * np.random.default_rng(92).standard_normal(M), dtype=torch.float32)
    beta = 0.3
    dev = [t.cuda() for t in (H, W, targets, rows_t, lp_old, adv)]
    out = mw.logprob_loss_fwd(*dev, eps_lo=0.2, eps_hi=0.28, lp_ref=lp_refpol.cuda(), beta=beta)
    dH, dW = mw.logprob_loss_bwd(dev[0], dev[1], dev[2], dev[3], out["lse"], out["ws"], 1.0)
    torch.cuda.synchronize()
    ratio_r, _, loss_r, g_r = OL.policy_loss(lp_o, np64(lp_old), np64(adv), 0.2, 0.28, lp_ref=np64(lp_refpol),
                                             beta=beta)
    edge = np.minimum(np.abs(ratio_r - 0.8), np.abs(ratio_r - 1.28)) < 1e-3
    assert edge.sum() == 0
    loss = float(out["loss"].item())
    _, _, loss_plain, _ = OL.policy_loss(lp_o, np64(lp_old), np64(adv), 0.2, 0.28)
    assert abs(loss_r - loss_plain) > 1e-3   # the term is not negligible here
    assert abs(loss - loss_r) <= 1e-3 * max(abs(loss_r), np.mean(np.abs(ratio_r * np64(adv)))), (loss, loss_r)
    dHr, dWr = OL.logprob_loss_bwd(np64(H), np64(W), targets.numpy(), rows, lse_o, g_r)
    if dtype == torch.float32:
        assert_rel(np64(out["lp"]), lp_o, 1e-4, "lp")
        assert_rel(np64(dH), dHr, 1e-4, "dH")
        assert_rel(np64(dW), dWr, 1e-4, "dW")
    else:
        assert_maxabs(np64(out["lp"]), lp_o, 1e-2, "lp")
        assert_grad_bf16(np64(dH), dHr, "dH")
        assert_grad_bf16(np64(dW), dWr, "dW")


def test_config3_full_size_sampled():
    """N = 32,768, d = 1,536, V = 151,936, 70% loss rows, in the bench's launch
    configuration. lp / dH are checked on sampled rows, dW on sampled vocab
    rows (the oracle's lse covers every loss row)."""
    import paper_2609_00865_gb300 as mw
    c = synth.CONFIGS[3]
    N, d, V = c["N"], c["d"], c["V"]
    rows = synth.loss_rows_fraction(N, c["loss_frac"], 3000)
    M = len(rows)
    g = torch.Generator(device="cuda").manual_seed(33)
    H = torch.randn(N, d, device="cuda", generator=g).to(torch.bfloat16)
    W = (0.02 * torch.randn(V, d, device="cuda", generator=g)).to(torch.bfloat16)
    tg = torch.randint(0, V, (N,), device="cuda", generator=g, dtype=torch.int32)
    adv = torch.randn(M, device="cuda", generator=g)
    r_dev = torch.tensor(rows, dtype=torch.int32, device="cuda")
    H64, W64, t_np = np64(H), np64(W), tg.cpu().numpy()
    lp_ref, lse_ref = OL.logprob(H64, W64, t_np, rows)
    lp_old = torch.tensor(lp_ref + 0.05 * np.random.default_rng(3).standard_normal(M), dtype=torch.float32,
                          device="cuda")
    out = mw.logprob_loss_fwd(H, W, tg, r_dev, lp_old, adv, 0.2, 0.2)
    dH, dW = mw.logprob_loss_bwd(H, W, tg, r_dev, out["lse"], out["ws"])
    torch.cuda.synchronize()
    assert_maxabs(np64(out["lp"]), lp_ref, 1e-2, "lp")
    ratio_r, _, loss_r, g_r = OL.policy_loss(lp_ref, np64(lp_old), np64(adv), 0.2, 0.2)
    loss = float(out["loss"].item())
    assert abs(loss - loss_r) <= 1e-3 * max(abs(loss_r), np.mean(np.abs(ratio_r * np64(adv))))
    rng = np.random.default_rng(4)
    pick = np.sort(rng.choice(M, 48, replace=False))
    dHr, _ = OL.logprob_loss_bwd(H64, W64, t_np, rows[pick], lse_ref[pick], g_r[pick])
    assert_grad_bf16(np64(dH)[rows[pick]], dHr[rows[pick]], "dH (sampled rows)")
    notloss = np.setdiff1d(np.arange(N), rows)[:64]
    assert (np64(dH)[notloss] == 0).all()
    vocab = np.unique(np.concatenate([rng.integers(0, V, 40), t_np[rows[:8]], [0, V - 1]]))
    dWr = OL.logprob_loss_bwd_vocab(H64, W64, t_np, rows, lse_ref, g_r, vocab)
    assert_grad_bf16(np64(dW)[vocab], dWr, "dW (sampled vocab rows)")


@pytest.mark.parametrize("d", [256, 1536])
def test_logits_far_above_the_reference_are_repaired(d):
    """The bf16 forward measures each row's logits against a fixed reference,
    its largest logit over the first vocabulary entries; a logit more than
    2^96 (66 nats) above it flags the row, which is recomputed exactly. Here
    a third of the rows have one late vocabulary entry (id 4000, past the
    reference range) about 128 nats above all others, some of them as their
    target: lp, the loss, dH and dW must still match the oracle."""
    N, V = 300, 5003
    H = synth.normal((N, d), 91).to(torch.bfloat16)
    W = synth.normal((V, d), 92, std=0.02)
    sign = torch.sign(synth.normal((d,), 93))
    sign[sign == 0] = 1.0
    peaked = torch.arange(0, N, 3)
    H[peaked] = sign.to(torch.bfloat16)                 # rows aligned with W[4000]
    W[4000] = 0.5 * sign * (256.0 / d)                   # logit 128 for those rows
    W = W.to(torch.bfloat16)
    targets = synth.uniform_int(N, V, 94)
    targets[peaked[::2]] = 4000
    rows = np.arange(0, N, 1)
    M = len(rows)
    lp_ref, lse_ref = OL.logprob(np64(H), np64(W), targets.numpy(), rows)
    assert lse_ref[peaked.numpy()].min() > 127.0
    adv = synth.normal((M,), 95)
    lp_old = torch.tensor(lp_ref + 0.05 * np.random.default_rng(96).standard_normal(M), dtype=torch.float32)
    r = torch.tensor(rows, dtype=torch.int32)
    out, dH, dW = _run(H, W, targets, r, lp_old, adv, 0.2, 0.28)
    _check(H, W, targets, r, lp_old, adv, lp_ref, lse_ref, out, dH, dW, 0.2, 0.28, fp32=False)
