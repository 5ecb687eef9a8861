"""GPU masked attention (fwd + bwd) vs the per-segment oracle."""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, assert_rel, lifetime_keys, np64
from oracle import attention as OA

pytestmark = pytest.mark.gpu


def _tensors(T, Hq, Hkv, Dh, seed, dtype):
    Q = synth.normal((T, Hq, Dh), seed).to(dtype)
    K = synth.normal((T, Hkv, Dh), seed + 1).to(dtype)
    V = synth.normal((T, Hkv, Dh), seed + 2).to(dtype)
    dO = synth.normal((T, Hq, Dh), seed + 3).to(dtype)
    return Q, K, V, dO


def _run(seqlens, edits, Q, K, V, dO, scale):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_visibility(seqlens, edits)
    q, k, v, do = (t.cuda() for t in (Q, K, V, dO))
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, scale)
    dQ, dK, dV = mw.masked_attn_bwd(vis, q, k, v, O, do, LSE, scale)
    torch.cuda.synchronize()
    return O, LSE, dQ, dK, dV


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


def test_config1_fp32_full():
    """Config 1 (tiny fp32): every output within 1e-4 relative."""
    c = synth.CONFIGS[1]
    r = synth.config_record(1)
    Q, K, V, dO = _tensors(r.total, c["Hq"], c["Hkv"], c["Dh"], 11, torch.float32)
    scale = c["Dh"] ** -0.5
    O, LSE, dQ, dK, dV = _run(r.seqlens, r.edits, Q, K, V, dO, scale)
    Or, Lr = OA.attn_fwd(r.seqlens, r.edits, np64(Q), np64(K), np64(V), scale)
    assert_rel(np64(O), Or, 1e-4, "O")
    assert_rel(np64(LSE), Lr, 1e-4, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(r.seqlens, r.edits, np64(Q), np64(K), np64(V), np64(dO), scale)
    assert_rel(np64(dQ), dQr, 1e-4, "dQ")
    assert_rel(np64(dK), dKr, 1e-4, "dK")
    assert_rel(np64(dV), dVr, 1e-4, "dV")


@pytest.mark.parametrize("Dh", [64, 128])
def test_medium_fp32_gqa(Dh):
    seqlens, edits = _medium_record(5)
    Q, K, V, dO = _tensors(sum(seqlens), 8, 2, Dh, 21, torch.float32)
    scale = Dh ** -0.5
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale)
    assert_rel(np64(O), Or, 1e-4, "O")
    assert_rel(np64(LSE), Lr, 1e-4, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale)
    assert_rel(np64(dQ), dQr, 1e-4, "dQ")
    assert_rel(np64(dK), dKr, 1e-4, "dK")
    assert_rel(np64(dV), dVr, 1e-4, "dV")


def test_medium_bf16_gqa():
    seqlens, edits = _medium_record(6)
    Q, K, V, dO = _tensors(sum(seqlens), 8, 2, 128, 31, torch.bfloat16)
    scale = 128 ** -0.5
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


# trajectories of 1, 127, 0, 128, 129 and 300 tokens in one record: a lone row,
# one row short of a tile, an empty trajectory, an exact tile, a one-row second
# tile and a ragged third tile
_TILE_EDGE = (
    [1, 127, 0, 128, 129, 300],
    [[], [(100, [(10, 40)])], [], [(64, [(0, 32)]), (120, [(70, 100)])], [(128, [(5, 127)])],
     [(150, [(20, 140)]), (280, [(150, 260)])]],
)


@pytest.mark.parametrize("Hq,Hkv", [(4, 4), (6, 2)])
def test_bf16_tile_edges_and_group_sizes(Hq, Hkv):
    """Tensor-core path on the tile-edge record, with one query head per KV
    head and with groups of three."""
    seqlens, edits = _TILE_EDGE
    Q, K, V, dO = _tensors(sum(seqlens), Hq, Hkv, 128, 51 + Hq, torch.bfloat16)
    scale = 128 ** -0.5
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


def test_fp32_tile_edges():
    """The exact-fp32 path (Dh 64, groups of two) on the tile-edge record."""
    seqlens, edits = _TILE_EDGE
    Q, K, V, dO = _tensors(sum(seqlens), 4, 2, 64, 61, torch.float32)
    scale = 64 ** -0.5
    O, LSE, dQ, dK, dV = _run(seqlens, edits, Q, K, V, dO, scale)
    Or, Lr = OA.attn_fwd(seqlens, edits, np64(Q), np64(K), np64(V), scale)
    assert_rel(np64(O), Or, 1e-4, "O")
    assert_rel(np64(LSE), Lr, 1e-4, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, edits, np64(Q), np64(K), np64(V), np64(dO), scale)
    assert_rel(np64(dQ), dQr, 1e-4, "dQ")
    assert_rel(np64(dK), dKr, 1e-4, "dK")
    assert_rel(np64(dV), dVr, 1e-4, "dV")


def test_later_edit_leaves_earlier_rows_unchanged():
    """The conditioning invariant on the GPU path (§3.3): adding a junction at
    row 600 that evicts tokens 100..399 changes nothing for rows before 600 --
    their attention outputs, log-sum-exps and the log-probs scored from them
    are bitwise equal (same visible keys, same tiles, same arithmetic order)."""
    import paper_2609_00865_gb300 as mw
    T, Hq, Hkv, Dh = 700, 8, 2, 128
    base = [(200, [(20, 150)]), (450, [(160, 300)])]
    later = base + [(600, [(100, 400)])]
    Q, K, V, dO = _tensors(T, Hq, Hkv, Dh, 71, torch.bfloat16)
    out = []
    W = synth.normal((5000, Hq * Dh), 72, std=0.02).to(torch.bfloat16).cuda()
    tg = synth.uniform_int(T, 5000, 73).cuda()
    rows = torch.arange(0, 600, 3, dtype=torch.int32, device="cuda")
    zeros = torch.zeros(rows.numel(), dtype=torch.float32, device="cuda")
    for edits in (base, later):
        O, LSE, *_ = _run([T], [edits], Q, K, V, dO, Dh ** -0.5)
        lp = mw.logprob_loss_fwd(O.reshape(T, Hq * Dh), W, tg, rows, zeros, zeros)["lp"]
        torch.cuda.synchronize()
        out.append((O[:600].clone(), LSE[:, :600].clone(), lp.clone()))
    assert torch.equal(out[0][0], out[1][0])
    assert torch.equal(out[0][1], out[1][1])
    assert torch.equal(out[0][2], out[1][2])


def test_no_edits_is_causal_attention():
    """K = 0 reduces to ordinary causal attention (library SDPA on the GPU
    output's inputs, float64 on the CPU)."""
    T, H, Dh = 300, 2, 64
    Q, K, V, dO = _tensors(T, H, H, Dh, 41, torch.float32)
    O, LSE, *_ = _run([T], [[]], Q, K, V, dO, 0.125)
    ref = torch.nn.functional.scaled_dot_product_attention(
        Q.double().permute(1, 0, 2), K.double().permute(1, 0, 2), V.double().permute(1, 0, 2),
        is_causal=True, scale=0.125).permute(1, 0, 2).numpy()
    assert_rel(np64(O), ref, 1e-4, "O")


def _sample_rows(rec, rng, n_random=24):
    """Rows around every junction, trajectory ends, and random rows."""
    rows, base = set(), 0
    for t in rec.trajs:
        rows.update({base, base + t.T - 1, base + min(127, t.T - 1), base + min(128, t.T - 1)})
        for J, _ in t.edits[:3]:
            rows.update({base + J - 1, base + J, base + min(J + 1, t.T - 1)})
        base += t.T
    rows.update(rng.integers(0, base, n_random).tolist())
    return np.array(sorted(rows))


def _full_size_fwd(rec, c, seed):
    import paper_2609_00865_gb300 as mw
    T = rec.total
    g = torch.Generator(device="cuda").manual_seed(seed)
    q = torch.randn(T, c["Hq"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    k = torch.randn(T, c["Hkv"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    v = torch.randn(T, c["Hkv"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    scale = c["Dh"] ** -0.5
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, scale)
    torch.cuda.synchronize()
    vis.check_status()
    rng = np.random.default_rng(seed)
    rows = _sample_rows(rec, rng)
    heads = sorted(set(rng.integers(0, c["Hq"], 3).tolist()) | {0, c["Hq"] - 1})
    Or, Lr = OA.attn_fwd(rec.seqlens, rec.edits, np64(q), np64(k), np64(v), scale, rows=rows, heads=heads)
    assert_maxabs(np64(O[rows][:, heads]), Or, 2e-2, "O")
    assert_maxabs(np64(LSE[heads][:, rows]), Lr, 2e-2, "LSE")


@pytest.mark.parametrize("cfg", [2, 4])
def test_full_size_forward_sampled(cfg):
    """Full-size workloads in the bench's launch configuration; the oracle
    recomputes sampled rows (every head's compact view) one by one."""
    _full_size_fwd(synth.config_record(cfg), synth.CONFIGS[cfg], 100 + cfg)


@pytest.mark.parametrize("K,f", [(1, 0.3), (32, 0.9)])
def test_sweep_forward_sampled(K, f):
    _full_size_fwd(synth.config_record(5, K=K, f=f), synth.CONFIGS[5], 200 + K)


def _full_size_bwd(rec, c, seed, keys_mode, early=(1, 4)):
    import paper_2609_00865_gb300 as mw
    T = rec.total
    g = torch.Generator(device="cuda").manual_seed(seed)
    q = torch.randn(T, c["Hq"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    k = torch.randn(T, c["Hkv"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    v = torch.randn(T, c["Hkv"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    do = torch.randn(T, c["Hq"], c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    scale = c["Dh"] ** -0.5
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, scale)
    dQ, dK, dV = mw.masked_attn_bwd(vis, q, k, v, O, do, LSE, scale)
    torch.cuda.synchronize()
    vis.check_status()
    rng = np.random.default_rng(seed)
    Q64, K64, V64, dO64 = np64(q), np64(k), np64(v), np64(do)
    rows = _sample_rows(rec, rng, n_random=12)
    heads = sorted(set(rng.integers(0, c["Hq"], 2).tolist()) | {c["Hq"] - 1})
    dQr = OA.attn_bwd_rows(rec.seqlens, rec.edits, Q64, K64, V64, dO64, scale, rows, heads)
    assert_grad_bf16(np64(dQ[rows][:, heads]), dQr, "dQ (sampled rows)")
    grp = int(rng.integers(0, c["Hkv"]))
    t0 = rec.trajs[0]
    if keys_mode == "all":        # keys across every segment of trajectory 0
        keys = np.unique(np.concatenate([[0, 1, 127, 128, t0.T - 1],
                                         [a for J, sp in t0.edits for a, _ in sp[:2]],
                                         rng.integers(0, t0.T, 10)]))
    else:                          # keys whose lifetimes end at every junction, and never
        keys = lifetime_keys(t0.T, t0.edits, early=early, seed=seed)
    dkr, dvr = OA.attn_bwd_keys(rec.seqlens[:1], rec.edits[:1], Q64[: t0.T], K64[: t0.T], V64[: t0.T],
                                dO64[: t0.T], scale, grp, keys)
    assert_grad_bf16(np64(dK[keys, grp]), dkr, "dK (sampled keys)")
    assert_grad_bf16(np64(dV[keys, grp]), dvr, "dV (sampled keys)")


def test_full_size_backward_config2():
    _full_size_bwd(synth.config_record(2), synth.CONFIGS[2], 302, "all")


def test_full_size_backward_config4():
    """Keys whose lifetimes end at each of the 8 junctions (the PARTIAL-tile
    interval [j, omega(j)) of the dK/dV kernel), keys visible across a whole
    segment, and never-evicted keys."""
    _full_size_bwd(synth.config_record(4), synth.CONFIGS[4], 304, "lifetimes")


@pytest.mark.parametrize("K,f,early", [(1, 0.3, ()), (8, 0.6, (4,)), (32, 0.9, (1, 16))])
def test_sweep_backward_sampled(K, f, early):
    """The sweep's sparsest, middle and densest-eviction points."""
    _full_size_bwd(synth.config_record(5, K=K, f=f), synth.CONFIGS[5], 305 + K, "lifetimes", early)
