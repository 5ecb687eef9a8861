"""Rotary masked attention at the full attention workload vs the oracle on
sampled rows and keys (§4.2 row-wise positions; the launch configuration
that `bench.py --config 2 --rope` times)."""

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, np64
from oracle import attention as OA

pytestmark = pytest.mark.gpu


def test_rope_full_size_config2_sampled():
    """The attention workload at full size (8 x 16,384 tokens, 32/8 heads, 4
    junctions per trajectory) in the launch configuration that
    `bench.py --config 2 --rope` times: O, LSE and dQ on sampled rows (next to
    junctions, tile edges, random), dK and dV on keys of trajectory 0 taken
    across all its segments, whose positions differ between segments."""
    import paper_2609_00865_gb300 as mw
    rec, c = synth.config_record(2), synth.CONFIGS[2]
    T, theta = rec.total, 1e6
    g = torch.Generator(device="cuda").manual_seed(402)
    q, k, v, do = (torch.randn(T, h, c["Dh"], device="cuda", generator=g).to(torch.bfloat16)
                   for h in (c["Hq"], c["Hkv"], c["Hkv"], c["Hq"]))
    vis = mw.build_visibility(rec.seqlens, rec.edits)
    pos = mw.logical_positions(vis)
    table = mw.rope_table(mw.rope_n_pos(vis), c["Dh"], theta)
    scale = c["Dh"] ** -0.5
    O, LSE = mw.masked_attn_rope_fwd(vis, pos, table, q, k, v, scale)
    dQ, dK, dV = mw.masked_attn_rope_bwd(vis, pos, table, q, k, v, O, do, LSE, scale)
    torch.cuda.synchronize()
    vis.check_status()
    rng = np.random.default_rng(402)
    rows, base = set(), 0
    for t in rec.trajs:
        rows.update({base, base + t.T - 1, base + 127, base + 128})
        for J, _ in t.edits[:2]:
            rows.update({base + J - 1, base + J, base + J + 1})
        base += t.T
    rows = np.array(sorted(rows | set(rng.integers(0, base, 8).tolist())))
    heads = [0, c["Hq"] - 1]
    Q64, K64, V64, dO64 = np64(q), np64(k), np64(v), np64(do)
    Or, Lr = OA.attn_fwd(rec.seqlens, rec.edits, Q64, K64, V64, scale, rows=rows, heads=heads, rope_theta=theta)
    assert_maxabs(np64(O[rows][:, heads]), Or, 2e-2, "O")
    assert_maxabs(np64(LSE[heads][:, rows]), Lr, 2e-2, "LSE")
    dQr = OA.attn_bwd_rows(rec.seqlens, rec.edits, Q64, K64, V64, dO64, scale, rows, heads, rope_theta=theta)
    assert_grad_bf16(np64(dQ[rows][:, heads]), dQr, "dQ (sampled rows)")
    t0 = rec.trajs[0]
    keys = np.unique(np.concatenate([[0, 1, 127, 128, t0.T - 1], [a for J, sp in t0.edits for a, _ in sp[:2]],
                                     rng.integers(0, t0.T, 8)]))
    grp = c["Hkv"] - 1
    dkr, dvr = OA.attn_bwd_keys(rec.seqlens[:1], rec.edits[:1], Q64[: t0.T], K64[: t0.T], V64[: t0.T],
                                dO64[: t0.T], scale, grp, keys, rope_theta=theta)
    assert_grad_bf16(np64(dK[keys, grp]), dkr, "dK (sampled keys)")
    assert_grad_bf16(np64(dV[keys, grp]), dvr, "dV (sampled keys)")
