"""GPU views of records whose events also bring spans back (MemexRL's offload /
retrieve, App. F): the builder's segments, compact views, view bits and pair
counts bit for bit against ``oracle.nonmonotone.build``, and the bf16 masked
attention (forward and backward) on those views against the oracle's compact
per-segment computation."""

import json
import os

import numpy as np
import pytest
import torch

import synth
from helpers import assert_grad_bf16, assert_maxabs, np64
from oracle import attention as OA
from oracle import nonmonotone as N

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(__file__)


def _memex_record(rng, T, n_events):
    """Offload whole observation-sized spans (60-300 tokens, so they cross
    tiles) and retrieve earlier offloaded spans in later events."""
    events, out_spans = [], []
    Js = sorted(rng.choice(np.arange(200, T - 1), size=n_events, replace=False).tolist())
    in_view_free = 0                       # offloads take spans after the previous retrievals
    for J in Js:
        sp_in = []
        if out_spans and rng.random() < 0.6:
            sp_in.append(out_spans.pop(int(rng.integers(0, len(out_spans)))))
        sp_out = []
        a = int(rng.integers(in_view_free, max(in_view_free + 1, J - 60)))
        b = int(min(J, a + rng.integers(60, 300)))
        if a < b and all(not (x < b and a < y) for x, y in sp_in + out_spans):
            sp_out.append((a, b))
            out_spans.append((a, b))
        events.append((int(J), sp_out, sp_in))
    return events


def _panel():
    with open(os.path.join(HERE, "golden", "memexrl_panel.json")) as f:
        g = json.load(f)
    return len(g["tokens"]), [(J, [tuple(s) for s in o], [tuple(s) for s in i]) for J, o, i in g["events"]]


def _compare(seqlens, events):
    import paper_2609_00865_gb300 as mw
    vis = mw.build_views_events(seqlens, events)
    torch.cuda.synchronize()
    vis.check_status()
    got = vis.arrays()
    want = N.build(seqlens, events)
    for key in ("seg", "seg_len", "cpos", "keymask"):
        np.testing.assert_array_equal(got[key], want[key], err_msg=key)
    defined = want["csrc"] != -2
    np.testing.assert_array_equal(got["csrc"][defined], want["csrc"][defined], err_msg="csrc")
    np.testing.assert_array_equal(got["pairs"], want["pairs"], err_msg="pairs")
    assert got["pairs_total"] == want["pairs_total"]
    assert len(got["fwd_idx"]) == 0 and len(got["bwd_idx"]) == 0    # no tile lists for such views
    return vis


def test_panel_views():
    T, events = _panel()
    _compare([T], [events])


@pytest.mark.parametrize("seed", range(4))
def test_random_event_records(seed):
    rng = np.random.default_rng(4000 + seed)
    seqlens = [int(rng.integers(300, 1500)) for _ in range(int(rng.integers(1, 4)))]
    events = [_memex_record(rng, T, int(rng.integers(1, 6))) for T in seqlens]
    _compare(seqlens, events)


def test_empty_trajectory_and_no_events():
    _compare([300, 0, 129], [[(100, [(0, 50)], []), (200, [], [(0, 50)])], [], []])


def test_attention_on_event_views():
    """bf16, 8 / 2 heads, Dh 128: re-entered spans sit at the end of a view,
    after tokens decoded meanwhile; the compact kernels read them in that
    order. Forward within 2e-2, gradients within the bf16 bar."""
    import paper_2609_00865_gb300 as mw
    rng = np.random.default_rng(4100)
    seqlens = [1100, 700]
    events = [_memex_record(rng, T, 5) for T in seqlens]
    assert any(ev[2] for e in events for ev in e)             # some span comes back
    vis = _compare(seqlens, events)
    T = sum(seqlens)
    Q, K, Vx, dO = (synth.normal((T, h, 128), 4200 + n).to(torch.bfloat16) for n, h in enumerate((8, 2, 2, 8)))
    q, k, v, do = (t.cuda() for t in (Q, K, Vx, dO))
    O, LSE = mw.masked_attn_fwd(vis, q, k, v, 128 ** -0.5)
    dQ, dK, dV = mw.masked_attn_bwd(vis, q, k, v, O, do, LSE, 128 ** -0.5)
    torch.cuda.synchronize()
    vis.check_status()
    Or, Lr = OA.attn_fwd(seqlens, events, np64(Q), np64(K), np64(Vx), 128 ** -0.5, views=N.live_views)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, events, np64(Q), np64(K), np64(Vx), np64(dO), 128 ** -0.5,
                                views=N.live_views)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


def test_event_records_rejected_where_lifetimes_are_needed():
    import paper_2609_00865_gb300 as mw
    T, events = _panel()
    vis = mw.build_views_events([T], [events])
    Q = torch.zeros(T, 2, 64, device="cuda")
    with pytest.raises(mw.MWError) as e:               # the fp32 path walks tile lists
        mw.masked_attn_fwd(vis, Q, Q, Q)
    assert e.value.status == 3
    with pytest.raises(mw.MWError) as e:
        mw.diverging_rows(vis)
    assert e.value.status == 3
    with pytest.raises(mw.MWError) as e:               # retrieving a position that is in the view
        mw.build_views_events([50], [[(10, [], [(2, 4)])]])
    assert e.value.status == 2


def test_rotary_attention_on_event_views():
    """Rotary positions on event views are list indices (reading 3): a
    re-entered span takes positions after the tokens decoded meanwhile. The
    bf16 rotary attention (keys turned by their rank as they are gathered)
    forward and backward against the oracle's compact computation with
    rotary positions on the same views."""
    import paper_2609_00865_gb300 as mw
    rng = np.random.default_rng(4300)
    seqlens = [900, 600]
    events = [_memex_record(rng, T, 4) for T in seqlens]
    assert any(ev[2] for e in events for ev in e)
    vis = _compare(seqlens, events)
    T = sum(seqlens)
    Q, K, Vx, dO = (synth.normal((T, h, 128), 4400 + n).to(torch.bfloat16) for n, h in enumerate((8, 2, 2, 8)))
    q, k, v, do = (t.cuda() for t in (Q, K, Vx, dO))
    theta, scale = 1e4, 128 ** -0.5
    pos = mw.logical_positions(vis)              # the build's ranks: list indices
    table = mw.rope_table(mw.rope_n_pos(vis), 128, theta)
    O, LSE = mw.masked_attn_rope_fwd(vis, pos, table, q, k, v, scale)
    dQ, dK, dV = mw.masked_attn_rope_bwd(vis, pos, table, q, k, v, O, do, LSE, scale)
    torch.cuda.synchronize()
    vis.check_status()
    Or, Lr = OA.attn_fwd(seqlens, events, np64(Q), np64(K), np64(Vx), scale, rope_theta=theta, views=N.live_views)
    assert_maxabs(np64(O), Or, 2e-2, "O")
    assert_maxabs(np64(LSE), Lr, 2e-2, "LSE")
    dQr, dKr, dVr = OA.attn_bwd(seqlens, events, np64(Q), np64(K), np64(Vx), np64(dO), scale, rope_theta=theta,
                                views=N.live_views)
    assert_grad_bf16(np64(dQ), dQr, "dQ")
    assert_grad_bf16(np64(dK), dKr, "dK")
    assert_grad_bf16(np64(dV), dVr, "dV")


def test_dense_mask_export_on_event_views():
    """mw_export_dense_mask on offload / retrieve views against both oracle
    formulations of their dense mask (view order, and the per-key replay)."""
    import paper_2609_00865_gb300 as mw
    rng = np.random.default_rng(4100)
    T0, ev0 = _panel()
    seqlens = [T0] + [int(rng.integers(300, 1500)) for _ in range(2)]
    events = [ev0] + [_memex_record(rng, T, int(rng.integers(1, 6))) for T in seqlens[1:]]
    vis = _compare(seqlens, events)
    for b, (T, e) in enumerate(zip(seqlens, events)):
        got = mw.export_dense_mask(vis, seqlens, b).cpu().numpy()
        np.testing.assert_array_equal(got, N.dense_mask(T, e), err_msg=f"trajectory {b}")
        np.testing.assert_array_equal(got, N.replay_mask(T, e), err_msg=f"trajectory {b} (replay)")
