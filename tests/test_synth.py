"""The seeded workload generator follows the input recipe it states: valid
records, junctions at their targets, evictions of whole still-visible
observation spans (half of them, or at least a fraction f of the visible
observation tokens), summaries after every junction that no edit evicts, and
loss rows on policy-generated targets."""

import numpy as np
import pytest

import synth
from oracle import visibility as OV


def _check_traj(t, K, evict, summary, prompt):
    T = t.T
    OV.validate_edits(T, t.edits)
    assert len(t.edits) <= K
    assert (t.kinds[: min(prompt, T)] == synth.PROMPT).all()
    evicted = np.zeros(T, dtype=bool)
    for k, (J, spans) in enumerate(t.edits):
        assert J >= ((k + 1) * T) // (K + 1)                 # fires at or after its target
        assert t.kinds[J] == synth.POLICY                    # at the end of a policy span
        visible_obs_tokens = int(((t.kinds[:J] == synth.OBSERVATION) & ~evicted[:J]).sum())
        gone = 0
        for a, b in spans:
            assert (t.kinds[a:b] == synth.OBSERVATION).all()  # whole observation spans only
            assert not evicted[a:b].any()                     # still visible when evicted
            assert a == 0 or t.kinds[a - 1] != synth.OBSERVATION or evicted[a - 1]
            assert b == T or t.kinds[b] != synth.OBSERVATION
            evicted[a:b] = True
            gone += b - a
        if isinstance(evict, float):
            assert gone >= evict * visible_obs_tokens - 1e-9
        s_end = min(J + 1 + summary, T)
        assert (t.kinds[J + 1: s_end] == synth.SUMMARY).all()
    assert not evicted[t.kinds == synth.SUMMARY].any()
    lr = t.loss_rows
    assert (t.kinds[lr + 1] == synth.POLICY).all()
    assert len(lr) == int((t.kinds[1:] == synth.POLICY).sum())


@pytest.mark.parametrize("cfg", [1, 2, 4])
def test_config_records_follow_the_recipe(cfg):
    c = synth.CONFIGS[cfg]
    rec = synth.config_record(cfg)
    assert len(rec.trajs) == c["n_traj"] and all(t.T == c["T"] for t in rec.trajs)
    for t in rec.trajs:
        _check_traj(t, c["K"], c["evict"], c["summary"], c["prompt"])
        assert len(t.edits) == c["K"]


@pytest.mark.parametrize("K,f", [(1, 0.3), (32, 0.9)])
def test_sweep_records_follow_the_recipe(K, f):
    c = synth.CONFIGS[5]
    rec = synth.config_record(5, K=K, f=f)
    _check_traj(rec.trajs[0], K, f, c["summary"], c["prompt"])


def test_half_span_eviction_count():
    t = synth.config_record(1).trajs[0]
    visible = 0
    seen = set()
    for J, spans in t.edits:
        obs_before = [(a, b) for a, b in _obs_spans(t.kinds[:J]) if (a, b) not in seen]
        assert len(spans) == int(round(0.5 * len(obs_before)))
        seen.update(spans)
        visible += len(obs_before)
    assert visible > 0


def _obs_spans(kinds):
    out, a = [], None
    for i, k in enumerate(kinds):
        if k == synth.OBSERVATION and a is None:
            a = i
        if k != synth.OBSERVATION and a is not None:
            out.append((a, i))
            a = None
    if a is not None:
        out.append((a, len(kinds)))
    return out


def test_generation_is_deterministic():
    a, b = synth.config_record(2), synth.config_record(2)
    assert a.edits == b.edits
    assert all((x.kinds == y.kinds).all() for x, y in zip(a.trajs, b.trajs))
    r1 = synth.loss_rows_fraction(1000, 0.7, 5)
    assert (r1 == synth.loss_rows_fraction(1000, 0.7, 5)).all() and len(r1) == 700
    assert (np.diff(r1) > 0).all()


def test_on_policy_summaries():
    """AgentFold-style records: every junction is the last token of an m-token
    policy span (the summary), whose rows carry loss; no inserted summaries."""
    r = synth.record(2, 900, 3, 0.6, 48, 32, 40, 30, 77, on_policy_summary=True)
    for t in r.trajs:
        assert (t.kinds != synth.SUMMARY).all()
        rows = set(t.loss_rows.tolist())
        for J, _ in t.edits:
            assert (t.kinds[J - 47: J + 1] == synth.POLICY).all()
            assert all(i in rows for i in range(J - 48, J))     # rows predicting the summary tokens


def test_events_record_offloads_and_retrieves_valid_spans():
    """The offload / retrieve stand-in keeps each compression's evicted spans
    as out-spans and brings earlier offloaded spans back: every event is
    valid (a retrieved span is out of the view when its event fires), some
    spans come back, and with retrieve = 0 the views equal the compression
    record's."""
    from oracle import nonmonotone as N
    rec = synth.config_record(2)
    ev = synth.events_record(rec, 0.3, 7)
    n_back = 0
    for t, e in zip(rec.trajs, ev):
        N.validate_events(t.T, e)
        assert [(J, list(o)) for J, o, _ in e] == [(J, list(map(tuple, s))) for J, s in t.edits]
        n_back += sum(len(i) for _, _, i in e)
    assert n_back > 0
    small = synth.record(2, 700, 3, 0.6, 16, 16, 20, 30, 11)
    none = synth.events_record(small, 0.0, 7)
    for t, e in zip(small.trajs, none):
        assert all(not i for _, _, i in e)
        np.testing.assert_array_equal(N.dense_mask(t.T, e), OV.dense_mask(t.T, t.edits))


def test_debug_workload_records_are_valid():
    """The records the debug-library workload runs on the GPU are valid
    records for the oracle (edits and events), so a failure there is the
    library's, not the input's."""
    import debug_workload as D
    from oracle import nonmonotone as N
    for seqlens, edits in (D.EDGE, D.MEDIUM):
        for T, e in zip(seqlens, edits):
            OV.validate_edits(T, e)
    for T, e in zip(*D.EVENTS):
        N.validate_events(T, e)
    assert any(i for e in D.EVENTS[1] for _, _, i in e)      # some span comes back
