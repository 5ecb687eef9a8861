"""Shared test helpers: tolerances, tensor plumbing and sample choice (no
method arithmetic)."""

import numpy as np
import torch


def np64(t):
    """Exact float64 copy of a CPU/GPU tensor (bf16 and f32 upcast exactly)."""
    return t.detach().to("cpu", torch.float64).numpy()


def rel_frobenius(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-300))


def assert_rel(got, ref, rtol, what=""):
    """Elementwise |got - ref| <= rtol * (|ref| + rms(ref)).

    The rms term keeps the bound meaningful for entries near zero, where a
    purely elementwise relative error is undefined.
    """
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    rms = np.sqrt(np.mean(ref * ref)) if ref.size else 0.0
    err = np.abs(got - ref)
    bound = rtol * (np.abs(ref) + rms)
    bad = err > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} beyond rtol {rtol}; "
                           f"max err {err.max():.3g}, max rel {np.max(err / (np.abs(ref) + rms)):.3g}")


def assert_maxabs(got, ref, atol, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = float(np.abs(got - ref).max()) if ref.size else 0.0
    assert err <= atol, f"{what}: max abs err {err:.3g} > {atol}"


def assert_grad_bf16(got, ref, what=""):
    """bf16 gradient bar: relative Frobenius <= 1e-2 and every element within
    5e-2 of the reference's largest magnitude."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    rf = rel_frobenius(got, ref)
    assert rf <= 1e-2, f"{what}: relative Frobenius {rf:.3g} > 1e-2"
    scale = float(np.abs(ref).max()) if ref.size else 0.0
    assert_maxabs(got, ref, 5e-2 * scale, what)


def lifetime_keys(T, edits, early=(1, 4), n_late=3, seed=0):
    """Keys of one trajectory chosen by where their lifetimes end: for every
    junction the last key it evicts (its visible rows end at that junction,
    inside a PARTIAL q-tile), for the junctions numbered in ``early`` (0-based)
    also a key it evicts from before the previous junction (visible rows
    spanning a whole segment), and never-evicted keys late in the last segment
    plus the last token. The oracle's cost for a key grows with the rows that
    see it, so the choice keeps every key's visible row range to about one
    segment."""
    from oracle.visibility import lifetimes   # the record's lifetimes pick the sample
    om = lifetimes(T, edits)
    Js = [J for J, _ in edits]
    keys = {T - 1}
    for k, J in enumerate(Js):
        ev = np.nonzero(om == J)[0]
        if ev.size:
            keys.add(int(ev.max()))
            if k >= 1 and k in early:
                early = ev[ev < Js[k - 1]]
                if early.size:
                    keys.add(int(early.max()))
    lo = max(Js[-1] if Js else 0, T - 2048)
    keys.update(np.random.default_rng(seed).integers(lo, T, n_late).tolist())
    return np.array(sorted(keys), dtype=np.int64)
