"""Seeded synthetic workloads: compression records and input tensors.

This module only draws inputs. It holds none of the method's arithmetic and is
shared by the tests, the benchmark and the oracle's tests; neither the oracle
nor the CUDA path depends on anything else here.

Each trajectory stands in for a compressed agent rollout (the paper's live
web-search rollouts are not available): a prompt, then turns of
[policy span ~ Geometric(mean Lp), observation span ~ Geometric(mean Lo)].
The k-th junction target is ``floor((k+1) T / (K+1))``; the junction fires at
the end of the first policy span that reaches the target (the compression
call, e.g. TC-RAG's ``pop``), evicts whole still-visible observation spans
chosen in seeded random order, and is followed by an inserted summary of
``summary`` tokens (never evicted, never in the loss). Rows whose next token is
policy-generated carry the loss.
"""

from dataclasses import dataclass, field

import numpy as np

PROMPT, POLICY, OBSERVATION, SUMMARY = 0, 1, 2, 3


@dataclass
class Trajectory:
    T: int
    edits: list                      # [(J, [(a, b), ...]), ...]
    kinds: np.ndarray                # int8 [T]: PROMPT/POLICY/OBSERVATION/SUMMARY

    @property
    def loss_rows(self):
        """Rows i whose target token i+1 is policy-generated."""
        nxt = np.zeros(self.T, dtype=bool)
        nxt[:-1] = self.kinds[1:] == POLICY
        return np.nonzero(nxt)[0]


@dataclass
class Record:
    trajs: list = field(default_factory=list)

    @property
    def seqlens(self):
        return [t.T for t in self.trajs]

    @property
    def edits(self):
        return [t.edits for t in self.trajs]

    @property
    def total(self):
        return int(sum(self.seqlens))

    def loss_rows(self):
        out, base = [], 0
        for t in self.trajs:
            out.append(t.loss_rows + base)
            base += t.T
        return np.concatenate(out).astype(np.int64) if out else np.zeros(0, np.int64)


def _rng(seed):
    return np.random.Generator(np.random.Philox(int(seed)))


def trajectory(T, K, evict, summary, prompt, Lp, Lo, seed, on_policy_summary=False):
    """One synthetic trajectory (see module docstring).

    ``evict`` is ``"half_spans"`` (evict round(0.5 x count) whole spans) or a
    float f (evict spans in shuffled order until at least f x the visible
    observation tokens are gone).

    ``on_policy_summary`` (AgentFold, App. F harness notes: the policy
    summarises the foldable prefix and the summary is trained): the
    ``summary`` tokens are policy tokens decoded before the fold, right after
    the policy span that reaches the target, and the junction is their last
    token, so they are scored under the pre-fold view and carry loss; later
    rows see the summary but not the folded spans.
    """
    rng = _rng(seed)
    kinds = np.full(T, PROMPT, dtype=np.int8)
    targets = [((k + 1) * T) // (K + 1) for k in range(K)]
    visible_obs = []
    edits = []
    pos = min(prompt, T)
    k = 0
    while pos < T:
        end = min(pos + int(rng.geometric(1.0 / Lp)), T)
        kinds[pos:end] = POLICY
        J = end - 1
        if on_policy_summary and k < K and J >= targets[k]:
            # the summary is decoded by the policy under the pre-fold view;
            # the fold fires at its last token
            s_end = min(end + summary, T)
            kinds[end:s_end] = POLICY
            J = s_end - 1
        if k < K and J >= targets[k] and J <= T - 1:
            order = rng.permutation(len(visible_obs))
            if evict == "half_spans":
                take = order[: int(round(0.5 * len(visible_obs)))]
            else:
                total = sum(b - a for a, b in visible_obs)
                take, gone = [], 0
                for o in order:
                    if gone >= evict * total:
                        break
                    take.append(o)
                    gone += visible_obs[o][1] - visible_obs[o][0]
            chosen = sorted(visible_obs[o] for o in take)
            visible_obs = [s for n, s in enumerate(visible_obs) if n not in set(int(t) for t in take)]
            edits.append((int(J), [(int(a), int(b)) for a, b in chosen]))
            if on_policy_summary:
                pos = J + 1
            else:
                s_end = min(J + 1 + summary, T)
                kinds[J + 1 : s_end] = SUMMARY
                pos = s_end
            k += 1
            continue
        pos = end
        if pos >= T:
            break
        oend = min(pos + int(rng.geometric(1.0 / Lo)), T)
        kinds[pos:oend] = OBSERVATION
        visible_obs.append((pos, oend))
        pos = oend
    return Trajectory(T=T, edits=edits, kinds=kinds)


# --- the five workloads -----------------------------------------------------

CONFIGS = {
    1: dict(name="tiny fp32: 1x512 tokens, 2 junctions (50% of spans), 32-token summaries, "
                 "2 heads Dh 64, LM head d=128 V=1024",
            n_traj=1, T=512, K=2, evict="half_spans", summary=32, prompt=32, Lp=32, Lo=24,
            Hq=2, Hkv=2, Dh=64, d=128, V=1024, dtype="f32"),
    2: dict(name="bf16 attention: 8x16384 tokens, 32/8 heads Dh 128, 4 junctions at 60%, "
                 "512-token summaries",
            n_traj=8, T=16384, K=4, evict=0.6, summary=512, prompt=256, Lp=200, Lo=400,
            Hq=32, Hkv=8, Dh=128, dtype="bf16"),
    3: dict(name="bf16 fused log-prob loss: N=32768, d=1536, V=151936, 70% loss rows, clip 0.2/0.28",
            N=32768, d=1536, V=151936, loss_frac=0.7, dtype="bf16"),
    4: dict(name="7B-shaped layer step: 2x65536 tokens, 28/4 heads Dh 128, 8 junctions at 70%, "
                 "1024-token summaries, LM head d=3584 V=152064",
            n_traj=2, T=65536, K=8, evict=0.7, summary=1024, prompt=256, Lp=200, Lo=400,
            Hq=28, Hkv=4, Dh=128, d=3584, V=152064, dtype="bf16"),
    5: dict(name="eviction-density sweep: 1x131072 tokens, 32/8 heads Dh 128",
            n_traj=1, T=131072, summary=0, prompt=256, Lp=200, Lo=400,
            Hq=32, Hkv=8, Dh=128, dtype="bf16",
            sweep_K=(1, 4, 8, 16, 32), sweep_f=(0.3, 0.6, 0.9)),
}


def record(n_traj, T, K, evict, summary, prompt, Lp, Lo, seed_base, on_policy_summary=False):
    """``n_traj`` trajectories; trajectory b uses seed ``seed_base + b``."""
    lens = T if isinstance(T, (list, tuple)) else [T] * n_traj
    return Record([trajectory(lens[b], K, evict, summary, prompt, Lp, Lo, seed_base + b, on_policy_summary)
                   for b in range(n_traj)])


def events_record(rec, retrieve, seed):
    """An offload / retrieve (MemexRL) record from a compression record: each
    junction offloads the spans the compression evicts (its out-spans), and
    every span offloaded at an earlier junction and still out comes back at a
    later junction with probability ``retrieve`` (its in-spans, in the order
    they were offloaded). Returns ``events_per_traj``: per trajectory a list
    of (J, out_spans, in_spans)."""
    rng = _rng(seed)
    out = []
    for t in rec.trajs:
        ev, offloaded = [], []
        for J, spans in t.edits:
            back = [s for s in offloaded if rng.random() < retrieve]
            offloaded = [s for s in offloaded if s not in back] + list(spans)
            ev.append((int(J), [tuple(s) for s in spans], [tuple(s) for s in back]))
        out.append(ev)
    return out


def config_record(cfg, K=None, f=None):
    """The record of workload ``cfg`` (1, 2, 4 or 5); seed = 1000*cfg + traj."""
    c = CONFIGS[cfg]
    if cfg == 5:
        return record(1, c["T"], K, f, c["summary"], c["prompt"], c["Lp"], c["Lo"],
                      1000 * cfg + 100 * K + int(round(10 * f)))
    return record(c["n_traj"], c["T"], c["K"], c["evict"], c["summary"], c["prompt"],
                  c["Lp"], c["Lo"], 1000 * cfg)


def loss_rows_fraction(N, frac, seed):
    """``round(frac * N)`` distinct rows drawn by a seeded permutation, sorted."""
    M = int(round(frac * N))
    return np.sort(_rng(seed).permutation(N)[:M]).astype(np.int64)


# --- tensors ----------------------------------------------------------------

def normal(shape, seed, std=1.0):
    """float32 N(0, std^2) tensor on the CPU from a seeded torch generator."""
    import torch
    g = torch.Generator().manual_seed(int(seed))
    t = torch.randn(*shape, generator=g, dtype=torch.float32)
    return t.mul_(std) if std != 1.0 else t


def uniform_int(n, high, seed):
    """int32 tensor of n values uniform over [0, high)."""
    import torch
    g = torch.Generator().manual_seed(int(seed))
    return torch.randint(0, high, (n,), generator=g, dtype=torch.int64).to(torch.int32)
