"""Benchmark: view-consistent scored tokens/s (fwd+bwd) of the whole hot path.

Default workload (N=1): the 7B-shaped layer step -- 2 x 65,536 tokens, 8
junctions per trajectory at 70% eviction with 1,024-token summaries, masked
GQA attention 28/4 heads Dh 128 fwd+bwd chained into the fused LM-head
log-prob + clipped loss (d = 3,584, V = 152,064) fwd+bwd. One step runs every
step of the path: visibility build, attention fwd, LM-head fwd + loss,
LM-head bwd, attention bwd (dO = dH). Scored tokens are the loss rows.
Other workloads: ``--config 2`` (attention op, 8 x 16,384), ``--config 3``
(log-prob loss, N = 32,768), ``--config 5 --K k --f f`` (one sweep point).

``--impl reference`` times the CPU oracle (the only reference this method has)
on a bounded sample of the same workload. Under torchrun every rank runs its
own replica (trajectories are independent): weak scaling, no collective on
the data path; rank 0 prints one JSON line.
"""

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "view-consistent scored tokens/sec (fwd+bwd)"


# PPO / GRPO clip range of the loss: App. F.1 trains with the asymmetric 0.2 / 0.28
EPS_LO, EPS_HI = 0.2, 0.28
# Device-resident model state, not re-uploaded by the end-to-end leg
RESIDENT = ("W",)


def _peaks():
    """(bf16 burst TFLOP/s, bf16 sustained TFLOP/s, HBM GB/s, source)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), float(p["bf16_tflops_sustained"]), float(p["hbm_gbs"]), "measured"
    except Exception:
        return 1900.0, 1700.0, 6800.0, "fallback"


# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per call of a
# dominant C-ABI call, from one ncu capture of the same bench command (summaries
# in profiles/). Reported only while the kernel source still hashes to the
# value it had when the counters were taken.
TRAFFIC = {
    (4, "mw_logprob_loss_bwd"): {
        "bytes": 456960 + (85569901056 + 14106740992) + (807919104 + 246921728),   # par, dW pass, dH from E
        "source": "paper_2609_00865_gb300/csrc/lmhead_bwd_tc.cu",
        "sha256": "56a02b5f128d1f4b9db9970e594ef9bf271e86f7f2ebd358a2e4d32f744c1b29",
    },
    (4, "mw_masked_attn_bwd"): {
        # lsd, compact gather, dQ (main + junction items), dK/dV, per-key reduce
        "bytes": (1894792704 + 28215296) + (457391872 + 700431872) + (4153245696 + 902921984) +
                 (515885568 + 6489344) + (2745335296 + 1457336064) + (1502192128 + 262524160),
        "source": "paper_2609_00865_gb300/csrc/attn_tc.cu",
        "sha256": "48d36168ce7bd2c054b9c265005945bbb82edcd5661adb8804942cc689e65178",
    },
}


def _traffic(cfg, call):
    import hashlib
    t = TRAFFIC.get((cfg, call))
    if t is None:
        return None
    try:
        with open(os.path.join(ROOT, t["source"]), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != t["sha256"]:
                return None
    except OSError:
        return None
    return t["bytes"]


class Clocks:
    """nvidia-smi sampler running while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = tempfile.mktemp(suffix=".csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx = max(mx, float(p[2]))
            except ValueError:
                continue
            for n, v in zip(names, p[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- workloads

def replica_seed(cfg, rank):
    """Seed of rank ``rank``'s replica: every rank scores its own independent
    synthetic batch (weak scaling)."""
    return 1000 * cfg + 17 + rank


def reduce_max(x, world, device=None):
    """Max of ``x`` over the ranks of the default process group (identity at
    world 1): the job's time is its slowest rank's."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(scored_per_rank, world, ms):
    """Whole-job throughput: the units all ranks processed over the job's time."""
    return scored_per_rank * world / (ms * 1e-3)


def make_workload(cfg, K=None, f=None, seed_offset=0, n_traj=None, pin=True, rope=None, events=None):
    """Host-side inputs of one workload (CPU tensors, pinned unless ``pin`` is
    False, + record).

    ``n_traj`` keeps only the first trajectories of the record (a smaller
    case of the same kernels, for profiler captures). ``rope`` (a rotary
    theta) runs the attention with row-wise logical rotary positions.
    ``events`` (a retrieve probability) turns the record into an offload /
    retrieve record (``synth.events_record``): the compressions' evicted spans
    are offloaded and come back at later junctions."""
    import numpy as np
    import torch

    import synth
    c = synth.CONFIGS[cfg]
    g = torch.Generator().manual_seed(replica_seed(cfg, seed_offset))
    w = {"cfg": cfg}
    if rope is not None and cfg in (2, 4, 5):
        w["rope"] = float(rope)
    bf = torch.bfloat16

    def randn(*shape, std=1.0):
        t = torch.randn(*shape, generator=g, dtype=torch.float32)
        if std != 1.0:
            t.mul_(std)
        t = t.to(bf)
        return t.pin_memory() if pin else t

    if cfg == 5:
        w["sweep"] = (K, f)
    if cfg in (2, 4, 5):
        rec = synth.config_record(cfg, K=K, f=f)
        if n_traj:
            rec = synth.Record(rec.trajs[:n_traj])
        w["record"] = rec
        if events is not None:
            w["events"] = synth.events_record(rec, float(events), 7000 + cfg)
            w["events_p"] = float(events)
        T = rec.total
        w["Q"] = randn(T, c["Hq"], c["Dh"])
        w["K"] = randn(T, c["Hkv"], c["Dh"])
        w["V"] = randn(T, c["Hkv"], c["Dh"])
        w["heads"] = (c["Hq"], c["Hkv"], c["Dh"])
        if cfg != 4:
            w["dO"] = randn(T, c["Hq"], c["Dh"])
    if cfg in (3, 4):
        if cfg == 3:
            N, d = c["N"], c["d"]
            rows = synth.loss_rows_fraction(N, c["loss_frac"], 3000)
            w["H"] = randn(N, d)
        else:
            N, d = w["record"].total, c["Hq"] * c["Dh"]
            rows = w["record"].loss_rows()
        w["N"], w["d"], w["Vocab"] = N, d, c["V"]
        w["W"] = randn(c["V"], d, std=0.02)
        w["targets"] = torch.randint(0, c["V"], (N,), generator=g, dtype=torch.int32)
        w["rows"] = torch.tensor(rows, dtype=torch.int32)
        M = len(rows)
        w["adv"] = torch.randn(M, generator=g)
        w["noise"] = 0.05 * torch.randn(M, generator=g)
        if pin:
            for k in ("targets", "rows", "adv", "noise"):
                w[k] = w[k].pin_memory()
    return w


def e2e_inputs(w, device_keys):
    """The host tensors the end-to-end leg uploads every step: the workload's
    per-step inputs that the step holds on the device, not the resident model
    state (RESIDENT)."""
    import torch
    return {k: v for k, v in w.items()
            if isinstance(v, torch.Tensor) and k in device_keys and k not in RESIDENT}


def describe(w):
    import synth
    c = synth.CONFIGS[w["cfg"]]
    d = {"workload": c["name"]}
    if "record" in w:
        r = w["record"]
        d.update(trajectories=len(r.trajs), tokens=r.total,
                 junctions=sum(len(e) for e in r.edits), heads=f"{w['heads'][0]}/{w['heads'][1]}",
                 head_dim=w["heads"][2])
    if "rows" in w:
        d.update(loss_rows=int(w["rows"].numel()), hidden=w["d"], vocab=w["Vocab"])
    if "sweep" in w:
        d.update(sweep_K=w["sweep"][0], evicted_fraction=w["sweep"][1])
    if "rope" in w:
        d["rope_theta"] = w["rope"]
    if "events" in w:
        d["views"] = "offload / retrieve events (MemexRL): evicted spans offloaded, " \
                     f"each brought back at a later junction with p = {w['events_p']}"
        d["retrieved_spans"] = sum(len(i) for e in w["events"] for _, _, i in e)
    d["l2"] = "inputs larger than L2 (129 MB); no flush"
    return d


class Step:
    """Device buffers and one pass of the hot path through the public API."""

    def __init__(self, w, device):
        import torch

        import paper_2609_00865_gb300 as mw
        self.mw = mw
        self.w = w
        self.dev = device
        self.stream = torch.cuda.current_stream(device)
        self.d = {k: v.to(device, non_blocking=True) for k, v in w.items() if isinstance(v, torch.Tensor)}
        self.events = {}
        self.timing = False
        if "record" in w:
            r = w["record"]
            if "events" in w:
                self.flat = mw.flatten_events(r.seqlens, w["events"])
                self.L = mw.mw_events_layout(self.flat[0], self.flat[2], len(self.flat[-1]))
            else:
                self.flat = mw.flatten_record(r.seqlens, r.edits)
                cu, J, jt, off, spans = self.flat
                self.L = mw.mw_visibility_layout(cu, jt, len(spans))
            self.vis = mw.Visibility(self.L, torch.empty(self.L.vis_bytes, dtype=torch.uint8, device=device),
                                     torch.empty(max(self.L.ws_bytes, 1), dtype=torch.uint8, device=device))
            Hq, Hkv, Dh = w["heads"]
            self.scale = Dh ** -0.5
            T = r.total
            self.O = torch.empty(T, Hq, Dh, dtype=torch.bfloat16, device=device)
            self.LSE = torch.empty(Hq, T, dtype=torch.float32, device=device)
            self.dQ = torch.empty_like(self.O)
            self.dK = torch.empty(T, Hkv, Dh, dtype=torch.bfloat16, device=device)
            self.dV = torch.empty_like(self.dK)
            if "rope" in w:
                # positions per (segment, key) and the cos/sin table (built once,
                # like weights); one workspace serves both calls (shared prefix)
                self.pos = torch.empty(max(self.L.n_keymask * mw.TILE, 1), dtype=torch.int32, device=device)
                self.table = mw.rope_table(mw.TILE * self.L.max_tiles, Dh, w["rope"], device=device)
                nb = mw.mw_masked_attn_rope_ws(self.vis, Hq, Hkv, Dh, mw.MW_BF16)[1]
            else:
                nb = mw.mw_masked_attn_bwd_ws(self.vis, Hq, Hkv, Dh, mw.MW_BF16)
                nf = mw.mw_masked_attn_fwd_ws(self.vis, Hkv, Dh, mw.MW_BF16)
                self.attn_fwd_ws = torch.empty(max(nf, 1), dtype=torch.uint8, device=device)
            self.attn_ws = torch.empty(max(nb, 1), dtype=torch.uint8, device=device)
        if "rows" in w:
            M = int(w["rows"].numel())
            N, d, V = w["N"], w["d"], w["Vocab"]
            self.lm_ws = torch.empty(max(mw.mw_logprob_ws(N, M, d, V, mw.MW_BF16), 1), dtype=torch.uint8,
                                     device=device)
            self.lp = torch.empty(M, dtype=torch.float32, device=device)
            self.ratio = torch.empty_like(self.lp)
            self.lse = torch.empty_like(self.lp)
            self.loss = torch.empty(1, dtype=torch.float32, device=device)
            self.dH = torch.empty(N, d, dtype=torch.bfloat16, device=device)
            self.dW = torch.empty(V, d, dtype=torch.float32, device=device)
            self.lp_old = torch.empty(M, dtype=torch.float32, device=device)

    def _ev(self, name, fn):
        import torch
        if not self.timing:
            return fn()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(self.stream)
        r = fn()
        b.record(self.stream)
        self.events.setdefault(name, []).append((a, b))
        return r

    def H(self):
        return self.O.view(self.O.shape[0], -1) if self.w["cfg"] == 4 else self.d["H"]

    def prime(self):
        """lp_old = current log-prob + N(0, 0.05) (computed once, untimed)."""
        if "rows" not in self.w:
            return
        if "record" in self.w:
            self.build()
            self.attn_fwd()
        self.d["lp_old"] = self.lp_old
        self.lp_old.zero_()
        self.lm_fwd()
        self.lp_old.copy_(self.lp + self.d["noise"])

    def build(self):
        if "events" in self.w:
            cu, J, jt, oo, io, spans = self.flat
            self._ev("mw_build_views_events", lambda: self.mw.mw_build_views_events(
                self.L, cu, J, jt, oo, io, spans, self.vis.ws, self.vis.vis, self.stream))
        else:
            cu, J, jt, off, spans = self.flat
            self._ev("mw_build_visibility", lambda: self.mw.mw_build_visibility(
                self.L, cu, J, jt, off, spans, self.vis.ws, self.vis.vis, self.stream))
        if "rope" in self.w:
            self._ev("mw_logical_positions", lambda: self.mw.mw_logical_positions(self.vis, self.pos, self.stream))

    def attn_fwd(self):
        if "rope" in self.w:
            self._ev("mw_masked_attn_rope_fwd", lambda: self.mw.mw_masked_attn_rope_fwd(
                self.vis, self.pos, self.table, self.d["Q"], self.d["K"], self.d["V"], self.O, self.LSE,
                self.scale, self.attn_ws, self.stream))
            return
        self._ev("mw_masked_attn_fwd", lambda: self.mw.mw_masked_attn_fwd(
            self.vis, self.d["Q"], self.d["K"], self.d["V"], self.O, self.LSE, self.scale, self.attn_fwd_ws,
            self.stream))

    def attn_bwd(self, dO):
        if "rope" in self.w:
            self._ev("mw_masked_attn_rope_bwd", lambda: self.mw.mw_masked_attn_rope_bwd(
                self.vis, self.pos, self.table, self.d["Q"], self.d["K"], self.d["V"], self.O, dO, self.LSE,
                self.dQ, self.dK, self.dV, self.scale, self.attn_ws, self.stream))
            return
        self._ev("mw_masked_attn_bwd", lambda: self.mw.mw_masked_attn_bwd(
            self.vis, self.d["Q"], self.d["K"], self.d["V"], self.O, dO, self.LSE, self.dQ, self.dK, self.dV,
            self.scale, self.attn_ws, self.stream))

    def lm_fwd(self):
        self._ev("mw_logprob_loss_fwd", lambda: self.mw.mw_logprob_loss_fwd(
            self.H(), self.d["W"], self.d["targets"], self.d["rows"], self.lp_old, self.d["adv"], EPS_LO, EPS_HI,
            self.lp, self.ratio, self.lse, self.loss, self.lm_ws, self.stream))

    def lm_bwd(self):
        self._ev("mw_logprob_loss_bwd", lambda: self.mw.mw_logprob_loss_bwd(
            self.H(), self.d["W"], self.d["targets"], self.d["rows"], self.lse, self.lm_ws, 1.0, self.dH, self.dW,
            self.stream))

    def run(self):
        cfg = self.w["cfg"]
        if cfg in (2, 5):
            self.build()
            self.attn_fwd()
            self.attn_bwd(self.d["dO"])
        elif cfg == 3:
            self.lm_fwd()
            self.lm_bwd()
        else:
            self.build()
            self.attn_fwd()
            self.lm_fwd()
            self.lm_bwd()
            self.attn_bwd(self.dH.view_as(self.O))

    def upload(self, host):
        """e2e: copy this step's inputs from pinned host memory."""
        for k, v in host.items():
            if k in self.d:
                self.d[k].copy_(v, non_blocking=True)

    def scored(self):
        return int(self.w["rows"].numel()) if "rows" in self.w else self.w["record"].total

    def tile_stats(self):
        """Attention work skipped by the visibility structure, against plain
        causal attention of the same trajectory lengths: 128x128 tiles listed
        (non-empty) vs causal tiles, visible pairs vs causal pairs."""
        if "record" not in self.w or "events" in self.w:   # event views have no tile lists
            return None
        import numpy as np
        L = self.vis.layout
        listed = int(self.vis._arr(L.off_fwd_ptr + 4 * L.n_tiles, 1, np.int32)[0])
        causal_pairs = sum(t * (t + 1) // 2 for t in self.w["record"].seqlens)
        return {"tiles_listed": listed, "tiles_causal": int(L.n_tri),
                "skipped_tile_frac": 1.0 - listed / max(1, int(L.n_tri)),
                "visible_pairs": int(self.vis.pairs_total), "causal_pairs": int(causal_pairs),
                "visible_pair_frac": int(self.vis.pairs_total) / max(1, causal_pairs)}

    def call_flops(self):
        """Algorithmic FLOPs of each timed C-ABI call of the step."""
        f = self.flops()
        return {"mw_masked_attn_fwd": 4.0 / 14.0 * f.get("attn", 0),
                "mw_masked_attn_bwd": 10.0 / 14.0 * f.get("attn", 0),
                "mw_masked_attn_rope_fwd": 4.0 / 14.0 * f.get("attn", 0),
                "mw_masked_attn_rope_bwd": 10.0 / 14.0 * f.get("attn", 0),
                # the forward forms the logits and E = sum_v p_v W_v (the dH
                # product); the backward recomputes the logits for dW
                "mw_logprob_loss_fwd": 4.0 / 8.0 * f.get("lm", 0),
                "mw_logprob_loss_bwd": 4.0 / 8.0 * f.get("lm", 0)}

    def flops(self):
        """Visible FLOPs per step: attention 14 P Dh Hq, LM head 8 M d V."""
        f = {}
        if "record" in self.w:
            Hq, _, Dh = self.w["heads"]
            f["attn"] = 14.0 * self.vis.pairs_total * Dh * Hq
        if "rows" in self.w:
            f["lm"] = 8.0 * self.w["rows"].numel() * self.w["d"] * self.w["Vocab"]
        return f


class PackedStep(Step):
    """One layer of the stacked-layer step (App. G's branch-replicated
    packing, the design for more than one layer): every segment's live view
    is packed as a branch of its own (mw_branch_pack of Q, K, V and the
    upstream dO, through the compact maps of the record's visibility build),
    the layer's attention runs causally over the packed branches (one build of
    the packed record: a trajectory per branch, no junctions), and the packed
    copies' gradients are summed back per token (mw_branch_unpack_add of dQ,
    dK, dV). A stack of L layers repeats the attention L times between one
    pack and one unpack. The branch lengths are structure of the record,
    read once (untimed); both builds are timed."""

    def __init__(self, w, device):
        import torch
        super().__init__(w, device)
        mw = self.mw
        Hq, Hkv, Dh = w["heads"]
        self.build()
        lens = mw.branch_lengths(self.vis)
        torch.cuda.synchronize()
        self.n = n = int(sum(lens))
        self.flat_p = mw.flatten_record(lens, [[] for _ in lens])
        cu, J, jt, off, spans = self.flat_p
        self.L_p = mw.mw_visibility_layout(cu, jt, len(spans))
        self.vis_p = mw.Visibility(self.L_p, torch.empty(self.L_p.vis_bytes, dtype=torch.uint8, device=device),
                                   torch.empty(max(self.L_p.ws_bytes, 1), dtype=torch.uint8, device=device))
        bf = torch.bfloat16
        self.Qp = torch.empty(n, Hq, Dh, dtype=bf, device=device)
        self.dOp = torch.empty_like(self.Qp)
        self.Kp = torch.empty(n, Hkv, Dh, dtype=bf, device=device)
        self.Vp = torch.empty_like(self.Kp)
        self.Op = torch.empty_like(self.Qp)
        self.LSEp = torch.empty(Hq, n, dtype=torch.float32, device=device)
        self.dQp = torch.empty_like(self.Qp)
        self.dKp = torch.empty_like(self.Kp)
        self.dVp = torch.empty_like(self.Kp)
        self.attn_fwd_ws_p = torch.empty(max(mw.mw_masked_attn_fwd_ws(self.vis_p, Hkv, Dh, mw.MW_BF16), 1),
                                         dtype=torch.uint8, device=device)
        self.attn_ws_p = torch.empty(max(mw.mw_masked_attn_bwd_ws(self.vis_p, Hq, Hkv, Dh, mw.MW_BF16), 1),
                                     dtype=torch.uint8, device=device)
        torch.cuda.synchronize()

    def run(self):
        mw = self.mw
        self.build()
        cu, J, jt, off, spans = self.flat_p
        self._ev("mw_build_visibility (packed)", lambda: mw.mw_build_visibility(
            self.L_p, cu, J, jt, off, spans, self.vis_p.ws, self.vis_p.vis, self.stream))
        for X, Xp in ((self.d["Q"], self.Qp), (self.d["K"], self.Kp), (self.d["V"], self.Vp),
                      (self.d["dO"], self.dOp)):
            self._ev("mw_branch_pack", lambda: mw.mw_branch_pack(self.vis, X, Xp, self.stream))
        self._ev("mw_masked_attn_fwd", lambda: mw.mw_masked_attn_fwd(
            self.vis_p, self.Qp, self.Kp, self.Vp, self.Op, self.LSEp, self.scale, self.attn_fwd_ws_p, self.stream))
        self._ev("mw_masked_attn_bwd", lambda: mw.mw_masked_attn_bwd(
            self.vis_p, self.Qp, self.Kp, self.Vp, self.Op, self.dOp, self.LSEp, self.dQp, self.dKp, self.dVp,
            self.scale, self.attn_ws_p, self.stream))
        for dXp, dX in ((self.dQp, self.dQ), (self.dKp, self.dK), (self.dVp, self.dV)):
            self._ev("mw_branch_unpack_add", lambda: mw.mw_branch_unpack_add(self.vis, dXp, dX, self.stream))

    def tile_stats(self):
        return None

    def flops(self):
        """Visible FLOPs of the layer: 14 P Dh Hq over the packed branches
        (P counts every packed row's causal keys, trunk copies included)."""
        Hq, _, Dh = self.w["heads"]
        return {"attn": 14.0 * self.vis_p.pairs_total * Dh * Hq}


class SdccStep(Step):
    """SDCC training step on the 7B-shaped layer (§5, Eq. "soft_loss"): the
    teacher is the masked attention under each row's live view (forward
    only, gradients stopped); the student is causal attention over each
    trajectory's final compressed walk, with the clipped task loss on the
    loss rows whose token survives on the walk (each predicted by the walk row
    before it) plus lam * KL(teacher || student) at the diverging ones; the
    summed gradients run back through the student's attention. The walk and
    the diverging rows are structure of the record, found once (untimed) with
    mw_final_walk / mw_diverging_rows; the student's own Q / K / V are
    synthetic inputs of the walk's length."""

    LAM = 0.1

    def __init__(self, w, device):
        import numpy as np
        import torch
        super().__init__(w, device)
        mw = self.mw
        r = w["record"]
        Hq, Hkv, Dh = w["heads"]
        self.build()
        wi, sr, wl = mw.final_walk(self.vis)
        div = mw.diverging_rows(self.vis)
        torch.cuda.synchronize()
        wi, sr, div = wi.cpu().numpy(), sr.cpu().numpy(), div.cpu().numpy()
        wl = wl.cpu().numpy()[: len(r.trajs)].astype(np.int64)
        woff = np.concatenate([[0], np.cumsum(wl)])
        tok = np.concatenate([[0], np.cumsum(r.seqlens)])
        rows = w["rows"].numpy().astype(np.int64)
        leaves, srow, p_t, p_s = [], [], [], []
        for m, rr in enumerate(rows):
            b = int(np.searchsorted(tok, rr, side="right") - 1)
            if rr + 1 >= tok[b + 1] or wi[rr + 1] < 0:
                continue                      # the leaf is evicted: no student score
            s_row = int(woff[b] + sr[rr])
            leaves.append(m)
            srow.append(s_row)
            if div[rr]:
                p_t.append(int(rr))
                p_s.append(s_row)
        self.Tw = int(woff[-1])
        self.walk_lens = [int(x) for x in wl]
        self.n_leaves, self.n_pairs = len(leaves), len(p_t)
        g = torch.Generator().manual_seed(4242)
        pin = lambda t: t.pin_memory()   # noqa: E731
        tgt = torch.zeros(self.Tw, dtype=torch.int32)
        tgt[torch.tensor(srow, dtype=torch.int64)] = w["targets"][torch.tensor(rows[leaves], dtype=torch.int64)]
        host = {"Qs": torch.randn(self.Tw, Hq, Dh, generator=g).to(torch.bfloat16),
                "Ks": torch.randn(self.Tw, Hkv, Dh, generator=g).to(torch.bfloat16),
                "Vs": torch.randn(self.Tw, Hkv, Dh, generator=g).to(torch.bfloat16),
                "tgt_s": tgt, "rows_s": torch.tensor(srow, dtype=torch.int32),
                "adv_s": w["adv"][torch.tensor(leaves, dtype=torch.int64)].clone(),
                "noise_s": w["noise"][torch.tensor(leaves, dtype=torch.int64)].clone(),
                "pair_t": torch.tensor(p_t, dtype=torch.int32), "pair_s": torch.tensor(p_s, dtype=torch.int32)}
        for k, v in host.items():
            w[k] = pin(v)
            self.d[k] = w[k].to(device, non_blocking=True)
        # student record: the walks, no edits
        self.flat_s = mw.flatten_record(self.walk_lens, [[] for _ in self.walk_lens])
        cu, J, jt, off, spans = self.flat_s
        self.Ls = mw.mw_visibility_layout(cu, jt, 0)
        self.vis_s = mw.Visibility(self.Ls, torch.empty(self.Ls.vis_bytes, dtype=torch.uint8, device=device),
                                   torch.empty(max(self.Ls.ws_bytes, 1), dtype=torch.uint8, device=device))
        mk = lambda *sh, dt=torch.bfloat16: torch.empty(*sh, dtype=dt, device=device)   # noqa: E731
        self.Os, self.LSEs = mk(self.Tw, Hq, Dh), mk(Hq, self.Tw, dt=torch.float32)
        self.dQs, self.dKs, self.dVs = mk(self.Tw, Hq, Dh), mk(self.Tw, Hkv, Dh), mk(self.Tw, Hkv, Dh)
        self.ws_fs = mk(max(mw.mw_masked_attn_fwd_ws(self.vis_s, Hkv, Dh, mw.MW_BF16), 1), dt=torch.uint8)
        self.ws_bs = mk(max(mw.mw_masked_attn_bwd_ws(self.vis_s, Hq, Hkv, Dh, mw.MW_BF16), 1), dt=torch.uint8)
        d, V, M = w["d"], w["Vocab"], self.n_leaves
        self.lm_ws_s = mk(max(mw.mw_logprob_ws(self.Tw, M, d, V, mw.MW_BF16), 1), dt=torch.uint8)
        f32 = lambda n: mk(max(n, 1), dt=torch.float32)   # noqa: E731
        self.lp_s, self.ratio_s, self.lse_s, self.lp_old_s = f32(M), f32(M), f32(M), f32(M)
        self.dHs = mk(self.Tw, d)
        self.kl_ws = mk(max(mw.mw_forward_kl_ws(self.n_pairs, d, V, mw.MW_BF16), 1), dt=torch.uint8)
        self.kl, self.loss_kl = f32(self.n_pairs), f32(1)

    def build_student(self):
        cu, J, jt, off, spans = self.flat_s
        self._ev("mw_build_visibility (student)", lambda: self.mw.mw_build_visibility(
            self.Ls, cu, J, jt, off, spans, self.vis_s.ws, self.vis_s.vis, self.stream))

    def prime(self):
        """Student lp_old = its current log-prob + N(0, 0.05) (once, untimed)."""
        self.build()
        self.build_student()
        self.attn_fwd_student()
        self.lp_old_s.zero_()
        self.d["lp_old_s"] = self.lp_old_s
        self.lm_fwd_student()
        self.lp_old_s.copy_(self.lp_s + self.d["noise_s"])

    def attn_fwd_student(self):
        self._ev("mw_masked_attn_fwd (student)", lambda: self.mw.mw_masked_attn_fwd(
            self.vis_s, self.d["Qs"], self.d["Ks"], self.d["Vs"], self.Os, self.LSEs, self.scale, self.ws_fs,
            self.stream))

    def lm_fwd_student(self):
        self._ev("mw_logprob_loss_fwd", lambda: self.mw.mw_logprob_loss_fwd(
            self.Os.view(self.Tw, -1), self.d["W"], self.d["tgt_s"], self.d["rows_s"], self.lp_old_s,
            self.d["adv_s"], EPS_LO, EPS_HI, self.lp_s, self.ratio_s, self.lse_s, self.loss, self.lm_ws_s,
            self.stream))

    def run(self):
        mw = self.mw
        T = self.w["record"].total
        self.build()
        self.build_student()
        self.attn_fwd()                       # teacher (live views), no backward
        self.attn_fwd_student()
        self.lm_fwd_student()
        self._ev("mw_forward_kl_fwd", lambda: mw.mw_forward_kl_fwd(
            self.O.view(T, -1), self.d["pair_t"], self.Os.view(self.Tw, -1), self.d["pair_s"], self.d["W"], self.kl,
            self.loss_kl, self.kl_ws, self.LAM, self.stream))
        self._ev("mw_logprob_loss_bwd", lambda: self.mw.mw_logprob_loss_bwd(
            self.Os.view(self.Tw, -1), self.d["W"], self.d["tgt_s"], self.d["rows_s"], self.lse_s, self.lm_ws_s,
            1.0, self.dHs, self.dW, self.stream))
        self._ev("mw_forward_kl_bwd", lambda: mw.mw_forward_kl_bwd(
            self.O.view(T, -1), self.d["pair_t"], self.Os.view(self.Tw, -1), self.d["pair_s"], self.d["W"],
            self.kl_ws, self.dHs, self.dW, self.LAM, 1.0, True, self.stream))
        self._ev("mw_masked_attn_bwd (student)", lambda: self.mw.mw_masked_attn_bwd(
            self.vis_s, self.d["Qs"], self.d["Ks"], self.d["Vs"], self.Os, self.dHs.view_as(self.Os), self.LSEs,
            self.dQs, self.dKs, self.dVs, self.scale, self.ws_bs, self.stream))

    def scored(self):
        return self.n_leaves

    def flops(self):
        """Visible FLOPs: student attention 14 P_walk Dh Hq (causal over the
        walks), teacher forward 4 P Dh Hq, LM head 8 M d V on the surviving
        leaves, KL 12 M_kl d V (both logit products forward; recomputed, dH
        and dW backward)."""
        Hq, _, Dh = self.w["heads"]
        P_w = sum(n * (n + 1) // 2 for n in self.walk_lens)
        d, V = self.w["d"], self.w["Vocab"]
        return {"attn": 14.0 * P_w * Dh * Hq, "teacher": 4.0 * int(self.vis.pairs_total) * Dh * Hq,
                "lm": 8.0 * self.n_leaves * d * V, "kl": 12.0 * self.n_pairs * d * V}

    def call_flops(self):
        f = self.flops()
        return {"mw_masked_attn_fwd (student)": 4.0 / 14.0 * f["attn"],
                "mw_masked_attn_bwd (student)": 10.0 / 14.0 * f["attn"],
                "mw_masked_attn_fwd": f["teacher"],
                "mw_logprob_loss_fwd": 0.5 * f["lm"], "mw_logprob_loss_bwd": 0.5 * f["lm"],
                "mw_forward_kl_fwd": f["kl"] / 3.0, "mw_forward_kl_bwd": 2.0 * f["kl"] / 3.0}


# ----------------------------------------------------------------------------- reference arm (CPU oracle)

def cpu_sample(w, budget_s=15.0, seed=5, detail=False):
    """Time the oracle on a bounded sample of loss rows of this workload
    (rows drawn by ``seed``: the cost of a row grows with its view, so every
    sample draws its own rows).

    Per sampled row: attention fwd and the row's whole attention backward over
    all query heads (its segment's compact view: dQ and its contributions to
    dK and dV), LM-head log-prob over the full vocabulary and the dH/dW
    contributions of that row. Returns (tokens/s, cores, description), or
    with ``detail`` (tokens, seconds, cores, parts).
    """
    import numpy as np
    import torch

    from oracle import attention as OA
    from oracle import logprob as OL
    from oracle import nonmonotone as ON
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    if "_f64" not in w:   # exact float64 copies of the bf16 inputs, made once
        w["_f64"] = {k: w[k].to(torch.float64).numpy() for k in ("Q", "K", "V", "dO", "H", "W") if k in w}
    x = w["_f64"]
    rng = np.random.default_rng(seed)
    if "rows" in w:
        pool = w["rows"].numpy().astype(np.int64)
    else:
        pool = np.arange(w["record"].total)
    batch = 8

    def one_batch(rows):
        parts = []
        O = None
        if "record" in w:
            r = w["record"]
            Hq, Hkv, Dh = w["heads"]
            parts.append("attention fwd + bwd (dQ, dK, dV contributions), all heads")
            th = w.get("rope")
            rec, views = (w["events"], ON.live_views) if "events" in w else (r.edits, None)
            O, _ = OA.attn_fwd(r.seqlens, rec, x["Q"], x["K"], x["V"], Dh ** -0.5, rows=rows, rope_theta=th,
                               views=views)
            OA.attn_bwd_rows(r.seqlens, rec, x["Q"], x["K"], x["V"], x.get("dO", x["Q"]), Dh ** -0.5,
                             rows, list(range(Hq)), rope_theta=th, with_kv=True, views=views)
        if "rows" in w:
            parts.append("LM-head fwd over the full vocabulary + dH/dW")
            if "H" in x:
                H = x["H"]
            else:       # chained: H rows are the oracle's own attention outputs
                H = np.zeros((w["N"], w["d"]))
                H[rows] = O.reshape(len(rows), -1)
            lp, lse = OL.logprob(H, x["W"], w["targets"].numpy(), rows)
            g = OL.policy_loss(lp, lp + 0.01, np.ones_like(lp), EPS_LO, EPS_HI)[3]
            OL.logprob_loss_bwd(H, x["W"], w["targets"].numpy(), rows, lse, g)
        return parts

    # one untimed batch on the first call: the first batch of a process pays
    # one-time costs (thread pools, first touch of the float64 copies) that no
    # later batch does
    if not w.get("_warm"):
        one_batch(np.sort(rng.choice(pool, size=batch, replace=False)))
        w["_warm"] = True
    done, t0 = 0, time.perf_counter()
    parts = []
    while time.perf_counter() - t0 < budget_s and done < 4096:
        parts = one_batch(np.sort(rng.choice(pool, size=batch, replace=False)))
        done += batch
    dt = time.perf_counter() - t0
    if detail:
        return done, dt, cores, parts
    return done / dt, cores, f"{done} sampled scored tokens ({' + '.join(parts)}), {dt:.1f} s"


def run_reference(args, rank, world):
    if rank != 0:
        return
    w = make_workload(args.config, args.K, args.f, n_traj=args.n_traj, pin=False,   # the oracle runs on the host
                      rope=args.rope, events=args.events)
    # every step samples its own rows; the value is all timed steps' tokens
    # over their time (whole-job throughput, as the bench's own CPU baseline)
    tok, sec = 0, 0.0
    for i in range(args.warmup + args.steps):
        done, dt, cores, parts = cpu_sample(w, budget_s=args.cpu_seconds / max(1, args.steps), seed=5 + i,
                                            detail=True)
        if i >= args.warmup:
            tok, sec = tok + done, sec + dt
    v = tok / sec
    desc = f"{tok} sampled scored tokens over {args.steps} steps ({' + '.join(parts)}), {sec:.1f} s"
    scored = int(w["rows"].numel()) if "rows" in w else w["record"].total
    # one whole step at the sampled rate (extrapolated: each timed step is a sample)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * scored / v,
            "ms_per_step_kind": f"extrapolated: {scored} scored tokens per step at the sampled rate",
            "ms_per_scored_token": 1e3 / v, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": describe(w),
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": desc},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- GPU arm

def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    import paper_2609_00865_gb300 as mw
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = make_workload(args.config, args.K, args.f, seed_offset=rank, n_traj=args.n_traj, rope=args.rope,
                      events=args.events)
    step = SdccStep(w, dev) if args.sdcc else PackedStep(w, dev) if args.packed else Step(w, dev)
    step.prime()
    for _ in range(args.warmup):
        step.run()
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            dist.barrier()

    clocks = Clocks(local_rank)
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    step.timing = True
    n0 = mw.kernel_launches()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(step.stream)
    for _ in range(args.steps):
        step.run()
    ev1.record(step.stream)
    torch.cuda.synchronize()
    launches = mw.kernel_launches() - n0
    step.timing = False
    ms = ev0.elapsed_time(ev1) / args.steps
    clk = clocks.stop()
    barrier()
    ms = reduce_max(ms, world, dev)
    per_call = {k: sum(a.elapsed_time(b) for a, b in v) / len(v) for k, v in step.events.items()}

    # e2e: pinned host inputs -> device, step, loss/metric read back, every
    # step. The per-step inputs are uploaded; the LM-head weight W is model
    # state, resident on the device across steps as in a training loop.
    host = e2e_inputs(w, step.d)
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    out = step.loss if hasattr(step, "loss") else step.LSE[0, :1]
    d2h = out.numel() * out.element_size()
    pinned_out = torch.empty(out.shape, dtype=out.dtype).pin_memory()

    def e2e_prefetch():
        """As a training loop that prefetches its next batch does, step i + 1's
        inputs are copied on a copy stream while step i computes, into the
        other of two device input sets. (Measured against copying each step's
        inputs on its own stream right before it: that schedule also pays the
        copies' occasional slow runs, e.g. one 2.68 GB upload in 195 ms
        against 12.7 ms at the usual 211 GB/s, and measured 101.9 / 258.2 ms
        per step at the attention / 7B-layer workloads against 58.7 / 217.5.)"""
        base = step.d
        sets = [base, dict(base)]
        for k in host:
            sets[1][k] = torch.empty_like(base[k])
        copy = torch.cuda.Stream(dev)
        ready = [torch.cuda.Event(), torch.cuda.Event()]
        used = [torch.cuda.Event(), torch.cuda.Event()]

        def upload(i):
            with torch.cuda.stream(copy):
                for k, v in host.items():
                    sets[i % 2][k].copy_(v, non_blocking=True)
                ready[i % 2].record(copy)

        barrier()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(step.stream)
        copy.wait_event(e0)
        upload(0)
        for i in range(args.steps):
            if i + 1 < args.steps:
                if i >= 1:
                    copy.wait_event(used[(i + 1) % 2])   # step i - 1 read that set
                upload(i + 1)
            step.stream.wait_event(ready[i % 2])
            step.d = sets[i % 2]
            step.run()
            used[i % 2].record(step.stream)
            pinned_out.copy_(out, non_blocking=True)
        e1.record(step.stream)
        torch.cuda.synchronize()
        step.d = base
        return reduce_max(e0.elapsed_time(e1) / args.steps, world, dev)

    e2e_ms = e2e_prefetch()

    if rank != 0:
        return
    scored = step.scored()
    flops = step.flops()
    peak_tf, peak_sus, hbm, peak_kind = _peaks()
    dom = max(per_call, key=per_call.get)
    dom_flops = step.call_flops().get(dom, 0.0)
    achieved = dom_flops / (per_call[dom] * 1e-3) / 1e12
    total_tf = sum(flops.values()) / (ms * 1e-3) / 1e12
    cpu = None
    if world == 1 and not args.no_cpu and not args.sdcc and not args.packed:   # the oracle sample times the 4D-mask path
        v, cores, desc = cpu_sample(w, budget_s=args.cpu_seconds)
        cpu = {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": desc}
    line = {
        "metric": METRIC, "value": job_value(scored, world, ms), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": describe(w),
        "visible_tflops": total_tf, "visible_frac_of_peak": total_tf / peak_tf,
        "visible_frac_of_sustained_peak": total_tf / peak_sus,
        # the dominant call is timed inside the step loop (seconds of back-to-back
        # work under the power cap): the sustained peak is its denominator
        "roofline": {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peak_sus,
                     "unit": "TFLOP/s", "frac": achieved / peak_sus, "traffic": _traffic(w["cfg"], dom),
                     "peak_kind": f"bf16 dense sustained, {peak_kind} (burst {peak_tf})"},
        "per_call_ms": per_call,
        "cpu_baseline": cpu,
        "e2e": {"value": job_value(scored, world, e2e_ms), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                "upload": "pinned host -> device, every per-step input (W stays resident as model state); "
                          "step i + 1's inputs on a copy stream during step i"},
        "gpu_launches": launches,
        "clocks": clk,
    }
    if args.sdcc:
        line["config"].update(method="SDCC (§5): student over the final walks + lam KL at diverging leaves",
                              walk_tokens=step.Tw, scored_leaves=step.n_leaves, kl_pairs=step.n_pairs,
                              lam=step.LAM)
    if args.packed:
        line["config"].update(method="one stacked layer over branch-replicated packing (App. G): pack Q, K, V, dO; "
                                     "attention fwd + bwd over the packed branches; unpack dQ, dK, dV",
                              packed_rows=step.n, packed_visible_pairs=int(step.vis_p.pairs_total),
                              visible_pairs_4d_mask=int(step.vis.pairs_total))
    ts = step.tile_stats()
    if ts is not None:
        line["attention_tiles"] = ts
    print(json.dumps(line), flush=True)


BUILDER_BATCH = 64


def run_builder(args, rank, world, local_rank):
    """The visibility builder alone, batched: 64 sweep-shaped trajectories of
    131,072 tokens (K junctions at eviction fraction f) per build. One
    trajectory is a few MB of structure and launch-bound, so the builder's
    bandwidth is measured on the batch. HBM roofline over the builder's
    algorithmic bytes: the packed record read once (12 B per evicted span,
    the per-trajectory and per-junction tables) and the structure written
    once (all of it but the compact source lists past each segment's last
    compact tile, which stay unspecified). The record is host data by the builder's API (the
    call packs it and uploads the span list), so the timed call includes that
    upload: ``value`` and ``e2e`` are the same measurement."""
    import numpy as np
    import torch

    import paper_2609_00865_gb300 as mw
    import synth
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    c = synth.CONFIGS[5]
    seed = 1000 * 5 + 100 * args.K + int(round(10 * args.f)) + 10000 * (rank + 1)
    rec = synth.record(BUILDER_BATCH, c["T"], args.K, args.f, c["summary"], c["prompt"], c["Lp"], c["Lo"], seed)
    cu, J, jt, off, spans = mw.flatten_record(rec.seqlens, rec.edits)
    L = mw.mw_visibility_layout(cu, jt, len(spans))
    vis = mw.Visibility(L, torch.empty(L.vis_bytes, dtype=torch.uint8, device=dev),
                        torch.empty(max(L.ws_bytes, 1), dtype=torch.uint8, device=dev))
    stream = torch.cuda.current_stream(dev)

    def build():
        mw.mw_build_visibility(L, cu, J, jt, off, spans, vis.ws, vis.vis, stream)

    for _ in range(args.warmup):
        build()
    torch.cuda.synchronize()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    clocks = Clocks(local_rank)
    torch.cuda.synchronize()
    clocks.start()
    n0 = mw.kernel_launches()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        build()
    e1.record(stream)
    torch.cuda.synchronize()
    launches = mw.kernel_launches() - n0
    clk = clocks.stop()
    ms = reduce_max(e0.elapsed_time(e1) / args.steps, world, dev)
    if rank != 0:
        return
    # dense-mask export (bit-packed T x T per trajectory; T^2 / 8 bytes written)
    # of the attention workload's record, 8 trajectories of 16,384 tokens
    r2 = synth.config_record(2)
    vis2 = mw.build_visibility(r2.seqlens, r2.edits)
    masks = [torch.empty(T * ((T + 31) // 32), dtype=torch.int32, device=dev) for T in r2.seqlens]
    cu2 = np.zeros(len(r2.seqlens) + 1, dtype=np.int32)
    cu2[1:] = np.cumsum(r2.seqlens)

    def export_all():
        for b, m in enumerate(masks):
            mw.mw_export_dense_mask(vis2, cu2, b, m, stream)

    for _ in range(args.warmup):
        export_all()
    torch.cuda.synchronize()
    m0 = torch.cuda.Event(enable_timing=True)
    m1 = torch.cuda.Event(enable_timing=True)
    m0.record(stream)
    for _ in range(args.steps):
        export_all()
    m1.record(stream)
    torch.cuda.synchronize()
    mask_ms = m0.elapsed_time(m1) / args.steps
    mask_bytes = sum(m.numel() * 4 for m in masks)

    n_spans = int(L.n_spans)
    # written: the whole structure except csrc past each segment's last compact
    # tile (left unspecified); read: the packed span list and the small tables
    seg_len = vis.seg_len.astype(np.int64)
    csrc_used = 4 * mw.TILE * int(((seg_len + mw.TILE - 1) // mw.TILE).sum())
    nbytes = (int(L.vis_bytes) - 4 * mw.TILE * int(L.n_keymask) + csrc_used
              + 12 * n_spans + 4 * (len(rec.seqlens) + 1) + 8 * int(L.n_junc))
    peak_tf, peak_sus, hbm, peak_kind = _peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    tokens = rec.total
    value = job_value(tokens, world, ms)
    line = {
        "metric": "visibility-build tokens/sec", "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": f"visibility builder batched: {BUILDER_BATCH}x{c['T']} tokens, "
                               f"{args.K} junctions at {args.f}",
                   "trajectories": len(rec.seqlens), "tokens": tokens, "junctions": int(L.n_junc),
                   "evicted_spans": n_spans, "listed_tiles": int(L.n_tiles), "structure_bytes": int(L.vis_bytes),
                   "l2": "structure larger than L2 (129 MB); no flush"},
        "roofline": {"bound": "hbm", "kernel": "mw_build_visibility (all kernels + host packing)",
                     "achieved": gbs, "peak": hbm, "unit": "GB/s", "frac": gbs / hbm, "traffic": None,
                     "algorithmic_bytes": nbytes, "peak_kind": f"copy bandwidth, {peak_kind}"},
        "e2e": {"value": value, "unit": "tokens/s", "ms_per_step": ms,
                "note": "host record in, device structure out: the timed call packs and uploads the record"},
        "gpu_launches": launches,
        "clocks": clk,
        "dense_mask_export": {"workload": "8 x 16384-token trajectories of the attention workload",
                              "ms": mask_ms, "bytes_written": mask_bytes,
                              "gbs": mask_bytes / (mask_ms * 1e-3) / 1e9,
                              "frac_of_copy_peak": mask_bytes / (mask_ms * 1e-3) / 1e9 / hbm},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mw", choices=["mw", "reference"])
    ap.add_argument("--config", type=int, default=4, choices=[2, 3, 4, 5])
    ap.add_argument("--K", type=int, default=8)
    ap.add_argument("--f", type=float, default=0.6)
    ap.add_argument("--n-traj", type=int, default=None,
                    help="keep only the first trajectories (smaller case for profiler captures)")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--sdcc", action="store_true",
                    help="config 4: time SDCC's training step (§5) instead of the 4D-mask step")
    ap.add_argument("--rope", type=float, default=None, metavar="THETA",
                    help="attention with row-wise logical rotary positions (theta of the rotary table)")
    ap.add_argument("--builder", action="store_true",
                    help="time the visibility builder alone on 64 sweep trajectories (131,072 tokens, --K, --f)")
    ap.add_argument("--packed", action="store_true",
                    help="config 2: one stacked layer over branch-replicated packing (pack, attention over the "
                         "packed branches, unpack)")
    ap.add_argument("--events", type=float, default=None, metavar="P",
                    help="offload / retrieve views: the record's evicted spans are offloaded and each comes "
                         "back at a later junction with probability P (configs 2, 4, 5)")
    args = ap.parse_args()
    if args.sdcc and (args.config != 4 or args.rope is not None or args.events is not None):
        ap.error("--sdcc times the 7B-shaped layer step (config 4) without rotary positions or events")
    if args.packed and (args.config != 2 or args.sdcc or args.rope is not None or args.events is not None):
        ap.error("--packed runs config 2's attention on edits views without rotary positions")
    if args.events is not None and (args.config == 3 or args.builder or not 0.0 <= args.events <= 1.0):
        ap.error("--events P (0 <= P <= 1) needs a record: configs 2, 4, 5")
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", args.gpus if args.gpus == 1 else 1))
    local_rank = int(os.environ.get("LOCAL_RANK", 0))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if args.impl == "mw" else "gloo")
    if args.impl == "reference":
        run_reference(args, rank, world)
    elif args.builder:
        run_builder(args, rank, world, local_rank)
    else:
        run_gpu(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
