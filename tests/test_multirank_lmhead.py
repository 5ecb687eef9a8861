"""The LM head's exchange steps if the path were sharded over GPUs, run as two
gloo ranks on CPU (no GPU, no NCCL).

One box has one GPU, so the bench runs replicas; the sharded design is
recorded and its arithmetic checked here against the single-process oracle:

* vocabulary-parallel log-probs: each rank holds a slice of W, computes its
  slice's logits, and the ranks exchange three numbers per loss row: the max
  (all-reduce MAX), the sum of exp(z - max) rescaled to the global max
  (all-reduce SUM) and the target logit (all-reduce MAX, -inf on ranks that
  do not hold the target);
* row-parallel backward: each rank holds half of the loss rows; dH rows are
  disjoint and dW is summed (all-reduce SUM).

Both are the same merges the single-GPU kernels do over vocabulary chunks and
row tiles.
"""

import os
import socket
import sys

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _case():
    g = np.random.default_rng(31)
    N, d, V, M = 24, 8, 101, 17
    H = g.standard_normal((N, d))
    W = g.standard_normal((V, d)) * 0.5
    targets = g.integers(0, V, N)
    rows = np.sort(g.permutation(N)[:M])
    lp_old = g.standard_normal(M) * 0.1 - 4.0
    adv = g.standard_normal(M)
    return H, W, targets, rows, lp_old, adv


def _rank_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    from oracle import logprob as LP
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        H, W, targets, rows, lp_old, adv = _case()
        V = W.shape[0]
        # --- vocabulary-parallel forward
        lo, hi = rank * V // world, (rank + 1) * V // world
        z = LP.logits(H, W[lo:hi], rows)                     # this rank's slice of the logits
        m = torch.from_numpy(z.max(axis=1))
        dist.all_reduce(m, op=dist.ReduceOp.MAX)
        s = torch.from_numpy(np.exp(z - m.numpy()[:, None]).sum(axis=1))
        dist.all_reduce(s, op=dist.ReduceOp.SUM)
        t = targets[rows]
        own = (t >= lo) & (t < hi)
        zt = np.where(own, z[np.arange(len(rows)), np.clip(t - lo, 0, hi - lo - 1)], -np.inf)
        zt = torch.from_numpy(zt)
        dist.all_reduce(zt, op=dist.ReduceOp.MAX)
        lse = m.numpy() + np.log(s.numpy())
        lp = zt.numpy() - lse
        # --- row-parallel backward: this rank's half of the loss rows
        _, _, _, g = LP.policy_loss(lp, lp_old, adv, 0.2, 0.28)
        mine = np.arange(len(rows)) % world == rank
        dH, dW = LP.logprob_loss_bwd(H, W, targets, rows[mine], lse[mine], g[mine])
        dW = torch.from_numpy(dW)
        dist.all_reduce(dW, op=dist.ReduceOp.SUM)
        np.savez(os.path.join(out_dir, f"rank{rank}.npz"), lp=lp, lse=lse, dW=dW.numpy(), dH=dH)
    finally:
        dist.destroy_process_group()


def test_sharded_lm_head_over_two_gloo_ranks(tmp_path):
    sys.path.insert(0, ROOT)
    from oracle import logprob as LP
    mp.start_processes(_rank_main, args=(2, _free_port(), str(tmp_path)), nprocs=2, start_method="spawn",
                       join=True)
    H, W, targets, rows, lp_old, adv = _case()
    lp_ref, lse_ref = LP.logprob(H, W, targets, rows)
    _, _, _, g = LP.policy_loss(lp_ref, lp_old, adv, 0.2, 0.28)
    dH_ref, dW_ref = LP.logprob_loss_bwd(H, W, targets, rows, lse_ref, g)
    outs = [np.load(tmp_path / f"rank{r}.npz") for r in range(2)]
    for o in outs:
        np.testing.assert_allclose(o["lp"], lp_ref, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(o["lse"], lse_ref, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(o["dW"], dW_ref, rtol=1e-10, atol=1e-12)
    # dH: each rank writes only its own loss rows; together they are the full dH
    np.testing.assert_allclose(outs[0]["dH"] + outs[1]["dH"], dH_ref, rtol=1e-10, atol=1e-12)
