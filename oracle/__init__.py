"""CPU oracle for view-consistent scoring of compressed agent rollouts.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package. The product path (the CUDA library and its Python binding) never
imports, calls or links it, and this package imports nothing from the product.

What it computes follows the paper (MemoryWalker, arXiv 2609.00865) literally
and slowly, in float64:

* ``visibility`` -- each generation segment's live view materialised as a
  Python list (§3.2 live view; App. B Def. "trajectory tree"), and from those
  lists the dense visibility mask, 128x128 tile classes, tile lists, pair
  counts and segment ids; plus the lifetime form of the 4D mask (§4.2, the
  M = M^causal (+) M^logical equation) as a second, independent formulation.
* ``attention`` -- per-segment compact causal softmax attention (§4.1
  LogitTree: one forward per branch on that branch's own sequence), forward
  and textbook backward, scattered back to physical rows; optionally with
  rotary positions taken from each row's gap-free logical positions (§4.2).
* ``visibility.logical_positions`` -- the rank of every key in every segment's
  live view (§4.2 row-wise position reassignment).
* ``logprob`` -- LM-head log-softmax, target gather, importance ratio and the
  clipped PPO/GRPO surrogate with its gradient (App. B.4 "Pitfall A, RL view";
  App. F.1 clip range), forward and backward.
* ``nonmonotone`` -- live views when edits also bring spans back (MemexRL's
  offload / retrieve, App. F): ordered view lists, a per-key replay as second
  formulation, rotary positions in view order, compact attention.
* ``sdcc`` -- SDCC (§5): the final compressed walk, diverging rows, the
  teacher-prefix reconstruction, the forward KL(teacher || student) over the
  vocabulary with the student's gradients, and the lambda ramp (App. F.1).

Every function names the passage it follows in its docstring.
"""

from . import visibility, attention, logprob, nonmonotone, sdcc, multilayer  # noqa: F401
