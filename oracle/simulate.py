"""Algorithm 1's main loop with trace completion, for tournament accounting.

Runs the loop of Algorithm 1 (left column) over slot-indexed traces with
seeded synthetic scores and completion lengths:

  while traces are running and |F| < C:
      Generate (one thought of `interval` tokens for every active trace, then
      the running-mean update with the thought's score);
      Tournament (Case 1 when N < C, Case 2 when N = C);
      move completed traces to F.

It counts roots, branches (children created), pruned traces and completed
traces, so that the node accounting of the paper's runtime example
(Appendix, "Runtime Example": 256 roots + 1,339 branches = 1,595 nodes) and
the zero-sum property of Case 2 (Section 3.1, after Eq. 3) can be checked.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from oracle.probe import running_mean_update
from oracle.tournament import tournament


@dataclass
class Accounting:
    roots: int = 0
    branches: int = 0
    pruned: int = 0
    completed: int = 0
    active_end: int = 0
    case2_rounds: list = field(default_factory=list)   # (pruned, branched, active after)
    case1_rounds: list = field(default_factory=list)   # (vacant before, branched)

    @property
    def nodes(self) -> int:
        return self.roots + self.branches


def simulate(C: int, K: int, fanout: int = 2, interval: int = 200, warmup: int = 0, seed: int = 0,
             mean_len: int = 20000, max_iters: int = 10000) -> Accounting:
    rng = np.random.default_rng(seed)
    active = np.zeros(C, dtype=bool)
    mean = np.zeros(C, dtype=np.float32)
    nsteps = np.zeros(C, dtype=np.int64)
    gen = np.zeros(C, dtype=np.int64)        # tokens since creation
    length = np.zeros(C, dtype=np.int64)     # tokens in the trace (prefix included)
    target = np.zeros(C, dtype=np.int64)     # completion length
    acc = Accounting(roots=C)
    active[:] = True
    target[:] = rng.integers(mean_len // 2, 3 * mean_len // 2, size=C)
    it = 0
    while active.any() and acc.completed < C and it < max_iters:
        it += 1
        # Generate one thought and score it.
        for b in np.flatnonzero(active):
            length[b] += interval
            gen[b] += interval
            x = np.float32(rng.random())
            mean[b], nsteps[b] = running_mean_update(mean[b], int(nsteps[b]), x)
        # Tournament.
        eligible = active & (gen >= warmup)
        plan = tournament(mean, active, eligible, C, K, fanout)
        if plan.case == 2:
            acc.pruned += len(plan.pruned)
            for s in plan.pruned:
                active[s] = False
        elif plan.case == 1:
            acc.case1_rounds.append((C - int(active.sum()), len(plan.children)))
        for s, p in plan.children:
            active[s] = True
            mean[s], nsteps[s] = mean[p], nsteps[p]
            length[s] = length[p]
            gen[s] = 0
            target[s] = length[p] + rng.integers(mean_len // 4, mean_len)
        acc.branches += len(plan.children)
        if plan.case == 2:
            acc.case2_rounds.append((len(plan.pruned), len(plan.children), int(active.sum())))
        # Move completed traces to F.
        for b in np.flatnonzero(active & (length >= target)):
            active[b] = False
            acc.completed += 1
            if acc.completed >= C:
                break
    acc.active_end = int(active.sum())
    return acc
