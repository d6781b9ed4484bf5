"""Algorithm 1's main loop on the oracle pool, with memory-pressure eviction.

Follows Algorithm 1 (left column) on ``oracle.pool.PoolOracle``:

  while traces run and |F| < C:
      Generate one thought (``interval`` tokens) for every running trace.  When the
      pool cannot hold it, the trace ranked last (lowest running mean; ties: the
      higher slot; NaN last) is evicted (Algorithm 1, the KV-saturation branch):
      its pages are released but it stays in the Tree view as a ghost, so it
      keeps counting against the capacity C (Section 3.2), and the thought is
      retried;
      update each running trace's mean with its thought score (fp32, Alg. 1);
      Tournament: Case 1 while running + ghosts < C, else Case 2 (Eq. 2, Eq. 3);
      move completed traces to F.

A thought is appended all or nothing: if any of its tokens cannot get a page,
the pool is left as it was before the thought.  Scores and completion lengths
come from the caller.  Returns the run's counts and every round's Case 1 /
Case 2 record, and the final pool.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import copy

import numpy as np

from oracle.pool import PoolOracle
from oracle.probe import running_mean_update
from oracle.tournament import rank_order


def tournament_loop(C: int, K: int, fanout: int, interval: int, warmup: int, page_size: int, num_pages: int,
                    max_pages: int, prompt_len: int, initial_targets, score_fn, target_fn,
                    max_rounds: int = 100000) -> dict:
    pool = PoolOracle(num_pages, C, max_pages, page_size)
    pool.seed(C, prompt_len)
    length = np.zeros(C, dtype=np.int64)              # generated tokens (after the prompt)
    target = np.asarray(initial_targets, dtype=np.int64).copy()
    out = {"roots": C, "branches": 0, "pruned": 0, "completed": 0, "ghosts": 0, "case1": [], "case2": []}
    rnd = 0
    while pool.active.any() and out["completed"] < C and rnd < max_rounds:
        rnd += 1
        while True:                                   # Generate, evicting under memory pressure
            before = copy.deepcopy(pool)
            if all(pool.begin_step() for _ in range(interval)):
                break
            pool = before
            victim = rank_order(pool.mean, pool.active)[-1]
            pool.release([victim])
            out["ghosts"] += 1
            pool.capacity = C - out["ghosts"]
            if not pool.active.any():
                out["pool"] = pool
                return out
        run = [int(b) for b in np.flatnonzero(pool.active)]
        length[run] += interval
        for b, x in zip(run, np.asarray(score_fn(run), dtype=np.float32)):
            pool.mean[b], pool.nsteps[b] = running_mean_update(pool.mean[b], int(pool.nsteps[b]), np.float32(x))
        counted = len(run) + out["ghosts"]
        plan, parent_of, pruned = pool.prune_branch(K, fanout, warmup)
        children = sorted(s for s, _ in plan.children)
        for s in children:
            length[s] = length[int(parent_of[s])]
        if children:
            target[children] = np.asarray(target_fn(children, length[children]), dtype=np.int64)
        out["branches"] += len(children)
        out["pruned"] += len(plan.pruned)
        if counted >= C:
            out["case2"].append((len(plan.pruned), len(children), int(pool.active.sum())))
        else:
            out["case1"].append((C - counted, len(children)))
        done = [b for b in np.flatnonzero(pool.active) if length[b] >= target[b]][: C - out["completed"]]
        if done:
            pool.release(done)
            out["completed"] += len(done)
    out["running"] = int(pool.active.sum())
    out["pool"] = pool
    return out
