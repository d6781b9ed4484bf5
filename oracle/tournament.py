"""Ranking and prune/branch routing of the Tournament function.

Follows Algorithm 1 (right column, ``Tournament(T_act, S, C, K)``) and the two
routing cases of Section 3.1:

* rank the active traces by running mean score, descending;
* eligible parents ``B``: traces that have generated at least ``w`` tokens
  since their own creation (Section 3.1, the definition of B);
* Case 1, under capacity (N < C, Eq. 2): branch the top ``min(C - N, |B|)``
  eligible traces, one child each;
* Case 2, at capacity (N = C, Eq. 3): prune the bottom ``K`` and branch the
  top ``K``; pruning and branching are paired so |T_act| stays C.

Readings where the paper is silent:

* ties in the ranking keep ascending slot order (the lower slot ranks
  higher), +0 and -0 compare equal, and a NaN mean ranks after every number;
* fan-out ``f``: every parent gets ``f - 1`` children (the last parent the
  remainder); parents are the first ``ceil(K/(f-1))`` eligible survivors in
  rank order.  ``f = 2`` is exactly Eq. 3;
* parents are never drawn from the pruned set; when the eligible survivors
  cannot supply ``K`` children only ``K_eff = min(K, (f-1)|B_surv|)`` traces
  are pruned (the bottom ``K_eff``), so that the active count stays C;
* child ``k`` (children ordered by parent rank, then child index) takes the
  ``k``-th smallest freed slot (Case 2: the pruned slots; Case 1: the
  inactive slots).

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np


def rank_order(mean: np.ndarray, active: np.ndarray) -> list[int]:
    """Active slots best-first: higher mean first, ties by slot, NaN last."""
    def key(s: int):
        m = float(mean[s])
        if math.isnan(m):
            return (1, 0.0, s)
        return (0, -m, s)
    return sorted((s for s in range(len(mean)) if active[s]), key=key)


@dataclass
class TournamentPlan:
    case: int                      # 0: nothing to do, 1: under capacity, 2: at capacity
    order: list[int]               # active slots best-first
    pruned: list[int] = field(default_factory=list)             # ascending slot ids
    children: list[tuple[int, int]] = field(default_factory=list)  # (child slot, parent slot)


def tournament(mean: np.ndarray, active: np.ndarray, eligible: np.ndarray,
               capacity: int, K: int, fanout: int) -> TournamentPlan:
    """Decide which traces are pruned and which are branched, and where children go."""
    if fanout < 2:
        raise ValueError("fan-out must be at least 2")
    order = rank_order(mean, active)
    N = len(order)
    if N == 0:
        return TournamentPlan(0, order)
    if N < capacity:
        # Case 1 (Eq. 2): fill vacant slots from the top eligible traces.
        B = [s for s in order if eligible[s]]
        m = min(capacity - N, len(B))
        vacant = [s for s in range(capacity) if not active[s]][:m]
        return TournamentPlan(1, order, [], [(vacant[k], B[k]) for k in range(m)])
    # Case 2 (Eq. 3): zero-sum swap, generalised to fan-out f.
    K = max(0, min(int(K), N))
    survivors = order[:N - K]
    B = [s for s in survivors if eligible[s]]
    k_eff = min(K, (fanout - 1) * len(B))
    if k_eff == 0:
        return TournamentPlan(2, order)
    pruned = sorted(order[N - k_eff:])
    children = [(pruned[k], B[k // (fanout - 1)]) for k in range(k_eff)]
    return TournamentPlan(2, order, pruned, children)
