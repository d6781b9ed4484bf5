"""Pins for oracle.tournament (Algorithm 1, Eq. 2 / Eq. 3) and the paper's tree accounting."""
import itertools
import json
import math
from pathlib import Path

import numpy as np
import pytest

from oracle.simulate import simulate
from oracle.tournament import rank_order, tournament
from oracle import backends

NAMES = {'rank_order': 'rank_order', 'tournament': 'tournament'}

@pytest.fixture(autouse=True, params=backends.NAMES)
def oracle_backend(request, monkeypatch):
    """Every pin runs on both oracles: the C++ one and its numpy twin."""
    B = backends.get(request.param)
    monkeypatch.setattr(backends, "DEFAULT", request.param)
    for name, attr in NAMES.items():
        monkeypatch.setitem(globals(), name, getattr(B, attr))
    return B


GOLDEN = Path(__file__).parent / "golden"


def _brute_force_case2(values, K, f):
    """Independent statement: prune the K_eff lowest by value, parents are the highest by value."""
    C = len(values)
    by_value_desc = list(np.argsort(-np.asarray(values), kind="stable"))
    k_eff = min(K, (f - 1) * (C - K))
    pruned = set(by_value_desc[C - k_eff:]) if k_eff else set()
    n_par = math.ceil(k_eff / (f - 1)) if k_eff else 0
    parents = by_value_desc[:n_par]
    return pruned, parents, k_eff


@pytest.mark.parametrize("f", [2, 3, 4])
def test_case2_brute_force_over_all_orders(f):
    C = 6
    base = [0.11, 0.27, 0.38, 0.52, 0.69, 0.93]
    active = np.ones(C, bool)
    for perm in itertools.permutations(range(C)):
        values = np.array([base[i] for i in perm], dtype=np.float32)
        for K in range(C + 1):
            plan = tournament(values, active, active, C, K, f)
            pruned, parents, k_eff = _brute_force_case2(values, K, f)
            assert plan.case == 2
            assert set(plan.pruned) == pruned
            assert plan.pruned == sorted(plan.pruned)
            # children fill the pruned slots ascending; parents in rank order, f-1 children each
            assert [s for s, _ in plan.children] == sorted(pruned)
            got_parents = [p for _, p in plan.children]
            assert got_parents == [parents[k // (f - 1)] for k in range(k_eff)]
            assert not (set(got_parents) & pruned)
            # zero-sum: active count unchanged
            assert C - len(plan.pruned) + len(plan.children) == C


def test_eq3_exactly_for_fanout_two():
    # Eq. 3: prune tau_(N-k+1), branch tau_(k) for k = 1..K.
    values = np.array([0.9, 0.1, 0.5, 0.7, 0.3, 0.8, 0.2, 0.6], dtype=np.float32)
    active = np.ones(8, bool)
    plan = tournament(values, active, active, 8, 3, 2)
    assert plan.order == [0, 5, 3, 7, 2, 4, 6, 1]
    assert plan.pruned == sorted([4, 6, 1])
    assert plan.children == [(1, 0), (4, 5), (6, 3)]


def test_ties_keep_slot_order_and_prune_highest_slots_first():
    values = np.array([0.5] * 6, dtype=np.float32)
    active = np.ones(6, bool)
    plan = tournament(values, active, active, 6, 2, 2)
    assert plan.order == [0, 1, 2, 3, 4, 5]
    assert plan.pruned == [4, 5]
    assert plan.children == [(4, 0), (5, 1)]


def test_nan_ranks_last_and_signed_zeros_tie():
    values = np.array([np.nan, 0.0, -0.0, 0.25, np.nan, -1.0], dtype=np.float32)
    active = np.ones(6, bool)
    assert rank_order(values, active) == [3, 1, 2, 5, 0, 4]


def test_infinities_rank_in_place():
    values = np.array([-np.inf, np.inf, 0.0, np.nan], dtype=np.float32)
    assert rank_order(values, np.ones(4, bool)) == [1, 2, 0, 3]


def test_ineligible_top_traces_are_skipped_as_parents():
    values = np.array([0.9, 0.8, 0.7, 0.6, 0.5, 0.4], dtype=np.float32)
    active = np.ones(6, bool)
    eligible = np.array([False, True, False, True, True, True])
    plan = tournament(values, active, eligible, 6, 2, 2)
    assert plan.pruned == [4, 5]
    assert plan.children == [(4, 1), (5, 3)]


def test_too_few_eligible_parents_prunes_less():
    values = np.array([0.9, 0.8, 0.7, 0.6, 0.5, 0.4], dtype=np.float32)
    active = np.ones(6, bool)
    eligible = np.array([False, False, True, False, False, False])
    plan = tournament(values, active, eligible, 6, 3, 2)
    # one eligible survivor, fan-out 2 -> only one child, so only the last-ranked trace is pruned
    assert plan.pruned == [5]
    assert plan.children == [(5, 2)]
    assert tournament(values, active, np.zeros(6, bool), 6, 3, 2).children == []


def test_fanout_remainder_goes_to_the_last_parent():
    values = np.linspace(1, 0, 8).astype(np.float32)
    active = np.ones(8, bool)
    plan = tournament(values, active, active, 8, 5, 4)  # 5 children, 3 per parent -> 3 + 2
    assert [p for _, p in plan.children] == [0, 0, 0, 1, 1]
    assert plan.pruned == [3, 4, 5, 6, 7]


def test_case1_fills_vacant_slots_from_the_top():
    values = np.array([0.2, 0.9, 0.0, 0.5, 0.0, 0.7], dtype=np.float32)
    active = np.array([True, True, False, True, False, True])
    eligible = active.copy()
    eligible[1] = False
    plan = tournament(values, active, eligible, 6, 3, 2)
    assert plan.case == 1 and plan.pruned == []
    assert plan.children == [(2, 5), (4, 3)]   # Eq. 2: top min(C-N, |B|) eligible, vacant slots ascending
    plan = tournament(values, active, np.array([False, False, False, False, False, True]), 6, 3, 2)
    assert plan.children == [(2, 5)]


def test_paper_runtime_example_accounting():
    g = json.loads((GOLDEN / "runtime_example.json").read_text())
    assert g["roots"] + g["branches"] == g["nodes"]
    # every node ends pruned, completed or still active; the active pool is C (zero-sum)
    assert g["nodes"] - g["pruned"] - g["completed"] == g["capacity_C"]


def test_simulated_main_loop_accounting():
    acc = simulate(C=32, K=4, fanout=2, interval=200, mean_len=6000, seed=3)
    assert acc.nodes == acc.roots + acc.branches
    assert acc.nodes == acc.pruned + acc.completed + acc.active_end
    assert 0 <= acc.active_end <= 32
    assert acc.completed == 32
    assert acc.case2_rounds, "expected at-capacity rounds"
    for pruned, branched, active_after in acc.case2_rounds:
        assert pruned == branched and active_after == 32      # Eq. 3: zero-sum, |T_act| = C
    for vacant, branched in acc.case1_rounds:
        assert branched <= vacant                              # Eq. 2: at most C - N children
