"""Host-side Tree view (Section 3.2): node accounting from tournament outputs, on CPU."""
import numpy as np
import pytest

from paper_2608_08020_gb300.tree import COMPLETED, GHOST, TreeView


def test_rounds_completions_and_ghosts():
    t = TreeView(capacity=4)
    t.add_roots(range(4), [0, 1, 2, 3])
    L = np.array([10, 10, 10, 10])
    # Case 2: slots 2 and 3 pruned; their slots take children of 0 and 1.
    ch = t.apply_round(1, parent_out=[0, 1, 0, 1], pruned_out=[0, 0, 1, 1], lineage_out=[0, 1, 4, 5], lengths=L)
    assert ch == [2, 3] and t.roots == 4 and t.branches == 2 and t.case2_rounds == [(2, 2, 4)]
    # Slot 1 completes, slot 3 is evicted as a ghost: 2 running + 1 ghost count against C = 4.
    t.finish([1], L)
    t.finish([3], L, GHOST)
    assert t.running() == 2 and t.counted() == 3 and t.count(COMPLETED) == 1 and t.count(GHOST) == 1
    # Case 1: one vacancy, one child of slot 0 into slot 1.
    ch = t.apply_round(2, parent_out=[0, 0, 2, -1], pruned_out=[0, 0, 0, 0], lineage_out=[0, 6, 4, 5], lengths=L)
    assert ch == [1] and t.case1_rounds == [(1, 1)]
    t.check()
    assert len(t.nodes) == 7 and t.nodes[6].parent == t.nodes[0].id


def test_zero_sum_violation_is_caught():
    t = TreeView(capacity=2)
    t.add_roots(range(2), [0, 1])
    t.case2_rounds.append((1, 0, 1))
    with pytest.raises(AssertionError):
        t.check()
