"""Pins for oracle.loop (Algorithm 1's loop on the oracle pool, with ghost eviction)."""
import numpy as np
import pytest

from oracle.loop import tournament_loop
from oracle.simulate import simulate


def _drive(C, K, fanout, warmup, num_pages, seed=5, interval=200, mean_len=3000, P=64):
    rng = np.random.default_rng(seed)
    init = rng.integers(mean_len // 2, 3 * mean_len // 2, size=C)
    return tournament_loop(C, K, fanout, interval, warmup, P, num_pages, 2048, 64, init,
                           lambda run: np.array([np.float32(rng.random()) for _ in run], dtype=np.float32),
                           lambda ch, plen: np.array([int(p) + int(rng.integers(mean_len // 4, mean_len))
                                                      for p in plen]))


@pytest.mark.parametrize("C,K,fanout,warmup", [(32, 8, 2, 0), (32, 12, 4, 400)])
def test_ample_memory_reproduces_the_simulation(C, K, fanout, warmup):
    """Two codings of Algorithm 1 (arrays in oracle.simulate, the page pool here) agree."""
    out = _drive(C, K, fanout, warmup, num_pages=C * 512)
    ref = simulate(C, K, fanout=fanout, interval=200, warmup=warmup, seed=5, mean_len=3000)
    assert out["ghosts"] == 0
    assert (out["branches"], out["pruned"], out["completed"], out["running"]) == \
        (ref.branches, ref.pruned, ref.completed, ref.active_end)
    assert out["case1"] == ref.case1_rounds and out["case2"] == ref.case2_rounds


def test_memory_pressure_makes_ghosts_and_keeps_the_accounting():
    out = _drive(32, 8, 2, 0, num_pages=600)
    assert out["ghosts"] > 0
    nodes = out["roots"] + out["branches"]
    assert nodes == out["running"] + out["pruned"] + out["completed"] + out["ghosts"]
    for pr, br, _ in out["case2"]:
        assert pr == br                       # zero-sum
    pool = out["pool"]
    pool.check_invariants()
    assert pool.capacity == 32 - out["ghosts"]
    assert int(pool.active.sum()) + out["ghosts"] <= 32
