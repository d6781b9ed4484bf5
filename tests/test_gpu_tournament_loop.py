"""Algorithm 1's main loop on the GPU pool against the oracle's simulation of it.

``TournamentLoop`` runs Generate / Tournament (Case 1 and Case 2, warm-up) / completion on
the device pool, fed with the same seeded synthetic scores and completion lengths as
``oracle.simulate``; the two must agree on every count (roots, branches, pruned,
completed, traces left) and on every round's Case 1 / Case 2 record, and the Tree view's
node accounting must hold (zero-sum Case-2 rounds; nodes = roots + branches).
"""
import numpy as np
import pytest

from oracle.simulate import simulate

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("C,K,fanout,warmup", [
    (64, 16, 2, 0),
    (64, 24, 4, 400),
    (256, 16, 2, 0),
])
def test_gpu_loop_matches_simulation(cuda, C, K, fanout, warmup):
    from paper_2608_08020_gb300.pool import BeamPool
    from paper_2608_08020_gb300.tree import COMPLETED, PRUNED, TournamentLoop
    seed, interval, mean_len = 7, 200, 3000
    ref = simulate(C, K, fanout=fanout, interval=interval, warmup=warmup, seed=seed, mean_len=mean_len)

    rng = np.random.default_rng(seed)                 # the simulation's draws, in its order
    initial = rng.integers(mean_len // 2, 3 * mean_len // 2, size=C)
    pool = BeamPool(num_layers=1, num_q_heads=2, num_kv_heads=1, head_dim=64, page_size=64, kv_dtype="f32",
                    num_pages=C * 1024, max_beams=C, max_pages_per_beam=2048)
    loop = TournamentLoop(pool, C, K, fanout=fanout, interval=interval, warmup=warmup, prompt_len=64)
    loop.seed(initial)
    tree = loop.run(lambda slots: np.array([np.float32(rng.random()) for _ in slots], dtype=np.float32),
                    lambda children, plen: np.array([int(p) + int(rng.integers(mean_len // 4, mean_len)) for p in plen]))
    tree.check()
    assert loop.evictions == 0
    assert tree.roots == ref.roots == C
    assert tree.branches == ref.branches
    assert tree.count(PRUNED) == ref.pruned
    assert tree.count(COMPLETED) == ref.completed
    assert tree.running() == ref.active_end
    assert tree.case2_rounds == ref.case2_rounds
    assert tree.case1_rounds == ref.case1_rounds
    assert pool.status() == 0


@pytest.mark.parametrize("C,K,num_pages", [(32, 8, 600), (64, 16, 1400)])
def test_gpu_loop_with_ghosts_matches_oracle_loop(cuda, C, K, num_pages):
    """Memory pressure: both evict the same traces as ghosts, make the same tournaments and
    end with the same pool, bit for bit (tables, refcounts, free pages, means, lineage)."""
    from oracle.loop import tournament_loop
    from paper_2608_08020_gb300.pool import BeamPool
    from paper_2608_08020_gb300.tree import COMPLETED, GHOST, PRUNED, TournamentLoop
    from tests.parity import assert_pool_equal
    seed, interval, mean_len, P = 5, 200, 3000, 64

    def drivers():
        rng = np.random.default_rng(seed)
        init = rng.integers(mean_len // 2, 3 * mean_len // 2, size=C)
        return (init, lambda run: np.array([np.float32(rng.random()) for _ in run], dtype=np.float32),
                lambda ch, plen: np.array([int(p) + int(rng.integers(mean_len // 4, mean_len)) for p in plen]))

    init, score_fn, target_fn = drivers()
    ref = tournament_loop(C, K, 2, interval, 0, P, num_pages, 2048, 64, init, score_fn, target_fn)
    assert ref["ghosts"] > 0

    init, score_fn, target_fn = drivers()
    pool = BeamPool(num_layers=1, num_q_heads=2, num_kv_heads=1, head_dim=64, page_size=P, kv_dtype="f32",
                    num_pages=num_pages, max_beams=C, max_pages_per_beam=2048)
    loop = TournamentLoop(pool, C, K, fanout=2, interval=interval, warmup=0, prompt_len=64)
    loop.seed(init)
    tree = loop.run(score_fn, target_fn)
    tree.check()
    assert loop.evictions == tree.count(GHOST) == ref["ghosts"]
    assert tree.branches == ref["branches"] and tree.count(PRUNED) == ref["pruned"]
    assert tree.count(COMPLETED) == ref["completed"] and tree.running() == ref["running"]
    assert tree.case1_rounds == ref["case1"] and tree.case2_rounds == ref["case2"]
    assert_pool_equal(pool.read_state(), ref["pool"], P, means="exact")
