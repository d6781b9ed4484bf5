"""Tournament rounds through the C ABI with scores pushed as exact fp32 inputs, so the GPU and
the oracle rank identical means: ties, NaN, eligibility, warm-up, fan-out, large pools.
Tables, refcounts, free bitmap, parents, pruned flags and lineage must be bit-exact."""
import dataclasses

import numpy as np
import pytest

from oracle.trajectory import OracleRun
from tests.parity import assert_pool_equal
from workload import gen
from workload.configs import QWEN3_8B_LAYER, TINY

pytestmark = pytest.mark.gpu


def _round(g, o, scores32, K, fanout, warmup=0, eligible=None, mask=None):
    import torch
    dev = g.dev
    g.pool.push_scores(torch.from_numpy(scores32).to(dev),
                       None if mask is None else torch.from_numpy(mask.astype(np.uint8)).to(dev))
    o.push_scores(scores32, mask)
    e_dev = None if eligible is None else torch.from_numpy(eligible.astype(np.uint8)).to(dev)
    parent, pruned, lineage = (t.cpu().numpy() for t in g.prune(K, fanout, warmup, e_dev))
    plan, parent_o, pruned_o = o.prune(K, fanout, warmup, eligible)
    assert np.array_equal(parent, parent_o), (parent, parent_o)
    assert np.array_equal(pruned, pruned_o)
    act = o.pool.active
    assert np.array_equal(lineage.view(np.uint32)[act], o.pool.lineage[act])
    assert_pool_equal(g.pool.read_state(), o.pool, g.wl.page_size, means="exact")
    return plan


def _setup(wl, grow=40, device_gen=False):
    from workload.driver import GpuRun
    g, o = GpuRun(wl, device_gen=device_gen), OracleRun(wl, literal_kv=False)
    g.seed()
    o.seed()
    g.append(grow)
    o.append(grow)
    return g, o


def test_ties_nan_and_signed_zero(cuda):
    wl = dataclasses.replace(TINY, context=400)
    g, o = _setup(wl)
    s = np.array([0.5, 0.5, np.nan, 0.25, 0.5, np.nan, 0.0, -0.0], np.float32)
    plan = _round(g, o, s, K=4, fanout=2)
    assert set(plan.pruned) == {2, 5, 6, 7}
    g.append(17)
    o.append(17)
    plan = _round(g, o, np.full(8, 0.3, np.float32), K=3, fanout=2)


@pytest.mark.parametrize("fanout,K", [(2, 4), (3, 5), (4, 6), (2, 0), (2, 8), (4, 20)])
def test_fanout_and_swap_sizes(cuda, fanout, K):
    wl = dataclasses.replace(TINY, context=400)
    g, o = _setup(wl, grow=50)
    for r in range(4):
        s = gen.uniform([r, 77, fanout, K], wl.beams)
        _round(g, o, s, K=K, fanout=fanout)
        g.append(23)
        o.append(23)


def test_eligibility_mask_and_warmup(cuda):
    wl = dataclasses.replace(TINY, context=400)
    g, o = _setup(wl, grow=30)
    s = gen.uniform([5, 1], wl.beams)
    elig = np.array([1, 0, 1, 0, 0, 0, 1, 0], bool)
    _round(g, o, s, K=4, fanout=2, eligible=elig)
    g.append(10)
    o.append(10)
    # children were created 10 tokens ago; warm-up 20 makes only older beams eligible
    _round(g, o, gen.uniform([5, 2], wl.beams), K=4, fanout=2, warmup=20)
    _round(g, o, gen.uniform([5, 3], wl.beams), K=2, fanout=2, mask=np.array([1, 1, 0, 0, 1, 1, 0, 0], bool))


def test_large_pool_random_trees(cuda):
    # 512 slots, 16-token pages, long tables: many rounds with K=384 / fan-out 4 and K=256 / fan-out 2.
    wl = dataclasses.replace(QWEN3_8B_LAYER, beams=512, prompt_len=64, context=2048, hidden=256)
    g, o = _setup(wl, grow=200, device_gen=True)
    for r in range(6):
        K, f = (384, 4) if r % 2 == 0 else (256, 2)
        _round(g, o, gen.uniform([9, r], wl.beams), K=K, fanout=f)
        g.append(37 + 16 * r)
        o.append(37 + 16 * r)
    assert g.pool.status() == 0


@pytest.mark.parametrize("scores", [
    [0.5, 0.5, np.nan, 0.25, 0.5, np.nan, 0.0, -0.0],   # NaN ranks last: the higher NaN slot
    [0.5, 0.1, 0.3, 0.1, 0.9, 0.1, 0.2, 0.7],           # ties on the lowest mean: the higher slot
    [0.0, -0.0, 0.25, 0.0, 0.5, 0.75, -0.0, 1.0],       # +0 and -0 tie
])
def test_last_ranked_is_the_tournaments_last(cuda, scores):
    """gb_pool_last_ranked (the eviction victim) is the last slot of the oracle's tournament order,
    also after a release leaves a slot inactive."""
    import torch
    from oracle import backends
    wl = dataclasses.replace(TINY, context=400)
    g, o = _setup(wl)
    s = np.array(scores, np.float32)
    g.pool.push_scores(torch.from_numpy(s).to(g.dev))
    o.push_scores(s, None)
    out = torch.full((1,), -7, dtype=torch.int32, device=g.dev)
    for released in ([], [int(backends.get().rank_order(o.pool.mean, o.pool.active)[-1])]):
        if released:
            g.pool.release(torch.tensor(released, dtype=torch.int32, device=g.dev))
            o.pool.release(released)
        g.pool.last_ranked(out)
        want = backends.get().rank_order(o.pool.mean, o.pool.active)[-1]
        assert int(out.item()) == want, (scores, released)
    assert g.pool.status() == 0
