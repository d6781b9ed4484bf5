"""Tiny fp32 workload (8 beams, 1 layer, 4/2 heads, D=64, P=16): every decode step, probe and
tournament round through the C ABI against the oracle (attention and scores within 1e-5;
tables, refcounts, free bitmap, parents, pruned flags and lineage bit-exact)."""
import numpy as np
import pytest

from oracle.trajectory import OracleRun
from tests.parity import assert_close, assert_pool_equal
from workload.configs import TINY

pytestmark = pytest.mark.gpu


def test_tiny_trajectory_matches_oracle(cuda):
    from workload.driver import GpuRun
    wl = TINY
    g, o = GpuRun(wl), OracleRun(wl, literal_kv=True)
    g.seed()
    o.seed()
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size)
    rounds = set(wl.rounds(include_final=True))
    assert rounds == {160, 256}
    worst = 0.0
    while g.pos < wl.context:
        out = g.decode_step().cpu().numpy()
        ref = o.decode_step()
        for (layer, b), r in ref.items():
            worst = max(worst, assert_close(out[layer, b], r, "f32", f"attention L={o.pos} slot {b}")[0])
        if g.pos in rounds:
            s_gpu = g.probe().cpu().numpy()
            s_ref = o.probe()
            for b, x in s_ref.items():
                assert_close(s_gpu[b], x, "f32", f"probe slot {b}")
            parent, pruned, lineage = (t.cpu().numpy() for t in g.prune())
            plan, parent_o, pruned_o = o.prune()
            assert np.array_equal(parent, parent_o), (parent, parent_o)
            assert np.array_equal(pruned, pruned_o)
            assert np.array_equal(lineage.view(np.uint32), o.pool.lineage)
            assert len(plan.children) == wl.K
            assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol", dtype="f32")
    assert g.pool.status() == 0
    assert worst < 1e-5
