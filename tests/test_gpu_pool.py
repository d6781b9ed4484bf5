"""Pool edge cases through the C ABI against the oracle: out of pages, release errors,
Case 1 refills after release, copy-on-write, host-side call-order checks."""
import dataclasses

import numpy as np
import pytest

from oracle.pool import ERR_INVALID, ERR_OOM, ERR_STATE
from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload.configs import TINY

pytestmark = pytest.mark.gpu


def _runs(wl, num_pages=None):
    from workload.driver import GpuRun
    g = GpuRun(wl, num_pages=num_pages)
    o = OracleRun(wl, literal_kv=True, num_pages=num_pages)
    g.seed()
    o.seed()
    return g, o


def test_out_of_pages_step_is_a_no_op_and_reports(cuda):
    import torch
    wl = dataclasses.replace(TINY, beams=4, prompt_len=16, context=64)
    g, o = _runs(wl, num_pages=4)                 # prompt uses 1 page; the next step needs 4
    out = g.decode_step().cpu().numpy()
    assert o.decode_step() is None
    assert g.pool.status() == ERR_OOM == o.pool.status
    assert (out == 0).all()
    g.pos -= 1                                    # the failed step did not advance the pool
    o.pos = g.pos
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size)
    g.pool.clear_status()
    assert g.pool.status() == 0
    g.pool.release(torch.tensor([3], dtype=torch.int32, device=cuda))   # 3 beams left: 3 pages needed, 3 free
    o.pool.release([3])
    out = g.decode_step().cpu().numpy()
    ref = o.decode_step()
    for (layer, b), r in ref.items():
        assert_close(out[layer, b], r, "f32", f"slot {b}")
    assert g.pool.status() == 0
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size)


def test_table_full_is_out_of_pages(cuda):
    from workload.driver import GpuRun
    wl = dataclasses.replace(TINY, beams=2, prompt_len=32, context=32)  # max_pages_per_beam = 2 + 1
    g = GpuRun(wl)
    g.seed()
    g.append(16)
    assert g.pool.status() == 0
    g.append(1)                                   # would need a 4th page
    assert g.pool.status() == ERR_OOM


def test_release_errors_and_case1_refill(cuda):
    import torch
    wl = dataclasses.replace(TINY, context=200)
    g, o = _runs(wl)
    g.append(30)
    o.append(30)
    g.pool.release(torch.tensor([9], dtype=torch.int32, device=cuda))
    assert g.pool.status() == ERR_INVALID
    g.pool.clear_status()
    g.pool.release(torch.tensor([6, 1, 6], dtype=torch.int32, device=cuda))
    o.pool.release([6, 1, 6])
    assert g.pool.status() == ERR_STATE == o.pool.status
    g.pool.clear_status()
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size)
    # Case 1 (Eq. 2): two vacant slots are refilled from the top eligible beams.
    g.probe()
    o.probe()
    parent, pruned, lineage = (t.cpu().numpy() for t in g.prune())
    plan, parent_o, pruned_o = o.prune()
    assert plan.case == 1 and [s for s, _ in plan.children] == [1, 6]
    assert np.array_equal(parent, parent_o) and not pruned.any()
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol")
    out = g.decode_step().cpu().numpy()
    for (layer, b), r in o.decode_step().items():
        assert_close(out[layer, b], r, "f32", f"slot {b}")


def test_layers_must_come_in_order(cuda):
    from workload.driver import GpuRun
    wl = dataclasses.replace(TINY, num_layers=2, context=100)
    g = GpuRun(wl)
    g.seed()
    with pytest.raises(B.GambitError) as e:
        g.pool.decode_attention(1, g.q, g.k_new, g.v_new, 1.0, g.out[1])
    assert e.value.code == B.GB_ERR_STATE
    g.decode_step()
    assert g.pool.status() == 0


def test_multi_layer_steps_match_oracle(cuda):
    wl = dataclasses.replace(TINY, num_layers=3, prompt_len=24, context=90, interval=30)
    g, o = _runs(wl)
    rounds = set(wl.rounds())
    while g.pos < wl.context:
        out = g.decode_step().cpu().numpy()
        for (layer, b), r in o.decode_step().items():
            assert_close(out[layer, b], r, "f32", f"layer {layer} slot {b}")
        if g.pos in rounds:
            g.probe(); o.probe(); g.prune(); o.prune()
            assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol")
    assert g.pool.status() == 0


def test_bf16_grouped_step_out_of_pages_and_all_released(cuda):
    """The bf16 path (grouped + per-beam kernels on two streams): a step that runs out of pages
    changes nothing, reports GB_ERR_OOM and gives zero outputs; after every slot is released a
    step has no work and gives zeros with the status clean."""
    import torch
    from workload.configs import QWEN3_8B_LAYER
    wl = dataclasses.replace(QWEN3_8B_LAYER, beams=32, prompt_len=64, context=80, hidden=256)
    g, o = _runs(wl, num_pages=4 + 32 + 31)       # prompt: 4 shared pages; one page per beam at L = 64
    g.append(15)
    o.append(15)                                  # tokens 64..78 in each beam's new page, 31 pages free
    out = g.decode_step().cpu().numpy()
    assert (np.abs(out) > 0).any() and g.pool.status() == 0   # token 79 still fits the page
    o.decode_step(compute=False)
    assert int(g.pool.read_state()["seg_cover"].sum()) > 0    # the shared prompt goes through the grouped path
    out = g.decode_step().cpu().numpy()           # position 80 needs a new page per beam: 32 > 31 free
    assert o.decode_step() is None
    assert g.pool.status() == ERR_OOM == o.pool.status
    assert (out == 0).all()
    g.pos -= 1
    o.pos = g.pos
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="exact", dtype="bf16")
    g.pool.clear_status()
    g.pool.release(torch.arange(32, dtype=torch.int32, device=cuda))
    out = g.decode_step().cpu().numpy()
    assert (out == 0).all() and g.pool.status() == 0
    st = g.pool.read_state()
    assert not st["active"].any() and (st["refcnt"] == 0).all()
