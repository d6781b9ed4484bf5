"""The slot limit: a pool of 1024 slots (one planner thread per slot; the tournament ranks 1024
means) grown through tournament rounds with exact fp32 scores pushed to both sides (Case 2,
fan-out 2 and 4, forks off page boundaries).  The pool state and the shared-prefix segments must
equal the oracle's bit for bit, and decode steps on the default path (grouped + per-beam side by
side) must match the oracle's fp64 attention on sampled beams."""
import dataclasses

import numpy as np
import pytest

from oracle.segments import segments
from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload import gen
from workload.configs import QWEN3_8B_LAYER

pytestmark = pytest.mark.gpu


def test_1024_slots_match_oracle(cuda):
    import torch
    from workload.driver import GpuRun
    wl = dataclasses.replace(QWEN3_8B_LAYER, beams=1024, prompt_len=40, context=400, hidden=256)
    g, o = GpuRun(wl, device_gen=True), OracleRun(wl, literal_kv=False)
    g.seed()
    o.seed()
    g.append(60)
    o.append(60)
    for r in range(4):
        K, f = (768, 4) if r % 2 == 0 else (512, 2)
        s = gen.uniform([11, r], wl.beams)
        g.pool.push_scores(torch.from_numpy(s).to(g.dev))
        o.push_scores(s, None)
        parent = g.prune(K, f, 0)[0].cpu().numpy()
        _, parent_o, _ = o.prune(K, f, 0)
        assert np.array_equal(parent, parent_o)
        g.append(41 + 16 * r)
        o.append(41 + 16 * r)
    st = g.pool.read_state()
    assert_pool_equal(st, o.pool, wl.page_size, means="exact")
    cover, nseg, _ = segments(o.pool, 2)
    act = o.pool.active
    assert act.sum() == 1024 and cover.sum() > 0
    assert np.array_equal(st["seg_cover"][act], cover[act]) and np.array_equal(st["seg_nseg"][act], nseg[act])
    sample = list(range(0, 1024, 41)) + [1023]
    for _ in range(2):
        out = g.decode_step(B.GB_PATH_AUTO).cpu().numpy()
        ref = o.decode_step(slots=sample)
        assert set(b for _, b in ref) == set(sample)
        for (layer, b), r in ref.items():
            assert_close(out[layer, b], r, "bf16", f"1024 slots L={o.pos} slot {b}")
    assert g.pool.status() == 0
