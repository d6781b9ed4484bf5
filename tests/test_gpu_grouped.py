"""Grouped shared-prefix path (tcgen05) against the oracle: beams that share a segment of full
pages are stacked into one query tile per KV head; outputs must match the oracle within the bf16
tolerance and agree with the per-beam path.  Covers segments of one and several 128-row tiles,
several depths, unaligned forks and a ragged per-beam remainder."""
import dataclasses

import numpy as np
import pytest

from oracle.segments import segments
from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload.configs import QWEN3_8B_LAYER

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("beams,group_min,prompt,context,interval,K", [
    (32, 4, 100, 520, 100, 16),     # 32 beams x 4 heads = one 128-row tile for the prompt
    (64, 16, 200, 700, 150, 32),    # 256 rows = two tiles; only the widest segments grouped
    (48, 2, 37, 400, 70, 24),       # small segments, unaligned prompt and forks
])
def test_grouped_matches_oracle(cuda, beams, group_min, prompt, context, interval, K):
    from workload.driver import GpuRun
    wl = dataclasses.replace(QWEN3_8B_LAYER, beams=beams, prompt_len=prompt, context=context, interval=interval,
                             K=K, hidden=256)
    g = GpuRun(wl, group_min_beams=group_min)
    o = OracleRun(wl, literal_kv=False)
    g.build(upto=context - 3)
    o.build(upto=context - 3)
    st = g.pool.read_state()
    assert_pool_equal(st, o.pool, wl.page_size, means="tol", dtype="bf16")
    cover, nseg, _ = segments(o.pool, group_min)
    act = o.pool.active
    assert np.array_equal(st["seg_cover"][act], cover[act]), (st["seg_cover"][act], cover[act])
    assert np.array_equal(st["seg_nseg"][act], nseg[act])
    assert cover.sum() > 0 and nseg.max() >= 1, "the grouped path must cover something here"
    for step in range(3):
        out = g.decode_step(B.GB_PATH_AUTO).cpu().numpy()
        ref = o.decode_step()
        for (layer, b), r in ref.items():
            assert_close(out[layer, b], r, "bf16", f"grouped L={o.pos} slot {b}")
    assert g.pool.status() == 0


def test_grouped_equals_per_beam_path(cuda):
    from workload.driver import GpuRun
    wl = dataclasses.replace(QWEN3_8B_LAYER, beams=64, prompt_len=256, context=900, interval=128, K=32, hidden=256)
    a = GpuRun(wl, group_min_beams=4, device_gen=True)
    b = GpuRun(wl, group_min_beams=4, device_gen=True)
    a.build(upto=wl.context - 2)
    b.build(upto=wl.context - 2)
    for _ in range(2):
        oa = a.decode_step(B.GB_PATH_AUTO).cpu().numpy().copy()
        ob = b.decode_step(B.GB_PATH_PER_BEAM).cpu().numpy()
        err = np.abs(oa - ob)
        assert (err <= 2e-3 + 1e-2 * np.abs(ob)).all(), float(err.max())
    assert a.pool.status() == 0 and b.pool.status() == 0
