"""Parity at the benchmark's full sizes, in the configuration bench.py times.

The Qwen3-8B layer (64 beams, 4096 tokens), parallel-sampling (512 beams, 16384 tokens,
fan-out 4) and long-context (256 beams, 32768 tokens, 32-token pages) trees are built on
the GPU exactly as bench.py builds them (device-generated inputs, the same pool sizing,
the default path and grouping threshold), through the method's schedule up to and
including the tournament round at the full context.  The oracle replays the same
schedule (tournaments from its own fp64 probe scores and fp32 running means) and
rebuilds each sampled beam's K/V from its writer history, so every expected value comes
from the oracle and the seeded generator.  Checked: the whole pool state bit-exact
(tables, refcounts, free bitmap, lineage, counters; means within the bf16 tolerance),
then one decode step: sampled beams element by element against the oracle's fp64
attention over the full context, every output finite.
"""
import numpy as np
import pytest

from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload.configs import BY_INDEX

pytestmark = pytest.mark.gpu

WARMUP = 8  # bench.py's default warm-up steps


@pytest.mark.parametrize("config,path", [(2, "auto"), (2, "per_beam"), (3, "auto"), (4, "auto")])
def test_full_size_sampled_beams_match_oracle(cuda, config, path):
    from workload.driver import GpuRun
    wl = BY_INDEX[config - 1]
    K = wl.interval                                   # bench.py's default timed steps
    max_context = wl.context + WARMUP + 2 * K + 1     # bench.py's pool sizing (timed + end-to-end steps)
    g = GpuRun(wl, device_gen=True, max_context=max_context)
    o = OracleRun(wl, literal_kv=False, max_context=max_context)
    g.build(upto=wl.context, final_round=True)
    o.build(upto=wl.context, final_round=True)
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol", dtype="bf16")

    flags = B.GB_PATH_AUTO if path == "auto" else B.GB_PATH_PER_BEAM
    out = g.decode_step(flags).cpu().numpy()
    C = wl.beams
    sample = sorted({0, 1, C // 3, C // 2 + 1, C - 1})
    ref = o.decode_step(compute=True, slots=sample)
    assert len(ref) == len(sample) * wl.num_layers
    for (layer, b), r in ref.items():
        assert_close(out[layer, b], r, "bf16", f"{wl.name} L={o.pos} slot {b}")
    assert np.isfinite(out).all()
    assert g.pool.status() == 0
