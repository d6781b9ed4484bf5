"""Parity at the benchmark's full sizes, in the configuration bench.py times.

The Qwen3-8B layer (64 beams, 4096 tokens), parallel-sampling (512 beams, 16384 tokens,
fan-out 4), long-context (256 beams, 32768 tokens, 32-token pages) and memory-capped
(36 layers, 198 beams, 8192 tokens in a 120 GB pool of 50,862 pages) trees, and the
unshared workload (64 independent traces of 16384 tokens), are built on the GPU exactly as
bench.py builds them (device-generated inputs, the same pool sizing, the default path and
grouping threshold), through the method's schedule up to and including the tournament round
at the full context.  The oracle replays the same schedule (tournaments from its own fp64
probe scores and fp32 running means) and rebuilds each sampled beam's K/V from its writer
history, so every expected value comes from the oracle and the seeded generator.  Checked:
the whole pool state bit-exact (tables, refcounts, free bitmap, lineage, counters; means
within the bf16 tolerance), then one decode step: sampled beams (and, for 36 layers, the
first, a middle and the last layer) element by element against the oracle's fp64 attention
over the full context, every output finite.
"""
import numpy as np
import pytest

from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload.configs import BY_INDEX

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("config,path", [(2, "auto"), (2, "per_beam"), (3, "auto"), (4, "auto"), (5, "auto"),
                                         (6, "auto"), (6, "per_beam")])
def test_full_size_sampled_beams_match_oracle(cuda, config, path):
    _check_full_size(BY_INDEX[config - 1], path)


# Query heads per KV head G = 2 and 8 on the 64-beam tree (the attention launch's two roles side
# by side on their shares of the SMs) and on the 512-beam tree (the per-beam CTAs following the
# grouped ones: 2-4 GB of attention reads per step).
@pytest.mark.parametrize("config,hq,hkv", [(2, 16, 8), (2, 32, 4), (3, 16, 8), (3, 32, 4)])
def test_full_size_group_sizes_match_oracle(cuda, config, hq, hkv):
    import dataclasses

    base = BY_INDEX[config - 1]
    _check_full_size(dataclasses.replace(base, name=f"{base.name}-G{hq // hkv}", num_q_heads=hq, num_kv_heads=hkv),
                     "auto")


# Page sizes 32 and 64 on the 512-beam tree (the per-beam CTAs following the grouped ones): the
# grouped role's page boxes (4 and 2 pages per 128-token tile) and the per-beam role's chunks
# inside larger pages.
@pytest.mark.parametrize("P", [32, 64])
def test_full_size_page_sizes_match_oracle(cuda, P):
    import dataclasses

    base = BY_INDEX[3 - 1]
    _check_full_size(dataclasses.replace(base, name=f"{base.name}-P{P}", page_size=P), "auto")


def _check_full_size(wl, path):
    import torch

    from workload.driver import GpuRun
    max_context = wl.context + 1                      # bench.py's pool sizing (every phase ends at the context)
    g = GpuRun(wl, device_gen=True, max_context=max_context)
    o = OracleRun(wl, literal_kv=False, max_context=max_context)
    assert g.pool.num_pages == o.pool.num_pages == wl.pool_pages(max_context)
    g.build(upto=wl.context, final_round=True)
    o.build(upto=wl.context, final_round=True)
    assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol", dtype="bf16")

    flags = B.GB_PATH_AUTO if path == "auto" else B.GB_PATH_PER_BEAM
    out = g.decode_step(flags).cpu().numpy()
    C = wl.beams
    sample = sorted({0, 1, C // 3, C // 2 + 1, C - 1})
    layers = sorted({0, wl.num_layers // 2 - 1, wl.num_layers - 1}) if wl.num_layers > 1 else None
    ref = o.decode_step(compute=True, slots=sample, layers=layers)
    assert len(ref) == len(sample) * (len(layers) if layers else wl.num_layers)
    for (layer, b), r in ref.items():
        assert_close(out[layer, b], r, "bf16", f"{wl.name} L={o.pos} layer {layer} slot {b}")
    assert np.isfinite(out).all()
    assert g.pool.status() == 0
    del g
    torch.cuda.empty_cache()
