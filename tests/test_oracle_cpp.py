"""The C++ oracle against its numpy twin (``oracle.backends``): two codings of the same
definitions, each pinned on its own by the other oracle tests, must agree - bit for bit on
block tables, reference counts, free pages, lengths, counters, lineage and running means,
and within 1e-12 on fp64 attention - over the tiny workload's whole trajectory (every decode
step, literal copy-on-fork KV) and over a 16-beam sample of the Qwen3-8B layer at full context."""
import dataclasses

import numpy as np
import pytest

from oracle import backends
from oracle.trajectory import OracleRun
from workload.configs import QWEN3_8B_LAYER, TINY


def _same_pool(a, b, what):
    assert [list(t) for t in a.tables] == [list(t) for t in b.tables], f"{what}: tables"
    for name in ("seq_len", "active", "gen", "nsteps", "lineage", "refcnt"):
        assert np.array_equal(np.asarray(getattr(a, name)), np.asarray(getattr(b, name))), f"{what}: {name}"
    assert np.array_equal(np.asarray(a.mean).view(np.uint32), np.asarray(b.mean).view(np.uint32)), f"{what}: mean bits"
    assert np.array_equal(a.free_bits(), b.free_bits()), f"{what}: free pages"
    assert a.history == b.history, f"{what}: writer histories"
    assert a.status == b.status and a.num_free() == b.num_free()


def test_backends_are_distinct_codings():
    c, n = backends.get("cpp"), backends.get("numpy")
    assert c.decode_attention is not n.decode_attention and c.Pool is not n.Pool


@pytest.mark.parametrize("over", [dict(), dict(prompt_len=40, interval=50, fanout=3, K=5)])
def test_tiny_trajectory_every_step(over):
    wl = dataclasses.replace(TINY, **over)
    runs = [OracleRun(wl, literal_kv=True, backend=b) for b in backends.NAMES]
    for r in runs:
        r.seed()
    rounds = set(wl.rounds(include_final=True))
    steps = 0
    while runs[0].pos < wl.context:
        outs = [r.decode_step() for r in runs]
        assert outs[0].keys() == outs[1].keys()
        for key in outs[0]:
            np.testing.assert_allclose(outs[0][key], outs[1][key], rtol=0, atol=1e-12, err_msg=str(key))
        steps += 1
        if runs[0].pos in rounds:
            s = [r.probe() for r in runs]
            for b in s[0]:
                assert abs(s[0][b] - s[1][b]) <= 1e-15
            plans = [r.prune() for r in runs]
            assert plans[0][0].children == plans[1][0].children
            assert np.array_equal(plans[0][1], plans[1][1]) and np.array_equal(plans[0][2], plans[1][2])
        _same_pool(runs[0].pool, runs[1].pool, f"L={runs[0].pos}")
    assert steps == wl.context - wl.prompt_len
    runs[0].pool.check_invariants()


def test_qwen3_layer_sample_at_full_context():
    wl = QWEN3_8B_LAYER
    runs = [OracleRun(wl, literal_kv=False, max_context=wl.context + 1, backend=b) for b in backends.NAMES]
    for r in runs:
        r.build(upto=wl.context, final_round=True)
    _same_pool(runs[0].pool, runs[1].pool, "after the schedule")
    sample = list(range(0, wl.beams, 4))[:16]
    outs = [r.decode_step(compute=True, slots=sample) for r in runs]
    assert len(outs[0]) == 16
    for key in outs[0]:
        np.testing.assert_allclose(outs[0][key], outs[1][key], rtol=0, atol=1e-12, err_msg=str(key))
    _same_pool(runs[0].pool, runs[1].pool, "after one more step")
