"""bf16 Qwen3-8B-shaped decode attention (32/8 heads, D=128) against the oracle on small trees:
unaligned prompt (copy-on-write of the shared tail page), ragged tails, several chunks per
(beam, head) split over several warps, forks by real tournament rounds."""
import dataclasses

import numpy as np
import pytest

from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload.configs import QWEN3_8B_LAYER, TINY

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("prompt,context,interval,beams,K", [
    (40, 300, 100, 8, 4),     # partial shared prompt page, ragged end
    (512, 700, 96, 16, 8),    # page-aligned prompt, forks off page boundaries
])
def test_bf16_decode_steps_match_oracle(cuda, prompt, context, interval, beams, K):
    from workload.driver import GpuRun
    wl = dataclasses.replace(QWEN3_8B_LAYER, beams=beams, prompt_len=prompt, context=context, interval=interval,
                             K=K, hidden=256)
    g, o = GpuRun(wl), OracleRun(wl, literal_kv=True)
    g.seed()
    o.seed()
    rounds = set(wl.rounds(include_final=True))
    check_every = 7
    step = 0
    while g.pos < wl.context:
        want = (step % check_every == 0) or (g.pos + 1 == wl.context) or (g.pos + 1 in rounds)
        out = g.decode_step().cpu().numpy()
        ref = o.decode_step(compute=want)
        for (layer, b), r in ref.items():
            assert_close(out[layer, b], r, "bf16", f"attention L={o.pos} slot {b}")
        if g.pos in rounds:
            g.probe()
            o.probe()
            g.prune()
            o.prune()
            assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol", dtype="bf16")
        step += 1
    assert g.pool.status() == 0


def test_per_beam_flag_matches_auto(cuda):
    from workload.driver import GpuRun
    wl = dataclasses.replace(TINY, context=120)
    a, b = GpuRun(wl), GpuRun(wl)
    a.seed()
    b.seed()
    while a.pos < wl.context:
        oa = a.decode_step(B.GB_PATH_AUTO).cpu().numpy().copy()
        ob = b.decode_step(B.GB_PATH_PER_BEAM).cpu().numpy()
        np.testing.assert_array_equal(oa, ob)


def test_inactive_rows_are_zero(cuda):
    import torch
    from workload.driver import GpuRun
    wl = dataclasses.replace(TINY, context=90)
    g = GpuRun(wl)
    g.seed()
    g.append(10)
    g.pool.release(torch.tensor([2, 5], dtype=torch.int32, device=cuda))
    out = g.decode_step().cpu().numpy()
    assert (out[0, 2] == 0).all() and (out[0, 5] == 0).all()
    assert np.abs(out[0, 0]).max() > 0
    assert g.pool.status() == 0
