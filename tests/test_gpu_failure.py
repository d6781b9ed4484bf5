"""Failure detection on the GPU without a fault: a bounded device-side wait that runs out.

gb_pool_wait_selftest enqueues one warp that waits, with the attention launch's merge wait, for
a record count that no kernel raises.  The wait must end by its limit (2 s), record
GB_ERR_TIMEOUT in the pool's status word, and leave the context and the pool usable: after the
status is cleared, the next decode steps match the oracle."""
import time

import pytest

from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close
from workload.configs import QWEN3_8B_LAYER, TINY

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("wl", [TINY, QWEN3_8B_LAYER], ids=["tiny-fp32", "qwen3-8b-layer"])
def test_bounded_wait_runs_out_and_the_pool_stays_usable(cuda, wl):
    import torch

    from workload.driver import GpuRun
    literal = wl is TINY
    g = GpuRun(wl) if literal else GpuRun(wl, device_gen=True, max_context=wl.prompt_len + 4)
    o = OracleRun(wl, literal_kv=literal, max_context=None if literal else wl.prompt_len + 4)
    g.seed()
    o.seed()
    g.decode_step()
    o.decode_step(compute=False)
    assert g.pool.status() == B.GB_OK

    torch.cuda.synchronize()
    t0 = time.perf_counter()
    B.gb_pool_wait_selftest(g.pool.handle)
    status = g.pool.status()              # synchronises the stream
    waited = time.perf_counter() - t0
    assert status == B.GB_ERR_TIMEOUT
    assert 1.5 < waited < 30.0, waited     # the 2 s limit, not a hang

    g.pool.clear_status()
    assert g.pool.status() == B.GB_OK
    for _ in range(2):                     # the pool still decodes, and correctly
        out = g.decode_step().cpu().numpy()
        ref = o.decode_step(compute=True, slots=[0, wl.beams - 1])
        for (layer, b), r in ref.items():
            assert_close(out[layer, b], r, wl.kv_dtype, f"{wl.name} after the timeout, slot {b}")
    assert g.pool.status() == B.GB_OK
