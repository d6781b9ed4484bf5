"""bf16 decode attention over every query-group size and page size the library takes
(G = Hq / Hkv in {2, 4, 8}; P in {16, 32, 64}), on the default path (grouped shared
prefixes beside the per-beam kernel) and on the per-beam path, against the oracle: an
unaligned prompt (copy-on-write of the shared tail page), ragged tails, forks by real
tournament rounds.  The per-beam kernel's MMA fragments hold G heads in 8 columns and its
TMA coordinates depend on P and on the layer, so each shape is a distinct case."""
import dataclasses

import pytest

from oracle.trajectory import OracleRun
from paper_2608_08020_gb300 import binding as B
from tests.parity import assert_close, assert_pool_equal
from workload.configs import QWEN3_8B_LAYER

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("Hq,Hkv,P,layers", [(4, 2, 16, 1), (16, 2, 16, 1), (8, 1, 32, 1), (32, 8, 64, 1),
                                             (16, 2, 64, 1), (32, 8, 16, 3)])
@pytest.mark.parametrize("flags", ["auto", "per_beam"])
def test_bf16_shapes_match_oracle(cuda, Hq, Hkv, P, layers, flags):
    from workload.driver import GpuRun
    wl = dataclasses.replace(QWEN3_8B_LAYER, num_layers=layers, num_q_heads=Hq, num_kv_heads=Hkv, page_size=P, beams=8,
                             prompt_len=72, context=72 + 3 * P + 40, interval=P + 24, K=4, hidden=256)
    path = B.GB_PATH_AUTO if flags == "auto" else B.GB_PATH_PER_BEAM
    g, o = GpuRun(wl), OracleRun(wl, literal_kv=True)
    g.seed()
    o.seed()
    rounds = set(wl.rounds(include_final=True))
    step = 0
    while g.pos < wl.context:
        want = (step % 5 == 0) or (g.pos + 1 == wl.context) or (g.pos + 1 in rounds)
        out = g.decode_step(path).cpu().numpy()
        ref = o.decode_step(compute=want)
        for (layer, b), r in ref.items():
            assert_close(out[layer, b], r, "bf16", f"G={Hq // Hkv} P={P} {flags}: attention L={o.pos} slot {b}")
        if g.pos in rounds:
            g.probe()
            o.probe()
            g.prune()
            o.prune()
            assert_pool_equal(g.pool.read_state(), o.pool, wl.page_size, means="tol", dtype="bf16")
        step += 1
    assert g.pool.status() == 0
