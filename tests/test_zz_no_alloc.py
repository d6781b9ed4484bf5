"""gb_paged_decode_noalloc: decode attention for callers that cannot allocate device memory.

Its working memory is the library's fixed device array, so it is checked against the pool's own
gb_decode_attention on the same pages, tables and queries, on two calls in a row (the second call
finds the first call's leftovers in the shared array).  The file name makes pytest collect it last.
"""
import dataclasses

import pytest

from tests.parity import assert_close
from workload.configs import QWEN3_8B_LAYER, TINY

pytestmark = pytest.mark.gpu


def _args(B, g, tables, seq_len, out):
    wl = g.wl
    return B.GbPagedDecodeArgs(g.pool.kv.data_ptr(), tables.data_ptr(), seq_len.data_ptr(), g.q.data_ptr(),
                               out.data_ptr(), wl.beams, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                               wl.page_size, B.GB_BF16 if wl.kv_dtype == "bf16" else B.GB_F32,
                               g.pool.max_pages, g.pool.num_pages, wl.attn_scale)


@pytest.mark.parametrize("base,over", [
    (TINY, dict(prompt_len=40, context=200, interval=50)),
    (QWEN3_8B_LAYER, dict(beams=24, prompt_len=100, context=420, interval=120, K=10, hidden=256)),
])
def test_noalloc_matches_pool_decode_on_two_calls(cuda, base, over):
    import torch

    from paper_2608_08020_gb300 import binding as B
    from workload.driver import GpuRun
    wl = dataclasses.replace(base, **over)
    g = GpuRun(wl)
    g.build(upto=wl.context - 2)                       # a tree with forks, unaligned ends
    released = torch.tensor([3], dtype=torch.int32, device=cuda)
    g.pool.release(released)                           # one empty row: its output must be zero
    for call in range(2):
        ref = g.decode_step()[0].clone()               # the pool's entry point (appends, then attends)
        st = g.pool.read_state()
        tables = torch.from_numpy(st["tables"]).to(cuda)
        seq_len = torch.from_numpy(st["seq_len"]).to(cuda)
        out = torch.full_like(ref, float("nan"))
        B.gb_paged_decode_noalloc(_args(B, g, tables, seq_len, out))
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert_close(got, ref.cpu().numpy(), wl.kv_dtype, f"call {call}")
        assert (got[3] == 0).all()
    assert g.pool.status() == 0


def test_noalloc_rejects_what_does_not_fit(cuda):
    import torch

    from paper_2608_08020_gb300 import binding as B
    buf = torch.zeros(1 << 16, dtype=torch.uint8, device=cuda)
    p = buf.data_ptr()
    # 1024 rows x 8 KV heads with G = 8 needs more than the fixed 32 MiB.
    big = B.GbPagedDecodeArgs(p, p, p, p, p, 1024, 64, 8, 128, 16, B.GB_BF16, 4, 16, 0.1)
    with pytest.raises(B.GambitError) as e:
        B.gb_paged_decode_noalloc(big)
    assert e.value.code == B.GB_ERR_TOO_LARGE
    bad = B.GbPagedDecodeArgs(p, p, p, p, p, 2048, 32, 8, 128, 16, B.GB_BF16, 4, 16, 0.1)
    with pytest.raises(B.GambitError) as e:
        B.gb_paged_decode_noalloc(bad)
    assert e.value.code == B.GB_ERR_INVALID
