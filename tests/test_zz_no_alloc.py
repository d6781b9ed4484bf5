"""gb_paged_decode_noalloc: decode attention for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc where they decode: a serving process whose allocator took
the GPU's memory when it started, or code running inside a framework that owns the device
memory.  They own their pages, tables, lengths, queries and outputs and pass only those; the
call's working memory is the library's fixed device array.

Each case builds caller-owned pages and block tables directly (no pool): rows that share pages
as a fork would, a row that fills its whole table, ragged tails, a released (zero-length) row.
Every row is checked against the oracle's fp64 attention over that row's K/V, gathered on the
host from the same pages, on two calls in a row (the second call finds the first call's
leftovers in the shared array).  The file name makes pytest collect it last.
"""
import numpy as np
import pytest

from oracle.attention import decode_attention
from tests.parity import assert_close
from workload import gen

pytestmark = pytest.mark.gpu


def _case(dtype, G, P, seed, Hkv=2, beams=7, max_pages=6, num_pages=48):
    """Pages [num_pages][K|V][Hkv][P][D], tables [beams][max_pages], lengths, queries (host)."""
    D = 128 if dtype == "bf16" else 64
    rng = np.random.default_rng(seed)
    kv = gen.round_to_dtype(rng.standard_normal((num_pages, 2, Hkv, P, D)).astype(np.float32), dtype)
    perm = rng.permutation(num_pages)
    tables = perm[:beams * max_pages].reshape(beams, max_pages).astype(np.int32)
    tables[1, :3] = tables[0, :3]            # row 1 shares row 0's first three pages (a fork)
    tables[2, :2] = tables[0, :2]
    full = max_pages * P
    seq_len = np.array([full, 3 * P + 5, 0, 1, 2 * P, P - 1, 2 * P + 7], dtype=np.int32)[:beams]
    q = gen.round_to_dtype(rng.standard_normal((beams, G * Hkv, D)).astype(np.float32), dtype)
    return dict(kv=kv, tables=tables, seq_len=seq_len, q=q, D=D, Hkv=Hkv, G=G, P=P, dtype=dtype,
                scale=1.0 / np.sqrt(D), max_pages=max_pages, num_pages=num_pages)


def _row_kv(c, b):
    """The row's full K and V [L][Hkv][D], gathered from its pages by the table (host, oracle side)."""
    L = int(c["seq_len"][b])
    pages = c["tables"][b][np.arange(L) // c["P"]]
    rows = np.arange(L) % c["P"]
    return c["kv"][pages, 0, :, rows, :], c["kv"][pages, 1, :, rows, :]


def _device(c, cuda):
    import torch
    tdt = torch.bfloat16 if c["dtype"] == "bf16" else torch.float32
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(cuda).to(dt)
    return dict(kv=t(c["kv"], tdt), tables=t(c["tables"], torch.int32), seq_len=t(c["seq_len"], torch.int32),
                q=t(c["q"], tdt), out=torch.full(c["q"].shape, float("nan"), dtype=torch.float32, device=cuda))


def _call(B, c, d):
    args = B.GbPagedDecodeArgs(d["kv"].data_ptr(), d["tables"].data_ptr(), d["seq_len"].data_ptr(),
                               d["q"].data_ptr(), d["out"].data_ptr(), len(c["seq_len"]), c["G"] * c["Hkv"],
                               c["Hkv"], c["D"], c["P"], B.GB_BF16 if c["dtype"] == "bf16" else B.GB_F32,
                               c["max_pages"], c["num_pages"], float(c["scale"]))
    B.gb_paged_decode_noalloc(args)
    return B.gb_paged_decode_noalloc_status()


def _check_rows(c, got, what):
    for b in range(len(c["seq_len"])):
        if c["seq_len"][b] <= 0:
            assert (got[b] == 0).all(), f"{what}: row {b} of length {c['seq_len'][b]} must be zero"
            continue
        K, V = _row_kv(c, b)
        assert_close(got[b], decode_attention(c["q"][b], K, V, c["scale"]), c["dtype"], f"{what} row {b}")


SHAPES = [("f32", G, 16) for G in (2, 4, 8)] + [("bf16", G, P) for G in (2, 4, 8) for P in (16, 32, 64)]


@pytest.mark.parametrize("dtype,G,P", SHAPES)
def test_noalloc_matches_oracle_on_caller_tables_two_calls(cuda, dtype, G, P):
    from paper_2608_08020_gb300 import binding as B
    for call in range(2):
        c = _case(dtype, G, P, seed=100 * G + P + call)
        if call == 1:
            c["seq_len"][[1, 4]] = [c["max_pages"] * P - 3, P + 2]   # other lengths than the first call
        d = _device(c, cuda)
        assert _call(B, c, d) == B.GB_OK
        _check_rows(c, d["out"].cpu().numpy(), f"{dtype} G={G} P={P} call {call}")


@pytest.mark.parametrize("dtype,G,P", [("f32", 4, 16), ("bf16", 4, 16), ("bf16", 8, 64)])
def test_noalloc_is_invariant_to_physical_page_placement(cuda, dtype, G, P):
    """The same logical K/V stored in other physical pages (the pool permuted, the tables
    renumbered to follow) gives bit-identical outputs: only the table decides which page holds
    which tokens."""
    from paper_2608_08020_gb300 import binding as B
    c = _case(dtype, G, P, seed=7 * G + P)
    d = _device(c, cuda)
    assert _call(B, c, d) == B.GB_OK
    first = d["out"].cpu().numpy()
    perm = np.random.default_rng(11).permutation(c["num_pages"])   # new page of old page i: perm[i]
    c2 = dict(c)
    kv2 = np.empty_like(c["kv"])
    kv2[perm] = c["kv"]
    c2["kv"] = kv2
    c2["tables"] = perm[c["tables"]].astype(np.int32)
    d2 = _device(c2, cuda)
    assert _call(B, c2, d2) == B.GB_OK
    second = d2["out"].cpu().numpy()
    assert np.array_equal(first, second), np.abs(first - second).max()


def test_noalloc_row_longer_than_its_table_is_refused_and_reported(cuda):
    from paper_2608_08020_gb300 import binding as B
    c = _case("bf16", 4, 16, seed=7)
    c["seq_len"][3] = c["max_pages"] * 16 + 1                       # one token more than the table holds
    d = _device(c, cuda)
    assert _call(B, c, d) == B.GB_ERR_INVALID
    got = d["out"].cpu().numpy()
    assert (got[3] == 0).all()
    c["seq_len"][3] = 0                                              # every other row is still right
    _check_rows(c, got, "with one refused row")
    c = _case("bf16", 4, 16, seed=8)                                 # the next call starts from GB_OK
    d = _device(c, cuda)
    assert _call(B, c, d) == B.GB_OK
    _check_rows(c, d["out"].cpu().numpy(), "after a refused row")


def test_noalloc_page_id_out_of_range_is_reported(cuda):
    from paper_2608_08020_gb300 import binding as B
    c = _case("f32", 2, 16, seed=9)
    c["tables"][4, 1] = c["num_pages"] + 5                           # row 4 reads 2 pages; the second is bad
    c["seq_len"][4] = 2 * 16
    d = _device(c, cuda)
    assert _call(B, c, d) == B.GB_ERR_INVALID                        # not dereferenced; recorded
    got = d["out"].cpu().numpy()
    assert np.isfinite(got).all()
    c["seq_len"][4] = 0
    got[4] = 0
    _check_rows(c, got, "rows beside the bad page id")


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
    huge = B.GbPagedDecodeArgs(p, p, p, p, p, 1024, 32, 8, 128, 64, B.GB_BF16, 1 << 20, 16, 0.1)
    with pytest.raises(B.GambitError) as e:                          # chunk counts would overflow 32 bits
        B.gb_paged_decode_noalloc(huge)
    assert e.value.code == B.GB_ERR_INVALID
