"""Comparison helpers for GPU-vs-oracle parity tests."""
from __future__ import annotations

import numpy as np

# Tolerances (|got - ref| <= atol + rtol * |ref| for every element).
TOL = {"f32": (1e-5, 1e-5), "bf16": (2e-3, 1e-2)}


def assert_close(got, ref, dtype: str, what: str = "") -> tuple[float, float]:
    atol, rtol = TOL[dtype]
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    err = np.abs(got - ref)
    bound = atol + rtol * np.abs(ref)
    max_abs = float(err.max()) if err.size else 0.0
    max_rel = float((err / np.maximum(np.abs(ref), 1e-30)).max()) if err.size else 0.0
    bad = ~(err <= bound)
    if bad.any():
        i = np.unravel_index(int(np.argmax(err - bound)), err.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} elements out of tolerance; worst at {i}: "
                             f"got {got[i]!r} ref {ref[i]!r}; max-abs {max_abs:.3g} max-rel {max_rel:.3g}")
    return max_abs, max_rel


def assert_pool_equal(st: dict, pool, P: int, means: str = "exact", dtype: str = "f32") -> None:
    """Bit-exact comparison of the library's pool state with oracle.pool.PoolOracle."""
    C = len(pool.tables)
    act = np.asarray(st["active"]) != 0
    assert np.array_equal(act, pool.active), ("active", np.flatnonzero(act ^ pool.active))
    assert np.array_equal(st["seq_len"][act], pool.seq_len[act]), "seq_len"
    for b in range(C):
        if pool.active[b]:
            n = -(-int(pool.seq_len[b]) // P)
            got = [int(x) for x in st["tables"][b][:n]]
            assert got == pool.tables[b], f"table of slot {b}: {got} vs {pool.tables[b]}"
    assert np.array_equal(st["refcnt"], pool.refcnt), f"refcnt differs at {np.flatnonzero(st['refcnt'] != pool.refcnt)[:10]}"
    assert np.array_equal(st["free_bits"], pool.free_bits()), "free bitmap"
    assert np.array_equal(st["gen"][act], pool.gen[act]), "gen"
    assert np.array_equal(st["nsteps"][act], pool.nsteps[act]), "nsteps"
    assert np.array_equal(st["lineage"][act], pool.lineage[act]), "lineage"
    if means == "exact":
        assert np.array_equal(st["mean"][act].view(np.uint32), pool.mean[act].view(np.uint32)), "mean bits"
    else:
        assert_close(st["mean"][act], pool.mean[act], dtype, "mean")
