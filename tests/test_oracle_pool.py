"""Pins for oracle.pool and oracle.beams: page accounting, allocation, copy-on-write, fork semantics."""
import dataclasses

import numpy as np
import pytest

from oracle.attention import decode_attention
from oracle.pool import ERR_INVALID, ERR_OOM, ERR_STATE, PoolOracle
from oracle import backends
from oracle.trajectory import OracleRun
from workload.configs import TINY

NAMES = {'PoolOracle': 'Pool', 'decode_attention': 'decode_attention'}

@pytest.fixture(autouse=True, params=backends.NAMES)
def oracle_backend(request, monkeypatch):
    """Every pin runs on both oracles: the C++ one and its numpy twin."""
    B = backends.get(request.param)
    monkeypatch.setattr(backends, "DEFAULT", request.param)
    for name, attr in NAMES.items():
        monkeypatch.setitem(globals(), name, getattr(B, attr))
    return B


rng = np.random.default_rng(4)


def test_seed_shares_the_lowest_pages():
    p = PoolOracle(num_pages=100, max_beams=8, max_pages_per_beam=20, page_size=16)
    p.seed(8, 64)
    assert all(p.tables[b] == [0, 1, 2, 3] for b in range(8))
    assert list(p.refcnt[:4]) == [8] * 4 and p.refcnt[4:].sum() == 0
    p.check_invariants()


def test_lowest_free_page_in_slot_order_matches_first_fit():
    p = PoolOracle(num_pages=64, max_beams=4, max_pages_per_beam=16, page_size=16)
    p.seed(4, 16)                      # page 0 shared, length 16 -> next step needs a page per beam
    assert p.begin_step()
    assert [p.tables[b][-1] for b in range(4)] == [1, 2, 3, 4]
    # free pages 2 and 4 by releasing slots 1 and 3, then grow: first fit gives 2 then 4
    p.release([1, 3])
    for _ in range(15):
        assert p.begin_step()
    assert p.begin_step()
    assert [p.tables[0][-1], p.tables[2][-1]] == [2, 4]
    p.check_invariants()


def test_prune_frees_only_unshared_pages_and_conserves_refcounts():
    p = PoolOracle(num_pages=200, max_beams=4, max_pages_per_beam=32, page_size=16)
    p.seed(4, 32)                                   # pages 0,1 shared by 4
    for _ in range(32):
        p.begin_step()                              # each beam: 2 private pages
    p.mean[:] = np.array([0.4, 0.3, 0.2, 0.1], np.float32)
    free_before = p.num_free()
    plan, parent_of, pruned = p.prune_branch(K=2, fanout=2)
    assert plan.children == [(2, 0), (3, 1)]
    assert p.num_free() == free_before + 4          # slots 2,3 private pages freed, shared prompt kept
    assert list(parent_of) == [0, 1, 0, 1] and list(pruned) == [0, 0, 1, 1]
    assert p.tables[2] == p.tables[0] and p.tables[3] == p.tables[1]
    assert list(p.refcnt[:2]) == [4, 4]
    p.check_invariants()


def test_fork_of_a_partial_tail_page_copies_on_first_write():
    p = PoolOracle(num_pages=50, max_beams=4, max_pages_per_beam=8, page_size=16)
    p.seed(4, 20)                                   # page 1 is a partial tail (4 tokens), shared by 4
    assert p.begin_step()
    # holders copy in slot order while shared: slots 0,1,2 copy, slot 3 writes in place
    assert [ev[0] for ev in p.cow_events] == [0, 1, 2]
    assert all(ev[1] == 1 and ev[3] == 4 for ev in p.cow_events)
    assert p.tables[3][1] == 1 and p.refcnt[1] == 1
    assert sorted(p.tables[b][1] for b in range(3)) == [2, 3, 4]
    p.check_invariants()


def test_out_of_pages_is_all_or_nothing():
    p = PoolOracle(num_pages=4, max_beams=4, max_pages_per_beam=8, page_size=16)
    p.seed(4, 16)                                   # 1 page used, 3 free, the step needs 4
    before = (p.refcnt.copy(), [list(t) for t in p.tables], p.seq_len.copy())
    assert not p.begin_step()
    assert p.status == ERR_OOM
    assert np.array_equal(before[0], p.refcnt) and before[1] == [list(t) for t in p.tables]
    assert np.array_equal(before[2], p.seq_len)


def test_release_errors():
    p = PoolOracle(num_pages=10, max_beams=2, max_pages_per_beam=4, page_size=16)
    p.seed(2, 16)
    p.release([7])
    assert p.status == ERR_INVALID
    p.status = 0
    p.release([1, 1])
    assert p.status == ERR_STATE and not p.active[1]
    p.check_invariants()


def test_random_operations_keep_invariants():
    for seed in range(5):
        r = np.random.default_rng(seed)
        p = PoolOracle(num_pages=400, max_beams=8, max_pages_per_beam=64, page_size=16)
        p.seed(8, int(r.integers(1, 40)))
        for it in range(120):
            op = r.random()
            if op < 0.7:
                p.begin_step()
            elif op < 0.9:
                p.mean[:] = r.random(8).astype(np.float32)
                p.prune_branch(K=int(r.integers(0, 5)), fanout=int(r.integers(2, 4)))
            else:
                live = np.flatnonzero(p.active)
                if len(live) > 1:
                    p.release([int(r.choice(live))])
            p.check_invariants()


def _tiny(**kw):
    return dataclasses.replace(TINY, **kw)


def test_literal_copy_model_equals_history_rebuild():
    wl = _tiny(prompt_len=20, interval=30, context=100)   # unaligned forks
    run = OracleRun(wl, literal_kv=True)
    run.build(final_round=True)
    hist = OracleRun(wl, literal_kv=False)
    hist.build(final_round=True)
    for b in range(wl.beams):
        K1, V1 = run.beam_kv(b, 0)
        K2, V2 = hist.beam_kv(b, 0)
        np.testing.assert_array_equal(K1, K2)
        np.testing.assert_array_equal(V1, V2)
        assert len(K1) == run.pool.seq_len[b]


def test_branching_leaves_the_parent_unchanged_and_child_matches_parent():
    wl = _tiny()
    run = OracleRun(wl, literal_kv=True)
    run.seed()
    run.append(40)
    run.probe()
    q = run.q(0, 0, run.pos)
    before = {b: decode_attention(q, *run.beam_kv(b, 0), wl.attn_scale) for b in range(wl.beams)}
    plan, parent_of, _ = run.prune()
    for b in range(wl.beams):
        if parent_of[b] == b:   # survivors
            np.testing.assert_array_equal(decode_attention(q, *run.beam_kv(b, 0), wl.attn_scale), before[b])
    for s, p in plan.children:  # a child queried with its parent's q gives the parent's output
        np.testing.assert_array_equal(decode_attention(q, *run.beam_kv(s, 0), wl.attn_scale), before[p])


def test_fork_slots_replays_a_tournament_decided_elsewhere():
    """A second pool that applies the first pool's parent_of ends in the same page state
    as the first (same tables up to page renaming is not enough: both allocate alike, so
    the tables, refcounts and free pages are equal), and a slot whose parent_of is its
    own slot or -1 is untouched."""
    import copy
    for seed in range(6):
        r = np.random.default_rng(seed)
        a = PoolOracle(num_pages=400, max_beams=12, max_pages_per_beam=40, page_size=16)
        a.seed(9, 20)
        for _ in range(int(r.integers(1, 40))):
            a.begin_step()
        b = copy.deepcopy(a)
        a.mean[:] = r.random(12).astype(np.float32)
        _, parent_of, _ = a.prune_branch(K=int(r.integers(0, 5)), fanout=int(r.integers(2, 4)))
        b.fork_slots(parent_of)
        assert a.tables == b.tables
        assert np.array_equal(a.refcnt, b.refcnt) and sorted(a._free) == sorted(b._free)
        assert np.array_equal(a.active, b.active) and np.array_equal(a.seq_len, b.seq_len)
        assert np.array_equal(a.lineage, b.lineage) and np.array_equal(a.gen, b.gen)
        b.check_invariants()
        for _ in range(20):                          # both grow alike afterwards
            a.begin_step()
            b.begin_step()
        assert a.tables == b.tables


def test_fork_slots_by_hand():
    p = PoolOracle(num_pages=50, max_beams=4, max_pages_per_beam=8, page_size=16)
    p.seed(3, 16)                                   # page 0 shared by slots 0..2, lineages 1..3
    for _ in range(16):
        p.begin_step()                              # private pages 1, 2, 3 of slots 0, 1, 2
    p.fork_slots([0, 0, 2, 2])                      # slot 1 <- slot 0; vacant slot 3 <- slot 2
    assert p.tables == [[0, 1], [0, 1], [0, 3], [0, 3]]
    assert list(p.refcnt[:4]) == [4, 2, 0, 2] and p.num_free() == 47
    assert list(p.lineage) == [1, 4, 3, 5] and list(p.seq_len) == [32] * 4 and list(p.gen) == [16, 0, 16, 0]
    p.check_invariants()
    p.fork_slots([-1, 9, -1, -1])                   # a parent out of range is an error, nothing changes
    assert p.status == ERR_INVALID and p.tables[1] == [0, 1]
