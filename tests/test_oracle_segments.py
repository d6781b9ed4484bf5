"""Pins for oracle.segments: hand-built trees with known shared runs."""
import numpy as np

from oracle.pool import PoolOracle
from oracle.segments import segments


def _pool(C=8, P=16):
    return PoolOracle(num_pages=4096, max_beams=C, max_pages_per_beam=64, page_size=P)


def test_prompt_shared_by_all():
    p = _pool()
    p.seed(8, 70)                       # 4 full pages + a partial one, shared by all 8
    cover, nseg, segs = segments(p, group_min=4)
    assert list(cover) == [4] * 8 and list(nseg) == [1] * 8
    assert segs[0][0][0] == 0 and segs[0][0][1] == 4 and len(segs[0][0][2]) == 8
    cover, nseg, _ = segments(p, group_min=9)
    assert cover.sum() == 0 and nseg.sum() == 0


def test_two_levels_after_a_round():
    p = _pool()
    p.seed(8, 32)                       # 2 shared pages
    for _ in range(32):
        p.begin_step()                  # each beam: 2 private pages
    p.mean[:] = np.linspace(0.9, 0.2, 8).astype(np.float32)
    p.prune_branch(K=4, fanout=2)       # beams 0-3 keep, 4-7 become their children
    for _ in range(16):
        p.begin_step()                  # each beam: 1 more private page
    cover, nseg, segs = segments(p, group_min=2)
    # prompt pages shared by 8, then 2 pages shared by each (parent, child) pair, then private
    assert list(cover) == [4] * 8 and list(nseg) == [2] * 8
    assert [s[1] for s in segs[0]] == [2, 2]
    assert segs[0][1][2] == frozenset({0, 4})
    cover, nseg, _ = segments(p, group_min=3)
    assert list(cover) == [2] * 8 and list(nseg) == [1] * 8


def test_depth_cap_and_partial_pages():
    p = _pool(C=4)
    p.seed(4, 16)
    for r in range(6):                  # a chain of forks: pairs share ever deeper prefixes
        for _ in range(16):
            p.begin_step()
        p.mean[:] = np.array([0.9, 0.1, 0.2, 0.3], np.float32)
        p.prune_branch(K=1, fanout=2)
    cover, nseg, segs = segments(p, group_min=2, max_depth=3)
    assert all(n <= 3 for n in nseg)
    full = [int(p.seq_len[b]) // 16 for b in range(4)]
    assert all(cover[b] <= full[b] for b in range(4))
    # the partial tail page (none here, lengths are page aligned) is never part of a segment
    p.begin_step()
    cover2, _, _ = segments(p, group_min=2, max_depth=3)
    assert all(cover2[b] <= int(p.seq_len[b]) // 16 for b in range(4))
