"""Shared-prefix segments of a beam tree, by their definition.

A branched child shares its parent's KV prefix (Section 3.1, after Eq. 3), so
several beams can hold the same page at the same block-table index.  For a
beam b and a full page index i, the sharer set is every active beam whose
table holds the same page at index i.  A segment of b is a maximal run of
consecutive full-page indices with one and the same sharer set, of at least
``group_min`` beams, starting from index 0; b's covered prefix ends at the
first index whose sharer set is smaller than ``group_min``, or after
``max_depth`` segments.

This is computed here from the sharer sets themselves (set equality over all
beams), not from refcounts, so it checks the kernels' refcount-based shortcut.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import numpy as np

from oracle.pool import PoolOracle


def segments(pool: PoolOracle, group_min: int, max_depth: int = 16) -> tuple[np.ndarray, np.ndarray, list]:
    """Returns (cover[b] in pages, nseg[b], per-beam list of (start, length, frozenset sharers))."""
    C = pool.max_beams
    cover = np.zeros(C, dtype=np.int64)
    nseg = np.zeros(C, dtype=np.int64)
    segs = [[] for _ in range(C)]
    active = [b for b in range(C) if pool.active[b]]
    for b in active:
        nfull = int(pool.seq_len[b]) // pool.P
        runs = []
        i = 0
        while i < nfull:
            page = pool.tables[b][i]
            sharers = frozenset(x for x in active
                                if len(pool.tables[x]) > i and pool.tables[x][i] == page)
            if len(sharers) < group_min:
                break
            if runs and runs[-1][2] == sharers:
                runs[-1][1] += 1
            else:
                if len(runs) == max_depth:
                    break
                runs.append([i, 1, sharers])
            i += 1
        cover[b] = sum(r[1] for r in runs) if runs else 0
        nseg[b] = len(runs)
        segs[b] = [tuple(r) for r in runs]
    return cover, nseg, segs
