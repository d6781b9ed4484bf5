"""The paged, refcounted KV pool as plain Python state.

What the paper fixes (Section 3.1, the paragraph after Eq. 3; Section 3.2):

* branching spawns a child that inherits the parent's KV through prefix
  caching - no KV is copied;
* pruning terminates a trace and frees only its non-shared KV blocks;
* the active count stays C (zero-sum).

What this model adds, as the definition the CUDA pool must reproduce bit for
bit (each a reading of a passage where the paper is silent):

* a page holds ``P`` consecutive token positions of one beam's context for
  every layer; a slot's block table lists its pages in position order;
* ``refcnt[p]`` is the number of active slots whose table holds page ``p``;
  a page is free exactly when ``refcnt[p] == 0``;
* allocation always takes the lowest free page id; within one decode step
  beams allocate in ascending slot order, and a multi-token append is that
  many decode steps in sequence;
* a branched child shares every page of its parent, including a partly
  filled tail page; the first append to a tail page that is still shared
  copies it to a fresh page (copy-on-write).  Beams take that decision in
  ascending slot order against the current refcount, so every holder but
  the highest-numbered one copies, and that one writes in place;
* a step that cannot get every page it needs changes nothing and reports
  out-of-memory.

Each slot also records its writer history: the list of ``(writer, start,
end)`` runs saying which slot wrote positions ``[start, end)`` of its
context (``workload.gen.PROMPT_WRITER`` for the prompt), which is what the
seeded input generator is keyed by.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import heapq

import numpy as np

from oracle.tournament import TournamentPlan, tournament

# Status codes, same meaning as the library's.
OK, ERR_INVALID, ERR_OOM, ERR_STATE = 0, 1, 2, 4

PROMPT_WRITER = 0xFFFFFFFF


class PoolOOM(Exception):
    pass


class PoolOracle:
    def __init__(self, num_pages: int, max_beams: int, max_pages_per_beam: int, page_size: int):
        self.num_pages = num_pages
        self.max_beams = max_beams
        self.capacity = max_beams   # the tree's capacity C for the tournament (Section 3.2: ghosts count)
        self.max_pages = max_pages_per_beam
        self.P = page_size
        self.refcnt = np.zeros(num_pages, dtype=np.int64)
        self._free = list(range(num_pages))  # min-heap of free page ids
        heapq.heapify(self._free)
        self.tables: list[list[int]] = [[] for _ in range(max_beams)]
        self.seq_len = np.zeros(max_beams, dtype=np.int64)
        self.active = np.zeros(max_beams, dtype=bool)
        self.gen = np.zeros(max_beams, dtype=np.int64)        # tokens since own creation
        self.mean = np.zeros(max_beams, dtype=np.float32)     # running mean score
        self.nsteps = np.zeros(max_beams, dtype=np.int64)     # scored steps n
        self.lineage = np.zeros(max_beams, dtype=np.uint32)
        self.next_lineage = 1
        self.history: list[list[list[int]]] = [[] for _ in range(max_beams)]
        self.status = OK
        self.cow_events: list[tuple[int, int, int, int]] = []  # (slot, old, new, tokens copied)

    # -- page bookkeeping --------------------------------------------------
    def _alloc(self) -> int:
        p = heapq.heappop(self._free)
        assert self.refcnt[p] == 0
        self.refcnt[p] = 1
        return p

    def _unref(self, p: int) -> None:
        self.refcnt[p] -= 1
        assert self.refcnt[p] >= 0
        if self.refcnt[p] == 0:
            heapq.heappush(self._free, p)

    def _ref(self, p: int) -> None:
        assert self.refcnt[p] >= 1, "a shared page is always already referenced"
        self.refcnt[p] += 1

    def num_free(self) -> int:
        return len(self._free)

    def free_bits(self) -> np.ndarray:
        """Bit p of word p//32 is set when page p is free."""
        words = np.zeros((self.num_pages + 31) // 32, dtype=np.uint32)
        for p in np.flatnonzero(self.refcnt == 0):
            words[p // 32] |= np.uint32(1 << (p % 32))
        return words

    def _set_error(self, code: int) -> None:
        if self.status == OK:
            self.status = code

    # -- operations --------------------------------------------------------
    def seed(self, n_beams: int, prompt_len: int) -> None:
        """n_beams root traces sharing one prompt of prompt_len tokens."""
        assert 1 <= n_beams <= self.max_beams and prompt_len >= 1
        npg = -(-prompt_len // self.P)
        if npg > self.max_pages or npg > self.num_free():
            raise PoolOOM
        pages = [self._alloc() for _ in range(npg)]
        for p in pages:
            self.refcnt[p] = n_beams
        for b in range(n_beams):
            self.tables[b] = list(pages)
            self.seq_len[b] = prompt_len
            self.active[b] = True
            self.gen[b] = 0
            self.mean[b] = np.float32(0.0)
            self.nsteps[b] = 0
            self.lineage[b] = self.next_lineage + b
            self.history[b] = [[PROMPT_WRITER, 0, prompt_len]]
        self.next_lineage += n_beams

    def _step_needs(self) -> int:
        """Pages one decode step needs (new pages + copy-on-write copies)."""
        need = 0
        shared_tail = {}
        for b in np.flatnonzero(self.active):
            L = int(self.seq_len[b])
            if L % self.P == 0:
                need += 1
            else:
                t = self.tables[b][L // self.P]
                shared_tail[t] = shared_tail.get(t, 0) + 1
        for t, holders in shared_tail.items():
            # holders copy in slot order while the page is still shared
            need += min(holders, int(self.refcnt[t]) - 1)
        return need

    def begin_step(self) -> bool:
        """Reserve position seq_len[b] for every active beam; True on success."""
        act = [int(b) for b in np.flatnonzero(self.active)]
        for b in act:
            L = int(self.seq_len[b])
            if L % self.P == 0 and L // self.P >= self.max_pages:
                self._set_error(ERR_OOM)
                return False
        if self._step_needs() > self.num_free():
            self._set_error(ERR_OOM)
            return False
        for b in act:
            L = int(self.seq_len[b])
            if L % self.P == 0:
                self.tables[b].append(self._alloc())
            else:
                old = self.tables[b][L // self.P]
                if self.refcnt[old] > 1:
                    new = self._alloc()
                    self.refcnt[old] -= 1
                    self.tables[b][L // self.P] = new
                    self.cow_events.append((b, old, new, L % self.P))
            self.seq_len[b] = L + 1
            self.gen[b] += 1
            h = self.history[b]
            if h and h[-1][0] == b and h[-1][2] == L:
                h[-1][2] = L + 1
            else:
                h.append([b, L, L + 1])
        return True

    def eligible(self, warmup: int, mask: np.ndarray | None) -> np.ndarray:
        e = self.gen >= warmup
        if mask is not None:
            e = e & (np.asarray(mask) != 0)
        return e & self.active

    def prune_branch(self, K: int, fanout: int, warmup: int = 0,
                     mask: np.ndarray | None = None) -> tuple[TournamentPlan, np.ndarray, np.ndarray]:
        """One tournament round; returns (plan, parent_of, pruned flags)."""
        plan = tournament(self.mean, self.active, self.eligible(warmup, mask),
                          self.capacity, K, fanout)
        was_active = self.active.copy()
        self._make_children(plan.children)
        parent_of = np.where(was_active, np.arange(self.max_beams), -1).astype(np.int64)
        for s, par in plan.children:
            parent_of[s] = par
        pruned = np.zeros(self.max_beams, dtype=np.uint8)
        pruned[plan.pruned] = 1
        return plan, parent_of, pruned

    def fork_slots(self, parent_of) -> None:
        """Apply a tournament decided on another pool (its parent_of): every slot s with
        parent_of[s] >= 0 and != s becomes a child of parent_of[s] (Section 3.1: a branch
        continues from its parent's cached prefix), in ascending slot order."""
        children = [(s, int(p)) for s, p in enumerate(parent_of) if p >= 0 and p != s]
        if any(p >= self.max_beams for _, p in children):
            self._set_error(ERR_INVALID)
        self._make_children([(s, p) for s, p in children if p < self.max_beams])

    def _make_children(self, children) -> None:
        """Each (slot, parent): the slot drops its references and takes the parent's table
        (no copy), length, mean and step count, gen 0 and a fresh lineage id."""
        for s, _ in children:               # the slot's old references go first
            if self.active[s]:
                for p in self.tables[s]:
                    self._unref(p)
        for k, (s, par) in enumerate(children):
            self.tables[s] = list(self.tables[par])
            for p in self.tables[s]:
                self._ref(p)
            self.seq_len[s] = self.seq_len[par]
            self.mean[s] = self.mean[par]
            self.nsteps[s] = self.nsteps[par]
            self.gen[s] = 0
            self.lineage[s] = self.next_lineage + k
            self.active[s] = True
            self.history[s] = [list(r) for r in self.history[par]]
        self.next_lineage += len(children)

    def release(self, slots) -> None:
        """Completed or evicted traces drop their page references."""
        for s in slots:
            s = int(s)
            if s < 0 or s >= self.max_beams:
                self._set_error(ERR_INVALID)
                continue
            if not self.active[s]:
                self._set_error(ERR_STATE)
                continue
            for p in self.tables[s]:
                self._unref(p)
            self.tables[s] = []
            self.active[s] = False
            self.seq_len[s] = 0
            self.gen[s] = 0
            self.history[s] = []

    # -- invariants ----------------------------------------------------------
    def check_invariants(self) -> None:
        """Refcount conservation and the free-page identity."""
        counted = np.zeros(self.num_pages, dtype=np.int64)
        for b in np.flatnonzero(self.active):
            assert len(self.tables[b]) == -(-int(self.seq_len[b]) // self.P)
            for p in self.tables[b]:
                counted[p] += 1
        assert np.array_equal(counted, self.refcnt)
        assert self.refcnt.sum() == sum(len(self.tables[b]) for b in np.flatnonzero(self.active))
        assert self.num_free() == self.num_pages - int((self.refcnt > 0).sum())
        assert sorted(self._free) == list(np.flatnonzero(self.refcnt == 0))
