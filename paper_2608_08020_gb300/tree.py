"""Algorithm 1's main loop on the GPU beam pool, with the method's Tree view.

Gambit keeps two views of its traces (Section 3.2): the Scheduler view (the traces
that run and hold KV) and the Tree view (every trace the search created, with its
parent, whether it was pruned, completed, or evicted as a "ghost" under memory
pressure).  The device holds the Scheduler view (``BeamPool``); ``TreeView`` is the
host-side Tree view, updated from the outputs of each tournament
(``gb_prune_branch``: parent slot, pruned flag and lineage id per slot) and from
the caller's completions and evictions.

``TournamentLoop`` runs Algorithm 1's loop on the pool:

    while traces run and |F| < C:
        Generate: one thought (``interval`` tokens) for every running trace, then
                  the running-mean update with that thought's score (gb_push_scores);
        on KV saturation, evict the running trace with the lowest mean as a ghost
                  (gb_release; the tree's capacity drops by one, gb_pool_set_capacity);
        Tournament: Case 1 while fewer than C traces count, else Case 2 (gb_prune_branch);
        move completed traces to F (gb_release).

Scores and completion lengths come from the caller (``score_fn``, ``target_fn``),
so a run is driven by seeded synthetic values and reproducible.  Token K/V values
do not matter to the loop's accounting; appends write zeros.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from paper_2608_08020_gb300 import binding as B
from paper_2608_08020_gb300.pool import BeamPool, TORCH_DT

RUNNING, PRUNED, COMPLETED, GHOST = "running", "pruned", "completed", "ghost"


@dataclass
class Node:
    id: int
    parent: int          # node id of the parent, -1 for a root
    lineage: int         # the pool's lineage id
    born: int            # round of creation (0 for roots)
    state: str = RUNNING
    slot: int = -1       # pool slot while running
    length: int = 0      # tokens when it stopped running


@dataclass
class TreeView:
    """Every trace of one search: roots, branches, their states, and the slot map."""
    capacity: int
    nodes: list = field(default_factory=list)
    slot_node: dict = field(default_factory=dict)   # running slot -> node id
    case1_rounds: list = field(default_factory=list)  # (vacant before, branched)
    case2_rounds: list = field(default_factory=list)  # (pruned, branched, running after)

    def add_roots(self, slots, lineages) -> None:
        for s, lin in zip(slots, lineages):
            n = Node(len(self.nodes), -1, int(lin), 0, RUNNING, int(s))
            self.nodes.append(n)
            self.slot_node[int(s)] = n.id

    def apply_round(self, rnd: int, parent_out, pruned_out, lineage_out, lengths) -> list:
        """Record one tournament from the pool's outputs; returns the new children's slots."""
        counted = self.counted()
        pruned = [s for s in range(len(pruned_out)) if pruned_out[s]]
        for s in pruned:
            n = self.nodes[self.slot_node.pop(s)]
            n.state, n.slot, n.length = PRUNED, -1, int(lengths[s])
        children = [s for s in range(len(parent_out)) if parent_out[s] >= 0 and parent_out[s] != s]
        for s in children:
            p = self.slot_node[int(parent_out[s])]
            n = Node(len(self.nodes), p, int(lineage_out[s]), rnd, RUNNING, s)
            self.nodes.append(n)
            self.slot_node[s] = n.id
        if counted >= self.capacity:
            self.case2_rounds.append((len(pruned), len(children), self.running()))
        else:
            self.case1_rounds.append((self.capacity - counted, len(children)))
        return children

    def finish(self, slots, lengths, state: str = COMPLETED) -> None:
        for s in slots:
            n = self.nodes[self.slot_node.pop(int(s))]
            n.state, n.slot, n.length = state, -1, int(lengths[s])

    def count(self, state: str) -> int:
        return sum(1 for n in self.nodes if n.state == state)

    def running(self) -> int:
        return len(self.slot_node)

    def counted(self) -> int:
        """Traces counted against the capacity: the running ones and the ghosts."""
        return self.running() + self.count(GHOST)

    @property
    def roots(self) -> int:
        return sum(1 for n in self.nodes if n.parent < 0)

    @property
    def branches(self) -> int:
        return sum(1 for n in self.nodes if n.parent >= 0)

    def check(self) -> None:
        """Node accounting: nodes = roots + branches = running + pruned + completed + ghosts,
        every Case-2 round branches exactly as many traces as it prunes (zero-sum), and
        the traces counted against the capacity never exceed it."""
        assert len(self.nodes) == self.roots + self.branches
        assert len(self.nodes) == self.running() + self.count(PRUNED) + self.count(COMPLETED) + self.count(GHOST)
        for pr, br, _ in self.case2_rounds:
            assert pr == br, (pr, br)
        assert self.counted() <= self.capacity
        for s, nid in self.slot_node.items():
            assert self.nodes[nid].slot == s and self.nodes[nid].state == RUNNING


class TournamentLoop:
    """Algorithm 1's main loop over a ``BeamPool`` (one layer is enough for the loop)."""

    def __init__(self, pool: BeamPool, C: int, K: int, fanout: int = 2, interval: int = 200, warmup: int = 0,
                 prompt_len: int = 64):
        self.pool, self.C, self.K, self.fanout = pool, C, K, fanout
        self.interval, self.warmup, self.prompt_len = interval, warmup, prompt_len
        cfg = pool.cfg
        self.dev = pool.device
        self.dt = TORCH_DT[pool.kv_dtype]
        self.kv_shape = (cfg.max_beams, cfg.num_kv_heads, cfg.head_dim)
        self.k_zero = torch.zeros((interval,) + self.kv_shape, dtype=self.dt, device=self.dev)
        self.scores = torch.zeros(cfg.max_beams, dtype=torch.float32, device=self.dev)
        self.parent = torch.empty(cfg.max_beams, dtype=torch.int32, device=self.dev)
        self.pruned = torch.empty(cfg.max_beams, dtype=torch.uint8, device=self.dev)
        self.lineage = torch.empty(cfg.max_beams, dtype=torch.int32, device=self.dev)
        self.length = np.zeros(cfg.max_beams, dtype=np.int64)   # generated tokens (after the prompt)
        self.target = np.zeros(cfg.max_beams, dtype=np.int64)   # completion length in generated tokens
        self.tree = TreeView(C)
        self.evictions = 0
        self.victim = torch.zeros(1, dtype=torch.int32, device=self.dev)   # slot chosen by gb_pool_last_ranked

    def _append(self) -> bool:
        """One thought for every running trace; False (and nothing appended) if the pool ran
        out of pages: the pool reserves the whole step's pages or none."""
        for layer in range(self.pool.cfg.num_layers):
            self.pool.append_kv(layer, self.interval, self.k_zero, self.k_zero)
        return self.pool.status() == 0

    def _evict_lowest(self) -> None:
        """Memory pressure: the running trace with the lowest mean becomes a ghost (Alg. 1, Section 3.2).
        The device picks it (the tournament's ranking read from its end) and releases it; the
        host reads back only the slot id, for the Tree view."""
        self.pool.last_ranked(self.victim)
        self.pool.release(self.victim)
        victim = int(self.victim.item())
        assert victim in self.tree.slot_node, (victim, "the pool's active slots are the running traces")
        self.tree.finish([victim], self.length, GHOST)
        self.evictions += 1
        self.pool.set_capacity(self.C - self.tree.count(GHOST))

    def seed(self, initial_targets) -> None:
        cfg = self.pool.cfg
        T = self.prompt_len
        kp = torch.zeros((cfg.num_layers, T, cfg.num_kv_heads, cfg.head_dim), dtype=self.dt, device=self.dev)
        self.pool.seed(self.C, T, kp, kp)
        self.pool.set_capacity(self.C)
        st = self.pool.read_state()
        self.tree.add_roots(range(self.C), st["lineage"][: self.C])
        self.length[: self.C] = 0
        self.target[: self.C] = initial_targets

    def run(self, score_fn, target_fn, max_rounds: int = 100000, on_round=None) -> TreeView:
        """score_fn(slots) -> fp32 score per listed running slot (slot order);
        target_fn(child_slots, parent_lengths) -> completion length of each new child."""
        tree = self.tree
        rnd = 0
        while tree.running() > 0 and tree.count(COMPLETED) < self.C and rnd < max_rounds:
            rnd += 1
            # Generate one thought per running trace; evict under memory pressure.
            while not self._append():
                self.pool.clear_status()
                if tree.running() == 0:
                    return tree
                self._evict_lowest()
            run = sorted(tree.slot_node)
            self.length[run] += self.interval
            sc = np.zeros(self.pool.cfg.max_beams, dtype=np.float32)
            sc[run] = np.asarray(score_fn(run), dtype=np.float32)
            self.scores.copy_(torch.from_numpy(sc))
            self.pool.push_scores(self.scores)
            # Tournament.
            self.pool.prune_branch(self.K, self.fanout, self.warmup, None, self.parent, self.pruned, self.lineage)
            parent = self.parent.cpu().numpy()
            pruned = self.pruned.cpu().numpy()
            lineage = self.lineage.cpu().numpy().view(np.uint32)
            children = tree.apply_round(rnd, parent, pruned, lineage, self.length)
            for s in children:
                self.length[s] = self.length[parent[s]]
            if children:
                self.target[children] = np.asarray(target_fn(children, self.length[children]), dtype=np.int64)
            # Move completed traces to F.
            done = [s for s in sorted(tree.slot_node) if self.length[s] >= self.target[s]]
            done = done[: self.C - tree.count(COMPLETED)]
            if done:
                tree.finish(done, self.length, COMPLETED)
                self.pool.release(torch.tensor(done, dtype=torch.int32, device=self.dev))
            if on_round is not None:
                on_round(rnd, tree)
        return tree
