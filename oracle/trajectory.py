"""Run a workload schedule on the oracle.

Mirrors the schedule of ``workload.configs`` on the oracle's pool (``oracle.cpp.CppPool``, or
``oracle.pool.PoolOracle`` with the numpy backend):
seeding, decode steps (every layer), chunked appends, the probe with the
running-mean update, and tournament rounds.  Attention outputs come from each
beam's full KV: the literal copy-on-fork arrays (``CppBeamKV`` / ``oracle.beams.BeamKV``) for
small cases, or the KV rebuilt from the writer history for sampled beams of
large cases.  Every input is regenerated here from the seeded generator; no
value is taken from the CUDA path.  The arithmetic (attention, probe, running mean,
tournament, pool) comes from the chosen oracle backend (``oracle.backends``): the C++
oracle by default, or its numpy twin.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import numpy as np

from oracle import backends
from oracle.beams import kv_from_history
from workload import gen
from workload.configs import Workload


class OracleRun:
    def __init__(self, wl: Workload, literal_kv: bool = True, num_pages: int | None = None,
                 max_context: int | None = None, backend: str | None = None):
        self.wl = wl
        self.B = backends.get(backend or backends.DEFAULT)
        self.pool = self.B.Pool(num_pages if num_pages is not None else wl.pool_pages(max_context), wl.beams,
                                wl.table_width(max_context), wl.page_size)
        self.kv = self.B.BeamKV(wl.num_layers, wl.beams, wl.num_kv_heads, wl.head_dim) if literal_kv else None
        self.hscale = None
        if wl.head_scale is not None:
            self.hscale = [gen.head_scales(wl.seed, l, wl.num_kv_heads, *wl.head_scale)
                           for l in range(wl.num_layers)]
        self.w = gen.probe_weight(wl.seed, wl.hidden, wl.w_scale)
        self.pos = 0

    def _kv(self, which, layer, writers, positions):
        wl = self.wl
        return gen.kv_rows(wl.seed, which, layer, writers, positions, wl.num_kv_heads, wl.head_dim, wl.kv_dtype,
                           self.hscale[layer] if self.hscale else None)

    def q(self, layer: int, slot: int, pos: int) -> np.ndarray:
        wl = self.wl
        return gen.q_rows(wl.seed, layer, slot, pos, wl.num_q_heads, wl.head_dim, wl.kv_dtype, wl.q_scale)

    def seed(self) -> None:
        wl = self.wl
        T = wl.prompt_len
        self.pool.seed(wl.beams, T)
        if self.kv is not None:
            pos = np.arange(T, dtype=np.uint64)
            kp = [self._kv(gen.TAG_KV_K, l, gen.PROMPT_WRITER, pos) for l in range(wl.num_layers)]
            vp = [self._kv(gen.TAG_KV_V, l, gen.PROMPT_WRITER, pos) for l in range(wl.num_layers)]
            self.kv.seed(wl.beams, kp, vp)
        self.pos = T

    def beam_kv(self, slot: int, layer: int) -> tuple[np.ndarray, np.ndarray]:
        """The full K, V of a beam: literal arrays when kept, else rebuilt from its writer history."""
        if self.kv is not None:
            return self.kv.get(slot, layer)
        wl = self.wl
        return kv_from_history(self.pool.history[slot], wl.seed, layer, wl.num_kv_heads, wl.head_dim,
                               wl.kv_dtype, self.hscale[layer] if self.hscale else None)

    def attention(self, slot: int, layer: int, pos: int) -> np.ndarray:
        K, V = self.beam_kv(slot, layer)
        return self.B.decode_attention(self.q(layer, slot, pos), K, V, self.wl.attn_scale)

    def decode_step(self, compute: bool = True, slots=None, layers=None) -> dict | None:
        """One token per active beam and layer; returns {(layer, slot): o} when compute, for the
        given slots and layers (default: every active slot and every layer).

        Returns None (and changes nothing) when the pool is out of pages.
        """
        wl = self.wl
        pos = self.pos
        if not self.pool.begin_step():
            return None
        active = [int(b) for b in np.flatnonzero(self.pool.active)]
        want = active if slots is None else [s for s in slots if s in active]
        outs = {}
        for layer in range(wl.num_layers):
            if self.kv is not None:
                k = self._kv(gen.TAG_KV_K, layer, np.asarray(active, np.uint64), pos)
                v = self._kv(gen.TAG_KV_V, layer, np.asarray(active, np.uint64), pos)
                for i, b in enumerate(active):
                    self.kv.append(b, layer, k[i], v[i])
            if compute and (layers is None or layer in layers):
                for b in want:
                    outs[(layer, b)] = self.attention(b, layer, pos)
        self.pos += 1
        return outs

    def append(self, n: int) -> None:
        wl = self.wl
        active = [int(b) for b in np.flatnonzero(self.pool.active)]
        for _ in range(n):
            if not self.pool.begin_step():
                raise RuntimeError("oracle pool out of pages")
        if self.kv is not None:
            pos = np.arange(self.pos, self.pos + n, dtype=np.uint64)
            for layer in range(wl.num_layers):
                for b in active:
                    self.kv.append_rows(b, layer, self._kv(gen.TAG_KV_K, layer, b, pos),
                                        self._kv(gen.TAG_KV_V, layer, b, pos))
        self.pos += n

    def probe_scores(self, slots=None) -> dict:
        """fp64 probe score of each active slot at the current position."""
        wl = self.wl
        slots = [int(b) for b in np.flatnonzero(self.pool.active)] if slots is None else slots
        h = gen.hidden_rows(wl.seed, np.asarray(slots), self.pos, wl.hidden, wl.hidden_dtype)
        s = self.B.probe_score(h, self.w, wl.bias)
        return dict(zip(slots, s))

    def probe(self, mask=None) -> dict:
        """Probe every active slot and apply the fp32 running-mean update to the masked ones."""
        scores = self.probe_scores()
        for b, x in scores.items():
            if mask is None or mask[b]:
                m, n = self.B.running_mean_update(self.pool.mean[b], int(self.pool.nsteps[b]), np.float32(x))
                self.pool.mean[b] = m
                self.pool.nsteps[b] = n
        return scores

    def push_scores(self, scores32: np.ndarray, mask=None) -> None:
        for b in np.flatnonzero(self.pool.active):
            if mask is None or mask[b]:
                m, n = self.B.running_mean_update(self.pool.mean[b], int(self.pool.nsteps[b]),
                                                  np.float32(scores32[b]))
                self.pool.mean[b] = m
                self.pool.nsteps[b] = n

    def prune(self, K: int | None = None, fanout: int | None = None, warmup: int | None = None, eligible=None):
        wl = self.wl
        plan, parent_of, pruned = self.pool.prune_branch(wl.K if K is None else K,
                                                         wl.fanout if fanout is None else fanout,
                                                         wl.warmup if warmup is None else warmup, eligible)
        if self.kv is not None:
            for s, p in plan.children:
                self.kv.branch(s, p)
        return plan, parent_of, pruned

    def build(self, upto: int | None = None, final_round: bool = False) -> None:
        wl = self.wl
        upto = wl.context if upto is None else upto
        self.seed()
        for L in wl.rounds(include_final=final_round):
            if L > upto:
                break
            self.append(L - self.pos)
            self.probe()
            self.prune()
        if upto > self.pos:
            self.append(upto - self.pos)

    def decision_margin(self) -> float:
        """Smallest gap between fp32 means at the tournament's decision boundaries (for tie diagnostics)."""
        order = sorted(np.flatnonzero(self.pool.active), key=lambda s: -float(self.pool.mean[s]))
        m = [float(self.pool.mean[s]) for s in order]
        gaps = [abs(m[i] - m[i + 1]) for i in range(len(m) - 1) if m[i] != m[i + 1]]
        return min(gaps) if gaps else float("inf")
