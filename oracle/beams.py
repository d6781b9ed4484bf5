"""Every beam's full KV context, two ways.

``BeamKV`` is the literal reading of Section 3.1 (Eq. 3 and the paragraph
after it): a branched child continues from a copy of its parent's context.
It keeps, per slot and layer, the full K and V arrays ``[L][Hkv][D]`` and
copies the parent's arrays when a child is branched; nothing is paged or
shared.  It is meant for small cases.

``kv_from_history`` rebuilds the same arrays for one beam from its writer
history (``oracle.pool.PoolOracle.history``) by regenerating every position
from the seeded input generator.  It is how large cases are checked on a
sample of beams; ``tests/test_oracle_pool.py`` checks both give identical
arrays.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import numpy as np

from workload import gen


class BeamKV:
    def __init__(self, num_layers: int, max_beams: int, num_kv_heads: int, head_dim: int):
        self.layers = num_layers
        self.Hkv = num_kv_heads
        self.D = head_dim
        empty = lambda: np.zeros((0, num_kv_heads, head_dim), dtype=np.float32)
        self.K = [[empty() for _ in range(num_layers)] for _ in range(max_beams)]
        self.V = [[empty() for _ in range(num_layers)] for _ in range(max_beams)]

    def seed(self, n_beams: int, k_prompt: list, v_prompt: list) -> None:
        """k_prompt[layer]: [T][Hkv][D]; every root beam gets its own copy."""
        for b in range(n_beams):
            self.K[b] = [np.array(k, dtype=np.float32) for k in k_prompt]
            self.V[b] = [np.array(v, dtype=np.float32) for v in v_prompt]

    def append(self, slot: int, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        self.K[slot][layer] = np.concatenate([self.K[slot][layer], k[None].astype(np.float32)])
        self.V[slot][layer] = np.concatenate([self.V[slot][layer], v[None].astype(np.float32)])

    def append_rows(self, slot: int, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        """Append n rows k, v [n][Hkv][D] to the slot's layer."""
        self.K[slot][layer] = np.concatenate([self.K[slot][layer], np.asarray(k, np.float32)])
        self.V[slot][layer] = np.concatenate([self.V[slot][layer], np.asarray(v, np.float32)])

    def get(self, slot: int, layer: int) -> tuple[np.ndarray, np.ndarray]:
        return self.K[slot][layer], self.V[slot][layer]

    def branch(self, child: int, parent: int) -> None:
        self.K[child] = [a.copy() for a in self.K[parent]]
        self.V[child] = [a.copy() for a in self.V[parent]]

    def release(self, slot: int) -> None:
        self.K[slot] = [a[:0] for a in self.K[slot]]
        self.V[slot] = [a[:0] for a in self.V[slot]]


def kv_from_history(history, seed: int, layer: int, num_kv_heads: int, head_dim: int,
                    dtype: str, hscale=None) -> tuple[np.ndarray, np.ndarray]:
    """K, V ``[L][Hkv][D]`` of one beam rebuilt from its ``(writer, start, end)`` runs."""
    Ks, Vs = [], []
    for writer, start, end in history:
        pos = np.arange(start, end, dtype=np.uint64)
        Ks.append(gen.kv_rows(seed, gen.TAG_KV_K, layer, writer, pos, num_kv_heads, head_dim,
                              dtype, hscale))
        Vs.append(gen.kv_rows(seed, gen.TAG_KV_V, layer, writer, pos, num_kv_heads, head_dim,
                              dtype, hscale))
    return np.concatenate(Ks), np.concatenate(Vs)
