"""Decode attention, textbook definition, in fp64.

Gambit (Section 3.1, Algorithm 1 "Generate") advances every active trace by
one token per decode step; a branched child attends over the KV it inherited
from its parent's prefix (Section 3.1, the paragraph after Eq. 3: "the child
inherits the parent's KV-cache via prefix caching").  The attention itself is
standard scaled dot-product attention with grouped KV heads: query head ``h``
reads KV head ``h // G`` with ``G = Hq / Hkv``.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import numpy as np


def softmax_weights(q: np.ndarray, K: np.ndarray, scale: float) -> np.ndarray:
    """Softmax weights p[t] = exp(s_t - max s) / sum exp(...), s_t = scale * q.K_t.

    q: [D], K: [L][D]; computed in fp64 with the two-pass (max, then sum) form.
    """
    s = float(scale) * (K.astype(np.float64) @ q.astype(np.float64))
    m = s.max()
    e = np.exp(s - m)
    return e / e.sum()


def decode_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, scale: float) -> np.ndarray:
    """One decode step of GQA attention for one beam.

    q: [Hq][D]; K, V: [L][Hkv][D] (the beam's full context, already rounded to
    the storage dtype); returns o: [Hq][D] in fp64 with
    ``o[h] = sum_t p_h[t] V[t, h // G]`` and ``p_h = softmax(scale * K[:, h//G] q[h])``.
    """
    Hq, D = q.shape
    L, Hkv, D2 = K.shape
    assert D == D2 and V.shape == K.shape and L >= 1 and Hq % Hkv == 0
    G = Hq // Hkv
    o = np.empty((Hq, D), dtype=np.float64)
    for h in range(Hq):
        kh = h // G
        p = softmax_weights(q[h], K[:, kh, :], scale)
        o[h] = p @ V[:, kh, :].astype(np.float64)
    return o
