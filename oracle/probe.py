"""Scorer probe and running mean score (Algorithm 1 "Generate"; Section 3.1).

The paper scores a trace at each thought boundary with a scorer
``f_theta(h_n)`` on the last-layer hidden state and keeps the running average
``s_bar <- s_bar + (f_theta(h_n) - s_bar) / n`` (Algorithm 1), which equals
``(1/n) * sum_j f_theta(h_j)`` (Section 3.1, the ranking paragraph).  The
probe used here is the linear-plus-sigmoid form ``sigma(w.h + b)``.

Precision: the probe is evaluated in fp64.  The running mean is kept in fp32
(the precision the ranking decision is taken in) with each of the three
operations - subtract, divide, add - rounded separately, in the order the
update is written.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import numpy as np


def probe_score(h: np.ndarray, w: np.ndarray, bias: float) -> np.ndarray:
    """sigma(w.h + b) in fp64.  h: [..., H], w: [H] -> [...]."""
    z = h.astype(np.float64) @ w.astype(np.float64) + float(bias)
    return 1.0 / (1.0 + np.exp(-z))


def mlp_probe_score(h: np.ndarray, w1: np.ndarray, b1: np.ndarray, w2: np.ndarray, b2: float) -> np.ndarray:
    """The two-layer MLP scorer sigma(w2 . relu(W1 h + b1) + b2) in fp64 (Section 4 uses a
    2-layer MLP scorer; ReLU between the layers).  h: [..., H], w1: [d_h, H], b1, w2: [d_h]."""
    z = h.astype(np.float64) @ w1.astype(np.float64).T + b1.astype(np.float64)
    y = np.maximum(z, 0.0) @ w2.astype(np.float64) + float(b2)
    return 1.0 / (1.0 + np.exp(-y))


def running_mean_update(mean: np.float32, n: int, x: np.float32) -> tuple[np.float32, int]:
    """One step of s_bar <- s_bar + (x - s_bar)/n with n counting this score.

    Returns (new_mean, new_n).  ``n`` is the number of scores seen so far
    (before this one); the division uses the incremented count.
    """
    n1 = n + 1
    d = np.float32(np.float32(x) - np.float32(mean))
    q = np.float32(d / np.float32(n1))
    return np.float32(np.float32(mean) + q), n1
