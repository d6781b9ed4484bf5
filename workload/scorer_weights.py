"""Seeded random weights for the sequence scorer (no trained scorer exists here).

Matrices are drawn N(0, 1/fan_in) and rounded to bf16 (held as fp32 so both the oracle
and the device see the same values); LayerNorm gains 1 + N(0, 0.01), biases N(0, 0.01);
the output vector N(0, 1/d).  Numbers only: no part of the scorer's arithmetic.
"""
from __future__ import annotations

import numpy as np


def _bf16(x: np.ndarray) -> np.ndarray:
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return u.astype(np.uint32).view(np.float32)


def seqscorer_weights(seed: int, hidden: int, d_model: int, ffn: int, layers: int, n_q_heads: int,
                      n_kv_heads: int, head_dim: int = 128) -> dict:
    rng = np.random.default_rng(seed)
    mat = lambda rows, cols: _bf16(rng.standard_normal((rows, cols)) / np.sqrt(cols))
    ln = lambda n: ((1.0 + 0.1 * rng.standard_normal(n)).astype(np.float32),
                    (0.1 * rng.standard_normal(n)).astype(np.float32))
    out = {"ln_in": ln(hidden), "w_in": mat(d_model, hidden), "layers": []}
    for _ in range(layers):
        out["layers"].append({
            "ln1": ln(d_model), "wq": mat(n_q_heads * head_dim, d_model), "wk": mat(n_kv_heads * head_dim, d_model),
            "wv": mat(n_kv_heads * head_dim, d_model), "wo": mat(d_model, d_model), "ln2": ln(d_model),
            "w1": mat(ffn, d_model), "w3": mat(ffn, d_model), "w2": mat(d_model, ffn)})
    out["ln_out"] = ln(d_model)
    out["w_out"] = (rng.standard_normal(d_model) / np.sqrt(d_model)).astype(np.float32)
    out["b_out"] = 0.0
    out["n_q_heads"], out["n_kv_heads"] = n_q_heads, n_kv_heads
    return out
