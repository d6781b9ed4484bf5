"""The history-aware sequence scorer (Appendix, "Evaluating Search Generalization", Eq. 4-6)
in fp64, by its definition.

For a trace's sequence of step hidden states h_1 .. h_T:
    x_t = GELU(W_in LN(h_t))                                               (Eq. 4)
    z_1 .. z_T = SequenceTransformer(x_1 .. x_T)                           (Eq. 5)
    y_t = sigmoid(w_out . LN(z_t) + b_out)                                 (Eq. 6)
The transformer has L pre-norm layers, each multi-head causal self-attention with rotary
position embeddings followed by a SwiGLU feed-forward network:
    a = x + W_o Attn(RoPE(W_q LN1(x)), RoPE(W_k LN1(x)), W_v LN1(x))
    x = a + W_2 (SiLU(W_1 LN2(a)) * W_3 LN2(a))
Readings where the appendix is silent: LayerNorm with gain and bias (eps 1e-5); exact
(erf) GELU; grouped-query attention with Hq query heads of 128 dims over Hkv key/value
heads (query head h reads key/value head h // (Hq / Hkv)); rotary embedding on
(dim i, dim i + 64) pairs with angle t * 10000^(-i / 64); softmax scale 1 / sqrt(128); an
output bias b_out.  Position t counts steps from 0, and every trace's sequence starts with
the hidden state at the end of the shared prompt (step 0).

Weights are inputs (``SeqScorerWeights``); the matrices are bf16 values held in fp32.
Every position is computed from the whole prefix (no cache), so causality is by
construction: y_t depends on h_1 .. h_t only.

This module is oracle code (test infrastructure), see ``oracle/__init__.py``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

HEAD_DIM = 128
EPS = 1e-5


@dataclass
class SeqScorerWeights:
    ln_in: tuple        # (gain [H], bias [H])
    w_in: np.ndarray    # [d, H]
    layers: list        # per layer: dict ln1, wq [Hq*128, d], wk [Hkv*128, d], wv [Hkv*128, d], wo [d, d],
                        #            ln2, w1 [F, d], w3 [F, d], w2 [d, F]
    ln_out: tuple       # (gain [d], bias [d])
    w_out: np.ndarray   # [d]
    b_out: float
    n_q_heads: int
    n_kv_heads: int


def layer_norm(x: np.ndarray, gain: np.ndarray, bias: np.ndarray) -> np.ndarray:
    x = x.astype(np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + EPS) * gain.astype(np.float64) + bias.astype(np.float64)


def gelu(x: np.ndarray) -> np.ndarray:
    erf = np.vectorize(math.erf)
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def rope(x: np.ndarray, pos: np.ndarray) -> np.ndarray:
    """Rotate (i, i + 64) pairs of the last axis by angle pos * 10000^(-i / 64).
    x: [T, heads, 128], pos: [T]."""
    half = HEAD_DIM // 2
    inv = 10000.0 ** (-np.arange(half, dtype=np.float64) / half)
    ang = pos.astype(np.float64)[:, None] * inv[None, :]            # [T, 64]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """q: [T, Hq, 128], k, v: [T, Hkv, 128] -> [T, Hq, 128]; position t sees 0..t."""
    T, Hq, _ = q.shape
    G = Hq // k.shape[1]
    out = np.zeros_like(q)
    for h in range(Hq):
        s = q[:, h, :] @ k[:, h // G, :].T / math.sqrt(HEAD_DIM)    # [T, T]
        s = np.where(np.tril(np.ones((T, T), dtype=bool)), s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, h // G, :]
    return out


def seq_scores(hs: np.ndarray, w: SeqScorerWeights) -> np.ndarray:
    """Scores y_1 .. y_T (Eq. 6) of one step sequence hs [T, H], fp64."""
    f64 = lambda a: np.asarray(a, dtype=np.float64)
    T = hs.shape[0]
    pos = np.arange(T)
    x = gelu(layer_norm(hs, *w.ln_in) @ f64(w.w_in).T)              # Eq. 4
    for L in w.layers:                                              # Eq. 5
        u = layer_norm(x, *L["ln1"])
        q = rope((u @ f64(L["wq"]).T).reshape(T, w.n_q_heads, HEAD_DIM), pos)
        k = rope((u @ f64(L["wk"]).T).reshape(T, w.n_kv_heads, HEAD_DIM), pos)
        v = (u @ f64(L["wv"]).T).reshape(T, w.n_kv_heads, HEAD_DIM)
        x = x + causal_attention(q, k, v).reshape(T, -1) @ f64(L["wo"]).T
        u = layer_norm(x, *L["ln2"])
        x = x + (silu(u @ f64(L["w1"]).T) * (u @ f64(L["w3"]).T)) @ f64(L["w2"]).T
    z = layer_norm(x, *w.ln_out)                                    # Eq. 6
    return 1.0 / (1.0 + np.exp(-(z @ f64(w.w_out) + float(w.b_out))))
