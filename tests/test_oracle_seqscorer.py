"""Pins for oracle.seqscorer (Appendix Eq. 4-6): closed forms of its parts, causality, a
one-step sequence written out without the attention routine, and prefix consistency."""
import math

import numpy as np

from oracle.seqscorer import (SeqScorerWeights, causal_attention, gelu, layer_norm, rope, seq_scores)
from workload.scorer_weights import seqscorer_weights


def _weights(H=128, d=256, F=192, L=2, Hq=2, Hkv=1, seed=0):
    w = seqscorer_weights(seed, H, d, F, L, Hq, Hkv)
    return SeqScorerWeights(w["ln_in"], w["w_in"], w["layers"], w["ln_out"], w["w_out"], w["b_out"], Hq, Hkv)


def test_layer_norm_standardises_then_applies_gain_and_bias():
    x = np.random.default_rng(0).standard_normal((5, 64)) * 3 + 7
    y = layer_norm(x, np.ones(64), np.zeros(64))
    np.testing.assert_allclose(y.mean(axis=1), 0, atol=1e-12)
    np.testing.assert_allclose(y.var(axis=1), 1, atol=1e-4)            # eps 1e-5 against variance 9
    z = layer_norm(x, np.full(64, 2.0), np.full(64, 0.5))
    np.testing.assert_allclose(z, 2 * y + 0.5, atol=1e-12)


def test_gelu_values():
    np.testing.assert_allclose(gelu(np.array([0.0, 1.0, -1.0, 8.0, -8.0])),
                               [0.0, 0.8413447460685429, -0.15865525393145707, 8.0, 0.0], atol=1e-12)


def test_rope_keeps_norms_and_depends_on_relative_position_only():
    rng = np.random.default_rng(1)
    q, k = rng.standard_normal((1, 1, 128)), rng.standard_normal((1, 1, 128))
    np.testing.assert_allclose(rope(q, np.array([0])), q, atol=0)
    np.testing.assert_allclose(np.linalg.norm(rope(q, np.array([9]))), np.linalg.norm(q), rtol=1e-12)
    a = (rope(q, np.array([7])) * rope(k, np.array([3]))).sum()
    b = (rope(q, np.array([107])) * rope(k, np.array([103]))).sum()
    assert abs(a - b) < 1e-9


def test_attention_first_position_returns_its_value_and_is_causal():
    rng = np.random.default_rng(2)
    q, k, v = rng.standard_normal((4, 2, 128)), rng.standard_normal((4, 1, 128)), rng.standard_normal((4, 1, 128))
    o = causal_attention(q, k, v)
    np.testing.assert_allclose(o[0, 0], v[0, 0], atol=1e-12)
    np.testing.assert_allclose(o[0, 1], v[0, 0], atol=1e-12)           # query head 1 reads KV head 0
    v2 = v.copy()
    v2[3] += 5.0
    np.testing.assert_allclose(causal_attention(q, k, v2)[:3], o[:3], atol=0)


def test_one_step_sequence_written_out():
    """T = 1: every head attends to its own value, so the layer is x + Wo [v expanded] + FFN."""
    w = _weights()
    h = np.random.default_rng(3).standard_normal((1, 128))
    x = gelu(layer_norm(h, *w.ln_in) @ w.w_in.astype(np.float64).T)
    for L in w.layers:
        u = layer_norm(x, *L["ln1"])
        v = u @ L["wv"].astype(np.float64).T                              # [1, Hkv * 128]
        o = np.concatenate([v[:, (hq // 2) * 128:(hq // 2 + 1) * 128] for hq in range(2)], axis=1)
        x = x + o @ L["wo"].astype(np.float64).T
        u = layer_norm(x, *L["ln2"])
        g = u @ L["w1"].astype(np.float64).T
        x = x + (g / (1 + np.exp(-g)) * (u @ L["w3"].astype(np.float64).T)) @ L["w2"].astype(np.float64).T
    y = 1 / (1 + math.exp(-(layer_norm(x, *w.ln_out) @ w.w_out.astype(np.float64) + w.b_out)[0]))
    np.testing.assert_allclose(seq_scores(h, w), [y], atol=1e-12)


def test_scores_are_causal_and_prefix_consistent():
    w = _weights()
    hs = np.random.default_rng(4).standard_normal((6, 128))
    y = seq_scores(hs, w)
    hs2 = hs.copy()
    hs2[3:] = np.random.default_rng(5).standard_normal((3, 128))        # a child that branched after step 3
    y2 = seq_scores(hs2, w)
    np.testing.assert_allclose(y2[:3], y[:3], atol=1e-13)
    assert np.all((y > 0) & (y < 1)) and abs(y2[5] - y[5]) > 1e-6
