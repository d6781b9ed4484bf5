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


# ---- The composition of Eq. 4-6, pinned by hand-built weights -------------------------------
# A LayerNorm with gain 0 outputs its bias whatever its input, so a layer whose norms have gain 0
# feeds chosen constant vectors to the attention and the FFN, and each term of the composition
# can be computed by hand.  A swapped gate/up pair, a post-norm layer, a misplaced or transposed
# W_o, or a head that skips its LayerNorm changes the printed numbers below.

def _hand_model(d=128, F=2, H=64):
    """One layer, one query and one key/value head (d = 128); every norm has gain 0 and bias 0,
    every matrix is zero: the caller fills in the parts under test."""
    z = lambda *s: np.zeros(s)
    layer = {"ln1": (z(d), z(d)), "wq": z(128, d), "wk": z(128, d), "wv": z(128, d), "wo": z(d, 128),
             "ln2": (z(d), z(d)), "w1": z(F, d), "w3": z(F, d), "w2": z(d, F)}
    return SeqScorerWeights((z(H), z(H)), z(d, H), [layer], (np.ones(d), z(d)), z(d), 0.0, 1, 1)


def _ln_coord(x, i):
    """Coordinate i of LayerNorm(x) with gain 1 and bias 0, eps 1e-5, for a vector given by hand."""
    mu = sum(x) / len(x)
    var = sum((e - mu) ** 2 for e in x) / len(x)
    return (x[i] - mu) / math.sqrt(var + 1e-5)


def test_head_with_zero_gain_gives_sigmoid_of_the_output_bias():
    w = _weights()
    w.ln_out = (np.zeros_like(w.ln_out[0]), np.zeros_like(w.ln_out[1]))
    w.b_out = 0.75
    hs = np.random.default_rng(6).standard_normal((4, 128))
    np.testing.assert_allclose(seq_scores(hs, w), np.full(4, 1 / (1 + math.exp(-0.75))), atol=1e-15)


def test_ffn_with_zero_up_projection_adds_nothing():
    """W_3 = 0 makes SiLU(W_1 u) * (W_3 u) zero, so the model equals the one without the FFN (W_2 = 0)."""
    w = _weights()
    hs = np.random.default_rng(7).standard_normal((5, 128))
    for L in w.layers:
        L["w3"] = np.zeros_like(L["w3"])
    y = seq_scores(hs, w)
    for L in w.layers:
        L["w2"] = np.zeros_like(L["w2"])
    np.testing.assert_allclose(seq_scores(hs, w), y, atol=0)


def test_swiglu_gate_and_up_order_by_hand():
    """LN2 outputs e_0; W_1 e_0 = (40, 40) (SiLU(40) = 40 in fp64), W_3 e_0 = (-1, 2), W_2 the identity
    onto coordinates 0 and 1: the layer writes (-40, 80) into a zero stream.  A swapped gate gives
    (SiLU(-1) * 40, SiLU(2) * 40) = (-10.76, 70.46) instead."""
    w = _hand_model()
    L = w.layers[0]
    L["ln2"] = (np.zeros(128), np.eye(128)[0])
    L["w1"][:, 0] = [40.0, 40.0]
    L["w3"][:, 0] = [-1.0, 2.0]
    L["w2"][0, 0] = L["w2"][1, 1] = 1.0
    w.w_out[0] = 1.0
    x = [-40.0, 80.0] + [0.0] * 126
    y = 1 / (1 + math.exp(-_ln_coord(x, 0)))
    assert abs(_ln_coord(x, 0) + 5.1031) < 1e-3                      # -40.3125 / sqrt(62.4024 + 1e-5)
    for T in (1, 3):
        np.testing.assert_allclose(seq_scores(np.ones((T, 64)), w), np.full(T, y), atol=1e-12)
    w.w_out[0], w.w_out[1] = 0.0, 1.0
    y1 = 1 / (1 + math.exp(-_ln_coord(x, 1)))
    np.testing.assert_allclose(seq_scores(np.ones((2, 64)), w), np.full(2, y1), atol=1e-12)


def test_attention_output_goes_through_w_o_before_the_residual():
    """LN1 outputs e_0 at every position, so q, k and v are the same at every position and the
    attention returns v = W_v e_0 = 3 e_0 whatever the softmax weights; W_o = 2 (e_5 e_0^T) moves it
    to coordinate 5, and the residual stream (x_0 = GELU(W_in 0) = 0) ends as 6 e_5.  A transposed W_o
    leaves the stream zero (score 1/2)."""
    w = _hand_model()
    L = w.layers[0]
    L["ln1"] = (np.zeros(128), np.eye(128)[0])
    L["wq"][0, 0] = L["wk"][0, 0] = 1.0
    L["wv"][0, 0] = 3.0
    L["wo"][5, 0] = 2.0
    w.w_out[5] = 1.0
    x = [0.0] * 128
    x[5] = 6.0
    y = 1 / (1 + math.exp(-_ln_coord(x, 5)))
    assert abs(_ln_coord(x, 5) - 11.2694) < 1e-3                     # (6 - 6/128) / sqrt(var + 1e-5)
    hs = np.random.default_rng(8).standard_normal((4, 64))
    np.testing.assert_allclose(seq_scores(hs, w), np.full(4, y), atol=1e-12)


def test_input_projection_is_gelu_of_w_in_after_layer_norm():
    """The stream starts as GELU(W_in LN_in(h)) (Eq. 4): LN_in with gain 0 and bias e_2 gives
    x_0 = GELU(W_in e_2); W_in e_2 = (1, -1, 0, ...) gives x_0 = (GELU(1), GELU(-1), 0, ...) =
    (0.8413, -0.1587, 0, ...), and an empty layer passes it to the head."""
    w = _hand_model()
    w.ln_in = (np.zeros(64), np.eye(64)[2])
    w.w_in[0, 2], w.w_in[1, 2] = 1.0, -1.0
    w.w_out[1] = 1.0
    x = [0.8413447460685429, -0.15865525393145707] + [0.0] * 126
    y = 1 / (1 + math.exp(-_ln_coord(x, 1)))
    np.testing.assert_allclose(seq_scores(np.random.default_rng(9).standard_normal((3, 64)), w), np.full(3, y),
                               atol=1e-12)
