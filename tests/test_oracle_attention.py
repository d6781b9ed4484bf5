"""Pins for oracle.attention: closed forms and invariants of softmax attention."""
import numpy as np
import pytest

from oracle.attention import decode_attention, softmax_weights
from oracle import backends

NAMES = {'decode_attention': 'decode_attention', 'softmax_weights': 'softmax_weights'}

@pytest.fixture(autouse=True, params=backends.NAMES)
def oracle_backend(request, monkeypatch):
    """Every pin runs on both oracles: the C++ one and its numpy twin."""
    B = backends.get(request.param)
    monkeypatch.setattr(backends, "DEFAULT", request.param)
    for name, attr in NAMES.items():
        monkeypatch.setitem(globals(), name, getattr(B, attr))
    return B


rng = np.random.default_rng(1)


def rand(*shape):
    return rng.standard_normal(shape).astype(np.float32)


def test_constant_keys_give_mean_of_values():
    L, Hkv, D = 37, 2, 16
    K = np.broadcast_to(rand(1, Hkv, D), (L, Hkv, D)).copy()
    V = rand(L, Hkv, D)
    q = rand(4, D)
    o = decode_attention(q, K, V, 0.7)
    for h in range(4):
        np.testing.assert_allclose(o[h], V[:, h // 2, :].astype(np.float64).mean(0), rtol=1e-12, atol=1e-12)


def test_single_key_gives_its_value():
    K, V, q = rand(1, 1, 8), rand(1, 1, 8), rand(3, 8)
    o = decode_attention(q, K, V, 1.0)
    for h in range(3):
        np.testing.assert_array_equal(o[h], V[0, 0].astype(np.float64))


def test_constant_values_give_that_value():
    L, D = 50, 8
    V = np.broadcast_to(rand(1, 1, D), (L, 1, D)).copy()
    o = decode_attention(rand(2, D), rand(L, 1, D), V, 3.0)
    np.testing.assert_allclose(o, np.broadcast_to(V[0, 0], (2, D)), rtol=1e-12, atol=1e-12)


def test_zero_query_gives_mean_of_values():
    K, V = rand(20, 1, 8), rand(20, 1, 8)
    o = decode_attention(np.zeros((1, 8), np.float32), K, V, 1.0)
    np.testing.assert_allclose(o[0], V[:, 0].astype(np.float64).mean(0), rtol=1e-12, atol=1e-12)


def test_huge_scale_selects_the_argmax_key_not_the_argmin():
    L, D = 30, 8
    K, V, q = rand(L, 1, D), rand(L, 1, D), rand(1, D)
    s = K[:, 0] @ q[0]
    o = decode_attention(q, K, V, 1e4)
    np.testing.assert_allclose(o[0], V[int(np.argmax(s)), 0], rtol=1e-6, atol=1e-6)


def test_two_tokens_closed_form():
    D = 8
    K, V, q = rand(2, 1, D), rand(2, 1, D), rand(1, D)
    scale = 0.3
    s0, s1 = scale * float(K[0, 0] @ q[0].astype(np.float64)), scale * float(K[1, 0] @ q[0].astype(np.float64))
    p0 = 1.0 / (1.0 + np.exp(s1 - s0))
    expect = p0 * V[0, 0] + (1 - p0) * V[1, 0]
    np.testing.assert_allclose(decode_attention(q, K, V, scale)[0], expect, rtol=1e-12, atol=1e-12)


def test_softmax_weights_sum_to_one_and_follow_exp_ratios():
    K, q = rand(100, 16), rand(16)
    p = softmax_weights(q, K, 0.25)
    assert abs(p.sum() - 1.0) < 1e-12
    s = 0.25 * (K.astype(np.float64) @ q.astype(np.float64))
    np.testing.assert_allclose(p[3] / p[7], np.exp(s[3] - s[7]), rtol=1e-10)


def test_gqa_equals_mha_with_replicated_kv():
    L, Hkv, G, D = 40, 3, 4, 16
    K, V, q = rand(L, Hkv, D), rand(L, Hkv, D), rand(Hkv * G, D)
    o_gqa = decode_attention(q, K, V, 0.5)
    o_mha = decode_attention(q, np.repeat(K, G, axis=1), np.repeat(V, G, axis=1), 0.5)
    np.testing.assert_allclose(o_gqa, o_mha, rtol=1e-12, atol=1e-12)
    # Head h reads KV head h // G (not h % Hkv): perturbing KV head 0 changes only heads 0..G-1.
    V2 = V.copy()
    V2[:, 0] += 1.0
    d = np.abs(decode_attention(q, K, V2, 0.5) - o_gqa).max(axis=1)
    assert (d[:G] > 0.5).all() and (d[G:] == 0).all()


def test_token_order_does_not_matter():
    K, V, q = rand(33, 2, 8), rand(33, 2, 8), rand(4, 8)
    perm = rng.permutation(33)
    np.testing.assert_allclose(decode_attention(q, K, V, 1.0), decode_attention(q, K[perm], V[perm], 1.0),
                               rtol=1e-12, atol=1e-12)


def test_scale_moves_between_query_and_scale():
    K, V, q = rand(25, 1, 8), rand(25, 1, 8), rand(1, 8)
    a = decode_attention(q, K, V, 0.5)
    b = decode_attention(q * np.float32(0.5), K, V, 1.0)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


def test_large_logits_do_not_overflow():
    K, V, q = rand(10, 1, 8) * 100, rand(10, 1, 8), rand(1, 8) * 100
    o = decode_attention(q, K, V, 1.0)
    assert np.isfinite(o).all()


@pytest.mark.parametrize("L", [1, 2, 17])
def test_output_is_convex_combination_of_values(L):
    K, V, q = rand(L, 1, 4), rand(L, 1, 4), rand(1, 4)
    o = decode_attention(q, K, V, 1.0)[0]
    assert (o <= V[:, 0].max(0) + 1e-12).all() and (o >= V[:, 0].min(0) - 1e-12).all()
