"""Pins for oracle.probe: sigmoid probe and the running mean of Algorithm 1."""
import math

import numpy as np
import pytest

from oracle.probe import probe_score, running_mean_update
from oracle import backends

NAMES = {'probe_score': 'probe_score', 'running_mean_update': 'running_mean_update'}

@pytest.fixture(autouse=True, params=backends.NAMES)
def oracle_backend(request, monkeypatch):
    """Every pin runs on both oracles: the C++ one and its numpy twin."""
    B = backends.get(request.param)
    monkeypatch.setattr(backends, "DEFAULT", request.param)
    for name, attr in NAMES.items():
        monkeypatch.setitem(globals(), name, getattr(B, attr))
    return B


rng = np.random.default_rng(2)


def test_zero_weight_zero_bias_is_one_half():
    assert probe_score(rng.standard_normal(64), np.zeros(64), 0.0) == 0.5


def test_unit_vector_picks_one_weight():
    w = rng.standard_normal(32)
    for i in (0, 5, 31):
        h = np.zeros(32)
        h[i] = 1.0
        assert abs(probe_score(h, w, 0.25) - 1 / (1 + math.exp(-(w[i] + 0.25)))) < 1e-15


def test_log_three_gives_three_quarters():
    h = np.zeros(8)
    h[0] = 1.0
    w = np.zeros(8)
    w[0] = math.log(3.0)
    assert abs(probe_score(h, w, 0.0) - 0.75) < 1e-15


def test_bias_sign_and_symmetry():
    h, w = rng.standard_normal(16), rng.standard_normal(16)
    assert abs(probe_score(h, w, 0.3) + probe_score(-h, w, -0.3) - 1.0) < 1e-14
    assert probe_score(h, w, 1.0) > probe_score(h, w, 0.0)


def test_batched_rows():
    h, w = rng.standard_normal((5, 16)), rng.standard_normal(16)
    s = probe_score(h, w, 0.1)
    for i in range(5):
        assert abs(s[i] - probe_score(h[i], w, 0.1)) < 1e-15


def test_running_mean_worked_example():
    # scores 0.2, 0.4, 0.9 -> means 0.2, 0.3, 0.5
    m, n = np.float32(0.0), 0
    expect = [0.2, 0.3, 0.5]
    for x, e in zip([0.2, 0.4, 0.9], expect):
        m, n = running_mean_update(m, n, np.float32(x))
        assert abs(float(m) - e) < 1e-7
    assert n == 3


def test_first_update_is_the_score_exactly():
    x = np.float32(0.123456789)
    m, n = running_mean_update(np.float32(0.0), 0, x)
    assert m == x and n == 1


def test_constant_scores_leave_mean_exact():
    x = np.float32(0.7312)
    m, n = np.float32(0.0), 0
    for _ in range(50):
        m, n = running_mean_update(m, n, x)
        assert m == x


def test_incremental_mean_equals_average_within_n_ulp():
    xs = rng.random(200).astype(np.float32)
    m, n = np.float32(0.0), 0
    for k, x in enumerate(xs, 1):
        m, n = running_mean_update(m, n, x)
        exact = float(np.mean(xs[:k].astype(np.float64)))
        assert abs(float(m) - exact) <= k * float(np.spacing(np.float32(1.0)))
    assert n == 200


def test_update_rounds_each_operation_in_fp32():
    m, n, x = np.float32(0.1), 2, np.float32(0.9)
    d = np.float32(x - m)
    q = np.float32(d / np.float32(3))
    assert running_mean_update(m, n, x)[0] == np.float32(m + q)


# -- the two-layer MLP scorer ------------------------------------------------------
def test_mlp_with_zero_first_layer_is_a_constant():
    from oracle.probe import mlp_probe_score
    rng = np.random.default_rng(0)
    h = rng.standard_normal((5, 64))
    b1 = np.array([0.5, -2.0, 1.5])
    w2 = np.array([2.0, 7.0, -1.0])
    got = mlp_probe_score(h, np.zeros((3, 64)), b1, w2, 0.25)
    want = 1.0 / (1.0 + np.exp(-(0.5 * 2.0 + 0.0 * 7.0 + 1.5 * -1.0 + 0.25)))   # relu(-2) = 0
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-15)


def test_mlp_reduces_to_the_linear_probe():
    """d_h = 1, a bias large enough that relu is the identity, and an output bias that
    cancels it: sigma(w.h) exactly as the linear probe."""
    from oracle.probe import mlp_probe_score, probe_score
    rng = np.random.default_rng(1)
    h = rng.standard_normal((7, 128))
    w = rng.standard_normal(128) / 8
    big = 1000.0
    got = mlp_probe_score(h, w[None, :], np.array([big]), np.array([1.0]), -big)
    np.testing.assert_allclose(got, probe_score(h, w, 0.0), rtol=0, atol=1e-12)


def test_mlp_relu_pair_gives_the_absolute_value():
    """Rows w and -w with unit output weights: relu(x) + relu(-x) = |x|."""
    from oracle.probe import mlp_probe_score
    rng = np.random.default_rng(2)
    h = rng.standard_normal((9, 96))
    w = rng.standard_normal(96) / 10
    got = mlp_probe_score(h, np.stack([w, -w]), np.zeros(2), np.ones(2), -0.5)
    want = 1.0 / (1.0 + np.exp(-(np.abs(h @ w) - 0.5)))
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
