"""Pins for oracle.probe: sigmoid probe and the running mean of Algorithm 1."""
import math

import numpy as np

from oracle.probe import probe_score, running_mean_update

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
