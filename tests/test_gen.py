"""The seeded input generator: published SplitMix64 outputs, determinism, distribution."""
import json
from pathlib import Path

import numpy as np

from workload import gen


def test_splitmix64_published_outputs():
    g = json.loads((Path(__file__).parent / "golden" / "generator_splitmix64.json").read_text())
    got = [int(x) for x in gen.raw_bits(np.uint64(g["seed"]), len(g["outputs_hex"]))]
    assert got == [int(h, 16) for h in g["outputs_hex"]]


def test_scalar_and_vector_keys_agree():
    ks = gen.stream_keys([7, gen.TAG_KV_K, 3, np.arange(5), 11])
    assert [int(k) for k in ks] == [gen.stream_key(7, gen.TAG_KV_K, 3, i, 11) for i in range(5)]


def test_deterministic_and_distinct_streams():
    a = gen.normal([0, 1, 2], 1000)
    assert np.array_equal(a, gen.normal([0, 1, 2], 1000))
    assert not np.array_equal(a, gen.normal([0, 1, 3], 1000))
    assert not np.array_equal(a, gen.normal([1, 1, 2], 1000))


def test_normal_moments_and_support():
    x = gen.normal([5, 9], 400_000).astype(np.float64)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    assert np.abs(x).max() <= np.sqrt(3.0) * 2 + 1e-6
    assert abs(((x - x.mean()) ** 4).mean() / x.var() ** 2 - 2.7) < 0.1   # Irwin-Hall(4): 3 - 6/20


def test_uniform_range():
    u = gen.uniform([1, 2], 100_000)
    assert u.min() >= 0 and u.max() < 1 and abs(u.mean() - 0.5) < 0.01


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.00390625, 1.005859375, 1.0078125, -2.5, 3.0e-5], np.float32)
    b = gen.f32_to_bf16_bits(x)
    assert list(b[:5]) == [0x3F80, 0x3F80, 0x3F81, 0x3F81, 0xC020]
    back = gen.bf16_bits_to_f32(b)
    assert np.all(np.abs(back - x) <= np.abs(x) * 2.0 ** -8)


def test_exact_scale_and_head_scale():
    x = gen.normal([0, 4], 64)
    assert np.array_equal(gen.normal([0, 4], 64, 0.125), x * np.float32(0.125))
    s = gen.head_scales(0, 0, 8, 0.5, 2.0)
    assert s.dtype == np.float32 and (s >= 0.5).all() and (s < 2.0).all()
