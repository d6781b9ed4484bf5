"""Seeded, counter-based synthetic input generator (host side, numpy).

This module is shared by the CPU oracle and by the harness that drives the
CUDA library.  It holds none of the beam-search arithmetic: it only turns
(seed, tag, field...) coordinates into reproducible pseudo-random numbers.
A bit-identical CUDA implementation lives in ``workload/gen.cu`` so that very
large inputs (long KV histories) can be produced directly in device memory;
``tests/test_gpu_gen.py`` checks the two agree bit for bit.

Generator definition
--------------------
* Mixing function: the 64-bit finaliser of SplitMix64 (Steele, Lea & Flood,
  "Fast splittable pseudorandom number generators", OOPSLA 2014; Stafford's
  "Mix13" constants).  ``mix64(z)``:
  ``z ^= z >> 30; z *= 0xBF58476D1CE4E5B9; z ^= z >> 27;
  z *= 0x94D049BB133111EB; z ^= z >> 31`` (all mod 2**64).
* Stream key for a coordinate tuple ``(f_0, ..., f_k)``: start from ``h = 0``
  and fold ``h = mix64((h + GAMMA) ^ f_i)`` over the fields, where
  ``GAMMA = 0x9E3779B97F4A7C15`` (the SplitMix64 increment).
* Element ``j`` of a stream is SplitMix64's ``(j+1)``-th output for initial
  state ``key``: ``r_j = mix64(key + (j + 1) * GAMMA)``.
* Approximate N(0,1) from ``r``: the four 16-bit fields of ``r`` are summed
  (Irwin-Hall with n = 4, mean 131070, variance (65536**2 - 1)/3), centred as
  an exact integer, converted exactly to fp32 and multiplied once (fp32,
  round-to-nearest-even) by ``C = fp32(sqrt(3)/65536)`` (bits 0x37DDB3D7).
  Only exactly specified IEEE operations are used, so numpy and CUDA agree.
* Optional fp32 scale: one more fp32 multiply by an exactly representable
  scale (e.g. 1/8) or by a per-row factor.
* Uniform in [0, 1): ``fp32(r >> 40) * 2**-24`` (exact).
* bf16 storage: round-to-nearest-even of the fp32 value (no NaN/Inf occurs).
"""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
M1 = 0xBF58476D1CE4E5B9
M2 = 0x94D049BB133111EB
NORMAL_SCALE_BITS = 0x37DDB3D7
NORMAL_SCALE = np.array([NORMAL_SCALE_BITS], dtype=np.uint32).view(np.float32)[0]
IRWIN_HALL_MEAN = 131070

# Stream tags.  Each input tensor kind draws from its own family of streams.
TAG_KV_K = 1       # K vector written at (layer, writer, position)
TAG_KV_V = 2       # V vector written at (layer, writer, position)
TAG_Q = 3          # query rows of a slot at (layer, slot, position)
TAG_HIDDEN = 4     # probe hidden state of a slot at (slot, position)
TAG_PROBE_W = 5    # probe weight vector
TAG_HEAD_SCALE = 6  # per-KV-head value scale at (layer)

# Writer id used for prompt tokens (shared by every root beam).
PROMPT_WRITER = 0xFFFFFFFF


def mix64_int(z: int) -> int:
    """SplitMix64 finaliser on a Python int (reference for the array form)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * M1) & MASK64
    z = ((z ^ (z >> 27)) * M2) & MASK64
    return z ^ (z >> 31)


def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser, elementwise on a uint64 array (wraps mod 2**64)."""
    z = np.array(z, dtype=np.uint64, ndmin=1)   # arrays wrap silently; scalars would warn
    t = np.empty_like(z)
    np.right_shift(z, np.uint64(30), out=t)
    z ^= t
    z *= np.uint64(M1)
    np.right_shift(z, np.uint64(27), out=t)
    z ^= t
    z *= np.uint64(M2)
    np.right_shift(z, np.uint64(31), out=t)
    z ^= t
    return z


def stream_key(*fields: int) -> int:
    """Fold coordinate fields into one 64-bit stream key."""
    h = 0
    for f in fields:
        h = mix64_int(((h + GAMMA) & MASK64) ^ (int(f) & MASK64))
    return h


def stream_keys(fields: list) -> np.ndarray:
    """Vectorised ``stream_key``: each field is an int or an integer array (broadcast)."""
    arrs = [np.asarray(f).astype(np.uint64) if not isinstance(f, (int, np.integer))
            else np.uint64(int(f) & MASK64) for f in fields]
    shape = np.broadcast_shapes(*[np.shape(a) for a in arrs])
    h = np.zeros(max(1, int(np.prod(shape))), dtype=np.uint64)
    for a in arrs:
        fa = np.broadcast_to(a, shape).reshape(-1) if shape else np.full(1, a, dtype=np.uint64)
        h = mix64((h + np.uint64(GAMMA)) ^ fa)
    return h.reshape(shape)


def raw_bits(keys: np.ndarray, n: int) -> np.ndarray:
    """64 random bits per element: shape keys.shape + (n,)."""
    keys = np.asarray(keys, dtype=np.uint64)
    j = np.arange(1, n + 1, dtype=np.uint64) * np.uint64(GAMMA)
    z = keys.reshape(keys.shape + (1,)) + j
    return mix64(z).reshape(keys.shape + (n,))


def bits_to_normal_f32(r: np.ndarray) -> np.ndarray:
    """Irwin-Hall(4) approximation of N(0,1), exactly specified in fp32."""
    s = ((r & np.uint64(0xFFFF)) + ((r >> np.uint64(16)) & np.uint64(0xFFFF))
         + ((r >> np.uint64(32)) & np.uint64(0xFFFF)) + (r >> np.uint64(48)))
    c = s.astype(np.int64) - IRWIN_HALL_MEAN
    return c.astype(np.float32) * NORMAL_SCALE


def bits_to_uniform_f32(r: np.ndarray) -> np.ndarray:
    """Uniform in [0, 1) with 24 random bits, exact in fp32."""
    return (r >> np.uint64(40)).astype(np.float32) * np.float32(2.0 ** -24)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (round to nearest, ties to even); returns uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to_dtype(x: np.ndarray, dtype: str) -> np.ndarray:
    """Value of ``x`` after storage in ``dtype`` ('f32' or 'bf16'), as fp32."""
    if dtype == "f32":
        return np.asarray(x, dtype=np.float32)
    if dtype == "bf16":
        return bf16_bits_to_f32(f32_to_bf16_bits(x))
    raise ValueError(dtype)


def storage_bits(x: np.ndarray, dtype: str) -> np.ndarray:
    """Raw storage of fp32 values in ``dtype``: float32 array or uint16 bf16 bits."""
    if dtype == "f32":
        return np.ascontiguousarray(x, dtype=np.float32)
    if dtype == "bf16":
        return f32_to_bf16_bits(x)
    raise ValueError(dtype)


def normal(fields: list, n: int, scale: float | None = None) -> np.ndarray:
    """fp32 approx-N(0,1) values: shape broadcast(fields) + (n,).

    ``scale`` (a Python float that must be exactly representable in fp32) is
    applied with a single fp32 multiply.
    """
    x = bits_to_normal_f32(raw_bits(stream_keys(fields), n))
    if scale is not None:
        s = np.float32(scale)
        assert float(s) == scale, "scale must be exact in fp32"
        x = x * s
    return x


def uniform(fields: list, n: int) -> np.ndarray:
    return bits_to_uniform_f32(raw_bits(stream_keys(fields), n))


# ---------------------------------------------------------------------------
# Named input families used by the workloads.
# ---------------------------------------------------------------------------

def head_scales(seed: int, layer: int, num_kv_heads: int, lo: float, hi: float) -> np.ndarray:
    """Per-KV-head value scale U(lo, hi): lo + (hi - lo) * u, two fp32 roundings."""
    u = uniform([seed, TAG_HEAD_SCALE, layer], num_kv_heads)
    return np.float32(lo) + np.float32(hi - lo) * u


def kv_rows(seed: int, which: int, layer: int, writers, positions, num_kv_heads: int,
            head_dim: int, dtype: str, hscale: np.ndarray | None = None) -> np.ndarray:
    """K (which=TAG_KV_K) or V (TAG_KV_V) vectors, fp32 values after storage rounding.

    ``writers`` and ``positions`` broadcast against each other; the result has
    shape broadcast + (num_kv_heads, head_dim).
    """
    w = np.asarray(writers, dtype=np.uint64)
    p = np.asarray(positions, dtype=np.uint64)
    x = normal([seed, which, layer, w, p], num_kv_heads * head_dim)
    x = x.reshape(x.shape[:-1] + (num_kv_heads, head_dim))
    if hscale is not None:
        x = x * np.asarray(hscale, dtype=np.float32)[:, None]
    return round_to_dtype(x, dtype)


def q_rows(seed: int, layer: int, slots, position: int, num_q_heads: int, head_dim: int,
           dtype: str, scale: float | None = None) -> np.ndarray:
    s = np.asarray(slots, dtype=np.uint64)
    x = normal([seed, TAG_Q, layer, s, position], num_q_heads * head_dim, scale)
    return round_to_dtype(x.reshape(x.shape[:-1] + (num_q_heads, head_dim)), dtype)


def hidden_rows(seed: int, slots, position: int, hidden: int, dtype: str) -> np.ndarray:
    s = np.asarray(slots, dtype=np.uint64)
    return round_to_dtype(normal([seed, TAG_HIDDEN, s, position], hidden), dtype)


def probe_weight(seed: int, hidden: int, scale: float) -> np.ndarray:
    return normal([seed, TAG_PROBE_W], hidden, scale)
