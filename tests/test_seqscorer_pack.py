"""The sequence scorer's weight buffer layout (gambit.h, gb_scorer_*), packed on the host: every
tensor at its offset in the stated order and type, W_qkv as the q, k, v rows stacked, W_13 as
the W_1 rows then the W_3 rows; a tensor that overflows its slot is refused."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2608_08020_gb300.seqscorer import pack_weights  # noqa: E402
from workload.scorer_weights import seqscorer_weights  # noqa: E402


def _layout(H, d, F, L, Hq, Hkv):
    sizes = [4 * H, 4 * H, 2 * d * H]
    for _ in range(L):
        sizes += [4 * d, 4 * d, 2 * (Hq + 2 * Hkv) * 128 * d, 2 * d * d, 4 * d, 4 * d, 2 * 2 * F * d, 2 * d * F]
    sizes += [4 * d, 4 * d, 4 * d, 4]
    offs, o = [], 0
    for n in sizes:
        offs.append(o)
        o += (n + 255) // 256 * 256
    return offs, o


def _bf16_of(buf, off, shape):
    n = int(np.prod(shape))
    u16 = buf[off:off + 2 * n].view(np.uint16).astype(np.uint32) << 16
    return u16.view(np.float32).reshape(shape)


def _f32_of(buf, off, n):
    return buf[off:off + 4 * n].view(np.float32)


def test_every_tensor_at_its_offset():
    H, F, L, Hq, Hkv = 128, 192, 2, 2, 1
    d = Hq * 128
    w = seqscorer_weights(1, H, d, F, L, Hq, Hkv)
    offs, total = _layout(H, d, F, L, Hq, Hkv)
    buf = pack_weights(w, offs, total)
    assert buf.dtype == np.uint8 and buf.size == total
    np.testing.assert_array_equal(_f32_of(buf, offs[0], H), w["ln_in"][0])
    np.testing.assert_array_equal(_f32_of(buf, offs[1], H), w["ln_in"][1])
    np.testing.assert_array_equal(_bf16_of(buf, offs[2], (d, H)), w["w_in"])      # bf16-exact values
    for l, lw in enumerate(w["layers"]):
        b = 3 + 8 * l
        np.testing.assert_array_equal(_f32_of(buf, offs[b], d), lw["ln1"][0])
        qkv = _bf16_of(buf, offs[b + 2], ((Hq + 2 * Hkv) * 128, d))
        np.testing.assert_array_equal(qkv[:Hq * 128], lw["wq"])
        np.testing.assert_array_equal(qkv[Hq * 128:(Hq + Hkv) * 128], lw["wk"])
        np.testing.assert_array_equal(qkv[(Hq + Hkv) * 128:], lw["wv"])
        np.testing.assert_array_equal(_bf16_of(buf, offs[b + 3], (d, d)), lw["wo"])
        np.testing.assert_array_equal(_f32_of(buf, offs[b + 5], d), lw["ln2"][1])
        w13 = _bf16_of(buf, offs[b + 6], (2 * F, d))
        np.testing.assert_array_equal(w13[:F], lw["w1"])
        np.testing.assert_array_equal(w13[F:], lw["w3"])
        np.testing.assert_array_equal(_bf16_of(buf, offs[b + 7], (d, F)), lw["w2"])
    t = 3 + 8 * L
    np.testing.assert_array_equal(_f32_of(buf, offs[t + 2], d), w["w_out"])
    assert _f32_of(buf, offs[t + 3], 1)[0] == np.float32(w["b_out"])


def test_a_tensor_larger_than_its_slot_is_refused():
    H, F, L, Hq, Hkv = 128, 192, 1, 2, 1
    w = seqscorer_weights(1, H, Hq * 128, F, L, Hq, Hkv)
    offs, total = _layout(H, Hq * 128, F, L, Hq, Hkv)
    offs[3] = offs[2] + 64                                   # W_in's slot cut short
    with pytest.raises(ValueError):
        pack_weights(w, offs, total)
    with pytest.raises(ValueError):
        pack_weights(w, offs[:-1], total)                   # wrong tensor count
