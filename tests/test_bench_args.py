"""bench.py's options and host-side choices that need no GPU: the scorer legs and which timed
steps carry kernel events."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_defaults_and_scorer_options():
    a = bench.parse_args([])
    assert a.config == 2 and a.gpus == 1 and a.probe == "linear" and a.event_stride == 0 and not a.eager
    a = bench.parse_args(["--probe", "seq", "--seq-shape", "3,8,2,2048"])
    assert a.probe == "seq" and [int(x) for x in a.seq_shape.split(",")] == [3, 8, 2, 2048]
    a = bench.parse_args(["--probe", "mlp", "--mlp-hidden", "256"])
    assert a.probe == "mlp" and a.mlp_hidden == 256


def test_about_32_bracketed_steps_by_default():
    for K in (64, 512, 1024, 2048):
        stride, steps = bench.bracketed_steps(8, K, 0, False)
        assert stride == K // 32 and len(steps) == 32
        assert steps[0] == 8 and all(b - a == stride for a, b in zip(steps, steps[1:]))
    assert bench.bracketed_steps(3, 10, 0, False) == (1, list(range(3, 13)))   # fewer than 32 steps: all
    assert bench.bracketed_steps(3, 100, 7, False)[1] == list(range(3, 103, 7))
    assert bench.bracketed_steps(3, 100, 7, True) == (1, list(range(3, 103)))  # --breakdown: every step
