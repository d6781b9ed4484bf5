"""bench.py's options and host-side choices that need no GPU: the default workload, the scorer
legs, and the layout of its phases (warm-up, end to end, profiled steps, timed window)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from workload.configs import BY_INDEX  # noqa: E402


def test_defaults_and_scorer_options():
    a = bench.parse_args([])
    assert a.config == 5 and a.gpus == 1 and a.probe == "linear" and a.profile_steps == 16 and not a.eager
    assert BY_INDEX[a.config - 1].num_layers == 36          # the largest single-GPU workload
    a = bench.parse_args(["--probe", "seq", "--seq-shape", "3,8,2,2048"])
    assert a.probe == "seq" and [int(x) for x in a.seq_shape.split(",")] == [3, 8, 2, 2048]
    a = bench.parse_args(["--probe", "mlp", "--mlp-hidden", "256"])
    assert a.probe == "mlp" and a.mlp_hidden == 256


def test_one_layer_copy_keeps_the_page_count():
    wl = bench.selected_workload(bench.parse_args(["--config", "5", "--layers", "1"]))
    full = BY_INDEX[4]
    assert wl.num_layers == 1 and wl.pool_pages() == full.pool_pages() == 50862 and wl.pool_bytes is None


@pytest.mark.parametrize("config", [1, 2, 3, 4, 5, 6])
@pytest.mark.parametrize("K,W", [(20, 5), (0, 8), (3, 3)])
def test_timed_window_ends_with_the_round_at_the_full_context(config, K, W):
    wl = BY_INDEX[config - 1]
    K = K or bench.default_steps(wl, W, 16, True, 0)
    lay = bench.step_layout(wl, K, 16, W, with_e2e=True)
    assert lay["timed"] == (wl.context - K, wl.context)
    # every tree workload's context is a round boundary (the unshared one has no tournament)
    assert bench.round_at(wl, wl.context) == (config != 6)
    phases = ["warmup", "e2e", "filler", "profile", "timed"]
    for a, b in zip(phases, phases[1:]):                     # contiguous, in order
        assert lay[a][1] == lay[b][0]
    assert lay["start"] == lay["warmup"][0] >= wl.prompt_len
    assert lay["warmup"][1] - lay["warmup"][0] == W and lay["e2e"][1] - lay["e2e"][0] == K
    assert lay["profile"][1] - lay["profile"][0] == 16
    filler = range(lay["filler"][0] + 1, lay["filler"][1] + 1)
    assert not any(bench.round_at(wl, L) for L in filler)   # no round is left untimed between the windows
    # the end-to-end window also ends at a round wherever one fits below the profiled steps
    if (lay["profile"][0] - wl.prompt_len) // wl.interval >= 1 and lay["e2e"][1] != lay["profile"][0]:
        assert bench.round_at(wl, lay["e2e"][1])


def test_layout_without_end_to_end_steps():
    wl = BY_INDEX[1]
    lay = bench.step_layout(wl, 20, 16, 5, with_e2e=False)
    assert lay["e2e"][0] == lay["e2e"][1] == lay["warmup"][1] == lay["profile"][0]
    assert lay["timed"] == (wl.context - 20, wl.context)
