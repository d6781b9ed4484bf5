"""bench.py's host logic for several ranks (one replica per GPU), on CPU with the gloo backend:
the job's time is the slowest rank's on every rank, the whole-job value counts every rank's
beams, each rank runs its own seeded replica, and the reference arm runs on rank 0 only."""
import io
import multiprocessing as mp
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, q) -> None:
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench as b
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        elapsed = b.max_over_ranks(10.0 + 5.0 * rank, world, "cpu")
        wl = b.selected_workload(b.parse_args(["--config", "2"]), rank)
        q.put((rank, elapsed, wl.seed, wl.beams))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_slowest_rank_and_per_rank_replicas(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    slowest = 10.0 + 5.0 * (world - 1)
    assert [e for _, e, _, _ in got] == [slowest] * world          # every rank sees the max
    seeds = [s for _, _, s, _ in got]
    assert len(set(seeds)) == world and seeds[0] == bench.selected_workload(bench.parse_args([]), 0).seed
    assert all(c == 64 for _, _, _, c in got)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5


def test_job_value_counts_every_rank():
    one = bench.job_value(1, 64, 512, 100.0)
    assert one == pytest.approx(64 * 512 / 0.1)
    assert bench.job_value(4, 64, 512, 100.0) == pytest.approx(4 * one)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    called = []
    monkeypatch.setattr(bench, "oracle_sample", lambda *a, **k: called.append(a))
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(bench.parse_args(["--impl", "reference", "--steps", "2", "--warmup", "1"]))
    assert buf.getvalue() == "" and not called
