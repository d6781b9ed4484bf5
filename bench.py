"""Benchmark of the beam-decode hot path of thought-level beam search on GB300.

The method's schedule: every decode step appends one token to every active
beam and attends over its context (page reservation + KV append, then one
attention launch per layer: grouped shared-prefix attention, per-beam split-KV
attention over the unshared tails, and the merge of their partial results);
every Delta tokens the probe scores every beam and one tournament round prunes
and branches (rank, fork block tables, free pages, rebuild shared-prefix
segments, in one launch).  The timed window is K decode steps that end at the
workload's full context with the round there, so every row of the hot path
runs in it and the beam tree is the one the schedule produces.

Default workload: 36 Qwen3-8B-shaped layers (32/8 heads, head dim 128, bf16
KV, 16-token pages) in a fixed 120 GB pool, 198 beams forked from one prompt
by real rounds (keep 50%, branch x2) up to 8192 tokens; ``--config`` picks
the others (1 tiny fp32, 2 one layer with 64 beams at 4096, 3 512 beams at
16384, 4 256 beams at 32768 with 32-token pages, 6 unshared traces).  Inputs
are seeded synthetic data generated on the device before the timed region.
The KV a step attends over is far larger than L2, so no flush is needed
between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config I]

N > 1 runs under torchrun: every rank runs an independent problem (its own
pool, seed + rank); nothing is exchanged (replicas), value = all ranks'
beam-tokens / max-over-ranks time.  ``--impl reference`` times the CPU
oracle (the only baseline this method has) on a bounded sample.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0,
                    help="timed decode steps (0: one tournament interval, or 64 where those inputs would not fit)")
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=5, choices=range(1, 7),
                    help="workload index 1..6 (default 5: the 36-layer memory-capped step, the largest "
                         "single-GPU workload; 6: independent roots with no shared KV)")
    ap.add_argument("--flags", choices=["auto", "per_beam"], default="auto")
    ap.add_argument("--group-min", type=int, default=0, help="beams a segment needs for the grouped path (0: library default, 2)")
    ap.add_argument("--cpu-steps", type=int, default=0,
                    help="steps of the oracle sample for cpu_baseline (0: 200 layer-steps, i.e. 200 / layers)")
    ap.add_argument("--cpu-beams", type=int, default=16, help="beams per step in the oracle sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--beams", type=int, default=0, help="override the workload's beam count (smaller profiling cases)")
    ap.add_argument("--context", type=int, default=0, help="override the workload's context length")
    ap.add_argument("--layers", type=int, default=0,
                    help="override the layer count, keeping the pool's page count (a one-layer copy of the "
                         "36-layer workload has the same tree and the same per-layer kernels)")
    ap.add_argument("--probe", choices=["linear", "mlp", "seq"], default="linear",
                    help="scorer at the tournament points: the linear probe of the workloads, the two-layer MLP, "
                         "or the history-aware sequence scorer")
    ap.add_argument("--mlp-hidden", type=int, default=512, help="hidden width of the two-layer MLP scorer")
    ap.add_argument("--seq-shape", default="2,4,2,1024",
                    help="sequence scorer layers,q-heads,kv-heads,ffn (128-dim heads; d_model = q-heads x 128)")
    ap.add_argument("--breakdown", action="store_true",
                    help="also time the planner, append and (fp32 pools) combine kernels in the profiled steps")
    ap.add_argument("--profile-steps", type=int, default=16,
                    help="steps before the timed window whose kernels the library brackets with CUDA events")
    ap.add_argument("--no-capacity", action="store_true", help="skip the memory-capped workload's capacity search")
    ap.add_argument("--eager", action="store_true",
                    help="launch the timed steps one by one instead of as one captured CUDA graph")
    return ap.parse_args(argv)


def selected_workload(args, rank: int = 0):
    from workload.configs import BY_INDEX
    wl = BY_INDEX[args.config - 1]
    over = {"seed": wl.seed + rank}
    if args.beams:
        over["beams"] = args.beams
        over["K"] = max(1, round(wl.K * args.beams / wl.beams))
    if args.context:
        over["context"] = args.context
    if args.layers and args.layers != wl.num_layers:
        over["num_layers"] = args.layers
        over["num_pages"] = wl.pool_pages()       # the same page count, so the same tree
        over["pool_bytes"] = None
    wl = dataclasses.replace(wl, **over)
    if args.beams or args.context or args.layers:
        wl = dataclasses.replace(wl, name=f"{wl.name}[beams={wl.beams},context={wl.context},layers={wl.num_layers}]")
    return wl


INPUT_BUDGET_BYTES = 16 * 2**30  # device memory for the pre-generated step inputs


def round_at(wl, L: int) -> bool:
    """A probe + tournament round follows the decode step that brings the context to L."""
    return L > wl.prompt_len and (L - wl.prompt_len) % wl.interval == 0


def default_steps(wl, W: int, Kp: int, with_e2e: bool, step_input_bytes: int) -> int:
    """Timed steps when --steps is 0: a tournament interval, at most 512 steps, 64 where the
    pre-generated inputs of more would not fit beside the pool, and fewer where the phases
    would not fit between the prompt and the context."""
    K = min(wl.interval, 512)
    if step_input_bytes * K > INPUT_BUDGET_BYTES:
        K = 64
    while K > 1:
        try:
            step_layout(wl, K, Kp, W, with_e2e)
            return K
        except SystemExit:
            K //= 2
    return K


def step_layout(wl, K: int, Kp: int, W: int, with_e2e: bool) -> dict:
    """Context lengths bounding each phase of the run, as (first, last) contexts of its steps
    (a phase of n steps takes the context from first to first + n).  The timed window is the
    last K steps: it ends at the workload's full context, where the schedule runs a probe +
    tournament round, so the window holds every row of the hot path whatever K is.  Before it,
    Kp profiled steps (kernels bracketed by events), and before those the K end-to-end steps,
    which end at the last round boundary below the profiled steps when there is room (so they
    hold a round too); untimed filler steps bridge the gap.  W warm-up steps come first."""
    ctx, P0, delta = wl.context, wl.prompt_len, wl.interval
    value = (ctx - K, ctx)
    prof = (value[0] - Kp, value[0])
    if with_e2e:
        n = (prof[0] - P0) // delta
        Re = P0 + n * delta if n >= 1 else None
        if Re is None or Re - K - W < P0:
            Re = prof[0]
        e2e = (Re - K, Re)
    else:
        e2e = (prof[0], prof[0])
    warm = (e2e[0] - W, e2e[0])
    if warm[0] < P0:
        raise SystemExit(f"{wl.name}: {W} warm-up + {K if with_e2e else 0} end-to-end + {Kp} profiled + {K} timed "
                         f"steps do not fit between the prompt ({P0}) and the context ({ctx})")
    return {"start": warm[0], "warmup": warm, "e2e": e2e, "filler": (e2e[1], prof[0]), "profile": prof,
            "timed": value}


# ---------------------------------------------------------------------------
# Clock sampling (nvidia-smi) during the timed region.
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.05)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.05)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        rows = []
        with open(self.file.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.file.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        pw = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None, "reasons": reasons, "samples": len(rows)}


def gpu_id_for_smi(local: int) -> str:
    """nvidia-smi -i accepts a UUID, which stays right whatever CUDA_VISIBLE_DEVICES maps."""
    import torch
    try:
        u = str(torch.cuda.get_device_properties(local).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        return vis.split(",")[local] if vis else str(local)


def captured_traffic(kernel: str, workload: str, path: str, bytes_per_launch: float):
    """DRAM bytes per launch from a committed ncu capture (profiles/traffic.json): a record of this
    kernel (or kernel pair), workload and path, whose kernel sources are unchanged since the
    capture and whose launch did the same algorithmic work (within 3%); None otherwise."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            records = json.load(f)["records"]
    except (OSError, KeyError, ValueError):
        return None
    for rec in records:
        try:
            if rec["kernel"] != kernel or rec["workload"] != workload or rec["path"] != path:
                continue
            if any(hashlib.sha256(open(os.path.join(ROOT, src), "rb").read()).hexdigest() != sha
                   for src, sha in rec["sources"].items()):
                continue
            alg = rec["algorithmic_bytes_per_launch"]
            if bytes_per_launch and abs(alg - bytes_per_launch) <= 0.03 * bytes_per_launch:
                return rec["dram_bytes_per_launch"]
        except (OSError, KeyError, TypeError):
            continue
    return None


def measured_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


# ---------------------------------------------------------------------------
# Oracle sample on host cores (cpu_baseline leg and the reference arm).
# ---------------------------------------------------------------------------
def _oracle_worker(wl_dict, slot_hist, positions, barrier, out_q):
    """Spawned process: for each layer, materialise its beams' KV (untimed), then time fp64 decode
    attention of every step; reports the timed seconds summed over layers."""
    from oracle import backends
    from oracle.beams import kv_from_history
    from workload import gen
    from workload.configs import Workload
    wl = Workload(**wl_dict)
    decode_attention = backends.get().decode_attention
    hscale = [gen.head_scales(wl.seed, l, wl.num_kv_heads, *wl.head_scale) for l in range(wl.num_layers)] \
        if wl.head_scale else None
    barrier.wait()
    timed = 0.0
    for l in range(wl.num_layers):
        kv = {s: kv_from_history(h, wl.seed, l, wl.num_kv_heads, wl.head_dim, wl.kv_dtype,
                                 hscale[l] if hscale else None) for s, h in slot_hist}
        t0 = time.perf_counter()
        for pos in positions:
            for s, _ in slot_hist:
                K, V = kv[s]
                q = gen.q_rows(wl.seed, l, s, pos, wl.num_q_heads, wl.head_dim, wl.kv_dtype, wl.q_scale)
                decode_attention(q, K, V, wl.attn_scale)
        timed += time.perf_counter() - t0
        del kv
    out_q.put((timed, len(positions) * len(slot_hist)))


def oracle_sample(wl, steps: int, sample_beams: int, workers: int | None = None) -> dict:
    """Time the CPU oracle on a bounded sample of the workload (host cores, spawn processes)."""
    import multiprocessing as mp

    import numpy as np

    from oracle.trajectory import OracleRun
    workers = workers or max(1, min(os.cpu_count() or 1, sample_beams))
    run = OracleRun(wl, literal_kv=False)
    run.build(upto=wl.context)
    L = run.pos
    sample = list(range(min(sample_beams, wl.beams)))
    chunks = [sample[i::workers] for i in range(workers)]
    chunks = [c for c in chunks if c]
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    ctx = mp.get_context("spawn")
    barrier = ctx.Barrier(len(chunks) + 1)
    out_q = ctx.Queue()
    positions = [L] * steps
    procs = []
    for c in chunks:
        p = ctx.Process(target=_oracle_worker, args=(dataclasses.asdict(wl), [(s, run.pool.history[s]) for s in c],
                                                     positions, barrier, out_q))
        p.start()
        procs.append(p)
    barrier.wait()
    results = [out_q.get() for _ in chunks]
    t_attn = max(t for t, _ in results)  # the workers run side by side, one per core
    for p in procs:
        p.join()
    # The tournament part of the schedule: one probe over all beams and one tournament round
    # every delta steps, timed once on the oracle pool and charged at that rate.
    t1 = time.perf_counter()
    run.probe()
    run.prune()
    t_round = time.perf_counter() - t1
    beams_done = sum(n for _, n in results)
    total = t_attn + t_round * steps / wl.interval
    return {"value": beams_done / total, "unit": "beam-tokens/s", "cores": len(chunks), "kind": "oracle",
            "seconds": round(total, 3), "wall_seconds": round(t_attn + t_round, 3),
            "sample": (f"{steps} steps x {len(sample)} of {wl.beams} beams: the C++ oracle's fp64 two-pass decode "
                       f"attention over all {wl.num_layers} layer(s) at "
                       f"L={L} over {len(chunks)} single-threaded spawn processes, plus the fp64 probe over all "
                       f"{wl.beams} beams and one tournament round on the oracle pool every {wl.interval} steps")}


# ---------------------------------------------------------------------------
# Several ranks (one replica per GPU): the job's time is the slowest rank's.
# ---------------------------------------------------------------------------
def max_over_ranks(x: float, world: int, device) -> float:
    """The largest of every rank's x, returned on every rank (x itself for one rank)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world: int, beams: int, steps: int, elapsed_ms: float) -> float:
    """Whole-job beam-tokens/s: every rank decodes `steps` tokens for its `beams` beams."""
    return world * beams * steps / (elapsed_ms / 1e3)


# ---------------------------------------------------------------------------
# Our arm.
# ---------------------------------------------------------------------------


def capacity_search(wl, dev) -> dict:
    """Beams of the workload's full context that a fixed pool holds: with every prefix copied
    (each beam owns all its pages) and with the method's forks sharing prefixes.  The forked
    count is found by running the whole schedule (seed 0: probe scores, tournaments, forks) in
    a pool of the same page count for growing beam counts; pages cover all layers, so one layer
    decides whether a tree fits."""
    import torch

    from workload.driver import GpuRun
    pages = wl.pool_pages()
    copied = pages // wl.pages_per_beam

    def fits(c: int) -> bool:
        w1 = dataclasses.replace(wl, num_layers=1, beams=c, K=max(1, round(wl.K * c / wl.beams)), pool_bytes=None,
                                 num_pages=pages)
        g = GpuRun(w1, device_gen=True, device=str(dev))
        g.build(upto=wl.context, final_round=True)
        ok = g.pool.status() == 0
        del g
        torch.cuda.empty_cache()
        return ok

    lo = wl.beams if fits(wl.beams) else 0   # the configured count (the worst-case bound) must fit
    hi = 1024                                # the library's slot limit
    if lo and fits(hi):
        lo = hi
    while hi - lo > 1 and lo:
        mid = (lo + hi) // 2
        if fits(mid):
            lo = mid
        else:
            hi = mid
    return {"pool_pages": pages, "pool_bytes": wl.pool_bytes, "copied_beams": copied,
            "forked_beams_configured": wl.beams, "forked_beams_configured_fit": lo >= wl.beams,
            "forked_beams_max_seed0": lo}
class _Cudart:
    """The CUDA runtime calls the end-to-end leg issues per step (copies between pinned host
    memory and the device, events between the compute and copy streams), called directly:
    from Python they cost a fraction of the equivalent torch calls."""
    H2D, D2H = 1, 2

    def __init__(self):
        import ctypes
        import ctypes.util
        lib = None
        for name in ("libcudart.so.13", "libcudart.so.12", ctypes.util.find_library("cudart") or "libcudart.so"):
            try:
                lib = ctypes.CDLL(name)
                break
            except OSError:
                continue
        if lib is None:
            raise RuntimeError("the CUDA runtime library is not loadable")
        P, Z, I, U = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_uint
        self._ct = ctypes
        self._copy = lib.cudaMemcpyAsync
        self._copy.argtypes = [P, P, Z, I, P]
        self._rec = lib.cudaEventRecord
        self._rec.argtypes = [P, P]
        self._wait = lib.cudaStreamWaitEvent
        self._wait.argtypes = [P, P, U]
        self._create = lib.cudaEventCreateWithFlags
        self._create.argtypes = [P, U]
        self._destroy = lib.cudaEventDestroy
        self._destroy.argtypes = [P]

    @staticmethod
    def _ok(code, what):
        if code != 0:
            raise RuntimeError(f"{what} failed with CUDA error {code}")

    def event(self):
        e = self._ct.c_void_p()
        self._ok(self._create(self._ct.byref(e), 2), "cudaEventCreateWithFlags")  # cudaEventDisableTiming
        return e.value

    def destroy(self, e):
        self._destroy(e)

    def copy(self, dst, src, n, kind, stream):
        self._ok(self._copy(dst, src, n, kind, stream), "cudaMemcpyAsync")

    def record(self, e, stream):
        self._ok(self._rec(e, stream), "cudaEventRecord")

    def wait(self, stream, e):
        self._ok(self._wait(stream, e, 0), "cudaStreamWaitEvent")


def build_seq_scorer(args, wl, g, dev, n_rounds_after: int):
    """The sequence scorer with seeded random weights and its step pool, seeded with the
    prompt's final hidden state and stepped once per tournament round already in the tree
    (hidden states of those rounds; no forks replayed, so every trace holds that many
    positions).  Returns the SeqScorer with ``history`` = positions per trace."""
    from paper_2608_08020_gb300.seqscorer import SeqScorer
    from workload import gen, gpu_gen
    from workload.scorer_weights import seqscorer_weights
    import torch
    if wl.hidden_dtype != "bf16" or wl.hidden % 64:
        raise SystemExit("--probe seq needs bf16 hidden states of a multiple of 64")
    n_layers, hq, hkv, ffn = (int(x) for x in args.seq_shape.split(","))
    w = seqscorer_weights(wl.seed + 2, wl.hidden, hq * 128, ffn, n_layers, hq, hkv)
    done = [L for L in wl.rounds() if L <= g.pos]
    sc = SeqScorer(w, hidden_dim=wl.hidden, ffn_dim=ffn, max_beams=wl.beams,
                   max_steps=len(done) + n_rounds_after + 2, device=dev)
    h = torch.empty(wl.beams, wl.hidden, dtype=torch.bfloat16, device=dev)
    gpu_gen.normal(h, "bf16", 1, wl.beams, wl.hidden, [wl.seed, gen.TAG_HIDDEN, (0, 0, 1), wl.prompt_len])
    sc.seed(h[0].contiguous(), wl.beams)
    score = torch.empty(wl.beams, dtype=torch.float32, device=dev)
    for L in done:
        gpu_gen.normal(h, "bf16", 1, wl.beams, wl.hidden, [wl.seed, gen.TAG_HIDDEN, (0, 0, 1), L])
        sc.step(h, score)
    sc.history = 1 + len(done)
    return sc


def run_ours(args) -> None:
    import torch
    import torch.distributed as dist

    from paper_2608_08020_gb300 import binding as B
    from workload import gen, gpu_gen
    from workload.driver import GpuRun

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    wl = selected_workload(args, rank)
    flags = B.GB_PATH_AUTO if args.flags == "auto" else B.GB_PATH_PER_BEAM
    W = args.warmup
    C, Hq, Hkv, D, NL = wl.beams, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.num_layers
    esz_in = 2 if wl.kv_dtype == "bf16" else 4
    step_input_bytes = NL * C * (Hq + 2 * Hkv) * D * esz_in
    Kp = max(1, args.profile_steps)
    with_e2e = not args.no_e2e
    K = args.steps if args.steps > 0 else default_steps(wl, W, Kp, with_e2e, step_input_bytes)
    lay = step_layout(wl, K, Kp, W, with_e2e)
    delta = wl.interval

    # Every phase ends at or before the workload's context, so the pool needs tables of that length.
    fixed_pool = wl.pool_bytes is not None
    g = GpuRun(wl, device_gen=True, device=str(dev), max_context=wl.context + 1, group_min_beams=args.group_min)
    t_build = time.perf_counter()
    g.build(upto=lay["start"])               # the schedule's rounds up to here, then plain appends
    torch.cuda.synchronize()
    t_build = time.perf_counter() - t_build
    pos0 = g.pos                             # context before the first (warm-up) step
    assert pos0 == lay["start"]
    S = wl.context - pos0                    # steps from here to the full context

    def is_round(i: int) -> bool:            # step i brings the context to pos0 + i + 1
        return round_at(wl, pos0 + i + 1)

    def steps_of(phase: str) -> range:
        first, last = lay[phase]
        return range(first - pos0, last - pos0)

    # Step inputs (q, k, v of every layer) for K steps, generated on the device before any timing;
    # every phase cycles through them (timing does not depend on their values).  The hidden states
    # at each round are the seeded ones of that position, so the tree is the schedule's.
    qs = torch.empty(K, NL, C, Hq, D, dtype=g.tdt, device=dev)
    ks = torch.empty(K, NL, C, Hkv, D, dtype=g.tdt, device=dev)
    vs = torch.empty_like(ks)
    for j in range(K):
        pos = lay["timed"][0] + j
        for l in range(NL):
            gpu_gen.normal(qs[j, l], wl.kv_dtype, 1, C, Hq * D, [wl.seed, gen.TAG_Q, l, (0, 0, 1), pos],
                           scale=wl.q_scale if wl.q_scale is not None else 1.0)
            for which, dst in ((gen.TAG_KV_K, ks), (gen.TAG_KV_V, vs)):
                gpu_gen.normal(dst[j, l], wl.kv_dtype, 1, C, Hkv * D, [wl.seed, which, l, (0, 0, 1), pos],
                               row_scale=g.hscale_dev[l] if g.hscale else None, row_scale_div=D)
    round_steps = [i for i in range(S) if is_round(i)]
    hs = torch.empty(max(1, len(round_steps)), C, wl.hidden, dtype=g.hidden.dtype, device=dev)
    h_index = {s: n for n, s in enumerate(round_steps)}
    for s_, n in h_index.items():
        gpu_gen.normal(hs[n], wl.hidden_dtype, 1, C, wl.hidden, [wl.seed, gen.TAG_HIDDEN, (0, 0, 1), pos0 + s_ + 1])
    out = torch.empty(NL, C, Hq, D, dtype=torch.float32, device=dev)
    pool = g.pool
    mlp = None
    if args.probe == "mlp":       # the two-layer MLP scorer, seeded random weights (no trained scorer here)
        if wl.hidden_dtype != "bf16" or wl.hidden % 64:
            raise SystemExit("--probe mlp needs bf16 hidden states of a multiple of 64")
        gen_w = torch.Generator(device=dev).manual_seed(wl.seed + 1)
        w1 = (torch.randn(args.mlp_hidden, wl.hidden, generator=gen_w, device=dev) / wl.hidden ** 0.5).to(torch.bfloat16)
        b1 = torch.randn(args.mlp_hidden, generator=gen_w, device=dev) * 0.1
        w2 = torch.randn(args.mlp_hidden, generator=gen_w, device=dev) / args.mlp_hidden ** 0.5
        mlp = (w1, b1, w2, 0.0)
    seq = None
    if args.probe == "seq":       # the sequence scorer, seeded random weights, its own step pool
        seq = build_seq_scorer(args, wl, g, dev, n_rounds_after=len(round_steps))
    stream = torch.cuda.current_stream()
    PROF = (B.GB_PROF_DECODE, B.GB_PROF_PROBE, B.GB_PROF_PRUNE, B.GB_PROF_GROUPED, B.GB_PROF_PLAN,
            B.GB_PROF_APPEND, B.GB_PROF_COMBINE, B.GB_PROF_ATTENTION)

    def clear_prof():
        for which in PROF:
            B.gb_pool_set_profile_events(pool.handle, which, None, None)
            if seq is not None:
                B.gb_pool_set_profile_events(seq.pool.handle, which, None, None)

    def inputs(i):
        j = i % K
        return qs[j], ks[j], vs[j], hs[h_index.get(i, 0)]

    def step(i, q, k, v, h, prof=None, o=None):
        o = out if o is None else o
        for l in range(NL):
            if prof is not None:
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_DECODE, *(prof["dec"][l] if "dec" in prof else (None, None)))
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_ATTENTION, *(prof["att"][l] if "att" in prof else (None, None)))
                if "app" in prof:
                    B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_APPEND, *prof["app"][l])
                    B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_COMBINE, *prof["comb"][l])
                    if l == 0:
                        B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PLAN, *prof["plan"])
            pool.decode_attention(l, q[l], k[l], v[l], wl.attn_scale, o[l], flags)
        if prof is not None:
            clear_prof()
        if is_round(i):
            if prof is not None and "probe" in prof:
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PROBE, *prof["probe"])
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PRUNE, *prof["prune"])
            if seq is not None:
                if prof is not None and "probe" in prof:
                    B.gb_pool_set_profile_events(seq.pool.handle, B.GB_PROF_PROBE, *prof["probe"])
                    B.gb_pool_set_profile_events(seq.pool.handle, B.GB_PROF_PRUNE, *prof["fork"])
                seq.step(h, g.scores)
                pool.push_scores(g.scores)
            elif mlp is None:
                pool.score_probe(h, wl.hidden_dtype, g.w, wl.bias, None, g.scores)
            else:
                pool.score_mlp(h, *mlp, score_out=g.scores)
            pool.prune_branch(wl.K, wl.fanout, wl.warmup, None, g.parent, g.pruned, g.lineage)
            if seq is not None:
                seq.fork(g.parent)
            if prof is not None:
                clear_prof()

    def ev_pair():
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        b.record(stream)
        return a, b

    # ---- warm-up --------------------------------------------------------------------------
    for i in steps_of("warmup"):
        step(i, *inputs(i))
    torch.cuda.synchronize()

    # ---- end to end through the C ABI with host buffers ----------------------------------------
    # Every step's q, k, v (and, at a round, the hidden states) come from pinned host memory in
    # one copy, and the step's attention output (and, at a round, the scores and the tournament's
    # outputs) go back to pinned host memory, inside the timed region.  Copies run on a second
    # stream into double buffers, overlapping the previous step.
    e2e = None
    sl = steps_of("e2e")
    if with_e2e:
        parts = (qs, ks, vs)
        nbytes = [t[0].numel() * t.element_size() for t in parts]
        offs = [0, nbytes[0], nbytes[0] + nbytes[1]]
        in_bytes = sum(nbytes)
        hin = torch.empty((K, in_bytes), dtype=torch.uint8).pin_memory()
        for n in range(K):
            for t, o0, nb in zip(parts, offs, nbytes):
                hin[n, o0:o0 + nb].copy_(t[n].reshape(-1).view(torch.uint8).cpu())
        hh = hs.cpu().pin_memory()
        din = [torch.empty(in_bytes, dtype=torch.uint8, device=dev) for _ in range(2)]
        views = [[din[b][o0:o0 + nb].view(t.dtype).view(t[0].shape) for t, o0, nb in zip(parts, offs, nbytes)]
                 for b in range(2)]
        h_d = [torch.empty_like(hs[0]) for _ in range(2)]
        dout = [torch.empty_like(out) for _ in range(2)]
        o_h = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(2)]
        r_h = {n: [torch.empty(C, dtype=t.dtype).pin_memory() for t in (g.scores, g.parent, g.pruned, g.lineage)]
               for n, i in enumerate(sl) if is_round(i)}
        cs = torch.cuda.Stream(device=dev)
        rt = _Cudart()
        SS, CS = stream.cuda_stream, cs.cuda_stream
        loaded, done, outfree = ([rt.event() for _ in range(2)] for _ in range(3))
        ev_fork, ev_join = rt.event(), rt.event()
        out_bytes = dout[0].numel() * dout[0].element_size()
        # Pointers of every buffer, layer and tensor, so a decode-only step is plain C calls.
        ptrs = [[(views[b][0][l].data_ptr(), views[b][1][l].data_ptr(), views[b][2][l].data_ptr(),
                  dout[b][l].data_ptr()) for l in range(NL)] for b in range(2)]
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        h2d = d2h = 0

        def load(n):                         # inputs of e2e step n into buffer n % 2 (copy stream)
            nonlocal h2d
            b = n % 2
            if n >= 2:
                rt.wait(CS, done[b])
            rt.copy(din[b].data_ptr(), hin[n % K].data_ptr(), in_bytes, rt.H2D, CS)
            h2d += in_bytes
            if is_round(sl[n]):
                nb = hh[0].numel() * hh.element_size()
                rt.copy(h_d[b].data_ptr(), hh[h_index[sl[n]]].data_ptr(), nb, rt.H2D, CS)
                h2d += nb
            rt.record(loaded[b], CS)

        e0.record(stream)
        t_host = time.perf_counter()
        rt.record(ev_fork, SS)
        rt.wait(CS, ev_fork)
        load(0)
        for n, i in enumerate(sl):
            b = n % 2
            if n + 1 < len(sl):
                load(n + 1)
            rt.wait(SS, loaded[b])
            if n >= 2:
                rt.wait(SS, outfree[b])
            if is_round(i):
                step(i, *views[b], h_d[b], o=dout[b])
            else:
                for l in range(NL):
                    qp, kp, vp, op = ptrs[b][l]
                    B.gb_decode_attention(pool.handle, l, qp, kp, vp, wl.attn_scale, op, flags, SS)
            rt.record(done[b], SS)
            rt.wait(CS, done[b])
            rt.copy(o_h[b].data_ptr(), dout[b].data_ptr(), out_bytes, rt.D2H, CS)
            d2h += out_bytes
            if is_round(i):
                for host, dev_t in zip(r_h[n], (g.scores, g.parent, g.pruned, g.lineage)):
                    nb = host.numel() * host.element_size()
                    rt.copy(host.data_ptr(), dev_t.data_ptr(), nb, rt.D2H, CS)
                    d2h += nb
            rt.record(outfree[b], CS)
        rt.record(ev_join, CS)
        rt.wait(SS, ev_join)
        e1.record(stream)
        t_host = time.perf_counter() - t_host
        torch.cuda.synchronize()
        for e in loaded + done + outfree + [ev_fork, ev_join]:
            rt.destroy(e)
        e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
        e2e_rounds = sum(1 for i in sl if is_round(i))
        e2e = {"value": job_value(world, C, len(sl), e_ms), "unit": "beam-tokens/s", "h2d_bytes_per_step": int(h2d // len(sl)),
               "d2h_bytes_per_step": int(d2h // len(sl)), "ms_per_step": e_ms / len(sl),
               "host_issue_us_per_step": t_host / len(sl) * 1e6,
               "context": [lay["e2e"][0], lay["e2e"][1]], "rounds": e2e_rounds,
               "path": "eager calls of the C API (gb_decode_attention per layer and step; probe and tournament "
                       "at a round); inputs copied from pinned host memory and outputs read back every step with "
                       "cudaMemcpyAsync, on a copy stream double-buffered against compute"}
        status = pool.status()
        if status != 0:
            raise RuntimeError(f"device status {status} after the e2e steps: the measurement is invalid")
        del hin, hh, din, views, dout, o_h

    # ---- filler: untimed steps up to the profiled steps ---------------------------------------
    for i in steps_of("filler"):
        step(i, *inputs(i))
    torch.cuda.synchronize()

    # ---- profiled steps: every kernel of the step bracketed by events ---------------------------
    # Each event record splits the step's chain of programmatically dependent launches, so the
    # kernel durations come from these steps and the timed window below carries no such records.
    pl = list(steps_of("profile"))
    profs = {i: {"dec": [ev_pair() for _ in range(NL)], "att": [ev_pair() for _ in range(NL)]} for i in pl}
    if args.breakdown:
        for i in pl:
            profs[i].update({"app": [ev_pair() for _ in range(NL)], "comb": [ev_pair() for _ in range(NL)],
                             "plan": ev_pair()})
    torch.cuda.synchronize()
    if args.eager:
        torch.cuda.nvtx.range_push("profiled")
        for i in pl:
            step(i, *inputs(i), prof=profs[i])
        torch.cuda.nvtx.range_pop()
    else:
        pgraph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(pgraph):
            for i in pl:
                step(i, *inputs(i), prof=profs[i])
        torch.cuda.nvtx.range_push("profiled")  # lets a profiler capture the profiled steps' kernels
        pgraph.replay()
        torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    stats = B.gb_pool_read_step_stats(pool.handle, max_steps=len(pl))   # one record per profiled step
    assert len(stats) == len(pl), (len(stats), len(pl))
    dec_ms = [a.elapsed_time(b) for i in pl for a, b in profs[i]["dec"]]
    att_ms = [a.elapsed_time(b) for i in pl for a, b in profs[i]["att"]]
    step_kernels_us = None
    if args.breakdown:
        step_kernels_us = {
            "plan": statistics.mean(profs[i]["plan"][0].elapsed_time(profs[i]["plan"][1]) for i in pl) * 1e3,
            "append": statistics.mean(a.elapsed_time(b) for i in pl for a, b in profs[i]["app"]) * 1e3,
            "attention": statistics.mean(dec_ms) * 1e3,
            # the bf16 kernels merge their records in the same launch; the fp32 one is followed by k_combine
            "combine": (statistics.mean(a.elapsed_time(b) for i in pl for a, b in profs[i]["comb"]) * 1e3
                        if not (wl.kv_dtype == "bf16" and D == 128) else None),
        }

    # ---- the timed window: K steps ending at the full context, then that context's round ---------
    tl = list(steps_of("timed"))
    timed_rounds = [i for i in tl if is_round(i)]
    rprof = {i: {} for i in tl}
    for i in timed_rounds:      # the round's probe and tournament (after the window's last decode step)
        rprof[i] = {"probe": ev_pair(), "prune": ev_pair(), "fork": ev_pair()}
    torch.cuda.synchronize()
    launches0 = B.gb_pool_launch_count(pool.handle)
    seq_launches0 = B.gb_pool_launch_count(seq.pool.handle) if seq is not None else 0
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    graph = None
    if not args.eager:
        # The K timed steps are captured once into a CUDA graph and launched once, so the
        # host's per-launch cost is out of the step (every kernel still runs, once, with the
        # arguments of its own step).
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for i in tl:
                step(i, *inputs(i), prof=rprof[i] or None)
        torch.cuda.synchronize()
    clocks = ClockSampler(gpu_id_for_smi(local))
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    torch.cuda.nvtx.range_push("timed")  # lets a profiler capture exactly the timed steps
    if graph is not None:
        graph.replay()
    else:
        for i in tl:
            step(i, *inputs(i), prof=rprof[i] or None)
    torch.cuda.nvtx.range_pop()
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    clear_prof()
    launches = B.gb_pool_launch_count(pool.handle) - launches0
    if seq is not None:
        launches += B.gb_pool_launch_count(seq.pool.handle) - seq_launches0
        if seq.pool.status() != 0:
            raise RuntimeError("sequence scorer's step pool reported an error: the measurement is invalid")
    elapsed_ms = max_over_ranks(t_start.elapsed_time(t_end), world, dev)
    status = pool.status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the timed steps: the measurement is invalid")
    prune_us = statistics.mean(rprof[i]["prune"][0].elapsed_time(rprof[i]["prune"][1]) for i in timed_rounds) * 1e3 \
        if timed_rounds else None
    probe_us = statistics.mean(rprof[i]["probe"][0].elapsed_time(rprof[i]["probe"][1]) for i in timed_rounds) * 1e3 \
        if timed_rounds else None
    fork_us = statistics.mean(rprof[i]["fork"][0].elapsed_time(rprof[i]["fork"][1]) for i in timed_rounds) * 1e3 \
        if (timed_rounds and seq is not None) else None
    grouped_on = flags != B.GB_PATH_PER_BEAM and wl.kv_dtype == "bf16" and D == 128
    # The attention launch of a layer-step: k_attention (the grouped tcgen05 role over shared
    # segments and the warp-MMA per-beam role over the tails) on the grouped path; the per-beam
    # kernel alone otherwise (warp-level MMAs for bf16 pools with 128-dim heads, paired fp32 FMAs
    # else).
    dec = "k_decode_mma" if wl.kv_dtype == "bf16" and D == 128 else "k_decode"

    # Algorithmic work per launch, from the library's per-step records of the profiled steps:
    #   per-beam role: the tokens it reads (all KV heads, K and V) + the queries;
    #   grouped role: unique bytes = every shared segment's pages once (K and V of every KV head);
    #                 bytes_read = the K/V tiles it reads (once per 128-row query tile);
    #                 useful flops = 4 * D per (query row, token) for Q.K^T and P.V.
    esz = 2 if wl.kv_dtype == "bf16" else 4
    kv_tok = 2 * Hkv * D * esz
    q_bytes = C * Hq * D * esz
    dec_tokens = [int(s[1] if grouped_on else s[0]) for s in stats]
    dec_bytes = statistics.mean(t * kv_tok + q_bytes for t in dec_tokens)
    eff_bytes = statistics.mean(int(s[0]) * kv_tok + q_bytes for s in stats)   # as if every beam read everything
    gr_read = statistics.mean(Hkv * int(s[3]) * 2 * D * esz for s in stats) if grouped_on else 0.0
    gr_unique = statistics.mean(int(s[8]) * kv_tok for s in stats) if grouped_on else 0.0
    gr_flops = statistics.mean(Hkv * int(s[2]) * 4 * D for s in stats) if grouped_on else 0.0
    dec_avg_s = statistics.mean(dec_ms) / 1e3
    att_avg_s = statistics.mean(att_ms) / 1e3
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs")
    peak_src = "measured" if peak else "fallback"
    peak = peak or 6800.0
    tpeak = peaks.get("bf16_tflops_sustained") or peaks.get("bf16_tflops")
    tpeak_src = "measured sustained" if tpeak else "fallback"
    tpeak = tpeak or 1700.0
    if grouped_on:
        kname = "k_attention"
        k_bytes = gr_unique + dec_bytes
        achieved = k_bytes / dec_avg_s / 1e9
        kernels = {kname: {"us": dec_avg_s * 1e6, "bytes": k_bytes, "gbps": achieved, "frac_hbm": achieved / peak,
                           "bytes_read": gr_read + dec_bytes,
                           "grouped_role": {"bytes": gr_unique, "bytes_read": gr_read, "flops": gr_flops,
                                            "tflops_over_launch": gr_flops / dec_avg_s / 1e12,
                                            "frac_tensor_over_launch": gr_flops / dec_avg_s / 1e12 / tpeak,
                                            "tensor_peak_source": tpeak_src,
                                            "segments": statistics.mean(int(s[4]) for s in stats),
                                            "work_units": statistics.mean(int(s[5]) * Hkv for s in stats)},
                           "per_beam_role": {"bytes": dec_bytes, "tokens": statistics.mean(dec_tokens)}}}
        role = "k_attention: grouped tcgen05 role over shared segments + warp-MMA per-beam role over the tails"
    else:
        kname = dec
        k_bytes = dec_bytes
        achieved = k_bytes / dec_avg_s / 1e9
        kernels = {kname: {"us": dec_avg_s * 1e6, "bytes": k_bytes, "gbps": achieved, "frac_hbm": achieved / peak}}
        role = f"{dec} (split-KV decode)"
    roofline = {"bound": "hbm", "kernel": role, "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": captured_traffic(kname, wl.name, args.flags, k_bytes),
                "bytes_per_launch": k_bytes, "peak_source": f"{peak_src} hbm_gbs"}

    value = job_value(world, C, K, elapsed_ms)
    ms_per_step = elapsed_ms / K

    # The capacity search builds and frees about a dozen one-layer pools; it runs after every timed
    # phase so that none of them runs in the state it leaves (host and device allocations).
    capacity = capacity_search(wl, dev) if (wl.pool_bytes is not None and rank == 0 and not args.no_capacity) else None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu_steps = args.cpu_steps or max(2, 200 // NL)
        cpu = oracle_sample(wl, cpu_steps, args.cpu_beams)
        one = oracle_sample(wl, max(1, cpu_steps // 8), 2, workers=1)   # the same oracle on one core
        cpu["single_core"] = {"value": one["value"], "unit": one["unit"], "seconds": one["seconds"],
                              "sample": one["sample"]}
    if rank == 0:
        line = {
            "metric": "beam-decode attn beam-tokens/s + achieved HBM TB/s vs peak; prune+branch us/step",
            "value": value, "unit": "beam-tokens/s", "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": wl.kv_dtype, "data": "synthetic (seeded counter-based generator, generated on device)",
            "config": {"workload": wl.name, "beams": C, "context_at_start": lay["timed"][0],
                       "context_at_end": lay["timed"][1], "layers": NL, "heads": f"{Hq}/{Hkv}", "head_dim": D,
                       "page_size": wl.page_size, "kv_dtype": wl.kv_dtype,
                       "schedule": f"decode every step; probe + tournament (K={wl.K}, fanout {wl.fanout}) every "
                                   f"{delta} tokens: {len(timed_rounds)} round(s) in the timed window (at its end)",
                       "path": args.flags, "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       "launch": "eager" if args.eager else "one CUDA graph of the timed steps",
                       "kernel_events": f"none in the timed window but the round's probe and tournament; kernel "
                                        f"durations from {len(pl)} profiled steps just before it "
                                        f"(contexts {lay['profile'][0]}-{lay['profile'][1]})",
                       "probe": {"linear": "linear", "mlp": f"mlp (hidden {args.mlp_hidden})",
                                 "seq": f"sequence scorer (layers, q heads, kv heads, ffn = {args.seq_shape}; "
                                        f"step pool of {seq.history} positions per trace before the window)"
                                 if seq is not None else None}[args.probe],
                       "l2": f"inputs larger than L2: {eff_bytes / 2**30:.2f} GiB of per-beam KV reads per layer-step",
                       "tree_build_s": round(t_build, 2),
                       "window": (f"steps end at the full context {wl.context} (fixed {wl.pool_bytes / 1e9:.0f} GB "
                                  f"pool)" if fixed_pool else f"steps end at the full context {wl.context}")},
            "attention_us": att_avg_s * 1e6,
            "attention_tbps": eff_bytes / att_avg_s / 1e12,
            "attention_tbps_note": "every beam's whole context (K and V of all KV heads) per attention time",
            "attention_kernel_us": dec_avg_s * 1e6,
            "step_kernels_us": step_kernels_us,
            "probe_us": probe_us,
            "prune_branch_us": prune_us,
            "prune_branch_note": "the whole gb_prune_branch call: rank, route, fork tables, refcounts, free, "
                                 "and the shared-prefix segment rebuild",
            "scorer_fork_us": fork_us,
            "kernels": kernels,
            "capacity": capacity,
            "roofline": roofline,
            "e2e": e2e,
            "gpu_launches": int(launches),
            "clocks": clk,
            "device_status": status,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_reference(args) -> None:
    """The CPU oracle on the host cores, same workload, metric and unit (rank 0 only)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = selected_workload(args)
    W = args.warmup
    K = args.steps if args.steps > 0 else wl.interval
    # Each step: a bounded sample (a few beams, every layer) so that the run ends within minutes:
    # at most 400 layer-steps per worker process.
    per_step_beams = max(1, min(args.cpu_beams, 16))
    steps_total = max(1, min(W + K, 400 // wl.num_layers))
    res = oracle_sample(wl, steps_total, per_step_beams)
    line = {
        "impl": "reference",
        "metric": "beam-decode attn beam-tokens/s + achieved HBM TB/s vs peak; prune+branch us/step",
        "value": res["value"], "unit": "beam-tokens/s", "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
        "steps": K, "warmup": W, "ms_per_step": wl.beams / res["value"] * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded counter-based generator)",
        "config": {"workload": wl.name, "beams": wl.beams, "context": wl.context, "layers": wl.num_layers,
                   "heads": f"{wl.num_q_heads}/{wl.num_kv_heads}", "head_dim": wl.head_dim,
                   "page_size": wl.page_size, "kv_dtype": wl.kv_dtype,
                   "sample_steps": steps_total, "sample_beams_per_step": per_step_beams},
        "cpu_baseline": {"value": res["value"], "unit": res["unit"], "cores": res["cores"], "kind": "oracle",
                         "sample": res["sample"]},
        "e2e": {"value": res["value"], "unit": "beam-tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
