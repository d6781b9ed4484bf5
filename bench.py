"""Benchmark of the beam-decode hot path of thought-level beam search on GB300.

The method's schedule: every decode step appends one token to every active
beam and attends over its context (page reservation + KV append + grouped
shared-prefix attention + per-beam split-KV attention + combine); every
Delta tokens the probe scores every beam and one tournament round prunes and
branches (rank, fork block tables, free pages, rebuild shared-prefix
segments).  The timed window is K decode steps and contains the rounds that
fall in it (by default one round: K = Delta), so every row of the hot path
runs in it and the beam tree is the one the schedule produces.

Default workload: the Qwen3-8B-shaped single layer (64 beams, 32/8 heads,
head dim 128, bf16 KV, 16-token pages), beam tree built by real rounds
(prune/branch every 512 tokens, keep 50%, branch x2) up to 4096 tokens;
the timed window runs from 4096 to 4608 tokens with the round at 4608.
Inputs are seeded synthetic data generated on the device before the timed
region.  The KV a step attends over (about 1 GiB as per-beam reads) is far
larger than L2, so no flush is needed between steps.

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
    ap.add_argument("--steps", type=int, default=0, help="timed decode steps (0: one tournament interval)")
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=2, help="workload index 1..5 (default 2: the metric's config)")
    ap.add_argument("--flags", choices=["auto", "per_beam"], default="auto")
    ap.add_argument("--group-min", type=int, default=0, help="beams a segment needs for the grouped path (0: library default, 2)")
    ap.add_argument("--cpu-steps", type=int, default=200, help="steps of the oracle sample for cpu_baseline")
    ap.add_argument("--cpu-beams", type=int, default=16, help="beams per step in the oracle sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--beams", type=int, default=0, help="override the workload's beam count (smaller profiling cases)")
    ap.add_argument("--context", type=int, default=0, help="override the workload's context length")
    ap.add_argument("--probe", choices=["linear", "mlp", "seq"], default="linear",
                    help="scorer at the tournament points: the linear probe of the workloads, the two-layer MLP, "
                         "or the history-aware sequence scorer")
    ap.add_argument("--mlp-hidden", type=int, default=512, help="hidden width of the two-layer MLP scorer")
    ap.add_argument("--seq-shape", default="2,4,2,1024",
                    help="sequence scorer layers,q-heads,kv-heads,ffn (128-dim heads; d_model = q-heads x 128)")
    ap.add_argument("--breakdown", action="store_true",
                    help="also time the planner, append and combine kernels (extra event records in the step)")
    ap.add_argument("--event-stride", type=int, default=0,
                    help="bracket the decode and grouped kernels with CUDA events on every n-th timed step "
                         "(each event record splits the step's chain of dependent launches; 0: about 32 "
                         "bracketed steps)")
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
    wl = dataclasses.replace(wl, **over)
    if args.beams or args.context:
        wl = dataclasses.replace(wl, name=f"{wl.name}[beams={wl.beams},context={wl.context}]")
    return wl


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


def captured_traffic(kernel: str, workload: str, path: str):
    """DRAM bytes per launch from the committed ncu capture, if it is of this kernel source and workload."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f).get(kernel)
        if not rec or rec["workload"] != workload or rec["path"] != path:
            return None
        with open(os.path.join(ROOT, rec["source"]), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != rec["source_sha256"]:
                return None
        return rec["dram_bytes_per_launch"]
    except (OSError, KeyError, ValueError):
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
    from oracle.attention import decode_attention
    from oracle.beams import kv_from_history
    from workload import gen
    from workload.configs import Workload
    wl = Workload(**wl_dict)
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
            "sample": (f"{steps} steps x {len(sample)} of {wl.beams} beams: fp64 two-pass decode attention at "
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
INPUT_BUDGET_BYTES = 16 * 2**30  # device memory for the pre-generated step inputs


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


def bracketed_steps(W: int, K: int, event_stride: int, breakdown: bool):
    """(stride, steps) of the timed steps whose kernels the library brackets with events:
    every step under --breakdown, else every event_stride-th (0: about 32 of the K)."""
    stride = 1 if breakdown else max(1, event_stride if event_stride > 0 else K // 32)
    return stride, [i for i in range(W, W + K) if (i - W) % stride == 0]


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
    from workload.configs import BY_INDEX
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
    if args.steps > 0:
        K = args.steps
    elif step_input_bytes * wl.interval > INPUT_BUDGET_BYTES:
        K = 64                               # pre-generated inputs of a whole interval would not fit beside the pool
    else:
        K = wl.interval
    S = W + (K if args.no_e2e else 2 * K)
    delta = wl.interval
    capacity = capacity_search(wl, dev) if (wl.pool_bytes is not None and rank == 0) else None

    # A fixed pool holds the tree up to the workload's context: the steps end there.  Otherwise
    # the timed window starts at the full context.
    fixed_pool = wl.pool_bytes is not None
    g = GpuRun(wl, device_gen=True, device=str(dev), max_context=wl.context + (0 if fixed_pool else S) + 1,
               group_min_beams=args.group_min)
    t_build = time.perf_counter()
    g.build(upto=wl.context - (S if fixed_pool else W))  # the schedule's rounds up to here, then plain appends
    torch.cuda.synchronize()
    t_build = time.perf_counter() - t_build
    pos0 = g.pos                             # context before the first (warm-up) step

    def is_round(step: int) -> bool:         # a round follows the step that brings the context to L
        L = pos0 + step + 1
        return L > wl.prompt_len and (L - wl.prompt_len) % delta == 0

    round_steps = [i for i in range(S) if is_round(i)]
    # Step inputs for every step (and hidden states for the round steps), generated before timing.
    qs = torch.empty(S, NL, C, Hq, D, dtype=g.tdt, device=dev)
    ks = torch.empty(S, NL, C, Hkv, D, dtype=g.tdt, device=dev)
    vs = torch.empty_like(ks)
    hs = torch.empty(max(1, len(round_steps)), C, wl.hidden, dtype=g.hidden.dtype, device=dev)
    h_index = {s: n for n, s in enumerate(round_steps)}
    for i in range(S):
        for l in range(NL):
            gpu_gen.normal(qs[i, l], wl.kv_dtype, 1, C, Hq * D, [wl.seed, gen.TAG_Q, l, (0, 0, 1), pos0 + i],
                           scale=wl.q_scale if wl.q_scale is not None else 1.0)
            for which, dst in ((gen.TAG_KV_K, ks), (gen.TAG_KV_V, vs)):
                gpu_gen.normal(dst[i, l], wl.kv_dtype, 1, C, Hkv * D, [wl.seed, which, l, (0, 0, 1), pos0 + i],
                               row_scale=g.hscale_dev[l] if g.hscale else None, row_scale_div=D)
    for s, n in h_index.items():
        gpu_gen.normal(hs[n], wl.hidden_dtype, 1, C, wl.hidden, [wl.seed, gen.TAG_HIDDEN, (0, 0, 1), pos0 + s + 1])
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

    def step(i, q, k, v, h, prof=None, o=None):
        o = out if o is None else o
        for l in range(NL):
            if prof is not None:
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_DECODE, *(prof["dec"][l] if "dec" in prof else (None, None)))
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_GROUPED, *(prof["gr"][l] if "gr" in prof else (None, None)))
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_ATTENTION, *(prof["att"][l] if "att" in prof else (None, None)))
                if "app" in prof:
                    B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_APPEND, *prof["app"][l])
                    B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_COMBINE, *prof["comb"][l])
                    if l == 0:
                        B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PLAN, *prof["plan"])
            pool.decode_attention(l, q[l], k[l], v[l], wl.attn_scale, o[l], flags)
        if is_round(i):
            if prof is not None:
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PROBE, *prof["probe"])
                B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PRUNE, *prof["prune"])
            if seq is not None:
                if prof is not None:
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

    for i in range(W):
        step(i, qs[i], ks[i], vs[i], hs[h_index.get(i, 0)])
    torch.cuda.synchronize()

    # Per-kernel events, recorded by the library on this stream around the kernels.
    def ev_pair():
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        b.record(stream)
        return a, b
    timed_rounds = [i for i in range(W, W + K) if is_round(i)]
    stride, inst = bracketed_steps(W, K, args.event_stride, args.breakdown)
    profs = {i: {} for i in range(W, W + K)}
    for i in inst:
        profs[i].update({"dec": [ev_pair() for _ in range(NL)], "gr": [ev_pair() for _ in range(NL)],
                         "att": [ev_pair() for _ in range(NL)]})
    if args.breakdown:  # every kernel of the step bracketed (the extra event records cost step time)
        for i in inst:
            profs[i].update({"app": [ev_pair() for _ in range(NL)], "comb": [ev_pair() for _ in range(NL)],
                             "plan": ev_pair()})
    for i in timed_rounds:
        profs[i]["probe"], profs[i]["prune"], profs[i]["fork"] = ev_pair(), ev_pair(), ev_pair()
    torch.cuda.synchronize()
    launches0 = B.gb_pool_launch_count(pool.handle)
    seq_launches0 = B.gb_pool_launch_count(seq.pool.handle) if seq is not None else 0
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    graph = None
    if not args.eager:
        # The K timed steps are captured once into a CUDA graph and launched once, so the
        # host's per-launch cost is out of the step (every kernel still runs, once, with the
        # arguments of its own step; the library's event records become graph nodes).
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for i in range(W, W + K):
                step(i, qs[i], ks[i], vs[i], hs[h_index.get(i, 0)], profs[i])
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
        for i in range(W, W + K):
            step(i, qs[i], ks[i], vs[i], hs[h_index.get(i, 0)], profs[i])
    torch.cuda.nvtx.range_pop()
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    for which in (B.GB_PROF_DECODE, B.GB_PROF_PROBE, B.GB_PROF_PRUNE, B.GB_PROF_GROUPED, B.GB_PROF_PLAN,
                  B.GB_PROF_APPEND, B.GB_PROF_COMBINE, B.GB_PROF_ATTENTION):
        B.gb_pool_set_profile_events(pool.handle, which, None, None)
        if seq is not None:
            B.gb_pool_set_profile_events(seq.pool.handle, which, None, None)
    stats = B.gb_pool_read_step_stats(pool.handle, max_steps=K)  # one record per timed step
    launches = B.gb_pool_launch_count(pool.handle) - launches0
    if seq is not None:
        launches += B.gb_pool_launch_count(seq.pool.handle) - seq_launches0
        if seq.pool.status() != 0:
            raise RuntimeError("sequence scorer's step pool reported an error: the measurement is invalid")
    elapsed_ms = max_over_ranks(t_start.elapsed_time(t_end), world, dev)
    status = pool.status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the timed steps: the measurement is invalid")
    dec_ms = [a.elapsed_time(b) for i in inst for a, b in profs[i]["dec"]]
    gr_ms = [a.elapsed_time(b) for i in inst for a, b in profs[i]["gr"]]
    att_ms = [a.elapsed_time(b) for i in inst for a, b in profs[i]["att"]]
    # In-stream duration of every kernel of a decode step (per layer; the planner once per step).
    step_kernels_us = None
    if args.breakdown:
        step_kernels_us = {
            "plan": statistics.mean(profs[i]["plan"][0].elapsed_time(profs[i]["plan"][1]) for i in inst) * 1e3,
            "append": statistics.mean(a.elapsed_time(b) for i in inst for a, b in profs[i]["app"]) * 1e3,
            "grouped": statistics.mean(gr_ms) * 1e3,
            "decode": statistics.mean(dec_ms) * 1e3,
            "combine": statistics.mean(a.elapsed_time(b) for i in inst for a, b in profs[i]["comb"]) * 1e3,
        }
    prune_us = statistics.mean(profs[i]["prune"][0].elapsed_time(profs[i]["prune"][1]) for i in timed_rounds) * 1e3 \
        if timed_rounds else None
    probe_us = statistics.mean(profs[i]["probe"][0].elapsed_time(profs[i]["probe"][1]) for i in timed_rounds) * 1e3 \
        if timed_rounds else None
    fork_us = statistics.mean(profs[i]["fork"][0].elapsed_time(profs[i]["fork"][1]) for i in timed_rounds) * 1e3 \
        if (timed_rounds and seq is not None) else None
    grouped_on = flags != B.GB_PATH_PER_BEAM and wl.kv_dtype == "bf16" and D == 128
    # The per-beam kernel: warp-level MMAs for bf16 pools with 128-dim heads, paired fp32 FMAs otherwise.
    dec = "k_decode_mma" if wl.kv_dtype == "bf16" and D == 128 else "k_decode"

    # Algorithmic work per launch, from the library's per-step records:
    #   per-beam:  tokens it reads (all KV heads, K and V) + the queries;
    #   k_grouped: K/V tiles it reads (once per 128-row query tile) and the useful flops
    #              4 * D per (query row, token) for Q.K^T and P.V.
    esz = 2 if wl.kv_dtype == "bf16" else 4
    kv_tok = 2 * Hkv * D * esz
    q_bytes = C * Hq * D * esz
    assert len(stats) == K, (len(stats), K)
    stats = [stats[i - W] for i in inst]       # the bracketed steps' work, to match their durations
    dec_tokens = [int(s[1] if grouped_on else s[0]) for s in stats]
    dec_bytes = statistics.mean(t * kv_tok + q_bytes for t in dec_tokens)
    eff_bytes = statistics.mean(int(s[0]) * kv_tok + q_bytes for s in stats)   # as if every beam read everything
    gr_bytes = statistics.mean(Hkv * int(s[3]) * 2 * D * esz for s in stats) if grouped_on else 0.0
    gr_flops = statistics.mean(Hkv * int(s[2]) * 4 * D for s in stats) if grouped_on else 0.0
    dec_avg_s = statistics.mean(dec_ms) / 1e3
    gr_avg_s = statistics.mean(gr_ms) / 1e3 if grouped_on else 0.0
    achieved = dec_bytes / dec_avg_s / 1e9
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs")
    peak_src = "measured" if peak else "fallback"
    peak = peak or 6800.0
    tpeak = peaks.get("bf16_tflops_sustained") or peaks.get("bf16_tflops")
    tpeak_src = "measured sustained" if tpeak else "fallback"
    tpeak = tpeak or 1700.0
    kernels = {dec: {"us": dec_avg_s * 1e6, "bytes": dec_bytes, "gbps": achieved, "frac_hbm": achieved / peak}}
    if grouped_on and gr_avg_s > 0:
        kernels["k_grouped"] = {"us": gr_avg_s * 1e6, "bytes": gr_bytes, "gbps": gr_bytes / gr_avg_s / 1e9,
                                "frac_hbm": gr_bytes / gr_avg_s / 1e9 / peak, "flops": gr_flops,
                                "tflops": gr_flops / gr_avg_s / 1e12, "frac_tensor": gr_flops / gr_avg_s / 1e12 / tpeak,
                                "segments": statistics.mean(int(s[4]) for s in stats),
                                "work_units": statistics.mean(int(s[5]) * Hkv for s in stats)}
    att_avg_s = statistics.mean(att_ms) / 1e3
    dominant = "k_grouped" if "k_grouped" in kernels and gr_avg_s > dec_avg_s else dec
    if "k_grouped" in kernels:
        # The grouped and per-beam kernels run concurrently on disjoint SMs: the pair is
        # one phase of the step, timed from before the fork to after the join.
        tr = [captured_traffic(k, wl.name, args.flags) for k in ("k_grouped", dec)]
        pair_bytes = gr_bytes + dec_bytes
        roofline = {"bound": "hbm", "kernel": f"k_grouped + {dec} (concurrent, disjoint SMs)",
                    "achieved": pair_bytes / att_avg_s / 1e9, "peak": peak, "unit": "GB/s",
                    "frac": pair_bytes / att_avg_s / 1e9 / peak,
                    "traffic": (tr[0] + tr[1]) if None not in tr else None, "bytes_per_launch": pair_bytes,
                    "phase_us": att_avg_s * 1e6, "peak_source": f"{peak_src} hbm_gbs"}
    elif dominant == dec:
        roofline = {"bound": "hbm", "kernel": f"{dec} (split-KV decode)", "achieved": achieved, "peak": peak,
                    "unit": "GB/s", "frac": achieved / peak, "traffic": captured_traffic(dec, wl.name, args.flags), "bytes_per_launch": dec_bytes,
                    "peak_source": f"{peak_src} hbm_gbs"}
    else:
        kg = kernels["k_grouped"]
        if kg["frac_tensor"] >= kg["frac_hbm"]:
            roofline = {"bound": "tensor", "kernel": "k_grouped (tcgen05 shared-prefix)", "achieved": kg["tflops"],
                        "peak": tpeak, "unit": "TFLOP/s", "frac": kg["frac_tensor"], "traffic": captured_traffic("k_grouped", wl.name, args.flags),
                        "flops_per_launch": gr_flops, "peak_source": f"{tpeak_src} bf16_tflops"}
        else:
            roofline = {"bound": "hbm", "kernel": "k_grouped (tcgen05 shared-prefix)", "achieved": kg["gbps"],
                        "peak": peak, "unit": "GB/s", "frac": kg["frac_hbm"], "traffic": captured_traffic("k_grouped", wl.name, args.flags),
                        "bytes_per_launch": gr_bytes, "peak_source": f"{peak_src} hbm_gbs"}

    value = job_value(world, C, K, elapsed_ms)
    ms_per_step = elapsed_ms / K

    # End to end through the C ABI with host buffers: each step's inputs copied in from pinned
    # memory and its outputs read back, inside the timed region.
    e2e = None
    if not args.no_e2e:
        # End to end: every step's q, k, v (and, at a round, the hidden states) come from
        # pinned host memory in one copy, and the step's attention output (and, at a round,
        # the scores and the tournament's outputs) go back to pinned host memory.  Copies
        # run on a second stream into double buffers, overlapping the previous step.
        sl = range(W + K, W + 2 * K)
        parts = (qs, ks, vs)
        nbytes = [t[0].numel() * t.element_size() for t in parts]
        offs = [0, nbytes[0], nbytes[0] + nbytes[1]]
        in_bytes = sum(nbytes)
        hin = torch.empty((K, in_bytes), dtype=torch.uint8).pin_memory()
        for n, i in enumerate(sl):
            for t, o0, nb in zip(parts, offs, nbytes):
                hin[n, o0:o0 + nb].copy_(t[i].reshape(-1).view(torch.uint8).cpu())
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
        S, CS = stream.cuda_stream, cs.cuda_stream
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
            rt.copy(din[b].data_ptr(), hin[n].data_ptr(), in_bytes, rt.H2D, CS)
            h2d += in_bytes
            if is_round(sl[n]):
                nb = hh[0].numel() * hh.element_size()
                rt.copy(h_d[b].data_ptr(), hh[h_index[sl[n]]].data_ptr(), nb, rt.H2D, CS)
                h2d += nb
            rt.record(loaded[b], CS)

        e0.record(stream)
        t_host = time.perf_counter()
        rt.record(ev_fork, S)
        rt.wait(CS, ev_fork)
        load(0)
        for n, i in enumerate(sl):
            b = n % 2
            if n + 1 < K:
                load(n + 1)
            rt.wait(S, loaded[b])
            if n >= 2:
                rt.wait(S, outfree[b])
            if is_round(i):
                step(i, *views[b], h_d[b], o=dout[b])
            else:
                for l in range(NL):
                    qp, kp, vp, op = ptrs[b][l]
                    B.gb_decode_attention(pool.handle, l, qp, kp, vp, wl.attn_scale, op, flags, S)
            rt.record(done[b], S)
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
        rt.wait(S, ev_join)
        e1.record(stream)
        t_host = time.perf_counter() - t_host
        torch.cuda.synchronize()
        for e in loaded + done + outfree + [ev_fork, ev_join]:
            rt.destroy(e)
        e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
        e2e = {"value": job_value(world, C, K, e_ms), "unit": "beam-tokens/s", "h2d_bytes_per_step": int(h2d // K),
               "d2h_bytes_per_step": int(d2h // K), "ms_per_step": e_ms / K,
               "host_issue_us_per_step": t_host / K * 1e6,
               "path": "eager calls of the C API (gb_decode_attention per layer and step); inputs copied from "
                       "pinned host memory and outputs read back every step with cudaMemcpyAsync, on a copy "
                       "stream double-buffered against compute"}
        status = pool.status()
        if status != 0:
            raise RuntimeError(f"device status {status} after the e2e steps: the measurement is invalid")

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = oracle_sample(wl, args.cpu_steps, args.cpu_beams)
        one = oracle_sample(wl, max(1, args.cpu_steps // 8), 2, workers=1)   # the same oracle on one core
        cpu["single_core"] = {"value": one["value"], "unit": one["unit"], "seconds": one["seconds"],
                              "sample": one["sample"]}
    if rank == 0:
        line = {
            "metric": "beam-decode attn beam-tokens/s + achieved HBM TB/s vs peak; prune+branch us/step",
            "value": value, "unit": "beam-tokens/s", "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": wl.kv_dtype, "data": "synthetic (seeded counter-based generator, generated on device)",
            "config": {"workload": wl.name, "beams": C, "context_at_start": pos0 + W, "context_at_end": pos0 + W + K,
                       "layers": NL, "heads": f"{Hq}/{Hkv}", "head_dim": D, "page_size": wl.page_size,
                       "kv_dtype": wl.kv_dtype,
                       "schedule": f"decode every step; probe + tournament (K={wl.K}, fanout {wl.fanout}) every "
                                   f"{delta} tokens: {len(timed_rounds)} round(s) in the timed window",
                       "path": args.flags, "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       "launch": "eager" if args.eager else "one CUDA graph of the timed steps",
                       "kernel_events": f"decode and grouped kernels bracketed by CUDA events on {len(inst)} of the "
                                        f"{K} timed steps (every {stride})",
                       "probe": {"linear": "linear", "mlp": f"mlp (hidden {args.mlp_hidden})",
                                 "seq": f"sequence scorer (layers, q heads, kv heads, ffn = {args.seq_shape}; "
                                        f"step pool of {seq.history} positions per trace before the window)"
                                 if seq is not None else None}[args.probe],
                       "l2": f"inputs larger than L2: {eff_bytes / 2**30:.2f} GiB of per-beam KV reads per step",
                       "tree_build_s": round(t_build, 2),
                       "window": (f"steps end at the full context {wl.context} (fixed {wl.pool_bytes / 1e9:.0f} GB pool)"
                                  if fixed_pool else f"steps start at the full context {wl.context}")},
            "attention_us": att_avg_s * 1e6,
            "attention_tbps": eff_bytes / att_avg_s / 1e12,
            "attention_tbps_note": "every beam's whole context (K and V of all KV heads) per attention time",
            "decode_kernel_us": dec_avg_s * 1e6,
            "grouped_kernel_us": gr_avg_s * 1e6,
            "step_kernels_us": step_kernels_us,
            "probe_us": probe_us,
            "prune_branch_us": prune_us,
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
    # Each step: a bounded sample (a few beams) so W + K steps end within minutes.
    per_step_beams = max(1, min(args.cpu_beams, 16))
    res = oracle_sample(wl, W + K, per_step_beams)
    steps_total = W + K
    line = {
        "impl": "reference",
        "metric": "beam-decode attn beam-tokens/s + achieved HBM TB/s vs peak; prune+branch us/step",
        "value": res["value"], "unit": "beam-tokens/s", "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
        "steps": K, "warmup": W, "ms_per_step": res["seconds"] * 1e3 / steps_total, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded counter-based generator)",
        "config": {"workload": wl.name, "beams": wl.beams, "context": wl.context},
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
