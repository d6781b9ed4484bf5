"""Benchmark of the beam-decode hot path of thought-level beam search on GB300.

One step = one pass of the whole hot path over the beam population:
  decode attention of every active beam (page reservation + KV append +
  split-KV attention + combine), the scorer probe with the running-mean
  update, and one tournament round (rank, prune, fork block tables, free).

Default workload: the Qwen3-8B-shaped single layer (64 beams, 32/8 heads,
head dim 128, bf16 KV, 16-token pages), its beam tree built by real rounds
(prune/branch every 512 tokens, keep 50%, branch x2) up to 4096 tokens of
context; timing starts there.  Inputs are seeded synthetic data generated
on the device before the timed region.  The KV read per step (1 GiB) is far
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


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=2, help="workload index 1..5 (default 2: the metric's config)")
    ap.add_argument("--flags", choices=["auto", "per_beam"], default="auto")
    ap.add_argument("--group-min", type=int, default=0, help="beams a segment needs for the grouped path (0: 16)")
    ap.add_argument("--cpu-steps", type=int, default=6, help="steps of the oracle sample for cpu_baseline")
    ap.add_argument("--cpu-beams", type=int, default=16, help="beams per step in the oracle sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


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
    """Spawned process: materialise its beams' KV, then time fp64 decode attention steps."""
    from oracle.attention import decode_attention
    from oracle.beams import kv_from_history
    from workload import gen
    from workload.configs import Workload
    wl = Workload(**wl_dict)
    hscale = [gen.head_scales(wl.seed, l, wl.num_kv_heads, *wl.head_scale) for l in range(wl.num_layers)] \
        if wl.head_scale else None
    kv = {(s, l): kv_from_history(h, wl.seed, l, wl.num_kv_heads, wl.head_dim, wl.kv_dtype,
                                  hscale[l] if hscale else None)
          for s, h in slot_hist for l in range(wl.num_layers)}
    barrier.wait()
    t0 = time.perf_counter()
    n = 0
    for pos in positions:
        for s, _ in slot_hist:
            for l in range(wl.num_layers):
                K, V = kv[(s, l)]
                q = gen.q_rows(wl.seed, l, s, pos, wl.num_q_heads, wl.head_dim, wl.kv_dtype, wl.q_scale)
                decode_attention(q, K, V, wl.attn_scale)
            n += 1
    out_q.put((time.perf_counter() - t0, n))


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
    t0 = time.perf_counter()
    results = [out_q.get() for _ in chunks]
    t_attn = time.perf_counter() - t0
    for p in procs:
        p.join()
    # The rest of the step runs once per step in this process: probe over all beams and one tournament.
    t1 = time.perf_counter()
    for _ in range(steps):
        run.probe()
        run.prune()
    t_tour = time.perf_counter() - t1
    beams_done = sum(n for _, n in results)
    total = t_attn + t_tour
    return {"value": beams_done / total, "unit": "beam-tokens/s", "cores": len(chunks), "kind": "oracle",
            "seconds": round(total, 3),
            "sample": (f"{steps} steps x {len(sample)} of {wl.beams} beams: fp64 two-pass decode attention at "
                       f"L={L} over {len(chunks)} single-threaded spawn processes, plus per step the fp64 probe "
                       f"over all {wl.beams} beams and one tournament round on the oracle pool")}


# ---------------------------------------------------------------------------
# Our arm.
# ---------------------------------------------------------------------------
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
    wl = dataclasses.replace(BY_INDEX[args.config - 1], seed=BY_INDEX[args.config - 1].seed + rank)
    flags = B.GB_PATH_AUTO if args.flags == "auto" else B.GB_PATH_PER_BEAM
    W, K = args.warmup, args.steps
    S = W + 2 * K

    g = GpuRun(wl, device_gen=True, device=str(dev), max_context=wl.context + S + 1, group_min_beams=args.group_min)
    t_build = time.perf_counter()
    g.build(upto=wl.context)
    torch.cuda.synchronize()
    t_build = time.perf_counter() - t_build
    C, Hq, Hkv, D, NL = wl.beams, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.num_layers
    pos0 = g.pos

    # Step inputs for every step, generated on the device before timing.
    qs = torch.empty(S, NL, C, Hq, D, dtype=g.tdt, device=dev)
    ks = torch.empty(S, NL, C, Hkv, D, dtype=g.tdt, device=dev)
    vs = torch.empty_like(ks)
    hs = torch.empty(S, C, wl.hidden, dtype=g.hidden.dtype, device=dev)
    for i in range(S):
        for l in range(NL):
            gpu_gen.normal(qs[i, l], wl.kv_dtype, 1, C, Hq * D, [wl.seed, gen.TAG_Q, l, (0, 0, 1), pos0 + i],
                           scale=wl.q_scale if wl.q_scale is not None else 1.0)
            for which, dst in ((gen.TAG_KV_K, ks), (gen.TAG_KV_V, vs)):
                gpu_gen.normal(dst[i, l], wl.kv_dtype, 1, C, Hkv * D, [wl.seed, which, l, (0, 0, 1), pos0 + i],
                               row_scale=g.hscale_dev[l] if g.hscale else None, row_scale_div=D)
        gpu_gen.normal(hs[i], wl.hidden_dtype, 1, C, wl.hidden, [wl.seed, gen.TAG_HIDDEN, (0, 0, 1), pos0 + i])
    out = torch.empty(NL, C, Hq, D, dtype=torch.float32, device=dev)
    pool = g.pool

    def step(i):
        for l in range(NL):
            pool.decode_attention(l, qs[i, l], ks[i, l], vs[i, l], wl.attn_scale, out[l], flags)
        pool.score_probe(hs[i], wl.hidden_dtype, g.w, wl.bias, None, g.scores)
        pool.prune_branch(wl.K, wl.fanout, wl.warmup, None, g.parent, g.pruned, g.lineage)

    stream = torch.cuda.current_stream()
    for i in range(W):
        step(i)
    torch.cuda.synchronize()

    # Per-kernel events (recorded by the library on this stream around the kernels).
    def events(n):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
        for e in evs:
            e.record(stream)
        return evs
    n_dec = K * NL
    dec_a, dec_b = events(n_dec), events(n_dec)
    gr_a, gr_b = events(n_dec), events(n_dec)
    pr_a, pr_b, pb_a, pb_b = events(K), events(K), events(K), events(K)
    torch.cuda.synchronize()
    launches0 = B.gb_pool_launch_count(pool.handle)
    clocks = ClockSampler(gpu_id_for_smi(local))
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(K):
        i = W + k
        B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PRUNE, pr_a[k], pr_b[k])
        B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_PROBE, pb_a[k], pb_b[k])
        for l in range(NL):
            B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_DECODE, dec_a[k * NL + l], dec_b[k * NL + l])
            B.gb_pool_set_profile_events(pool.handle, B.GB_PROF_GROUPED, gr_a[k * NL + l], gr_b[k * NL + l])
            pool.decode_attention(l, qs[i, l], ks[i, l], vs[i, l], wl.attn_scale, out[l], flags)
        pool.score_probe(hs[i], wl.hidden_dtype, g.w, wl.bias, None, g.scores)
        pool.prune_branch(wl.K, wl.fanout, wl.warmup, None, g.parent, g.pruned, g.lineage)
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    for which in (B.GB_PROF_DECODE, B.GB_PROF_PROBE, B.GB_PROF_PRUNE, B.GB_PROF_GROUPED):
        B.gb_pool_set_profile_events(pool.handle, which, None, None)
    stats = B.gb_pool_read_step_stats(pool.handle, max_steps=K)  # one record per timed step (layer 0 opens it)
    launches = B.gb_pool_launch_count(pool.handle) - launches0
    elapsed_ms = t_start.elapsed_time(t_end)
    if world > 1:
        t = torch.tensor([elapsed_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        elapsed_ms = float(t.item())
    dec_ms = [a.elapsed_time(b) for a, b in zip(dec_a, dec_b)]
    prune_us = statistics.mean(a.elapsed_time(b) for a, b in zip(pr_a, pr_b)) * 1e3
    probe_us = statistics.mean(a.elapsed_time(b) for a, b in zip(pb_a, pb_b)) * 1e3
    status = pool.status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the timed steps: the measurement is invalid")

    gr_ms = [a.elapsed_time(b) for a, b in zip(gr_a, gr_b)]
    grouped_on = flags != B.GB_PATH_PER_BEAM and wl.kv_dtype == "bf16" and D == 128

    # Algorithmic work per launch, from the library's per-step records:
    #   k_decode:  tokens it reads (all KV heads, K and V) + the queries;
    #   k_grouped: K/V tiles it reads (once per 128-row query tile) and the useful flops
    #              4 * D per (query row, token) for Q.K^T and P.V.
    esz = 2 if wl.kv_dtype == "bf16" else 4
    kv_tok = 2 * Hkv * D * esz
    q_bytes = C * Hq * D * esz
    assert len(stats) == K, (len(stats), K)
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
    kernels = {"k_decode": {"us": dec_avg_s * 1e6, "bytes": dec_bytes, "gbps": achieved, "frac_hbm": achieved / peak}}
    if grouped_on and gr_avg_s > 0:
        kernels["k_grouped"] = {"us": gr_avg_s * 1e6, "bytes": gr_bytes, "gbps": gr_bytes / gr_avg_s / 1e9,
                                "frac_hbm": gr_bytes / gr_avg_s / 1e9 / peak, "flops": gr_flops,
                                "tflops": gr_flops / gr_avg_s / 1e12, "frac_tensor": gr_flops / gr_avg_s / 1e12 / tpeak,
                                "segments": statistics.mean(int(s[4]) for s in stats),
                                "tiles": statistics.mean(int(s[5]) for s in stats)}
    dominant = "k_grouped" if "k_grouped" in kernels and gr_avg_s > dec_avg_s else "k_decode"
    if dominant == "k_decode":
        roofline = {"bound": "hbm", "kernel": "k_decode (split-KV decode)", "achieved": achieved, "peak": peak,
                    "unit": "GB/s", "frac": achieved / peak, "traffic": None, "bytes_per_launch": dec_bytes,
                    "peak_source": f"{peak_src} hbm_gbs"}
    else:
        kg = kernels["k_grouped"]
        if kg["frac_tensor"] >= kg["frac_hbm"]:
            roofline = {"bound": "tensor", "kernel": "k_grouped (tcgen05 shared-prefix)", "achieved": kg["tflops"],
                        "peak": tpeak, "unit": "TFLOP/s", "frac": kg["frac_tensor"], "traffic": None,
                        "flops_per_launch": gr_flops, "peak_source": f"{tpeak_src} bf16_tflops"}
        else:
            roofline = {"bound": "hbm", "kernel": "k_grouped (tcgen05 shared-prefix)", "achieved": kg["gbps"],
                        "peak": peak, "unit": "GB/s", "frac": kg["frac_hbm"], "traffic": None,
                        "bytes_per_launch": gr_bytes, "peak_source": f"{peak_src} hbm_gbs"}

    value = world * C * K / (elapsed_ms / 1e3)
    ms_per_step = elapsed_ms / K

    # End to end through the C ABI with host buffers: inputs copied in from pinned memory and
    # outputs read back every step, inside the timed region.
    e2e = None
    if not args.no_e2e:
        sl = slice(W + K, W + 2 * K)
        hq, hk, hv, hh = (t[sl].cpu().pin_memory() for t in (qs, ks, vs, hs))
        q_d, k_d, v_d, h_d = (torch.empty_like(t[0]) for t in (qs, ks, vs, hs))
        o_h = torch.empty(out.shape, dtype=out.dtype).pin_memory()
        s_h = torch.empty(C, dtype=torch.float32).pin_memory()
        p_h = torch.empty(C, dtype=torch.int32).pin_memory()
        pr_h = torch.empty(C, dtype=torch.uint8).pin_memory()
        ln_h = torch.empty(C, dtype=torch.int32).pin_memory()
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for k in range(K):
            q_d.copy_(hq[k], non_blocking=True)
            k_d.copy_(hk[k], non_blocking=True)
            v_d.copy_(hv[k], non_blocking=True)
            h_d.copy_(hh[k], non_blocking=True)
            for l in range(NL):
                pool.decode_attention(l, q_d[l], k_d[l], v_d[l], wl.attn_scale, out[l], flags)
            pool.score_probe(h_d, wl.hidden_dtype, g.w, wl.bias, None, g.scores)
            pool.prune_branch(wl.K, wl.fanout, wl.warmup, None, g.parent, g.pruned, g.lineage)
            o_h.copy_(out, non_blocking=True)
            s_h.copy_(g.scores, non_blocking=True)
            p_h.copy_(g.parent, non_blocking=True)
            pr_h.copy_(g.pruned, non_blocking=True)
            ln_h.copy_(g.lineage, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms = e0.elapsed_time(e1)
        if world > 1:
            t = torch.tensor([e_ms], device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e_ms = float(t.item())
        h2d = sum(t[0].numel() * t.element_size() for t in (hq, hk, hv, hh))
        d2h = sum(t.numel() * t.element_size() for t in (o_h, s_h, p_h, pr_h, ln_h))
        e2e = {"value": world * C * K / (e_ms / 1e3), "unit": "beam-tokens/s", "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h), "ms_per_step": e_ms / K}
        status = status or pool.status()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = oracle_sample(wl, args.cpu_steps, args.cpu_beams)
    if rank == 0:
        line = {
            "metric": "beam-decode attn beam-tokens/s + achieved HBM TB/s vs peak; prune+branch us/step",
            "value": value, "unit": "beam-tokens/s", "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": wl.kv_dtype, "data": "synthetic (seeded counter-based generator, generated on device)",
            "config": {"workload": wl.name, "beams": C, "context_at_start": pos0, "context_at_end": pos0 + K,
                       "layers": NL, "heads": f"{Hq}/{Hkv}", "head_dim": D, "page_size": wl.page_size,
                       "kv_dtype": wl.kv_dtype, "tournament": f"K={wl.K} fanout={wl.fanout} every step",
                       "path": args.flags, "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       "l2": f"inputs larger than L2: {C * pos0 * kv_tok / 2**30:.2f} GiB of KV read per step",
                       "tree_build_s": round(t_build, 2)},
            "attention_us": (dec_avg_s + gr_avg_s) * 1e6,
            "attention_tbps": eff_bytes / (dec_avg_s + gr_avg_s) / 1e12,
            "attention_tbps_note": "every beam's whole context (K and V of all KV heads) per attention time",
            "decode_kernel_us": dec_avg_s * 1e6,
            "grouped_kernel_us": gr_avg_s * 1e6,
            "probe_us": probe_us,
            "prune_branch_us": prune_us,
            "kernels": kernels,
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
    from workload.configs import BY_INDEX
    wl = BY_INDEX[args.config - 1]
    W, K = args.warmup, args.steps
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
