"""Benchmark of the DAVET step-conditioning hot path on one or more GPUs.

One bench step is one pass of the whole path over one batch: the evidence
pyramid of every request (once), then, for each of the workload's T
denoising steps, the view gather, the step attention and the unmasking.
`value` is denoising steps per second over all ranks, with inputs resident in
HBM; `e2e` is the same metric through the C ABI from pinned host buffers,
with every step's inputs copied in and the committed tokens copied out inside
the timed region.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME]
    python bench.py --impl reference ...   # the fp64 CPU oracle, bounded sample

Multi-GPU (torchrun): requests are independent, so every rank runs its own
batch (weak scaling, no collective on the data path); the per-pass times are
reduced with MAX across ranks only for reporting.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "step attention TFLOP/s (% bf16 peak); pyramid/unmask HBM GB/s; steps/s"
DEFAULT_CONFIG = "highres"
L2_FLUSH_BYTES = 512 << 20


def attention_source_hash() -> str:
    """sha256 of the attention kernel's sources (attention.cu, common.cuh)."""
    import hashlib
    h = hashlib.sha256()
    for f in ("attention.cu", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2608_01821_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def profiled_traffic(workload: str, fused: bool = True):
    """DRAM bytes per attention launch from the committed ncu summary of this
    workload's pass, or None when the summary is missing or was taken on
    different kernel sources."""
    kind = "view_attention" if fused else "attention"
    path = os.path.join(ROOT, "profiles", f"{kind}_{workload}_pass_traffic.txt")
    try:
        kv = {}
        for line in open(path):
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                kv[k.strip()] = v.strip()
        if kv.get("kernel_sources_sha256") != attention_source_hash():
            return None
        return float(kv["dram_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        time.sleep(0.25)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        time.sleep(0.15)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = max(mx, float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------- our arm
def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2608_01821_gb300 import davet, workloads
    from paper_2608_01821_gb300.pipeline import Pipeline

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    lib = davet.load()
    w = workloads.make(args.config)
    if args.schedule != "workload":
        workloads.set_static_view(w, args.schedule)
    if rank > 0:
        w.seed = w.seed + 1000 * rank  # each replica gets its own batch
    realizer = getattr(args, "realizer", "pool")
    pl = Pipeline(w, dev, lib, fused=not getattr(args, "unfused", False), realizer=realizer)
    feats = [workloads.features(w, b) for b in range(w.batch)]
    text = workloads.text_rows(w)
    scores = [workloads.token_scores(w, b) for b in range(w.batch)] if realizer == "prune" else None
    pl.load_inputs(feats, text, scores=scores)
    torch.cuda.synchronize()

    # step logits: a pool of distinct device buffers, step t uses t % P
    logit_bytes = w.total_resp * w.V * 2
    P = max(2, min(w.T, int((16 << 30) // max(logit_bytes, 1))))
    if args.logit_pool:
        P = max(1, min(P, args.logit_pool))
    pool = torch.empty((P, w.total_resp, w.V), dtype=torch.bfloat16, device=dev)
    for i in range(P):
        workloads.logits_device(w, i, dev, out=pool[i])
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(device=dev)

    # closed-loop policy (Eq. 6-9 on the device): each step's view comes from
    # the previous step's unmasking statistics
    policy = getattr(args, "policy", False)
    if policy:
        orient = 0 if args.orientation == "early" else 1
        view_level = workloads.policy_view_levels(w)
        lo = torch.empty((w.batch, w.T), dtype=torch.float64, device=dev)
        up = torch.empty_like(lo)
        demand = (None if args.uniform_demand else
                  torch.tensor(workloads.request_demands(w), dtype=torch.float64, device=dev))
        budget = torch.zeros((w.T, w.batch), dtype=torch.float64, device=dev)

    def policy_pass():
        lib.davet_policy_envelope(w.T, orient, args.budget, args.rho, demand, w.batch, lo, up)

    def policy_step(t):
        lib.davet_policy_step(t, w.T, lo, up, pl.stats[t - 1] if t else None, w.batch, args.alpha, view_level,
                              pl.schedule[t], budget[t])

    def one_pass():
        pl.reset_state()
        pl.build_pyramids()
        if policy:
            policy_pass()
        for t in range(w.T):
            if policy:
                policy_step(t)
            pl.step(t, pool[t % P])

    # eager warm-up (first calls resolve device addresses), then graph capture
    with torch.cuda.stream(stream):
        for _ in range(2):
            one_pass()
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        one_pass()
    torch.cuda.synchronize()

    # correctness guard: every answer position committed or still masked sensibly
    st, flags = lib.davet_device_status()
    if st != 0:
        raise RuntimeError(f"device error word {flags:#x} after warm-up")

    # --------------------------------------------------- timed region
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks:
        wall0 = time.perf_counter()
        with torch.cuda.stream(stream):
            for i in range(args.steps):
                flush.fill_(i & 0xFF)  # evict L2 between timed passes (not timed)
                starts[i].record(stream)
                graph.replay()
                ends[i].record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
    barrier(world)
    pass_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    total_s = sum(pass_ms) / 1e3
    total_s = allreduce_max(total_s, world, dev)
    st, flags = lib.davet_device_status()
    if st != 0:
        raise RuntimeError(f"device error word {flags:#x} after the timed region")

    # ------------------------------------ per-kernel times (eager, events)
    comp = kernel_times(pl, w, pool, P, stream, flush, policy_pass=policy_pass if policy else None,
                        policy_step=policy_step if policy else None)
    comp["pass_ms"] = statistics.mean(pass_ms)
    comp["sum_vs_pass"] = comp["sum_ms"] / comp["pass_ms"]

    # ---------------------------------------------------------- e2e
    e2e = None if args.no_e2e else run_e2e(args, pl, w, dev, stream, world,
                                           policy_pass=policy_pass if policy else None,
                                           policy_step=policy_step if policy else None)

    out = None
    if rank == 0:
        peaks = measured_peaks()
        value = whole_job_rate(w.T * args.steps, world, total_s)
        # per request the view-block build (realizer + fill kernels) or the
        # pyramid; per step the fused view attention (or gather and attention)
        # and the two unmask kernels
        launches_per_pass = build_launches(w, pl.realizer, pl.fused) + w.T * (3 if pl.fused else 4)
        if policy:
            launches_per_pass += 1 + w.T  # envelope, then one policy step per denoising step
        akey = "view_attention" if pl.fused else "attention"
        attn_flops_launch = comp[akey]["flops"] / comp[akey]["launches"]
        attn_ms = comp[akey]["ms"] / comp[akey]["launches"]
        achieved = attn_flops_launch / (attn_ms * 1e-3) / 1e12
        out = {
            "metric": METRIC,
            "value": round(value, 3),
            "unit": "denoising steps/s",
            "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup,
            "ms_per_step": round(statistics.mean(pass_ms), 4),
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "bf16",
            "data": "synthetic (seeded N(0,1) features/text, N(0,2) logits; no weights)",
            "config": {
                **workload_config(w),
                "parallelism": f"replicas x{world} (independent requests)",
                "timing": "CUDA events per pass on the launching stream; one CUDA graph per pass",
                "l2": f"{L2_FLUSH_BYTES >> 20} MiB write between timed passes (not timed)",
                "logit_pool": P,
                "realizer": pl.realizer,
            },
            "components": {
                k: ({kk: (round(vv, 4) if isinstance(vv, float) else vv) for kk, vv in v.items()}
                    if isinstance(v, dict) else v)
                for k, v in comp.items()
            },
            "roofline": {
                "kernel": "view_attention (fused gather and step attention)" if pl.fused else "step_attention",
                "bound": "tensor",
                "achieved": round(achieved, 2),
                "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s",
                "frac": round(achieved / peaks["bf16_tflops"], 4),
                "peak_source": f"{peaks['source']} bf16 burst (MEASURED_PEAKS.json)",
                "traffic": profiled_traffic(w.name, pl.fused),
                "traffic_unit": "bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum)",
                "flops_per_launch": attn_flops_launch,
            },
            "clocks": clocks.summary(),
            "gpu_launches": launches_per_pass * args.steps,
            "e2e": e2e,
            "wall_s_timed": round(wall, 3),
        }
        if policy:
            out["config"]["schedule"] = "closed-loop policy (Eq. 6-9 on the device)"
            out["policy"] = policy_summary(args, w, pl.schedule.cpu().numpy(), budget)
        elif args.schedule != "workload":
            out["config"]["schedule"] = f"static {args.schedule} view"
    return out


def run_backbone(args, rank, world, local_rank):
    """The full backbone step (`--model full`): every denoising step runs
    `--layers` synthetic-weight layers over the step sequence, the LM head
    over the answer rows and the unmasking, in one CUDA graph per pass."""
    import torch

    from paper_2608_01821_gb300 import davet, workloads
    from paper_2608_01821_gb300.model import Backbone

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    lib = davet.load()
    w = workloads.make(args.config)
    if args.schedule != "workload":
        workloads.set_static_view(w, args.schedule)
    if rank > 0:
        w.seed = w.seed + 1000 * rank
    bb = Backbone(w, args.layers, dev, lib)
    if args.policy:
        bb.use_policy(args.orientation, args.budget, args.rho, args.alpha, args.uniform_demand)
    feats = [workloads.normal_bf16((w.tiles[b], w.grid, w.grid, bb.C),
                                   workloads.derive_seed(w.seed, workloads.KIND_FEAT, b)) for b in range(w.batch)]
    prompts = [workloads.normal_bf16((w.prompt[b], bb.C), workloads.derive_seed(w.seed, workloads.KIND_TEXT, b))
               for b in range(w.batch)]
    bb.load_inputs(feats, prompts)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def one_pass(timed=None):
        bb.begin_pass()
        bb.build_pyramids()
        for t in range(w.T):
            bb.step(t, timed=timed)

    with torch.cuda.stream(stream):
        one_pass()
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        one_pass()
    torch.cuda.synchronize()
    st, flags = lib.davet_device_status()
    if st != 0:
        raise RuntimeError(f"device error word {flags:#x} after warm-up")
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks:
        with torch.cuda.stream(stream):
            for i in range(args.steps):
                flush.fill_(i & 0xFF)
                starts[i].record(stream)
                graph.replay()
                ends[i].record(stream)
        torch.cuda.synchronize()
    barrier(world)
    pass_ms = [a.elapsed_time(b) for a, b in zip(starts, ends)]
    total_s = allreduce_max(sum(pass_ms) / 1e3, world, dev)
    st, flags = lib.davet_device_status()
    if st != 0:
        raise RuntimeError(f"device error word {flags:#x} after the timed region")

    # per-kind device time of one pass: a graph with an event pair around every call
    calls = []

    def timed(kind, fn):
        a, b = torch.cuda.Event(enable_timing=True, external=True), torch.cuda.Event(enable_timing=True,
                                                                                     external=True)
        a.record(stream)
        fn()
        b.record(stream)
        calls.append((kind, a, b))

    g2 = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g2, stream=stream):
        one_pass(timed)
    g2.replay()
    torch.cuda.synchronize()
    kinds = {}
    for kind, a, b in calls:
        kinds[kind] = kinds.get(kind, 0.0) + a.elapsed_time(b)
    n_gemm = sum(1 for k, _, _ in calls if k == "gemm")
    # the views every step ran (the policy's choices are read back after the pass)
    sched = bb.schedule.cpu().numpy()
    step_rows = [bb.rows_of(sched[t]) for t in range(w.T)]
    gemm_flops = sum(bb.gemm_flops(t, step_rows[t]) for t in range(w.T))

    # end to end: visual hidden states and prompt rows from pinned host memory,
    # committed tokens back to the host, every pass
    e2e = None
    if not args.no_e2e:
        pf = [f.pin_memory() for f in feats]
        pp = [p.pin_memory() for p in prompts]
        tok_host = torch.empty(w.total_resp, dtype=torch.int32).pin_memory()
        n = max(1, min(args.steps, 3))
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            s0.record(stream)
            for _ in range(n):
                bb.load_inputs(pf, pp, non_blocking=True)
                graph.replay()
                tok_host.copy_(bb.tokens, non_blocking=True)
            s1.record(stream)
        torch.cuda.synchronize()
        te = allreduce_max(s0.elapsed_time(s1) / 1e3, world, dev)
        h2d = sum(f.numel() * 2 for f in pf) + sum(p.numel() * 2 for p in pp)
        d2h = w.total_resp * 4
        e2e = {"value": round(w.T * n * world / te, 3), "unit": "denoising steps/s",
               "h2d_bytes_per_step": int(round(h2d / w.T)), "d2h_bytes_per_step": int(round(d2h / w.T)),
               "h2d_bytes_per_pass": int(h2d), "d2h_bytes_per_pass": int(d2h), "passes": n,
               "bytes_note": "per denoising step = per pass / T (inputs and tokens cross once per pass)"}

    if rank != 0:
        return None
    peaks = measured_peaks()
    achieved = gemm_flops / (kinds["gemm"] * 1e-3) / 1e12
    peak = peaks.get("bf16_tflops_sustained") or peaks["bf16_tflops"]
    n_steps = w.T
    return {
        "metric": METRIC,
        "value": round(whole_job_rate(w.T * args.steps, world, total_s), 3),
        "unit": "denoising steps/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(pass_ms), 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) visual hidden states and prompt rows; random N(0,1/fan_in) weights)",
        "config": {
            "workload": w.name,
            "model": "full backbone step (synthetic weights)",
            "layers": args.layers,
            "hidden": bb.C,
            "heads": w.H,
            "head_dim": w.D,
            "mlp": bb.F,
            "vocab": w.V,
            "batch": w.batch,
            "denoising_steps_per_pass": n_steps,
            "parallelism": f"replicas x{world} (independent requests)",
            "timing": "CUDA events per pass on the launching stream; one CUDA graph per pass",
            "l2": f"{L2_FLUSH_BYTES >> 20} MiB write between timed passes (not timed); weights stream from HBM",
            "schedule": ("closed-loop policy (Eq. 6-9 on the device)" if args.policy else
                         "workload level schedule" if args.schedule == "workload" else f"static {args.schedule} view"),
            "mean_rows_per_step": round(sum(step_rows) / w.T, 2),
        },
        "components": {k: {"ms_per_pass": round(v, 3), "share": round(v / sum(kinds.values()), 4)}
                       for k, v in kinds.items()},
        "roofline": {
            "kernel": "davet_linear (tcgen05 GEMM, all projections and the LM head)",
            "bound": "tensor",
            "achieved": round(achieved, 2),
            "peak": peak,
            "unit": "TFLOP/s",
            "frac": round(achieved / peak, 4),
            "peak_source": f"{peaks['source']} bf16 sustained (MEASURED_PEAKS.json)",
            "traffic": None,
            "flops_per_launch": gemm_flops / max(n_gemm, 1),
        },
        "clocks": clocks.summary(),
        "gpu_launches": (sum(1 for x in w.tiles if x > 0) + sum(bb.launches(t) for t in range(w.T))
                         + (1 if args.policy else 0)) * args.steps,
        "e2e": e2e,
        **({"policy": policy_summary(args, w, sched, bb.budget)} if args.policy else {}),
    }


def policy_summary(args, w, sched, budget):
    """The policy's settings and what it chose over one pass."""
    import numpy as np

    from paper_2608_01821_gb300 import workloads
    views, counts = np.unique(sched, return_counts=True)
    return {"orientation": args.orientation, "B": args.budget, "rho": args.rho, "alpha": args.alpha,
            "view_levels": workloads.policy_view_levels(w),
            "demand": [1.0] * w.batch if args.uniform_demand else workloads.request_demands(w),
            "mean_budget": round(float(budget.mean().item()), 4),
            "steps_per_view": {int(v): int(c) for v, c in zip(views, counts)}}


def merge_round_count(grid: int, n_levels: int) -> int:
    """Bipartite matching rounds the merging realizer runs per tile: level l
    is reached from n tokens by rounds of r = min(n - G_l^2, ceil(n/2))."""
    sides, g = [], grid
    for _ in range(n_levels):
        sides.append(g)
        g = (g + 1) // 2
    n, rounds = grid * grid, 0
    for g in sides[1:]:
        while n > g * g:
            n -= min(n - g * g, (n + 1) // 2)
            rounds += 1
    return rounds


def workload_config(w) -> dict:
    """The workload's defining sizes, reported by both arms."""
    return {"workload": w.name, "batch": w.batch, "heads": w.H, "head_dim": w.D, "grid": w.grid,
            "levels": w.n_levels, "tiles": w.tiles if w.batch <= 16 else sum(w.tiles),
            "denoising_steps_per_pass": w.T, "vocab": w.V, "k": w.k}


def build_launches(w, realizer: str, fused: bool) -> int:
    """Kernels the view construction of one pass launches (all requests)."""
    if not fused:
        return sum(1 for t in w.tiles if t > 0)
    n = 0
    for b in range(w.batch):
        has_text = w.prompt[b] + w.resp[b] > 0
        if w.tiles[b] > 0:
            if realizer == "merge":
                R = merge_round_count(w.grid, w.n_levels)
                n += 1 + 3 * R + (w.n_levels - 1)  # init, rounds, level rows
            else:
                n += 1  # pyramid or pruning kernel
        if has_text or (w.mixed and realizer != "prune" and w.tiles[b] > 0):
            n += 1  # text (and mixed) fill
    return n


def kernel_times(pl, w, pool, P, stream, flush, reps=3, policy_pass=None, policy_step=None):
    """Average device time of each kind of kernel over one pass.

    Every kind's calls of one pass are captured into a CUDA graph of their
    own, in pass order and with nothing between them (so the kernels chain
    with programmatic dependent launch as they do in the pass): the view
    construction; the T step attentions (or gathers and attentions); the
    answer-state reset followed by the T unmaskings; the allocation policy's
    steps when it runs.  Each graph is replayed `reps` times between CUDA
    events on the launching stream, L2 evicted before every replay as before
    every timed pass.  The answer-state reset (three fills) is timed alone
    and taken out of the unmasking.  `sum_ms` against the pass time shows
    how well the parts add up."""
    import torch

    def graph_of(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        return g

    def time_graph(g):
        t = 0.0
        with torch.cuda.stream(stream):
            for i in range(reps):
                flush.fill_(i & 0xFF)
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                g.replay()
                b.record(stream)
                b.synchronize()
                t += a.elapsed_time(b)
        return t / reps

    def attn_all():
        for t in range(w.T):
            if pl.fused:
                pl.view_attention(t)
            else:
                pl.gather(t)
                pl.attention()

    def gather_all():
        for t in range(w.T):
            pl.gather(t)

    def unmask_all():
        pl.reset_state()
        for t in range(w.T):
            pl.unmask(t, pool[t % P])

    def policy_all():
        policy_pass()
        for t in range(w.T):
            policy_step(t)

    graphs = {"pyramid": graph_of(pl.build_pyramids), "reset": graph_of(pl.reset_state),
              "unmask": graph_of(unmask_all)}
    scratch = []
    if pl.fused and pl.realizer == "pool":
        # the pyramid kernel alone (the view-block build also runs the text
        # fill): each request's level 0 copied into a level-major scratch
        # pyramid, pooled there with davet_build_pyramid (the same kernel and
        # bytes as inside davet_build_views)
        for b in range(w.batch):
            if w.tiles[b] > 0:
                buf = torch.empty((w.pyramid_rows(b), w.C), dtype=torch.bfloat16, device=pl.dev)
                l0 = pl.level0(b)
                buf[:l0.shape[0]].copy_(l0)
                scratch.append((b, buf))

        def pyramid_kernels():
            for b, buf in scratch:
                pl.lib.davet_build_pyramid(buf, buf, w.tiles[b], w.grid, w.n_levels, w.C, None, stream)

        graphs["pyramid_kernel"] = graph_of(pyramid_kernels)
    if pl.fused:
        graphs["view_attention"] = graph_of(attn_all)
    else:
        graphs["gather"] = graph_of(gather_all)
        graphs["gather+attention"] = graph_of(attn_all)
    if policy_pass is not None:
        graphs["policy"] = graph_of(policy_all)
    torch.cuda.synchronize()
    totals = {k: time_graph(g) for k, g in graphs.items()}
    pk_ms = totals.pop("pyramid_kernel", None)
    del scratch
    totals["unmask"] = max(totals["unmask"] - totals["reset"], 0.0)
    if not pl.fused:
        totals["attention"] = max(totals.pop("gather+attention") - totals["gather"], 0.0)
    mode = "per-kind CUDA graphs (the pass's calls of one kind, chained as in the pass)"
    ms = totals
    flops = sum(w.attention_flops(t) for t in range(w.T))
    gbytes = sum(w.gather_bytes(t) for t in range(w.T))
    ubytes = sum(w.unmask_bytes(t) for t in range(w.T))
    pbytes = w.pyramid_bytes()
    nb = build_launches(w, pl.realizer, pl.fused)
    if pl.realizer == "pool":
        out = {
            "timing_mode": mode,
            "pyramid": {"launches": nb, "ms": ms["pyramid"], "bytes": pbytes,
                        "GBps": pbytes / (ms["pyramid"] * 1e-3) / 1e9,
                        # with the view blocks' text copies (and mixed rows) the fill adds
                        "bytes_with_fill": pbytes + w.view_fill_bytes(),
                        "GBps_with_fill": (pbytes + w.view_fill_bytes()) / (ms["pyramid"] * 1e-3) / 1e9},
        }
        if pk_ms:
            out["pyramid"]["pyramid_kernel"] = {
                "launches": sum(1 for t in w.tiles if t > 0), "ms": pk_ms, "bytes": pbytes,
                "GBps": pbytes / (pk_ms * 1e-3) / 1e9,
                "what": "the pyramid kernel alone (davet_build_pyramid on a level-major copy of level 0)"}
    else:
        out = {
            "timing_mode": mode,
            "views_build": {"realizer": pl.realizer, "launches": nb, "ms": ms["pyramid"],
                            "ms_per_request": ms["pyramid"] / max(w.batch, 1)},
        }
    if pl.fused:
        out["view_attention"] = {"launches": w.T, "ms": ms["view_attention"], "flops": flops,
                                 "TFLOPs": flops / (ms["view_attention"] * 1e-3) / 1e12}
    else:
        out["gather"] = {"launches": w.T, "ms": ms["gather"], "bytes": gbytes,
                         "GBps": gbytes / (ms["gather"] * 1e-3) / 1e9}
        out["attention"] = {"launches": w.T, "ms": ms["attention"], "flops": flops,
                            "TFLOPs": flops / (ms["attention"] * 1e-3) / 1e12}
    out["unmask"] = {"launches": 2 * w.T, "ms": ms["unmask"], "bytes": ubytes,
                     "GBps": ubytes / (ms["unmask"] * 1e-3) / 1e9}
    out["reset"] = {"launches": 3, "ms": ms["reset"], "what": "answer-state reset (torch fills)"}
    if "policy" in ms:
        out["policy"] = {"launches": 1 + w.T, "ms": ms["policy"]}
    out["sum_ms"] = sum(v for k, v in ms.items())
    return out


def run_e2e(args, pl, w, dev, stream, world, policy_pass=None, policy_step=None):
    """Same pass through the C ABI with pinned host inputs: features and text
    copied in, every step's logits read from pinned host memory, committed
    tokens copied out.

    Mode "staged" (default): on a second stream, davet_stage_masked_rows
    copies the rows of step t's logits that were still masked after step t-2
    (a superset of the rows step t reads) from pinned host memory into a ring
    of three device buffers, overlapping the kernels of step t-1; step t's
    unmasking reads the staged rows.  Mode "mapped": the unmasking kernel
    reads each step's logits straight from pinned host memory (only rows still
    masked cross the host link), in line with the step's other kernels.  Mode
    "copy": every step's full logits are copied on the second stream, the copy
    for step t+1 overlapping the kernels of step t.  The timed region spans
    both streams; events order them."""
    import torch

    from paper_2608_01821_gb300 import workloads
    feats = [workloads.features(w, b).pin_memory() for b in range(w.batch)]
    text = workloads.text_rows(w).pin_memory()
    scores = ([workloads.token_scores(w, b).pin_memory() for b in range(w.batch)] if pl.realizer == "prune"
              else None)
    P = 4
    host_logits = [workloads.logits(w, t).pin_memory() for t in range(P)]
    NB = 3
    mode = getattr(args, "e2e_mode", "staged")
    mapped = mode == "mapped"
    dev_logits = [] if mapped else [torch.empty((w.total_resp, w.V), dtype=torch.bfloat16, device=dev)
                                    for _ in range(NB)]
    tokens_host = torch.empty(w.total_resp, dtype=torch.int32).pin_memory()
    if mode == "mapped":
        logit_rows = sum(w.masked_rows(t) for t in range(w.T))
    elif mode == "staged":
        logit_rows = sum(w.masked_rows(max(t - 1, 0)) for t in range(w.T))
    else:
        logit_rows = w.T * w.total_resp
    h2d = sum(f.numel() * 2 for f in feats) + text.numel() * 2 + logit_rows * w.V * 2
    if scores is not None:
        h2d += sum(x.numel() * 4 for x in scores)
    d2h = w.total_resp * 4
    copy_stream = torch.cuda.Stream(device=dev)
    ready = [torch.cuda.Event() for _ in range(NB)]
    free = [torch.cuda.Event() for _ in range(NB)]
    pass_start = torch.cuda.Event()

    def issue_copy(t):
        slot = t % NB
        with torch.cuda.stream(copy_stream):
            if t >= NB:
                copy_stream.wait_event(free[slot])
            dev_logits[slot].copy_(host_logits[t % P], non_blocking=True)
            ready[slot].record(copy_stream)

    def one_mapped():
        pl.reset_state()
        pl.load_inputs(feats, text, non_blocking=True, scores=scores)
        pl.build_pyramids()
        if policy_pass:
            policy_pass()
        for t in range(w.T):
            if policy_step:
                policy_step(t)
            pl.step(t, host_logits[t % P])
        tokens_host.copy_(pl.tokens, non_blocking=True)

    def one_copy():
        pass_start.record(stream)
        copy_stream.wait_event(pass_start)  # no copy starts before the pass (or under the previous one)
        for t in range(min(NB, w.T)):
            issue_copy(t)
        pl.reset_state()
        pl.load_inputs(feats, text, non_blocking=True, scores=scores)
        pl.build_pyramids()
        if policy_pass:
            policy_pass()
        for t in range(w.T):
            slot = t % NB
            stream.wait_event(ready[slot])
            if policy_step:
                policy_step(t)
            pl.step(t, dev_logits[slot])
            free[slot].record(stream)
            if t + NB < w.T:
                issue_copy(t + NB)
        tokens_host.copy_(pl.tokens, non_blocking=True)

    lib = pl.lib
    reset_done = torch.cuda.Event()
    step_done = [torch.cuda.Event() for _ in range(NB)]

    def issue_stage(t):
        # rows masked now (after step t-2's commits, or all at the start of the pass)
        with torch.cuda.stream(copy_stream):
            lib.davet_stage_masked_rows(host_logits[t % P], w.V, pl.masked, w.total_resp, dev_logits[t % NB],
                                        copy_stream)
            ready[t % NB].record(copy_stream)

    def one_staged():
        pl.reset_state()
        reset_done.record(stream)
        copy_stream.wait_event(reset_done)
        for t in range(min(2, w.T)):
            issue_stage(t)
        pl.load_inputs(feats, text, non_blocking=True, scores=scores)
        pl.build_pyramids()
        if policy_pass:
            policy_pass()
        for t in range(w.T):
            slot = t % NB
            stream.wait_event(ready[slot])
            if policy_step:
                policy_step(t)
            pl.step(t, dev_logits[slot])
            step_done[slot].record(stream)
            if t + 2 < w.T:
                # step t's commits are done and step t-1 no longer reads slot (t+2) % 3
                copy_stream.wait_event(step_done[slot])
                issue_stage(t + 2)
        tokens_host.copy_(pl.tokens, non_blocking=True)

    one = {"mapped": one_mapped, "copy": one_copy, "staged": one_staged}[mode]
    with torch.cuda.stream(stream):
        one()
    torch.cuda.synchronize()
    n = max(1, min(args.steps, 5))
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    with torch.cuda.stream(stream):
        s.record(stream)
        for _ in range(n):
            one()
        e.record(stream)
    torch.cuda.synchronize()
    t = allreduce_max(s.elapsed_time(e) / 1e3, world, dev)
    return {"value": round(w.T * n * world / t, 3), "unit": "denoising steps/s",
            "h2d_bytes_per_step": int(round(h2d / w.T)), "d2h_bytes_per_step": int(round(d2h / w.T)),
            "h2d_bytes_per_pass": int(h2d), "d2h_bytes_per_pass": int(d2h), "passes": n, "mode": mode,
            "h2d_GBps": round(h2d * n / t / 1e9, 1)}


# ----------------------------------------------------------- CPU oracle
ATTN_SAMPLE_ITEMS = 32768


def _to_bf16_bits(x):
    """Round an fp64 array to bf16 (nearest even) and return its bits."""
    import numpy as np
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x)).float().to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _sampled_attention_time(oracle, packed, cu, w):
    """Oracle attention time for the whole step, from at most
    ATTN_SAMPLE_ITEMS (row, head) outputs spread uniformly over the rows."""
    import numpy as np
    N = int(cu[-1])
    items = N * w.H
    n = min(items, ATTN_SAMPLE_ITEMS)
    idx = np.linspace(0, items - 1, n).astype(np.int64)
    rows, heads = idx // w.H, (idx % w.H).astype(np.int32)
    t0 = time.perf_counter()
    oracle.attention_rows(packed, cu, w.H, w.D, w.scale, rows, heads)
    dt = time.perf_counter() - t0
    return dt, dt * items / n

def oracle_sample(w, budget_s=20.0):
    """Times the fp64 oracle on a bounded sample of the workload and
    extrapolates to the whole pass: the pyramid of the first request (scaled
    to every request by tile count), then for each distinct scheduled view
    combination (most frequent first, until the budget is spent) the gather
    and the attention on at most ATTN_SAMPLE_ITEMS (row, head) outputs
    (scaled by the output count), and the unmasking of the first step (every
    answer row masked), scaled to each step by its masked-row count.
    Returns (denoising steps/s, cores, description, seconds, parts)."""
    import numpy as np

    import oracle
    from paper_2608_01821_gb300 import workloads
    cores = oracle.max_threads()
    text = workloads.text_rows(w)
    b0 = next(b for b in range(w.batch) if w.tiles[b] > 0)
    f0 = workloads.features(w, b0)
    t0 = time.perf_counter()
    ref = oracle.pyramid(f0, w.tiles[b0], w.grid, w.n_levels, w.C)
    t_pyr1 = time.perf_counter() - t0
    pyr0 = _to_bf16_bits(ref)
    # the other requests' pyramids are not timed: their rows only feed the
    # gather, whose cost does not depend on the values
    pyr = []
    for b in range(w.batch):
        if b == b0 or w.tiles[b] == w.tiles[b0]:
            pyr.append(pyr0)
        else:
            pyr.append(np.zeros((w.pyramid_rows(b), w.C), np.uint16))
    t_pyr = t_pyr1 * sum(w.tiles) / w.tiles[b0]
    lg = workloads.logits(w, 0)
    t2 = time.perf_counter()
    masked = np.ones(w.total_resp, np.uint8)
    tokens = np.full(w.total_resp, -1, np.int32)
    argmax = np.full(w.total_resp, -1, np.int32)
    oracle.unmask(lg, w.V, w.cu_resp(), w.k, masked, tokens, argmax)
    t_unmask0 = time.perf_counter() - t2
    spent = t_pyr1 + t_unmask0
    keys = {}
    for t in range(w.T):
        keys.setdefault(tuple(int(x) for x in w.schedule[t]), []).append(t)
    per_key = {}
    for key, ts in sorted(keys.items(), key=lambda kv: -len(kv[1])):
        t = ts[0]
        t1 = time.perf_counter()
        packed, cu = oracle.gather(pyr, w.tiles, text, w.text_offsets(), w.prompt, w.resp, w.schedule[t], w.grid,
                                   w.n_levels, w.C)
        t_gather = time.perf_counter() - t1
        t_attn_spent, t_attn = _sampled_attention_time(oracle, packed, cu, w)
        per_key[key] = t_gather + t_attn
        spent += t_gather + t_attn_spent
        if spent > budget_s:
            break
    mean_dt = sum(per_key.values()) / len(per_key)
    unmask_total = sum(t_unmask0 * w.masked_rows(t) / max(w.total_resp, 1) for t in range(w.T))
    total = t_pyr + sum(per_key.get(k, mean_dt) * len(ts) for k, ts in keys.items()) + unmask_total
    desc = (f"fp64 oracle: pyramid of request {b0} (scaled to all {sum(w.tiles)} tiles), one gather + attention "
            f"for {len(per_key)} of {len(keys)} distinct view combinations (attention on at most "
            f"{ATTN_SAMPLE_ITEMS} sampled (row, head) outputs, scaled by the output count), the unmasking of the "
            f"first step (scaled by each step's masked rows); extrapolated over the {w.T}-step schedule")
    parts = {"pyramid_one_request_s": round(t_pyr1, 3), "unmask_first_step_s": round(t_unmask0, 3),
             "gather_plus_attention_s": {"/".join(map(str, k[:4])) + ("..." if len(k) > 4 else ""): round(v, 3)
                                         for k, v in per_key.items()}}
    return w.T / total, cores, desc, spent, parts


def backbone_oracle_sample(w, n_layers: int):
    """The fp64 layer oracle on one layer of one step of the workload (its
    first step's sequence), scaled to n_layers and the whole schedule by the
    steps' GEMM work.  Returns (denoising steps/s, cores, description, s)."""
    import numpy as np

    import oracle
    from oracle import layer as L
    cores = oracle.max_threads()
    C = w.H * w.D
    F = 3 * C
    rng = np.random.default_rng(0)
    lens = w.step_lengths(0)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    x = rng.standard_normal((int(cu[-1]), C))
    wts = dict(g1=np.ones(C), wq=rng.standard_normal((C, C)) / 64, wk=rng.standard_normal((C, C)) / 64,
               wv=rng.standard_normal((C, C)) / 64, wo=rng.standard_normal((C, C)) / 64, g2=np.ones(C),
               wg=rng.standard_normal((F, C)) / 64, wu=rng.standard_normal((F, C)) / 64,
               wd=rng.standard_normal((C, F)) / 110)
    t0 = time.perf_counter()
    L.layer(x, wts, cu, w.H, w.D, 500000.0, 1e-5)
    dt = time.perf_counter() - t0
    rows0 = float(cu[-1])
    per_step = [dt * n_layers * sum(w.step_lengths(t)) / rows0 for t in range(w.T)]
    desc = (f"fp64 layer oracle (numpy): one layer of step 0 ({int(rows0)} rows) timed, scaled by rows to "
            f"{n_layers} layers and the {w.T}-step schedule; LM head and unmasking not included")
    return w.T / sum(per_step), cores, desc, dt


def run_reference(args, rank, world):
    """The oracle arm: each timed step is one denoising step of the workload
    run by the fp64 CPU oracle (levels taken in schedule order, cycling
    through a bounded set of distinct levels); the pyramid build is timed
    once and amortized over the schedule."""
    import numpy as np

    import oracle
    from paper_2608_01821_gb300 import workloads
    if rank != 0:
        return None
    w = workloads.make(args.config)
    feats = [workloads.features(w, b) for b in range(w.batch)]
    text = workloads.text_rows(w)
    t0 = time.perf_counter()
    pyr = []
    for b in range(w.batch):
        ref = oracle.pyramid(feats[b], w.tiles[b], w.grid, w.n_levels, w.C)
        pyr.append(_to_bf16_bits(ref))
    t_pyr = time.perf_counter() - t0
    lg = workloads.logits(w, 0)
    # distinct step levels, coarsest first so a bounded run covers cheap and costly steps
    order = list(range(w.T))
    picks = order[:: max(1, w.T // max(1, args.steps + args.warmup))]

    def step(t):
        packed, cu = oracle.gather(pyr, w.tiles, text, w.text_offsets(), w.prompt, w.resp, w.schedule[t], w.grid,
                                   w.n_levels, w.C)
        if int(cu[-1]) * w.H <= ATTN_SAMPLE_ITEMS or w.name == "tiny":
            oracle.attention(packed, cu, w.H, w.D, w.scale)
        else:
            # bounded sample: a spread of (row, head) outputs, timed and scaled to the full step
            actual, scaled = _sampled_attention_time(oracle, packed, cu, w)
            extra.append(scaled - actual)
        masked = np.ones(w.total_resp, np.uint8)
        tokens = np.full(w.total_resp, -1, np.int32)
        argmax = np.full(w.total_resp, -1, np.int32)
        oracle.unmask(lg, w.V, w.cu_resp(), w.k, masked, tokens, argmax)

    extra = []
    for i in range(args.warmup):
        step(picks[i % len(picks)])
    extra.clear()
    t1 = time.perf_counter()
    for i in range(args.steps):
        step(picks[(args.warmup + i) % len(picks)])
    # the sampled attention ran inside the loop: add what the unsampled outputs would take
    dt = time.perf_counter() - t1 + t_pyr * args.steps / w.T + sum(extra)
    value = args.steps / dt
    cores = oracle.max_threads()
    sample = (f"{args.steps} denoising steps of workload '{w.name}' at schedule positions spread over the "
              f"{w.T}-step schedule, fp64 oracle, plus the pyramid build amortized over the schedule")
    return {"metric": METRIC, "value": round(value, 5), "unit": "denoising steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt / args.steps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded N(0,1) features/text, N(0,2) logits; no weights)",
            "config": workload_config(w), "impl": "reference",
            "cpu_baseline": {"value": round(value, 5), "unit": "denoising steps/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 5), "unit": "denoising steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def run_profile(args):
    """Minimal launch sequence for profilers: the workload's inputs for one
    step and `--steps` launches of one kernel (after `--warmup` launches).
    `--profile-view V` runs the step at view V for every request.  With
    `--profile-time`, the `--steps` launches are then captured as one CUDA
    graph and replayed three times (an L2 flush before each replay, not
    timed); the line reports the best replay's time per launch."""
    import torch

    from paper_2608_01821_gb300 import davet, workloads
    from paper_2608_01821_gb300.pipeline import Pipeline
    dev = torch.device("cuda", 0)
    lib = davet.load()
    w = workloads.make(args.config)
    realizer = getattr(args, "realizer", "pool")
    pl = Pipeline(w, dev, lib, realizer=realizer)
    pl.load_inputs([workloads.features(w, b) for b in range(w.batch)], workloads.text_rows(w),
                   scores=[workloads.token_scores(w, b) for b in range(w.batch)] if realizer == "prune" else None)
    t = args.profile_step
    if args.profile_view is not None:
        if not 0 <= args.profile_view < w.n_levels + (1 if w.mixed else 0):
            raise SystemExit(f"--profile-view {args.profile_view}: no such view in workload {w.name}")
        pl.schedule[t].fill_(args.profile_view)
    lg = workloads.logits_device(w, t, dev)
    pl.build_pyramids()
    pl.gather(t)
    fn = {"pyramid": pl.build_pyramids, "gather": lambda: pl.gather(t), "attention": pl.attention,
          "view_attention": lambda: pl.view_attention(t),
          "unmask": lambda: (pl.reset_state(), pl.unmask(t, lg))}[args.profile]
    for _ in range(args.warmup + args.steps):
        fn()
    torch.cuda.synchronize()
    us = None
    if args.profile_time and args.profile != "unmask":
        stream = torch.cuda.Stream(device=dev)
        flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            fn()  # first use on this stream, outside the capture
        torch.cuda.synchronize()
        with torch.cuda.graph(graph, stream=stream):
            for _ in range(args.steps):
                fn()
        best = None
        for rep in range(3):
            with torch.cuda.stream(stream):
                flush.fill_(rep)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                graph.replay()
                e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            best = ms if best is None else min(best, ms)
        us = round(best * 1000.0 / max(args.steps, 1), 2)
    st, flags = lib.davet_device_status()
    views = sorted(set(int(v) for v in pl.schedule[t].cpu().tolist()))
    print(json.dumps({"profile": args.profile, "workload": w.name, "step": t, "views": views, "status": st,
                      "flags": flags, "us_per_launch": us}))
    return 0 if st == 0 else 1


# ------------------------------------------------------------ dist glue
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


_pg = {"init": False}


def init_dist(world, backend):
    if world > 1 and not _pg["init"]:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)
        _pg["init"] = True


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def whole_job_rate(units_per_rank: float, world: int, max_seconds: float) -> float:
    """Units processed by all ranks divided by the slowest rank's time."""
    return units_per_rank * world / max_seconds


def allreduce_max(x: float, world: int, device) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--logit-pool", type=int, default=0, help="cap on distinct device logit buffers")
    ap.add_argument("--e2e-mode", choices=["staged", "mapped", "copy"], default="staged",
                    help="e2e logits: masked rows staged on a second stream one step ahead, read from pinned host "
                         "memory by the unmasking kernel, or full logits copied to the device")
    ap.add_argument("--unfused", action="store_true",
                    help="pack each step with davet_gather_view, then davet_step_attention (instead of the fused call)")
    ap.add_argument("--profile", choices=["pyramid", "gather", "attention", "view_attention", "unmask"], default=None,
                    help="only set up one step and launch this kernel --steps times (for ncu captures)")
    ap.add_argument("--profile-step", type=int, default=0)
    ap.add_argument("--profile-view", type=int, default=None,
                    help="with --profile: run the step at this view for every request")
    ap.add_argument("--profile-time", action="store_true",
                    help="with --profile: time the --steps launches as one CUDA graph (best of 3 replays)")
    ap.add_argument("--policy", action="store_true",
                    help="choose every step's view with the closed-loop allocation policy on the device")
    ap.add_argument("--schedule", choices=["workload", "high", "mid", "low"], default="workload",
                    help="the level schedule without --policy: the workload's own, or one static view for every step")
    ap.add_argument("--orientation", choices=["early", "late"], default="early")
    ap.add_argument("--budget", type=float, default=0.75, help="average budget B")
    ap.add_argument("--rho", type=float, default=0.20)
    ap.add_argument("--alpha", type=float, default=1.0)
    ap.add_argument("--uniform-demand", action="store_true",
                    help="with --policy: d(o) = 1 for every request instead of the Table A prior")
    ap.add_argument("--model", choices=["core", "full"], default="core",
                    help="core: the step-conditioning path (attention core); full: every step runs --layers "
                         "synthetic-weight backbone layers and the LM head")
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--realizer", choices=["pool", "prune", "merge"], default="pool",
                    help="evidence realizer of the view blocks (Sec. 4.3): pooling (default), pruning or merging")
    args = ap.parse_args(argv)
    rank, world, local = dist_env()
    if args.profile:
        return run_profile(args)
    if args.impl == "reference":
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out), flush=True)
        return 0
    init_dist(world, "nccl")
    if args.model == "full":
        out = run_backbone(args, rank, world, local)
        if rank == 0:
            if not args.no_cpu_baseline:
                from paper_2608_01821_gb300 import workloads
                v, cores, desc, spent = backbone_oracle_sample(workloads.make(args.config), args.layers)
                out["cpu_baseline"] = {"value": round(v, 6), "unit": "denoising steps/s", "cores": cores,
                                       "kind": "oracle", "sample": desc, "cpu_seconds": round(spent, 1)}
            print(json.dumps(out), flush=True)
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return 0
    out = run_ours(args, rank, world, local)
    if rank == 0:
        if not args.no_cpu_baseline:
            from paper_2608_01821_gb300 import workloads
            v, cores, desc, spent, parts = oracle_sample(workloads.make(args.config))
            out["cpu_baseline"] = {"value": round(v, 5), "unit": "denoising steps/s", "cores": cores,
                                   "kind": "oracle", "sample": desc, "cpu_seconds": round(spent, 1),
                                   "parts": parts}
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
