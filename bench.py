#!/usr/bin/env python3
"""Benchmark of the GB300 PCED decode step.

Metric: PCED decode tokens/s (one token per query per step) on the
Llama-3-8B-shaped workload with N=8 document experts + amateur (and, as a
secondary line item, N=32 ragged experts), plus the achieved HBM bandwidth of
the dominant kernel against the measured copy peak.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun each rank runs an independent replica of the workload on its
own GPU (the queries of PCED never interact), timed between barriers; rank 0
prints one JSON line with the whole-job throughput.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "PCED decode tokens/s at N=8/32 experts; achieved HBM GB/s vs ~8 TB/s peak"
UNIT = "tokens/s"
NOMINAL_HBM_GBS = 8000.0
GRAPH_STEPS = 8  # decode steps per captured CUDA graph (at most)


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=64)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="llama8")
    p.add_argument("--layers", type=int, default=0,
                   help="override the workload's layer count (small cases for multi-pass ncu captures; "
                        "not the headline configuration)")
    p.add_argument("--secondary", default="llama32", help="second workload timed on the value path ('none' skips)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--paged", type=int, default=0,
                   help="store the caches paged with blocks of this many rows (a multiple of 64; 0: slabs)")
    p.add_argument("--rope-theta", type=float, default=0.0,
                   help="rotate queries and appended keys with this rotary base (0: none)")
    p.add_argument("--aggregation", choices=["max", "moe", "poe"], default="max",
                   help="how experts are combined: Eq. 3's max (default) or the MoE / PoE variants")
    p.add_argument("--raw-logits", action="store_true", help="Eq. 2 on raw logits instead of log-probabilities")
    p.add_argument("--no-dynamic-beta", action="store_true",
                   help="skip timing the first step with dynamic contrast strength")
    p.add_argument("--profile-steps", type=int, default=4, help="replays with per-launch events (roofline)")
    return p.parse_args()


# ----------------------------------------------------------------------- dist
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


class Dist:
    def __init__(self, world: int, local_rank: int):
        import torch
        self.world = world
        self.pg = None
        if world > 1:
            import torch.distributed as td
            td.init_process_group("gloo")
            self.td = td

    def barrier(self):
        if self.world > 1:
            self.td.barrier()

    def max(self, x: float) -> float:
        if self.world == 1:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64)
        self.td.all_reduce(t, op=self.td.ReduceOp.MAX)
        return float(t.item())

    def sum(self, x: float) -> float:
        if self.world == 1:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64)
        self.td.all_reduce(t, op=self.td.ReduceOp.SUM)
        return float(t.item())

    def close(self):
        if self.world > 1:
            self.td.destroy_process_group()


# --------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.3)
        self.proc.terminate()
        self.proc.wait()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) != 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[2], parts[3], parts[4:]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[4]) if v.lower() == "active"})
        busy = [r[0] for r in rows if r[0] > 0.5 * r[1]] or [r[0] for r in rows]
        return {"sm_mhz": statistics.median(busy), "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows)}


# ---------------------------------------------------------------------- utils
def measured_peaks() -> dict:
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        return {}


def source_hash(files) -> str:
    h = hashlib.sha256()
    for f in files:
        h.update(open(os.path.join(ROOT, f), "rb").read())
    return h.hexdigest()[:16]


KERNEL_SOURCES = {
    "attention": ["paper_2601_08670_gb300/csrc/attention.cu", "paper_2601_08670_gb300/csrc/attention.cuh",
                   "paper_2601_08670_gb300/csrc/common.cuh"],
    "lm_head": ["paper_2601_08670_gb300/csrc/lm_head.cu", "paper_2601_08670_gb300/csrc/lm_head.cuh",
                "paper_2601_08670_gb300/csrc/common.cuh", "paper_2601_08670_gb300/csrc/select_key.cuh"],
}


def ncu_traffic(kind: str, workload: str):
    """DRAM bytes per launch of `kind` from the committed ncu summary, or None
    when missing or taken on a different version of the kernel source.  A
    capture of the same shapes with fewer layers is scaled by the layer count
    (the attention launch streams every layer once)."""
    import synth
    try:
        rec = json.load(open(os.path.join(ROOT, "profiles", "ncu_traffic.json")))[kind]
    except (OSError, ValueError, KeyError):
        return None
    if rec.get("source_hash") != source_hash(KERNEL_SOURCES[kind]):
        return None
    got = rec.get("dram_bytes_per_launch")
    if rec.get("workload") == workload or got is None:
        return got
    wc, w = synth.get(rec["workload"]), synth.get(workload)
    if kind == "attention" and replace_layers(wc, w.L) == replace_layers(w, w.L):
        return got * w.L / wc.L
    if kind == "lm_head" and (wc.S, wc.d, wc.V) == (w.S, w.d, w.V):
        return got
    return None


def replace_layers(w, L):
    from dataclasses import replace
    return replace(w, L=L, name=None, steps=None, description=None) if w else w


def step_bytes(w, lens_after) -> int:
    import synth
    return synth.algorithmic_bytes_per_step(w, lens_after)


# --------------------------------------------------------------- our GPU path
AGGREGATIONS = {"max": 0, "moe": 1, "poe": 2}


def build_decoder(w, dev, capacity_steps, paged=0, rope_theta=0.0, aggregation="max", raw_logits=False):
    import paper_2601_08670_gb300 as pced
    import synth
    t = synth.device_inputs(w, dev, extra_steps=capacity_steps, paged=paged)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=capacity_steps, bos=w.bos, rope_theta=rope_theta,
                                   aggregation=AGGREGATIONS[aggregation], score_mode=1 if raw_logits else 0)
    return dec, t


def steps_per_graph(steps, most=GRAPH_STEPS):
    """Decode steps captured in one CUDA graph: the largest divisor of the
    timed step count up to `most`, so the timed region is exactly `steps`."""
    return max(k for k in range(1, most + 1) if steps % k == 0)


def graph_capacity(steps, warmup):
    """Steps time_graph runs: eager warm-up, warm-up graph replays, timed steps."""
    k = steps_per_graph(steps)
    return max(1, warmup) + k * (-(-warmup // k)) + steps


def time_graph(dec, dist, steps, warmup, dev, clocks=None):
    """Returns (elapsed ms of `steps` decode steps replayed from CUDA graphs of
    steps_per_graph(steps) steps each, lengths before the timed region, the
    graph, its stream, the clock record, the median ms per step over the
    graphs).  Every
    step in a graph is a full pced_step; several per graph only save the
    launch of a graph between steps, as a serving loop would."""
    import torch
    s = torch.cuda.Stream(device=dev)
    for _ in range(max(1, warmup)):  # eager warm-up (also configures the kernels)
        dec.step()
    torch.cuda.synchronize(dev)
    k = steps_per_graph(steps)
    s.wait_stream(torch.cuda.current_stream(dev))
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for _ in range(k):
            dec.step()
    # capture does not execute: state is unchanged
    with torch.cuda.stream(s):
        for _ in range(-(-warmup // k)):
            g.replay()
    torch.cuda.synchronize(dev)
    lens0 = dec.seq_len.cpu().numpy().copy()
    # an event after every graph: the total is the metric, the median graph
    # gives the median step time as well
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps // k + 1)]
    if clocks:
        clocks.start()
    dist.barrier()
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(s):
        ev[0].record(s)
        for i in range(steps // k):
            g.replay()
            ev[i + 1].record(s)
    torch.cuda.synchronize(dev)
    dist.barrier()
    clk = clocks.stop() if clocks else None
    med = statistics.median(ev[i].elapsed_time(ev[i + 1]) for i in range(steps // k)) / k
    return ev[0].elapsed_time(ev[-1]), lens0, g, s, clk, med


def profile_launches(dec, g_unused, dev, reps):
    """Per-launch device times from stage events recorded inside a captured step."""
    import torch
    kinds = dec.launch_kinds()
    n = len(kinds)
    events = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    dec.set_stage_events(events)
    s = torch.cuda.Stream(device=dev)
    s.wait_stream(torch.cuda.current_stream(dev))
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        dec.step()
    dec.set_stage_events(None)
    per = [[] for _ in range(n)]
    lens = []
    for _ in range(reps):
        lens.append(dec.seq_len.cpu().numpy() + 1)
        with torch.cuda.stream(s):
            g.replay()
        torch.cuda.synchronize(dev)
        for i in range(n):
            per[i].append(events[i].elapsed_time(events[i + 1]))
    return kinds, per, lens


def run_e2e(dec, w, dev, steps):
    """End to end through the C ABI with host buffers (pced_step_host_io), as a
    serving loop runs it: every step uploads beta and r from page-locked host
    memory, runs the decode step and copies the chosen token / expert / score
    back; the host reads each step's choice while the next step runs (two
    host slots used in turn).  Timed twice by the wall clock over `steps`
    steps: with one captured CUDA graph of the call per slot (a replay is one
    step with its copies) and with eager calls.  Returns both times, the
    bytes copied per step and whether the tokens read on the host are the
    device history."""
    import torch
    B = w.B
    # beta and r side by side, and the choice as one [3, B] block, as on the
    # device: one upload and one read-back per step
    beta_r = torch.stack([dec.beta.cpu(), dec.r.cpu()]).pin_memory()
    beta_h, r_h = beta_r[0], beta_r[1]
    slots = [dict(zip(("token", "expert", "score"), dec.choice_buffers())) for _ in range(2)]
    graphs = [dec.capture_host_io(beta_h, r_h, **sl) for sl in slots]
    events = [torch.cuda.Event(), torch.cuda.Event()]

    def loop(run):
        run(0)  # warm-up steps (a graph's first replay also uploads it)
        run(1)
        torch.cuda.synchronize(dev)
        t_first = int(dec.step_t.item())
        got = []
        t0 = time.perf_counter()
        for i in range(steps + 1):
            if i < steps:
                run(i % 2)
                events[i % 2].record()
            if i:  # the previous step's choice, read while this one runs
                events[(i - 1) % 2].synchronize()
                sl = slots[(i - 1) % 2]
                got.append((sl["token"].tolist(), sl["expert"].tolist(), sl["score"].tolist()))
        el = time.perf_counter() - t0
        hist = dec.history[:, t_first:t_first + steps].cpu().T.tolist()
        return el, [g[0] for g in got] == hist

    el_graph, ok_graph = loop(lambda k: graphs[k].replay())
    el_eager, ok_eager = loop(lambda k: dec.step_host_io(beta_h, r_h, **slots[k]))
    del graphs
    h2d = beta_h.numel() * 4 + r_h.numel() * 4
    d2h = B * (4 + 4 + 4)
    return el_graph, el_eager, h2d, d2h, ok_graph and ok_eager


def time_dynamic_beta_first_step(w, dev, reps=3):
    """Device time of the first step of a decode with dynamic contrast strength,
    of the regular step after it, and of the first step of a decode with a
    fixed beta (eager calls, CUDA events), median of `reps` fresh decoders
    each.  The extra cost of dynamic beta is the difference of the two first
    steps: both start on freshly written caches, which the second step of a
    decode does not."""
    import torch
    import paper_2601_08670_gb300 as pced
    import synth
    S = w.B * (w.N + 1)
    pced.adacad_beta(torch.zeros((S, w.V), dtype=torch.float32, device=dev), w.B, w.N)  # load the kernel
    first, regular, fixed_first, status = [], [], [], 0
    for _ in range(reps):
        for dyn in (True, False):
            t = synth.device_inputs(w, dev, extra_steps=4)
            dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
            dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=4, bos=w.bos, dynamic_beta=dyn)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            torch.cuda.synchronize()
            ev[0].record()
            dec.step()
            ev[1].record()
            dec.step()
            ev[2].record()
            torch.cuda.synchronize()
            if dyn:
                first.append(ev[0].elapsed_time(ev[1]) * 1e3)
                regular.append(ev[1].elapsed_time(ev[2]) * 1e3)
            else:
                fixed_first.append(ev[0].elapsed_time(ev[1]) * 1e3)
            status |= dec.status()
            del dec, t
    f, r, ff = statistics.median(first), statistics.median(regular), statistics.median(fixed_first)
    return {"first_step_us": f, "fixed_beta_first_step_us": ff, "next_step_us": r, "extra_us": f - ff,
            "extra_vs_next_step_us": f - r, "reps": reps,
            "path": "pced_step with beta_from_step: the LM head writes raw logits and per-tile log-sum-exp records, "
                    "lse_finalize, the beta kernel, then Eq. 3 over the stored logits with that beta "
                    "(no second LM-head pass)"}, status


def cpu_baseline(w, budget_s=20.0, max_steps=3):
    import oracle
    from oracle.run import OracleRun
    run = OracleRun(w)
    t0 = time.perf_counter()
    n = 0
    while n < max_steps:
        run.step()
        n += 1
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    return {"value": w.B * n / el, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
            "sample": f"{n} full decode step(s) of the {w.name} workload (all {w.S} sequences, {w.L} layers, "
                      f"vocab {w.V}), fp64 scalar C, caches generated before timing",
            "ms_per_step": 1e3 * el / n}


def workload_config(w, graph=True, paged=0, rope_theta=0.0, aggregation="max", raw_logits=False):
    import synth
    bl = synth.base_lengths(w)
    return {"workload": f"{w.name}: {w.description}", "B": w.B, "N": w.N, "S": w.S, "L": w.L, "Hq": w.Hq,
            "Hkv": w.Hkv, "D": w.D, "V": w.V, "kv_tokens_at_start": int(bl.sum()), "beta": w.beta,
            "gamma": w.gamma, "seed": w.seed,
            "l2": (f"no flush: every step reads {step_bytes(w, bl + 1) / 1e9:.2f} GB, larger than the 129 MB L2"
                   if step_bytes(w, bl + 1) > 129e6 else "step working set fits in L2 (not a bandwidth workload)"),
            "cuda_graph": graph, "parallelism": "one independent replica per GPU",
            "kv_layout": f"paged, {paged}-row blocks in a shuffled pool" if paged else "one slab per (sequence, kv-head)",
            "rotary": f"queries and appended keys rotated, base {rope_theta:g}" if rope_theta > 0 else "none",
            "aggregation": {"max": "max over experts (Eq. 3)", "moe": "mixture of experts (weighted sum)",
                            "poe": "product of experts (weighted product)"}[aggregation],
            "scores": "raw logits" if raw_logits else "log-probabilities"}


def run_ours(args):
    import torch
    import synth
    rank, world, local = dist_env()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    dist = Dist(world, local)
    peaks = measured_peaks()
    hbm_peak = peaks.get("hbm_gbs")
    w = synth.get(args.workload, **({"L": args.layers} if args.layers > 0 else {}))
    e2e_steps = 0 if args.no_e2e else args.steps
    cap_steps = graph_capacity(args.steps, args.warmup) + 1 + args.profile_steps + 2
    dec, _ = build_decoder(w, dev, cap_steps, paged=args.paged, rope_theta=args.rope_theta,
                           aggregation=args.aggregation, raw_logits=args.raw_logits)
    launches = dec.launches_per_step()

    clocks = ClockSampler(local)
    ms, lens0, g, s, clk, med = time_graph(dec, dist, args.steps, args.warmup, dev, clocks)
    ms = dist.max(ms)
    status = dec.status()
    # algorithmic bytes of every timed step (lengths grow by one per step)
    tot_bytes = sum(step_bytes(w, lens0 + 1 + i) for i in range(args.steps))
    tokens = dist.sum(w.B * args.steps)
    value = tokens / (ms / 1e3)
    ms_step = ms / args.steps

    # roofline of the dominant kernel from per-launch events
    kinds, per, plens = profile_launches(dec, g, dev, args.profile_steps)
    by_kind = {}
    for k, times in zip(kinds, per):
        d = by_kind.setdefault(k, {"launches_per_step": 0, "ms": []})
        d["launches_per_step"] += 1
        d["ms"].extend(times)
    prof_step_ms = sum(sum(t) for t in per) / args.profile_steps
    kernels = {k: {"launches_per_step": d["launches_per_step"],
                   "us_per_step": 1e3 * sum(d["ms"]) / args.profile_steps,
                   "share": sum(d["ms"]) / args.profile_steps / prof_step_ms} for k, d in by_kind.items()}
    # attention: one launch runs all L layers; its algorithmic bytes are the
    # K and V rows of every live position of every layer (at the profiled lengths)
    att_bytes = [float(sum(l.astype("int64")) * 2 * w.Hkv * w.D * 2 * w.L) for l in plens]
    att_ms = per[kinds.index("attention")]
    att_gbs = statistics.mean(b / (t / 1e3) / 1e9 for b, t in zip(att_bytes, att_ms))
    lm_ms = statistics.mean(per[kinds.index("lm_head")])
    lm_bytes = w.V * w.d * 2
    lm_gbs = lm_bytes / (lm_ms / 1e3) / 1e9
    dominant = max(("attention", "lm_head"), key=lambda k: kernels[k]["share"])
    if dominant == "attention":
        dom = {"kernel": f"attention (att_step_kernel<{w.D}>: embedding + {w.L} layers in one cooperative launch)",
               "achieved": att_gbs,
               "algorithmic_bytes_per_launch": statistics.mean(att_bytes),
               "avg_launch_us": 1e3 * statistics.mean(att_ms)}
    else:
        dom = {"kernel": "lm_head (lm_head_kernel)", "achieved": lm_gbs, "algorithmic_bytes_per_launch": lm_bytes,
               "avg_launch_us": 1e3 * lm_ms}
    roofline = {"bound": "hbm", **dom, "peak": hbm_peak, "unit": "GB/s",
                "frac": dom["achieved"] / hbm_peak if hbm_peak else None,
                "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured)" if hbm_peak else None,
                "traffic": ncu_traffic(dominant, w.name),
                "lm_head": {"achieved": lm_gbs, "frac": lm_gbs / hbm_peak if hbm_peak else None,
                            "avg_launch_us": 1e3 * lm_ms,
                            "tensor_tflops": 2.0 * w.S * w.V * w.d / (lm_ms / 1e3) / 1e12},
                "kernels": kernels}

    status |= dec.status()
    del dec, g
    torch.cuda.empty_cache()

    # end to end on a fresh decoder brought to the lengths at which the timed
    # region started, so its steps read the same bytes as the timed ones
    e2e = None
    if e2e_steps:
        pre = graph_capacity(args.steps, args.warmup) - args.steps
        dec, _ = build_decoder(w, dev, pre + 2 * (e2e_steps + 2) + 2, paged=args.paged, rope_theta=args.rope_theta,
                               aggregation=args.aggregation, raw_logits=args.raw_logits)
        for _ in range(pre):
            dec.step()
        el, el_eager, h2d, d2h, same = run_e2e(dec, w, dev, e2e_steps)
        el, el_eager = dist.max(el), dist.max(el_eager)
        e2e = {"value": dist.sum(w.B * e2e_steps) / el, "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "steps": e2e_steps,
               "path": "pced_step_host_io (C ABI, host buffers): beta and r uploaded from page-locked host "
                       "memory (one copy), the step, token / expert / score copied back (one copy), one "
                       "captured CUDA graph of the call per step; the host reads each step's choice while the "
                       "next runs; wall clock; a fresh decoder over the timed steps' cache lengths",
               "host_tokens_equal_device_history": same,
               "eager": {"value": dist.sum(w.B * e2e_steps) / el_eager, "unit": UNIT,
                         "path": "the same loop with eager pced_step_host_io calls, after the graph loop "
                                 f"(caches {e2e_steps + 2} rows longer)"}}
        if not same:
            status |= 1 << 16
        status |= dec.status()
        del dec
        torch.cuda.empty_cache()

    # first step with dynamic contrast strength (log-probs materialised, beta
    # from their divergences, then the fused path) against the next, regular step
    dyn = None
    if not args.no_dynamic_beta:
        dyn, st = time_dynamic_beta_first_step(w, dev)
        status |= st
        torch.cuda.empty_cache()

    secondary = None
    if args.secondary != "none":
        w2 = synth.get(args.secondary)
        k2 = min(args.steps, 32)
        dec2, _ = build_decoder(w2, dev, graph_capacity(k2, args.warmup) + 2)
        ms2, l2, g2, s2, _, _ = time_graph(dec2, dist, k2, args.warmup, dev)
        ms2 = dist.max(ms2)
        b2 = sum(step_bytes(w2, l2 + 1 + i) for i in range(k2))
        status |= dec2.status()
        secondary = {"workload": f"{w2.name}: {w2.description}", "value": dist.sum(w2.B * k2) / (ms2 / 1e3),
                     "unit": UNIT, "steps": k2, "ms_per_step": ms2 / k2,
                     "step_hbm_gbs": b2 / (ms2 / 1e3) / 1e9,
                     "frac_of_8tbps": b2 / (ms2 / 1e3) / 1e9 / NOMINAL_HBM_GBS}
        del dec2, g2
        torch.cuda.empty_cache()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w)

    step_gbs = tot_bytes / (ms / 1e3) / 1e9
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "median_ms_per_step": dist.max(med),
            "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded counter-based generator)",
            "config": dict(workload_config(w, paged=args.paged, rope_theta=args.rope_theta,
                                           aggregation=args.aggregation, raw_logits=args.raw_logits),
                           steps_per_graph=steps_per_graph(args.steps)),
            "step_hbm": {"achieved_gbs": step_gbs,
                                                       "frac_of_8tbps": step_gbs / NOMINAL_HBM_GBS,
                                                       "frac_of_measured": step_gbs / hbm_peak if hbm_peak else None,
                                                       "algorithmic_bytes_per_step": tot_bytes / args.steps},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches * args.steps,
            "clocks": clk, "device_status": status, "secondary": secondary, "dynamic_beta_first_step": dyn}
    if rank == 0:
        print(json.dumps(line), flush=True)
    dist.close()
    return 0 if status == 0 else 1


# ----------------------------------------------------------- reference arm
def run_reference(args):
    """The CPU oracle timed as the reference implementation (rank 0 only)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    import synth
    from oracle.run import OracleRun
    w = synth.get(args.workload, **({"L": args.layers} if args.layers > 0 else {}))
    run = OracleRun(w, extra_steps=args.warmup + args.steps + 1)
    t0 = time.perf_counter()
    run.step()
    est = time.perf_counter() - t0
    for _ in range(max(0, min(args.warmup, 1) - 1)):
        run.step()
    budget = 150.0
    k = max(1, min(args.steps, int(budget / max(est, 1e-3))))
    t0 = time.perf_counter()
    for _ in range(k):
        run.step()
    el = time.perf_counter() - t0
    value = w.B * k / el
    sample = (f"{k} of the {args.steps} requested full decode steps of the {w.name} workload (bounded to about "
              f"{budget:.0f} s), fp64 scalar C on the host cores")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": k,
            "warmup": 1, "ms_per_step": 1e3 * el / k, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded counter-based generator)",
            "config": workload_config(w, graph=False),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse_args()
    world = dist_env()[1]
    if args.gpus != world:
        # one rank per GPU comes from the launcher (torchrun); a mismatch
        # would silently time fewer GPUs than asked for
        print(f"bench.py: --gpus {args.gpus} but WORLD_SIZE={world}; launch one rank per GPU with "
              f"python -m torch.distributed.run --nproc-per-node {args.gpus} bench.py --gpus {args.gpus}",
              file=sys.stderr)
        return 2
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
