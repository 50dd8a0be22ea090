#!/usr/bin/env python
"""Benchmark of the fused RoI mask forward + backward on a Qwen2.5-shaped layer set.

One step = roi_mask_fwd over every tensor of the layer set (forward order), then
roi_mask_bwd over every tensor (reverse order), with step-keyed noise (the step
index is the Philox counter word), all on one CUDA stream.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--set qwen2.5-7b] [--nm 2:4] [--tau 1.0]

Under torchrun every rank runs its own full layer set (independent problems, no
collective on the data path: weak scaling); rank 0 prints the max-over-ranks time.
--impl reference times the CPU oracle (the plain statement of the method) on the
host cores instead.
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
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as WL  # noqa: E402

METRIC = "fused RoI mask fwd+bwd groups/s and HBM GB/s (% of GB300 peak), 1 GPU"
FWD_BYTES = 4 + 2 + 2 + 1 / 8     # logits, W in; Wm, hard bits out
BWD_BYTES = 4 + 2 + 2 + 4         # logits, W, dWm in; dlogits out
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=("ours", "reference"), default="ours")
    p.add_argument("--set", default="qwen2.5-7b", choices=sorted(WL.LAYER_SETS))
    p.add_argument("--nm", default="2:4")
    p.add_argument("--tau", type=float, default=None)
    p.add_argument("--e2e-steps", type=int, default=5)
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-configs", action="store_true",
                   help="skip the timed records of the other configurations (default: after the headline)")
    p.add_argument("--layers", type=int, default=None, help="only the first L layers (profiling cases)")
    p.add_argument("--proj", default=None, help="comma-separated projections to keep, e.g. gate")
    p.add_argument("--op", choices=("mask", "st", "adamw", "export2of4", "linear"), default="mask",
                   help="mask: the fwd+bwd step (default); st: the straight-through pair with dW; "
                        "adamw: fwd + the backward fused with the logits' AdamW step; "
                        "export2of4: the compressed 2:4 export; linear: the masked linear forward "
                        "(mask formed in a tensor-core GEMM's prologue) over --tokens tokens (one GPU)")
    p.add_argument("--tokens", type=int, default=256, help="tokens per layer for --op linear (1..256)")
    p.add_argument("--per-tensor", action="store_true",
                   help="one roi_mask_fwd_ex / roi_mask_bwd call per tensor instead of one batched call per "
                        "direction (adds the per-projection breakdown)")
    return p.parse_args()


def selected_tensors(args):
    """[(layer, proj_index, rows, cols)] of the layer set, optionally restricted."""
    lset = WL.LAYER_SETS[args.set]
    keep = set(args.proj.split(",")) if args.proj else set(WL.PROJS)
    out = []
    for layer, p, rows, cols in lset.tensors():
        if args.layers is not None and layer >= args.layers:
            continue
        if WL.PROJS[p] in keep:
            out.append((layer, p, rows, cols))
    return out


def config_for(args):
    lset = WL.LAYER_SETS[args.set]
    cfg = WL.CONFIGS[args.set]
    N, M = map(int, args.nm.split(":"))
    tau = args.tau if args.tau is not None else cfg.taus[0]
    sel = selected_tensors(args)
    E = sum(r * c for _, _, r, c in sel)
    h, kv, i = lset.hidden, lset.kv, lset.inter
    layers = lset.layers if args.layers is None else min(args.layers, lset.layers)
    projs = "{q,o %dx%d; k,v %dx%d; gate,up %dx%d; down %dx%d}" % (h, h, kv, h, i, h, h, i)
    if args.proj:
        projs = "{" + ",".join(f"{q} {'x'.join(map(str, lset.shape(q)))}" for q in args.proj.split(",")) + "}"
    return {
        "workload": (f"{args.set}-shaped layer set, {N}:{M}, tau={tau}, {layers} layers x {projs}, "
                     f"logits {cfg.logits}, step-keyed noise"),
        "layer_set": args.set, "N": N, "M": M, "tau": tau, "lambda": 1.0,
        "elements": E, "groups": E // M, "tensors": len(sel),
        "l2": "inputs larger than L2: every step streams the whole set (>90 GB for the 7B set)",
        "calls": ("one roi_mask_fwd_ex + one roi_mask_bwd per tensor" if getattr(args, "per_tensor", False) else
                  "one roi_mask_fwd_batch + one roi_mask_bwd_batch per step (all tensors)"),
    }


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [ln for ln in out.splitlines() if ln.strip()]
        else:
            self.lines = []

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for name, val in zip(names, f[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------------
# roofline denominators and counters
# --------------------------------------------------------------------------
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e, nominal (the measured copy bandwidth is the peak used)


# Special-function-unit work per element of the general-tau path, in ex2 issue slots
# (lg2 and rcp take two: 32 ex2 or 16 lg2 / rcp per clock per SM on this part).
# Algorithmic counts: the Gumbel sample needs two logs; each of the N relaxation
# steps one exp per element and one reciprocal per group, each step but the last a
# log per element; the backward re-forms all of it and divides by 1 - mu once per
# element in each of its N - 1 earlier steps.
SFU_SLOTS_PER_CLK_SM = 32
SFU_CLOCK_MHZ = 2070  # maximum SM clock


def sfu_slots(N, M):
    fwd = 2 * 2 + N + 2 * (N - 1) + 2 * N / M
    return fwd, fwd + 2 * (N - 1)


def sfu_peak(dev):
    import torch
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    return SFU_SLOTS_PER_CLK_SM * sms * SFU_CLOCK_MHZ * 1e6 / 1e9  # G slots/s


def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash():
    d = os.path.join(ROOT, "paper_2608_23048_gb300", "csrc")
    h = hashlib.sha256()
    for name in sorted(os.listdir(d)):
        with open(os.path.join(d, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel_tag: str):
    """DRAM bytes per element of `kernel_tag` from profiles/dram_traffic.txt, if the
    kernel sources are unchanged since that capture; else None."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    try:
        lines = open(path).read().splitlines()
    except OSError:
        return None
    want = kernel_source_hash()
    for ln in lines:
        if ln.startswith("#") or not ln.strip():
            continue
        kv = dict(x.split("=", 1) for x in ln.split() if "=" in x)
        if kv.get("kernel") == kernel_tag and kv.get("sources") == want:
            return float(kv["dram_bytes_per_element"])
    return None


# --------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and --impl reference)
# --------------------------------------------------------------------------
def _oracle_chunk(job):
    """Runs in a spawned worker: oracle fwd + bwd over `rows` rows of a tensor."""
    import numpy as np
    import workloads as W
    from oracle import roi_oracle as O
    rows, cols, N, M, tau, kind, seed, step, row_offset = job
    Wt, phi, dWm = W.make_inputs(rows, cols, kind, seed)
    ph, Wb, dWb = phi.numpy(), W.bf16_bits(Wt), W.bf16_bits(dWm)
    t0 = time.perf_counter()
    O.mask_fwd(ph, Wb, N, M, tau, seed, step, row_offset=row_offset)
    O.mask_bwd(ph, Wb, dWb, N, M, tau, seed, step, row_offset=row_offset)
    return time.perf_counter() - t0, rows * cols // M


def oracle_pool(cores):
    import multiprocessing as mp
    return mp.get_context("spawn").Pool(cores)


def time_oracle(pool, cores, cfg, cols, rows_per_job, jobs, step=0):
    N, M, tau = cfg["N"], cfg["M"], cfg["tau"]
    kind = WL.CONFIGS[cfg["layer_set"]].logits
    work = [(rows_per_job, cols, N, M, tau, kind, 1000 + j, step, j * rows_per_job) for j in range(jobs)]
    res = pool.map(_oracle_chunk, work, chunksize=1)
    groups = sum(g for _, g in res)
    # the jobs run side by side, one per process: the slowest bounds the wall time
    return groups, max(t for t, _ in res)


def calibrate_rows(pool, cores, cfg, cols, target_s, max_rows):
    """Rows per job so that one job of the oracle takes about target_s seconds:
    grow the job until it takes a quarter of the target, then scale linearly."""
    rows = 4
    time_oracle(pool, cores, cfg, cols, rows, cores)      # workers pay their imports here
    while True:
        _, t = time_oracle(pool, cores, cfg, cols, rows, cores)
        if t >= target_s / 4 or rows * 4 > max_rows:
            break
        rows *= 4
    return max(1, min(max_rows, int(rows * target_s / max(t, 1e-6))))


def cpu_baseline(cfg, seconds, cores=None):
    """Oracle (float64, as it stands) on the host cores over rows of the set's largest tensor."""
    cores = cores or os.cpu_count() or 1
    lset = WL.LAYER_SETS[cfg["layer_set"]]
    rows_full, cols = lset.shape("gate")
    pool = oracle_pool(cores)
    try:
        rows_per_job = calibrate_rows(pool, cores, cfg, cols, seconds, rows_full // cores)
        g, wall = time_oracle(pool, cores, cfg, cols, rows_per_job, cores)
    finally:
        pool.close()
        pool.join()
    return {"value": g / wall, "unit": "groups/s", "cores": cores, "kind": "oracle",
            "sample": (f"{cores} x {rows_per_job} rows of the {cfg['layer_set']} gate_proj shape "
                       f"({rows_per_job * cores} x {cols}, {g} groups), float64 oracle fwd+bwd, "
                       f"{wall:.1f} s wall on {cores} processes")}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cfg = config_for(args)
    cores = os.cpu_count() or 1
    lset = WL.LAYER_SETS[cfg["layer_set"]]
    _, cols = lset.shape("gate")
    pool = oracle_pool(cores)
    budget = 120.0  # seconds of oracle work for the whole --steps/--warmup run
    try:
        per_step = min(10.0, budget / max(1, args.steps + args.warmup))
        rows_per_job = calibrate_rows(pool, cores, cfg, cols, per_step, 4096)
        for w in range(args.warmup):
            time_oracle(pool, cores, cfg, cols, rows_per_job, cores, step=w)
        tot_g, tot_t = 0, 0.0
        for s in range(args.steps):
            g, wall = time_oracle(pool, cores, cfg, cols, rows_per_job, cores, step=args.warmup + s)
            tot_g += g
            tot_t += wall
    finally:
        pool.close()
        pool.join()
    value = tot_g / tot_t
    sample = (f"each step: {cores} x {rows_per_job} rows of the gate_proj shape x {cols} "
              f"({tot_g // max(1, args.steps)} groups), float64 oracle fwd+bwd")
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "groups/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / max(1, args.steps),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "config": cfg,
           "cpu_baseline": {"value": value, "unit": "groups/s", "cores": cores, "kind": "oracle", "sample": sample},
           "e2e": {"value": value, "unit": "groups/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# --------------------------------------------------------------------------
# our arm
# --------------------------------------------------------------------------
def make_set_tensors(roi, set_name, sel, dev, rank=0):
    """Device tensors of the selected layers of a layer set (inputs and outputs)."""
    import torch
    kind = WL.CONFIGS[set_name].logits
    tensors = []
    for layer, p, rows, cols in sel:
        W, phi, dWm = WL.make_inputs(rows, cols, kind, WL.tensor_seed(layer, p) + 7919 * rank, device=dev)
        tensors.append({
            "id": layer * len(WL.PROJS) + p, "rows": rows, "cols": cols, "phi": phi, "W": W, "dWm": dWm,
            "Wm": torch.empty_like(W), "dphi": torch.empty_like(phi),
            "hard": torch.empty(roi.hard_words(rows, cols), dtype=torch.int32, device=dev)})
    torch.cuda.synchronize()
    return tensors


class MaskStep:
    """One step: roi_mask_fwd over every tensor (forward order), then roi_mask_bwd over
    every tensor (reverse order), step-keyed noise, on one stream; batched calls (one
    per direction) unless per_tensor.  step(s, ev) records events around each call
    into ev = (fwd start, fwd end, bwd start, bwd end) lists when given."""

    def __init__(self, roi, tensors, N, M, tau, stream, per_tensor=False):
        self.roi, self.tensors, self.N, self.M, self.tau = roi, tensors, N, M, tau
        self.stream, self.per_tensor = stream, per_tensor
        self.states = {t["id"]: roi.NoiseState(0, 0, t["id"], 1.0, 0) for t in tensors}
        self.fwd_items = roi.make_fwd_items([(t["phi"], t["W"], self.states[t["id"]], t["Wm"], None, t["hard"])
                                             for t in tensors])
        self.bwd_items = roi.make_bwd_items([(t["phi"], t["W"], self.states[t["id"]], t["dWm"], t["dphi"], None)
                                             for t in reversed(tensors)])

    def _mark(self, lst, ev):
        import torch
        if ev is not None:
            lst.append(torch.cuda.Event(enable_timing=True))
            lst[-1].record(self.stream)

    def __call__(self, s, ev=None):
        roi, N, M, tau, stream = self.roi, self.N, self.M, self.tau, self.stream
        e = ev if ev is not None else (None,) * 4
        if not self.per_tensor:
            for arr in (self.fwd_items, self.bwd_items):
                for k in range(len(arr)):
                    arr[k].st.step = s
            self._mark(e[0], ev)
            roi.roi_mask_fwd_batch(self.fwd_items, N, M, tau, stream=stream)
            self._mark(e[1], ev)
            self._mark(e[2], ev)
            roi.roi_mask_bwd_batch(self.bwd_items, N, M, tau, stream=stream)
            self._mark(e[3], ev)
            return
        for t in self.tensors:
            st = self.states[t["id"]]
            st.step = s
            self._mark(e[0], ev)
            roi.roi_mask_fwd_ex(t["phi"], t["W"], N, M, tau, st, t["Wm"], None, t["hard"], stream=stream)
            self._mark(e[1], ev)
        for t in reversed(self.tensors):
            st = self.states[t["id"]]
            self._mark(e[2], ev)
            roi.roi_mask_bwd(t["phi"], t["W"], st, N, M, t["dWm"], tau, t["dphi"], None, stream=stream)
            self._mark(e[3], ev)


def time_steps(roi, step, stream, steps, warmup, world, local):
    """W untimed warm-up steps, then K timed steps bracketed by a barrier and a device
    synchronisation, with per-call CUDA events on the launch stream and the clocks
    sampled meanwhile.  Returns the timings (max over ranks for the whole region)."""
    import torch
    import torch.distributed as dist
    with torch.cuda.stream(stream):
        for w in range(warmup):
            step(w)
    torch.cuda.synchronize()
    roi.roi_device_status(stream)
    ev = ([], [], [], [])
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = roi.roi_launch_count()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clocks:
        start.record(stream)
        for s in range(steps):
            step(warmup + s, ev)
        end.record(stream)
        torch.cuda.synchronize()
    launches = roi.roi_launch_count() - launches0
    if world > 1:
        dist.barrier()
    roi.roi_device_status(stream)
    elapsed = start.elapsed_time(end) / 1e3
    if world > 1:
        tt = torch.tensor([elapsed], device=torch.device("cuda", local))
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        elapsed = float(tt.item())
    fwd_t = sum(a.elapsed_time(b) for a, b in zip(ev[0], ev[1])) / 1e3
    bwd_t = sum(a.elapsed_time(b) for a, b in zip(ev[2], ev[3])) / 1e3
    # per-step device time: first forward launch to last backward launch of each step
    T = len(ev[0]) // steps  # events per step and direction: one per call
    step_ms = sorted(ev[0][s * T].elapsed_time(ev[3][s * T + T - 1]) for s in range(steps))
    pct = lambda q: round(step_ms[min(len(step_ms) - 1, int(q * (len(step_ms) - 1) + 0.5))], 3)
    return {"elapsed": elapsed, "fwd_t": fwd_t, "bwd_t": bwd_t, "ev": ev, "launches": int(launches),
            "clocks": clocks.summary(), "step_ms": {"p10": pct(0.1), "median": pct(0.5), "p90": pct(0.9)}}


def mask_roofline(E, N, M, tau, tm, steps, world, dev, ntensors, per_tensor=False, per_projection=None):
    """Roofline object of the dominant kernel of a mask step: HBM for the tile
    kernels, the special-function units for the warp-slice configurations."""
    fwd_t, bwd_t = tm["fwd_t"], tm["bwd_t"]
    step_gbs = world * E * (FWD_BYTES + BWD_BYTES) * steps / tm["elapsed"] / 1e9
    peak, peak_kind = hbm_peak()
    fwd_gbs = E * FWD_BYTES * steps / fwd_t / 1e9
    bwd_gbs = E * BWD_BYTES * steps / bwd_t / 1e9
    dom = "bwd" if bwd_t >= fwd_t else "fwd"
    tag = f"roi_{dom}_kernel<{N},{M},{'tau1' if tau == 1.0 else 'tau'}>"
    traffic = recorded_traffic(tag)
    per_elem = BWD_BYTES if dom == "bwd" else FWD_BYTES
    achieved = bwd_gbs if dom == "bwd" else fwd_gbs
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4),
                "traffic": (None if traffic is None else traffic * E / ntensors),
                "kernel": tag, "peak_kind": peak_kind,
                "algorithmic_bytes_per_element": per_elem,
                "units_per_launch": (f"{E / ntensors:.0f} elements (mean over the {ntensors} tensors"
                                     + ("" if per_tensor else
                                        "; batched calls, chained launches, one per large tensor and one per run of "
                                        "small tensors, achieved from the call's time") + ")"),
                "fwd_gbs": round(fwd_gbs, 1), "bwd_gbs": round(bwd_gbs, 1),
                "fwd_frac": round(fwd_gbs / peak, 4), "bwd_frac": round(bwd_gbs / peak, 4),
                "fwd_ms_per_step": round(1e3 * fwd_t / steps, 3),
                "bwd_ms_per_step": round(1e3 * bwd_t / steps, 3),
                "step_gbs": round(step_gbs / world, 1), "step_frac": round(step_gbs / world / peak, 4),
                "nominal_hbm_gbs": NOMINAL_HBM_GBS, "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
                "step_frac_of_nominal": round(step_gbs / world / NOMINAL_HBM_GBS, 4)}
    if per_projection:
        roofline["per_projection"] = per_projection
    if M >= 16 and tau != 1.0:
        # the warp-slice configurations bind on the special-function units, not HBM:
        # the binding roofline is the SFU issue rate (the HBM figures stay beside it)
        sf, sb = sfu_slots(N, M)
        sp = sfu_peak(dev)
        t_dom = bwd_t if dom == "bwd" else fwd_t
        ach = E * (sb if dom == "bwd" else sf) * steps / t_dom / 1e9
        step_ach = E * (sf + sb) * steps / (fwd_t + bwd_t) / 1e9
        roofline = {"bound": "alu", "achieved": round(ach, 1), "peak": round(sp, 1), "unit": "G SFU slots/s",
                    "frac": round(ach / sp, 4), "traffic": roofline["traffic"], "kernel": tag,
                    "peak_kind": (f"derived: {SFU_SLOTS_PER_CLK_SM} ex2 slots per clock per SM x SMs x "
                                  f"{SFU_CLOCK_MHZ} MHz (lg2 / rcp take two slots)"),
                    "sfu_slots_per_element": {"fwd": sf, "bwd": sb},
                    "units_per_launch": roofline["units_per_launch"],
                    "fwd_ms_per_step": roofline["fwd_ms_per_step"], "bwd_ms_per_step": roofline["bwd_ms_per_step"],
                    "fwd_sfu_frac": round(E * sf * steps / fwd_t / 1e9 / sp, 4),
                    "bwd_sfu_frac": round(E * sb * steps / bwd_t / 1e9 / sp, 4),
                    "step_sfu_frac": round(step_ach / sp, 4), "hbm": {k: roofline[k] for k in (
                        "achieved", "peak", "unit", "frac", "algorithmic_bytes_per_element", "fwd_gbs", "bwd_gbs",
                        "step_gbs", "step_frac")}}
        if per_projection:
            roofline["per_projection"] = per_projection
    return roofline, step_gbs


def near_ties(roi, t, N, M, step):
    """Groups of tensor t whose N-th and (N+1)-th perturbed keys (lambda = 1) differ
    by less than 1e-6 at `step`: the keys are the library's, phi + g in float32 with g
    from roi_gumbel_noise (the noise the kernels regenerate)."""
    import torch
    rows, cols = t["rows"], t["cols"]
    g = torch.empty(rows * cols, dtype=torch.float32, device=t["phi"].device)
    roi.roi_gumbel_noise(roi.NoiseState(0, step, t["id"], 1.0, 0), rows, cols, g)
    keys = (t["phi"].reshape(-1) + g).view(-1, M)
    top = torch.topk(keys, N + 1, dim=1).values
    n = int((top[:, N - 1] - top[:, N] < 1e-6).sum())
    return {"tensor": f"{t['id']} ({rows}x{cols})", "step": step, "groups": rows * cols // M, "near_tie_groups": n}


# The remaining configurations of the benchmark's configuration list, timed after the
# headline (one GPU): (layer set, N, M, tau, timed steps).
CONFIG_SWEEP = [
    ("qwen2.5-7b", 4, 8, 1.0, 10),
    ("qwen2.5-0.5b", 2, 4, 1.0, 50),
    ("qwen2.5-0.5b", 2, 4, 0.1, 50),
    ("qwen2.5-1.5b", 4, 8, 0.5, 20),
    ("qwen2.5-3b", 8, 16, 0.2, 10),
    ("qwen2.5-3b", 16, 32, 0.2, 10),
]


def config_sweep(roi, stream, dev, local, cache, warmup=3):
    """One record per configuration of CONFIG_SWEEP: the full layer set, batched calls,
    ms/step, groups/s, roofline, clocks and near ties of the set's first gate tensor.
    `cache` maps a layer set to its tensors (the headline's, to reuse); the sweep
    empties it when it moves to another set, so only one set is resident at a time."""
    import torch
    out = []
    for set_name, N, M, tau, steps in CONFIG_SWEEP:
        if set_name not in cache:
            cache.clear()
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
            cache[set_name] = make_set_tensors(roi, set_name, WL.LAYER_SETS[set_name].tensors(), dev)
        tensors = cache[set_name]
        E = sum(t["rows"] * t["cols"] for t in tensors)
        step = MaskStep(roi, tensors, N, M, tau, stream)
        tm = time_steps(roi, step, stream, steps, warmup, 1, local)
        roofline, step_gbs = mask_roofline(E, N, M, tau, tm, steps, 1, dev, len(tensors))
        gate = next(t for t in tensors if t["id"] % len(WL.PROJS) == WL.PROJS.index("gate"))
        lset = WL.LAYER_SETS[set_name]
        h, kv, i = lset.hidden, lset.kv, lset.inter
        out.append({
            "workload": (f"{set_name}-shaped layer set, {N}:{M}, tau={tau}, {lset.layers} layers x "
                         f"{{q,o {h}x{h}; k,v {kv}x{h}; gate,up {i}x{h}; down {h}x{i}}}, "
                         f"logits {WL.CONFIGS[set_name].logits}, step-keyed noise"),
            "N": N, "M": M, "tau": tau, "elements": E, "groups": E // M, "steps": steps, "warmup": warmup,
            "ms_per_step": round(1e3 * tm["elapsed"] / steps, 3), "groups_per_s": (E // M) * steps / tm["elapsed"],
            "hbm_gbs": round(step_gbs, 1), "step_ms": tm["step_ms"], "gpu_launches": tm["launches"],
            "roofline": roofline, "clocks": tm["clocks"],
            "near_ties": near_ties(roi, gate, N, M, warmup + steps - 1)})
    cache.clear()
    return out


def run_ours(args):
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    cfg = config_for(args)
    N, M, tau = cfg["N"], cfg["M"], cfg["tau"]

    # the oracle pool is spawned before the first CUDA call
    base = None
    if rank == 0 and not args.no_cpu_baseline:
        base = cpu_baseline(cfg, args.cpu_seconds)

    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2608_23048_gb300 import _build
    if rank == 0:
        _build.build()
    if world > 1:
        dist.barrier()
    import paper_2608_23048_gb300 as roi
    roi.lib()

    lset = WL.LAYER_SETS[args.set]
    tensors = make_set_tensors(roi, args.set, selected_tensors(args), dev, rank)
    stream = torch.cuda.Stream(device=dev)
    step = MaskStep(roi, tensors, N, M, tau, stream, per_tensor=args.per_tensor)

    # timed region: K steps, per-call events for the per-kernel roofline
    tm = time_steps(roi, step, stream, args.steps, args.warmup, world, local)
    elapsed, ev = tm["elapsed"], tm["ev"]
    # per projection, summed over layers, per step: fwd ms, bwd ms, fraction of the roofline
    # (per-tensor calls only)
    per_proj = {}
    nt = len(tensors) if args.per_tensor else 10 ** 9
    for i, (a, b) in enumerate(zip(ev[0], ev[1]) if args.per_tensor else ()):
        t = tensors[i % nt]
        per_proj.setdefault(WL.PROJS[t["id"] % len(WL.PROJS)], [0.0, 0.0, 0])[0] += a.elapsed_time(b) / args.steps
    for i, (a, b) in enumerate(zip(ev[2], ev[3]) if args.per_tensor else ()):
        t = tensors[nt - 1 - i % nt]
        per_proj[WL.PROJS[t["id"] % len(WL.PROJS)]][1] += a.elapsed_time(b) / args.steps
    for t in tensors if args.per_tensor else ():
        per_proj[WL.PROJS[t["id"] % len(WL.PROJS)]][2] += t["rows"] * t["cols"]
    pk = hbm_peak()[0]
    per_projection = {k: {"fwd_ms": round(f, 3), "bwd_ms": round(b, 3),
                          "frac": round(n * (FWD_BYTES + BWD_BYTES) / ((f + b) * 1e-3) / 1e9 / pk, 3)}
                      for k, (f, b, n) in per_proj.items()}

    E = cfg["elements"]
    groups_all = world * (E // M) * args.steps
    value = groups_all / elapsed
    roofline, step_gbs = mask_roofline(E, N, M, tau, tm, args.steps, world, dev, len(tensors),
                                       args.per_tensor, per_projection)
    peak = hbm_peak()[0]

    # the hard masks change with the step and each step reproduces (outside the timed region)
    t0 = tensors[0]
    last = args.warmup + args.steps - 1
    h_last = t0["hard"].clone()
    scratch_Wm = torch.empty_like(t0["Wm"])
    h_again = torch.empty_like(t0["hard"])
    h_prev = torch.empty_like(t0["hard"])
    other = last - 1 if last > 0 else last + 1
    for s_, out_h in ((last, h_again), (other, h_prev)):
        st = roi.NoiseState(0, s_, t0["id"], 1.0, 0)
        roi.roi_mask_fwd_ex(t0["phi"], t0["W"], N, M, tau, st, scratch_Wm, None, out_h, stream=stream)
    torch.cuda.synchronize()
    gate = [t for t in tensors if t["id"] % len(WL.PROJS) == WL.PROJS.index("gate")]
    checks = {"step_reproducible": bool(torch.equal(h_again, h_last)),
              "masks_differ_across_steps": bool(not torch.equal(h_prev, h_last)),
              "checked_on": f"tensor {t0['id']} ({t0['rows']}x{t0['cols']}), steps {other} and {last}",
              "near_ties": [near_ties(roi, t, N, M, last) for t in [t0] + gate[:1]],
              "near_ties_rule": ("groups whose N-th and (N+1)-th perturbed keys (the library's float32 keys) "
                                 "differ by less than 1e-6, at the last timed step")}

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, roi, tensors, lset, N, M, tau, dev, world)

    configs = None
    if (world == 1 and not args.no_configs and args.set == "qwen2.5-7b" and args.layers is None
            and args.proj is None and not args.per_tensor):
        holder = {args.set: tensors}
        del step, tensors, t0, gate
        configs = config_sweep(roi, stream, dev, local, holder)

    if rank == 0:
        out = {"metric": METRIC, "value": value, "unit": "groups/s", "n_gpus": world, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": 1e3 * elapsed / args.steps, "higher_is_better": True,
               "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": cfg,
               "hbm_gbs": round(step_gbs, 1), "hbm_frac": round(step_gbs / world / peak, 4),
               "roofline": roofline, "cpu_baseline": base, "e2e": e2e,
               "gpu_launches": tm["launches"], "step_ms": tm["step_ms"], "checks": checks, "clocks": tm["clocks"],
               "clocks_note": "sampled with nvidia-smi every 100 ms during the timed region",
               "configs": configs,
               "configs_note": ("the other configurations of the benchmark list, each its full layer set with "
                                "batched calls, timed after the headline on the same GPU (one GPU runs only)")}
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_e2e(args, roi, tensors, lset, N, M, tau, dev, world):
    """Same step through the C ABI with host buffers: per tensor, copy logits, W and
    dWm from pinned host memory, run fwd + bwd, copy Wm, the hard bits and the logit
    gradients back.  Three streams form a pipeline (host->device copies, kernels,
    device->host copies) ordered by per-tensor events, so both copy directions and
    the kernels overlap."""
    import torch
    host = {}
    for t in tensors:
        p = t["id"] % len(WL.PROJS)
        if p in host:
            continue
        host[p] = {
            "phi": t["phi"].cpu().pin_memory(), "W": t["W"].cpu().pin_memory(), "dWm": t["dWm"].cpu().pin_memory(),
            "Wm": torch.empty_like(t["Wm"], device="cpu").pin_memory(),
            "hard": torch.empty_like(t["hard"], device="cpu").pin_memory(),
            "dphi": torch.empty_like(t["dphi"], device="cpu").pin_memory()}
    s_in, s_run, s_out = (torch.cuda.Stream(device=dev) for _ in range(3))
    ev_in = [torch.cuda.Event() for _ in tensors]
    ev_run = [torch.cuda.Event() for _ in tensors]
    ev_out = [torch.cuda.Event() for _ in tensors]
    h2d = sum(t["rows"] * t["cols"] * 8 for t in tensors)
    d2h = sum(t["rows"] * t["cols"] * 6 + t["hard"].numel() * 4 for t in tensors)
    started = [False]

    def one(s):
        for i, t in enumerate(tensors):
            hs = host[t["id"] % len(WL.PROJS)]
            st = roi.NoiseState(0, s, t["id"], 1.0, 0)
            with torch.cuda.stream(s_in):
                if started[0]:
                    s_in.wait_event(ev_out[i])  # the previous step is done with this tensor's buffers
                t["phi"].copy_(hs["phi"], non_blocking=True)
                t["W"].copy_(hs["W"], non_blocking=True)
                t["dWm"].copy_(hs["dWm"], non_blocking=True)
                ev_in[i].record(s_in)
            with torch.cuda.stream(s_run):
                s_run.wait_event(ev_in[i])
                roi.roi_mask_fwd_ex(t["phi"], t["W"], N, M, tau, st, t["Wm"], None, t["hard"], stream=s_run)
                roi.roi_mask_bwd(t["phi"], t["W"], st, N, M, t["dWm"], tau, t["dphi"], None, stream=s_run)
                ev_run[i].record(s_run)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_run[i])
                hs["Wm"].copy_(t["Wm"], non_blocking=True)
                hs["hard"].copy_(t["hard"], non_blocking=True)
                hs["dphi"].copy_(t["dphi"], non_blocking=True)
                ev_out[i].record(s_out)
        started[0] = True

    one(10_000)
    torch.cuda.synchronize()
    steps = max(1, args.e2e_steps)
    t0 = time.perf_counter()
    for s in range(steps):
        one(10_001 + s)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    if world > 1:
        import torch.distributed as dist
        tt = torch.tensor([wall], device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        wall = float(tt.item())
    groups = world * (sum(t["rows"] * t["cols"] for t in tensors) // M) * steps
    return {"value": groups / wall, "unit": "groups/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": steps, "ms_per_step": 1e3 * wall / steps,
            "note": "host buffers: one layer's tensors in pinned memory, reused for all layers"}


ST_FWD_BYTES = FWD_BYTES
ST_BWD_BYTES = BWD_BYTES + 2 + 1 / 8   # + dW out, + the forward's hard bits in
EXPORT_2OF4_BYTES = 4 + 2 + 1 + 1 / 8  # logits, W in; kept values, index codes out
ADAMW_BWD_BYTES = 4 + 2 + 2 + 4 + 4 + 4 + 4 + 4  # logits, W, dWm, m, v in; logits, m, v out


def run_variant(args):
    """The straight-through pair (roi_mask_fwd_st + roi_mask_bwd_st with dW) or the
    compressed 2:4 export over the layer set: device-resident inputs, per-launch CUDA
    events, algorithmic bytes against the measured copy bandwidth.  One GPU."""
    import torch
    if int(os.environ.get("RANK", "0")) != 0:
        return
    cfg = config_for(args)
    N, M, tau = cfg["N"], cfg["M"], cfg["tau"]
    if args.op == "export2of4" and (N, M) != (2, 4):
        raise SystemExit("--op export2of4 needs --nm 2:4")
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2608_23048_gb300 import _build
    _build.build()
    import paper_2608_23048_gb300 as roi
    kind = WL.CONFIGS[args.set].logits
    tensors = []
    for layer, p, rows, cols in selected_tensors(args):
        W, phi, dWm = WL.make_inputs(rows, cols, kind, WL.tensor_seed(layer, p), device=dev)
        t = {"id": layer * len(WL.PROJS) + p, "rows": rows, "cols": cols, "phi": phi, "W": W, "dWm": dWm}
        if args.op in ("st", "adamw"):
            t.update(Wm=torch.empty_like(W), dphi=torch.empty_like(phi), dW=torch.empty_like(W),
                     hard=torch.empty(roi.hard_words(rows, cols), dtype=torch.int32, device=dev))
        if args.op == "adamw":
            t.update(m=torch.zeros_like(phi), v=torch.zeros_like(phi))
        else:
            t.update(values=torch.empty(rows, cols // 2, dtype=torch.bfloat16, device=dev),
                     meta=torch.empty(rows * cols // 32, dtype=torch.int32, device=dev))
        tensors.append(t)
    stream = torch.cuda.Stream(device=dev)
    if args.op == "st":
        st_fwd = roi.make_fwd_items([(t["phi"], t["W"], roi.NoiseState(0, 0, t["id"], 1.0, 0), t["Wm"], None,
                                      t["hard"]) for t in tensors])
        st_bwd = roi.make_bwd_st_items([(t["phi"], t["W"], roi.NoiseState(0, 0, t["id"], 1.0, 0), t["dWm"], t["hard"],
                                         t["dphi"], t["dW"]) for t in reversed(tensors)])
    if args.op == "adamw":
        adamw_fwd = roi.make_fwd_items([(t["phi"], t["W"], roi.NoiseState(0, 0, t["id"], 1.0, 0), t["Wm"], None,
                                         t["hard"]) for t in tensors])
        adamw_bwd = roi.make_adamw_items([(t["phi"], t["W"], roi.NoiseState(0, 0, t["id"], 1.0, 0), t["dWm"], t["m"],
                                           t["v"], None, None) for t in reversed(tensors)])

    def launches(s, ev):
        def rec(lst):
            if ev is not None:
                lst.append(torch.cuda.Event(enable_timing=True))
                lst[-1].record(stream)
        if args.op == "st" and not args.per_tensor:
            for arr in (st_fwd, st_bwd):
                for k in range(len(arr)):
                    arr[k].st.step = s
            rec(ev[0] if ev else None)
            roi.roi_mask_fwd_st_batch(st_fwd, N, M, tau, stream=stream)
            rec(ev[1] if ev else None)
            rec(ev[2] if ev else None)
            roi.roi_mask_bwd_st_batch(st_bwd, N, M, tau, stream=stream)
            rec(ev[3] if ev else None)
            return
        if args.op == "adamw" and not args.per_tensor:
            # the training step's two calls: every forward, then every backward fused
            # with the logits' AdamW step (chained launches)
            for arr in (adamw_fwd, adamw_bwd):
                for k in range(len(arr)):
                    arr[k].st.step = s
            rec(ev[0] if ev else None)
            roi.roi_mask_fwd_batch(adamw_fwd, N, M, tau, stream=stream)
            rec(ev[1] if ev else None)
            rec(ev[2] if ev else None)
            roi.roi_mask_bwd_adamw_batch(adamw_bwd, N, M, tau, roi.AdamW(1e-3, 0.9, 0.95, 1e-8, 0.05, s + 1),
                                         stream=stream)
            rec(ev[3] if ev else None)
            return
        for t in tensors:
            st = roi.NoiseState(0, s, t["id"], 1.0, 0)
            rec(ev[0] if ev else None)
            if args.op == "st":
                roi.roi_mask_fwd_st(t["phi"], t["W"], N, M, tau, st, t["Wm"], None, t["hard"], stream=stream)
            elif args.op == "adamw":
                roi.roi_mask_fwd_ex(t["phi"], t["W"], N, M, tau, st, t["Wm"], None, t["hard"], stream=stream)
            else:
                roi.roi_export_compressed_2of4(t["phi"], t["W"], t["values"], t["meta"], stream=stream)
            rec(ev[1] if ev else None)
        if args.op in ("st", "adamw"):
            for t in reversed(tensors):
                st = roi.NoiseState(0, s, t["id"], 1.0, 0)
                rec(ev[2] if ev else None)
                if args.op == "st":
                    roi.roi_mask_bwd_st(t["phi"], t["W"], st, N, M, t["dWm"], t["hard"], tau, t["dphi"], t["dW"],
                                        stream=stream)
                else:
                    opt = roi.AdamW(1e-3, 0.9, 0.95, 1e-8, 0.05, s + 1)
                    roi.roi_mask_bwd_adamw(t["phi"], t["W"], st, N, M, t["dWm"], tau, t["m"], t["v"], opt,
                                           stream=stream)
                rec(ev[3] if ev else None)

    for w in range(args.warmup):
        launches(w, None)
    torch.cuda.synchronize()
    roi.roi_device_status(stream)
    ev = ([], [], [], [])
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clocks:
        start.record(stream)
        for s in range(args.steps):
            launches(args.warmup + s, ev)
        end.record(stream)
        torch.cuda.synchronize()
    roi.roi_device_status(stream)
    elapsed = start.elapsed_time(end) / 1e3
    a_t = sum(x.elapsed_time(y) for x, y in zip(ev[0], ev[1])) / 1e3
    b_t = sum(x.elapsed_time(y) for x, y in zip(ev[2], ev[3])) / 1e3
    E = cfg["elements"]
    peak, peak_kind = hbm_peak()
    if args.op in ("st", "adamw"):
        fb, bb = (ST_FWD_BYTES, ST_BWD_BYTES) if args.op == "st" else (FWD_BYTES, ADAMW_BWD_BYTES)
        a_gbs = E * fb * args.steps / a_t / 1e9
        b_gbs = E * bb * args.steps / b_t / 1e9
        dom = "bwd" if b_t >= a_t else "fwd"
        achieved, per = (b_gbs, bb) if dom == "bwd" else (a_gbs, fb)
        step_bytes = fb + bb
        extra = {"fwd_gbs": round(a_gbs, 1), "bwd_gbs": round(b_gbs, 1),
                 "fwd_ms_per_step": round(1e3 * a_t / args.steps, 3), "bwd_ms_per_step": round(1e3 * b_t / args.steps, 3)}
        what = "straight-through" if args.op == "st" else "backward fused with AdamW"
        kernel = f"roi_{dom}_kernel<{N},{M},{'tau1' if tau == 1.0 else 'tau'}> ({what})"
        metric = ("straight-through RoI mask fwd+bwd (dW on) groups/s and HBM GB/s, 1 GPU" if args.op == "st" else
                  "RoI mask fwd + bwd fused with the logits' AdamW step, groups/s and HBM GB/s, 1 GPU")
    else:
        achieved = E * EXPORT_2OF4_BYTES * args.steps / a_t / 1e9
        per, step_bytes = EXPORT_2OF4_BYTES, EXPORT_2OF4_BYTES
        extra = {"ms_per_step": round(1e3 * a_t / args.steps, 3)}
        kernel = "roi_export_2of4_kernel"
        metric = "compressed 2:4 export groups/s and HBM GB/s, 1 GPU"
    step_gbs = E * step_bytes * args.steps / elapsed / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": None, "kernel": kernel, "peak_kind": peak_kind,
                "algorithmic_bytes_per_element": per, "step_gbs": round(step_gbs, 1),
                "step_frac": round(step_gbs / peak, 4), **extra}
    cfg = dict(cfg, op=args.op)
    print(json.dumps({"metric": metric, "value": (E // M) * args.steps / elapsed, "unit": "groups/s",
                      "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                      "ms_per_step": 1e3 * elapsed / args.steps, "higher_is_better": True, "scaling": "weak",
                      "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": cfg,
                      "roofline": roofline, "clocks": clocks.summary()}), flush=True)


def bf16_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_BF16_TFLOPS, "fallback"


def run_linear(args):
    """Masked linear forward over the layer set: every tensor's Y = X Wm^T for
    --tokens tokens with the mask formed in the GEMM's prologue
    (roi_masked_linear_fwd), device-resident inputs, per-launch CUDA events.  Beside
    it, the unfused pair the fusion replaces: roi_mask_fwd_ex writing Wm, then a
    cuBLAS bf16 GEMM (torch.mm) reading it.  One GPU."""
    import torch
    if int(os.environ.get("RANK", "0")) != 0:
        return
    cfg = config_for(args)
    N, M, tau, T = cfg["N"], cfg["M"], cfg["tau"], args.tokens
    if not 1 <= T <= 256:
        raise SystemExit("--tokens must be in 1..256")
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    from paper_2608_23048_gb300 import _build
    _build.build()
    import paper_2608_23048_gb300 as roi
    kind = WL.CONFIGS[args.set].logits
    tensors, ws_bytes = [], 16
    for layer, p, rows, cols in selected_tensors(args):
        seed = WL.tensor_seed(layer, p)
        W, phi, _ = WL.make_inputs(rows, cols, kind, seed, device=dev)
        t = {"id": layer * len(WL.PROJS) + p, "rows": rows, "cols": cols, "phi": phi, "W": W,
             "X": WL.make_tokens(T, cols, seed, device=dev),
             "Y": torch.empty(T, rows, dtype=torch.float32, device=dev)}
        ws_bytes = max(ws_bytes, roi.roi_masked_linear_workspace_size(T, rows, cols))
        tensors.append(t)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    Wm = torch.empty(max(t["rows"] * t["cols"] for t in tensors), dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def fused(s, ev):
        for t in tensors:
            st = roi.NoiseState(0, s, t["id"], 1.0, 0)
            if ev is not None:
                ev[0].append(torch.cuda.Event(enable_timing=True))
                ev[0][-1].record(stream)
            roi.roi_masked_linear_fwd(t["X"], t["phi"], t["W"], N, M, tau, st, t["Y"], ws, stream=stream)
            if ev is not None:
                ev[1].append(torch.cuda.Event(enable_timing=True))
                ev[1][-1].record(stream)

    def unfused(s, ev=None):
        with torch.cuda.stream(stream):
            for t in tensors:
                st = roi.NoiseState(0, s, t["id"], 1.0, 0)
                wm = Wm[:t["rows"] * t["cols"]].view(t["rows"], t["cols"])
                if ev is not None:
                    ev[0].append(torch.cuda.Event(enable_timing=True))
                    ev[0][-1].record(stream)
                roi.roi_mask_fwd_ex(t["phi"], t["W"], N, M, tau, st, wm, stream=stream)
                torch.mm(t["X"], wm.t())
                if ev is not None:
                    ev[1].append(torch.cuda.Event(enable_timing=True))
                    ev[1][-1].record(stream)

    for w in range(args.warmup):
        fused(w, None)
    torch.cuda.synchronize()
    roi.roi_device_status(stream)
    ev = ([], [])
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clocks:
        start.record(stream)
        for s in range(args.steps):
            fused(args.warmup + s, ev)
        end.record(stream)
        torch.cuda.synchronize()
    roi.roi_device_status(stream)
    elapsed = start.elapsed_time(end) / 1e3
    k_t = sum(x.elapsed_time(y) for x, y in zip(ev[0], ev[1])) / 1e3
    # the unfused pair, same inputs and steps
    for w in range(args.warmup):
        unfused(w)
    u0, u1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    uev = ([], [])
    u0.record(stream)
    for s in range(args.steps):
        unfused(args.warmup + s, uev)
    u1.record(stream)
    torch.cuda.synchronize()
    unfused_t = u0.elapsed_time(u1) / 1e3
    # per projection (summed over layers), per step: fused kernel vs the unfused pair
    per_proj = {}
    for i, (x, y) in enumerate(zip(ev[0], ev[1])):
        name = WL.PROJS[tensors[i % len(tensors)]["id"] % len(WL.PROJS)]
        per_proj.setdefault(name, [0.0, 0.0])[0] += x.elapsed_time(y) / args.steps
    for i, (x, y) in enumerate(zip(uev[0], uev[1])):
        name = WL.PROJS[tensors[i % len(tensors)]["id"] % len(WL.PROJS)]
        per_proj.setdefault(name, [0.0, 0.0])[1] += x.elapsed_time(y) / args.steps
    E = cfg["elements"]
    bytes_step = sum(6 * t["rows"] * t["cols"] + 2 * T * t["cols"] + 4 * T * t["rows"] for t in tensors)
    flops_step = sum(2 * T * t["rows"] * t["cols"] for t in tensors)
    peak, peak_kind = hbm_peak()
    tpeak, tpeak_kind = bf16_peak()
    gbs = bytes_step * args.steps / k_t / 1e9
    tflops = flops_step * args.steps / k_t / 1e12
    bound = "hbm" if bytes_step / (peak * 1e9) >= flops_step / (tpeak * 1e12) else "tensor"
    tag = f"roi_masked_linear_kernel<{N},{M},{'tau1' if tau == 1.0 else 'tau'}>"
    traffic = recorded_traffic(tag)  # DRAM bytes per weight element (one 256-token capture)
    roofline = {"bound": bound, "achieved": round(gbs, 1), "peak": peak, "unit": "GB/s",
                "frac": round(gbs / peak, 4),
                "traffic": (None if traffic is None or T != 256 else traffic * E / len(tensors)),
                "kernel": tag,
                "peak_kind": peak_kind, "algorithmic_bytes_per_element": 6,
                "algorithmic_bytes_per_step": bytes_step, "tensor_tflops": round(tflops, 1),
                "tensor_peak_tflops": tpeak, "tensor_frac": round(tflops / tpeak, 4),
                "tensor_peak_kind": tpeak_kind, "kernel_ms_per_step": round(1e3 * k_t / args.steps, 3),
                "unfused_ms_per_step": round(1e3 * unfused_t / args.steps, 3),
                "unfused": "roi_mask_fwd_ex (Wm written) + cuBLAS bf16 GEMM reading Wm (torch.mm)",
                "per_projection_ms_fused_unfused": {k: [round(a, 3), round(b, 3)] for k, (a, b) in per_proj.items()}}
    cfg = dict(cfg, op="linear", tokens=T, y_dtype="f32")
    print(json.dumps({"metric": "masked linear forward (RoI mask in the GEMM prologue) groups/s and HBM GB/s, 1 GPU",
                      "value": (E // M) * args.steps / elapsed, "unit": "groups/s",
                      "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                      "ms_per_step": 1e3 * elapsed / args.steps, "higher_is_better": True, "scaling": "weak",
                      "vs_baseline": None, "dtype": "bf16 (products) / f32 (mask, accumulation)",
                      "data": "synthetic", "config": cfg, "roofline": roofline, "clocks": clocks.summary()}),
          flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    elif args.op == "linear":
        run_linear(args)
    elif args.op != "mask":
        run_variant(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
