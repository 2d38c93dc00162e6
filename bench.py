#!/usr/bin/env python3
"""Throughput of the GB300 chunkwise GLA forward (GTR token mixer).

One step = one forward pass over one batch of the workload: the whole hot path
(scan-order gather, in-chunk cumulative log-decay, chunk summaries, state
carry, intra-chunk gated scores, outputs and the final state) in the library's
kernels.  Default workload: the batched 1600-token mixer (B=32, 40x40 grid,
H=12, Dk=Dv=64, bf16, scan order alternating per step across the four
orders).  Prints ONE JSON line on rank 0.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload ID] [--impl reference]
                  [--launch graph|eager]

The K timed steps are captured once into one CUDA graph and replayed between two CUDA
events (the default, --launch graph); the same steps as eager calls, each between its
own events, are timed as well and reported as roofline.eager.

Multi-GPU (torchrun, one rank per GPU): every rank runs its own batch of the
same workload (weak scaling, no collective on the data path); value = tokens
of all ranks / max-over-ranks time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_26590_gb300 import workloads as wl  # noqa: E402

METRIC = "GLA-forward tokens/s (GB300, device-timed) and % of roofline at 1600 tokens"
DEFAULT_WORKLOAD = 2
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", type=int, default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--schedule", default="auto", choices=["auto", "simt", "tc"])
    ap.add_argument("--gated", action="store_true",
                    help="time the mixer with its output gate u = SiLU(r) * RMSNorm(o) (Sec. 3.1) instead of o")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--launch", default="graph", choices=["graph", "eager"],
                    help="graph (default): the K timed steps are captured once into one CUDA graph "
                         "(through the caller-workspace entry points) and replayed, as the paper times its "
                         "operator (Sec. 3.3); the eager per-step loop is timed as well and reported beside it. "
                         "eager: one eager call per step, each bracketed by CUDA events")
    ap.add_argument("--graph", action="store_true", help="same as --launch graph")
    ap.add_argument("--op", default="mixer", choices=["mixer", "sswiglu"],
                    help="mixer: the chunkwise GLA token mixer (default); sswiglu: the Spatial SwiGLU "
                         "gate-and-depthwise-conv step (Eq. spatial_swiglu) on --sw-workload")
    ap.add_argument("--sw-workload", type=int, default=2)
    ap.add_argument("--gate-producer", action="store_true",
                    help="compute the retention gate in the kernel from its rank-16 projection "
                         "(gtr_gla_fwd_lowrank_gate, Sec. 3.1) instead of reading a stored log-gate")
    ap.add_argument("--no-secondary", action="store_true",
                    help="skip the 6400-token workload the default run also times")
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's batch size (smaller cases for profiling)")
    args = ap.parse_args()
    if args.graph:
        args.launch = "graph"
    if args.schedule != "auto":  # the graph is captured through the automatic schedule's entry points
        args.launch = "eager"
    return args


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_seed(w: wl.Workload, rank: int) -> int:
    """Seed of rank r's batch: every rank draws its own batch of the same workload
    (same distributions), so N ranks process N independent batches."""
    return 1234 + w.wid + 1000 * rank


def max_over_ranks(ms: float, pg, device) -> float:
    """The slowest rank's time (all-reduce MAX); `ms` itself without a process group."""
    if pg is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank_step: int, world: int, ms_per_step: float) -> float:
    """Whole-job throughput: the tokens of all ranks over the max-over-ranks step time."""
    return tokens_per_rank_step * world / (ms_per_step * 1e-3)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


# GB300 L2 size.  The buffer-rotation plan below is computed from this constant in
# both arms, so that they print the same config; the GPU arm also records the size
# the device reports.
L2_NOMINAL_BYTES = 129_000_000


def rotation_sets(step_bytes: int) -> int:
    """Input/output buffer sets a timed loop rotates through: enough that their
    total exceeds twice the L2 size, so that every step reads its inputs from HBM
    rather than from the L2 copy the previous step left behind."""
    if step_bytes >= 2 * L2_NOMINAL_BYTES:
        return 1
    return -(-2 * L2_NOMINAL_BYTES // step_bytes)


def l2_note(w: wl.Workload, n_sets: int) -> str:
    mb = w.algorithmic_bytes() / 1e6
    if n_sets == 1:
        return "inputs larger than L2 (%.0f MB per step > 2 x 129 MB)" % mb
    return ("rotating %d input/output buffer sets (%.2f MB per step, %.0f MB in all > 2 x 129 MB L2)"
            % (n_sets, mb, n_sets * mb))


def workload_config(w: wl.Workload, world: int, args=None, extra=None):
    """The `config` object of a JSON line; both arms print the same keys and values
    for the same command-line arguments."""
    cfg = {"workload": w.name, "B": w.B, "H": w.H, "grid": [w.grid_h, w.grid_w], "T": w.T,
           "Dk": w.Dk, "Dv": w.Dv, "tokens_per_step_per_gpu": w.B * w.T,
           "scan_orders": "alternating " + "/".join(wl.ORDER_NAMES[o] for o in w.orders),
           "final_state": w.final_state,
           "l2": l2_note(w, rotation_sets(w.algorithmic_bytes())),
           "parallelism": f"replicas x{world} (independent batches, no collective)"}
    if args is not None:
        cfg["schedule"] = args.schedule
        cfg["launch"] = ("one CUDA graph of the timed steps, replayed once" if args.launch == "graph"
                         else "eager, CUDA events around each step")
        if args.gated:
            cfg["epilogue"] = "output gate u = SiLU(r) * RMSNorm(o), second kernel right after the mixer"
        if getattr(args, "gate_producer", False):
            cfg["gate"] = ("computed in the kernel: g = logsigmoid(a W2 + b) / tau from a = x W1 (rank 16), "
                           "tau %g" % w.tau)
    if extra:
        cfg.update(extra)
    return cfg


# --------------------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, enabled: bool = True):
        self.gpu_index = gpu_index
        self.enabled = enabled
        self.proc = None
        self.path = None

    def __enter__(self):
        if not self.enabled:
            return self
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu_index}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            # the timed region starts once the sampler is running (its first sample written):
            # nvidia-smi's start-up overlapping the timed steps slowed them by ~2 %
            t0 = time.time()
            while time.time() - t0 < 5.0 and os.path.getsize(self.path) == 0:
                time.sleep(0.05)
            time.sleep(0.15)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        return False

    def summary(self):
        if not self.enabled or self.proc is None or not self.path:
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append(parts)
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            for n, val in zip(names, r[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(rows)}


# --------------------------------------------------------------------------------------
# CPU baseline: the fp64 oracle as it stands, on the host cores
# --------------------------------------------------------------------------------------

def time_oracle(w: wl.Workload, inp64, order: int, budget_s: float = 10.0, max_pairs=None):
    """Time the oracle over (b, h) pairs of the workload until ~budget_s of wall
    time is spent (at least one full pass over the chosen pairs)."""
    import oracle
    pairs_all = [(b, h) for b in range(w.B) for h in range(w.H)]
    pairs = pairs_all if max_pairs is None else pairs_all[:max_pairs]
    n_done, t0 = 0, time.perf_counter()
    while True:
        oracle.recurrence(inp64["q"], inp64["k"], inp64["v"], inp64["g"], w.grid_h, w.grid_w,
                          order, pairs=pairs)
        n_done += len(pairs)
        el = time.perf_counter() - t0
        if el >= budget_s or (max_pairs is None and el > 0.5 * budget_s):
            break
    tokens = n_done / w.H * w.T      # (b, h) pairs -> image tokens (all heads of a batch item)
    return tokens / el, el, n_done, oracle.max_threads()


def run_reference(args, w: wl.Workload, rank: int, world: int):
    """--impl reference: the oracle timed on the host cores, per step a bounded
    sample of the same workload (a prefix of its (b, h) pairs)."""
    if rank != 0:
        return
    import oracle
    inp = wl.workload_inputs(w)
    inp64 = {n: wl.storage_to_f64(inp[n], w.dtype) for n in ("q", "k", "v", "g")}
    del inp
    n_pairs = min(w.B * w.H, max(1, oracle.max_threads()))
    gp = None
    if args.gate_producer:  # the sampled images' gates come from the rank-16 projection, in the step
        nb = (n_pairs + w.H - 1) // w.H
        gpi = wl.gate_producer_inputs(w.B, w.H, w.T, w.Dk, w.dtype, rank_seed(w, rank) + 29, z_mean=w.z_mean,
                                       bias_std=0.0)
        gp = (wl.storage_to_f64(gpi["a"][:nb], w.dtype), wl.storage_to_f64(gpi["w2"], w.dtype),
              gpi["bias"].astype(np.float64), nb)

    def gates():
        if gp is None:
            return inp64["g"]
        g = np.zeros_like(inp64["g"])
        g[:gp[3]] = oracle.gate_producer(gp[0], gp[1], gp[2], w.tau)
        return g

    for i in range(args.warmup):
        oracle.recurrence(inp64["q"], inp64["k"], inp64["v"], gates(), w.grid_h, w.grid_w,
                          w.orders[i % len(w.orders)],
                          pairs=[(b, h) for b in range(w.B) for h in range(w.H)][:n_pairs])
    times = []
    for i in range(args.steps):
        order = w.orders[i % len(w.orders)]
        pairs = [(b, h) for b in range(w.B) for h in range(w.H)][:n_pairs]
        t0 = time.perf_counter()
        oracle.recurrence(inp64["q"], inp64["k"], inp64["v"], gates(), w.grid_h, w.grid_w,
                          order, pairs=pairs)
        times.append(time.perf_counter() - t0)
    per_step = sum(times) / len(times)
    tokens = n_pairs / w.H * w.T
    value = tokens / per_step
    sample = f"{n_pairs} of {w.B * w.H} (b,h) sequences of {w.T} tokens per step"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": per_step * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded, workload recipe)",
            "config": workload_config(w, world, args),
            "reference": "fp64 CPU oracle (oracle/), as it stands",
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.max_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------------------

def run_sswiglu(args, rank: int, world: int, local: int):
    """The Spatial SwiGLU step between its projections (Sec. 3.1, Eq. spatial_swiglu) on
    one S-SwiGLU workload: device-resident timing, roofline, CPU oracle and end to end."""
    if world > 1:
        raise SystemExit("--op sswiglu runs on one GPU")
    sw = wl.SWIGLU_WORKLOADS[args.sw_workload]
    inp = wl.sswiglu_inputs(sw.B, sw.grid_h, sw.grid_w, sw.F, sw.dtype, seed=2609 + sw.wid)
    metric = "tokens/s (Spatial SwiGLU gate-and-conv step)"
    cfg = {"workload": sw.name, "B": sw.B, "grid": [sw.grid_h, sw.grid_w], "T": sw.T, "F": sw.F,
           "layout": "one [B, T, 2F] projection output (gate | value)",
           "l2": "inputs larger than L2 (%.0f MB per step > 129 MB)" % (sw.algorithmic_bytes() / 1e6),
           "parallelism": "single GPU"}

    def time_cpu(budget_s=10.0):
        import oracle
        h64 = wl.storage_to_f64(inp["h"], sw.dtype)
        F, n, t0 = sw.F, 0, time.perf_counter()
        while True:  # one image at a time, all channels, until the budget is spent
            b = n % sw.B
            oracle.sswiglu_dwconv(h64[b:b + 1, :, :F], h64[b:b + 1, :, F:], inp["weight"], inp["bias"],
                                  sw.grid_h, sw.grid_w)
            n += 1
            el = time.perf_counter() - t0
            if el >= budget_s or n >= 4 * sw.B:
                return n * sw.T / el, el, n

    if args.impl == "reference":
        val, el, n = time_cpu(budget_s=max(5.0, 2.0 * args.steps))
        print(json.dumps({"impl": "reference", "metric": metric, "value": val, "unit": "tokens/s", "n_gpus": world,
                          "steps": args.steps, "warmup": args.warmup, "ms_per_step": sw.B * sw.T / val * 1e3,
                          "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                          "data": "synthetic", "config": cfg,
                          "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                                           "sample": f"{n} images x {sw.T} tokens x {sw.F} channels ({el:.1f} s)"},
                          "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                                  "d2h_bytes_per_step": 0}}), flush=True)
        return

    import torch
    from paper_2609_26590_gb300 import gla
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    gla.load()
    dt = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[sw.dtype]
    hh = torch.from_numpy(inp["h"].view(np.int16)).view(torch.bfloat16) if sw.dtype == "bf16" \
        else torch.from_numpy(inp["h"])
    h = hh.to(dev)
    wt = torch.from_numpy(inp["weight"]).to(dev)
    bs = torch.from_numpy(inp["bias"]).to(dev)
    out = torch.empty((sw.B, sw.T, sw.F), dtype=dt, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        gla.sswiglu_dwconv(h[:, :, :sw.F], h[:, :, sw.F:], wt, bs, sw.grid_h, sw.grid_w, out=out)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    with ClockSampler(local, enabled=not args.no_clocks) as clk:
        t_begin, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t_begin.record(stream)
        for i in range(args.steps):
            starts[i].record(stream)
            step()
            ends[i].record(stream)
        t_end.record(stream)
        torch.cuda.synchronize()
    if gla.sync_status() != 0:
        raise RuntimeError("device status word set during the timed region")
    ms_per_step = t_begin.elapsed_time(t_end) / args.steps
    value = sw.B * sw.T / (ms_per_step * 1e-3)
    kernel_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / args.steps
    peak, src = load_peaks()
    achieved = sw.algorithmic_bytes() / (kernel_ms * 1e-3) / 1e9
    traffic = None
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tpath):
        with open(tpath) as f:
            entry = json.load(f).get(f"{sw.name}:sswiglu")
            if isinstance(entry, dict):
                traffic = entry.get("dram_bytes")
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": traffic, "peak_source": f"{src} (MEASURED_PEAKS.json hbm_gbs)" if src == "measured"
                else "fallback", "kernel": "sswiglu_kernel (TMA value box with zero-padding halo, TMA gate box)",
                "kernel_ms": kernel_ms, "algorithmic_bytes_per_launch": sw.algorithmic_bytes()}
    # end to end: pinned host input -> device, the call, output -> pinned host, every step
    e2e = None
    if args.e2e_steps > 0:
        hin = hh.pin_memory()
        hout = torch.empty(out.shape, dtype=dt).pin_memory()
        for _ in range(2):
            h.copy_(hin, non_blocking=True); step(); hout.copy_(out, non_blocking=True)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.e2e_steps):
            h.copy_(hin, non_blocking=True)
            step()
            hout.copy_(out, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms = e0.elapsed_time(e1) / args.e2e_steps
        e2e = {"value": sw.B * sw.T / (e_ms * 1e-3), "unit": "tokens/s",
               "h2d_bytes_per_step": hin.numel() * hin.element_size(),
               "d2h_bytes_per_step": hout.numel() * hout.element_size()}
    cpu = None
    if not args.no_cpu_baseline:
        val, el, n = time_cpu()
        cpu = {"value": val, "unit": "tokens/s", "cores": 1, "kind": "oracle",
               "sample": f"{n} images x {sw.T} tokens x {sw.F} channels ({el:.1f} s wall, numpy fp64)"}
    print(json.dumps({"metric": metric, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
                      "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
                      "scaling": "weak", "vs_baseline": None, "dtype": sw.dtype,
                      "data": "synthetic (seeded, recipe in workloads.py)", "config": cfg, "roofline": roofline,
                      "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": args.steps, "clocks": clk.summary()}),
          flush=True)


def to_device(a: np.ndarray, dtype: str, dev):
    import torch
    if dtype == "bf16":
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev)
    return torch.from_numpy(a).to(dev)


def device_l2_bytes(dev) -> int:
    import torch
    return int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0))


def mixer_sets(w: wl.Workload, inp, dev, n_sets: int, gated: bool, seed: int):
    """n_sets device copies of the step's inputs and outputs (the same values at
    different addresses); the timed loop rotates through them."""
    import torch
    base = {n: to_device(inp[n], w.dtype, dev) for n in ("q", "k", "v", "g")}
    extra = {}
    if gated:
        rng = np.random.Generator(np.random.PCG64(seed + 17))
        extra["r"] = to_device(wl.round_to_storage(rng.standard_normal((w.B, w.T, w.H, w.Dv)) * 1.5, w.dtype),
                               w.dtype, dev)
        extra["w"] = torch.from_numpy((1.0 + 0.2 * rng.standard_normal(w.Dv)).astype(np.float32)).to(dev)
    sets = []
    for j in range(n_sets):
        s = {n: (t if j == 0 else t.clone()) for n, t in base.items()}
        if gated:
            s["r"] = extra["r"] if j == 0 else extra["r"].clone()
            s["w"] = extra["w"]
        s["out"] = torch.empty_like(s["v"])
        s["fs"] = (torch.empty((w.B, w.H, w.Dk, w.Dv), dtype=torch.float32, device=dev)
                   if w.final_state else None)
        sets.append(s)
    return sets


def timed_loop(run, steps: int, stream, clocks_enabled: bool, local: int, pg=None):
    """Time `steps` calls of run(i) on `stream` with CUDA events (one pair per step and
    one around the loop), bracketed by a barrier and a synchronize on both sides;
    nvidia-smi clocks are sampled during the loop."""
    import torch
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local, enabled=clocks_enabled) as clk:
        t_begin = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_begin.record(stream)
        for i in range(steps):
            starts[i].record(stream)
            run(i)
            ends[i].record(stream)
        t_end.record(stream)
        torch.cuda.synchronize()
    if pg:
        pg.barrier()
    per_launch = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    return t_begin.elapsed_time(t_end), per_launch, clk.summary()


TORCH_DT_NAMES = {"f32": "float32", "f16": "float16", "bf16": "bfloat16"}
SECONDARY_WORKLOAD = 3   # the 6400-token workload, timed after the headline in the same run


def time_mixer(args, w: wl.Workload, rank: int, world: int, local: int, dev, pg):
    """Device-resident timing of one mixer workload: warm-up, `args.steps` timed steps
    rotating through enough buffer sets to defeat the L2, the roofline of the step's
    kernel(s) and the clocks seen.  Returns a dict (the sets and host inputs stay in it
    for the end-to-end leg)."""
    import math

    import torch
    from paper_2609_26590_gb300 import gla

    dt = getattr(torch, TORCH_DT_NAMES[w.dtype])
    seed = rank_seed(w, rank)
    inp = wl.workload_inputs(w, B=w.B, seed=seed)
    n_sets = rotation_sets(w.algorithmic_bytes())
    sets = mixer_sets(w, inp, dev, n_sets, args.gated, seed)
    if args.gate_producer:  # the gate's low-rank inputs instead of the stored log-gate
        gp = wl.gate_producer_inputs(w.B, w.H, w.T, w.Dk, w.dtype, seed + 29, z_mean=w.z_mean, bias_std=0.0)
        for j, st in enumerate(sets):
            st["a"] = to_device(gp["a"], w.dtype, dev)
            st["w2"] = to_device(gp["w2"], w.dtype, dev)
            st["bias"] = torch.from_numpy(gp["bias"]).to(dev)
            del st["g"]
    stream = torch.cuda.current_stream(dev)
    orders = w.orders
    schedule = args.schedule
    tc = gla.tc_supported(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, orders[0], dt)
    kernel_name = "tensor-core chunkwise (tcgen05/TMEM/TMA)" if (tc and schedule != "simt") else "simt recurrence"
    ws_n = gla.workspace_bytes(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, dt) if tc and schedule != "simt" else 0
    split = not args.gate_producer and ws_n > 0 and gla.split_plan(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv,
                                         torch.cuda.get_device_properties(dev).multi_processor_count)[0] > 1
    launches_per_step = 2 if split else 1
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    if split:
        kernel_name += ", segment-summary pass + output pass"
    elif ws_n > 0 and not args.gate_producer and gla.balanced_plan(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, n_sm):
        kernel_name += ", balanced ranges (one CTA per SM, state hand-offs between them)"
    # the library fuses the output gate into the tensor-core kernel's stores for one key half and one
    # value slice when the sequences fill at most half of the SMs; otherwise it is one more kernel
    gate_fused = tc and schedule != "simt" and w.Dk <= 64 and w.Dv <= 64 and 2 * w.B * w.H <= n_sm
    if args.gated and gate_fused:
        kernel_name += ", output gate fused into the output stores"
    elif args.gated:
        launches_per_step += 1
        kernel_name += " + output-gate kernel"
    if args.gate_producer:
        if args.gated:
            raise SystemExit("--gate-producer runs without the output gate")
        kernel_name += ", retention gate computed in the kernel"

    def call(s, order, strm=None, ws=None, graph=False):
        if args.gate_producer:
            gla.forward_lowrank_gate(s["q"], s["k"], s["v"], s["a"], s["w2"], s["bias"], w.tau, w.grid_h, w.grid_w,
                                     order, out=s["out"], final_state=s["fs"], stream=strm)
        elif args.gated:
            gla.forward_gated(s["q"], s["k"], s["v"], s["g"], s["r"], s["w"], 1e-5, w.grid_h, w.grid_w, order,
                              out=s["out"], final_state=s["fs"], stream=strm, workspace=ws)
        elif graph:
            gla.forward_ws(s["q"], s["k"], s["v"], s["g"], w.grid_h, w.grid_w, order, s["out"], s["fs"], ws,
                           stream=strm)
        else:
            gla.forward(s["q"], s["k"], s["v"], s["g"], w.grid_h, w.grid_w, order, out=s["out"],
                        final_state=s["fs"], schedule=schedule)

    def step(i):
        call(sets[i % n_sets], orders[i % len(orders)])

    for i in range(max(3, args.warmup)):
        step(i)
    torch.cuda.synchronize()
    if gla.sync_status() != 0:
        raise RuntimeError("device status word set during warm-up")

    if args.launch == "graph":
        # the K timed steps captured once into one CUDA graph through the caller-workspace entry
        # points (no allocation, no synchronisation), rotating buffer sets and scan orders as
        # the eager loop does; replayed once untimed (upload), then once timed
        ws = torch.empty(ws_n, dtype=torch.uint8, device=dev) if ws_n else None
        for i in range(max(3, args.warmup)):
            s = sets[i % n_sets]
            call(s, orders[i % len(orders)], ws=ws, graph=True)
        torch.cuda.synchronize()
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cap):
            with torch.cuda.graph(graph, stream=cap):
                for i in range(args.steps):
                    call(sets[i % n_sets], orders[i % len(orders)], strm=cap, ws=ws, graph=True)
        stream.wait_stream(cap)
        graph.replay()
        torch.cuda.synchronize()
        if gla.sync_status() != 0:
            raise RuntimeError("device status word set during graph warm-up")
        total_ms, _, clocks = timed_loop(lambda i: graph.replay(), 1, stream, not args.no_clocks, local, pg)
        per_launch_ms = [total_ms / args.steps] * args.steps
        timing = "CUDA events around one replay of the graph of all timed steps, divided by the steps"
        # the same steps as eager calls, for comparison (not the headline)
        e_total, e_per, _ = timed_loop(step, args.steps, stream, False, local, pg)
        eager = {"ms_per_step": max_over_ranks(e_total, pg, dev) / args.steps,
                 "kernel_ms": sum(e_per) / len(e_per),
                 "timing": "CUDA events around each eager step"}
    else:
        total_ms, per_launch_ms, clocks = timed_loop(step, args.steps, stream, not args.no_clocks, local, pg)
        timing = "CUDA events around each step on the launching stream"
        eager = None
    if gla.sync_status() != 0:
        raise RuntimeError("device status word set during the timed region")
    total_ms = max_over_ranks(total_ms, pg, dev)
    ms_per_step = total_ms / args.steps
    value = job_tokens_per_s(w.B * w.T, world, ms_per_step)

    hbm_peak, peak_src = load_peaks()
    alg_bytes = w.algorithmic_bytes()
    if args.gated:  # the gate's pre-activation is read once more per token-head (u replaces o)
        alg_bytes += w.B * w.T * w.H * w.Dv * wl.ELEM_SIZE[w.dtype]
    if args.gate_producer:  # no g tensor; a (rank 16 per token), W2 and the bias instead
        es = wl.ELEM_SIZE[w.dtype]
        alg_bytes += (- w.B * w.T * w.H * w.Dk * es + w.B * w.T * wl.GATE_RANK * es
                      + w.H * wl.GATE_RANK * w.Dk * es + w.H * w.Dk * 4)
    kernel_ms = sum(per_launch_ms) / len(per_launch_ms)
    achieved = alg_bytes / (kernel_ms * 1e-3) / 1e9
    traffic, traffic_note = None, None
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tpath) and not args.gated and not args.gate_producer and args.batch is None:
        with open(tpath) as f:
            tj = json.load(f)
        entry = tj.get(f"{w.name}:{'tc' if (tc and schedule != 'simt') else 'simt'}")
        if isinstance(entry, dict):
            traffic, traffic_note = entry.get("dram_bytes"), entry.get("note")
    roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                "frac": achieved / hbm_peak, "traffic": traffic,
                "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured" else "fallback",
                "kernel": kernel_name, "kernel_ms": kernel_ms, "algorithmic_bytes_per_launch": alg_bytes,
                "timing": timing}
    if eager is not None:
        roofline["eager"] = dict(eager, frac=alg_bytes / (eager["kernel_ms"] * 1e-3) / 1e9 / hbm_peak)
    if traffic_note:
        roofline["traffic_note"] = traffic_note
    return {"w": w, "inp": inp, "sets": sets, "value": value, "ms_per_step": ms_per_step,
            "roofline": roofline, "clocks": clocks, "launches": args.steps * launches_per_step,
            "n_sets": n_sets, "dt": dt, "tc": tc}


def time_e2e(args, res, world: int, dev, pg):
    """End to end through gtr_gla_fwd_host: pinned host inputs in, outputs back to
    pinned host memory, every step inside the timed region.  Beside it, the host
    link's own rate: plain pinned copies of the same bytes, each direction alone and
    both at once, so that the e2e number can be read against what the link gives."""
    import torch
    from paper_2609_26590_gb300 import gla

    w, inp, dt = res["w"], res["inp"], res["dt"]
    stream = torch.cuda.current_stream(dev)
    orders = w.orders
    host = {n: (torch.from_numpy(inp[n].view(np.int16)).view(torch.bfloat16) if w.dtype == "bf16"
                else torch.from_numpy(inp[n])).pin_memory() for n in ("q", "k", "v", "g")}
    hout = torch.empty(host["v"].shape, dtype=host["v"].dtype).pin_memory()
    hfs = torch.empty((w.B, w.H, w.Dk, w.Dv), dtype=torch.float32).pin_memory() if w.final_state else None
    nbytes = gla.host_buffer_bytes(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, dt, w.final_state)
    dbuf = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    for i in range(2):
        gla.forward_host(host["q"], host["k"], host["v"], host["g"], w.grid_h, w.grid_w,
                         orders[i % len(orders)], hout, hfs, dbuf)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(args.e2e_steps):
        gla.forward_host(host["q"], host["k"], host["v"], host["g"], w.grid_h, w.grid_w,
                         orders[i % len(orders)], hout, hfs, dbuf)
    e1.record(stream)
    torch.cuda.synchronize()
    if gla.sync_status() != 0:
        raise RuntimeError("device status word set during the end-to-end leg")
    e_ms = max_over_ranks(e0.elapsed_time(e1), pg, dev) / args.e2e_steps
    h2d = sum(host[n].numel() * host[n].element_size() for n in ("q", "k", "v", "g"))
    d2h = hout.numel() * hout.element_size() + (hfs.numel() * 4 if hfs is not None else 0)

    # the link alone: one cudaMemcpyAsync per tensor (torch copy_ of pinned memory)
    s0 = res["sets"][0]
    dins = [s0[n] for n in ("q", "k", "v", "g")]
    douts = [(hout, s0["out"])] + ([(hfs, s0["fs"])] if hfs is not None else [])
    side = torch.cuda.Stream(dev)
    reps = 3

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    def up():
        for d, n in zip(dins, ("q", "k", "v", "g")):
            d.copy_(host[n], non_blocking=True)

    def down():
        for h, d in douts:
            h.copy_(d, non_blocking=True)

    def both():  # uploads on the launching stream, downloads on a second one at the same time
        side.wait_stream(stream)
        up()
        with torch.cuda.stream(side):
            down()
        stream.wait_stream(side)

    up_ms, down_ms, both_ms = timed(up), timed(down), timed(both)
    tokens = w.B * w.T
    return {"value": job_tokens_per_s(tokens, world, e_ms), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e_ms,
            "api": "gtr_gla_fwd_host (pinned host buffers)",
            "link": {"e2e_gbs": (h2d + d2h) / (e_ms * 1e-3) / 1e9,
                     "h2d_alone_gbs": h2d / (up_ms * 1e-3) / 1e9,
                     "d2h_alone_gbs": d2h / (down_ms * 1e-3) / 1e9,
                     "both_at_once_gbs": (h2d + d2h) / (both_ms * 1e-3) / 1e9,
                     "copies_only_ms_per_step": both_ms,
                     "how": "plain pinned cudaMemcpyAsync of the step's bytes, one per tensor, in the same run"}}


def main():
    args = parse()
    rank, world, local = dist_env()
    if args.op == "sswiglu":
        run_sswiglu(args, rank, world, local)
        return
    w = wl.WORKLOADS[args.workload]
    if args.batch is not None:
        import dataclasses
        w = dataclasses.replace(w, B=args.batch, name=f"{w.name}_b{args.batch}")
    if args.impl == "reference":
        run_reference(args, w, rank, world)
        return

    import torch
    from paper_2609_26590_gb300 import gla

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    gla.load()

    res = time_mixer(args, w, rank, world, local, dev, pg)
    head = {k: res[k] for k in ("value", "ms_per_step", "roofline", "clocks", "launches")}
    # the host-buffer entry point runs the plain mixer: no end-to-end leg for the gated and
    # gate-producer variants, and the oracle baseline times the plain mixer's inputs
    e2e = (time_e2e(args, res, world, dev, pg)
           if args.e2e_steps > 0 and not args.gated and not args.gate_producer else None)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not args.gate_producer:
        inp64 = {n: wl.storage_to_f64(res["inp"][n], w.dtype) for n in ("q", "k", "v", "g")}
        val, el, n_pairs, cores = time_oracle(w, inp64, w.orders[0], budget_s=10.0)
        cpu = {"value": val, "unit": "tokens/s", "cores": cores, "kind": "oracle",
               "sample": f"{n_pairs} (b,h) sequences x {w.T} tokens ({el:.1f} s wall), "
                         f"order {wl.ORDER_NAMES[w.orders[0]]}"}
        del inp64

    secondary = None
    if (args.workload == DEFAULT_WORKLOAD and args.batch is None and not args.gated and not args.no_secondary
            and args.schedule == "auto"):
        # the 6400-token workload in the same run (the second length of the target)
        del res
        torch.cuda.empty_cache()
        w2 = wl.WORKLOADS[SECONDARY_WORKLOAD]
        r2 = time_mixer(args, w2, rank, world, local, dev, pg)
        secondary = {"workload": w2.name, "metric": "GLA-forward tokens/s (GB300, device-timed) and % of roofline "
                                                    "at 6400 tokens",
                     "value": r2["value"], "unit": "tokens/s", "ms_per_step": r2["ms_per_step"],
                     "steps": args.steps, "dtype": w2.dtype, "roofline": r2["roofline"], "clocks": r2["clocks"],
                     "gpu_launches": r2["launches"],
                     "config": workload_config(w2, world, args), "token_heads_per_s": r2["value"] * w2.H}
    if rank == 0:
        line = {"metric": METRIC, "value": head["value"], "unit": "tokens/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": head["ms_per_step"],
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": w.dtype, "data": "synthetic (seeded, workload recipe in workloads.py)",
                "config": workload_config(w, world, args),
                "roofline": head["roofline"], "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": head["launches"], "clocks": head["clocks"],
                "token_heads_per_s": head["value"] * w.H, "l2_device_bytes": device_l2_bytes(dev),
                "secondary": secondary}
        print(json.dumps(line), flush=True)
    if pg:
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
