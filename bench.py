#!/usr/bin/env python
"""Optimizer steps/s of the MALT update over the GPT-2 Large 2-D parameter set.

One step = one malt_step over all 144 matrices (36 layers x {1280x3840,
1280x1280, 1280x5120, 5120x1280}, bf16 weights, fp32 state and gradients,
5 Newton-Schulz iterations): statistics + momentum, preconditioners,
prescale, the Newton-Schulz GEMMs, graft and apply.  The working set
(about 15 GB) is far larger than L2, so no flush is needed between steps.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference]

N > 1 runs under torch.distributed.run with one process per GPU; each rank
updates its own replica of the parameter set (independent problems, no
collective on the data path) and the value is N * K / (max over ranks of the
timed region).  Prints one JSON line on rank 0.
"""
from __future__ import annotations

import argparse
import dataclasses
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

METRIC = "optimizer steps/sec (full GPT-2 param set, 1 GB300)"
UNIT = "steps/s"
DEFAULT_WORKLOAD = "gpt2_large"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
NCU_SUMMARY = os.path.join(ROOT, "profiles", "ns_gemm_gpt2_large_ncu.json")
# The sources the Newton-Schulz kernel compiles from: the traffic figure of
# the committed ncu summary holds only while all of them are unchanged.
NS_SOURCES = [os.path.join(ROOT, "paper_2608_05088_gb300", "csrc", f)
              for f in ("ns_gemm.cu", "common.cuh", "ptx.cuh")]


def ns_sources_sha256() -> str:
    h = hashlib.sha256()
    for path in NS_SOURCES:
        with open(path, "rb") as f:
            h.update(hashlib.sha256(f.read()).digest())
    return h.hexdigest()
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# --------------------------------------------------------------------- ranks
def rank_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def init_dist(backend: str):
    import torch.distributed as dist
    rank, world, _ = rank_env()
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return rank, world


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def host_link_bound(g_host, g_dev, w_dev, w_host, step_ms, e2e_per_gpu, reps=5):
    """The host link's bound on the end-to-end rate: the same per-tensor
    copies as one host step (every gradient in, every weight out), timed
    alone in each direction and both directions at once, with no kernels
    running.  A pipelined host step can go no faster than the slower of the
    device-resident step and the concurrent copies."""
    import torch
    up, down = torch.cuda.Stream(), torch.cuda.Stream()

    def h2d():
        with torch.cuda.stream(up):
            for d, h in zip(g_dev, g_host):
                d.copy_(h, non_blocking=True)

    def d2h():
        with torch.cuda.stream(down):
            for h, d in zip(w_host, w_dev):
                h.copy_(d, non_blocking=True)

    def both():
        h2d()
        d2h()

    def wall_ms(fn):
        # median of single runs: the host link on these machines now and then
        # stalls a copy for tens of milliseconds
        fn()
        torch.cuda.synchronize()
        times = []
        for _ in range(reps):
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            times.append((time.perf_counter() - t0) * 1e3)
        return statistics.median(times)

    bi = sum(t.numel() * t.element_size() for t in g_host)
    bo = sum(t.numel() * t.element_size() for t in w_host)
    t_in, t_out, t_both = wall_ms(h2d), wall_ms(d2h), wall_ms(both)
    bound_ms = max(step_ms, t_both)
    return {"h2d_gbs": bi / t_in / 1e6, "d2h_gbs": bo / t_out / 1e6,
            "concurrent_ms": t_both, "device_step_ms": step_ms,
            "bound_steps_per_s": 1e3 / bound_ms,
            "frac": e2e_per_gpu * bound_ms / 1e3,
            "bound": "host link" if t_both > step_ms else "device step"}


def max_over_ranks(x: float, device=None) -> float:
    """Maximum of a host scalar over all ranks (timing only, never data)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# -------------------------------------------------------------------- clocks
THROTTLE_REASONS = {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}


class ClockSampler:
    """nvidia-smi sampled every 50 ms around the timed region; the summary
    keeps the samples whose timestamps fall inside it (begin() .. end()).
    The sampler starts before the region so that its own start-up does not
    eat into it.  If no timestamp can be read, every sample counts."""

    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    INTERVAL_MS = 50
    STARTUP_S = 0.5

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None
        self.t0 = None
        self.t1 = None

    def start(self):
        """Start sampling (call before the timed region)."""
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", str(self.INTERVAL_MS)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(self.STARTUP_S)
        except Exception:
            self.proc = None

    def begin(self):
        self.t0 = time.time()

    def end(self):
        self.t1 = time.time()

    @staticmethod
    def _stamp(v):
        from datetime import datetime
        try:
            return datetime.strptime(v.strip(), "%Y/%m/%d %H:%M:%S.%f").timestamp()
        except ValueError:
            return None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(2.0 * self.INTERVAL_MS / 1e3)      # the sample after end()
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 10:
                    rows.append(parts)
        os.unlink(self.path)
        try:
            return self.summarise(rows, self.t0, self.t1)
        except Exception:
            return self.summarise(rows, None, None)

    @classmethod
    def summarise(cls, rows, t0, t1):
        """Median SM clock, maximum clock and the throttle reasons seen in the
        samples taken between t0 and t1 (all samples if none is dated)."""
        if not rows:
            return None
        window = "timed region"
        inside = rows
        stamps = [cls._stamp(r[0]) for r in rows]
        if t0 is not None and t1 is not None and all(t is not None for t in stamps):
            inside = [r for r, t in zip(rows, stamps) if t0 <= t <= t1]
            if not inside:     # region shorter than the interval: the sample nearest its middle
                mid = 0.5 * (t0 + t1)
                inside = [min(zip(rows, stamps), key=lambda rt: abs(rt[1] - mid))[0]]
                window = "nearest sample to the timed region"
        else:
            window = "all samples (timestamps unreadable)"

        def num(v):
            try:
                return float(v)
            except ValueError:
                return float("nan")
        sm = [num(r[2]) for r in inside]
        mx = max(num(r[3]) for r in rows)
        reasons = set()
        for r in inside:
            for name, v in zip(("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                                "sw_power_cap"), r[6:10]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        good = [x for x in sm if not math.isnan(x)]
        return {"sm_mhz": statistics.median(good) if good else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(inside), "samples_total": len(rows),
                "interval_ms": cls.INTERVAL_MS, "window": window}


# -------------------------------------------------------------------- peaks
def peaks():
    try:
        with open(PEAKS_FILE) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return FALLBACK_PEAKS, "fallback"


def ncu_tensor_pipe():
    """Tensor-pipe busy % of peak of the Gram, Poly and B*X launches from the
    committed ncu summary, weighted by their captured durations (the NS mix
    of one iteration), or None when a kernel source changed since."""
    try:
        with open(NCU_SUMMARY) as f:
            s = json.load(f)
        if s.get("ns_sources_sha256") != ns_sources_sha256():
            return None
        tp = s["tensor_pipe_pct_of_peak_elapsed"]
        dur = tp["durations_us"]
        kinds = ("gram", "poly", "bx")
        mix = sum(tp[k] * dur[k] for k in kinds) / sum(dur[k] for k in kinds)
        return {"per_product": {k: tp[k] for k in kinds}, "duration_weighted": round(mix, 2),
                "source": "ncu, first 12 GPT-2 Large layers (profiles/ns_gemm_gpt2_large_first12l.md)"}
    except Exception:
        return None


def ncu_traffic_per_launch(persistent: bool):
    """DRAM bytes per NS GEMM launch (of the schedule the timed steps used)
    from the committed ncu summary, or None when a kernel source changed
    since the capture or the summary has no figure for the schedule."""
    try:
        with open(NCU_SUMMARY) as f:
            s = json.load(f)
        if s.get("ns_sources_sha256") != ns_sources_sha256():
            return None
        key = "persistent_dram_bytes_per_launch_full_size" if persistent else \
              "dram_bytes_per_launch_full_size"
        return float(s[key])
    except Exception:
        return None


# ------------------------------------------------------------ CPU baseline
def oracle_full_step_time(wl, step=0):
    """Seconds of one oracle step over EVERY matrix of the workload (fp64,
    numpy's BLAS on all host cores), each matrix from zero state with its
    gradient of `step`.  Inputs are drawn before each matrix's clock starts;
    only the malt_step_ref calls are timed.  One matrix is held at a time."""
    import numpy as np
    import oracle.malt_ref as ref
    from paper_2608_05088_gb300 import inputs
    hp = ref.Hyper(lr=wl.lr, ns_steps=wl.ns_steps)
    total = 0.0
    for i, shape in enumerate(wl.shapes):
        W = inputs.initial_weight(wl, i).astype(np.float64)
        G = inputs.gradient(wl, i, step).astype(np.float64)
        st = ref.State.zeros(*shape)
        t0 = time.perf_counter()
        ref.malt_step_ref(W, G, st, hp, variant=wl.variant, weight_dtype=wl.weight_dtype)
        total += time.perf_counter() - t0
    return total


def oracle_warmup(wl, matrices=4):
    """One untimed oracle step of the first matrices (BLAS threads and pages)."""
    import numpy as np
    import oracle.malt_ref as ref
    from paper_2608_05088_gb300 import inputs
    hp = ref.Hyper(lr=wl.lr, ns_steps=wl.ns_steps)
    for i in range(min(matrices, len(wl.shapes))):
        ref.malt_step_ref(inputs.initial_weight(wl, i).astype(np.float64),
                          inputs.gradient(wl, i, 0).astype(np.float64),
                          ref.State.zeros(*wl.shapes[i]), hp, variant=wl.variant,
                          weight_dtype=wl.weight_dtype)


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


# ----------------------------------------------------------------- reference
def run_reference(args):
    """The fp64 oracle timed on the host cores: one warm-up step over one
    layer's matrices, then ONE timed step over the whole parameter set (about
    a minute for GPT-2 Large on 16 cores; the requested step count would take
    many minutes).  The line reports the steps actually timed."""
    rank, world, _ = rank_env()
    if rank != 0:
        return
    from paper_2608_05088_gb300 import inputs
    wl = inputs.WORKLOADS[args.workload]
    oracle_warmup(wl)
    t_step = oracle_full_step_time(wl)
    value = 1.0 / t_step
    sample = (f"one full step of all {len(wl.shapes)} matrices of {wl.name} (each from zero "
              f"state), after one warm-up step of 4 matrices")
    out = {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference",
           "n_gpus": world, "steps": 1, "warmup": 1,
           "requested": getattr(args, "requested", {"steps": args.steps, "warmup": args.warmup}),
           "ms_per_step": t_step * 1e3, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": dict(workload_config(wl), ns_schedule=args.ns_schedule),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(),
                            "kind": "oracle", "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def workload_config(wl):
    return {"workload": wl.name, "matrices": len(wl.shapes),
            "shapes": sorted(set(f"{m}x{n}" for m, n in wl.shapes)),
            "elements": wl.elements, "variant": wl.variant, "ns_steps": wl.ns_steps,
            "weights": wl.weight_dtype, "state": "f32", "gradients": "f32",
            "lr": wl.lr, "l2": "inputs larger than L2 (working set ~%.0f GB)" % (
                wl.elements * 26 / 1e9)}


# ------------------------------------------------------- cuBLAS comparison
def run_compare_cublas(args):
    """The GEMM shape of GPT-2 Large's B*X product for its 36 1280x5120
    matrices, timed through cuBLAS and through the library (context for the
    Newton-Schulz kernel's tensor-pipe efficiency; not a bench line)."""
    import torch
    import paper_2608_05088_gb300.malt as malt
    from paper_2608_05088_gb300 import build, inputs
    build.build()
    dev = torch.device("cuda:0")
    flops = 2.0 * 36 * 1280 * 1280 * 5120
    a = torch.randn(36, 1280, 1280, device=dev, dtype=torch.bfloat16)
    b = torch.randn(36, 1280, 5120, device=dev, dtype=torch.bfloat16)
    for _ in range(args.warmup):
        torch.matmul(a, b)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        torch.matmul(a, b)
    e1.record()
    torch.cuda.synchronize()
    cub_ms = e0.elapsed_time(e1) / args.steps
    del a, b
    wl = inputs.Workload("bx36", 81, ((1280, 5120),) * 36, "bf16", 1.5, 0.0007, "malt", 1)
    W = [torch.from_numpy(w).to(dev).to(torch.bfloat16) for w in inputs.initial_weights(wl)]
    G = [torch.from_numpy(g).to(dev) for g in inputs.gradients_for_step(wl, 0)]
    M = [torch.empty(s_, dtype=torch.float32, device=dev) for s_ in wl.shapes]
    l = [torch.empty(s_[0], dtype=torch.float32, device=dev) for s_ in wl.shapes]
    r = [torch.empty(s_[1], dtype=torch.float32, device=dev) for s_ in wl.shapes]
    opt = malt.MaltOptimizer(list(zip(W, G, M, l, r)))
    opt.set_ns_schedule(malt.MALT_NS_PHASED)
    hp = malt.hparams(lr=wl.lr)
    for _ in range(args.warmup):
        opt.step(hp)
    torch.cuda.synchronize()
    opt.profile(True)
    opt.profile_read()
    for _ in range(max(1, args.steps // 5)):
        opt.step(hp)
    prof = opt.profile_read()
    opt.profile(False)
    ours_ms = prof["ns_bx"][0] / prof["ns_bx"][1]
    opt.close()
    print(json.dumps({"compare": "B*X product, 36 x (1280x1280 @ 1280x5120) bf16",
                      "cublas_ms": cub_ms, "cublas_tflops": flops / cub_ms / 1e9,
                      "library_ms": ours_ms, "library_tflops": flops / ours_ms / 1e9}), flush=True)


STRESS_SHAPES = ((4096, 4096), (4096, 16384), (16384, 4096))


def run_stress_sweep(args):
    """The shape / anisotropy stress set: one large bf16 matrix with fp32
    state per case (4096^2, 4096x16384, 16384x4096; row / column scale sigma
    in {0, 1, 3}; 5 or 8 Newton-Schulz iterations).  Per case, one JSON line:
    steps/s, the Newton-Schulz products' rate against the measured sustained
    bf16 peak, and the statistics / prescale / apply kernels' HBM rate
    against the measured copy bandwidth (device-resident inputs, CUDA events
    of the library's per-kernel profiling).  Not a bench line."""
    import torch
    import paper_2608_05088_gb300.malt as malt
    from paper_2608_05088_gb300 import build, inputs
    build.build()
    dev = torch.device("cuda:0")
    pk, pk_src = peaks()
    sigmas = (0.0, 1.0, 3.0) if args.stress_sigma is None else (args.stress_sigma,)
    ks = (5, 8) if args.stress_k is None else (args.stress_k,)
    for rows, cols in STRESS_SHAPES:
        for sigma in sigmas:
            for k in ks:
                wl = inputs.stress_workload(rows, cols, sigma, k)
                W = [torch.from_numpy(w).to(dev).to(torch.bfloat16) for w in inputs.initial_weights(wl)]
                G = [torch.from_numpy(g).to(dev) for g in inputs.gradients_for_step(wl, 0)]
                M = [torch.empty(s_, dtype=torch.float32, device=dev) for s_ in wl.shapes]
                l = [torch.empty(s_[0], dtype=torch.float32, device=dev) for s_ in wl.shapes]
                r = [torch.empty(s_[1], dtype=torch.float32, device=dev) for s_ in wl.shapes]
                opt = malt.MaltOptimizer(list(zip(W, G, M, l, r)))
                hp = malt.hparams(lr=wl.lr, ns_steps=k)
                for _ in range(args.warmup):
                    opt.step(hp)
                torch.cuda.synchronize()
                opt.profile(True)
                opt.profile_read()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                for _ in range(args.steps):
                    opt.step(hp)
                e1.record()
                torch.cuda.synchronize()
                prof = opt.profile_read()
                opt.profile(False)
                if opt.check() != malt.MALT_OK:
                    raise SystemExit(f"stress step failed: {wl.name}")
                t_ms = e0.elapsed_time(e1) / args.steps
                ns_ms = sum(prof[x][0] for x in malt.NS_KINDS) / args.steps
                ns_tf = wl.ns_flops_min() / (ns_ms / 1e3) / 1e12
                elems = wl.elements
                mem = {}
                for kind, bpe in (("stats", 12.0), ("prescale", 6.0), ("apply", 6.0)):
                    ms = prof[kind][0] / args.steps
                    gbs = bpe * elems / (ms / 1e3) / 1e9
                    mem[kind] = {"ms": round(ms, 4), "GB/s": round(gbs, 1),
                                 "frac_of_hbm": round(gbs / float(pk["hbm_gbs"]), 3)}
                print(json.dumps({
                    "case": wl.name, "shape": f"{rows}x{cols}", "sigma": sigma, "ns_steps": k,
                    "steps_per_s": round(1e3 / t_ms, 2), "ms_per_step": round(t_ms, 4),
                    "ns": {"ms": round(ns_ms, 4), "tflops_symmetric": round(ns_tf, 1),
                           "frac_of_sustained_bf16": round(ns_tf / float(pk["bf16_tflops_sustained"]), 3),
                           "schedule": "persistent" if prof["ns_persistent"][1] > 0 else "phased"},
                    "hbm": mem, "peaks": pk_src}), flush=True)
                opt.close()
                del W, G, M, l, r
                torch.cuda.empty_cache()


# ----------------------------------------------------------- whole optimizer
ADAMW_BYTES_PER_ELEM = 30.0     # g 4, w 4+4, m 4+4, v 4+4, bf16 copy 2


def run_whole_optimizer_leg(args, wl, G, dev, stream):
    """The whole optimizer step of the model (Section 5.1 parameter grouping):
    MALT on the 2-D matrices with fp32 master weights, their bf16 copies and
    decoupled weight decay 0.1 (appendix table), plus AdamW on the other
    tensors (embeddings, tied head, LayerNorms, biases) at the AdamW learning
    rate, both on one stream.  The matrices read the timed workload's
    gradients G.  Reports ms per whole step, the AdamW launch's own time and
    HBM rate, and the apply pass (which now also writes the copies)."""
    import torch
    import paper_2608_05088_gb300.malt as malt
    from paper_2608_05088_gb300 import inputs
    base = wl.name.split("_first")[0]
    if base not in inputs.ADAMW_SETS:
        return None
    aset = inputs.ADAMW_SETS[base]
    W = [torch.from_numpy(w).to(dev) for w in inputs.initial_weights(
        dataclasses.replace(wl, weight_dtype="f32"))]
    copies = [torch.empty(s_, dtype=torch.bfloat16, device=dev) for s_ in wl.shapes]
    M = [torch.empty(s_, dtype=torch.float32, device=dev) for s_ in wl.shapes]
    l = [torch.empty(s_[0], dtype=torch.float32, device=dev) for s_ in wl.shapes]
    r = [torch.empty(s_[1], dtype=torch.float32, device=dev) for s_ in wl.shapes]
    others = []
    for i, (_, shape, wd) in enumerate(aset.tensors):
        w = torch.from_numpy(inputs.adamw_initial(aset, i)).to(dev)
        others.append((w, torch.empty(shape, dtype=torch.bfloat16, device=dev),
                       torch.from_numpy(inputs.adamw_gradient(aset, i, 0)).to(dev),
                       torch.empty(shape, dtype=torch.float32, device=dev),
                       torch.empty(shape, dtype=torch.float32, device=dev), wd))
    whole = malt.WholeOptimizer(list(zip(W, G, M, l, r)), others, copies=copies)
    hp = malt.hparams(lr=wl.lr, ns_steps=wl.ns_steps, weight_decay=0.1)
    ahp = malt.adamw_hparams(lr=aset.lr)
    malter = wl.variant == "malter"
    for _ in range(args.warmup):
        whole.step(hp, ahp, malter=malter)
    torch.cuda.synchronize()
    if whole.check() != malt.MALT_OK:
        raise SystemExit("whole-optimizer warm-up step failed")
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        whole.step(hp, ahp, malter=malter)
    e1.record(stream)
    torch.cuda.synchronize()
    t_whole = max_over_ranks(e0.elapsed_time(e1), dev) / args.steps
    # the AdamW launches alone, and the MALT apply pass, from their own events
    whole.malt.profile(True)
    whole.malt.profile_read()
    a0 = torch.cuda.Event(enable_timing=True)
    a1 = torch.cuda.Event(enable_timing=True)
    t_adam = 0.0
    for _ in range(args.steps):
        whole.malt.step(hp, malter=malter)
        a0.record(stream)
        whole.adamw.step(ahp)
        a1.record(stream)
        torch.cuda.synchronize()
        t_adam += a0.elapsed_time(a1)
    prof = whole.malt.profile_read()
    whole.malt.profile(False)
    if whole.check() != malt.MALT_OK:
        raise SystemExit("whole-optimizer step failed")
    t_adam /= args.steps
    pk, pk_src = peaks()
    gbs = ADAMW_BYTES_PER_ELEM * aset.elements / (t_adam / 1e3) / 1e9
    apply_ms = prof["apply"][0] / args.steps
    apply_bpe = 4.0 + 4.0 + 2.0 + 2.0            # W fp32 read+write, O read, copy write
    out = {"ms_per_step": t_whole, "value": world_size() / (t_whole / 1e3), "unit": UNIT,
           "matrices": len(wl.shapes), "matrix_elements": wl.elements,
           "adamw_tensors": len(aset.tensors), "adamw_elements": aset.elements,
           "parameters": wl.elements + aset.elements,
           "malt": f"{wl.variant}, fp32 master weights with bf16 copies, weight decay 0.1, lr {wl.lr}",
           "adamw": f"betas (0.9, 0.95), eps 1e-8, lr {aset.lr}, weight decay 0.1 on the "
                    f"embeddings, 0 on vectors, bf16 copies",
           "adamw_kernel": {"ms_per_step": t_adam, "bytes_per_elem": ADAMW_BYTES_PER_ELEM,
                            "achieved_gbs": gbs, "frac_of_hbm": gbs / float(pk["hbm_gbs"])},
           "apply_with_copies": {"ms_per_step": apply_ms, "bytes_per_elem": apply_bpe,
                                 "achieved_gbs": apply_bpe * wl.elements / (apply_ms / 1e3) / 1e9},
           "peaks": pk_src}
    whole.close()
    return out


def world_size():
    return rank_env()[1]


# --------------------------------------------------------------------- MALT
def run_malt(args):
    import numpy as np
    import torch
    rank, world = init_dist("nccl")
    _, _, local = rank_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import paper_2608_05088_gb300.malt as malt
    from paper_2608_05088_gb300 import build, inputs
    build.build()
    wl = inputs.WORKLOADS[args.workload]
    if args.layers:
        wl = inputs.first_layers(wl, args.layers)
    n = len(wl.shapes)
    wdt = torch.bfloat16 if wl.weight_dtype == "bf16" else torch.float32

    # Inputs: drawn on the host once, made resident in HBM before timing.
    W0 = inputs.initial_weights(wl)
    G_host = [torch.from_numpy(g).pin_memory() for g in inputs.gradients_for_step(wl, 0)]
    W = [torch.from_numpy(w).to(dev).to(wdt) for w in W0]
    G = [g.to(dev) for g in G_host]
    M = [torch.empty(s, dtype=torch.float32, device=dev) for s in wl.shapes]
    l = [torch.empty(s[0], dtype=torch.float32, device=dev) for s in wl.shapes]
    r = [torch.empty(s[1], dtype=torch.float32, device=dev) for s in wl.shapes]
    params = list(zip(W, G, M, l, r))
    opt = malt.MaltOptimizer(params)
    hp = malt.hparams(lr=wl.lr, ns_steps=wl.ns_steps)
    malter = wl.variant == "malter"
    stream = torch.cuda.current_stream()
    sched_code = {"auto": malt.MALT_NS_AUTO, "phased": malt.MALT_NS_PHASED,
                  "persistent": malt.MALT_NS_PERSISTENT}[args.ns_schedule]
    opt.set_ns_schedule(sched_code)

    for _ in range(args.warmup):
        opt.step(hp, malter=malter)
    torch.cuda.synchronize()
    status = opt.check()
    if status != malt.MALT_OK:
        raise SystemExit(f"warm-up step failed: {malt.status_string(status)}")

    # ---- device-resident timed region
    def timed_region():
        opt.profile(True)
        opt.profile_read()
        clocks = ClockSampler(local)
        clocks.start()
        barrier()
        torch.cuda.synchronize()
        clocks.begin()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            opt.step(hp, malter=malter)
        e1.record(stream)
        torch.cuda.synchronize()
        clocks.end()
        barrier()
        clk = clocks.stop()
        prof = opt.profile_read()
        opt.profile(False)
        status = opt.check()
        if status != malt.MALT_OK:
            raise SystemExit(f"timed step failed: {malt.status_string(status)}")
        return max_over_ranks(e0.elapsed_time(e1), dev), clk, prof

    t_ms, clk, prof = timed_region()
    # A region that saw the GPU slowed by hardware or thermal limits is
    # measured once more (the power cap alone is normal under a dense GEMM).
    throttled = sorted(set((clk or {}).get("reasons", [])) & THROTTLE_REASONS)
    if throttled:
        t_ms, clk, prof = timed_region()
        if clk is not None:
            clk["remeasured_after"] = throttled
    value = world * args.steps / (t_ms / 1e3)

    # ---- the same step with each Newton-Schulz schedule forced (one launch
    # per product, or one persistent launch for all products), for
    # comparison with the default, which picks one per launch group.
    sched = None
    if not args.no_muon:
        sched = {"timed": args.ns_schedule + (" (persistent for shallow products, phased for "
                                              "deep ones)" if args.ns_schedule == "auto" else ""),
                 "timed_ms_per_step": t_ms / args.steps}
        for name, code in (("phased", malt.MALT_NS_PHASED), ("persistent", malt.MALT_NS_PERSISTENT)):
            opt.set_ns_schedule(code)
            for _ in range(2):
                opt.step(hp, malter=malter)
            torch.cuda.synchronize()
            barrier()
            p0 = torch.cuda.Event(enable_timing=True)
            p1 = torch.cuda.Event(enable_timing=True)
            p0.record(stream)
            for _ in range(args.steps):
                opt.step(hp, malter=malter)
            p1.record(stream)
            torch.cuda.synchronize()
            sched[f"{name}_ms_per_step"] = max_over_ranks(p0.elapsed_time(p1), dev) / args.steps
            if opt.check() != malt.MALT_OK:
                raise SystemExit(f"{name}-schedule step failed")
        opt.set_ns_schedule(sched_code)

    # ---- the same step replayed from a CUDA graph: one step captured once
    # (binding kernel, statistics, Newton-Schulz launches, apply), then K
    # replays.  The device work is the same; the host-side argument
    # marshalling and the per-launch enqueue cost are gone.
    graph_leg = None
    if not args.no_graph:
        gs = torch.cuda.Stream()
        gs.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(gs):
            with torch.cuda.graph(graph, stream=gs):
                opt.step(hp, malter=malter, stream=gs)
        torch.cuda.synchronize()
        for _ in range(2):
            graph.replay()
        torch.cuda.synchronize()
        barrier()
        g0 = torch.cuda.Event(enable_timing=True)
        g1 = torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for _ in range(args.steps):
            graph.replay()
        g1.record(stream)
        torch.cuda.synchronize()
        tg = max_over_ranks(g0.elapsed_time(g1), dev) / args.steps
        if opt.check() != malt.MALT_OK:
            raise SystemExit("graph-replayed step failed")
        graph_leg = {"ms_per_step": tg, "value": world / (tg / 1e3), "unit": UNIT,
                     "schedule": args.ns_schedule}
        del graph

    # ---- the same engine as Muon (identity preconditioners, no statistics):
    # the optimizer-only counterpart of the paper's MALT-vs-Muon overhead table.
    # Muon and MALT run in alternating blocks of steps on the same state, so
    # that both see the same clocks under the power cap.
    muon = None
    if not args.no_muon:
        for _ in range(2):
            opt.step(hp, muon=True)
        torch.cuda.synchronize()
        barrier()
        block = max(1, args.steps // 2)
        t_muon = t_malt = 0.0
        for _ in range(4):
            for is_muon in (True, False):
                m0 = torch.cuda.Event(enable_timing=True)
                m1 = torch.cuda.Event(enable_timing=True)
                m0.record(stream)
                for _ in range(block):
                    if is_muon:
                        opt.step(hp, muon=True)
                    else:
                        opt.step(hp, malter=malter)
                m1.record(stream)
                torch.cuda.synchronize()
                if is_muon:
                    t_muon += m0.elapsed_time(m1)
                else:
                    t_malt += m0.elapsed_time(m1)
        tm = max_over_ranks(t_muon, dev) / (4 * block)
        tmalt = max_over_ranks(t_malt, dev) / (4 * block)
        muon = {"ms_per_step": tm, "malt_ms_per_step": tmalt,
                "malt_overhead_vs_muon": tmalt / tm - 1.0,
                "method": f"4 alternating blocks of {block} Muon and {block} "
                          f"{'MALTER' if malter else 'MALT'} steps on one state"}
        if opt.check() != malt.MALT_OK:
            raise SystemExit("muon step failed")

    # ---- the whole optimizer (MALT on the matrices + AdamW on the rest)
    whole = None
    if not args.no_whole:
        whole = run_whole_optimizer_leg(args, wl, G, dev, stream)

    # ---- end to end through the C ABI with host buffers (malt_step_host):
    # every step copies all gradients in from pinned host memory and all
    # updated weights back out; the library overlaps those copies with the
    # neighbouring steps' kernels.  Wall clock between full synchronisations.
    e2e = None
    if not args.no_e2e:
        W_host = [torch.empty(w.shape, dtype=w.dtype, pin_memory=True) for w in W]
        h2d = sum(g.numel() * g.element_size() for g in G_host)
        d2h = sum(w.numel() * w.element_size() for w in W)
        # Two device gradient sets, alternated, so step i+1's copy-in overlaps step i.
        G2 = [torch.empty_like(g) for g in G]
        param_sets = [params, list(zip(W, G2, M, l, r))]
        for s_ in range(max(2, args.warmup // 2)):
            opt.step_host(hp, G_host, W_host, malter=malter, params=param_sets[s_ % 2])
        if opt.check() != malt.MALT_OK:
            raise SystemExit("e2e warm-up step failed")
        torch.cuda.synchronize()
        barrier()
        t0 = time.perf_counter()
        ends = []
        for s_ in range(args.steps):
            opt.step_host(hp, G_host, W_host, malter=malter, params=param_sets[s_ % 2])
            ends.append(torch.cuda.Event(enable_timing=True))
            ends[-1].record(stream)           # the end of the step's kernels
        status = opt.check()                  # waits for the compute and both copy streams
        torch.cuda.synchronize()
        te = time.perf_counter() - t0
        barrier()
        te = max_over_ranks(te, dev)
        e2e = {"value": world * args.steps / te, "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "api": "malt_step_host (copies overlapped with compute)"}
        if status != malt.MALT_OK:
            raise SystemExit("e2e step failed")
        link = host_link_bound(G_host, G2, W, W_host, t_ms / args.steps, e2e["value"] / world)
        # Steady state: the spacing of consecutive steps' ends, once the
        # pipeline is full (the timed region also holds its fill and drain:
        # the first step's gradient copy and the last step's weight copy).
        gaps = [a.elapsed_time(b) for a, b in zip(ends[1:], ends[2:])]
        if gaps:
            link["pipelined_ms_per_step"] = statistics.median(gaps)
            link["pipelined_frac_of_bound"] = 1e3 / link["bound_steps_per_s"] / link["pipelined_ms_per_step"]
        e2e["link"] = link

    if rank != 0:
        return

    # ---- roofline of the dominant kernel (the Newton-Schulz GEMMs)
    pk, pk_src = peaks()
    ns_ms = sum(prof[k][0] for k in malt.NS_KINDS)
    ns_launches = sum(prof[k][1] for k in malt.NS_KINDS)
    # Algorithmic work: the Newton-Schulz flops with the symmetry of the Gram
    # matrix and of the polynomial used (3 p^2 q + p^3 per matrix and iteration),
    # which is what the kernels compute (upper-triangle tiles only).
    flops = wl.ns_flops_min() * args.steps
    achieved = flops / (ns_ms / 1e3) / 1e12
    dense_equiv = wl.ns_flops_dense() * args.steps / (ns_ms / 1e3) / 1e12
    peak = float(pk["bf16_tflops_sustained"])
    persistent_timed = prof["ns_persistent"][1] > 0 and prof["ns_bx"][1] == 0
    # the committed capture is of the 144-matrix GPT-2 Large set only
    traffic = ncu_traffic_per_launch(persistent_timed) if (
        wl.name == "gpt2_large" and not args.layers) else None
    roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "traffic": traffic,
                "kernel": ("ns_gemm_kernel, persistent schedule (every Gram, Poly and BX "
                           "product of the k iterations in one launch)"
                           if prof["ns_persistent"][1] > 0 else
                           "ns_gemm_kernel, phased schedule (one launch per Gram, Poly and BX "
                           "product)"),
                "peak_source": f"{pk_src}: bf16_tflops_sustained",
                "flops_per_step": wl.ns_flops_min(),
                "flops_counted": "3p^2q + p^3 per matrix and NS iteration (symmetric Gram and polynomial)",
                "dense_equivalent_tflops": dense_equiv,
                # what the tensor cores execute: symmetric products as whole
                # 256 x 256 tiles on and above the diagonal
                "issued_tflops": wl.ns_flops_issued() * args.steps / (ns_ms / 1e3) / 1e12,
                "tensor_pipe_pct_ncu": ncu_tensor_pipe() if wl.name.startswith("gpt2_large") else None,
                "launch_avg_ms": ns_ms / max(ns_launches, 1)}
    elems = wl.elements
    wbytes = 2 if wl.weight_dtype == "bf16" else 4
    mem = {}
    for kind, bytes_per_elem in (("stats", 12.0), ("prescale", 6.0 + (4.0 if malter else 0.0)),
                                 ("apply", 2.0 * wbytes + 2.0)):
        ms = prof[kind][0]
        gbs = bytes_per_elem * elems * args.steps / (ms / 1e3) / 1e9 if ms > 0 else None
        mem[kind] = {"ms_per_step": ms / args.steps, "bytes_per_elem": bytes_per_elem,
                     "achieved_gbs": gbs,
                     "frac_of_hbm": (gbs / float(pk["hbm_gbs"])) if gbs else None}
    # finalize: per matrix, the per-block partial sums of G^2 (one per 256-column
    # block for each row, one per 64-row block for each column: the statistics
    # kernel's tile) in, l and r in and out, L and R out, all fp32
    fin_bytes = 0.0
    for m_, n_ in wl.shapes:
        m8, n8 = -(-m_ // 8) * 8, -(-n_ // 8) * 8
        fin_bytes += 4.0 * (m8 * -(-n8 // 256) + n8 * -(-m8 // 64)) + 16.0 * (m8 + n8)
    ms = prof["finalize"][0]
    gbs = fin_bytes * args.steps / (ms / 1e3) / 1e9 if ms > 0 else None
    mem["finalize"] = {"ms_per_step": ms / args.steps, "bytes_per_step": fin_bytes,
                       "achieved_gbs": gbs,
                       "frac_of_hbm": (gbs / float(pk["hbm_gbs"])) if gbs else None,
                       "note": "about 0.1 B per element: latency-bound, not bandwidth-bound"}
    breakdown = {k: round(v[0] / args.steps, 4) for k, v in prof.items()}
    launches = sum(v[1] for v in prof.values())

    cpu = None
    if not args.no_cpu_baseline and world == 1:
        oracle_warmup(wl)
        t_cpu = oracle_full_step_time(wl)
        cpu = {"value": 1.0 / t_cpu, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "ms_per_step": t_cpu * 1e3,
               "sample": f"one fp64 step of all {len(wl.shapes)} matrices of {wl.name} "
                         f"(each from zero state), timed once, no scaling"}

    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_ms / args.steps,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "bf16", "data": "synthetic",
           "config": dict(workload_config(wl), ns_schedule=args.ns_schedule),
           "clocks": clk, "e2e": e2e, "gpu_launches": launches, "roofline": roofline,
           "hbm_kernels": mem, "ms_per_step_by_kernel": breakdown,
           "cpu_baseline": cpu, "muon_same_engine": muon, "ns_schedules": sched,
           "whole_optimizer": whole,
           "cuda_graph": graph_leg, "workspace_bytes": opt.workspace_bytes()}
    print(json.dumps(out), flush=True)
    opt.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("malt", "reference"), default="malt")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-muon", action="store_true")
    ap.add_argument("--no-whole", action="store_true",
                    help="skip the whole-optimizer leg (MALT + AdamW on every parameter)")
    ap.add_argument("--no-graph", action="store_true",
                    help="skip the CUDA-graph replay of the timed step")
    ap.add_argument("--ns-schedule", choices=("auto", "phased", "persistent"),
                    default="auto",
                    help="schedule of the timed steps (default: the library's auto)")
    ap.add_argument("--layers", type=int, default=0,
                    help="profiling only: the first N layers of the workload")
    ap.add_argument("--compare-cublas", action="store_true",
                    help="one B*X-shaped product (36 x 1280^2 @ 1280x5120, bf16) through "
                         "cuBLAS (torch.matmul) and through this library's phased B*X launch")
    ap.add_argument("--stress-sweep", action="store_true",
                    help="the shape / anisotropy stress set, one JSON line per case (not a bench line)")
    ap.add_argument("--stress-sigma", type=float, default=None,
                    help="stress sweep: only this row / column scale sigma")
    ap.add_argument("--stress-k", type=int, default=None,
                    help="stress sweep: only this Newton-Schulz iteration count")
    args = ap.parse_args()
    args.requested = {"steps": args.steps, "warmup": args.warmup}
    if args.warmup < 3:
        args.warmup = 3
    if args.compare_cublas:
        run_compare_cublas(args)
    elif args.stress_sweep:
        run_stress_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_malt(args)


if __name__ == "__main__":
    main()
