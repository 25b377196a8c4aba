"""Benchmark of one GMC / GMC+ step on GB300: worker-parameters per second.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl gmc|reference]

A step is one pass of the whole hot path (accumulator, compression, residual,
aggregate and update) for the K simulated workers of the workload over one
batch of synthetic gradients already resident in HBM. ``value`` is
K*d*steps*ranks / (max over ranks of the device time of the timed steps).
``workloads`` holds the same timing for the other configurations the metric is
quoted on (d >= 11 M, K >= 8: resnet18, and resnet50 with shared and per-worker
RBGS blocks), each measured in the same invocation.
``e2e`` is the same metric through the host-memory entry point (host->device
copy of the step's gradients and device->host read of the step's counters
inside the timed region). ``roofline`` reports the dominant kernel's
algorithmic bytes per launch over its CUDA-event duration (events around it on
every EVENTS_EVERY-th timed step) against the measured HBM copy peak. ``cpu_baseline`` times the oracle on the host cores on a bounded
sample of the same workload.

Multi-GPU: the step does not shard (K workers are simulated on one GPU), so
N > 1 runs N independent replicas, one per rank, and reports their aggregate.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workloads  # noqa: E402

METRIC = "GMC step throughput (worker-params/sec) and achieved HBM GB/s vs 8 TB/s, 1 GB300"
UNIT = "worker-params/s"
DEFAULT_WORKLOAD = "vgg16"
DEFAULT_EXTRA = "resnet18,resnet50,resnet50_pw"
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129e6
EVENTS_EVERY = 5  # timed steps per step whose dominant kernel is bracketed by events


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    """Samples SM clock and throttle reasons of one GPU while running: NVML
    through ctypes (read-only queries) when available, else nvidia-smi."""

    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown",
               0x4: "sw_power_cap", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, index: int, period_s: float = 0.01):
        self.index = index
        self.period = period_s
        self.samples = []  # (sm_mhz, reasons_mask)
        self.max_mhz = None
        self._stop = threading.Event()
        self._nvml = None
        self._handle = None
        self._proc = None
        self._csv = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() == 0:
                h = ctypes.c_void_p()
                if nv.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(index), ctypes.byref(h)) == 0:
                    self._nvml, self._handle = nv, h
                    mx = ctypes.c_uint()
                    if nv.nvmlDeviceGetMaxClockInfo(h, ctypes.c_int(1), ctypes.byref(mx)) == 0:
                        self.max_mhz = mx.value
        except OSError:
            self._nvml = None

    def _sample_nvml(self):
        nv, h = self._nvml, self._handle
        clk, reasons = ctypes.c_uint(), ctypes.c_ulonglong()
        if nv.nvmlDeviceGetClockInfo(h, ctypes.c_int(1), ctypes.byref(clk)) == 0:
            nv.nvmlDeviceGetCurrentClocksThrottleReasons(h, ctypes.byref(reasons))
            self.samples.append((clk.value, reasons.value))

    def _loop(self):
        while not self._stop.is_set():
            self._sample_nvml()
            time.sleep(self.period)

    def start(self):
        if self._nvml is not None:
            self._sample_nvml()
            self._thread = threading.Thread(target=self._loop, daemon=True)
            self._thread.start()
        else:
            self._csv = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            q = ("clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,"
                 "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
                 "clocks_event_reasons.sw_power_cap")
            try:
                self._proc = subprocess.Popen(
                    ["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                     "--format=csv,noheader,nounits", "-lms", "50"],
                    stdout=self._csv, stderr=subprocess.DEVNULL)
            except OSError:
                self._proc = None

    def stop(self) -> dict:
        if self._nvml is not None:
            self._stop.set()
            self._thread.join()
            self._sample_nvml()
        elif self._proc is not None:
            time.sleep(0.1)
            self._proc.terminate()
            self._proc.wait()
            self._csv.seek(0)
            names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
            bits = [0x8, 0x40, 0x20, 0x4]
            for line in self._csv.read().splitlines():
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 6 or not parts[0].isdigit():
                    continue
                mask = sum(b for b, v in zip(bits, parts[2:6]) if v.lower() == "active")
                self.samples.append((int(parts[0]), mask))
                self.max_mhz = int(parts[1]) if parts[1].isdigit() else self.max_mhz
            del names
            os.unlink(self._csv.name)
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [], "samples": 0}
        mask = 0
        for _, m in self.samples:
            mask |= m
        return {"sm_mhz": statistics.median(s for s, _ in self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": [n for b, n in self.REASONS.items() if mask & b],
                "samples": len(self.samples)}


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------
def measured_hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def _code_only(text: str) -> str:
    """C++/CUDA source without its comments and blank lines: what the
    compiler sees (the sources hold no string literal with a comment marker)."""
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    return "\n".join(line.rstrip() for line in text.splitlines() if line.strip())


def kernel_source_hash() -> str:
    """Hash of the kernel sources' code (comments ignored): a recorded ncu
    figure stays valid while the code it measured is unchanged."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_1905_12948_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name), encoding="utf-8") as f:
                h.update(_code_only(f.read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel sources (profiles/<kernel>_<workload>.md holds lines
    `traffic_bytes_per_launch: N` and `source_hash: H`)."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    hsh = re.search(r"source_hash:\s*([0-9a-f]+)", text)
    if not m or not hsh or hsh.group(1) != kernel_source_hash():
        return None
    return float(m.group(1))


def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl"
        try:
            import torch
            if not torch.cuda.is_available():
                backend = "gloo"
        except ImportError:
            backend = "gloo"
        dist.init_process_group(backend=backend)
    return world, rank, local


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------------------
# CPU oracle on a bounded sample of the workload
# ---------------------------------------------------------------------------
def _oracle_kind(wl) -> str:
    """The C++ oracle states Alg. 1 / Alg. 2 with top-s or RBGS; the appendix
    variants and the approximate top-s are in the numpy oracle only."""
    return "cpp" if wl.variant == "gmc" and wl.compressor in ("topk", "rbgs") else "numpy"


def oracle_sample(wl, budget_s: float = 12.0, max_steps: int = 50, workers: int = 0,
                  d_sample: int = 1 << 24, first_step: int = 0, threads: int = 0):
    """Time the oracle (as it stands) on a bounded sample of the workload:
    `workers` of its workers (0: all K) over the leading `d_sample` parameters
    (same per-parameter gradient scales, same compression ratio), running
    steps until `budget_s` of wall time is spent. The C++ oracle runs one
    thread per worker, at most `threads` (0: the host's cores); the numpy
    oracle one thread. Two gradient batches are drawn beforehand and
    alternate; drawing them is not timed."""
    import oracle
    from oracle import cref
    K_s = wl.K if workers <= 0 else min(workers, wl.K)
    d_s = min(wl.d, d_sample)
    kind = _oracle_kind(wl)
    gen = workloads.NumpyGradients(wl, seed=0, d=d_s, K=K_s)
    batches = [gen(first_step + i) for i in range(2)]
    args = dict(compressor=wl.compressor, ratio=wl.ratio, block=wl.block, lam=wl.lam, seed=0,
                per_worker=wl.per_worker, variant=wl.variant)
    if kind == "cpp":
        o = cref.CGMC(d_s, K_s, wl.beta, wl.eta, threads=threads or (os.cpu_count() or 1), **args)
        cores = o.threads
    else:
        o = oracle.GMC(d_s, K_s, wl.beta, wl.eta, **args)
        cores = 1
    o.set_params(workloads.init_params(wl.d)[:d_s])
    spent, steps = 0.0, 0
    while steps < max_steps and (spent < budget_s or steps == 0):
        t0 = time.perf_counter()
        o.step(batches[steps % 2])
        spent += time.perf_counter() - t0
        steps += 1
    what = ((f"C++ oracle, {cores} threads, one worker each" if cores > 1 else "C++ oracle, one thread")
            if kind == "cpp"
            else "numpy oracle, one thread")
    return {"value": K_s * d_s * steps / spent, "unit": UNIT, "cores": cores, "kind": "oracle",
            "host_cores": os.cpu_count(),
            "sample": f"{steps} oracle step(s) of {K_s} of the {wl.K} workers over the first "
                      f"{d_s:,} of d={wl.d:,} parameters ({what}), {spent:.1f} s",
            "seconds": spent, "d_sample": d_s, "steps": steps}


def cpu_baseline(wl, budget_s: float):
    """The oracle on the host's cores, with its one-thread figure beside it."""
    many = oracle_sample(wl, budget_s=budget_s)
    many.pop("seconds", None)
    if many["cores"] > 1:
        one = oracle_sample(wl, budget_s=budget_s / 2, threads=1)
        many["one_thread"] = {"value": one["value"], "sample": one["sample"]}
    return many


# ---------------------------------------------------------------------------
# arms
# ---------------------------------------------------------------------------
def run_reference(args, wl, world, rank):
    """The reference arm: the oracle (the paper has no code to install), as it
    stands, on the host's cores; each step one oracle step of all K workers
    over the first `--ref-params` parameters of the workload."""
    if rank != 0:
        return None
    import oracle
    from oracle import cref
    d_s = min(wl.d, args.ref_params)
    kind = _oracle_kind(wl)
    gen = workloads.NumpyGradients(wl, seed=0, d=d_s, K=wl.K)
    batches = [gen(i) for i in range(2)]
    kw = dict(compressor=wl.compressor, ratio=wl.ratio, block=wl.block, lam=wl.lam, seed=0,
              per_worker=wl.per_worker, variant=wl.variant)
    if kind == "cpp":
        o = cref.CGMC(d_s, wl.K, wl.beta, wl.eta, threads=os.cpu_count() or 1, **kw)
        cores = o.threads
    else:
        o = oracle.GMC(d_s, wl.K, wl.beta, wl.eta, **kw)
        cores = 1
    o.set_params(workloads.init_params(wl.d)[:d_s])
    for i in range(args.warmup):
        o.step(batches[i % 2])
    t0 = time.perf_counter()
    for i in range(args.steps):
        o.step(batches[(args.warmup + i) % 2])
    spent = time.perf_counter() - t0
    value = wl.K * d_s * args.steps / spent
    what = ((f"C++ oracle, {cores} threads, one worker each" if cores > 1 else "C++ oracle, one thread")
            if kind == "cpp"
            else "numpy oracle, one thread")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * spent / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": config_of(wl, args),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "host_cores": os.cpu_count(),
                         "sample": f"each step: one oracle step of all {wl.K} workers over the "
                                   f"first {d_s:,} of d={wl.d:,} parameters ({what}); two "
                                   f"gradient batches alternate"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    return line


def step_bytes(wl) -> float:
    """Algorithmic bytes of one step's dense work: read g and e, write e
    (12 B per worker-parameter, 10 with bf16 gradients); the local momentum
    adds its read and write (8 B), Alg. 3's dense server pass 20 B per parameter."""
    b = (8.0 + (2.0 if wl.grad_dtype == "bf16" else 4.0)) * wl.K * wl.d
    if wl.variant in ("local_momentum", "local_momentum_mfm"):
        b += 8.0 * wl.K * wl.d
    if wl.variant == "server_momentum":
        b += 20.0 * wl.d
    return b


def config_of(wl, args):
    return {"workload": f"{wl.name}: d={wl.d:,}, K={wl.K}, {wl.compressor}"
                        + (f" ratio {wl.ratio:.6g}" if wl.compressor != "rbgs"
                           else f" block {wl.block}, {wl.ratio:.0%} of blocks, lambda {wl.lam}")
                        + f", beta {wl.beta}, eta {wl.eta}"
                        + ("" if wl.variant == "gmc" else f", variant {wl.variant}")
                        + ("" if wl.grad_dtype == "f32" else f", {wl.grad_dtype} gradients"),
            "d": wl.d, "K": wl.K, "compressor": wl.compressor, "ratio": wl.ratio,
            "block": wl.block if wl.compressor == "rbgs" else None,
            "per_worker_blocks": wl.per_worker if wl.compressor == "rbgs" else None,
            "lambda": wl.lam, "variant": wl.variant, "grad_dtype": wl.grad_dtype,
            "l2": "inputs larger than L2 (gradient batches rotate)",
            "parallelism": f"replicas x{args.gpus}"}


def measure(args, wl, world, rank, local, breakdown=True):
    """Time `args.steps` steps of one workload on this rank's GPU, with its
    gradients already in HBM: the device time of the steps (max over ranks),
    the dominant kernel's CUDA-event time, the clocks during the timed region
    and, with `breakdown`, the per-kernel split from untimed steps after it.
    Returns (the handle, w0, the result dict)."""
    import torch
    from paper_1905_12948_gb300 import GMC
    dev = torch.device("cuda", local)
    gpu = GMC(wl.d, wl.K, wl.beta, wl.eta, compressor=wl.compressor, ratio=wl.ratio,
              block=wl.block, lam=wl.lam if wl.compressor == "rbgs" else None, seed=0,
              per_worker=wl.per_worker, variant=wl.variant, device=dev)
    w0 = torch.from_numpy(workloads.init_params(wl.d)).to(dev)
    gen = workloads.TorchGradients(wl, dev, seed=rank)
    bf16 = wl.grad_dtype == "bf16"
    gb = (2.0 if bf16 else 4.0) * wl.K * wl.d  # gradient bytes per step
    n_batches = 2 if gb > 2 * L2_BYTES else max(2, math.ceil(4 * L2_BYTES / gb))
    batches = [gen(t).to(torch.bfloat16) if bf16 else gen(t) for t in range(n_batches)]
    del gen
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()

    gpu.set_params(w0)
    for i in range(args.warmup):
        gpu.step(batches[i % n_batches])
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    dom = "rbgs_step" if wl.compressor == "rbgs" else "accumulate"
    # events around the dominant kernel only, on every EVENTS_EVERY-th timed
    # step: an event between two launches ends the programmatic overlap of
    # their scheduling (bracketing every step added 9 us to a resnet18 step,
    # every fifth step 1.7 us; the kernel's own duration reads the same)
    gpu.profile(True, kernels=[dom])
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for i in range(args.steps):
        gpu.profile_mask([dom] if i % EVENTS_EVERY == 0 else [])
        gpu.step(batches[(args.warmup + i) % n_batches])
    ev1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier(world)
    ms = ev0.elapsed_time(ev1)
    prof = gpu.profile_read()
    gpu.profile(False)
    # the per-kernel breakdown and launch count, from untimed steps with every
    # launch bracketed (those events lengthen a step slightly)
    n_bd = min(args.steps, 10) if breakdown else 2
    gpu.profile(True)
    for i in range(n_bd):
        gpu.step(batches[(args.warmup + args.steps + i) % n_batches])
    bd = gpu.profile_read()
    gpu.profile(False)
    status = gpu.check()
    totals = gpu.stats()
    ms_max = max_over_ranks(ms, world, dev)
    value = wl.K * wl.d * args.steps * world / (ms_max / 1e3)

    p = prof.get(dom, {"ms": float("nan"), "launches": 1, "bytes": float("nan")})
    per_launch_bytes = p["bytes"] / p["launches"]
    avg_s = p["ms"] / p["launches"] / 1e3
    achieved = per_launch_bytes / avg_s / 1e9
    peak, peak_kind = measured_hbm_peak()
    step_ms = ms_max / args.steps
    kernels = {k: {"ms_per_step": round(v["ms"] / n_bd, 4),
                   "share": round(v["ms"] / max(sum(x["ms"] for x in bd.values()), 1e-12), 4)}
               for k, v in bd.items()}
    del batches
    torch.cuda.synchronize()
    launches_per_step = sum(v["launches"] for v in bd.values()) / n_bd
    res = {
        "value": value, "ms_per_step": step_ms,
        "hbm_gbs_step": step_bytes(wl) / (step_ms / 1e3) / 1e9,
        "frac_of_8tbs": step_bytes(wl) / (step_ms / 1e3) / 8e12,
        "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak,
                     "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": recorded_traffic(dom, wl.name),
                     "algorithmic_bytes_per_launch": per_launch_bytes,
                     "avg_launch_ms": avg_s * 1e3,
                     "launches_timed": int(p["launches"]), "events_every": EVENTS_EVERY},
        "clocks": clk, "kernels": kernels, "status": status,
        "gpu_launches": int(round(launches_per_step * args.steps)),
        "select_fallbacks": totals["fallbacks"], "steps_run": totals["steps"],
    }
    return gpu, w0, res


def run_gmc(args, wl, world, rank, local):
    import torch
    from paper_1905_12948_gb300 import build as gbuild
    if rank == 0:
        gbuild.build()
    barrier(world)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    gpu, w0, res = measure(args, wl, world, rank, local)
    bf16 = wl.grad_dtype == "bf16"
    gb = (2.0 if bf16 else 4.0) * wl.K * wl.d

    e2e = None
    if not args.no_e2e:
        host = torch.empty((wl.K, wl.d), dtype=torch.bfloat16 if bf16 else torch.float32).pin_memory()
        host.copy_(torch.from_numpy(workloads.NumpyGradients(wl, seed=rank, K=wl.K)(0))
                   if wl.K * wl.d <= 50_000_000 else
                   workloads.TorchGradients(wl, dev, seed=rank)(0).cpu())
        stats = torch.zeros(8, dtype=torch.int64).pin_memory()
        gpu.set_params(w0)
        for _ in range(max(1, min(args.warmup, 3))):
            gpu.step_host(host, stats)
        torch.cuda.synchronize()
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            gpu.step_host(host, stats)
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
        e2e = {"value": wl.K * wl.d * args.steps * world / (e_ms / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(gb), "d2h_bytes_per_step": 8 * 8,
               "ms_per_step": e_ms / args.steps}
        del host
    gpu.close()
    del gpu, w0
    torch.cuda.empty_cache()

    # the other configurations the metric is quoted on (d >= 11 M, K >= 8), each
    # timed the same way in this invocation
    others = {}
    extra = args.extra if args.extra is not None else (DEFAULT_EXTRA if wl.name == DEFAULT_WORKLOAD else "")
    for name in ([] if args.no_extra else [n for n in extra.split(",") if n and n != wl.name]):
        owl = workloads.workload(name)
        g2, _, r2 = measure(args, owl, world, rank, local, breakdown=False)
        g2.close()
        del g2
        torch.cuda.empty_cache()
        others[name] = {"config": config_of(owl, args)["workload"], **{
            k: r2[k] for k in ("ms_per_step", "value", "hbm_gbs_step", "frac_of_8tbs", "roofline",
                               "clocks", "status", "gpu_launches")}}

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, args.cpu_budget)

    line = {
        "metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": config_of(wl, args),
        "hbm_gbs_step": res["hbm_gbs_step"], "frac_of_8tbs": res["frac_of_8tbs"],
        "roofline": res["roofline"],
        "cpu_baseline": cpu, "e2e": e2e, "clocks": res["clocks"],
        "gpu_launches": res["gpu_launches"] + sum(o["gpu_launches"] for o in others.values()),
        "gpu_launches_headline": res["gpu_launches"],
        "kernels": res["kernels"], "status": res["status"],
        "select_fallbacks": res["select_fallbacks"], "steps_run": res["steps_run"],
        "workloads": others,
    }
    return line if rank == 0 else None


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gmc", "reference"], default="gmc")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    help="one of " + ", ".join(w.name for w in workloads.WORKLOADS))
    ap.add_argument("--extra", default=None,
                    help="comma-separated workloads also timed in the same run (key `workloads`); "
                         f"default {DEFAULT_EXTRA} with the default workload, none otherwise")
    ap.add_argument("--no-extra", action="store_true", help="time the one workload only")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle CPU time")
    ap.add_argument("--ref-params", type=int, default=1 << 22,
                    help="reference arm: parameters of the oracle sample per step")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "gmc":
        ap.error("--warmup must be >= 3")
    wl = workloads.workload(args.workload)
    world, rank, local = dist_setup(args.gpus)
    if args.impl == "reference":
        line = run_reference(args, wl, world, rank)
    else:
        line = run_gmc(args, wl, world, rank, local)
    if line is not None:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
