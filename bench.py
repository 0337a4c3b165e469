#!/usr/bin/env python
"""Benchmark: validation throughput on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--config c1|c2|c3|c4|c5]

A step is one nmv_validate call (nmv_validate_batch for c3) on one seeded
synthetic workload resident in HBM; the default workload is the largest one
that fits one GPU: the fp32 [32768, 65536] candidate/reference pair with a
2^31-element operator input (the candidate passes half of it through), 24 GiB
read per call.  The metric is GB/s of candidate + reference bytes read; the
roofline counts every byte the call must read (the input included).  Prints
ONE JSON line on rank 0.

Under torchrun (N > 1) every rank validates its own replica (independent
problems, no collective on the data path); the timed region is bracketed by
a barrier and a device synchronize on every rank and the slowest rank's time
is used.  ``--impl reference`` times the CPU oracle (the reference arm: one
host core, a bounded sample of the same workload per step).
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "validation GB/s (cand+ref bytes read) and % of GB300 HBM peak, 1 GPU"
L2_BYTES = 129 * 1024 * 1024
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="c5",
                    choices=["c1", "c2", "c3", "c4", "c5", "stats", "forensics", "sweep"],
                    help="c1-c5: nmv_validate / nmv_validate_batch on the five workloads; stats: "
                         "nmv_stats of the c5 candidate (tile 128x128); forensics: nmv_forensics of the "
                         "c5 pair along its rows; sweep: nmv_sweep with 48 clean lightweight cases "
                         "escalating to the 512-case c3 set")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--c2-batch", type=int, default=8,
                    help="leading dimension of the c2 workload (8 = full size); smaller "
                         "values give the small cases used for profiler captures")
    ap.add_argument("--c5-rows", type=int, default=32768,
                    help="rows of the c5 workload (32768 = full size, 65536 columns)")
    ap.add_argument("--no-inputs", action="store_true",
                    help="drop the cases' inputs (c5 as a plain cand/ref pair, same data)")
    return ap.parse_args()


# ------------------------------------------------------------- workloads
def make_cases(config: str, device, seed_shift: int = 0, c2_batch: int = 8, c5_rows: int = 32768,
               no_inputs: bool = False):
    cases = _make_cases(config, device, seed_shift, c2_batch, c5_rows)
    if not no_inputs:
        return cases
    # the same pairs without their inputs, named for what is read
    out = []
    for c in cases:
        name = c.get("name", "")
        out.append(dict(c, inputs=[], name=name[:-len("_input")] if name.endswith("_input") else name))
    return out


def _make_cases(config, device, seed_shift, c2_batch, c5_rows):
    from paper_2608_02712_gb300 import workloads as W
    if config == "c1":
        return [W.c1(seed=0 + seed_shift, device=device)]
    if config == "c2":
        return [W.c2(seed=1 + seed_shift, device=device, shape=(c2_batch, 4096, 4096))]
    if config == "c3":
        return W.c3(seed=2 + seed_shift, device=device)
    if config == "c4":
        return [W.c4(seed=3 + seed_shift, device=device)]
    return [W.c5(seed=4 + seed_shift, device=device, shape=(c5_rows, 65536))]


def case_bytes(c, with_inputs=False):
    b = c["cand"].numel() * c["cand"].element_size() * 2
    if with_inputs:
        b += sum(x.numel() * x.element_size() for x in c["inputs"])
    return b


def describe(config, cases):
    c = cases[0]
    if config == "c3":
        name = "c3_batch%d_rank1-5_fp32/fp16/bf16" % len(cases)
        return {"workload": name, "cases": len(cases),
                "elements": int(sum(x["cand"].numel() for x in cases)),
                "tolerance": "torch.testing defaults per dtype", "tile": [64, 64],
                "first_k": 256}
    return {"workload": c["name"], "shape": list(c["cand"].shape),
            "dtype_in": str(c["cand"].dtype).split(".")[-1], "rtol": c["rtol"],
            "atol": c["atol"], "tile": list(c["tile"]), "first_k": c["first_k"],
            "inputs": len(c["inputs"])}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """Samples SM clock and throttle reasons through NVML while running."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, device_index: int):
        self.samples, self.reasons, self.max_mhz = [], set(), None
        self._stop = threading.Event()
        self._nvml = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                return
            handle = ctypes.c_void_p()
            import torch
            bus = None
            try:
                p = torch.cuda.get_device_properties(device_index)
                bus = "%08x:%02x:%02x.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
            except Exception:
                bus = None
            ok = bus is not None and nv.nvmlDeviceGetHandleByPciBusId_v2(
                bus.encode(), ctypes.byref(handle)) == 0
            if not ok and nv.nvmlDeviceGetHandleByIndex_v2(device_index, ctypes.byref(handle)) != 0:
                return
            self._nv, self._h = nv, handle
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(handle, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = mx.value
            self._nvml = True
        except OSError:
            self._nvml = None

    def sample(self):
        if not self._nvml:
            return
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        if self._nv.nvmlDeviceGetClockInfo(self._h, 1, ctypes.byref(clk)) == 0:
            self.samples.append(clk.value)
        if self._nv.nvmlDeviceGetCurrentClocksEventReasons(self._h, ctypes.byref(rs)) == 0:
            for bit, name in self.REASONS.items():
                if rs.value & bit:
                    self.reasons.add(name)

    def _run(self):
        while not self._stop.is_set():
            self.sample()
            time.sleep(0.02)

    def __enter__(self):
        self.sample()
        self._t = threading.Thread(target=self._run, daemon=True)
        self._t.start()
        return self

    def __exit__(self, *a):
        self._stop.set()
        self._t.join()
        self.sample()

    def report(self):
        if not self._nvml:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvml unavailable"]}
        return {"sm_mhz": statistics.median(self.samples) if self.samples else None,
                "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                "samples": len(self.samples)}


# ---------------------------------------------------------------- peaks
def measured_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs)"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def full_size(args) -> bool:
    """The workload at the size and with the inputs that the benchmark names."""
    return args.c2_batch == 8 and args.c5_rows == 32768 and not args.no_inputs


def profiled_traffic(config: str):
    """DRAM bytes per scan launch from the committed ncu summary, when it was
    taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "scan_kernel_%s_traffic.txt" % config)
    src = os.path.join(ROOT, "paper_2608_02712_gb300", "csrc", "nmv_scan.cuh")
    try:
        info = {}
        for line in open(path):
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                info[k.strip()] = v.strip()
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
        if info.get("kernel_source_sha256") != digest:
            return None
        return int(info["dram_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


# ------------------------------------------------------------ ranks
def max_over_ranks(value: float, world: int, device) -> float:
    """The slowest rank's figure (every rank passes its own; all get the max)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_gbs(nbytes_per_rank: int, world: int, ms: float) -> float:
    """Whole-job throughput: every rank's bytes over the slowest rank's time
    (replicas: each rank validates its own copy of the workload)."""
    return world * nbytes_per_rank / (ms * 1e-3) / 1e9


# ------------------------------------------------------------ reference
def sample_units(cases):
    """What a bounded oracle sample counts: rows of the [M, N] view of a single
    case, or whole cases of a batch."""
    if len(cases) > 1:
        return len(cases)
    c = cases[0]["cand"]
    return c.reshape(-1, c.shape[-1]).shape[0] if c.dim() else 1


def sample_text(cases, units, nbytes):
    what = "cases of the batch" if len(cases) > 1 else "rows of the [M, N] view"
    return "first %d %s (%d bytes of cand+ref)" % (units, what, nbytes)


def oracle_step_time(cases, units):
    """Run the oracle on a sample: the first `units` rows of the [M, N] view
    of a single case (its inputs cut to the same elements), or the first
    `units` cases of a batch."""
    import oracle
    t0 = time.perf_counter()
    nbytes = 0
    if len(cases) > 1:
        for c in cases[:units]:
            oracle.validate(c["cand"], c["ref"], inputs=c["inputs"], rtol=c["rtol"], atol=c["atol"],
                            tile=c["tile"], first_k=c["first_k"])
            nbytes += case_bytes(c)
    else:
        c = cases[0]
        n = c["cand"].shape[-1] if c["cand"].dim() else 1
        cv = c["cand"].reshape(-1, n)[:units]
        rv = c["ref"].reshape(-1, n)[:units]
        xs = [x.reshape(-1)[:cv.numel()] for x in c["inputs"]]
        oracle.validate(cv, rv, inputs=xs, rtol=c["rtol"], atol=c["atol"], tile=c["tile"],
                        first_k=c["first_k"])
        nbytes = cv.numel() * cv.element_size() * 2
    return time.perf_counter() - t0, nbytes


def host_copy(cases):
    return [dict(c, cand=c["cand"].cpu(), ref=c["ref"].cpu(),
                 inputs=[x.cpu() for x in c["inputs"]]) for c in cases]


def cpu_baseline(cases_host, budget_s=12.0):
    """The oracle as it stands, on one host core, on a bounded row sample."""
    n = sample_units(cases_host)
    units = min(n, 4 if len(cases_host) > 1 else 256)
    t, b = oracle_step_time(cases_host, units)
    units = int(min(n, max(units, units * budget_s / max(t, 1e-6))))
    t, b = oracle_step_time(cases_host, units)
    return {"value": b / t / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
            "sample": "%s, one pass, %.1f s" % (sample_text(cases_host, units, b), t)}


def run_reference(args, rank, world):
    import torch
    if rank != 0:
        return None
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    cases = host_copy(make_cases(args.config, dev, c2_batch=args.c2_batch, c5_rows=args.c5_rows,
                                 no_inputs=args.no_inputs))
    n = sample_units(cases)
    probe = min(n, 4 if len(cases) > 1 else 64)
    t, _ = oracle_step_time(cases, probe)
    per_step = 150.0 / max(1, args.steps + args.warmup)
    units = int(min(n, max(1, probe * per_step / max(t, 1e-6))))
    for _ in range(args.warmup):
        oracle_step_time(cases, units)
    times, nbytes = [], 0
    for _ in range(args.steps):
        dt, nbytes = oracle_step_time(cases, units)
        times.append(dt)
    total = sum(times)
    value = nbytes * args.steps / total / 1e9
    sample = sample_text(cases, units, nbytes) + " per step"
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": total / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": describe(args.config, cases),
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


# ------------------------------------------------------------------ ours
def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    import paper_2608_02712_gb300 as nmv
    from paper_2608_02712_gb300 import nmv as nmvmod

    torch.cuda.set_device(local_rank)
    cases = make_cases(args.config, "cuda", seed_shift=0, c2_batch=args.c2_batch, c5_rows=args.c5_rows,
                       no_inputs=args.no_inputs)
    torch.cuda.synchronize()
    nbytes = sum(case_bytes(c) for c in cases)
    algo_bytes = sum(case_bytes(c, with_inputs=True) for c in cases)
    stream = torch.cuda.current_stream()
    prep = nmv.Prepared(cases, stream=stream)

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(max(3, args.warmup)):
        prep.call()
    # Every SAMPLE-th timed step records CUDA events around the scan kernel
    # (its duration for the roofline); the others run without them.
    SAMPLE = 8
    scan_ms, launches = [], 0
    sampler = ClockSampler(local_rank)
    barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    per_step = None
    with sampler:
        ev0.record(stream)
        for i in range(args.steps):
            sample = i % SAMPLE == 0
            if sample:
                nmvmod.profile_enable(nmvmod.PROFILE_TIMING)
            prep.call()
            if sample:
                pr = nmvmod.profile_last()
                nmvmod.profile_enable(False)
                scan_ms.append(pr["scan_ms"])
                per_step = pr["kernel_launches"]
            launches += per_step
        ev1.record(stream)
        torch.cuda.synchronize()
    barrier()
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), world, "cuda")
    ms_per_step = elapsed_ms / args.steps
    # one more call with the exact-path counters (kept out of the timed loop)
    nmvmod.profile_enable(nmvmod.PROFILE_TIMING | nmvmod.PROFILE_COUNTERS)
    prep.call()
    pr = nmvmod.profile_last()
    nmvmod.profile_enable(False)
    value = job_gbs(nbytes, world, ms_per_step)

    # e2e: pinned host buffers -> device copies -> validate -> results back
    # (one pinned host copy of the workload, also the CPU baseline's source)
    def pinned(t):
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h

    host = [dict(c, cand=pinned(c["cand"]), ref=pinned(c["ref"]),
                 inputs=[pinned(x) for x in c["inputs"]]) for c in cases]
    dev_bufs = [dict(c, cand=torch.empty_like(c["cand"]), ref=torch.empty_like(c["ref"]),
                     inputs=[torch.empty_like(x) for x in c["inputs"]]) for c in cases]
    desc = describe(args.config, cases)
    del prep
    cases = None  # the device copies of the workload are released
    torch.cuda.empty_cache()
    prep2 = nmv.Prepared(dev_bufs, stream=stream)
    copied = sum(case_bytes(c, with_inputs=True) for c in host)

    def e2e_step():
        for h, d in zip(host, dev_bufs):
            d["cand"].copy_(h["cand"], non_blocking=True)
            d["ref"].copy_(h["ref"], non_blocking=True)
            for hx, dx in zip(h["inputs"], d["inputs"]):
                dx.copy_(hx, non_blocking=True)
        prep2.call()

    for _ in range(2):
        e2e_step()
    nmvmod.profile_enable(True)
    e2e_step()
    pr_e2e = nmvmod.profile_last()
    lib_h2d, lib_d2h = pr_e2e["h2d_bytes"], pr_e2e["d2h_bytes"]
    nmvmod.profile_enable(False)
    ke = max(1, min(args.e2e_steps, args.steps))
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(ke):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / ke, world, "cuda")

    if rank != 0:
        return None
    peak, peak_src = measured_peak()
    scan_mean = statistics.fmean(scan_ms)
    achieved = algo_bytes / (scan_mean * 1e-3) / 1e9
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32+f64", "data": "synthetic",
        "config": dict(desc,
                       l2="inputs (%d B) larger than the %d B L2; no flush between steps"
                          % (algo_bytes, L2_BYTES) if algo_bytes > L2_BYTES else
                          "inputs smaller than L2 (cache-warm)",
                       parallelism="replicas" if world > 1 else "1 GPU",
                       pct_of_hbm_peak=100.0 * value / world / peak),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": profiled_traffic(args.config) if full_size(args) else None,
                     "kernel": "scan_kernel", "peak_source": peak_src,
                     "algorithmic_bytes_per_launch": algo_bytes,
                     "scan_ms_mean": scan_mean, "scan_ms_min": min(scan_ms),
                     "slow_steps": pr["slow_steps"], "light_steps": pr["light_steps"],
                     "exact_abs": pr["exact_abs"],
                     "exact_rel": pr["exact_rel"], "exact_pred": pr["exact_pred"]},
        "e2e": {"value": job_gbs(nbytes, world, e2e_ms), "unit": "GB/s",
                "h2d_bytes_per_step": copied + lib_h2d, "d2h_bytes_per_step": lib_d2h,
                "ms_per_step": e2e_ms},
        "gpu_launches": launches,
        "clocks": sampler.report(),
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(host)
    return line


# ------------------------------------------------------- other entry points
AUX_METRIC = {"stats": "diagnostic statistics GB/s (bytes read), 1 GPU",
              "forensics": "deep forensics GB/s (cand+ref bytes read), 1 GPU",
              "sweep": "full-coverage sweep GB/s (cand+ref bytes of the cases validated), 1 GPU"}


def aux_workload(args):
    """The data, the call and what a bounded oracle sample of it costs."""
    from paper_2608_02712_gb300 import workloads as W
    import paper_2608_02712_gb300 as nmv
    if args.config == "stats":
        x = W.c5(device="cuda", shape=(args.c5_rows, 65536))["cand"]
        nbytes = x.numel() * 4
        desc = {"workload": "stats_fp32_%dx65536" % args.c5_rows, "tile": [128, 128]}

        def call():
            return nmv.stats(x, tile=(128, 128))

        def sample(rows):
            import oracle
            xs = x[:rows].cpu()
            t0 = time.perf_counter()
            oracle.stats(xs, tile=(128, 128))
            return time.perf_counter() - t0, xs.numel() * 4
        return call, nbytes, desc, sample, x.shape[0]
    if args.config == "forensics":
        case = W.c5(device="cuda", shape=(args.c5_rows, 65536))
        c, r = case["cand"], case["ref"]
        nbytes = c.numel() * 8
        kw = dict(rtol=case["rtol"], atol=case["atol"], axis=0)
        desc = {"workload": "forensics_fp32_%dx65536_axis0" % args.c5_rows}

        def call():
            return nmv.forensics(c, r, **kw)

        def sample(rows):
            import oracle
            ch, rh = c[:rows].cpu(), r[:rows].cpu()
            t0 = time.perf_counter()
            oracle.forensics(ch, rh, **kw)
            return time.perf_counter() - t0, ch.numel() * 8
        return call, nbytes, desc, sample, c.shape[0]
    light = W.c3(seed=20, device="cuda", count=96, cap=1 << 20)[0::2]
    ext = W.c3(device="cuda")
    nbytes = sum(case_bytes(x) for x in light + ext)
    desc = {"workload": "sweep_light48_c3ext512", "light": len(light), "extended": len(ext),
            "call": "nmv_sweep through the C ABI, case arrays marshalled once"}
    prep = nmv.PreparedSweep(light, ext)

    def call():
        return prep.call()

    def sample(n):
        import oracle
        hl = host_copy(light[:1])
        he = host_copy(ext[:n])
        t0 = time.perf_counter()
        for cs in (hl, he):
            for c in cs:
                oracle.validate(c["cand"], c["ref"], rtol=c["rtol"], atol=c["atol"], tile=c["tile"],
                                first_k=c["first_k"])
        return time.perf_counter() - t0, sum(case_bytes(x) for x in hl + he)
    return call, nbytes, desc, sample, len(ext)


def run_aux(args):
    """One JSON line for an entry point other than the validation itself:
    the whole call timed with CUDA events (inputs resident), every step."""
    import torch
    call, nbytes, desc, sample, units = aux_workload(args)
    torch.cuda.synchronize()
    for _ in range(max(3, args.warmup)):
        call()
    sampler = ClockSampler(0)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = max(1, min(args.steps, 200))
    with sampler:
        torch.cuda.synchronize()
        ev0.record()
        for _ in range(steps):
            call()
        ev1.record()
        torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / steps
    value = nbytes / (ms * 1e-3) / 1e9
    peak, peak_src = measured_peak()
    line = {"metric": AUX_METRIC[args.config], "value": value, "unit": "GB/s", "n_gpus": 1, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32+f64", "data": "synthetic",
            "config": dict(desc, l2="inputs larger than L2; no flush between steps"),
            "roofline": {"bound": "hbm", "achieved": value, "peak": peak, "unit": "GB/s", "frac": value / peak,
                         "traffic": None, "kernel": "whole call (kernels and finalize)",
                         "peak_source": peak_src, "algorithmic_bytes_per_launch": nbytes},
            "clocks": sampler.report()}
    if not args.no_cpu_baseline:
        probe = max(1, units // 512)
        t, b = sample(probe)
        n = int(min(units, max(probe, probe * 12.0 / max(t, 1e-6))))
        t, b = sample(n)
        line["cpu_baseline"] = {"value": b / t / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                "sample": "first %d %s, one pass, %.1f s" % (
                                    n, "cases of the extended set" if args.config == "sweep" else "rows", t)}
    return line


def main():
    args = parse()
    if args.config in AUX_METRIC:
        if args.impl == "reference" or int(os.environ.get("RANK", "0")) != 0:
            return
        print(json.dumps(run_aux(args)), flush=True)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        if world > 1:
            import torch
            import torch.distributed as dist
            torch.cuda.set_device(local_rank)
            dist.init_process_group("nccl")
        line = run_ours(args, rank, world, local_rank)
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
