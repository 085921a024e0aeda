"""Throughput of the differential-oracle hot path on GB300.

One step = one pass of the whole hot path over one batch of synthetic
input: the Tier 1 guarded fill of the workload's input regions followed by
the equivalence check of the reference output against every candidate
(AsmEvo Sec. 3.4 and Eq. 1).  Default workload: a 16 GiB guarded fill of
GEMM input buffers, then one fp16 [32768, 32768] reference checked against
8 candidates carrying 0..8 ULP of noise.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mine|reference]
                       [--workload NAME] [--no-e2e] [--no-cpu] [--no-eq]

Beside the step, the line carries `snapshot_4096`: the 4096-region replay
snapshot's fill and check, each kernel timed alone with CUDA events;
`eq1`: Eq. 1 as a whole (the exact sums of the cosine term over the same
reference and candidates); `eq1_f64`: the same for binary64 outputs of the
reference's size; and `restore`: the Tier 2 restore of the step's input
regions from a captured snapshot, timed the same way.  `--impl reference`
times the CPU oracle alone on host-built samples of the same workload (no
GPU library is loaded).
For N > 1 launch under torchrun; every rank runs its own replica (weak
scaling, no data-path collective) and rank 0 prints one JSON line.
"""
import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verify GB/s (ref+cand bytes compared per s) and fill GB/s, % of GB300 HBM peak"
UNIT = "GB/s"
FALLBACK_HBM_GBS = 6800.0
# bounded CPU samples: the cpu_baseline leg's check bytes, and one reference-arm step's
CPU_SAMPLE_VERIFY_BYTES = 2 << 30
REF_STEP_VERIFY_BYTES = 1 << 30


# ------------------------------------------------------------------ helpers
def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle samples during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.out = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
        time.sleep(0.25)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        if not self.out:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        # median over samples taken under load (the busiest half)
        loaded = sorted(sm)[len(sm) // 2:] if len(sm) > 3 else sm
        return {"sm_mhz": float(np.median(loaded)), "sm_max_mhz": float(max(smax)),
                "samples": len(sm), "reasons": sorted(reasons)}


def kernel_traffic(kernel, workload):
    """dram read+write bytes per launch from a committed ncu summary, if it
    was taken on the kernel source as it is now."""
    path = os.path.join(ROOT, "profiles", "%s_%s.md" % (kernel, workload))
    if not os.path.exists(path):
        return None, None
    txt = open(path).read()
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    h = re.search(r"source_sha256:\s*([0-9a-f]+)", txt)
    if not m or not h or h.group(1) != source_hash(kernel):
        return None, path
    return float(m.group(1)), path


# the source files each kernel is compiled from
KERNEL_SOURCES = {"fill": ("fill.cu", "fill_math.cuh", "fill_tables.h", "device.cuh", "ln_table.h",
                           "plan.h"),
                  "compare": ("compare.cu", "device.cuh", "plan.h"),
                  "eqsum": ("eqsum.cu", "device.cuh", "plan.h"),
                  "copy": ("copy.cu", "device.cuh", "plan.h"),
                  "eq64": ("eq64.cu", "eq64.h", "device.cuh", "plan.h")}


def _code_only(src):
    """A source's code with comments, blank lines and indentation removed:
    an edit to comments alone leaves the compiled kernel, and so the hash,
    unchanged."""
    tok = re.compile(r'"(?:\\.|[^"\\])*"|\'(?:\\.|[^\'\\])*\'|/\*.*?\*/|//[^\n]*', re.S)
    src = tok.sub(lambda m: m.group(0) if m.group(0)[0] in "\"'" else " ", src)
    return "\n".join(line.strip() for line in src.splitlines() if line.strip())


def source_hash(kernel):
    d = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_20711_gb300", "csrc")
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(csrc, f)) as fh:
            d.update(f.encode() + _code_only(fh.read()).encode())
    return d.hexdigest()[:16]


# ------------------------------------------------------------------ workload
def fill_specs_of(wl):
    """The regions a step fills: the input buffers, or the outputs themselves."""
    return wl.input_regions if wl.input_regions else wl.regions


def step_bytes(wl):
    """(fill bytes, physical verify bytes, logical verify bytes) of one step:
    the fill writes payload + guards; the check reads the reference once and
    every candidate once, guards included (logical: reference per candidate)."""
    fill = sum(r.alloc_bytes if r.dist != "none" else r.guard_lo + r.guard_hi
               for r in fill_specs_of(wl))
    payload = sum(r.payload_bytes for r in wl.regions)
    guards = sum(r.guard_lo + r.guard_hi for r in wl.regions)
    k = wl.n_cands
    return fill, payload * (1 + k) + guards * (1 + k), 2 * payload * k


def step_config(wl, world):
    fill, vp, vl = step_bytes(wl)
    return {"workload": wl.name, "description": wl.description, "fill_bytes": fill,
            "verify_bytes_physical": vp, "verify_bytes_logical": vl, "candidates": wl.n_cands,
            "l2": "inputs larger than L2 (129 MB); no flush",
            "parallelism": "replica per GPU" if world > 1 else "1 GPU"}


def make_candidates(wl, ref):
    """The workload's candidate outputs: copies of the reference arena (a
    torch uint8 tensor, on any device) perturbed by the workload's recipe."""
    W = _workloads()
    rng = np.random.default_rng(wl.seed + 77)
    recipe = wl.name.split("_8kx16k")[0].split("_4kx16k")[0]   # size variants share the recipe
    cands = []
    for j in range(wl.n_cands):
        c = ref.clone()
        if recipe == "batched_gemm_fp16":
            W.perturb_uniform_ulps(c, wl.regions[0], seed=wl.seed * 100 + j,
                                   magnitude=wl.ulp_magnitudes[j])
        elif recipe == "fp32_1m":
            W.perturb_fp32_single(c, wl)
        elif recipe == "attention_bf16":
            for r in wl.regions:
                W.perturb_ulp_noise(c, r, seed=wl.seed * 10 + r.region_id)
        elif recipe == "int_exact":
            for r in wl.regions:
                W.flip_bit(c, r, rng)
        elif recipe == "snapshot_4096":
            for r in wl.regions:
                W.perturb_sparse(c, r, rng, rate=1e-6)
            for k in rng.choice(len(wl.regions), 3, replace=False):
                W.corrupt_guard(c, wl.regions[int(k)], rng, "hi")
        cands.append(c)
    return cands


def _workloads():
    from paper_2608_20711_gb300 import workloads as W
    return W


class Setup:
    """Device buffers and region tables of one workload replica."""

    def __init__(self, name, device):
        import torch
        from paper_2608_20711_gb300 import asmv
        from paper_2608_20711_gb300 import workloads as W
        self.torch, self.asmv, self.W = torch, asmv, W
        self.name = name
        self.device = device
        wl = W.WORKLOADS[name]()
        self.wl = wl
        self.ctx = asmv.Context(device.index or 0)
        dev = device
        self.ref = torch.empty(wl.arena_bytes, dtype=torch.uint8, device=dev)
        self.ref_regs = asmv.regions_in_arena(wl.regions, self.ref.data_ptr())
        self.ctx.fill(self.ref_regs, seed=wl.seed)
        if wl.input_regions:
            self.inp = torch.empty(wl.input_arena_bytes, dtype=torch.uint8, device=dev)
            self.fill_regs = asmv.regions_in_arena(wl.input_regions, self.inp.data_ptr())
            self.fill_specs = wl.input_regions
        else:
            self.inp = None
            self.fill_regs = self.ref_regs
            self.fill_specs = wl.regions
        # candidates (input construction, outside the timed region)
        self.cands = make_candidates(wl, self.ref)
        self.cand_regs = [asmv.regions_in_arena(wl.regions, c.data_ptr()) for c in self.cands]
        torch.cuda.synchronize(dev)
        self.fill_bytes, self.verify_physical, self.verify_logical = step_bytes(wl)
        self.tol = wl.tol

    def step(self):
        """Fill, then check every candidate (K <= 8 share one reference read)."""
        self.ctx.fill(self.fill_regs, seed=self.wl.seed)
        if len(self.cands) == 1:
            return [self.ctx.compare(self.ref_regs, self.cand_regs[0], self.tol)]
        return self.ctx.compare_batched(self.ref_regs, self.cand_regs, self.tol)


# ------------------------------------------------------------------ CPU oracle
def _timed_until(budget_s, fn, n0, nmax):
    """Run fn(n) (which returns the work it did) with n growing until one
    run takes >= budget_s; at n == nmax, repeat until the budget is spent.
    Returns (n, seconds, work) summed over the measured runs."""
    n = n0
    while True:
        t0 = time.perf_counter()
        work = fn(n)
        dt = time.perf_counter() - t0
        if dt >= budget_s:
            return n, dt, work
        if n >= nmax:
            break
        n = min(nmax, n * max(2, int(budget_s / max(dt, 1e-3) * 0.7)))
    total_t, total_w = dt, work
    while total_t < budget_s:
        t0 = time.perf_counter()
        total_w += fn(n)
        total_t += time.perf_counter() - t0
    return n, total_t, total_w


class OracleSample:
    """A bounded sample of one step of a workload, built and checked on the
    host by the CPU oracle alone (no GPU library is loaded): every region of
    the workload scaled down by the same factor (at least one element each),
    the fill regions scaled so that the sample's fill and verify bytes keep
    the full step's ratio.  The reference arena comes from the oracle's fill,
    the candidates from the workload's recipe on host tensors; run() times the
    oracle's fill of the fill sample plus its check of every candidate."""

    def __init__(self, name, verify_bytes, threads):
        import copy
        import torch
        from oracle import oracle as O
        W = _workloads()
        self.O = O
        self.threads = int(threads)
        wl = W.WORKLOADS[name]()
        fill_full, verify_full, _ = step_bytes(wl)
        f = min(1.0, verify_bytes / verify_full)
        sample = copy.deepcopy(wl)
        for r in sample.regions:
            r.n_elems = max(1, int(r.n_elems * f))
        sample.arena_bytes = W.layout(sample.regions)
        if wl.input_regions:              # the same factor keeps the fill : verify ratio
            for r in sample.input_regions:
                r.n_elems = max(1, int(r.n_elems * f))
            sample.input_arena_bytes = W.layout(sample.input_regions)
        self.wl = sample
        self.ref = torch.zeros(sample.arena_bytes, dtype=torch.uint8)
        host = self.ref.numpy()
        for r in sample.regions:
            O.fill_region(host[r.offset:r.offset + r.alloc_bytes], r.n_elems, O.CODE_OF_DTYPE[r.dtype],
                          O.CODE_OF_DIST[r.dist], r.guard_lo, r.guard_hi, r.region_id, r.canary,
                          r.p0, r.p1, sample.seed, threads=self.threads)
        self.cands = [c.numpy() for c in make_candidates(sample, self.ref)]
        self.fill_specs = fill_specs_of(sample)
        self.fill_arena = np.zeros(W.layout(self.fill_specs) + 256, np.uint8)
        self.fill_bytes, self.verify_bytes, _ = step_bytes(sample)
        self.kinds = len({(r.dtype, r.dist) for r in self.fill_specs})

    def run(self):
        """(seconds of fill, seconds of check, mismatches found)."""
        O, wl, th = self.O, self.wl, self.threads
        t0 = time.perf_counter()
        for r in self.fill_specs:
            O.fill_region(self.fill_arena[r.offset:r.offset + r.alloc_bytes], r.n_elems,
                          O.CODE_OF_DTYPE[r.dtype], O.CODE_OF_DIST[r.dist], r.guard_lo, r.guard_hi,
                          r.region_id, r.canary, r.p0, r.p1, wl.seed, threads=th)
        t1 = time.perf_counter()
        ref = self.ref.numpy()
        mism = 0
        for c in self.cands:
            for r in wl.regions:
                t = wl.tol.get(r.dtype, _workloads().Tolerance(0.0, 0.0))
                a = ref[r.offset:r.offset + r.alloc_bytes]
                b = c[r.offset:r.offset + r.alloc_bytes]
                st = O.compare_region(a, r.guard_lo, r.guard_hi, r.canary, b, r.guard_lo, r.guard_hi,
                                      r.canary, r.n_elems, O.CODE_OF_DTYPE[r.dtype], t.atol, t.rtol,
                                      threads=th if r.n_elems >= (1 << 16) else 1)
                mism += int(st["mismatches"])
        t2 = time.perf_counter()
        return t1 - t0, t2 - t1, mism

    def describe(self, seconds):
        return ("oracle on host-built inputs: fill of %.1f MB (%d region kinds) and check of "
                "%.1f MB (reference + %d candidates, %d regions), %d threads, %.2f s"
                % (self.fill_bytes / 1e6, self.kinds, self.verify_bytes / 1e6, len(self.cands),
                   len(self.wl.regions), self.threads, seconds))


def cpu_oracle_sample(name, verify_bytes, threads=None, repeats=1):
    """The oracle as it stands on the host cores over a bounded sample of the
    workload (OracleSample): rate = sample bytes / measured seconds."""
    from oracle import oracle as O
    threads = O.host_threads() if threads is None else int(threads)
    smp = OracleSample(name, verify_bytes, threads)
    tf = tc = 0.0
    for _ in range(repeats):
        a, b, _ = smp.run()
        tf, tc = tf + a, tc + b
    nb = (smp.fill_bytes + smp.verify_bytes) * repeats
    return {"value": round(nb / (tf + tc) / 1e9, 4), "unit": UNIT, "cores": threads,
            "kind": "oracle", "sample": smp.describe(tf + tc),
            "fill_gbs": round(smp.fill_bytes * repeats / tf / 1e9, 4),
            "verify_gbs": round(smp.verify_bytes * repeats / tc / 1e9, 4),
            "seconds": round(tf + tc, 2)}


# ------------------------------------------------------------------ runs
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_mine(args):
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    setup = Setup(args.workload, device)
    ctx = setup.ctx
    stream = torch.cuda.current_stream(device)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(device)

    for _ in range(args.warmup):
        stats = setup.step()
    barrier()
    # kernel durations: CUDA events around each launch (one step at a time)
    ctx.set_timing(True)
    fill_ms, cmp_ms = [], []
    for _ in range(max(3, args.steps)):
        ctx.fill(setup.fill_regs, seed=setup.wl.seed)
        fill_ms.append(ctx.kernel_ms())
        if len(setup.cands) == 1:
            ctx.compare(setup.ref_regs, setup.cand_regs[0], setup.tol)
        else:
            ctx.compare_batched(setup.ref_regs, setup.cand_regs, setup.tol)
        cmp_ms.append(ctx.kernel_ms())
    ctx.set_timing(False)
    barrier()
    # the timed region: K whole steps
    launches0 = ctx.launches
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        barrier()
        ev0.record(stream)
        for _ in range(args.steps):
            stats = setup.step()
        ev1.record(stream)
        barrier()
    elapsed = ev0.elapsed_time(ev1) / 1e3
    launches = ctx.launches - launches0
    if world > 1:
        import torch.distributed as dist
        t = torch.tensor([elapsed], device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        elapsed = float(t.item())
    step_bytes = setup.fill_bytes + setup.verify_physical
    value = world * step_bytes * args.steps / elapsed / 1e9
    # e2e: the public API with host buffers (pinned), copies inside the timed region
    e2e = None
    if args.e2e:
        e2e = run_e2e(setup, args, device, world, barrier)
    peak, peak_kind = measured_peaks()
    f_ms, c_ms = float(np.mean(fill_ms)), float(np.mean(cmp_ms))
    fill_gbs = setup.fill_bytes / (f_ms / 1e3) / 1e9
    verify_gbs = setup.verify_physical / (c_ms / 1e3) / 1e9
    # the roofline of the step's dominant kernel: HBM, algorithmic bytes per launch over the
    # kernel's CUDA-event time, against the measured copy bandwidth
    kern = "compare" if c_ms >= f_ms else "fill"
    nbytes, ms = (setup.verify_physical, c_ms) if kern == "compare" else (setup.fill_bytes, f_ms)
    achieved = nbytes / (ms / 1e3) / 1e9
    traffic, _ = kernel_traffic(kern, args.workload)
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": traffic, "kernel": kern + "_kernel",
                "peak_kind": peak_kind + " (copy bandwidth, burst)",
                "algorithmic_bytes_per_launch": nbytes, "avg_launch_ms": round(ms, 4),
                "other_kernel": {"kernel": ("fill" if kern == "compare" else "compare") + "_kernel",
                                 "frac": round((fill_gbs if kern == "compare" else verify_gbs) / peak, 4)}}
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(elapsed / args.steps * 1e3, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": dtype_label(setup.wl),
        "data": "synthetic (seeded Philox fill; seeded candidate perturbations)",
        "config": step_config(setup.wl, world),
        "fill_gbs": round(fill_gbs, 1), "verify_gbs": round(verify_gbs, 1),
        "fill_frac": round(fill_gbs / peak, 4), "verify_frac": round(verify_gbs / peak, 4),
        "clocks": clk.summary(), "gpu_launches": launches, "roofline": roofline,
        "e2e": e2e,
    }
    if args.snapshot and args.workload != "snapshot_4096":
        line["snapshot_4096"] = run_snapshot(args, device, peak)
    if args.eq:
        line["eq1"] = run_eq1(setup, args, peak)
        line["eq1_f64"] = run_eq1_f64(setup, args, peak)
    if args.restore:
        line["restore"] = run_restore(setup, args, peak)
    if rank == 0 and world == 1 and args.cpu:
        line["cpu_baseline"] = cpu_oracle_sample(args.workload, CPU_SAMPLE_VERIFY_BYTES)
        one = cpu_oracle_sample(args.workload, CPU_SAMPLE_VERIFY_BYTES // 16, threads=1)
        line["cpu_baseline"]["single_thread"] = {k: one[k] for k in ("value", "fill_gbs", "verify_gbs",
                                                                      "seconds", "sample")}
    if rank == 0:
        mism = sum(int(s["mismatches"]) for cs in stats for s in cs)
        line["check"] = {"total_mismatches": mism}
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def dtype_label(wl):
    """What the path computes: the stored formats of the payloads it fills
    and checks, and the exact fp64 statistics."""
    fmts = sorted({r.dtype for r in fill_specs_of(wl)} | {r.dtype for r in wl.regions})
    return "/".join(fmts) + " payloads; statistics exact in fp64"


def run_snapshot(args, device, peak):
    """The 4096-region replay snapshot: its fill and its check of one
    candidate, each kernel timed alone with CUDA events around its launches
    (the same protocol as the step's kernels)."""
    import torch
    snap = Setup("snapshot_4096", device)
    ctx = snap.ctx
    ctx.fill(snap.fill_regs, seed=snap.wl.seed)
    ctx.compare(snap.ref_regs, snap.cand_regs[0], snap.tol)
    ctx.set_timing(True)
    fill_ms, cmp_ms = [], []
    for _ in range(max(5, args.steps)):
        ctx.fill(snap.fill_regs, seed=snap.wl.seed)
        fill_ms.append(ctx.kernel_ms())
        st = ctx.compare(snap.ref_regs, snap.cand_regs[0], snap.tol)
        cmp_ms.append(ctx.kernel_ms())
    ctx.set_timing(False)
    f_ms, c_ms = float(np.mean(fill_ms)), float(np.mean(cmp_ms))
    fill_gbs = snap.fill_bytes / (f_ms / 1e3) / 1e9
    verify_gbs = snap.verify_physical / (c_ms / 1e3) / 1e9
    out = {"regions": len(snap.wl.regions), "fill_bytes": snap.fill_bytes,
           "verify_bytes_physical": snap.verify_physical,
           "fill_avg_launch_ms": round(f_ms, 4), "verify_avg_launch_ms": round(c_ms, 4),
           "fill_gbs": round(fill_gbs, 1), "verify_gbs": round(verify_gbs, 1),
           "fill_frac": round(fill_gbs / peak, 4), "verify_frac": round(verify_gbs / peak, 4),
           "fill_traffic": kernel_traffic("fill", "snapshot_4096")[0],
           "verify_traffic": kernel_traffic("compare", "snapshot_4096")[0],
           "mismatches": int(sum(s["mismatches"] for s in st)),
           "bad_guard_bytes": int(sum(s["guard_bad_bytes"] for s in st))}
    ctx.close()
    del snap
    torch.cuda.empty_cache()
    return out


def run_eq1(setup, args, peak):
    """Eq. 1 as a whole over the step's reference and candidates
    (asmv_compare_eq); the kernel that adds the exact cosine sums is timed
    alone, with CUDA events around its launches on the call's stream."""
    ctx = setup.ctx
    floats = ("f32", "bf16", "f16", "f8e4m3")
    k = len(setup.cands)
    ctx.compare_eq(setup.ref_regs, setup.cand_regs, setup.tol)
    ctx.set_timing(True)
    ms = []
    for _ in range(max(3, args.steps)):
        _, eqs = ctx.compare_eq(setup.ref_regs, setup.cand_regs, setup.tol)
        ms.append(ctx.kernel_ms())
    ctx.set_timing(False)
    payload = sum(r.payload_bytes for r in setup.wl.regions if r.dtype in floats)
    nbytes = payload * (1 + k)                 # the reference once, every candidate once
    elems = sum(r.n_elems for r in setup.wl.regions if r.dtype in floats)
    avg = float(np.mean(ms))
    gbs = nbytes / (avg / 1e3) / 1e9
    traffic, _ = kernel_traffic("eqsum", args.workload)
    return {"kernel": "eq_kernel", "avg_launch_ms": round(avg, 4),
            "algorithmic_bytes_per_launch": nbytes, "element_pairs_per_launch": elems * k,
            "gbs": round(gbs, 1), "hbm_frac": round(gbs / peak, 4), "traffic": traffic,
            "pairs_per_s": round(elems * k / (avg / 1e3), 1),
            "theta": setup.asmv.THETA, "tau": setup.asmv.TAU,
            "passing": int(sum(e["eq"] for cs in eqs for e in cs)), "checks": k * len(eqs[0])}


def run_eq1_f64(setup, args, peak, k=2):
    """Eq. 1 over binary64 outputs of the same size as the step's reference
    (a N(0, 1) reference from the guarded fill, k candidates with the last
    bit flipped at every 7th element), through asmv_compare_eq; its binary64
    sums kernel timed alone with CUDA events around its launches."""
    torch, ctx, asmv = setup.torch, setup.ctx, setup.asmv
    floats = ("f32", "bf16", "f16", "f8e4m3")
    n = max(1, sum(r.payload_bytes for r in setup.wl.regions if r.dtype in floats) // 8)
    ref = torch.empty(n, dtype=torch.float64, device=setup.device)

    def table(t):
        return [asmv.make_region(t.data_ptr(), n, "f64", "normal", 0, 0, region_id=1, p0=0.0, p1=1.0)]
    ctx.fill(table(ref), seed=11)
    cands = []
    for j in range(k):
        c = ref.clone()
        c.view(torch.int64)[j::7] ^= 1
        cands.append(c)
    tol = {"f64": (1e-9, 1e-9)}
    ctx.compare_eq(table(ref), [table(c) for c in cands], tol)
    ctx.set_timing(True)
    ms = []
    for _ in range(max(3, args.steps)):
        _, eqs = ctx.compare_eq(table(ref), [table(c) for c in cands], tol)
        ms.append(ctx.kernel_ms())
    ctx.set_timing(False)
    avg = float(np.mean(ms))
    nbytes = 8 * n * (1 + k)
    gbs = nbytes / (avg / 1e3) / 1e9
    traffic, _ = kernel_traffic("eq64", args.workload)
    del ref, cands
    return {"kernel": "eq64_kernel", "values": n, "candidates": k, "avg_launch_ms": round(avg, 4),
            "algorithmic_bytes_per_launch": nbytes, "gbs": round(gbs, 1),
            "hbm_frac": round(gbs / peak, 4), "traffic": traffic,
            "pairs_per_s": round(n * k / (avg / 1e3), 1),
            "passing": int(sum(e[0]["eq"] for e in eqs)), "cos": [e[0]["cos"] for e in eqs]}


def run_restore(setup, args, peak):
    """Tier 2 restore of the step's input regions (asmv_restore) from a
    snapshot taken with asmv_capture; the copy kernel timed alone with CUDA
    events around its launch."""
    torch = setup.torch
    ctx = setup.ctx
    specs = setup.fill_specs
    offs, total = [], 0
    for r in specs:
        total = (total + 255) // 256 * 256
        offs.append(total)
        total += r.payload_bytes
    snap = torch.empty(max(total, 1), dtype=torch.uint8, device=setup.device)
    src = [snap.data_ptr() + o for o in offs]
    ctx.capture(setup.fill_regs, src)
    ctx.restore(setup.fill_regs, src)
    ctx.set_timing(True)
    ms = []
    for _ in range(max(3, args.steps)):
        ctx.restore(setup.fill_regs, src)
        ms.append(ctx.kernel_ms())
    ctx.set_timing(False)
    torch.cuda.synchronize(setup.device)
    payload = sum(r.payload_bytes for r in specs)
    guards = sum(r.guard_lo + r.guard_hi for r in specs)
    nbytes = 2 * payload + guards                # source read, payload written, guards written
    avg = float(np.mean(ms))
    gbs = nbytes / (avg / 1e3) / 1e9
    traffic, _ = kernel_traffic("copy", args.workload)
    del snap
    return {"kernel": "copy_kernel", "regions": len(specs), "avg_launch_ms": round(avg, 4),
            "algorithmic_bytes_per_launch": nbytes, "gbs": round(gbs, 1),
            "hbm_frac": round(gbs / peak, 4), "traffic": traffic,
            "peak_kind": "measured copy bandwidth (read + write bytes)"}


def run_e2e(setup, args, device, world, barrier):
    """Host buffers through the public API: every step copies the reference
    and candidate outputs from pinned host memory, fills, checks, and reads
    the statistics back.  The copies run on a copy stream while the fill
    (which writes other buffers) runs on the compute stream; the check waits
    for both.  Each step's copies wait for the previous step's check, which
    reads the same device buffers."""
    import torch
    ctx = setup.ctx
    host_ref = setup.ref.cpu().pin_memory()
    host_cands = [c.cpu().pin_memory() for c in setup.cands]
    stream = torch.cuda.current_stream(device)
    copy_stream = torch.cuda.Stream(device)
    h2d = host_ref.numel() + sum(h.numel() for h in host_cands)
    nstat = len(setup.wl.regions) * len(setup.cands)
    d2h = 64 * nstat
    pairs = [(setup.ref, host_ref)] + list(zip(setup.cands, host_cands))

    def e2e_step():
        copy_stream.wait_stream(stream)
        with torch.cuda.stream(copy_stream):
            for d, h in pairs:
                d.copy_(h, non_blocking=True)
        ctx.fill(setup.fill_regs, seed=setup.wl.seed)
        stream.wait_stream(copy_stream)
        if len(setup.cands) == 1:
            return [ctx.compare(setup.ref_regs, setup.cand_regs[0], setup.tol)]
        return ctx.compare_batched(setup.ref_regs, setup.cand_regs, setup.tol)   # stats to the host

    for _ in range(2):
        e2e_step()
    # the same host-to-device copies alone: the link's rate for these buffers
    torch.cuda.synchronize(device)
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    h2d_ms = []
    for _ in range(2):
        c0.record(copy_stream)
        with torch.cuda.stream(copy_stream):
            for d, h in pairs:
                d.copy_(h, non_blocking=True)
        c1.record(copy_stream)
        c1.synchronize()
        h2d_ms.append(c0.elapsed_time(c1))
    h2d_s = min(h2d_ms) / 1e3
    barrier()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        e2e_step()
    ev1.record(stream)
    barrier()
    el = ev0.elapsed_time(ev1) / 1e3
    step_bytes = setup.fill_bytes + setup.verify_physical
    return {"value": round(world * step_bytes * args.steps / el / 1e9, 1), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": round(el / args.steps * 1e3, 3),
            "h2d_gbs": round(h2d / h2d_s / 1e9, 1), "h2d_ms": round(h2d_s * 1e3, 3),
            "overlap": "host-to-device copies on a copy stream, concurrent with the fill"}


def run_reference(args):
    """The oracle (the plain CPU program) on the same workload, metric and
    config: every step is one OracleSample of the workload run on the host
    cores, with inputs the oracle built on the host (no GPU library is
    loaded); value = sample bytes / measured seconds."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from oracle import oracle as O
    W = _workloads()
    wl = W.WORKLOADS[args.workload]()
    threads = O.host_threads()
    smp = OracleSample(args.workload, REF_STEP_VERIFY_BYTES, threads)
    for _ in range(args.warmup):
        smp.run()
    secs = []
    for _ in range(args.steps):
        tf, tc, _ = smp.run()
        secs.append(tf + tc)
    total = float(np.sum(secs))
    nb = (smp.fill_bytes + smp.verify_bytes) * args.steps
    value = nb / total / 1e9
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total / args.steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": dtype_label(wl),
            "data": "synthetic (the oracle's seeded fill and the workload's candidate recipe, on the host)",
            "config": step_config(wl, world),
            "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": threads,
                             "kind": "oracle", "sample": smp.describe(total / args.steps) + " per step"},
            "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mine", choices=["mine", "reference"])
    ap.add_argument("--workload", default="batched_gemm_fp16")
    ap.add_argument("--no-e2e", dest="e2e", action="store_false")
    ap.add_argument("--no-cpu", dest="cpu", action="store_false")
    ap.add_argument("--no-eq", dest="eq", action="store_false")
    ap.add_argument("--no-restore", dest="restore", action="store_false")
    ap.add_argument("--no-snapshot", dest="snapshot", action="store_false")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    if args.impl == "reference":
        from oracle import build as oracle_build      # the oracle only: no GPU library
        oracle_build.build()
        run_reference(args)
    else:
        import __graft_entry__
        __graft_entry__.build()
        run_mine(args)


if __name__ == "__main__":
    main()
