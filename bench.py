"""Throughput of the differential-oracle hot path on GB300.

One step = one pass of the whole hot path over one batch of synthetic
input: the Tier 1 guarded fill of the workload's input regions followed by
the equivalence check of the reference output against every candidate
(AsmEvo Sec. 3.4 and Eq. 1).  Default workload: a 16 GiB guarded fill of
GEMM input buffers, then one fp16 [32768, 32768] reference checked against
8 candidates carrying 0..8 ULP of noise.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mine|reference]
                       [--workload NAME] [--no-e2e] [--no-cpu] [--no-eq]

Beside the step, the line carries `eq1`: Eq. 1 as a whole (the exact sums
of the cosine term over the same reference and candidates), its kernel
timed alone with CUDA events; `eq1_f64`: the same for binary64 outputs of
the reference's size; and `restore`: the Tier 2 restore of the step's input
regions from a captured snapshot, timed the same way.
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
KERNEL_SOURCES = {"fill": ("fill.cu", "fill_math.cuh", "device.cuh", "ln_table.h", "plan.h"),
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


# Algorithmic operations of the fill per 16-byte chunk, counted from the
# operation sequences the fill's specification states (include/asmv.h); one
# op is one 32-bit integer or fp32 operation: a 32x32->64 product, a
# three-input XOR, an IEEE add/mul/fma/sqrt, a conversion, a shift or mask.
PHILOX_BLOCK_OPS = 40          # 10 rounds x (2 wide products + 2 three-input XORs)
BOX_MULLER_PAIR_OPS = 54       # word prep 3, ln 20, rho 2, sincos 23, z 2, mean+std*z 4
UNIFORM_ELEM_OPS = 5           # shift, int->float, scale, multiply, add
INT_RANGE_ELEM_OPS = 2         # wide product, add
# GB300: 152 SMs x 128 fp32/int32 lanes x 2070 MHz (maximum SM clock)
ALU_PEAK_TOPS = 152 * 128 * 2.070e9 / 1e12


def fill_ops_per_chunk(dtype, dist):
    size = {"f32": 4, "bf16": 2, "f16": 2, "f8e4m3": 1, "i32": 4, "i8": 1, "u8": 1}[dtype]
    elems = 16 // size
    blocks = max(1, elems // 4) if dist != "raw" else 1
    packs = elems // 2 if size < 4 else 0          # packed conversions to 16/8-bit
    if dist == "raw":
        return PHILOX_BLOCK_OPS
    if dist == "none":
        return 0
    if dist == "int_range":
        return blocks * PHILOX_BLOCK_OPS + elems * INT_RANGE_ELEM_OPS
    if dist == "uniform":
        return blocks * PHILOX_BLOCK_OPS + elems * UNIFORM_ELEM_OPS + packs
    return blocks * PHILOX_BLOCK_OPS + (elems // 2) * BOX_MULLER_PAIR_OPS + packs


def fill_algorithmic_ops(regions):
    return sum(((r.payload_bytes + 15) // 16) * fill_ops_per_chunk(r.dtype, r.dist)
               for r in regions)


# ------------------------------------------------------------------ workload
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
        rng = np.random.default_rng(wl.seed + 77)
        self.cands = []
        ncand = wl.n_cands
        recipe = wl.name               # the recipe, shared by the size variants
        for j in range(ncand):
            c = self.ref.clone()
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
            self.cands.append(c)
        self.cand_regs = [asmv.regions_in_arena(wl.regions, c.data_ptr()) for c in self.cands]
        torch.cuda.synchronize(dev)
        self.fill_bytes = sum(r.alloc_bytes if r.dist != "none" else r.guard_lo + r.guard_hi
                              for r in self.fill_specs)
        ref_payload = sum(r.payload_bytes for r in wl.regions)
        guards = sum(r.guard_lo + r.guard_hi for r in wl.regions)
        self.verify_physical = ref_payload * (1 + ncand) + guards * (1 + ncand)
        self.verify_logical = 2 * ref_payload * ncand
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


def cpu_oracle_sample(setup, budget_s=12.0, threads=None):
    """The oracle as it stands, on the host cores (all of them unless
    `threads` is given), over a bounded sample of the same workload: element
    prefixes of the fill regions (one of each dtype/distribution kind) and
    of the reference/candidate payloads.  The two measured rates are
    combined over the step's byte mix."""
    from oracle import oracle as O
    ORACLE_DTYPE, ORACLE_DIST = O.CODE_OF_DTYPE, O.CODE_OF_DIST
    W = setup.W
    threads = O.host_threads() if threads is None else int(threads)
    kinds = {}
    for r in setup.fill_specs:
        kinds.setdefault((r.dtype, r.dist), r)
    cap_bytes = 256 << 20
    bufs = {k: np.zeros(min(r.payload_bytes, cap_bytes), np.uint8) for k, r in kinds.items()}

    def fill(n_bytes):
        done = 0
        for (dt, dist), r in kinds.items():
            sz = W.DTYPE_SIZE[dt]
            n = min(n_bytes // sz, bufs[(dt, dist)].size // sz)
            O.fill_region(bufs[(dt, dist)], n, ORACLE_DTYPE[dt], ORACLE_DIST[dist], 0, 0,
                          r.region_id, r.canary, r.p0, r.p1, setup.wl.seed, threads=threads)
            done += n * sz
        return done

    _, t_fill, fill_done = _timed_until(budget_s / 2, fill, 1 << 16, cap_bytes)
    # reference/candidate payload prefixes of the first region
    r = setup.wl.regions[0]
    nb = min(r.payload_bytes, cap_bytes // max(1, len(setup.cands)))
    a = setup.ref[r.payload_offset:r.payload_offset + nb].cpu().numpy()
    cs = [c[r.payload_offset:r.payload_offset + nb].cpu().numpy() for c in setup.cands]
    t = setup.tol.get(r.dtype, W.Tolerance(0.0, 0.0))
    sz = W.DTYPE_SIZE[r.dtype]

    def compare(n_bytes):
        n = min(n_bytes, nb) // sz
        for c in cs:
            O.compare_payload(a, c, ORACLE_DTYPE[r.dtype], n, t.atol, t.rtol, threads=threads)
        return n * sz * (1 + len(cs))

    _, t_cmp, cmp_done = _timed_until(budget_s / 2, compare, 1 << 16, nb)
    fill_rate = fill_done / t_fill
    cmp_rate = cmp_done / t_cmp
    step_s = setup.fill_bytes / fill_rate + setup.verify_physical / cmp_rate
    value = (setup.fill_bytes + setup.verify_physical) / step_s / 1e9
    sample = ("oracle fill of %.1f MB over %d region kinds and compare of %.1f MB of "
              "reference + %d candidate payload prefixes, %d threads; rates combined over the "
              "step's fill/verify byte mix" % (fill_done / 1e6, len(kinds), cmp_done / 1e6,
                                               len(cs), threads))
    return {"value": round(value, 4), "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": sample, "fill_gbs": round(fill_rate / 1e9, 4),
            "verify_gbs": round(cmp_rate / 1e9, 4), "seconds": round(t_fill + t_cmp, 2)}


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
    fill_ops = fill_algorithmic_ops(setup.fill_specs)
    fill_alu_ms = fill_ops / (ALU_PEAK_TOPS * 1e12) * 1e3
    fill_hbm_ms = setup.fill_bytes / (peak * 1e9) * 1e3
    if c_ms >= f_ms:
        traffic, _ = kernel_traffic("compare", args.workload)
        achieved = setup.verify_physical / (c_ms / 1e3) / 1e9
        roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                    "frac": round(achieved / peak, 4), "traffic": traffic, "kernel": "compare",
                    "peak_kind": peak_kind + " (copy bandwidth, burst)",
                    "algorithmic_bytes_per_launch": setup.verify_physical,
                    "avg_launch_ms": round(c_ms, 4)}
    else:
        traffic, _ = kernel_traffic("fill", args.workload)
        # the fill's roof is the ALU when its operations take longer than its bytes
        if fill_alu_ms >= fill_hbm_ms:
            achieved = fill_ops / (f_ms / 1e3) / 1e12
            roofline = {"bound": "alu", "achieved": round(achieved, 3), "peak": round(ALU_PEAK_TOPS, 3),
                        "unit": "Top/s", "frac": round(achieved / ALU_PEAK_TOPS, 4),
                        "traffic": traffic, "kernel": "fill",
                        "peak_kind": "derived: 152 SMs x 128 lanes x 2070 MHz",
                        "algorithmic_ops_per_launch": fill_ops, "avg_launch_ms": round(f_ms, 4),
                        "hbm_gbs": round(fill_gbs, 1), "hbm_frac": round(fill_gbs / peak, 4)}
        else:
            achieved = setup.fill_bytes / (f_ms / 1e3) / 1e9
            roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                        "frac": round(achieved / peak, 4), "traffic": traffic, "kernel": "fill",
                        "peak_kind": peak_kind + " (copy bandwidth, burst)",
                        "algorithmic_bytes_per_launch": setup.fill_bytes,
                        "avg_launch_ms": round(f_ms, 4)}
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(elapsed / args.steps * 1e3, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded Philox fill; seeded candidate perturbations)",
        "config": {"workload": args.workload, "description": setup.wl.description,
                   "fill_bytes": setup.fill_bytes, "verify_bytes_physical": setup.verify_physical,
                   "verify_bytes_logical": setup.verify_logical, "candidates": len(setup.cands),
                   "l2": "inputs larger than L2 (129 MB); no flush",
                   "parallelism": "replica per GPU" if world > 1 else "1 GPU"},
        "fill_gbs": round(fill_gbs, 1), "verify_gbs": round(verify_gbs, 1),
        "fill_frac": round(fill_gbs / peak, 4), "verify_frac": round(verify_gbs / peak, 4),
        "clocks": clk.summary(), "gpu_launches": launches, "roofline": roofline,
        "e2e": e2e,
    }
    if args.eq:
        line["eq1"] = run_eq1(setup, args, peak)
        line["eq1_f64"] = run_eq1_f64(setup, args, peak)
    if args.restore:
        line["restore"] = run_restore(setup, args, peak)
    if rank == 0 and world == 1 and args.cpu:
        line["cpu_baseline"] = cpu_oracle_sample(setup)
        one = cpu_oracle_sample(setup, budget_s=4.0, threads=1)
        line["cpu_baseline"]["single_thread"] = {k: one[k] for k in ("value", "fill_gbs", "verify_gbs",
                                                                      "seconds")}
    if rank == 0:
        mism = sum(int(s["mismatches"]) for cs in stats for s in cs)
        line["check"] = {"total_mismatches": mism}
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


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
            "overlap": "host-to-device copies on a copy stream, concurrent with the fill"}


def run_reference(args):
    """The oracle (plain CPU program) on the same workload: each step is a
    bounded sample, extrapolated to the step's byte mix."""
    world, rank, local = dist_env()
    if rank != 0:
        return
    import torch
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    setup = Setup(args.workload, device)
    for _ in range(args.warmup):
        pass
    vals, secs = [], []
    for _ in range(args.steps):
        r = cpu_oracle_sample(setup, budget_s=max(2.0, 60.0 / max(1, args.steps)))
        vals.append(r["value"])
        secs.append(r["seconds"])
    step_bytes = setup.fill_bytes + setup.verify_physical
    value = float(np.median(vals))
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(step_bytes / (value * 1e9) * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": args.workload},
            "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": r["cores"],
                             "kind": "oracle", "sample": r["sample"]},
            "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
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
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    import __graft_entry__
    __graft_entry__.build()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_mine(args)


if __name__ == "__main__":
    main()
