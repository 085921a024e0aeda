"""Seeded synthetic workloads: region tables, arena layout and candidate
construction.

This module is the one input generator shared by the tests, the bench and
the oracle-side checks.  It holds none of the method's arithmetic: no
Philox, no fill, no predicate.  It only describes *which* regions exist
(sizes, dtypes, distributions, guard bands) and builds candidate outputs
by perturbing a reference copy (ULP steps, bit flips, NaN/Inf injection,
guard corruption) with numpy's / torch's own generators.

The five workloads stand in for the paper's captured dispatches (AsmEvo
Sec. 3.4, Tier 1 synthetic inputs and Tier 2 referenced-memory regions);
the captured binaries are not available, so shapes follow the kernels the
paper evaluates (attention outputs, block tables, quantised weights, a GEMM
output, a pointer-rich replay snapshot).
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence

import numpy as np

DTYPES = ("f32", "bf16", "f16", "f8e4m3", "i32", "i8", "u8", "f8e5m2", "f8e4m3fnuz",
          "f8e5m2fnuz", "f64", "i16", "i64")
DTYPE_SIZE = {"f32": 4, "bf16": 2, "f16": 2, "f8e4m3": 1, "i32": 4, "i8": 1, "u8": 1,
              "f8e5m2": 1, "f8e4m3fnuz": 1, "f8e5m2fnuz": 1, "f64": 8, "i16": 2, "i64": 8}
FLOAT_DTYPES = ("f32", "bf16", "f16", "f8e4m3", "f8e5m2", "f8e4m3fnuz", "f8e5m2fnuz", "f64")
DISTS = ("raw", "uniform", "normal", "int_range", "none")

# largest finite value's bit pattern, per float format (sign-magnitude)
_MAX_FINITE_BITS = {"f32": 0x7F7FFFFF, "bf16": 0x7F7F, "f16": 0x7BFF, "f8e4m3": 0x7E,
                    "f8e5m2": 0x7B, "f8e4m3fnuz": 0x7F, "f8e5m2fnuz": 0x7F,
                    "f64": 0x7FEFFFFFFFFFFFFF}
_BITS = {"f32": 32, "bf16": 16, "f16": 16, "f8e4m3": 8, "i32": 32, "i8": 8, "u8": 8,
         "f8e5m2": 8, "f8e4m3fnuz": 8, "f8e5m2fnuz": 8, "f64": 64, "i16": 16, "i64": 64}

ARENA_ALIGN = 256


@dataclasses.dataclass
class Region:
    """One guarded allocation: [guard_lo | payload | guard_hi]."""
    name: str
    dtype: str
    n_elems: int
    dist: str = "raw"
    p0: float = 0.0
    p1: float = 0.0
    guard_lo: int = 0
    guard_hi: int = 0
    canary: int = 0xA5
    region_id: int = 0
    offset: int = 0            # allocation start within its arena (set by layout)

    @property
    def payload_bytes(self) -> int:
        return self.n_elems * DTYPE_SIZE[self.dtype]

    @property
    def alloc_bytes(self) -> int:
        return self.guard_lo + self.payload_bytes + self.guard_hi

    @property
    def payload_offset(self) -> int:
        return self.offset + self.guard_lo


def layout(regions: Sequence[Region], align: int = ARENA_ALIGN, base: int = 0) -> int:
    """Place allocations back to back in one arena, each start aligned to
    `align` bytes; returns the arena size."""
    off = base
    for r in regions:
        off = (off + align - 1) // align * align
        r.offset = off
        off += r.alloc_bytes
    return (off + align - 1) // align * align


@dataclasses.dataclass
class Tolerance:
    atol: float
    rtol: float


@dataclasses.dataclass
class Workload:
    name: str
    seed: int
    regions: List[Region]
    arena_bytes: int
    tol: dict                      # dtype name -> Tolerance
    description: str = ""
    # bench-only extras (the batched case)
    input_regions: Optional[List[Region]] = None
    input_arena_bytes: int = 0
    n_cands: int = 1
    ulp_magnitudes: Optional[List[int]] = None

    @property
    def payload_bytes(self) -> int:
        return sum(r.payload_bytes for r in self.regions)


# torch.testing-style defaults per dtype (used where a workload states none)
DEFAULT_TOL = {
    "f32": Tolerance(1e-5, 1.3e-6),
    "bf16": Tolerance(1e-5, 1.6e-2),
    "f16": Tolerance(1e-5, 1e-3),
    "f8e4m3": Tolerance(1e-5, 0.125),
    "f8e5m2": Tolerance(1e-5, 0.25),
    "f8e4m3fnuz": Tolerance(1e-5, 0.125),
    "f8e5m2fnuz": Tolerance(1e-5, 0.25),
    "f64": Tolerance(1e-7, 1e-7),
}


def _tol(**over):
    t = dict(DEFAULT_TOL)
    t.update(over)
    return t


# --------------------------------------------------------------------------
# The five workloads
# --------------------------------------------------------------------------
def fp32_single(n: int = 1 << 20, guard: int = 4096) -> Workload:
    """One fp32 region, U[-1, 1) from seed 1, 4 KiB guard bands of 0xA5."""
    regs = [Region("x", "f32", n, "uniform", -1.0, 1.0, guard, guard, 0xA5, 0)]
    size = layout(regs)
    return Workload("fp32_1m", 1, regs, size, _tol(f32=Tolerance(1e-5, 1e-5)),
                    "single fp32 region, 37 seeded perturbations, one bad guard byte")


def attention_bf16(batch=16, heads=32, seq=2048, head_dim=128, guard=4096) -> Workload:
    """Attention outputs: O bf16 [B,H,S,D] and LSE fp32 [B,H,S], N(0,1)."""
    regs = [Region("O", "bf16", batch * heads * seq * head_dim, "normal", 0.0, 1.0,
                   guard, guard, 0xA5, 0),
            Region("LSE", "f32", batch * heads * seq, "normal", 0.0, 1.0,
                   guard, guard, 0xA5, 1)]
    size = layout(regs)
    return Workload("attention_bf16", 2, regs, size,
                    _tol(bf16=Tolerance(1e-2, 1.6e-2), f32=Tolerance(1e-5, 1e-5)),
                    "bf16 O [16,32,2048,128] + fp32 LSE [16,32,2048]; ULP noise")


def int_exact(scale: int = 1, guard: int = 4096) -> Workload:
    """Integer/index buffers that must be bit-exact: block table, int8
    weights, slot mapping.  `scale` divides the sizes for small cases."""
    regs = [Region("block_table", "i32", 256 * 512 // scale, "int_range", 0, 131072,
                   guard, guard, 0xA5, 0),
            Region("weights", "i8", 8192 * 8192 // scale, "raw", 0, 0, guard, guard, 0xA5, 1),
            Region("slot_mapping", "i32", 1048576 // scale, "int_range", 0, 1 << 20,
                   guard, guard, 0xA5, 2)]
    size = layout(regs)
    return Workload("int_exact", 3, regs, size, _tol(),
                    "int32 [256,512] + int8 [8192,8192] + int32 [1M]; one bit flip each")


SNAPSHOT_DTYPES = ("f32", "bf16", "f16", "f8e4m3", "i32", "i8")


def snapshot(n_regions: int = 4096, total_bytes: int = 8 << 30, median: int = 64 << 10,
             sigma: float = 2.6, cap: int = 256 << 20, guard: int = 256,
             seed: int = 4) -> Workload:
    """Pointer-rich replay snapshot: lognormal region sizes (median 64 KiB,
    cap 256 MiB, rescaled to ~total_bytes), dtypes uniform over six types,
    N(0,1) floats and full-range raw ints, 256 B guard bands."""
    rng = np.random.default_rng([seed, 3])
    raw = np.exp(rng.normal(math.log(median), sigma, n_regions))
    sizes = np.minimum(raw, cap)
    for _ in range(50):                      # rescale toward the target total
        s = total_bytes / sizes.sum()
        if abs(s - 1.0) < 1e-3:
            break
        sizes = np.minimum(sizes * s, cap)
    sizes = np.maximum(sizes, 16.0)
    dts = rng.integers(0, len(SNAPSHOT_DTYPES), n_regions)
    regs = []
    for i in range(n_regions):
        dt = SNAPSHOT_DTYPES[dts[i]]
        n = max(1, int(sizes[i]) // DTYPE_SIZE[dt])
        if dt in FLOAT_DTYPES:
            regs.append(Region("r%d" % i, dt, n, "normal", 0.0, 1.0, guard, guard, 0xA5, i))
        else:
            regs.append(Region("r%d" % i, dt, n, "raw", 0, 0, guard, guard, 0xA5, i))
    size = layout(regs)
    return Workload("snapshot_4096", seed, regs, size, _tol(),
                    "4096 mixed-dtype regions, lognormal sizes, 256 B guards")


def batched_gemm(rows: int = 32768, cols: int = 32768, n_cands: int = 8,
                 input_bytes: int = 16 << 30, input_regions: int = 64,
                 guard: int = 4096) -> Workload:
    """Batched candidate gating: one fp16 GEMM output [rows, cols] N(0, 0.5)
    against n_cands candidates with 0..8 ULP noise, preceded by a guarded
    fill of `input_bytes` of input buffers (fp16 N(0,1) activations and int8
    raw weights, alternating)."""
    ref = [Region("C", "f16", rows * cols, "normal", 0.0, 0.5, guard, guard, 0xA5, 1000)]
    size = layout(ref)
    per = input_bytes // input_regions
    ins = []
    for i in range(input_regions):
        if i % 2 == 0:
            ins.append(Region("in%d" % i, "f16", per // 2, "normal", 0.0, 1.0,
                              guard, guard, 0xA5, i))
        else:
            ins.append(Region("in%d" % i, "i8", per, "raw", 0, 0, guard, guard, 0xA5, i))
    in_size = layout(ins)
    mags = [0, 1, 2, 3, 4, 5, 6, 8][:n_cands] if n_cands <= 8 else \
        [k % 9 for k in range(n_cands)]
    return Workload("batched_gemm_fp16", 5, ref, size, _tol(f16=Tolerance(1e-5, 1e-3)),
                    "fp16 [32768,32768] ref x 8 candidates (0..8 ULP) after a 16 GiB fill",
                    input_regions=ins, input_arena_bytes=in_size, n_cands=n_cands,
                    ulp_magnitudes=mags)


WORKLOADS = {
    "fp32_1m": fp32_single,
    "attention_bf16": attention_bf16,
    "int_exact": int_exact,
    "snapshot_4096": snapshot,
    "batched_gemm_fp16": batched_gemm,
    # smaller cases of the same kernels (above L2, a few GB on the device)
    "batched_gemm_fp16_8kx16k": lambda: batched_gemm(rows=8192, cols=16384,
                                                     input_bytes=1 << 30, input_regions=8),
    "batched_gemm_fp16_4kx16k": lambda: batched_gemm(rows=4096, cols=16384,
                                                     input_bytes=512 << 20, input_regions=4),
    "snapshot_4096_1g": lambda: snapshot(total_bytes=1 << 30),
}


# --------------------------------------------------------------------------
# Candidate construction (bench/test input only; not part of the method)
# --------------------------------------------------------------------------
def _torch():
    import torch
    return torch


def _ordered(bits, dtype):
    """Sign-magnitude float bits -> position on the ordered integer line
    (two's complement; +0 and -0 both map to 0)."""
    nb = _BITS[dtype]
    sign = (bits >> (nb - 1)) & 1
    mag = bits & ((1 << (nb - 1)) - 1)
    return mag - 2 * sign * mag


def _from_ordered(o, dtype):
    torch = _torch()
    nb = _BITS[dtype]
    neg = o < 0
    mag = torch.where(neg, -o, o)
    return torch.where(neg, mag | (1 << (nb - 1)), mag)


def ulp_step(bits, steps, dtype):
    """Move float values (given as int64 bit patterns) by `steps` ULPs along
    the ordered line; finite values are clamped to the largest finite value,
    NaN and Inf are left alone."""
    torch = _torch()
    nb = _BITS[dtype]
    mag = bits & ((1 << (nb - 1)) - 1)
    if dtype == "f8e4m3":
        special = mag == 0x7F
    elif dtype == "f32":
        special = mag >= 0x7F800000
    elif dtype == "bf16":
        special = mag >= 0x7F80
    else:
        special = mag >= 0x7C00
    o = _ordered(bits, dtype) + steps
    mx = _MAX_FINITE_BITS[dtype]
    o = torch.clamp(o, -mx, mx)
    return torch.where(special, bits, _from_ordered(o, dtype))


def _elem_view(arena, region):
    """The region's payload as a tensor of its storage width, and that dtype."""
    torch = _torch()
    sz = DTYPE_SIZE[region.dtype]
    seg = arena[region.payload_offset:region.payload_offset + region.payload_bytes]
    tdt = {4: torch.int32, 2: torch.int16, 1: torch.uint8}[sz]
    return seg.view(tdt), tdt


def _bits_of(t, dtype):
    """Unsigned bit patterns (int64) of stored elements."""
    torch = _torch()
    return t.to(torch.int64) & ((1 << _BITS[dtype]) - 1)


def _to_storage(bits64, tdt, dtype):
    """Unsigned bit patterns -> tensor of the storage dtype."""
    torch = _torch()
    nb = _BITS[dtype]
    b = bits64 & ((1 << nb) - 1)
    if tdt == torch.uint8:
        return b.to(torch.uint8)
    b = torch.where(b >= (1 << (nb - 1)), b - (1 << nb), b)
    return b.to(tdt)


def _positions(rng, n, k):
    """k distinct positions in [0, n), sorted."""
    if k >= n:
        return np.arange(n)
    return np.sort(rng.choice(n, size=k, replace=False))


def corrupt_guard(arena, region, rng, side="hi"):
    """Overwrite one seeded guard byte with the bitwise complement of the
    canary; returns its offset from the allocation start."""
    if side == "hi":
        assert region.guard_hi > 0
        off = region.guard_lo + region.payload_bytes + int(rng.integers(0, region.guard_hi))
    else:
        assert region.guard_lo > 0
        off = int(rng.integers(0, region.guard_lo))
    bad = region.canary ^ 0xFF
    arena[region.offset + off] = bad
    return off


def perturb_fp32_single(cand, wl: Workload, seed: int = 101):
    """37 perturbations of the fp32 region: 20 inside the tolerance, 15
    outside it, one NaN, one +Inf; plus one corrupted high-guard byte.
    Returns the ground truth (positions and expected counts)."""
    torch = _torch()
    r = wl.regions[0]
    tol = wl.tol["f32"]
    rng = np.random.default_rng(seed)
    pos = _positions(rng, r.n_elems, 37)
    rng.shuffle(pos)
    inside, outside, nan_pos, inf_pos = pos[:20], pos[20:35], pos[35], pos[36]
    view, tdt = _elem_view(cand, r)
    vals = view.cpu().view(torch.float32).numpy().astype(np.float64)
    new = vals.copy()
    for p in inside:
        bound = tol.atol + tol.rtol * abs(vals[p])
        s = 1.0 if rng.random() < 0.5 else -1.0
        new[p] = vals[p] + s * 0.5 * bound * rng.uniform(0.1, 1.0)
    for p in outside:
        bound = tol.atol + tol.rtol * abs(vals[p])
        s = 1.0 if rng.random() < 0.5 else -1.0
        new[p] = vals[p] + s * (2.0 * bound + abs(vals[p]) * 2.0 ** -10 + 1e-3 * rng.uniform(0.1, 1.0))
    new32 = new.astype(np.float32)
    new32[nan_pos] = np.float32("nan")
    new32[inf_pos] = np.float32("inf")
    idx = np.concatenate([inside, outside, [nan_pos, inf_pos]])
    host = view.cpu().clone()
    host_f = host.view(torch.float32)
    host_f[torch.from_numpy(idx)] = torch.from_numpy(new32[idx])
    view.copy_(host.to(view.device))
    goff = corrupt_guard(cand, r, rng, "hi")
    bad_idx = np.concatenate([outside, [nan_pos, inf_pos]])
    return {"mismatches": 17, "nonfinite_mismatches": 2,
            "first_mismatch": int(bad_idx.min()), "guard_bad_bytes": 1,
            "first_guard_bad": goff, "inside": inside, "outside": outside,
            "nan": int(nan_pos), "inf": int(inf_pos)}


def perturb_ulp_noise(cand, region: Region, seed: int, rate_small=1e-3, ulp_small=1,
                      rate_large=1e-7, ulp_large=64):
    """Per element: with probability rate_small move +-ulp_small ULPs, else
    with probability rate_large move +-ulp_large ULPs (independent draws)."""
    torch = _torch()
    view, tdt = _elem_view(cand, region)
    g = torch.Generator(device=view.device)
    g.manual_seed(seed)
    n = region.n_elems
    chunk = 1 << 26
    for a in range(0, n, chunk):
        b = min(n, a + chunk)
        u1 = torch.rand(b - a, generator=g, device=view.device)
        u2 = torch.rand(b - a, generator=g, device=view.device)
        sgn = torch.randint(0, 2, (b - a,), generator=g, device=view.device) * 2 - 1
        steps = torch.where(u1 < rate_small, sgn * ulp_small,
                            torch.where(u2 < rate_large, sgn * ulp_large, 0))
        seg = _bits_of(view[a:b], region.dtype)
        new = torch.where(steps != 0, ulp_step(seg, steps, region.dtype), seg)
        view[a:b] = _to_storage(new, tdt, region.dtype)


def perturb_uniform_ulps(cand, region: Region, seed: int, magnitude: int):
    """Every element moves by a uniform integer in [-m, m] ULPs."""
    torch = _torch()
    if magnitude == 0:
        return
    view, tdt = _elem_view(cand, region)
    g = torch.Generator(device=view.device)
    g.manual_seed(seed)
    n = region.n_elems
    chunk = 1 << 27
    for a in range(0, n, chunk):
        b = min(n, a + chunk)
        seg = _bits_of(view[a:b], region.dtype)
        steps = torch.randint(-magnitude, magnitude + 1, (b - a,), generator=g,
                              device=view.device)
        view[a:b] = _to_storage(ulp_step(seg, steps, region.dtype), tdt, region.dtype)


def flip_bit(cand, region: Region, rng):
    """Flip one seeded bit of one seeded element; returns (index, bit)."""
    torch = _torch()
    view, tdt = _elem_view(cand, region)
    i = int(rng.integers(0, region.n_elems))
    bit = int(rng.integers(0, _BITS[region.dtype]))
    one = _bits_of(view[i:i + 1], region.dtype)
    view[i:i + 1] = _to_storage(one ^ (1 << bit), tdt, region.dtype)
    return i, bit


def perturb_sparse(cand, region: Region, rng, rate: float, max_ulps: int = 64):
    """Perturbations at `rate` per element: floats move 1..max_ulps ULPs
    (random sign), integers get one flipped bit.  Returns the positions."""
    torch = _torch()
    k = int(rng.binomial(region.n_elems, rate))
    if k == 0:
        return np.zeros(0, np.int64)
    pos = _positions(rng, region.n_elems, k)
    view, tdt = _elem_view(cand, region)
    idx = torch.from_numpy(pos).to(view.device)
    sel = _bits_of(view[idx], region.dtype)
    if region.dtype in FLOAT_DTYPES:
        mag = rng.integers(1, max_ulps + 1, k) * rng.choice([-1, 1], k)
        new = ulp_step(sel, torch.from_numpy(mag).to(view.device), region.dtype)
    else:
        b = rng.integers(0, _BITS[region.dtype], k)
        new = sel ^ (torch.ones_like(sel) << torch.from_numpy(b).to(view.device))
    view[idx] = _to_storage(new, tdt, region.dtype)
    return pos
