"""Splitting one comparison across processes, and merging its statistics.

The per-region statistics of the equivalence check (AsmEvo Eq. 1, per
element) are monoids: counts add, first indices take the minimum, and the
two maxima are maxima of non-negative doubles, whose IEEE bit patterns
order like integers.  A comparison can therefore be split into element
ranges on different GPUs (one process each) and merged exactly, whatever
the split.  This module does the host side of that: slice regions by rank,
shift indices back to region coordinates, and all-reduce the statistics
with torch.distributed (any backend; the tests use gloo on CPU).

The exact sums behind Eq. 1's cosine split the same way: every process
returns its sums as unrounded digit vectors (asmv_compare_eq_digits), the
vectors are added over the processes, and the verdict is formed once from
the total (asmv_eq_from_digits), so the cosine is that of the whole region.

Guard bands belong to whole allocations: the slice that starts the
payload keeps the low band, the slice that ends it keeps the high band,
and every other slice carries none, so each guard byte is checked once.
"""
from __future__ import annotations

import struct
from typing import Dict, List, Sequence, Tuple

STATS_FIELDS = ("mismatches", "first_mismatch", "max_abs_err", "max_rel_err",
                "nonfinite_mismatches", "guard_bad_bytes", "first_guard_bad",
                "ref_guard_bad_bytes")
U64_NONE = (1 << 64) - 1
_CHUNK = 16                      # slices start on 16-byte boundaries of the payload


def _bits(x: float) -> int:
    return struct.unpack("<q", struct.pack("<d", float(x)))[0]


def _double(b: int) -> float:
    return struct.unpack("<d", struct.pack("<q", int(b)))[0]


def empty_stats() -> Dict:
    return {"mismatches": 0, "first_mismatch": U64_NONE, "max_abs_err": 0.0,
            "max_rel_err": 0.0, "nonfinite_mismatches": 0, "guard_bad_bytes": 0,
            "first_guard_bad": U64_NONE, "ref_guard_bad_bytes": 0}


def merge_stats(a: Dict, b: Dict) -> Dict:
    """The exact merge of two partial results of one region."""
    return {
        "mismatches": a["mismatches"] + b["mismatches"],
        "first_mismatch": min(a["first_mismatch"], b["first_mismatch"]),
        "max_abs_err": _double(max(_bits(a["max_abs_err"]), _bits(b["max_abs_err"]))),
        "max_rel_err": _double(max(_bits(a["max_rel_err"]), _bits(b["max_rel_err"]))),
        "nonfinite_mismatches": a["nonfinite_mismatches"] + b["nonfinite_mismatches"],
        "guard_bad_bytes": a["guard_bad_bytes"] + b["guard_bad_bytes"],
        "first_guard_bad": min(a["first_guard_bad"], b["first_guard_bad"]),
        "ref_guard_bad_bytes": a["ref_guard_bad_bytes"] + b["ref_guard_bad_bytes"],
    }


def slice_bounds(n_elems: int, elem_size: int, rank: int, world: int) -> Tuple[int, int]:
    """Element range [a, b) of `rank` among `world`: contiguous, cut at
    16-byte boundaries of the payload so every slice keeps the payload's
    alignment."""
    chunk_elems = max(1, _CHUNK // elem_size)
    chunks = (n_elems + chunk_elems - 1) // chunk_elems
    a = min(n_elems, chunks * rank // world * chunk_elems)
    b = min(n_elems, chunks * (rank + 1) // world * chunk_elems)
    return a, b


def shard_region(region, elem_size: int, rank: int, world: int):
    """The slice of a region (an object with alloc, n_elems, guard_lo and
    guard_hi attributes; copied) that `rank` checks, the region index of
    its first element and the offset of its start from the region's
    allocation start.  The first slice keeps the low guard band, the last
    slice the high one."""
    import copy
    a, b = slice_bounds(region.n_elems, elem_size, rank, world)
    s = copy.copy(region)
    shift = 0
    if a > 0:
        shift = region.guard_lo + a * elem_size
        s.alloc = region.alloc + shift
        s.guard_lo = 0
    if b < region.n_elems:
        s.guard_hi = 0
    s.n_elems = b - a
    return s, a, shift


def to_region_coordinates(stats: Dict, first_index: int, alloc_shift: int) -> Dict:
    """Shift a slice's first mismatch and first bad guard byte back to the
    region's element index and allocation offset."""
    out = dict(stats)
    if out["first_mismatch"] != U64_NONE:
        out["first_mismatch"] += first_index
    if out["first_guard_bad"] != U64_NONE:
        out["first_guard_bad"] += alloc_shift
    return out


def allreduce_stats(per_region: Sequence[Dict], group=None) -> List[Dict]:
    """Merge every rank's partial statistics of the same regions (one dict
    per region, in the same order on every rank)."""
    import torch
    import torch.distributed as dist
    n = len(per_region)
    sums = torch.zeros((n, 4), dtype=torch.int64)
    mins = torch.zeros((n, 2), dtype=torch.int64)
    maxs = torch.zeros((n, 2), dtype=torch.int64)
    for i, s in enumerate(per_region):
        sums[i] = torch.tensor([s["mismatches"], s["nonfinite_mismatches"],
                                s["guard_bad_bytes"], s["ref_guard_bad_bytes"]])
        # UINT64_MAX ("none") as int64 max, so that MIN over ranks keeps real indices
        mins[i] = torch.tensor([min(s["first_mismatch"], (1 << 63) - 1),
                                min(s["first_guard_bad"], (1 << 63) - 1)])
        maxs[i] = torch.tensor([_bits(s["max_abs_err"]), _bits(s["max_rel_err"])])
    dist.all_reduce(sums, op=dist.ReduceOp.SUM, group=group)
    dist.all_reduce(mins, op=dist.ReduceOp.MIN, group=group)
    dist.all_reduce(maxs, op=dist.ReduceOp.MAX, group=group)
    out = []
    for i in range(n):
        f, g = int(mins[i, 0]), int(mins[i, 1])
        out.append({
            "mismatches": int(sums[i, 0]),
            "first_mismatch": U64_NONE if f == (1 << 63) - 1 else f,
            "max_abs_err": _double(int(maxs[i, 0])),
            "max_rel_err": _double(int(maxs[i, 1])),
            "nonfinite_mismatches": int(sums[i, 1]),
            "guard_bad_bytes": int(sums[i, 2]),
            "first_guard_bad": U64_NONE if g == (1 << 63) - 1 else g,
            "ref_guard_bad_bytes": int(sums[i, 3]),
        })
    return out


def normalize_digits(digits, ndigits: int = None):
    """Carry every digit vector along its last axis (ndigits digits, by
    default the length of that axis) so that each digit but the top one lies
    in [0, 2^32) (the integer it represents is unchanged): a sum over many
    processes then keeps every digit far inside int64."""
    import numpy as np
    d = np.asarray(digits, dtype=np.int64)
    ndigits = d.shape[-1] if ndigits is None else ndigits
    flat = d.reshape(-1, ndigits)
    out = np.zeros_like(flat)
    for r in range(flat.shape[0]):
        v = sum(int(flat[r, k]) << (32 * k) for k in range(ndigits))
        for k in range(ndigits - 1):
            out[r, k] = (v >> (32 * k)) & 0xFFFFFFFF
        out[r, ndigits - 1] = v >> (32 * (ndigits - 1))
    return out.reshape(d.shape)


def allreduce_digits(digits, group=None):
    """Sum the Eq. 1 digit vectors of every rank (numpy int64, the same
    shape on every rank), after normalising them: the exact sums of the
    whole split check."""
    import numpy as np
    import torch
    import torch.distributed as dist
    t = torch.from_numpy(np.ascontiguousarray(normalize_digits(digits)))
    dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return t.numpy()
