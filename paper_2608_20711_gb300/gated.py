"""GatedEval (AsmEvo Algorithm 1, Sec. 3.4) on top of the library's calls:
correctness strictly before timing, then the commit gate of Eq. 2.

For a candidate c against the original K0 over the evaluated inputs X:
  1. For each input x -- a Tier 1 dispatch (input regions and a seed) or a
     Tier 2 replay (captured regions and their pre-dispatch snapshots):
     - the inputs are prepared (Tier 1: filled from x's seed with asmv_fill;
       Tier 2: restored from the capture with asmv_restore, so kernels that
       update their inputs in place start from the same state every run),
       the reference output regions are overwritten with a poison pattern,
       and K0 runs once, giving O(x);
     - c runs `repeats` times (three in the paper, Sec. 5); before each run
       the inputs are prepared again and the candidate's output regions are
       poisoned with a fresh pattern, so that output c failed to write cannot
       match; each result is checked with Eq. 1 (asmv_compare_eq).  The first
       failing check ends the evaluation as "divergent".
  2. Timing on the first input (the representative launch): `warmup`
     untimed launches, then `reps` launches each timed with its own pair of
     CUDA events (asmv_time_launches), for K0 and for c; the latency T is the
     median; s(c) = T(K0) / T(c); cv is the larger of the two coefficients of
     variation.
  3. The commit gate of Eq. 2 against the current best speedup s_best.

Outcomes: "ok" (equivalent; `commit` says whether Eq. 2 accepts it, and
`reason` is "insufficient_speedup" when it does not), "divergent", and
"runtime_failure" (a launch callable raised).  The assembly and ABI gates
of Algorithm 1 concern rebuilding a binary and are outside this library.

Kernels are supplied as callables run(i, stream_handle) that enqueue the
kernel for input i on the given CUDA stream.  Everything on the device goes
through this library's kernels (fill, compare, Eq. 1 sums) and the
caller's own; this module only orders the calls.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable, List, Optional, Sequence

from . import asmv

POISON_TAG = 0x9E3779B97F4A7C15        # seeds of the poison fills differ from input seeds


@dataclass
class Dispatch:
    """One evaluated input x: regions to fill (asmv Region objects or dicts
    with device addresses) and the seed of the Tier 1 fill."""
    inputs: Sequence
    seed: int
    name: str = ""


@dataclass
class ReplayDispatch:
    """One evaluated input x captured from a real dispatch (Tier 2,
    Sec. 3.4): the referenced regions (asmv Region objects or dicts, at the
    addresses the kernel arguments point to) and, per region, the device
    address of its captured pre-dispatch payload.  Before every run the
    regions are restored from the capture (asmv_restore), guard bands
    included."""
    regions: Sequence
    snapshots: Sequence[int]
    name: str = ""


def _prepare(ctx, x, stream):
    if isinstance(x, ReplayDispatch):
        ctx.restore(x.regions, x.snapshots, stream=stream)
    else:
        ctx.fill(x.inputs, seed=x.seed, stream=stream)


@dataclass
class GateResult:
    outcome: str
    commit: bool = False
    reason: str = ""
    speedup: Optional[float] = None
    m_star: Optional[float] = None
    timing_original: Optional[dict] = None
    timing_candidate: Optional[dict] = None
    failed_at: Optional[dict] = None
    checks: List[dict] = field(default_factory=list)


def _poisoned(regions: Sequence, salt: int) -> List:
    """Copies of output regions whose fill writes random bytes over the
    payload and the canary over the guard bands."""
    arr = asmv.region_array(regions)
    return [asmv.make_region(arr[j].alloc, arr[j].n_elems, arr[j].dtype, asmv.DIST_RAW,
                             arr[j].guard_lo, arr[j].guard_hi,
                             (arr[j].region_id ^ salt) & 0xFFFFFFFF, arr[j].canary)
            for j in range(len(regions))]


def gated_eval(ctx: "asmv.Context", dispatches: Sequence[Dispatch],
               run_original: Callable[[int, int], None], run_candidate: Callable[[int, int], None],
               ref_out: Sequence, cand_out: Sequence, tol, *, theta: float = asmv.THETA,
               tau: float = asmv.TAU, repeats: int = 3, warmup: int = 3, reps: int = 20,
               s_best: float = 1.0, eps: float = asmv.GATE_EPS, k: float = asmv.GATE_K,
               s_floor: float = asmv.GATE_S_FLOOR, stream=None) -> GateResult:
    """Algorithm 1 for one candidate; see the module docstring."""
    import torch
    if not dispatches:
        raise ValueError("GatedEval needs at least one evaluated input")
    st = stream if stream is not None else torch.cuda.current_stream()
    handle = st.cuda_stream
    res = GateResult(outcome="ok")
    for i, x in enumerate(dispatches):
        salt = getattr(x, "seed", i)
        _prepare(ctx, x, st)
        ctx.fill(_poisoned(ref_out, 0x5EF), seed=salt ^ POISON_TAG, stream=st)
        try:
            run_original(i, handle)
        except Exception as e:           # the original must run; report, do not hide
            raise RuntimeError("the original kernel failed on input %d" % i) from e
        for rep in range(repeats):
            _prepare(ctx, x, st)
            ctx.fill(_poisoned(cand_out, 0xCA0 + rep), seed=salt ^ POISON_TAG ^ (rep + 1),
                     stream=st)
            try:
                run_candidate(i, handle)
            except Exception as e:
                res.outcome = "runtime_failure"
                res.failed_at = {"input": i, "repeat": rep, "error": repr(e)}
                return res
            stats, eqs = ctx.compare_eq(ref_out, [cand_out], tol, theta, tau, stream=st)
            res.checks.append({"input": i, "repeat": rep, "stats": stats[0], "eq": eqs[0]})
            bad = [j for j, e in enumerate(eqs[0]) if not e["eq"]]
            if bad:
                res.outcome = "divergent"
                res.failed_at = {"input": i, "repeat": rep, "region": bad[0],
                                 "flags": eqs[0][bad[0]]["flags"]}
                return res
    # timing on the representative launch (the first input), inputs in place
    _prepare(ctx, dispatches[0], st)
    t0 = asmv.time_launches(lambda h: run_original(0, h), reps, warmup, stream=st)
    t1 = asmv.time_launches(lambda h: run_candidate(0, h), reps, warmup, stream=st)
    res.timing_original = asmv.timing_summary(t0)
    res.timing_candidate = asmv.timing_summary(t1)
    res.speedup = res.timing_original["median_ms"] / res.timing_candidate["median_ms"]
    cv = max(res.timing_original["cv"], res.timing_candidate["cv"])
    res.m_star, res.commit = asmv.commit_gate(True, res.speedup, s_best, cv, eps, k, s_floor)
    if not res.commit:
        res.reason = "insufficient_speedup"
    return res
