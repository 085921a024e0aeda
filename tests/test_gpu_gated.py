"""GatedEval (Algorithm 1) end to end on the GPU with small torch kernels
as K0 and candidates: an equivalent rewrite, a wrong element, an
out-of-bounds write into a guard band, a candidate that differs only on a
repeated run, a candidate that does not write its output, one that raises,
and a genuinely faster rewrite that the commit gate of Eq. 2 accepts."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W
from paper_2608_20711_gb300.gated import Dispatch, gated_eval

from ._gpu import torch_cuda

pytestmark = pytest.mark.gpu

N = 1 << 20
GUARD = 256


@pytest.fixture(scope="module")
def env():
    torch = torch_cuda()
    ctx = asmv.Context(0)
    alloc = N * 2 + 2 * GUARD
    arena = torch.zeros(3 * alloc + 1024, dtype=torch.uint8, device="cuda")
    base = arena.data_ptr()
    offs = [0, alloc + 256 - (alloc % 256), 2 * (alloc + 256 - (alloc % 256))]

    def region(k, rid, dist="normal"):
        return asmv.make_region(base + offs[k], N, "f16", dist, GUARD, GUARD, rid, 0xA5, 0.0, 1.0)

    def view(k):
        return arena[offs[k] + GUARD:offs[k] + GUARD + 2 * N].view(torch.float16)

    e = {"torch": torch, "ctx": ctx, "arena": arena, "x": view(0), "y0": view(1), "y1": view(2),
         "inp": [region(0, 1)], "ref_out": [region(1, 2)], "cand_out": [region(2, 3)],
         "guard_hi_c": arena[offs[2] + GUARD + 2 * N:offs[2] + 2 * GUARD + 2 * N]}
    yield e
    ctx.close()


def _on(torch, handle):
    """Run torch ops on the stream GatedEval passes (0 is the default stream)."""
    if handle == 0:
        return torch.cuda.stream(torch.cuda.default_stream())
    return torch.cuda.stream(torch.cuda.ExternalStream(handle))


def _run(env, cand, **kw):
    torch = env["torch"]

    def original(i, h):
        with _on(torch, h):
            torch.mul(env["x"], 2, out=env["y0"])

    def candidate(i, h):
        with _on(torch, h):
            cand(env, i)
    xs = [Dispatch(env["inp"], seed=11), Dispatch(env["inp"], seed=12)]
    return gated_eval(env["ctx"], xs, original, candidate, env["ref_out"], env["cand_out"],
                      W.DEFAULT_TOL, reps=kw.pop("reps", 10), **kw)


def test_equivalent_rewrite_passes(env):
    torch = env["torch"]
    r = _run(env, lambda e, i: torch.add(e["x"], e["x"], out=e["y1"]))
    assert r.outcome == "ok" and len(r.checks) == 6
    assert all(c["eq"][0]["cos"] >= 0.9999 and c["eq"][0]["eq"] == 1 for c in r.checks)
    assert r.speedup > 0 and r.m_star >= 1.002
    assert r.commit == (r.speedup >= max(r.m_star, 1.0))


def test_wrong_value_is_divergent(env):
    torch = env["torch"]

    def cand(e, i):
        torch.mul(e["x"], 2, out=e["y1"])
        e["y1"][12345] += 1.0
    r = _run(env, cand)
    assert r.outcome == "divergent" and r.failed_at["repeat"] == 0
    assert r.failed_at["flags"] & asmv.EQ_LINF == 0


def test_out_of_bounds_write_is_divergent(env):
    torch = env["torch"]

    def cand(e, i):
        torch.mul(e["x"], 2, out=e["y1"])
        e["guard_hi_c"][3] = 0
    r = _run(env, cand)
    assert r.outcome == "divergent" and r.failed_at["flags"] == (asmv.EQ_COS | asmv.EQ_LINF |
                                                                 asmv.EQ_INT)


def test_difference_on_a_repeat_is_caught(env):
    torch = env["torch"]
    calls = {"n": 0}

    def cand(e, i):
        torch.mul(e["x"], 2, out=e["y1"])
        calls["n"] += 1
        if calls["n"] == 2:
            e["y1"][7] = float("nan")
    r = _run(env, cand)
    assert r.outcome == "divergent" and r.failed_at == {"input": 0, "repeat": 1, "region": 0,
                                                        "flags": r.failed_at["flags"]}


def test_missing_write_is_divergent(env):
    r = _run(env, lambda e, i: None)          # leaves the poison pattern in place
    assert r.outcome == "divergent"


def test_raising_candidate_is_a_runtime_failure(env):
    def cand(e, i):
        raise RuntimeError("launch failed")
    r = _run(env, cand)
    assert r.outcome == "runtime_failure" and "launch failed" in r.failed_at["error"]


def test_faster_rewrite_is_committed(env):
    """K0 here is a slow chain of 40 exact multiplications by one; the
    candidate computes the same bits in one kernel."""
    torch = env["torch"]

    def slow_original(i, h):
        with _on(torch, h):
            torch.mul(env["x"], 2, out=env["y0"])
            for _ in range(40):
                env["y0"].mul_(1)

    def fast(i, h):
        with _on(torch, h):
            torch.mul(env["x"], 2, out=env["y1"])
    xs = [Dispatch(env["inp"], seed=21)]
    r = gated_eval(env["ctx"], xs, slow_original, fast, env["ref_out"], env["cand_out"],
                   W.DEFAULT_TOL, reps=20)
    assert r.outcome == "ok" and r.speedup > 5.0 and r.commit and r.reason == ""
    # against a best that is already faster than this candidate, the gate refuses it
    r2 = gated_eval(env["ctx"], xs, slow_original, fast, env["ref_out"], env["cand_out"],
                    W.DEFAULT_TOL, reps=20, s_best=r.speedup * 2)
    assert r2.outcome == "ok" and not r2.commit and r2.reason == "insufficient_speedup"


def test_time_launches_counts_each_launch(env):
    torch = env["torch"]
    n = {"calls": 0}

    def fn(h):
        n["calls"] += 1
        with _on(torch, h):
            torch.mul(env["x"], 2, out=env["y1"])
    ms = asmv.time_launches(fn, 7, warmup=2)
    assert n["calls"] == 9 and len(ms) == 7 and all(m > 0 for m in ms)
    s = asmv.timing_summary(ms)
    assert s["r"] == 7 and s["median_ms"] == float(np.median(ms))


def test_replay_dispatch_restores_inputs(env):
    """Tier 2 replay: a kernel that updates its input in place (x += 1,
    y = 2x) is equivalent on every repeat only because the captured
    pre-state is restored before each run."""
    from paper_2608_20711_gb300.gated import ReplayDispatch
    torch = env["torch"]
    ctx = env["ctx"]
    ctx.fill(env["inp"], seed=31)
    snap = torch.empty(2 * N, dtype=torch.uint8, device="cuda")
    ctx.capture(env["inp"], [snap.data_ptr()])

    def original(i, h):
        with _on(torch, h):
            env["x"].add_(1)
            torch.mul(env["x"], 2, out=env["y0"])

    def candidate(i, h):
        with _on(torch, h):
            env["x"].add_(1)
            torch.add(env["x"], env["x"], out=env["y1"])
    x = ReplayDispatch(env["inp"], [snap.data_ptr()])
    r = gated_eval(ctx, [x], original, candidate, env["ref_out"], env["cand_out"],
                   W.DEFAULT_TOL, reps=5)
    assert r.outcome == "ok" and len(r.checks) == 3
    # without restoring, the second repeat would see x + 2 and diverge
    xs = [Dispatch(env["inp"], seed=31)]
    r2 = gated_eval(ctx, xs, original, candidate, env["ref_out"], env["cand_out"],
                    W.DEFAULT_TOL, reps=5)
    assert r2.outcome == "ok"                     # Tier 1 refills the input each run too
