"""GPU parity of the relative-error maximum where the screen decides it:
elements whose relative error ties with the running maximum (which the
screen does not send to the exact path), maxima that appear only late in a
region or in one lane, differences of tiny values near the bottom of the
fp32 range, and binary64 regions where every value differs (every element
takes the exact path, whose division is skipped when it cannot raise the
maximum).  Every statistic is compared with the oracle bit for bit."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from ._gpu import assert_stats_equal, oracle_region_stats, to_device, torch_cuda

pytestmark = pytest.mark.gpu

N = 3 * 8192 + 77                 # several compare tiles and a ragged tail


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _storage(values, dtype):
    import torch
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16,
           "f64": torch.float64}[dtype]
    return torch.from_numpy(np.asarray(values, np.float64)).to(tdt)


def _ulp_shift(t, k):
    """Each element moved k steps along its own bit pattern (same sign)."""
    import torch
    ib = {2: torch.int16, 4: torch.int32, 8: torch.int64}[t.element_size()]
    out = t.clone()
    out.view(ib).add_(k)
    return out


def _bytes(t):
    import torch
    ib = {2: torch.int16, 4: torch.int32, 8: torch.int64}[t.element_size()]
    return t.view(ib).numpy().view(np.uint8).copy()


def _check(ctx, oracle, dtype, ref_t, cands_t, tol):
    reg = W.Region("s", dtype, ref_t.numel(), "raw", 0, 0, 0, 0, 0xA5, 0)
    reg.offset = 0
    R = _bytes(ref_t)
    Cs = [_bytes(c) for c in cands_t]
    dref = to_device(R)
    dcs = [to_device(c) for c in Cs]
    n = ref_t.numel()
    got = ctx.compare_batched([asmv.make_region(dref.data_ptr(), n, dtype)],
                              [[asmv.make_region(d.data_ptr(), n, dtype)] for d in dcs], tol)
    for j, C in enumerate(Cs):
        want = oracle_region_stats(oracle, R, reg, C, reg, tol)
        assert_stats_equal(got[j][0], want, "%s cand %d" % (dtype, j))
    return got


@pytest.mark.parametrize("dtype", ["bf16", "f16", "f32"])
def test_ties_with_the_maximum_relative_error(ctx, oracle, dtype):
    """Powers of two moved by exactly k units in the last place: every
    element of a candidate has the same relative error, so after the first
    one every element ties with the running maximum."""
    rng = np.random.default_rng(3)
    e = rng.integers(-12, 12, N)
    ref = _storage(np.ldexp(rng.choice([-1.0, 1.0], N), e), dtype)
    cands = [_ulp_shift(ref, k) for k in (1, 2, 5)]
    tol = {dtype: (1e-6, 1e-3)}
    got = _check(ctx, oracle, dtype, ref, cands, tol)
    assert len({g[0]["max_rel_err"] for g in got}) == 3


@pytest.mark.parametrize("dtype", ["bf16", "f16", "f32"])
def test_maximum_found_late_and_in_one_lane(ctx, oracle, dtype):
    """Uniform small noise everywhere, a slightly larger relative error at
    a handful of scattered late positions, and one ties with it."""
    rng = np.random.default_rng(4)
    ref = _storage(rng.uniform(1.0, 2.0, N) * rng.choice([-1.0, 1.0], N), dtype)
    c = _ulp_shift(ref, 1)
    late = rng.choice(np.arange(N - 3000, N), 5, replace=False)
    import torch
    idx = torch.from_numpy(late)
    c[idx] = _ulp_shift(ref[idx], 3)
    c[N - 1] = _ulp_shift(ref[N - 1:N], 3)[0]
    _check(ctx, oracle, dtype, ref, [c, _ulp_shift(ref, 2)], {dtype: (0.0, 0.0)})


def test_tiny_values_near_the_bottom_of_fp32(ctx, oracle):
    """References of 2^-140 .. 2^-120 with differences of a few units of
    2^-149: the relative errors are large, distinct and close to each other."""
    rng = np.random.default_rng(5)
    ref = np.ldexp(rng.uniform(1.0, 2.0, N), rng.integers(-140, -120, N)).astype(np.float32)
    steps = rng.integers(-3, 4, N).astype(np.int32)
    cand = (ref.view(np.int32) + steps).view(np.float32)
    import torch
    _check(ctx, oracle, "f32", torch.from_numpy(ref), [torch.from_numpy(cand)],
           {"f32": (0.0, 0.5)})


@pytest.mark.parametrize("step", [1, 7])
def test_binary64_every_value_differs(ctx, oracle, step):
    """Binary64 with the last bit of every (or every 7th) value flipped:
    each differing element takes the exact path."""
    rng = np.random.default_rng(6)
    import torch
    ref = torch.from_numpy(rng.standard_normal(N) * np.ldexp(1.0, rng.integers(-30, 30, N)))
    cands = []
    for j in range(3):
        c = ref.clone()
        c.view(torch.int64)[j::step] ^= 1 + j
        cands.append(c)
    _check(ctx, oracle, "f64", ref, cands, {"f64": (1e-300, 1e-15)})
