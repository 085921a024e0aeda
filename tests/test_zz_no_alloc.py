"""asmv_compare_noalloc: the comparison for callers that must not allocate
device memory (for instance a harness that keeps its reserved address
space untouched between captured replays, or one that times candidates
and cannot take an allocation's synchronisation).  It has no context and
uses the library's fixed device scratch; its results must equal those of
asmv_compare on the same inputs, call after call.

Collected last (file name), so that a failure here does not hide other
results in a run that stops at the first failure."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

pytestmark = pytest.mark.gpu

TOL = {"f32": (1e-5, 1e-5), "bf16": (1e-2, 1.6e-2), "f16": (1e-5, 1e-3), "f8e4m3": (1e-5, 0.125)}


def _setup(seed):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    regs = []
    dts = ["f32", "bf16", "f16", "f8e4m3", "i32", "i8", "u8"]
    for i, dt in enumerate(dts * 2):
        n = [1, 1000, 40000, 70001][i % 4]
        dist = "normal" if dt in W.FLOAT_DTYPES else "raw"
        regs.append(W.Region("r%d" % i, dt, n, dist, 0.0, 1.0, 256 if i % 3 else 8, 4096, 0xA5, i))
    size = W.layout(regs) + 256
    ref = torch.zeros(size, dtype=torch.uint8, device="cuda")
    ctx = asmv.Context(0)
    rr = asmv.regions_in_arena(regs, ref.data_ptr())
    ctx.fill(rr, seed=seed)
    torch.cuda.synchronize()
    cand = ref.clone()
    rng = np.random.default_rng(seed)
    for r in regs:
        if r.dtype in W.FLOAT_DTYPES and r.n_elems > 10:
            W.perturb_uniform_ulps(cand, r, seed=seed * 7 + r.region_id, magnitude=3)
        else:
            W.perturb_sparse(cand, r, rng, rate=0.05)
    W.corrupt_guard(cand, regs[2], rng, "hi")
    torch.cuda.synchronize()
    cr = asmv.regions_in_arena(regs, cand.data_ptr())
    return ctx, rr, cr, (ref, cand)


def test_noalloc_matches_context_compare_twice():
    for seed in (3, 4):                       # two calls in a row, different inputs
        ctx, rr, cr, keep = _setup(seed)
        want = ctx.compare(rr, cr, TOL)
        got = asmv.compare_noalloc(rr, cr, TOL)
        again = asmv.compare_noalloc(rr, cr, TOL)
        for w, g, a in zip(want, got, again):
            for f in asmv.STATS_FIELDS:
                assert np.float64(g[f]).view(np.uint64) == np.float64(w[f]).view(np.uint64), f
                assert np.float64(a[f]).view(np.uint64) == np.float64(w[f]).view(np.uint64), f
        assert sum(w["mismatches"] for w in want) > 0
        ctx.close()


def test_noalloc_rejects_tables_beyond_its_scratch():
    ctx, rr, cr, keep = _setup(5)
    big_ref = [rr[0]] * 12000                 # 12000 regions need more than 1 MiB of plan
    big_cand = [cr[0]] * 12000
    with pytest.raises(asmv.AsmvError) as e:
        asmv.compare_noalloc(big_ref, big_cand, TOL)
    assert e.value.status == asmv.EINVAL
    ctx.close()
