"""The bounded waits of the compare pipeline.  With the producer's bound
set to 0 it stops issuing copies as soon as it needs a stage back; the
checking warps then wait for a tile that never comes until their own
(default) bound runs out, the kernel sets its error word, lets the copies
it issued land and returns, and the call reports ASMV_ETIMEOUT without
writing statistics.  The context stays usable: with the default bound
restored the same calls succeed and agree with the oracle.  Nothing here
faults or hangs the GPU: every wait is bounded and no copy outlives its
kernel."""
import ctypes

import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from ._gpu import assert_stats_equal, oracle_fill_arena, oracle_region_stats, to_device, torch_cuda

pytestmark = pytest.mark.gpu

TILE = 16 * 1024


def _arena():
    # region a alone spans 1024 tiles of 16 KiB, more than 4 per CTA of a
    # one-CTA-per-SM grid, so the producer of every CTA needs a stage back
    regs = [W.Region("a", "f32", 1024 * TILE // 4 + 5, "uniform", -1.0, 1.0, 64, 64, 0xA5, 1),
            W.Region("b", "f16", 5 * TILE // 2 + 3, "normal", 0.0, 1.0, 0, 256, 0x5A, 2),
            W.Region("c", "i32", 777, "int_range", 0, 1000, 16, 0, 0x11, 3)]
    off = 0
    for r in regs:
        off = (off + 255) // 256 * 256
        r.offset = off
        off += r.alloc_bytes
    return regs, off + 64


def test_wait_bound_zero_times_out_and_context_recovers(oracle):
    torch_cuda()
    regs, nbytes = _arena()
    ref = oracle_fill_arena(oracle, regs, nbytes, seed=3)
    cand = ref.copy()
    rng = np.random.default_rng(4)
    for r in regs:
        pos = r.payload_offset + rng.integers(0, r.payload_bytes, 20)
        cand[pos] ^= 0x40
    dref, dcand = to_device(ref), to_device(cand)
    rr = asmv.regions_in_arena(regs, dref.data_ptr())
    cc = asmv.regions_in_arena(regs, dcand.data_ptr())
    ctx = asmv.Context(0)
    try:
        ctx.set_wait_rounds(0)
        calls = (lambda: ctx.compare(rr, cc, W.DEFAULT_TOL),
                 lambda: ctx.compare_batched(rr, [cc, rr, cc], W.DEFAULT_TOL),
                 lambda: ctx.compare_eq(rr, [cc], W.DEFAULT_TOL))
        for call in calls:
            with pytest.raises(asmv.AsmvError) as e:
                call()
            assert e.value.status == asmv.ETIMEOUT
        # the raw call leaves out_host untouched
        L = asmv.lib()
        out = (asmv.Stats * len(regs))()
        ctypes.memset(out, 0x7B, ctypes.sizeof(out))
        before = bytes(out)
        rc = L.asmv_compare(ctx._h, asmv.region_array(rr), asmv.region_array(cc), len(regs),
                            asmv.tol_array(W.DEFAULT_TOL), out, None)
        assert rc == asmv.ETIMEOUT and bytes(out) == before
        # a table with no payload has no pipeline waits
        empty = [asmv.make_region(dref.data_ptr() + regs[0].offset, 0, "f32", guard_lo=64, guard_hi=64,
                                  canary=0xA5)]
        st = ctx.compare(empty, empty, W.DEFAULT_TOL)
        assert st[0]["mismatches"] == 0
        # back to the default bound: the same context checks correctly
        ctx.set_wait_rounds(None)
        got = ctx.compare(rr, cc, W.DEFAULT_TOL)
        for i, r in enumerate(regs):
            assert_stats_equal(got[i], oracle_region_stats(oracle, ref, r, cand, r, W.DEFAULT_TOL))
        stats, eqs = ctx.compare_eq(rr, [cc], W.DEFAULT_TOL)
        for i, r in enumerate(regs):
            assert_stats_equal(stats[0][i], got[i])
    finally:
        ctx.close()
