"""Helpers shared by the GPU parity tests: device arenas, host <-> device
copies and the oracle-side evaluation of the same regions."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import workloads as W

from oracle.oracle import CODE_OF_DIST as ORACLE_DIST
from oracle.oracle import CODE_OF_DTYPE as ORACLE_DTYPE


def torch_cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch


def device_arena(nbytes, fill_byte=0):
    torch = torch_cuda()
    t = torch.empty(max(nbytes, 1), dtype=torch.uint8, device="cuda")
    t.fill_(fill_byte)
    return t


def to_device(host_u8):
    torch = torch_cuda()
    return torch.from_numpy(np.ascontiguousarray(host_u8)).to("cuda")


def to_host(dev_u8):
    torch = torch_cuda()
    torch.cuda.synchronize()
    return dev_u8.cpu().numpy()


def oracle_fill_arena(oracle, regions, arena_bytes, seed, threads=None, base=None):
    """The oracle's guarded fill of every region into a host arena."""
    arena = np.zeros(arena_bytes, np.uint8) if base is None else base.copy()
    threads = threads or oracle.host_threads()
    for r in regions:
        oracle.fill_region(arena[r.offset:r.offset + r.alloc_bytes], r.n_elems,
                           ORACLE_DTYPE[r.dtype], ORACLE_DIST[r.dist], r.guard_lo, r.guard_hi,
                           r.region_id, r.canary, r.p0, r.p1, seed, threads=threads)
    return arena


def oracle_region_stats(oracle, ref_arena, ref_reg, cand_arena, cand_reg, tol, threads=1):
    t = tol.get(ref_reg.dtype, W.Tolerance(0.0, 0.0)) if isinstance(tol, dict) else tol
    if isinstance(t, tuple):
        t = W.Tolerance(*t)
    return oracle.compare_region(
        ref_arena[ref_reg.offset:], ref_reg.guard_lo, ref_reg.guard_hi, ref_reg.canary,
        cand_arena[cand_reg.offset:], cand_reg.guard_lo, cand_reg.guard_hi, cand_reg.canary,
        ref_reg.n_elems, ORACLE_DTYPE[ref_reg.dtype], t.atol, t.rtol, threads=threads)


def assert_stats_equal(got, want, where=""):
    """Field-by-field equality; doubles compared bit for bit."""
    for f, v in want.items():
        g = got[f]
        if isinstance(v, float):
            gb = np.float64(g).view(np.uint64)
            wb = np.float64(v).view(np.uint64)
            assert gb == wb, "%s %s: gpu %r != oracle %r" % (where, f, g, v)
        else:
            assert int(g) == int(v), "%s %s: gpu %r != oracle %r" % (where, f, g, v)
