"""The N > 1 host path on CPU: world_size-2 gloo ranks each check a slice
of every region (the oracle stands in for the GPU, which this host lacks)
and merge the statistics with torch.distributed; the merged result must
equal the unsplit result exactly."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

from paper_2608_20711_gb300 import distributed as D  # noqa: E402
from paper_2608_20711_gb300 import workloads as W  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _workload():
    from oracle import oracle as O
    regs = []
    for i, (dt, n) in enumerate([("f32", 100003), ("bf16", 7), ("f16", 65536), ("f8e4m3", 999),
                                 ("i32", 4097), ("i8", 1), ("u8", 123457), ("f64", 5001)]):
        dist_ = "normal" if dt in W.FLOAT_DTYPES else "raw"
        regs.append(W.Region("r%d" % i, dt, n, dist_, 0.0, 1.0, 64 + i, 128, 0xA5, i))
    size = W.layout(regs)
    ref = np.zeros(size, np.uint8)
    for r in regs:
        O.fill_region(ref[r.offset:r.offset + r.alloc_bytes], r.n_elems, O.CODE_OF_DTYPE[r.dtype],
                      O.CODE_OF_DIST[r.dist], r.guard_lo, r.guard_hi, r.region_id, r.canary,
                      r.p0, r.p1, 9)
    cand_t = torch.from_numpy(ref.copy())
    rng = np.random.default_rng(5)
    for r in regs:
        if r.dtype == "f64":              # low-bit flips at 1 % of the values
            v = cand_t[r.payload_offset:r.payload_offset + r.payload_bytes].numpy().view(np.uint64)
            v[rng.random(v.size) < 0.01] ^= np.uint64(3)
        else:
            W.perturb_sparse(cand_t, r, rng, rate=0.01)
        if r.guard_hi:
            W.corrupt_guard(cand_t, r, rng, "hi")
    W.corrupt_guard(cand_t, regs[2], rng, "lo")
    return regs, ref, cand_t.numpy()


TOL = {"f32": (1e-5, 1e-5), "bf16": (1e-2, 1.6e-2), "f16": (1e-5, 1e-3), "f8e4m3": (1e-5, 0.125),
       "f64": (1e-9, 1e-9)}


def _region_stats(O, ref, cand, r, shift_ref_alloc, s):
    """Oracle statistics of slice s of region r (allocation offsets in the arena)."""
    t = TOL.get(r.dtype, (0.0, 0.0))
    off = r.offset + shift_ref_alloc
    return O.compare_region(ref[off:], s.guard_lo, s.guard_hi, s.canary, cand[off:],
                            s.guard_lo, s.guard_hi, s.canary, s.n_elems,
                            O.CODE_OF_DTYPE[r.dtype], t[0], t[1])


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import oracle as O
        regs, ref, cand = _workload()
        partial = []
        for r in regs:
            r.alloc = 0                       # arena coordinates
            s, first, shift = D.shard_region(r, W.DTYPE_SIZE[r.dtype], rank, world)
            st = _region_stats(O, ref, cand, r, shift, s)
            partial.append(D.to_region_coordinates(st, first, shift))
        merged = D.allreduce_stats(partial)
        if rank == 0:
            out.put(merged)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_sharded_compare_merges_exactly(world):
    from oracle import oracle as O
    regs, ref, cand = _workload()
    whole = [_region_stats(O, ref, cand, r, 0, r) for r in regs]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(k, world, port, q)) for k in range(world)]
    for p in procs:
        p.start()
    merged = q.get(timeout=240)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r, w, m in zip(regs, whole, merged):
        for f in D.STATS_FIELDS:
            assert np.float64(m[f]).view(np.uint64) == np.float64(w[f]).view(np.uint64), (r.name, f)
    assert sum(w["mismatches"] for w in whole) > 0
    assert sum(w["guard_bad_bytes"] for w in whole) >= 2


def test_merge_is_order_independent():
    from oracle import oracle as O
    regs, ref, cand = _workload()
    r = regs[0]
    r.alloc = 0
    parts = []
    for k in range(5):
        s, first, shift = D.shard_region(r, 4, k, 5)
        parts.append(D.to_region_coordinates(_region_stats(O, ref, cand, r, shift, s), first, shift))
    a = D.empty_stats()
    for p in parts:
        a = D.merge_stats(a, p)
    b = D.empty_stats()
    for p in reversed(parts):
        b = D.merge_stats(p, b)
    assert a == b == _region_stats(O, ref, cand, r, 0, r)


def _eq_worker(rank, world, port, out):
    """Each rank: its element range of every float region, as unrounded Eq. 1
    digit vectors (built from the oracle's exact sums, in the library's
    layout) and statistics; both all-reduced."""
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import oracle as O
        from paper_2608_20711_gb300 import asmv
        from tests.test_eq_digits import full_stats, shard_digits
        regs, ref, cand = _workload()
        flt = [r for r in regs if r.dtype in W.FLOAT_DTYPES]
        nd = asmv.digits_per_slot([r.dtype for r in flt])
        digs, parts = [], []
        for r in flt:
            a, b = D.slice_bounds(r.n_elems, W.DTYPE_SIZE[r.dtype], rank, world)
            off = r.payload_offset
            rp, cp = ref[off:off + r.payload_bytes], cand[off:off + r.payload_bytes]
            digs.append(shard_digits(O, rp, [cp], r.dtype, a, b, nd=nd))
            t = TOL[r.dtype]
            parts.append(D.to_region_coordinates(full_stats(O, rp, cp, r.dtype, a, b, t), a, 0))
        merged_digits = D.allreduce_digits(np.stack(digs))
        merged_stats = D.allreduce_stats(parts)
        if rank == 0:
            out.put((merged_digits, merged_stats))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_sharded_eq1_verdict_is_exact(world):
    """Eq. 1 of regions split over gloo ranks, formed once from the summed
    digit vectors, equals the oracle's verdict on the whole regions."""
    from oracle import oracle as O
    from paper_2608_20711_gb300 import asmv
    from tests.test_eq_digits import ONAME, full_stats
    regs, ref, cand = _workload()
    flt = [r for r in regs if r.dtype in W.FLOAT_DTYPES]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_eq_worker, args=(k, world, port, q)) for k in range(world)]
    for p in procs:
        p.start()
    digits, stats = q.get(timeout=240)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    got = asmv.eq_from_digits([r.dtype for r in flt], [stats], digits)[0]
    for r, g in zip(flt, got):
        off = r.payload_offset
        rp, cp = ref[off:off + r.payload_bytes], cand[off:off + r.payload_bytes]
        code = getattr(O, ONAME[r.dtype])
        whole = full_stats(O, rp, cp, r.dtype, 0, r.n_elems, TOL[r.dtype])
        want = O.eq_verdict(whole, O.eq_sums(rp, cp, code, r.n_elems), code)
        for f in ("sum_rc", "sum_rr", "sum_cc", "cos", "flags", "eq"):
            assert g[f] == want[f], (r.name, f)
