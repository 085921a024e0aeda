"""GPU parity of the Tier 2 replay calls: restore (captured payload back
into each region, canary over its guard bands) and capture (region payload
out to a buffer), byte for byte against the oracle, over ragged sizes,
unaligned sources and destinations, guard bands longer than one segment and
empty regions; rejection of overlapping or host tables; device memory at a
chosen virtual address, and a capture -> modify -> restore replay there."""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from ._gpu import to_device, to_host, torch_cuda

pytestmark = pytest.mark.gpu

TILE = 16 * 1024


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _table(seed, count=24, skew=True):
    """Regions laid out in one arena (some payloads unaligned) and a
    matching snapshot buffer layout (some sources unaligned)."""
    rng = np.random.default_rng(seed)
    sizes = [0, 1, 15, 16, 17, 4099, TILE - 1, TILE, TILE + 3, 3 * TILE + 77, 300 * 1024 + 5]
    dts = ["f32", "bf16", "f16", "f8e4m3", "i32", "i8", "u8"]
    regs, srcs = [], []
    off = soff = 0
    for i in range(count):
        dt = dts[int(rng.integers(0, len(dts)))]
        sz = W.DTYPE_SIZE[dt]
        n = int(rng.choice(sizes)) // sz
        glo, ghi = [int(x) for x in rng.choice([0, 5, 256, 4096, 5000], 2)]
        r = W.Region("r%d" % i, dt, n, "raw", 0, 0, glo, ghi, int(rng.integers(0, 256)), i)
        off = (off + 255) // 256 * 256 + (int(rng.integers(0, 16)) if skew else 0)
        r.offset = off
        off += r.alloc_bytes
        regs.append(r)
        soff = (soff + 15) // 16 * 16 + (int(rng.integers(0, 16)) if skew and i % 3 == 0 else 0)
        srcs.append(soff)
        soff += r.payload_bytes
    return regs, off + 64, srcs, soff + 64


def test_restore_matches_oracle(ctx, oracle):
    regs, nbytes, srcs, sbytes = _table(1)
    rng = np.random.default_rng(2)
    arena_h = rng.integers(0, 256, nbytes, dtype=np.uint8)        # poisoned memory
    snap_h = rng.integers(0, 256, sbytes, dtype=np.uint8)         # captured pre-state
    arena, snap = to_device(arena_h), to_device(snap_h)
    ctx.restore(asmv.regions_in_arena(regs, arena.data_ptr()),
                [snap.data_ptr() + s for s in srcs])
    got = to_host(arena)
    want = arena_h.copy()
    for r, s in zip(regs, srcs):
        oracle.restore_region(want[r.offset:r.offset + r.alloc_bytes], r.payload_bytes,
                              r.guard_lo, r.guard_hi, r.canary, snap_h[s:s + r.payload_bytes])
    np.testing.assert_array_equal(got, want)


def test_capture_matches_payloads(ctx):
    regs, nbytes, srcs, sbytes = _table(3)
    rng = np.random.default_rng(4)
    arena_h = rng.integers(0, 256, nbytes, dtype=np.uint8)
    buf_h = rng.integers(0, 256, sbytes, dtype=np.uint8)
    arena, buf = to_device(arena_h), to_device(buf_h)
    ctx.capture(asmv.regions_in_arena(regs, arena.data_ptr()), [buf.data_ptr() + s for s in srcs])
    got = to_host(buf)
    want = buf_h.copy()
    for r, s in zip(regs, srcs):
        want[s:s + r.payload_bytes] = arena_h[r.payload_offset:r.payload_offset + r.payload_bytes]
    np.testing.assert_array_equal(got, want)
    np.testing.assert_array_equal(to_host(arena), arena_h)        # capture reads only


def test_capture_then_restore_round_trip(ctx):
    """Capture the pre-state, let a 'kernel' scribble over payloads and
    guards, restore: every byte is back."""
    torch = torch_cuda()
    regs, nbytes, srcs, sbytes = _table(5, skew=False)
    arena = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    dregs = asmv.regions_in_arena(regs, arena.data_ptr())
    for r in dregs:
        r.dist = asmv.DIST_RAW
    ctx.fill(dregs, seed=9)
    before = to_host(arena).copy()
    snap = torch.empty(sbytes, dtype=torch.uint8, device="cuda")
    ctx.capture(dregs, [snap.data_ptr() + s for s in srcs])
    arena.add_(3)                                            # the replayed kernel
    assert not np.array_equal(to_host(arena), before)
    ctx.restore(dregs, [snap.data_ptr() + s for s in srcs])
    after = to_host(arena)
    for r in regs:
        a, b = r.offset, r.offset + r.alloc_bytes
        np.testing.assert_array_equal(after[a:b], before[a:b], err_msg=r.name)


def test_rejections(ctx):
    torch = torch_cuda()
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    base = buf.data_ptr()
    a = asmv.make_region(base, 1000, "u8", guard_lo=16, guard_hi=16)
    b = asmv.make_region(base + 512, 100, "u8")
    src = base + 600 * 1024
    for regions, addrs in (([a, b], [src, src + 4096]),          # overlapping allocations
                           ([a], [base + 100]),                   # source inside the region
                           ([a], [0])):                           # null source
        with pytest.raises(asmv.AsmvError) as e:
            ctx.restore(regions, addrs)
        assert e.value.status == asmv.EINVAL
    host = np.zeros(4096, np.uint8)
    with pytest.raises(asmv.AsmvError):
        ctx.restore([a], [host.ctypes.data])
    with pytest.raises(asmv.AsmvError):                           # capture targets overlap
        ctx.capture([a, asmv.make_region(base + 8192, 1000, "u8")], [src, src + 10])
    ctx.restore([a], [src])                                       # the valid call passes
    ctx.restore([a, asmv.make_region(base + 8192, 1000, "u8")], [src, src + 10])   # sources may overlap


def test_fixed_virtual_address_replay(ctx, oracle):
    """Memory at a chosen address: map, note the address, unmap, map again
    at that address, restore a captured state there and check it."""
    torch = torch_cuda()
    g = asmv.va_granularity(0)
    assert g > 0 and g & (g - 1) == 0
    nbytes = 3 * g + 12345
    first = asmv.VaMapping(nbytes)
    addr = first.address
    assert addr % g == 0 and first.size == 4 * g
    first.unmap()
    with pytest.raises(asmv.AsmvError) as e:
        asmv.VaMapping(g, addr=addr + 1)                          # misaligned address
    assert e.value.status == asmv.EINVAL
    with asmv.VaMapping(nbytes, addr=addr) as m:
        assert m.address == addr
        with pytest.raises(asmv.AsmvError):                       # the range is now in use
            asmv.VaMapping(g, addr=addr)
        n = 777777
        reg = [asmv.make_region(addr + 64, n, "f16", "normal", 128, 256, 7, 0x5A, 0.0, 1.0)]
        rng = np.random.default_rng(8)
        snap_h = rng.integers(0, 256, 2 * n, dtype=np.uint8)
        snap = to_device(snap_h)
        ctx.restore(reg, [snap.data_ptr()])
        torch.cuda.synchronize()
        total = 128 + 2 * n + 256
        out = torch.empty(total, dtype=torch.uint8, device="cuda")
        ctx.capture([asmv.make_region(addr + 64, total, "u8")], [out.data_ptr()])   # the whole allocation
        want = np.zeros(total, np.uint8)
        oracle.restore_region(want, 2 * n, 128, 256, 0x5A, snap_h)
        np.testing.assert_array_equal(to_host(out), want)
        # the check of this memory against the captured state finds nothing
        stats = ctx.compare(reg, [asmv.make_region(addr + 64, n, "f16", "normal", 128, 256, 7, 0x5A)],
                            W.DEFAULT_TOL)
        assert stats[0]["mismatches"] == 0 and stats[0]["guard_bad_bytes"] == 0
        torch.cuda.synchronize()
