"""GPU parity at the full sizes of the five workloads, in the launch
configuration the bench uses (one context, persistent grid, K <= 8
candidates per launch).

- Fills: every byte for the workloads that fit comfortably on the host
  (1 Mi fp32, attention outputs, integer buffers); sampled element ranges
  computed one by one by the oracle for the 8 GiB snapshot and the 16 GiB
  input fill.
- Comparisons: all statistics of every region against the oracle on the
  same bytes.  The reference arena comes from the oracle's fill on the
  host and the candidates from the seeded input generator; neither is
  produced by the kernels under test.
"""
import numpy as np
import pytest

from paper_2608_20711_gb300 import asmv
from paper_2608_20711_gb300 import workloads as W

from ._gpu import (ORACLE_DIST, ORACLE_DTYPE, assert_stats_equal, oracle_fill_arena,
                   oracle_region_stats, to_device, to_host, torch_cuda)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    torch_cuda()
    c = asmv.Context(0)
    yield c
    c.close()


def _threads(oracle):
    return oracle.host_threads()


def _gpu_fill(ctx, wl, regions=None, arena_bytes=None):
    torch = torch_cuda()
    regions = regions or wl.regions
    dev = torch.zeros(arena_bytes or wl.arena_bytes, dtype=torch.uint8, device="cuda")
    ctx.fill(asmv.regions_in_arena(regions, dev.data_ptr()), seed=wl.seed)
    torch.cuda.synchronize()
    return dev


def _check_compare(ctx, oracle, wl, ref_host, cand_host, regions=None):
    regions = regions or wl.regions
    dref, dcand = to_device(ref_host), to_device(cand_host)
    got = ctx.compare(asmv.regions_in_arena(regions, dref.data_ptr()),
                      asmv.regions_in_arena(regions, dcand.data_ptr()), wl.tol)
    th = _threads(oracle)
    out = []
    for r, g in zip(regions, got):
        want = oracle_region_stats(oracle, ref_host, r, cand_host, r, wl.tol, threads=th)
        assert_stats_equal(g, want, r.name)
        out.append(want)
    return out


def _sampled_fill_check(oracle, wl, regions, dev, seed, samples=6, span=4099):
    """Oracle values for a few element ranges of every region (first,
    last and random), byte for byte against the device."""
    rng = np.random.default_rng(seed)
    for r in regions:
        sz = W.DTYPE_SIZE[r.dtype]
        starts = {0, max(0, r.n_elems - span)}
        for _ in range(samples):
            starts.add(int(rng.integers(0, max(1, r.n_elems - span))))
        for a in sorted(starts):
            b = min(r.n_elems, a + span)
            got = dev[r.payload_offset + a * sz:r.payload_offset + b * sz].cpu().numpy()
            want = np.zeros(b * sz, np.uint8)
            oracle.fill_payload(want, ORACLE_DTYPE[r.dtype], ORACLE_DIST[r.dist], a, b,
                                r.region_id, r.p0, r.p1, seed)
            np.testing.assert_array_equal(got, want[a * sz:], err_msg="%s [%d, %d)" % (r.name, a, b))
        # guard bands
        lo = dev[r.offset:r.offset + r.guard_lo].cpu().numpy()
        hi = dev[r.payload_offset + r.payload_bytes:r.offset + r.alloc_bytes].cpu().numpy()
        assert (lo == r.canary).all() and (hi == r.canary).all(), r.name


def test_fp32_single_full(ctx, oracle):
    torch = torch_cuda()
    wl = W.fp32_single()
    dev = _gpu_fill(ctx, wl)
    ref = oracle_fill_arena(oracle, wl.regions, wl.arena_bytes, wl.seed)
    np.testing.assert_array_equal(to_host(dev), ref)
    cand_t = torch.from_numpy(ref.copy())
    truth = W.perturb_fp32_single(cand_t, wl)
    s = _check_compare(ctx, oracle, wl, ref, cand_t.numpy())[0]
    assert (s["mismatches"], s["nonfinite_mismatches"], s["guard_bad_bytes"]) == (17, 2, 1)
    assert s["first_mismatch"] == truth["first_mismatch"]
    assert s["first_guard_bad"] == truth["first_guard_bad"]


def test_attention_bf16_full(ctx, oracle):
    torch = torch_cuda()
    wl = W.attention_bf16()
    dev = _gpu_fill(ctx, wl)
    ref = oracle_fill_arena(oracle, wl.regions, wl.arena_bytes, wl.seed)
    got = to_host(dev)
    assert np.array_equal(got, ref), "attention fill differs from the oracle"
    del got
    cand_t = torch.from_numpy(ref.copy())
    for r in wl.regions:
        W.perturb_ulp_noise(cand_t, r, seed=wl.seed * 10 + r.region_id)
    stats = _check_compare(ctx, oracle, wl, ref, cand_t.numpy())
    # +-1 bf16 ULP is inside rtol 1.6e-2; the +-64 ULP moves decide the count
    assert stats[0]["mismatches"] < 100 and stats[0]["max_abs_err"] > 0


def test_int_exact_full(ctx, oracle):
    torch = torch_cuda()
    wl = W.int_exact()
    dev = _gpu_fill(ctx, wl)
    ref = oracle_fill_arena(oracle, wl.regions, wl.arena_bytes, wl.seed)
    np.testing.assert_array_equal(to_host(dev), ref)
    cand_t = torch.from_numpy(ref.copy())
    rng = np.random.default_rng(wl.seed)
    flips = [W.flip_bit(cand_t, r, rng) for r in wl.regions]
    stats = _check_compare(ctx, oracle, wl, ref, cand_t.numpy())
    for s, (i, bit) in zip(stats, flips):
        assert (s["mismatches"], s["first_mismatch"], s["max_abs_err"]) == (1, i, 2.0 ** bit)


def test_snapshot_4096_full(ctx, oracle):
    torch = torch_cuda()
    wl = W.snapshot()
    assert len(wl.regions) == 4096
    assert abs(wl.payload_bytes / (8 << 30) - 1.0) < 0.02
    dev = _gpu_fill(ctx, wl)
    _sampled_fill_check(oracle, wl, wl.regions[::7], dev, wl.seed, samples=2, span=1031)
    # the comparison over all 4096 regions, on the oracle's own reference
    ref = oracle_fill_arena(oracle, wl.regions, wl.arena_bytes, wl.seed)
    cand_t = torch.from_numpy(ref.copy())
    rng = np.random.default_rng(44)
    for r in wl.regions:
        W.perturb_sparse(cand_t, r, rng, rate=1e-6)
    bad = rng.choice(len(wl.regions), 3, replace=False)
    for k in bad:
        W.corrupt_guard(cand_t, wl.regions[int(k)], rng, "hi")
    stats = _check_compare(ctx, oracle, wl, ref, cand_t.numpy())
    assert sum(s["guard_bad_bytes"] for s in stats) == 3
    assert sum(s["mismatches"] for s in stats) > 0


def test_batched_gemm_fp16_full(ctx, oracle):
    """The bench's step at full size: the 16 GiB guarded input fill
    (sampled), then the fp16 [32768, 32768] reference against 8 candidates
    in one batched launch group, every statistic against the oracle."""
    torch = torch_cuda()
    wl = W.batched_gemm()
    ins = _gpu_fill(ctx, wl, wl.input_regions, wl.input_arena_bytes)
    _sampled_fill_check(oracle, wl, wl.input_regions, ins, wl.seed, samples=3, span=2053)
    del ins
    torch.cuda.empty_cache()
    r = wl.regions[0]
    ref = oracle_fill_arena(oracle, wl.regions, wl.arena_bytes, wl.seed)
    dref = to_device(ref)
    cands = []
    for j in range(wl.n_cands):
        c = dref.clone()
        W.perturb_uniform_ulps(c, r, seed=wl.seed * 100 + j, magnitude=wl.ulp_magnitudes[j])
        cands.append(c)
    torch.cuda.synchronize()
    got = ctx.compare_batched(asmv.regions_in_arena(wl.regions, dref.data_ptr()),
                              [asmv.regions_in_arena(wl.regions, c.data_ptr()) for c in cands],
                              wl.tol)
    th = _threads(oracle)
    for j, c in enumerate(cands):
        ch = c.cpu().numpy()
        want = oracle_region_stats(oracle, ref, r, ch, r, wl.tol, threads=th)
        assert_stats_equal(got[j][0], want, "candidate %d" % j)
        if wl.ulp_magnitudes[j] == 0:
            assert want["mismatches"] == 0 and want["max_abs_err"] == 0.0
        del ch


def test_region_beyond_2_pow_32_elements(ctx, oracle):
    """One fp16 NORMAL region of 2^32 + 1029 elements (8 GiB): element
    indices and byte offsets past 2^32.  The GPU fill matches the oracle
    on sampled ranges including the tail; a compare whose reference is the
    oracle's own fill and whose candidate carries mismatches on both sides
    of element 2^32 gives the oracle's statistics (count, first index,
    exact maxima, guard damage past byte 2^33)."""
    n = (1 << 32) + 1029
    r = W.Region("big", "f16", n, "normal", 0.0, 1.0, 512, 4096, 0x5A, 3)
    r.offset = 0
    size = r.alloc_bytes + 64
    seed = 31
    torch = torch_cuda()
    dev = torch.zeros(size, dtype=torch.uint8, device="cuda")
    ctx.fill(asmv.regions_in_arena([r], dev.data_ptr()), seed=seed)
    torch.cuda.synchronize()
    _sampled_fill_check(oracle, None, [r], dev, seed, samples=4)
    del dev
    torch.cuda.empty_cache()
    ref = oracle_fill_arena(oracle, [r], size, seed)
    cand = ref.copy()
    pay = cand[r.payload_offset:r.payload_offset + r.payload_bytes].view(np.uint16)
    pos = np.array([5, 1 << 31, (1 << 32) - 1, 1 << 32, (1 << 32) + 7, n - 1], np.int64)
    pay[pos] ^= np.array([1, 0x40, 2, 0x300, 1, 0x7C00], np.uint16)
    cand[r.payload_offset + r.payload_bytes + 4000] ^= 0xFF          # high guard, past 2^33 bytes
    import types
    _check_compare(ctx, oracle, types.SimpleNamespace(tol=W.DEFAULT_TOL), ref, cand, regions=[r])


def test_philox_block_numbers_past_2_pow_32(ctx, oracle):
    """One int8 INT_RANGE region of 2^34 + 4099 elements (16 GiB): its
    chunks take four Philox blocks each, so the blocks of elements from 2^34
    on have a high counter word of 1.  Ranges on both sides of that element
    and the tail match the oracle byte for byte."""
    n = (1 << 34) + 4099
    r = W.Region("wide", "i8", n, "int_range", -100, 27, 256, 256, 0xC3, 9)
    r.offset = 0
    seed = 77
    torch = torch_cuda()
    dev = torch.zeros(r.alloc_bytes + 64, dtype=torch.uint8, device="cuda")
    ctx.fill(asmv.regions_in_arena([r], dev.data_ptr()), seed=seed)
    torch.cuda.synchronize()
    for a, b in (((1 << 34) - 4096, (1 << 34) + 4096), ((1 << 33) - 777, (1 << 33) + 333), (n - 5000, n)):
        got = dev[r.payload_offset + a:r.payload_offset + b].cpu().numpy()
        want = np.zeros(b, np.uint8)
        oracle.fill_payload(want, ORACLE_DTYPE[r.dtype], ORACLE_DIST[r.dist], a, b, r.region_id, r.p0, r.p1,
                            seed)
        np.testing.assert_array_equal(got, want[a:], err_msg="[%d, %d)" % (a, b))
    hi = dev[r.payload_offset + r.payload_bytes:r.offset + r.alloc_bytes].cpu().numpy()
    assert (hi == r.canary).all()
    del dev
    torch.cuda.empty_cache()
