"""Pins of the oracle's Philox4x32-10 (the counter-based generator behind
Tier 1 input synthesis) against two independent implementations run as
black boxes: triton's interpreter-mode `tl.philox` and PyTorch's header-only
engine.  Neither shares code with the oracle."""
import os
import subprocess

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


def _rand_u32(rng, shape):
    return rng.integers(0, 1 << 32, size=shape, dtype=np.uint64).astype(np.uint32)


def _triton_philox(ctr, key):
    """Run triton's Philox4x32 (10 rounds) on the CPU interpreter."""
    os.environ["TRITON_INTERPRET"] = "1"
    torch = pytest.importorskip("torch")
    triton = pytest.importorskip("triton")
    import triton.language as tl

    @triton.jit
    def kern(out_ptr, c_ptr, k_ptr, N: tl.constexpr):
        i = tl.arange(0, N)
        c0 = tl.load(c_ptr + 4 * i + 0)
        c1 = tl.load(c_ptr + 4 * i + 1)
        c2 = tl.load(c_ptr + 4 * i + 2)
        c3 = tl.load(c_ptr + 4 * i + 3)
        k0 = tl.load(k_ptr + 2 * i + 0).to(tl.uint64)
        k1 = tl.load(k_ptr + 2 * i + 1).to(tl.uint64)
        # triton's philox takes one 64-bit seed; its low/high halves are the key words
        a, b, c, d = tl.philox((k1 << 32) | k0, c0, c1, c2, c3, 10)
        tl.store(out_ptr + 4 * i + 0, a)
        tl.store(out_ptr + 4 * i + 1, b)
        tl.store(out_ptr + 4 * i + 2, c)
        tl.store(out_ptr + 4 * i + 3, d)

    n = ctr.shape[0]
    assert n & (n - 1) == 0
    c_t = torch.from_numpy(ctr.astype(np.uint32).view(np.int32).reshape(-1).copy())
    k_t = torch.from_numpy(key.astype(np.uint32).view(np.int32).reshape(-1).copy())
    c_t = c_t.view(torch.uint32)
    k_t = k_t.view(torch.uint32)
    out = torch.zeros(4 * n, dtype=torch.uint32)
    kern[(1,)](out, c_t, k_t, N=n)
    return out.view(torch.int32).numpy().view(np.uint32).reshape(n, 4)


def test_philox_matches_triton_interpreter(oracle):
    rng = np.random.default_rng(12345)
    n = 2048
    ctr = _rand_u32(rng, (n, 4))
    key = _rand_u32(rng, (n, 2))
    # structured counters too: small block indices, the layout the fill uses
    ctr[:64] = 0
    ctr[:64, 0] = np.arange(64)
    ctr[64:128, 2] = np.arange(64)
    key[:128] = 0
    got = oracle.philox(ctr, key)
    want = _triton_philox(ctr, key)
    np.testing.assert_array_equal(got, want)


def test_philox_matches_torch_engine(oracle, torch_philox):
    """The fill's counter layout (block lo, block hi, region_id, 0) under key
    (seed lo, seed hi) is torch's (offset, subsequence, seed) addressing."""
    rng = np.random.default_rng(777)
    n = 3000
    seeds = rng.integers(0, 1 << 63, size=n, dtype=np.uint64)
    regions = _rand_u32(rng, n).astype(np.uint64)
    blocks = rng.integers(0, 1 << 40, size=n, dtype=np.uint64)
    seeds[:8] = [0, 1, 2, 3, 4, 5, 1 << 32, (1 << 63) - 1]
    blocks[:8] = 0
    regions[:8] = 0
    lines = "\n".join("%d %d %d" % (s, r, b) for s, r, b in zip(seeds, regions, blocks))
    res = subprocess.run([torch_philox.exe], input=lines, capture_output=True, text=True,
                         check=True).stdout.split()
    want = np.array(res, dtype=np.uint64).astype(np.uint32).reshape(n, 4)
    ctr = np.stack([blocks & 0xFFFFFFFF, blocks >> 32, regions,
                    np.zeros(n, np.uint64)], axis=1).astype(np.uint32)
    key = np.stack([seeds & 0xFFFFFFFF, seeds >> 32], axis=1).astype(np.uint32)
    np.testing.assert_array_equal(oracle.philox(ctr, key), want)


def test_philox_counter_injective_sample(oracle):
    """Distinct counters under one key give distinct blocks (Philox is a
    bijection of the counter for a fixed key)."""
    n = 1 << 18
    ctr = np.zeros((n, 4), np.uint32)
    ctr[:, 0] = np.arange(n)
    key = np.tile(np.array([[0xDEADBEEF, 0x12345678]], np.uint32), (n, 1))
    out = oracle.philox(ctr, key)
    packed = out.view(np.dtype([("a", "<u4"), ("b", "<u4"), ("c", "<u4"), ("d", "<u4")]))
    assert np.unique(packed).size == n
    # every output word is roughly uniform: each byte value appears ~n*16/256 times
    counts = np.bincount(out.view(np.uint8).reshape(-1), minlength=256)
    expected = out.size * 4 / 256.0
    chi2 = ((counts - expected) ** 2 / expected).sum()
    assert chi2 < 400.0  # 255 dof; p ~ 1e-8 at 400
