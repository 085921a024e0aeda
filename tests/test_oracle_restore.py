"""Pins of the oracle's Tier 2 restore: the result is the captured payload
between two canary bands, built independently with numpy slicing."""
import numpy as np
import pytest


@pytest.mark.parametrize("glo,ghi,nb", [(0, 0, 0), (0, 0, 17), (5, 0, 100), (0, 4096, 1),
                                        (256, 256, 65536 + 3), (4097, 13, 999)])
def test_restore_is_guards_plus_capture(oracle, glo, ghi, nb):
    rng = np.random.default_rng(glo * 7 + ghi * 3 + nb)
    alloc = rng.integers(0, 256, glo + nb + ghi, dtype=np.uint8)
    captured = rng.integers(0, 256, nb, dtype=np.uint8)
    canary = int(rng.integers(0, 256))
    want = np.concatenate([np.full(glo, canary, np.uint8), captured,
                           np.full(ghi, canary, np.uint8)])
    oracle.restore_region(alloc, nb, glo, ghi, canary, captured)
    np.testing.assert_array_equal(alloc, want)


def test_restore_touches_nothing_outside(oracle):
    buf = np.full(1000, 0x77, np.uint8)
    oracle.restore_region(buf[100:100 + 64 + 32 + 64], 32, 64, 64, 0xA5, np.arange(32, dtype=np.uint8))
    assert (buf[:100] == 0x77).all() and (buf[260:] == 0x77).all()
    assert (buf[100:164] == 0xA5).all() and (buf[196:260] == 0xA5).all()
    np.testing.assert_array_equal(buf[164:196], np.arange(32, dtype=np.uint8))
