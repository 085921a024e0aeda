"""Pins of the plain commit-gate and timing-statistics oracle (Eq. 2;
GatedEval timing, Sec. 3.4): Python's statistics module, closed forms and
the paper's constants."""
import math
import random
import statistics

import pytest

from oracle import gate as G


def test_constants_are_the_papers():
    assert (G.EPS, G.K, G.S_FLOOR) == (0.002, 0.85, 1.0)


@pytest.mark.parametrize("r", [1, 2, 3, 10, 11, 50])
def test_summary_against_statistics(r):
    rng = random.Random(r)
    xs = [rng.uniform(0.5, 2.0) for _ in range(r)]
    med, mean, cv = G.timing_summary(xs)
    assert med == statistics.median(xs)
    assert abs(mean - math.fsum(xs) / r) <= 4 * r * 2.0 ** -53 * mean
    if r > 1:
        want = statistics.stdev(xs) / statistics.fmean(xs)
        assert abs(cv - want) <= 1e-12 * want
    else:
        assert cv == 0.0


def test_summary_closed_forms():
    assert G.timing_summary([2.0] * 7) == (2.0, 2.0, 0.0)
    med, mean, cv = G.timing_summary([1.0, 3.0])
    assert (med, mean) == (2.0, 2.0) and cv == math.sqrt(2.0) / 2.0
    assert G.timing_summary([5.0, 1.0, 3.0])[0] == 3.0       # median of unsorted samples
    for bad in ([], [1.0, 0.0], [1.0, -2.0], [float("nan")], [float("inf")]):
        with pytest.raises(ValueError):
            G.timing_summary(bad)


def test_margin_is_eps_below_the_crossover():
    # k cv < eps  <=>  cv < 0.002 / 0.85
    cross = 0.002 / 0.85
    assert G.m_star(1.0, 0.0) == 1.002
    assert G.m_star(1.0, cross * 0.99) == 1.002
    assert G.m_star(1.0, 0.01) == (1.0 + 0.85 * 0.01) * 1.0
    assert abs(G.m_star(1.0, 0.01) - 1.0085) < 1e-15
    assert abs(G.m_star(1.5, 0.1) - 1.5 * 1.085) < 1e-15


def test_commit_rule():
    # equivalent, speedup exactly m*: commits (>=)
    m, ok = G.commit(True, 1.002, 1.0, 0.0)
    assert m == 1.002 and ok
    assert not G.commit(True, 1.0019, 1.0, 0.0)[1]
    # never without equivalence
    assert not G.commit(False, 10.0, 1.0, 0.0)[1]
    # against a better current best the margin scales with it
    assert G.commit(True, 1.202, 1.2, 0.0)[1] is False      # m* = 1.2024
    assert G.commit(True, 1.2025, 1.2, 0.0)[1] is True
    # s_floor rejects a "speedup" below 1 even when the best so far is lower
    assert not G.commit(True, 0.9, 0.5, 0.0)[1]
    # noisy timing raises the bar
    assert not G.commit(True, 1.05, 1.0, 0.1)[1] and G.commit(True, 1.09, 1.0, 0.1)[1]
