"""The C ABI's timing statistics and commit gate (host code, no GPU)
against the plain oracle of Eq. 2, bit for bit."""
import random

import pytest

from oracle import gate as G
from paper_2608_20711_gb300 import asmv


@pytest.fixture(scope="module", autouse=True)
def lib():
    import os
    if not os.path.exists(asmv.LIB_PATH):
        from paper_2608_20711_gb300 import build
        build.build()
    asmv.lib()


@pytest.mark.parametrize("r", [1, 2, 5, 20, 101])
def test_summary_matches_oracle(r):
    rng = random.Random(100 + r)
    for _ in range(20):
        xs = [rng.lognormvariate(0.0, 0.3) for _ in range(r)]
        got = asmv.timing_summary(xs)
        med, mean, cv = G.timing_summary(xs)
        assert (got["median_ms"], got["mean_ms"], got["cv"], got["r"]) == (med, mean, cv, r)


def test_gate_matches_oracle():
    rng = random.Random(7)
    for _ in range(2000):
        all_eq = rng.random() < 0.8
        s_best = rng.choice([1.0, rng.uniform(0.5, 3.0)])
        cv = rng.choice([0.0, rng.uniform(0.0, 0.05), 0.002 / 0.85])
        s_cand = rng.choice([G.m_star(s_best, cv), rng.uniform(0.5, 3.5)])
        assert asmv.commit_gate(all_eq, s_cand, s_best, cv) == G.commit(all_eq, s_cand, s_best, cv)


def test_rejects_bad_arguments():
    for xs in ([], [0.0], [-1.0], [float("nan")], [float("inf")]):
        with pytest.raises(asmv.AsmvError):
            asmv.timing_summary(xs)
    for args in ((True, -1.0, 1.0, 0.0), (True, 1.0, 0.0, 0.0), (True, 1.0, 1.0, float("nan")),
                 (True, float("inf"), 1.0, 0.0)):
        with pytest.raises(asmv.AsmvError):
            asmv.commit_gate(*args)
