"""The commit gate of AsmEvo (Eq. 2) and the GatedEval timing statistics
(Sec. 3.4, Algorithm 1), restated plainly.  TEST INFRASTRUCTURE ONLY: only
tests/, __graft_entry__.smoke() and bench.py's CPU legs may use this module.

Readings (the paper states the formula and the constants only):
  - the latency of a kernel is the median of R event-timed launches after
    warm-up; for even R, the mean of the two middle samples;
  - cv is the sample standard deviation (divisor R - 1) over the mean, taken
    for each of the two kernels timed; the gate uses the larger one, since
    both latencies enter the speedup;
  - every quantity is one double operation after another in the order
    written below.
"""
import math

EPS, K, S_FLOOR = 0.002, 0.85, 1.0        # Sec. 5


def timing_summary(samples):
    """(median, mean, cv) of positive finite timing samples."""
    xs = [float(x) for x in samples]
    if not xs or any(not math.isfinite(x) or x <= 0.0 for x in xs):
        raise ValueError("timing samples must be finite and positive")
    r = len(xs)
    srt = sorted(xs)
    median = srt[r // 2] if r % 2 else (srt[r // 2 - 1] + srt[r // 2]) / 2.0
    total = 0.0
    for x in xs:
        total += x
    mean = total / r
    if r == 1:
        return median, mean, 0.0
    ss = 0.0
    for x in xs:
        d = x - mean
        ss += d * d
    return median, mean, math.sqrt(ss / (r - 1)) / mean


def m_star(s_best, cv, eps=EPS, k=K):
    """m* of Eq. 2: (1 + max(eps, k cv)) times the current best speedup."""
    return (1.0 + max(eps, k * cv)) * s_best


def commit(all_eq, s_cand, s_best, cv, eps=EPS, k=K, s_floor=S_FLOOR):
    """g(c) of Eq. 2: equivalent on every input, and a speedup of at least
    max(m*, s_floor)."""
    m = m_star(s_best, cv, eps, k)
    return m, bool(all_eq) and s_cand >= max(m, s_floor)
