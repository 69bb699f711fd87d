"""Pins of the oracle's top-k sampling (paper Sections 2-4: top-k sampling
with k = 50; top-p and min-p as second-stage logit processors) and of the
counter-based generator that gives each draw its uniform.

Each pin checks the oracle against something other than itself: published
known-answer vectors of the generator, closed forms of the sampling
distribution, an independent 50-digit evaluation, limits of the
temperature, and the frequencies of many draws."""
import math
import os
from fractions import Fraction

import mpmath
import numpy as np
import pytest

import oracle as default_oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def load_kat():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        w = [int(x, 16) for x in line.split()]
        rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


# ---------------------------------------------------------------------------
def pin_philox_known_answers(lib):
    kat = load_kat()
    assert len(kat) == 3
    for ctr, key, want in kat:
        got = [int(x) for x in lib.philox4x32_10(ctr, key)]
        assert got == want, (ctr, key, [hex(x) for x in got])


def pin_uniform_from_known_answer(lib):
    """Seed 0, step 0, query 0 is Philox counter (0, 0, 0, 0) with key
    (0, 0): its first published output word 0x6627e8d5, top 24 bits over 2^24."""
    (ctr, key, want), = [r for r in load_kat() if r[0] == [0, 0, 0, 0] and r[1] == [0, 0]]
    assert lib.uniform(0, 0, 0) == (want[0] >> 8) / 2**24 == 0x6627E8 / 2**24


def pin_uniform_is_24_bit_and_uniform(lib):
    us = np.array([lib.uniform(12345, step, 0) for step in range(20000)])
    assert np.all((us >= 0.0) & (us < 1.0))
    assert np.all(us * 2**24 == np.floor(us * 2**24))  # exact in fp32
    # Kolmogorov-Smirnov distance of 20000 draws from U[0, 1): 1.63/sqrt(n) is the 1 % point
    s = np.sort(us)
    n = s.size
    dplus = np.max(np.arange(1, n + 1) / n - s)
    dminus = np.max(s - np.arange(0, n) / n)
    assert max(dplus, dminus) < 1.63 / math.sqrt(n)
    # queries, steps and seeds give different streams
    a = np.array([lib.uniform(7, s, 0) for s in range(4000)])
    b = np.array([lib.uniform(7, s, 1) for s in range(4000)])
    c = np.array([lib.uniform(8, s, 0) for s in range(4000)])
    assert abs(np.corrcoef(a, b)[0, 1]) < 0.06 and abs(np.corrcoef(a, c)[0, 1]) < 0.06


def pin_equal_logits_draw_floor_uk(lib):
    """Equal logits, no truncation: p_j = 1/k, so the inverse CDF picks
    j = floor(u k) (u k in exact rational arithmetic), including at the
    boundaries u = m / k when 1/k is exact in binary (k a power of two)."""
    for k in (1, 2, 3, 4, 7, 8, 50, 64):
        z = np.full(k, 1.5)
        us = [0.0, 0.25, 0.5, 0.75, 0.999, 1.0 / 3.0, 0.1, 0.61]
        if k & (k - 1) == 0:
            us += [m / k for m in range(k)]
        for u in us:
            uk = Fraction(u) * k
            if k & (k - 1) and abs(uk - round(uk)) < Fraction(1, 10**12):
                continue  # a boundary the fp64 cumulative sums cannot place exactly
            j, prob, kept = lib.sample_sorted(z, 0.8, 1.0, 0.0, u)
            assert kept == k and j == min(math.floor(uk), k - 1), (k, u, j)
            assert abs(prob - 1.0 / k) < 1e-15


def pin_two_candidates_logistic(lib):
    """Two candidates a logit gap D apart: p_0 = 1 / (1 + exp(-D / T))."""
    for D, T in ((1.0, 1.0), (3.0, 0.5), (0.2, 2.0), (7.0, 1.3)):
        p0 = 1.0 / (1.0 + math.exp(-D / T))
        for u in (p0 - 1e-9, p0 + 1e-9, p0 * 0.5, (1 + p0) * 0.5):
            if not 0 <= u < 1:
                continue
            j, prob, kept = lib.sample_sorted([D, 0.0], T, 1.0, 0.0, u)
            assert kept == 2 and j == (0 if u < p0 else 1), (D, T, u)
            assert abs(prob - (p0 if j == 0 else 1 - p0)) < 1e-12


def pin_top_p_prefix(lib):
    """Equal logits, k = 4: each candidate holds exactly 1/4, so the top-p
    prefix is the smallest n with n/4 >= top_p."""
    z = np.zeros(4)
    for top_p, n in ((1.0, 4), (0.75, 3), (0.5, 2), (0.5000001, 3), (0.25, 1), (0.2, 1), (1e-12, 1)):
        _, _, kept = lib.sample_sorted(z, 1.0, top_p, 0.0, 0.3)
        assert kept == n, (top_p, kept)
    # a single candidate survives a tiny top-p: always the best, with probability 1
    for u in (0.0, 0.5, 0.9999):
        assert lib.sample_sorted([3.0, 2.9, 2.8], 1.0, 1e-12, 0.0, u) == (0, 1.0, 1)


def pin_min_p_in_log_space(lib):
    """p_j >= min_p p_0  <=>  z_0 - z_j <= -T ln(min_p): count in log space."""
    rng = np.random.default_rng(3)
    for _ in range(40):
        k = int(rng.integers(2, 60))
        z = np.sort(rng.normal(0, 3, k))[::-1]
        T = float(rng.uniform(0.3, 2.0))
        min_p = float(rng.uniform(0.01, 0.9))
        gap = -T * math.log(min_p)
        if np.min(np.abs((z[0] - z) - gap)) < 1e-9:
            continue  # too close to the boundary to decide in either form
        want = int(np.sum(z[0] - z <= gap))
        _, _, kept = lib.sample_sorted(z, T, 1.0, min_p, 0.5)
        assert kept == want, (k, T, min_p, kept, want)
    # min_p = 1 keeps only the maximum; min_p = 0 keeps everything
    assert lib.sample_sorted([5.0, 4.0, 3.0], 1.0, 1.0, 1.0, 0.99)[2] == 1
    assert lib.sample_sorted([5.0, 4.0, 3.0], 1.0, 1.0, 0.0, 0.99)[2] == 3


def _mp_draw(z, T, top_p, min_p, u):
    """The same definition evaluated with 50-digit arithmetic."""
    mpmath.mp.dps = 50
    e = [mpmath.exp(mpmath.mpf(x) / T - mpmath.mpf(z[0]) / T) for x in z]
    tot = mpmath.fsum(e)
    p = [x / tot for x in e]
    n_p = len(z)
    run = mpmath.mpf(0)
    for n in range(1, len(z) + 1):
        run += p[n - 1]
        if run >= top_p:
            n_p = n
            break
    n_m = sum(1 for x in p if x >= min_p * p[0])
    n = min(n_p, n_m)
    M = mpmath.fsum(p[:n])
    cum = mpmath.mpf(0)
    for j in range(n):
        cum += p[j]
        if cum > u * M:
            return j, p, n, M
    return n - 1, p, n, M


def pin_high_precision(lib):
    rng = np.random.default_rng(11)
    checked = 0
    for _ in range(60):
        k = int(rng.integers(1, 12))
        z = np.sort(rng.normal(0, 2, k))[::-1]
        T = float(rng.uniform(0.2, 3.0))
        top_p = float(rng.uniform(0.3, 1.0))
        min_p = float(rng.uniform(0.0, 0.5))
        u = float(rng.random())
        j_hp, p, n, M = _mp_draw(z, T, top_p, min_p, u)
        # skip draws within 1e-12 of a boundary of the kept set or of the CDF
        cums = [mpmath.fsum(p[:i + 1]) for i in range(k)]
        if any(abs(c - top_p) < 1e-12 for c in cums) or any(abs(x - min_p * p[0]) < 1e-12 for x in p):
            continue
        if any(abs(c - u * M) < 1e-12 for c in cums[:n]):
            continue
        j, prob, kept = lib.sample_sorted(z, T, top_p, min_p, u)
        assert (j, kept) == (j_hp, n), (z, T, top_p, min_p, u)
        assert abs(prob - float(p[j_hp] / M)) < 1e-12
        checked += 1
    assert checked >= 50


def pin_temperature_limits(lib):
    z = np.array([4.0, 3.5, 1.0, -2.0, -2.5])
    for u in (0.0, 0.3, 0.9, 0.999999):  # T -> 0: all mass on the best candidate
        assert lib.sample_sorted(z, 1e-6, 1.0, 0.0, u)[0] == 0
    for u in (0.05, 0.3, 0.55, 0.95):    # T -> infinity: uniform over the k
        assert lib.sample_sorted(z, 1e9, 1.0, 0.0, u)[0] == int(u * 5)


def pin_frequencies(lib):
    """40000 draws at consecutive steps: each candidate's share matches its
    renormalised probability within 5 standard deviations."""
    z = np.array([2.0, 1.6, 1.5, 0.4, -0.3])
    T, top_p, min_p = 0.7, 0.93, 0.05
    _, p, n, M = _mp_draw(z, T, top_p, min_p, 0.5)
    want = np.array([float(p[j] / M) for j in range(n)])
    N = 40000
    counts = np.zeros(len(z), int)
    for step in range(N):
        counts[lib.sample_sorted(z, T, top_p, min_p, lib.uniform(99, step, 3))[0]] += 1
    assert counts[n:].sum() == 0
    sd = np.sqrt(want * (1 - want) / N)
    assert np.all(np.abs(counts[:n] / N - want) < 5 * sd + 1e-4), (counts / N, want)


def pin_argument_errors(lib):
    for T, top_p, min_p, u in ((0.0, 1.0, 0.0, 0.5), (-1.0, 1.0, 0.0, 0.5), (1.0, 0.0, 0.0, 0.5),
                               (1.0, 1.5, 0.0, 0.5), (1.0, 1.0, -0.1, 0.5), (1.0, 1.0, 1.1, 0.5),
                               (1.0, 1.0, 0.0, 1.0), (1.0, 1.0, 0.0, -0.1)):
        with pytest.raises(ValueError):
            lib.sample_sorted([1.0, 0.0], T, top_p, min_p, u)


SAMPLING_PINS = [(f.__name__, f) for f in (
    pin_philox_known_answers, pin_uniform_from_known_answer, pin_uniform_is_24_bit_and_uniform, pin_equal_logits_draw_floor_uk,
    pin_two_candidates_logistic, pin_top_p_prefix, pin_min_p_in_log_space, pin_high_precision,
    pin_temperature_limits, pin_frequencies, pin_argument_errors)]


@pytest.mark.parametrize("name,pin", SAMPLING_PINS, ids=[n for n, _ in SAMPLING_PINS])
def test_sampling_pin(name, pin):
    pin(default_oracle._default())
