"""Pins for the oracle's Dynamic Partitioning (Section 4.1, Algorithm 1; Eq. 2, Eq. 3).

Each check ties the oracle to something other than its own code: hand-worked
partitions, closed-form invariants, and brute-force enumeration on tiny cases.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import partition as P

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "partition_examples.json")


def test_worked_examples():
    cases = json.load(open(GOLDEN))["cases"]
    assert len(cases) >= 5
    for c in cases:
        assert P.partition_sizes(c["cp"], c["N"]) == c["sizes"], c


def _random_cases(count=3000, seed=11):
    rng = np.random.default_rng(seed)
    for _ in range(count):
        m = int(rng.integers(1, 17))
        n = int(rng.integers(m, 20000))
        kind = rng.integers(0, 3)
        if kind == 0:
            cp = rng.lognormal(0.0, 1.0, m)
        elif kind == 1:
            cp = rng.integers(1, 7, m).astype(float)    # many exact ties
        else:
            cp = rng.uniform(0.01, 1.0, m)
        yield list(map(float, cp)), n


def test_sum_and_quota_bounds():
    for cp, n in _random_cases():
        sizes = P.partition_sizes(cp, n)
        assert sum(sizes) == n
        assert all(s >= 1 for s in sizes)
        q = P.quotas(cp, n)
        if all(v >= 1.0 for v in q):          # the >= 1 fix-up is inactive
            assert all(abs(s - v) < 1.0 for s, v in zip(sizes, q)), (cp, n, sizes)


def test_equal_weights_is_plain_data_parallelism():
    # Section 3: Sync-SGD splits the data uniformly, |D_i| ~ |D| / M.
    for m in range(1, 17):
        for n in (m, m + 1, 128, 1000, 16384, 16383):
            sizes = P.partition_sizes([2.5] * m, n)
            base, extra = divmod(n, m)
            assert sizes == [base + 1] * extra + [base] * (m - extra)
            assert P.even_sizes(m, n) == sizes


def test_scale_invariance():
    rng = np.random.default_rng(5)
    for cp, n in _random_cases(500, seed=3):
        for k in (2.0, 0.5, 1024.0, 2.0 ** -20):        # exact scalings in binary
            assert P.partition_sizes([c * k for c in cp], n) == P.partition_sizes(cp, n)
        # a generic factor changes the quotas by a few ulps: the result may only move where
        # two remainders sit within that rounding of each other
        k = float(rng.uniform(0.1, 10))
        q = P.quotas(cp, n)
        rem = sorted(v - math.floor(v) for v in q)
        if all(b - a > 1e-9 for a, b in zip(rem, rem[1:])) and all(v >= 1.0 for v in q):
            assert P.partition_sizes([c * k for c in cp], n) == P.partition_sizes(cp, n)


def test_predicted_times_equalised():
    # Eq. 3: X'_m = |D'_m| / CP_m; sizing |D'_m| ~ CP_m |D| makes them equal up to rounding.
    for cp, n in _random_cases(1000, seed=7):
        s = sum(cp)
        cpn = [c / s for c in cp]
        q = P.quotas(cp, n)
        if not all(v >= 1.0 for v in q):
            continue
        sizes = P.partition_sizes(cp, n)
        x = P.predicted_times(sizes, cpn)
        for xm, c in zip(x, cpn):
            assert abs(xm - n) < 1.0 / c + 1e-9


def test_compute_power_round_trip():
    # Workers of speed c_m that processed n_m samples take X_m = n_m / c_m (Eq. 2 inverted);
    # Algorithm 1 at t > 0 then sizes the next partition from c alone.
    rng = np.random.default_rng(9)
    for _ in range(300):
        m = int(rng.integers(1, 12))
        n = int(rng.integers(m, 5000))
        speed = rng.lognormal(0, 0.7, m)
        prev = P.even_sizes(m, n)
        times = [prev[i] / speed[i] for i in range(m)]
        cp = P.compute_power(prev, times)
        assert np.allclose(cp, speed, rtol=1e-13)
        assert P.dynamic_partitioning(1, times, prev, n, m) == P.partition_sizes(cp, n)
        assert P.dynamic_partitioning(0, times, prev, n, m) == P.even_sizes(m, n)


def test_brute_force_minimisers():
    """Among all non-negative integer vectors summing to N, the rule returns a minimiser of
    max |n - q| and of sum |n - q|, and the lowest-index one among tied minimisers."""
    rng = np.random.default_rng(1)
    checked = 0
    for _ in range(400):
        m = int(rng.integers(1, 5))
        n = int(rng.integers(m, 13))
        cp = [float(v) for v in rng.integers(1, 5, m)] if rng.random() < 0.5 \
            else [float(v) for v in rng.uniform(0.2, 1.0, m)]
        q = P.quotas(cp, n)
        if not all(v >= 1.0 for v in q):
            continue
        cands = []
        for vec in itertools.product(range(n + 1), repeat=m):
            if sum(vec) != n:
                continue
            key = (max(abs(v - w) for v, w in zip(vec, q)), sum(abs(v - w) for v, w in zip(vec, q)))
            cands.append((key, vec))
        kmin = min(k for k, _ in cands)
        tied = [v for k, v in cands if abs(k[0] - kmin[0]) < 1e-12 and abs(k[1] - kmin[1]) < 1e-12]
        got = tuple(P.partition_sizes(cp, n))
        assert got in tied, (cp, n, got, tied)
        # lowest-index choice: extra samples go to the earliest workers among equal remainders,
        # i.e. the lexicographically largest of the tied minimisers.  Remainders are compared in
        # fp64, so quotas that are equal only in exact arithmetic (4/9*12 vs 1/9*12) may differ in
        # the last ulp; the lexicographic check applies where fp64 ties are exact or clearly apart.
        rem = [v - math.floor(v) for v in q]
        fuzzy = any(0 < abs(a - b) < 1e-12 for a in rem for b in rem)
        if not fuzzy:
            assert got == max(tied), (cp, n, got, tied)
        checked += 1
    assert checked > 100


def test_offsets_and_index_map():
    sizes = [43, 85, 128, 256]
    off = P.offsets(sizes)
    assert off == [0, 43, 128, 256, 512]
    im = P.index_map(sizes)
    assert len(im) == 512
    for i, m in enumerate(im):
        assert off[m] <= i < off[m + 1]


@pytest.mark.parametrize("cp,n", [([], 4), ([1.0, 1.0], 1), ([1.0, -1.0], 4), ([1.0, 0.0], 4),
                                  ([1.0, math.inf], 4), ([1.0, math.nan], 4)])
def test_invalid_inputs_raise(cp, n):
    with pytest.raises(ValueError):
        P.partition_sizes(cp, n)


def test_cp_history_closed_forms():
    seq = [[1.0, 2.0], [3.0, 2.0], [5.0, 8.0], [7.0, 2.0]]
    last = P.CPHistory("last")
    assert [last.update(c) for c in seq][-1] == [7.0, 2.0]
    ema = P.CPHistory("ema", 0.5)
    outs = [ema.update(c) for c in seq]
    assert outs[0] == [1.0, 2.0] and outs[1] == [2.0, 2.0] and outs[2] == [3.5, 5.0] and outs[3] == [5.25, 3.5]
    win = P.CPHistory("window", 2)
    outs = [win.update(c) for c in seq]
    assert outs[0] == [1.0, 2.0] and outs[1] == [2.0, 2.0] and outs[2] == [4.0, 5.0] and outs[3] == [6.0, 5.0]
    # a constant history is its own estimate, so the partition equals the one-shot rule
    for h in (P.CPHistory("ema", 0.3), P.CPHistory("window", 3)):
        for _ in range(5):
            est = h.update([1.0, 3.0])
        assert P.partition_sizes(est, 128) == [32, 96]
