"""Host-side retention bookkeeping (no GPU): the per-layer counts of App. A and the synthetic
nested retained sets the tests and the bench use."""
import math
from fractions import Fraction

import numpy as np
import pytest

import workloads


def _lib_ss():
    ss = pytest.importorskip("paper_2509_24832_gb300")
    from paper_2509_24832_gb300 import build

    build.build()
    return ss


def _exact_retain(n_tok, nums, den):
    """Retain[i] = floor(T * prod_{j<=i} num_j / den) with Python's exact rationals."""
    out, p = [], Fraction(n_tok)
    for a in nums:
        p *= Fraction(a, den)
        out.append(math.floor(p))
    return out


def test_retain_counts_hand_cases():
    """Retain[i] = T * prod_{j<=i} alpha_retain[j] (App. A), rounded down, worked by hand."""
    ss = _lib_ss()
    assert ss.retain_counts(1000, [800, 500, 500], 1000) == [800, 400, 200]
    assert ss.retain_counts(5120, [1000] * 4, 1000) == [5120] * 4
    assert ss.retain_counts(10, [3, 3], 4) == [7, 5]              # 7.5 -> 7, 5.625 -> 5
    assert ss.retain_counts(7, [], 1000) == []
    # 0.7 and 0.1 have no exact binary form (1000 * 0.7 in doubles is 699.99999999999994): the
    # rational ratios keep these products exact
    assert ss.retain_counts(1000, [700], 1000) == [700]
    assert ss.retain_counts(100, [1, 1], 10) == [10, 1]
    assert ss.retain_counts(3, [1, 1, 1], 3) == [1, 0, 0]
    assert ss.retain_counts(0, [500, 500], 1000) == [0, 0]
    assert ss.retain_counts(5, [0, 1000], 1000) == [0, 0]


def test_retain_counts_against_exact_rationals():
    """Random schedules of up to 128 layers against Fraction arithmetic (a planted float rounding
    or a per-layer floor instead of one floor of the whole product fails this)."""
    ss = _lib_ss()
    g = np.random.default_rng(5)
    for trial in range(300):
        L = int(g.integers(0, 129))
        den = int(g.choice([1, 2, 3, 7, 10, 100, 1000, 4096, 99991, 2**31 - 1]))
        nums = [int(x) for x in g.integers(0 if trial % 3 else den // 2, den + 1, size=L)]
        T = int(g.choice([0, 1, 5, 1000, 5120, 65536, 2**31 - 1]))
        assert ss.retain_counts(T, nums, den) == _exact_retain(T, nums, den), (T, den, nums[:5])
    # the synthetic schedule of the 5k workload (0.8, then 0.98 per layer)
    nums = workloads.retain_alphas(32)
    assert ss.retain_counts(5120, nums, workloads.RETAIN_DEN) == _exact_retain(5120, nums, workloads.RETAIN_DEN)


def test_retain_counts_rejects_bad_arguments():
    ss = _lib_ss()
    for args in [(-1, [1], 2), (1 << 31, [1], 2), (10, [3], 2), (10, [-1], 2), (10, [1], 0), (10, [1] * 129, 2)]:
        with pytest.raises(ss.SemshareError):
            ss.retain_counts(*args)


def test_hd_count_is_the_ceiling_of_the_percentage():
    """Insight 1's 40%: k = ceil(0.4 T), checked against exact rationals for every T up to 5000
    and at the 5k and batched lengths."""
    ss = _lib_ss()
    for T in list(range(0, 5001)) + [5120, 2048, 4096, 65536, (1 << 40) - 1]:
        assert ss.hd_count(T) == math.ceil(Fraction(40 * T, 100)), T
    for pct in (0, 1, 33, 50, 99, 100):
        for T in (0, 1, 7, 100, 5120):
            assert ss.hd_count(T, pct) == math.ceil(Fraction(pct * T, 100))
    for bad in [(-1, 40), (1 << 40, 40), (10, -1), (10, 101)]:
        with pytest.raises(ss.SemshareError):
            ss.hd_count(*bad)


def test_synthetic_retained_sets_are_nested_and_sorted():
    counts = [80, 70, 70, 12, 0]
    ret = workloads.retained_tokens(100, counts, seed=3)
    assert [len(r) for r in ret] == counts
    for a, b in zip(ret, ret[1:]):
        assert set(b) <= set(a)
    assert all(np.all(np.diff(r) > 0) for r in ret)
    assert workloads.retain_alphas(3) == [800, 980, 980] and workloads.RETAIN_DEN == 1000
