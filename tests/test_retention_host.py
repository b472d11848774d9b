"""Host-side retention bookkeeping (no GPU): the per-layer counts of App. A and the synthetic
nested retained sets the tests and the bench use."""
import numpy as np
import pytest

import workloads


def test_retain_counts_helper():
    """Retain[i] = T * prod_{j<=i} alpha_retain[j] (App. A), rounded down."""
    ss = pytest.importorskip("paper_2509_24832_gb300")
    assert ss.retain_counts(1000, [0.8, 0.5, 0.5]) == [800, 400, 200]
    assert ss.retain_counts(5120, [1.0] * 4) == [5120] * 4
    assert ss.retain_counts(10, [0.75, 0.75]) == [7, 5]   # 7.5 -> 7, 5.625 -> 5
    assert ss.retain_counts(7, []) == []


def test_synthetic_retained_sets_are_nested_and_sorted():
    counts = [80, 70, 70, 12, 0]
    ret = workloads.retained_tokens(100, counts, seed=3)
    assert [len(r) for r in ret] == counts
    for a, b in zip(ret, ret[1:]):
        assert set(b) <= set(a)
    assert all(np.all(np.diff(r) > 0) for r in ret)
    assert workloads.retain_alphas(3) == [0.8, 0.98, 0.98]
