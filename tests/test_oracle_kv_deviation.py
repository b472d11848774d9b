"""Pins of the oracle's Key-Value deviation (SemShareKV App. A.4: sigma_K = ||K_reused -
K_recomputed||_2, sigma_V likewise, sigma_KV = sigma_K + sigma_V; read per layer and token over
all heads and head dimensions) and of its high-deviation token selection (Insight 1: the tokens
of highest deviation; ties to the lower token index, listed in ascending order)."""
import os

import numpy as np
import pytest

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden():
    arrs = {n: np.zeros((1, 2, 4, 2), dtype=np.float32) for n in ("k_reused", "v_reused", "k_recomp", "v_recomp")}
    expect, hd = {}, {}
    with open(os.path.join(GOLDEN, "kv_deviation_small.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            key, *v = line.split()
            if key in arrs:
                h, t, a, b = int(v[0]), int(v[1]), float(v[2]), float(v[3])
                arrs[key][0, h, t] = (a, b)
            elif key == "hd":
                hd[int(v[0])] = [int(x) for x in v[1:]]
            else:
                expect[key] = [float(x) for x in v]
    return arrs, expect, hd


def test_golden_small(oracle_mod):
    arrs, expect, hd = _golden()
    sk, sv, skv = oracle_mod.kv_deviation(arrs["k_reused"], arrs["v_reused"], arrs["k_recomp"], arrs["v_recomp"])
    np.testing.assert_allclose(sk[0], expect["sigma_k"], rtol=1e-15, atol=0)
    np.testing.assert_allclose(sv[0], expect["sigma_v"], rtol=1e-15, atol=0)
    np.testing.assert_allclose(skv[0], expect["sigma_kv"], rtol=1e-15, atol=0)
    for k, idx in hd.items():
        np.testing.assert_array_equal(oracle_mod.select_hd(skv, k)[0], idx)


def _bf16_arrays(shape, seed, n=4, spread=1.0):
    g = workloads.rng(seed, 7)
    base = g.standard_normal(shape, dtype=np.float32)
    out = []
    for i in range(n):
        x = base + spread * (i % 2) * g.standard_normal(shape, dtype=np.float32)
        out.append(workloads.f32_to_bf16_bits(x))
    return out


@pytest.mark.parametrize("shape", [(1, 8, 37, 128), (3, 2, 5, 64), (2, 1, 1, 16)])
def test_against_numpy_norm(oracle_mod, shape):
    """The norm is numpy's 2-norm of each token's [H][hd] difference block (a library routine)."""
    k_re, k_rc, v_re, v_rc = _bf16_arrays(shape, seed=sum(shape))
    sk, sv, skv = oracle_mod.kv_deviation(k_re, v_re, k_rc, v_rc)
    f = workloads.bf16_bits_to_f32
    dk = (f(k_re).astype(np.float64) - f(k_rc)).transpose(0, 2, 1, 3).reshape(shape[0], shape[2], -1)
    dv = (f(v_re).astype(np.float64) - f(v_rc)).transpose(0, 2, 1, 3).reshape(shape[0], shape[2], -1)
    np.testing.assert_allclose(sk, np.linalg.norm(dk, axis=2), rtol=1e-13)
    np.testing.assert_allclose(sv, np.linalg.norm(dv, axis=2), rtol=1e-13)
    np.testing.assert_allclose(skv, sk + sv, rtol=0, atol=0)


def test_invariants(oracle_mod):
    shape = (2, 4, 9, 32)
    k_re, k_rc, v_re, v_rc = _bf16_arrays(shape, seed=3)
    sk, sv, skv = oracle_mod.kv_deviation(k_re, v_re, k_rc, v_rc)
    # identical caches deviate by 0
    z = oracle_mod.kv_deviation(k_re, v_re, k_re, v_re)
    assert all(np.all(a == 0) for a in z)
    # symmetric in reused / recomputed
    s2 = oracle_mod.kv_deviation(k_rc, v_rc, k_re, v_re)
    np.testing.assert_array_equal(s2[2], skv)
    # K and V enter separately: swapping them swaps sigma_K and sigma_V
    s3 = oracle_mod.kv_deviation(v_re, k_re, v_rc, k_rc)
    np.testing.assert_array_equal(s3[0], sv)
    np.testing.assert_array_equal(s3[1], sk)
    # the squared norm over heads is the sum of the per-head squared norms
    per_head = [oracle_mod.kv_deviation(*(np.ascontiguousarray(a[:, h:h + 1]) for a in (k_re, v_re, k_rc, v_rc)))[0]
                for h in range(shape[1])]
    np.testing.assert_allclose(sk ** 2, sum(p ** 2 for p in per_head), rtol=1e-12)
    # scaling both caches by 2 (exact in float32) doubles every deviation exactly
    f = [workloads.bf16_bits_to_f32(a) for a in (k_re, v_re, k_rc, v_rc)]
    s1 = oracle_mod.kv_deviation(*f)
    s4 = oracle_mod.kv_deviation(*(2 * a for a in f))
    np.testing.assert_array_equal(s4[2], 2 * s1[2])
    np.testing.assert_array_equal(s1[2], skv)  # bf16 bits and their float32 values agree


def _brute_select(sigma, k):
    return np.array([sorted(sorted(range(len(row)), key=lambda t: (-row[t], t))[:k]) for row in sigma],
                    dtype=np.int64).reshape(len(sigma), k)


@pytest.mark.parametrize("T,k", [(10, 4), (37, 15), (100, 0), (100, 100), (1, 1), (513, 206)])
def test_select_brute_force(oracle_mod, T, k):
    g = np.random.default_rng(T + k)
    sigma = g.random((3, T))
    sigma[1] = np.round(sigma[1] * 4) / 4          # many ties
    sigma[2] = 0.5                                 # all equal: the first k tokens
    got = oracle_mod.select_hd(sigma, k)
    np.testing.assert_array_equal(got, _brute_select(sigma, k))
    np.testing.assert_array_equal(got[2], np.arange(k))
    assert all(np.all(np.diff(r) > 0) for r in got)


def _nan(bits: int) -> float:
    return float(np.array([bits], dtype=np.uint64).view(np.float64)[0])


def _total_order_key(v: float, t: int):
    """Python's own sort key of the selection order: NaN (any sign or payload) first, then larger
    values first (-0 and +0 equal: Python's == says so), then the lower token."""
    return (0, 0.0, t) if v != v else (1, -v, t)


def _brute_select_total(sigma, k):
    return np.array([sorted(sorted(range(len(row)), key=lambda t: _total_order_key(row[t], t))[:k]) for row in sigma],
                    dtype=np.int64).reshape(len(sigma), k)


@pytest.mark.parametrize("k", list(range(0, 14)))
def test_select_nan_inf_signed_zero(oracle_mod, k):
    """Special values at every k: NaNs of both signs and several payloads rank above +inf and tie
    with each other (lower token first), -inf ranks last, -0 ties with +0."""
    qnan, neg_qnan = _nan(0x7FF8000000000000), _nan(0xFFF8000000000000)
    payload, neg_payload = _nan(0x7FF0000000000123), _nan(0xFFF4000000000001)
    row = [0.5, neg_qnan, -0.0, np.inf, 0.0, qnan, -np.inf, 0.5, payload, 1e300, -0.0, neg_payload, 0.25]
    assert len(row) == 13
    sigma = np.array([row, row[::-1]], dtype=np.float64)
    got = oracle_mod.select_hd(sigma, min(k, 13))
    np.testing.assert_array_equal(got, _brute_select_total(sigma, min(k, 13)))
    # by hand: the four NaNs first (tokens 1, 5, 8, 11), then +inf (3), 1e300 (9), the two 0.5
    # (0, 7), 0.25 (12), the three zeros in token order (2, 4, 10), -inf (6)
    rank = [1, 5, 8, 11, 3, 9, 0, 7, 12, 2, 4, 10, 6]
    np.testing.assert_array_equal(got[0], sorted(rank[:min(k, 13)]))


def test_select_zeros_tie_by_token(oracle_mod):
    """-0 and +0 are one value: among them the lower tokens win, whatever their signs."""
    sigma = np.array([[0.0, -0.0, 0.0, -0.0, -0.0, 0.0]])
    for k in range(7):
        np.testing.assert_array_equal(oracle_mod.select_hd(sigma, k)[0], np.arange(k))
    sigma = np.array([[-0.0, 0.0, -0.0, 0.0, -0.0, 0.0]])
    np.testing.assert_array_equal(oracle_mod.select_hd(sigma, 3)[0], [0, 1, 2])


def test_select_random_special_values(oracle_mod):
    """Random rows drawn from a small pool of specials and ties, against the Python sort."""
    g = np.random.default_rng(77)
    pool = np.array([np.nan, -np.nan, np.inf, -np.inf, 0.0, -0.0, 1.0, 1.0, 2.0, -1.0, 3.5])
    pool[1] = _nan(0xFFF8000000000000)
    for T in (1, 2, 7, 64, 301):
        sigma = pool[g.integers(0, len(pool), size=(4, T))]
        for k in sorted({0, 1, T // 3, (40 * T + 99) // 100, T}):
            np.testing.assert_array_equal(oracle_mod.select_hd(sigma, k), _brute_select_total(sigma, k))


def test_kv_deviation_nan_and_inf_payloads(oracle_mod):
    """A NaN anywhere in a token's rows makes its deviation NaN; inf minus a finite value is inf;
    inf minus inf is NaN.  The other tokens are unaffected."""
    shape = (1, 2, 4, 8)
    k_re, k_rc, v_re, v_rc = _bf16_arrays(shape, seed=5)
    base = oracle_mod.kv_deviation(k_re, v_re, k_rc, v_rc)
    k_re2 = k_re.copy()
    k_re2[0, 1, 1, 3] = 0x7FC1          # NaN in token 1's K
    k_re2[0, 0, 2, 0] = 0x7F80          # +inf in token 2's K (the recomputed value is finite)
    v_re2, v_rc2 = v_re.copy(), v_rc.copy()
    v_re2[0, 1, 3, 5] = 0xFF80          # -inf - (-inf) = NaN in token 3's V
    v_rc2[0, 1, 3, 5] = 0xFF80
    sk, sv, skv = oracle_mod.kv_deviation(k_re2, v_re2, k_rc, v_rc2)
    assert np.isnan(sk[0, 1]) and np.isnan(skv[0, 1])
    assert np.isinf(sk[0, 2]) and np.isinf(skv[0, 2])
    assert np.isnan(sv[0, 3]) and np.isnan(skv[0, 3])
    np.testing.assert_array_equal(skv[0, 0], base[2][0, 0])
    # the selection ranks the NaN tokens first, then the inf token
    np.testing.assert_array_equal(oracle_mod.select_hd(skv, 2)[0], [1, 3])
    np.testing.assert_array_equal(oracle_mod.select_hd(skv, 3)[0], [1, 2, 3])
