"""Pins of the oracle's retention-aware rearrangement (SemShareKV Sec. 3.3.4; App. A:
Retain[i] = T * prod_{j<=i} alpha_retain[j], tokens not retained are evicted): each layer's
rearranged cache holds only its retained target tokens' rows, packed in list order."""
import os

import numpy as np
import pytest

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_golden_small(oracle_mod):
    ret, outs = {}, {}
    with open(os.path.join(GOLDEN, "gather_retained_small.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            key, *v = line.split()
            if key == "idx":
                idx = [int(x) for x in v]
            elif key == "retained":
                ret[int(v[0])] = [int(x) for x in v[1:]]
            else:
                outs[int(v[0])] = [float(x) for x in v[1:]]
    ref = np.array([[[[10 * l + r] for r in range(4)]] for l in range(2)], dtype=np.float32)  # [2][1][4][1]
    ok, ov, bad = oracle_mod.gather_kv_retained(ref, ref + 100, idx, [ret[0], ret[1]], cap=3)
    assert bad == 0
    for l in (0, 1):
        n = len(outs[l])
        np.testing.assert_array_equal(ok[l, 0, :n, 0], outs[l])
        np.testing.assert_array_equal(ov[l, 0, :n, 0], np.array(outs[l]) + 100)
        assert np.all(ok[l, 0, n:] == 0)


def _case(L=3, H=2, N=50, hd=8, T=40, seed=1):
    g = np.random.default_rng(seed)
    k = workloads.f32_to_bf16_bits(g.standard_normal((L, H, N, hd), dtype=np.float32))
    v = workloads.f32_to_bf16_bits(g.standard_normal((L, H, N, hd), dtype=np.float32))
    idx = g.integers(0, N, size=T).astype(np.int32)
    perm = g.permutation(T)
    counts = [T, 31, 0][:L] if L == 3 else [int(T * 0.8 ** (i + 1)) for i in range(L)]
    ret = [np.sort(perm[:c]).astype(np.int32) for c in counts]
    return k, v, idx, ret


def test_equals_full_rearrangement_then_row_selection(oracle_mod):
    k, v, idx, ret = _case()
    ok, ov, bad = oracle_mod.gather_kv_retained(k, v, idx, ret)
    fk, fv, fbad = oracle_mod.gather_kv(k, v, idx)  # [1][L][H][T][hd]
    assert bad == 0 and fbad == 0
    for l, r in enumerate(ret):
        np.testing.assert_array_equal(ok[l, :, :len(r)], fk[0, l][:, r])
        np.testing.assert_array_equal(ov[l, :, :len(r)], fv[0, l][:, r])
        assert np.all(ok[l, :, len(r):] == 0)


def test_all_retained_is_the_plain_rearrangement(oracle_mod):
    k, v, idx, _ = _case(seed=2)
    T = len(idx)
    ok, ov, _ = oracle_mod.gather_kv_retained(k, v, idx, [np.arange(T)] * k.shape[0])
    fk, fv, _ = oracle_mod.gather_kv(k, v, idx)
    np.testing.assert_array_equal(ok, fk[0])
    np.testing.assert_array_equal(ov, fv[0])


def test_brute_force_and_bad_entries(oracle_mod):
    k, v, idx, ret = _case(L=2, T=12, N=9, seed=5)
    idx[3] = 99                                # an index outside the reference
    ret = [np.array([5, 3, 11, 0], dtype=np.int32), np.array([12, 7], dtype=np.int32)]  # 12 is outside [0, T)
    ok, ov, bad = oracle_mod.gather_kv_retained(k, v, idx, ret, cap=5)
    assert bad == 2
    for l, r in enumerate(ret):
        for j, t in enumerate(r):
            for h in range(k.shape[1]):
                if 0 <= t < len(idx) and 0 <= idx[t] < k.shape[2]:
                    assert np.array_equal(ok[l, h, j], k[l, h, idx[t]]) and np.array_equal(ov[l, h, j], v[l, h, idx[t]])
                else:
                    assert np.all(ok[l, h, j] == 0) and np.all(ov[l, h, j] == 0)
