"""Pins of the oracle's LSH codes (SemShareKV Sec. 3.3, App. A.2) and its bf16 operand rounding."""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_hash():
    cases = {}
    with open(os.path.join(GOLDEN, "hash_unit.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            tag, key, *vals = line.split()
            cases.setdefault(tag, {})[key] = vals
    return cases


def _bf16(v):
    return workloads.f32_to_bf16_bits(np.asarray(v, dtype=np.float32))


def test_golden_case_a_sign_codes(oracle_mod):
    c = _golden_hash()["A"]
    x = np.array([[float(v) for v in c["x"]]], dtype=np.float32)
    R = np.zeros((32, 4), dtype=np.float32)
    for j in range(32):
        R[j, j % 4] = 1.0 if j < 16 else -1.0
    codes, proj = oracle_mod.hash_codes(x, [0], _bf16(R))
    assert codes[0, 0] == int(c["code"][0], 16)
    np.testing.assert_array_equal(proj[0, :4], x[0])


def test_golden_case_b_rotated_row(oracle_mod):
    c = _golden_hash()["B"]
    x = np.array([[float(v) for v in c["x"]]], dtype=np.float32)
    R = np.zeros((32, 4), dtype=np.float32)
    R[np.arange(4), np.arange(4)] = 1.0
    codes, proj = oracle_mod.hash_codes(x, [int(c["m"][0])], _bf16(R), base=(2.0 / math.pi) ** 2)
    np.testing.assert_array_equal(proj[0, :4], [float(v) for v in c["proj"]])
    assert codes[0, 0] == int(c["code"][0], 16)


def test_golden_case_c_operand_rounding(oracle_mod):
    c = _golden_hash()["C"]
    x = np.array([[float(v) for v in c["x"]]], dtype=np.float32)
    R = np.zeros((32, 4), dtype=np.float32)
    R[0, 0] = 1.0
    _, p_r = oracle_mod.hash_codes(x, [0], _bf16(R), round_operand=True)
    _, p_u = oracle_mod.hash_codes(x, [0], _bf16(R), round_operand=False)
    assert p_r[0, 0] == float(c["proj_rounded"][0])
    assert p_u[0, 0] == float(c["proj_unrounded"][0])


def test_integer_projection_brute_force(oracle_mod):
    # position 0 and small integers: every product and sum is exact, so p must equal the exact
    # integer dot product of each hyperplane row with x (catches a transposed operand)
    g = np.random.default_rng(7)
    n, d, nbits = 9, 12, 64
    x = g.integers(-8, 9, size=(n, d)).astype(np.float32)
    R = g.integers(-8, 9, size=(nbits, d)).astype(np.float32)
    codes, proj = oracle_mod.hash_codes(_bf16(x), np.zeros(n, np.int32), _bf16(R))
    for i in range(n):
        for j in range(nbits):
            p = sum(int(R[j, c]) * int(x[i, c]) for c in range(d))
            assert proj[i, j] == p
            bit = (int(codes[i, j // 32]) >> (j % 32)) & 1
            assert bit == (1 if p > 0 else 0)


def test_unit_hyperplanes_give_signs_of_rotated_row(oracle_mod):
    # r_j = e_j: p_j is coordinate j of bf16(RoPE(x)), so the code is its sign pattern
    g = np.random.default_rng(8)
    n, d = 6, 64
    x = g.standard_normal((n, d)).astype(np.float32)
    pos = g.integers(0, 3000, size=n).astype(np.int32)
    R = np.eye(d, dtype=np.float32)
    codes, proj = oracle_mod.hash_codes(x, pos, _bf16(R))
    y = oracle_mod.rope(x.astype(np.float64), pos)
    y_b = np.array([[oracle_mod.bf16_value(oracle_mod.bf16_round(v)) for v in row] for row in y])
    np.testing.assert_array_equal(proj, y_b.astype(np.float32))
    bits = np.unpackbits(codes.view(np.uint8), axis=1, bitorder="little")
    np.testing.assert_array_equal(bits, (y_b > 0).astype(np.uint8))


def test_power_of_two_scaling_invariance(oracle_mod):
    wl = workloads.WORKLOADS["tiny"].scaled(n_ref=40, d=128, nbits=64, emb_dtype="bf16")
    x = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    pos = np.arange(40, dtype=np.int32) * 37
    c1, p1 = oracle_mod.hash_codes(x, pos, R)
    x4 = workloads.f32_to_bf16_bits(workloads.bf16_bits_to_f32(x) * 4.0)
    c4, p4 = oracle_mod.hash_codes(x4, pos, R)
    np.testing.assert_array_equal(c1, c4)
    np.testing.assert_array_equal(p4, p1 * 4.0)


def test_negation_complements_codes(oracle_mod):
    wl = workloads.WORKLOADS["tiny"].scaled(n_ref=40, d=128, nbits=96, emb_dtype="f32")
    x = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    pos = np.arange(40, dtype=np.int32)
    c1, p1 = oracle_mod.hash_codes(x, pos, R)
    c2, p2 = oracle_mod.hash_codes(-x, pos, R)
    np.testing.assert_array_equal(p2, -p1)
    assert (p1 != 0).all()
    np.testing.assert_array_equal(c2, ~c1)


def test_null_positions_mean_row_index(oracle_mod):
    wl = workloads.WORKLOADS["tiny"].scaled(n_ref=20, d=64, nbits=32)
    x = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    a = oracle_mod.hash_codes(x, None, R)
    b = oracle_mod.hash_codes(x, np.arange(20), R)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])


def _bf16_nearest_exact(v: float) -> int:
    """Brute force: the bf16 pattern nearest to v by exact rational distance, ties to even."""
    if v == 0.0:
        return 0x8000 if math.copysign(1.0, v) < 0 else 0
    base = int(workloads.f32_to_bf16_bits(np.array([v], dtype=np.float32))[0]) & 0x7FFF
    sign = 0x8000 if v < 0 else 0
    best = None
    for h in range(max(0, base - 2), min(0x7F80, base + 3)):
        val = Fraction(float(workloads.bf16_bits_to_f32(np.array([h], dtype=np.uint16))[0]))
        dist = abs(Fraction(abs(v)) - val)
        key = (dist, h & 1)
        if best is None or key < best[0]:
            best = (key, h)
    return sign | best[1]


def test_bf16_round_is_nearest_even(oracle_mod):
    g = np.random.default_rng(9)
    vals = list(g.standard_normal(3000) * np.exp2(g.integers(-20, 20, size=3000)))
    # values around bf16 midpoints, including ones where float32 rounding lands on the midpoint
    for h in [0x3F80, 0x3F81, 0x4000, 0x4001, 0xBF85, 0x0081, 0x7F00]:
        lo = Fraction(float(workloads.bf16_bits_to_f32(np.array([h], dtype=np.uint16))[0]))
        hi = Fraction(float(workloads.bf16_bits_to_f32(np.array([h + 1], dtype=np.uint16))[0]))
        mid = (lo + hi) / 2
        for eps in [0, Fraction(1, 2 ** 60), -Fraction(1, 2 ** 60), Fraction(1, 2 ** 40), -Fraction(1, 2 ** 40)]:
            vals.append(float(mid * (1 + eps)))
    for v in vals:
        assert oracle_mod.bf16_round(v) == _bf16_nearest_exact(v), v


def test_bf16_round_matches_torch_on_float32(oracle_mod):
    torch = pytest.importorskip("torch")
    g = np.random.default_rng(10)
    v = (g.standard_normal(5000) * np.exp2(g.integers(-30, 30, size=5000))).astype(np.float32)
    want = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().astype(np.uint16)
    got = np.array([oracle_mod.bf16_round(float(t)) for t in v], dtype=np.uint16)
    np.testing.assert_array_equal(got, want)
