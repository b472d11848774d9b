"""Pins of the oracle's rotary encoding (SemShareKV Eq. 1, App. A.1; Sec. 3.3.1).

Each check comes from outside the oracle: a hand-derived golden case, a property the
rotation must have, or a special case with a known closed form."""
import math
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _quarter_turn_rows():
    rows = []
    with open(os.path.join(GOLDEN, "rope_quarter_turn.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                v = [float(t) for t in line.split()]
                rows.append((int(v[0]), v[1:5], v[5:9]))
    return rows


def test_golden_quarter_turn(oracle_mod):
    # direction, pairing and the exponent -2k/d of theta_k: any of these wrong breaks a row
    base = (2.0 / math.pi) ** 2
    for m, x, y_expected in _quarter_turn_rows():
        y = oracle_mod.rope(np.array([x]), [m], base)[0]
        np.testing.assert_allclose(y, y_expected, rtol=0, atol=1e-12, err_msg=f"m={m}")


def test_position_zero_is_identity(oracle_mod):
    x = np.random.default_rng(1).standard_normal((7, 64))
    y = oracle_mod.rope(x, 0)
    assert np.array_equal(y, x)


def test_pair_norms_preserved(oracle_mod):
    g = np.random.default_rng(2)
    x = g.standard_normal((32, 128))
    pos = g.integers(0, 70000, size=32)
    y = oracle_mod.rope(x, pos)
    nx = np.hypot(x[:, 0::2], x[:, 1::2])
    ny = np.hypot(y[:, 0::2], y[:, 1::2])
    np.testing.assert_allclose(ny, nx, rtol=1e-12, atol=0)


def test_composition_adds_positions(oracle_mod):
    g = np.random.default_rng(3)
    x = g.standard_normal((16, 96))
    m = g.integers(0, 5000, size=16)
    n = g.integers(0, 5000, size=16)
    twice = oracle_mod.rope(oracle_mod.rope(x, m), n)
    once = oracle_mod.rope(x, m + n)
    np.testing.assert_allclose(twice, once, rtol=0, atol=1e-9)


def test_relative_position_property(oracle_mod):
    # the reason Eq. 1 is used: <RoPE(q, m), RoPE(k, n)> depends only on m - n
    g = np.random.default_rng(4)
    d = 256
    q = g.standard_normal((1, d))
    k = g.standard_normal((1, d))
    for m, n in [(10, 3), (4000, 3990), (100, 0), (5119, 17)]:
        lhs = float(oracle_mod.rope(q, m)[0] @ oracle_mod.rope(k, n)[0])
        rhs = float(oracle_mod.rope(q, m - n)[0] @ k[0])
        assert abs(lhs - rhs) <= 1e-9 * max(1.0, abs(rhs)), (m, n, lhs, rhs)
        shifted = float(oracle_mod.rope(q, m + 77)[0] @ oracle_mod.rope(k, n + 77)[0])
        assert abs(shifted - lhs) <= 1e-9 * max(1.0, abs(lhs))


def test_frequencies_are_powers_of_base(oracle_mod):
    # d = 8, base 10^4: theta = 1, 0.1, 0.01, 0.001, so pair k at position 10^k*m turns exactly
    # as far as pair 0 at position m
    g = np.random.default_rng(5)
    pair = g.standard_normal(2)
    for m in [1, 3, 7]:
        ref = oracle_mod.rope(np.concatenate([pair, np.zeros(6)])[None], m)[0][0:2]
        for k in range(1, 4):
            x = np.zeros(8)
            x[2 * k:2 * k + 2] = pair
            y = oracle_mod.rope(x[None], m * 10 ** k)[0]
            np.testing.assert_allclose(y[2 * k:2 * k + 2], ref, rtol=0, atol=1e-11)
    assert oracle_mod.theta(0, 4096) == 1.0
    assert abs(oracle_mod.theta(1024, 4096) - 0.01) < 1e-17


def test_complex_rotation_form(oracle_mod):
    # Eq. 1 is multiplication of x[2k] + i x[2k+1] by the unit complex number of angle m*theta_k
    g = np.random.default_rng(6)
    d = 64
    x = g.standard_normal((5, d))
    pos = np.array([0, 1, 17, 999, 4095])
    ang = pos[:, None] * (10000.0 ** (-np.arange(0, d, 2) / d))[None, :]
    z = (x[:, 0::2] + 1j * x[:, 1::2]) * np.exp(1j * ang)
    y = oracle_mod.rope(x, pos)
    np.testing.assert_allclose(y[:, 0::2], z.real, rtol=0, atol=1e-12)
    np.testing.assert_allclose(y[:, 1::2], z.imag, rtol=0, atol=1e-12)


@pytest.mark.parametrize("wrong", ["sign", "rotate_half", "exponent"])
def test_pins_catch_planted_mistakes(oracle_mod, wrong):
    # a mistaken rotation (planted here, on the CPU) fails the golden quarter-turn rows
    base = (2.0 / math.pi) ** 2

    def mistaken(x, m):
        d = x.shape[0]
        y = np.empty_like(x)
        for k in range(d // 2):
            e = -k / d if wrong == "exponent" else -2 * k / d
            a = m * base ** e
            c, s = math.cos(a), math.sin(a)
            i0, i1 = (k, k + d // 2) if wrong == "rotate_half" else (2 * k, 2 * k + 1)
            sg = -1.0 if wrong == "sign" else 1.0
            y[i0] = x[i0] * c - sg * x[i1] * s
            y[i1] = sg * x[i0] * s + x[i1] * c
        return y

    failures = 0
    for m, x, y_expected in _quarter_turn_rows():
        if not np.allclose(mistaken(np.array(x), m), y_expected, rtol=0, atol=1e-9):
            failures += 1
    assert failures > 0
