"""Pins of the oracle's "rotate-half" rotary pairing, (k, k + d/2) turned by m * theta_k: an
alternative arrangement of Eq. 1's pairs (2k, 2k+1), offered as an option."""
import os

import numpy as np

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _interleave(x):
    """Q: columns (k, k + d/2) -> (2k, 2k+1)."""
    d = x.shape[-1]
    out = np.empty_like(x)
    out[..., 0::2] = x[..., : d // 2]
    out[..., 1::2] = x[..., d // 2:]
    return out


def _deinterleave(y):
    d = y.shape[-1]
    return np.concatenate([y[..., 0::2], y[..., 1::2]], axis=-1)


def test_golden_quarter_turn(oracle_mod):
    rows = []
    with open(os.path.join(GOLDEN, "rope_half_quarter_turn.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                rows.append([float(v) for v in line.split()])
    base = (2 / np.pi) ** 2
    for r in rows:
        y = oracle_mod.rope(np.array([r[1:5]]), [int(r[0])], base=base, layout="half")[0]
        np.testing.assert_allclose(y, r[5:9], rtol=1e-15, atol=1e-15)


def test_is_the_interleaved_rotation_of_permuted_columns(oracle_mod):
    g = np.random.default_rng(3)
    x = g.standard_normal((7, 64))
    pos = g.integers(0, 100000, size=7).astype(np.int32)
    half = oracle_mod.rope(x, pos, layout="half")
    inter = oracle_mod.rope(_interleave(x), pos)
    np.testing.assert_array_equal(half, _deinterleave(inter))
    assert not np.allclose(half, oracle_mod.rope(x, pos))  # a different pairing


def test_pair_norms_and_relative_position(oracle_mod):
    g = np.random.default_rng(4)
    d = 32
    q, k = g.standard_normal((2, d))
    yq = oracle_mod.rope(np.array([q]), [5], layout="half")[0]
    np.testing.assert_allclose(np.hypot(yq[: d // 2], yq[d // 2:]), np.hypot(q[: d // 2], q[d // 2:]), rtol=1e-14)
    dots = []
    for m, n in ((7, 3), (104, 100), (1004, 1000)):
        a = oracle_mod.rope(np.array([q]), [m], layout="half")[0]
        b = oracle_mod.rope(np.array([k]), [n], layout="half")[0]
        dots.append(a @ b)
    np.testing.assert_allclose(dots, dots[0], rtol=1e-11)


def test_hash_matches_permuted_interleaved_hash(oracle_mod):
    """Hashing with the half pairing = hashing the interleaved-permuted rows with the same
    permutation applied to the hyperplanes' columns (the projection is a sum over columns)."""
    wl = workloads.WORKLOADS["tiny"].scaled(n_ref=40, n_tgt=40, d=128)
    emb, pos, _ = workloads.prompt_rows(wl)
    R = workloads.hyperplanes(wl)
    ch, ph = oracle_mod.hash_codes(emb, pos, R, layout="half")
    ci, pi = oracle_mod.hash_codes(np.ascontiguousarray(_interleave(emb)), pos, np.ascontiguousarray(_interleave(R)))
    np.testing.assert_allclose(ph, pi, rtol=1e-6, atol=1e-9)
    band = np.abs(pi) < 1e-9
    bits_h = np.unpackbits(ch.view(np.uint8), axis=1, bitorder="little").astype(bool)
    bits_i = np.unpackbits(ci.view(np.uint8), axis=1, bitorder="little").astype(bool)
    assert np.all((bits_h == bits_i) | band)
