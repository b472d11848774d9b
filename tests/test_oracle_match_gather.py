"""Pins of the oracle's Hamming nearest-neighbour search and KV rearrangement (SemShareKV Sec. 3.3)."""
import os

import numpy as np
import pytest

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _brute_force_match(tgt, ref, nbits):
    """Bit by bit on unpacked codes, exhaustive, first minimum kept."""
    tb = np.unpackbits(tgt.view(np.uint8), axis=1, bitorder="little")[:, :nbits]
    rb = np.unpackbits(ref.view(np.uint8), axis=1, bitorder="little")[:, :nbits]
    idx, dist = [], []
    for t in range(tb.shape[0]):
        best, bj = None, None
        for j in range(rb.shape[0]):
            h = 0
            for q in range(nbits):
                h += int(tb[t, q] != rb[j, q])
            if best is None or h < best:
                best, bj = h, j
        idx.append(bj)
        dist.append(best)
    return np.array(idx), np.array(dist)


def test_golden_small(oracle_mod):
    ref, rows = None, []
    with open(os.path.join(GOLDEN, "match_small.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            parts = line.split()
            if parts[0] == "ref":
                ref = np.array([[int(h, 16)] for h in parts[1:]], dtype=np.uint32)
            else:
                rows.append((int(parts[0], 16), int(parts[1]), int(parts[2])))
    tgt = np.array([[r[0]] for r in rows], dtype=np.uint32)
    idx, dist = oracle_mod.match(tgt, ref)
    np.testing.assert_array_equal(idx, [r[1] for r in rows])
    np.testing.assert_array_equal(dist, [r[2] for r in rows])


@pytest.mark.parametrize("nbits,n_t,n_r", [(32, 40, 64), (64, 33, 17), (256, 12, 64)])
def test_brute_force(oracle_mod, nbits, n_t, n_r):
    g = np.random.default_rng(nbits)
    ref = workloads.random_codes(n_r, nbits, seed=nbits, stream=1)
    tgt = workloads.random_codes(n_t, nbits, seed=nbits, stream=2)
    # plant near-duplicates and exact duplicates so ties occur
    tgt[: n_t // 3] = ref[g.integers(0, n_r, size=n_t // 3)]
    ref[n_r // 2] = ref[1]
    tgt[-1] ^= np.uint32(1)
    idx, dist = oracle_mod.match(tgt, ref, nbits)
    bi, bd = _brute_force_match(tgt, ref, nbits)
    np.testing.assert_array_equal(idx, bi)
    np.testing.assert_array_equal(dist, bd)


def test_distance_axioms(oracle_mod):
    for nbits in (32, 64, 128, 256):
        c = workloads.random_codes(50, nbits, seed=3)
        for i in range(0, 50, 7):
            assert oracle_mod.hamming(c[i], c[i]) == 0
            assert oracle_mod.hamming(c[i], ~c[i]) == nbits
            for j in range(0, 50, 11):
                h = oracle_mod.hamming(c[i], c[j])
                assert h == oracle_mod.hamming(c[j], c[i])
                assert 0 <= h <= nbits


def test_identical_prompts_map_to_themselves(oracle_mod):
    c = workloads.random_codes(300, 128, seed=4)
    c[200] = c[17]  # a duplicate code resolves to its first occurrence
    idx, dist = oracle_mod.match(c, c)
    want = np.arange(300)
    want[200] = 17
    np.testing.assert_array_equal(idx, want)
    assert (dist == 0).all()


def test_all_equal_codes_tie_to_zero(oracle_mod):
    ref = np.full((77, 2), 0x12345678, dtype=np.uint32)
    tgt = workloads.random_codes(9, 64, seed=5)
    idx, dist = oracle_mod.match(tgt, ref)
    assert (idx == 0).all()


def test_pool_argmin_is_min_over_members(oracle_mod):
    pool = workloads.random_codes(4 * 50, 64, seed=6)
    tgt = workloads.random_codes(30, 64, seed=7)
    idx, dist = oracle_mod.match(tgt, pool)
    best = np.full(30, 1 << 30)
    bidx = np.full(30, -1)
    for s in range(4):
        i, d = oracle_mod.match(tgt, pool[s * 50:(s + 1) * 50])
        better = d < best
        best = np.where(better, d, best)
        bidx = np.where(better, i + s * 50, bidx)
    np.testing.assert_array_equal(idx, bidx)
    np.testing.assert_array_equal(dist, best)


# ---- gather --------------------------------------------------------------------------------

def test_gather_golden_small(oracle_mod):
    K = np.zeros((1, 2, 3, 2), dtype=np.uint16)
    for h in range(2):
        for r in range(3):
            K[0, h, r] = (10 * h + 2 * r, 10 * h + 2 * r + 1)
    V = K + 100
    exp = {}
    with open(os.path.join(GOLDEN, "gather_small.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                p = line.split()
                exp[(p[0], p[1] if p[0] != "idx" else "")] = [int(v) for v in p[1 if p[0] == "idx" else 2:]]
    idx = np.array(exp[("idx", "")], dtype=np.int32)
    ok, ov, bad = oracle_mod.gather_kv(K, V, idx)
    assert bad == 0
    for h in range(2):
        np.testing.assert_array_equal(ok[0, 0, h].reshape(-1), exp[("outK", f"h{h}")])
        np.testing.assert_array_equal(ov[0, 0, h].reshape(-1), exp[("outV", f"h{h}")])


def test_gather_per_element_loop(oracle_mod):
    g = np.random.default_rng(11)
    L, H, hd = 3, 2, 8
    segs = [g.integers(0, 65536, size=(L, H, n, hd), dtype=np.uint16) for n in (5, 0, 7, 3)]
    segv = [g.integers(0, 65536, size=s.shape, dtype=np.uint16) for s in segs]
    offs = np.cumsum([0] + [s.shape[2] for s in segs])
    idx = g.integers(0, offs[-1], size=(2, 9)).astype(np.int32)
    ok, ov, bad = oracle_mod.gather_kv(segs, segv, idx)
    assert bad == 0
    for b in range(2):
        for l in range(L):
            for h in range(H):
                for t in range(9):
                    r = int(idx[b, t])
                    s = int(np.searchsorted(offs, r, side="right") - 1)
                    for e in range(hd):
                        assert ok[b, l, h, t, e] == segs[s][l, h, r - offs[s], e]
                        assert ov[b, l, h, t, e] == segv[s][l, h, r - offs[s], e]


def test_gather_identity_and_permutation(oracle_mod):
    g = np.random.default_rng(12)
    K = g.integers(0, 65536, size=(4, 2, 50, 16), dtype=np.uint16)
    V = g.integers(0, 65536, size=(4, 2, 50, 16), dtype=np.uint16)
    ok, ov, _ = oracle_mod.gather_kv(K, V, np.arange(50, dtype=np.int32))
    np.testing.assert_array_equal(ok[0], K)
    np.testing.assert_array_equal(ov[0], V)
    perm = g.permutation(50).astype(np.int32)
    ok, ov, _ = oracle_mod.gather_kv(K, V, perm)
    for l in range(4):
        for h in range(2):
            a = sorted(map(bytes, ok[0, l, h]))
            b = sorted(map(bytes, K[l, h]))
            assert a == b


def test_gather_keeps_special_bf16_patterns(oracle_mod):
    special = np.array([0x7FC1, 0xFFFF, 0x8000, 0x0001, 0x7F80, 0xFF80, 0x807F, 0x7FA5], dtype=np.uint16)
    K = np.tile(special, (1, 1, 4, 1))
    V = K[..., ::-1].copy()
    ok, ov, _ = oracle_mod.gather_kv(K, V, np.array([3, 2, 1, 0, 0], dtype=np.int32))
    for t, r in enumerate([3, 2, 1, 0, 0]):
        assert ok[0, 0, 0, t].tobytes() == K[0, 0, r].tobytes()
        assert ov[0, 0, 0, t].tobytes() == V[0, 0, r].tobytes()


def test_gather_out_of_range_rows_untouched(oracle_mod):
    K = np.ones((1, 1, 4, 8), dtype=np.uint16)
    V = K * 2
    out_k = np.full((1, 1, 1, 3, 8), 7, dtype=np.uint16)
    out_v = np.full((1, 1, 1, 3, 8), 9, dtype=np.uint16)
    ok, ov, bad = oracle_mod.gather_kv(K, V, np.array([1, 4, -1], dtype=np.int32), out_k, out_v)
    assert bad == 2
    assert (ok[0, 0, 0, 0] == 1).all() and (ok[0, 0, 0, 1:] == 7).all()
    assert (ov[0, 0, 0, 0] == 2).all() and (ov[0, 0, 0, 1:] == 9).all()


def test_thread_count_does_not_change_results(oracle_mod):
    """The CPU baseline times the oracle on one thread and on all cores: same results either way."""
    g = np.random.default_rng(8)
    t = g.integers(0, 2**32, size=(300, 4), dtype=np.uint64).astype(np.uint32)
    r = g.integers(0, 2**32, size=(257, 4), dtype=np.uint64).astype(np.uint32)
    prev = oracle_mod.set_threads(1)
    try:
        a = oracle_mod.match(t, r)
    finally:
        oracle_mod.set_threads(prev)
    b = oracle_mod.match(t, r)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])
