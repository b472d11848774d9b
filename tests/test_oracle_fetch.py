"""Pins of the oracle's selected-row load (SemShareKV Sec. 3.2: the retrieved reference prompt's
KV cache is brought onto the GPU; Sec. 3.3: the rearrangement reads only the rows the match
selects).  Every selected row is copied, every other row is left alone, and the rearrangement of
the loaded copy equals the rearrangement of the source."""
import numpy as np

import workloads


def _segs(sizes, L=2, H=3, hd=8, seed=4):
    g = np.random.default_rng(seed)
    ks = [workloads.f32_to_bf16_bits(g.standard_normal((L, H, n, hd), dtype=np.float32)) for n in sizes]
    vs = [workloads.f32_to_bf16_bits(g.standard_normal((L, H, n, hd), dtype=np.float32)) for n in sizes]
    return ks, vs


def test_brute_force_rows(oracle_mod):
    # Definition by Python loops: row r of every (l, h) plane is copied iff r appears in idx.
    ks, vs = _segs([7])
    k, v = ks[0], vs[0]
    idx = [5, 0, 5, 5, 2]
    sent = np.full_like(k, 0xBEEF)
    dk, dv, bad = oracle_mod.fetch_rows(k, v, idx, sent.copy(), sent.copy())
    assert bad == 0
    L, H, N, _ = k.shape
    for l in range(L):
        for h in range(H):
            for r in range(N):
                if r in idx:
                    assert (dk[l, h, r] == k[l, h, r]).all() and (dv[l, h, r] == v[l, h, r]).all()
                else:
                    assert (dk[l, h, r] == 0xBEEF).all() and (dv[l, h, r] == 0xBEEF).all()


def test_segments_receive_their_own_rows(oracle_mod):
    # Global row r of segment s lands at local row r - offset[s] of that segment's copy only.
    ks, vs = _segs([4, 0, 6, 3])
    idx = [0, 4, 9, 12, 9, 3]  # offsets 0, 4, 4, 10
    dk, dv, bad = oracle_mod.fetch_rows(ks, vs, idx)
    assert bad == 0
    want = {0: [0, 3], 1: [], 2: [0, 5], 3: [2]}
    for s, rows in want.items():
        other = [r for r in range(ks[s].shape[2]) if r not in rows]
        np.testing.assert_array_equal(dk[s][:, :, rows], ks[s][:, :, rows])
        np.testing.assert_array_equal(dv[s][:, :, rows], vs[s][:, :, rows])
        assert not dk[s][:, :, other].any() and not dv[s][:, :, other].any()


def test_rearrangement_of_the_copy_equals_the_source(oracle_mod):
    ks, vs = _segs([30, 50, 20], seed=9)
    g = np.random.default_rng(2)
    idx = g.integers(0, 100, size=(2, 64)).astype(np.int32)
    dk, dv, bad = oracle_mod.fetch_rows(ks, vs, idx)
    assert bad == 0
    want_k, want_v, _ = oracle_mod.gather_kv(ks, vs, idx)
    got_k, got_v, _ = oracle_mod.gather_kv(dk, dv, idx)
    np.testing.assert_array_equal(got_k, want_k)
    np.testing.assert_array_equal(got_v, want_v)


def test_out_of_range_and_empty(oracle_mod):
    ks, vs = _segs([5, 5])
    dk, dv, bad = oracle_mod.fetch_rows(ks, vs, [-1, 10, 2**31 - 1, 7])
    assert bad == 3
    assert not dk[0].any() and not dv[0].any()
    np.testing.assert_array_equal(dk[1][:, :, 2], ks[1][:, :, 2])
    ek, ev, bad = oracle_mod.fetch_rows(ks, vs, np.zeros(0, dtype=np.int32))
    assert bad == 0 and not any(a.any() for a in ek + ev)
