"""Pins of the oracle's reference retrieval (SemShareKV Sec. 3.2; App. A.3: Similarity =
clip(1 - LSH_dist/30, 0, 1); Sec. 4.4: reuse applies above 0.8).  LSH_dist of a candidate is
read as the mean over the target's tokens of each token's nearest Hamming distance to the
candidate."""
import os
from fractions import Fraction

import numpy as np
import pytest

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _brute_force(tgt, pool, offs, nbits, dmax=30, threshold=Fraction(4, 5)):
    """Unpacked bits, exhaustive, exact rational arithmetic; first maximum kept."""
    tb = np.unpackbits(tgt.view(np.uint8), axis=1, bitorder="little")[:, :nbits]
    pb = np.unpackbits(pool.view(np.uint8), axis=1, bitorder="little")[:, :nbits]
    means, sims = [], []
    for c in range(len(offs) - 1):
        total = 0
        for t in range(tb.shape[0]):
            total += min(int((tb[t] != pb[j]).sum()) for j in range(offs[c], offs[c + 1]))
        m = Fraction(total, tb.shape[0])
        means.append(m)
        sims.append(min(max(1 - m / dmax, Fraction(0)), Fraction(1)))
    best = max(range(len(sims)), key=lambda c: (sims[c], -c))
    return means, sims, best, sims[best] > threshold


def test_golden_small(oracle_mod):
    fields = {}
    with open(os.path.join(GOLDEN, "retrieve_small.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                k, *v = line.split()
                fields[k] = v
    tgt = np.array([[int(h, 16)] for h in fields["target"]], dtype=np.uint32)
    pool = np.array([[int(h, 16)] for h in fields["pool"]], dtype=np.uint32)
    offs = [int(o) for o in fields["offsets"]]
    mean, sim, best, applies = oracle_mod.retrieve(tgt, pool, offs, 32)
    np.testing.assert_array_equal(mean, [float(m) for m in fields["mean"]])
    np.testing.assert_allclose(sim, [13 / 15, 1.0, 1 / 15, 0.6], rtol=0, atol=1e-15)
    assert best == int(fields["best"][0]) and applies == bool(int(fields["applies"][0]))
    # the comment's variant: the perfect candidate removed, the 13/15 one still applies
    keep = np.r_[0:2, 4:7]
    mean2, sim2, best2, applies2 = oracle_mod.retrieve(tgt, pool[keep], [0, 2, 3, 5], 32)
    np.testing.assert_array_equal(mean2, [4, 28, 12])
    assert best2 == 0 and applies2


@pytest.mark.parametrize("nbits,n_t,sizes", [(32, 9, [3, 1, 7, 2]), (64, 13, [5, 9, 1]), (256, 6, [4, 4, 11])])
def test_brute_force(oracle_mod, nbits, n_t, sizes):
    g = np.random.default_rng(nbits + n_t)
    offs = np.concatenate([[0], np.cumsum(sizes)])
    pool = workloads.random_codes(int(offs[-1]), nbits, seed=nbits, stream=3)
    tgt = workloads.random_codes(n_t, nbits, seed=nbits, stream=4)
    # candidate 1 gets copies of some target rows, so distances span 0..nbits/2
    take = g.choice(n_t, size=min(n_t, sizes[1]), replace=False)
    pool[offs[1]:offs[1] + len(take)] = tgt[take]
    mean, sim, best, applies = oracle_mod.retrieve(tgt, pool, offs, nbits)
    bm, bs, bb, ba = _brute_force(tgt, pool, list(offs), nbits)
    np.testing.assert_array_equal(mean, [float(m) for m in bm])
    # 1 - m/30 is rounded twice in fp64 (division, subtraction): within two half-ulps of 1
    np.testing.assert_allclose(sim, [float(s) for s in bs], rtol=0, atol=2.3e-16)
    assert best == bb and applies == ba


def test_identical_prompt_and_ties(oracle_mod):
    nbits = 64
    tgt = workloads.random_codes(40, nbits, seed=5, stream=1)
    other = workloads.random_codes(30, nbits, seed=5, stream=2)
    # candidates: unrelated, the target itself (shuffled), a copy of the target (tie), unrelated
    perm = np.random.default_rng(0).permutation(40)
    pool = np.concatenate([other, tgt[perm], tgt, other[:5]])
    offs = [0, 30, 70, 110, 115]
    mean, sim, best, applies = oracle_mod.retrieve(tgt, pool, offs, nbits)
    assert mean[1] == 0.0 and mean[2] == 0.0 and sim[1] == 1.0 and sim[2] == 1.0
    assert best == 1 and applies  # tie between 1 and 2 goes to the lower index
    # unrelated random 64-bit codes sit ~20 bits from their nearest of 30 rows: sim < 0.8
    assert sim[0] < 0.8 and sim[3] <= sim[0]


def test_clip_and_threshold(oracle_mod):
    nbits = 64
    tgt = workloads.random_codes(8, nbits, seed=9, stream=1)
    # a target of one repeated row against its complement: distance 64 > 30, similarity clipped to 0
    rep = np.repeat(tgt[:1], 8, axis=0)
    mean, sim, best, applies = oracle_mod.retrieve(rep, ~rep[:3], [0, 3], nbits)
    assert mean[0] == 64.0 and sim[0] == 0.0 and best == 0 and not applies
    # one flipped bit per target row: mean 1, similarity 1 - 1/30; the threshold decides
    one = tgt.copy()
    one[:, 0] ^= np.uint32(1)
    _, sim1, _, app = oracle_mod.retrieve(tgt, one, [0, 8], nbits)
    assert sim1[0] == 1.0 - 1.0 / 30.0 and app
    _, _, _, app_hi = oracle_mod.retrieve(tgt, one, [0, 8], nbits, threshold=1.0 - 1.0 / 30.0)
    assert not app_hi  # strictly above the threshold
    # mean 6 gives similarity exactly 0.8: not above 0.8
    six = tgt.copy()
    six[:, 0] ^= np.uint32(0x3F)
    _, sim6, _, app6 = oracle_mod.retrieve(tgt, six, [0, 8], nbits)
    assert sim6[0] == 1.0 - 6.0 / 30.0 and not app6


def test_single_candidate_matches_search(oracle_mod):
    """With one candidate the summed distance is the sum of the 1-NN distances of Sec. 3.3."""
    nbits = 128
    ref = workloads.random_codes(50, nbits, seed=3, stream=1)
    tgt = workloads.random_codes(20, nbits, seed=3, stream=2)
    tgt[:7] = ref[10:17]
    mean, _, _, _ = oracle_mod.retrieve(tgt, ref, [0, 50], nbits)
    _, dist = oracle_mod.match(tgt, ref, nbits)
    assert mean[0] * 20 == dist.sum()
