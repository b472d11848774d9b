"""Parity of semshare_retrieve (reference retrieval, Sec. 3.2; similarity of App. A.3; the 0.8
threshold of Sec. 4.4) with the oracle: per-candidate mean nearest distances and similarities
bit-exact (both sides divide the same integer sum in fp64), the chosen candidate and the
threshold decision identical, and the per-token match against the chosen candidate identical
to the oracle's 1-NN search over that candidate's rows."""
import numpy as np
import pytest

import workloads
from gpu_helpers import bf16_dev, check_hash, codes_host, emb_dev

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ss():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_24832_gb300 as ss

    ss.load()
    return ss


@pytest.fixture(scope="module")
def orc():
    import oracle

    oracle.build()
    return oracle


def _planted(nbits, n_tgt, sizes, seed):
    """Random pool and target codes; candidate 1 (and an exact copy of it, last) holds copies of
    target rows with a few flipped bits, so its distances are small and a tie is planted."""
    g = np.random.default_rng(seed)
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    pool = workloads.random_codes(int(offs[-1]), nbits, seed=seed, stream=1)
    tgt = workloads.random_codes(n_tgt, nbits, seed=seed, stream=2)
    if len(sizes) > 1:
        n1 = sizes[1]
        rows = tgt[g.integers(0, n_tgt, size=n1)].copy()
        flips = g.integers(0, nbits, size=(n1, 2))
        for i in range(n1):
            for b in flips[i]:
                rows[i, b // 32] ^= np.uint32(1 << (b % 32))
        pool[offs[1]:offs[2]] = rows
        if sizes[-1] == n1 and len(sizes) > 2:
            pool[offs[-2]:offs[-1]] = rows
    return tgt, pool, offs


def _check(ss, orc, tgt, pool, offs, nbits, **kw):
    dev = torch.device("cuda")
    t = torch.from_numpy(tgt.view(np.int32)).to(dev)
    p = torch.from_numpy(pool.view(np.int32)).to(dev)
    flag = ss.new_err_flag(dev)
    res = ss.semshare_retrieve(t, p, offs, err_flag=flag, nbits=nbits, **kw)
    torch.cuda.synchronize()
    ss.check_flag(flag, "retrieve")
    mean, sim, best, applies = orc.retrieve(tgt, pool, offs, nbits, **kw)
    np.testing.assert_array_equal(res.mean_dist.cpu().numpy(), mean)
    np.testing.assert_array_equal(res.similarity.cpu().numpy(), sim)
    assert int(res.best.item()) == best and bool(res.applies.item()) == applies
    oi, od = orc.match(tgt, pool[offs[best]:offs[best + 1]], nbits)
    np.testing.assert_array_equal(res.idx.cpu().numpy(), oi + offs[best])
    np.testing.assert_array_equal(res.dist.cpu().numpy(), od)
    return res, (mean, sim, best, applies)


CASES = [
    # boundaries inside 32-column chunks, a one-row candidate, chunk- and tile-sized ones
    (64, 300, [100, 37, 1, 31, 32, 33, 256, 200]),
    # boundaries exactly on 256-column tiles, a ragged target block
    (256, 129, [256, 256, 1, 255, 513, 256]),
    # many short candidates, several per chunk
    (128, 1000, [5] * 200),
    # the maximum number of candidates, one row each: a boundary at every column
    (32, 77, [1] * 256),
    # nbits not a multiple of the 128-bit chunk; candidates spanning several tiles
    (96, 200, [700, 300, 1100]),
    # a single candidate
    (160, 513, [999]),
]


@pytest.mark.parametrize("nbits,n_tgt,sizes", CASES)
def test_retrieve_random_codes(ss, orc, nbits, n_tgt, sizes):
    _check(ss, orc, *_planted(nbits, n_tgt, sizes, seed=nbits + n_tgt), nbits=nbits)


def test_retrieve_threshold_and_scale(ss, orc):
    tgt, pool, offs = _planted(64, 150, [40, 60, 60], seed=11)
    for kw in (dict(max_dist=64.0, threshold=0.5), dict(max_dist=2.5, threshold=0.0), dict(threshold=1.0)):
        _check(ss, orc, tgt, pool, offs, 64, **kw)


def test_retrieve_repeatable(ss, orc):
    """Two calls in a row through the same workspace give identical outputs."""
    tgt, pool, offs = _planted(256, 700, [300, 500, 64, 500], seed=5)
    dev = torch.device("cuda")
    t = torch.from_numpy(tgt.view(np.int32)).to(dev)
    p = torch.from_numpy(pool.view(np.int32)).to(dev)
    ws = torch.empty(ss.semshare_retrieve_workspace_size(700, int(offs[-1]), 4, 256), dtype=torch.uint8, device=dev)
    # max_dist 256: the similarities stay apart from 0 (with 30 every 256-bit mean here clips to 0)
    r1 = ss.semshare_retrieve(t, p, offs, workspace=ws, max_dist=256.0)
    r2 = ss.semshare_retrieve(t, p, offs, workspace=ws, max_dist=256.0)
    torch.cuda.synchronize()
    for a, b in zip(r1, r2):
        assert torch.equal(a, b)
    sim = r1.similarity.cpu().numpy()
    assert sim[1] == sim[3] and sim[1] > max(sim[0], sim[2])
    assert int(r1.best.item()) == 1  # the tie between candidates 1 and 3 goes to the lower index
    _, osim, obest, _ = orc.retrieve(tgt, pool, offs, 256, max_dist=256.0)
    np.testing.assert_array_equal(sim, osim)
    assert obest == 1


def test_retrieve_workload_full_size(ss, orc):
    """16 stored prompts of 4096 tokens and a rewritten target: hash every row without rotary
    encoding, retrieve, and compare with the oracle everywhere (codes on sampled rows)."""
    wl = workloads.RETRIEVAL_WORKLOADS["retrieve-16x4096"]
    emb, _, src = workloads.prompt_rows(wl)
    dev = torch.device("cuda")
    n_rows = emb.shape[0]
    zeros = np.zeros(n_rows, dtype=np.int32)
    R = workloads.hyperplanes(wl)
    table = ss.semshare_rope_table(wl.d, 10000.0, device=dev)
    proj = torch.empty((n_rows, wl.nbits), dtype=torch.float32, device=dev)
    flag = ss.new_err_flag(dev)
    codes = ss.semshare_hash(emb_dev(emb, dev), table, bf16_dev(R, dev), torch.from_numpy(zeros).to(dev),
                             proj_out=proj, err_flag=flag)
    offs = [s * wl.seg_len for s in range(wl.n_seg + 1)]
    res = ss.semshare_retrieve(codes[wl.n_ref:], codes[:wl.n_ref], offs, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, wl.name)

    g = np.random.default_rng(23)
    rows = np.sort(np.concatenate([g.choice(n_rows, 256, replace=False), [0, wl.n_ref - 1, wl.n_ref, n_rows - 1]]))
    gc = codes_host(codes)
    oc, op = orc.hash_codes(emb[rows], zeros[rows], R)
    check_hash(gc, proj.cpu().numpy(), oc, op, rows=rows)

    mean, sim, best, applies = orc.retrieve(gc[wl.n_ref:], gc[:wl.n_ref], offs, wl.nbits)
    np.testing.assert_array_equal(res.mean_dist.cpu().numpy(), mean)
    np.testing.assert_array_equal(res.similarity.cpu().numpy(), sim)
    assert int(res.best.item()) == best == workloads.retrieval_member(wl)
    assert bool(res.applies.item()) == applies
    oi, od = orc.match(gc[wl.n_ref:], gc[offs[best]:offs[best + 1]])
    np.testing.assert_array_equal(res.idx.cpu().numpy(), oi + offs[best])
    np.testing.assert_array_equal(res.dist.cpu().numpy(), od)
    copied = src[0] >= 0
    recall = float((res.idx.cpu().numpy()[copied] == src[0][copied]).mean())
    print(f"{wl.name}: best {best} similarity {sim[best]:.4f} (others <= {np.delete(sim, best).max():.4f}), "
          f"applies {applies}, recall {recall:.3f}")
