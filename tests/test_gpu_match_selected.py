"""Parity of semshare_match_tc_selected (token matching, Sec. 3.3, against the candidate that a
device value names -- the retrieval's choice, Sec. 3.2) with the oracle: idx equals the oracle's
1-NN over that candidate's rows shifted to pool rows, dist is identical, a shorter candidate's
tail is masked, and an invalid choice is flagged with every output -1."""
import numpy as np
import pytest

import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ss():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_24832_gb300 as ss

    ss.load()
    return ss


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()


def _expect(orc, tgt, pool, offs, c, nbits):
    idx, dist = orc.match(tgt, pool[offs[c]:offs[c + 1]], nbits)
    return idx + offs[c], dist


@pytest.mark.parametrize("nbits", [64, 128, 256])
def test_selected_parity_every_candidate(ss, oracle_mod, nbits):
    sizes = [300, 1, 513, 256, 77]  # several tiles, a ragged tail, a one-row candidate
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    tgt = workloads.random_codes(333, nbits, seed=nbits, stream=1)
    pool = workloads.random_codes(int(offs[-1]), nbits, seed=nbits, stream=2)
    pool[offs[2]:offs[2] + 40] = tgt[:40]  # exact copies: distance 0
    pool[offs[2] + 41] = tgt[5]            # a tie, resolved to the lower row
    t, p = _dev(tgt), _dev(pool)
    best = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(ss.semshare_match_tc_selected_workspace_size(len(tgt), offs, nbits), dtype=torch.uint8,
                     device="cuda")
    for c in range(len(sizes)):
        best.fill_(c)
        flag = ss.new_err_flag()
        idx, dist = ss.semshare_match_tc_selected(t, p, offs, best, workspace=ws, err_flag=flag, nbits=nbits)
        torch.cuda.synchronize()
        assert int(flag.item()) == 0
        ei, ed = _expect(oracle_mod, tgt, pool, offs, c, nbits)
        assert np.array_equal(idx.cpu().numpy(), ei), f"candidate {c}"
        assert np.array_equal(dist.cpu().numpy(), ed), f"candidate {c}"


def test_short_candidate_tail_is_masked(ss, oracle_mod):
    # every target is at distance nbits from the short candidate's rows; the longest candidate
    # sizes the search, and a zero (unmasked) padding row would sit at nbits/2 and win
    nbits = 128
    x = workloads.random_codes(1, nbits, seed=3)[0]
    tgt = np.tile(x, (200, 1))
    sizes = [3, 600]
    offs = np.array([0, 3, 603], dtype=np.int64)
    pool = workloads.random_codes(603, nbits, seed=4)
    pool[:3] = ~x
    idx, dist = ss.semshare_match_tc_selected(_dev(tgt), _dev(pool), offs, torch.zeros(1, dtype=torch.int32,
                                                                                        device="cuda"))
    torch.cuda.synchronize()
    assert (idx.cpu().numpy() == 0).all() and (dist.cpu().numpy() == nbits).all()
    ei, ed = _expect(oracle_mod, tgt, pool, offs, 0, nbits)
    assert np.array_equal(idx.cpu().numpy(), ei) and np.array_equal(dist.cpu().numpy(), ed)


@pytest.mark.parametrize("bad", [-1, 2, 1 << 30])
def test_invalid_choice_flagged(ss, bad):
    nbits = 64
    offs = np.array([0, 100, 250], dtype=np.int64)
    tgt = workloads.random_codes(70, nbits, seed=5)
    pool = workloads.random_codes(250, nbits, seed=6)
    flag = ss.new_err_flag()
    idx, dist = ss.semshare_match_tc_selected(_dev(tgt), _dev(pool), offs,
                                              torch.full((1,), bad, dtype=torch.int32, device="cuda"), err_flag=flag)
    torch.cuda.synchronize()
    assert int(flag.item()) & ss.FLAG_INDEX
    assert (idx.cpu().numpy() == -1).all() and (dist.cpu().numpy() == -1).all()


def test_retrieve_then_match_then_gather_without_sync(ss, oracle_mod):
    """The whole reuse path enqueued back to back: retrieval picks the candidate on the device,
    the selected match reads it there, the gather runs over the pool's segments with pool rows."""
    nbits = 128
    n_cand, seg = 8, 320
    offs = np.arange(n_cand + 1, dtype=np.int64) * seg
    pool = workloads.random_codes(n_cand * seg, nbits, seed=7)
    g = np.random.default_rng(8)
    tgt = pool[offs[5]:offs[5] + 300].copy()      # the target rewrites candidate 5
    flips = g.integers(0, nbits, size=(300, 3))
    for i in range(300):
        for b in flips[i]:
            tgt[i, b // 32] ^= np.uint32(1 << (b % 32))
    t, p = _dev(tgt), _dev(pool)
    res = ss.semshare_retrieve(t, p, offs, want_match=False)
    idx, dist = ss.semshare_match_tc_selected(t, p, offs, res.best)
    L, H, hd = 2, 2, 64
    ks = [torch.randn((L, H, seg, hd), device="cuda").to(torch.bfloat16) for _ in range(n_cand)]
    vs = [torch.randn((L, H, seg, hd), device="cuda").to(torch.bfloat16) for _ in range(n_cand)]
    out_k, out_v = ss.semshare_gather_kv(ks, vs, idx)
    torch.cuda.synchronize()
    assert int(res.best.item()) == 5
    ei, ed = _expect(oracle_mod, tgt, pool, offs, 5, nbits)
    assert np.array_equal(idx.cpu().numpy(), ei) and np.array_equal(dist.cpu().numpy(), ed)
    want_k = torch.stack([ks[5][:, :, int(r) - int(offs[5])] for r in ei], dim=2)
    assert torch.equal(out_k[0].view(torch.int16), want_k.view(torch.int16))


def test_selected_with_the_maximum_of_256_candidates(ss, oracle_mod):
    """256 one- to three-row candidates (the most a pool may have), each chosen in turn for a few."""
    nbits = 32
    g = np.random.default_rng(21)
    sizes = g.integers(1, 4, size=256)
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    pool = workloads.random_codes(int(offs[-1]), nbits, seed=22)
    tgt = workloads.random_codes(129, nbits, seed=23)
    t, p = _dev(tgt), _dev(pool)
    best = torch.zeros(1, dtype=torch.int32, device="cuda")
    for c in (0, 1, 127, 200, 255):
        best.fill_(c)
        idx, dist = ss.semshare_match_tc_selected(t, p, offs, best, nbits=nbits)
        torch.cuda.synchronize()
        ei, ed = _expect(oracle_mod, tgt, pool, offs, c, nbits)
        assert np.array_equal(idx.cpu().numpy(), ei) and np.array_equal(dist.cpu().numpy(), ed), c
