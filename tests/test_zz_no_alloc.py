"""semshare_match_static: the Hamming search for callers that cannot allocate device memory
(for example code hosted inside a framework that owns the whole device memory pool and forbids
allocations, or a serving loop that must not allocate on its hot path).  It uses a fixed
scratch array inside the library instead of a caller workspace.

Its results must equal semshare_match's, bit for bit, on two calls in a row, and both must
equal the CPU oracle's exhaustive search on the same codes: the scratch array keeps the first
call's keys, so the second call (a different, smaller problem) also checks that each call
resets what it uses.  Sizes beyond the array's capacity must be refused before anything is
enqueued.  This file is named to be collected last."""
import numpy as np
import pytest

import oracle
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


@pytest.fixture(scope="module", autouse=True)
def _oracle_built():
    oracle.build()


def _codes(n, nbits, seed, stream):
    return torch.from_numpy(workloads.random_codes(n, nbits, seed=seed, stream=stream).view(np.int32)).cuda()


def test_static_scratch_match_equals_workspace_match_on_two_calls(ss):
    for n_tgt, n_ref, nbits, seed in [(3000, 2000, 256, 11), (1200, 700, 64, 12)]:
        ref = _codes(n_ref, nbits, seed, 1)
        tgt = _codes(n_tgt, nbits, seed, 2)
        tgt[: n_tgt // 4] = ref[torch.randint(0, n_ref, (n_tgt // 4,), device="cuda")]  # exact matches
        ref[n_ref - 1] = ref[3]                                                        # a tie
        want_idx, want_dist = ss.semshare_match(tgt, ref)
        idx = torch.full((n_tgt,), -7, dtype=torch.int32, device="cuda")
        dist = torch.full((n_tgt,), -7, dtype=torch.int32, device="cuda")
        ss.semshare_match_static(tgt, ref, idx=idx, dist=dist)
        torch.cuda.synchronize()
        assert torch.equal(idx, want_idx), f"idx differs on the {n_tgt}-target call"
        assert torch.equal(dist, want_dist), f"dist differs on the {n_tgt}-target call"
        # both against the oracle's exhaustive scan (ties to the lowest reference index)
        oi, od = oracle.match(tgt.cpu().numpy().view(np.uint32), ref.cpu().numpy().view(np.uint32))
        np.testing.assert_array_equal(idx.cpu().numpy(), oi, err_msg=f"{n_tgt}-target call vs the oracle")
        np.testing.assert_array_equal(dist.cpu().numpy(), od, err_msg=f"{n_tgt}-target call vs the oracle")


def test_static_scratch_match_refuses_sizes_beyond_capacity(ss):
    cap = ss.MATCH_STATIC_MAX_TARGETS
    ref = _codes(10, 64, 13, 1)
    tgt = torch.zeros((cap + 1, 2), dtype=torch.int32, device="cuda")
    with pytest.raises(ss.SemshareError) as e:
        ss.semshare_match_static(tgt, ref)
    assert e.value.status == 6  # SEMSHARE_ETOOLARGE
