"""The path captured in a CUDA graph: every call enqueues only kernels on the caller's stream
(no allocation, no host synchronisation, kernels chained as programmatic dependents), so a whole
step -- hash, match, gather; or hash, retrieval, hash, selected match, gather -- records into one
graph, and replaying it gives the bits of the eager step."""
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


def _outputs(prob):
    return [t.detach().clone() for t in (prob.codes, prob.idx, prob.dist, prob.out_k.view(torch.int16),
                                         prob.out_v.view(torch.int16))]


def _scramble(prob):
    for t in (prob.codes, prob.idx, prob.dist):
        t.fill_(-7)
    prob.out_k.view(torch.int16).fill_(-7)
    prob.out_v.view(torch.int16).fill_(-7)


def _capture_and_compare(ss, prob):
    prob.step()
    torch.cuda.synchronize()
    want = _outputs(prob)
    _scramble(prob)
    g = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        prob.step()  # warm the side stream once outside capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    _scramble(prob)
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        prob.step()
    for _ in range(3):
        _scramble(prob)
        g.replay()
        torch.cuda.synchronize()
        got = _outputs(prob)
        for a, b in zip(got, want):
            assert torch.equal(a, b)
    ss.check_flag(prob.flag, "graph replay")


@pytest.mark.parametrize("name", ["llama8b-1k", "llama8b-5k"])
def test_matching_step_in_a_graph(ss, name):
    import bench

    wl = workloads.WORKLOADS[name]
    prob = bench.make_problem(wl, torch.device("cuda"), wl.base_seed, "tc")
    _capture_and_compare(ss, prob)


def test_retrieval_step_in_a_graph(ss):
    """Retrieval, the selected match and the gather with no host round trip: one graph."""
    import bench

    wl = workloads.RETRIEVAL_WORKLOADS["retrieve-16x4096"].scaled(name="retrieve-8x512", n_ref=8 * 512, n_seg=8,
                                                                    n_tgt=512, kv=(4, 2, 128))
    prob = bench.make_problem(wl, torch.device("cuda"), wl.base_seed, "tc")
    _capture_and_compare(ss, prob)
    assert prob.winner == workloads.retrieval_member(wl)


def test_prepared_calls_match_the_plain_calls(ss):
    """Prepared calls (arguments checked and marshalled once) give the plain calls' results, on
    the current stream or a given one, for a fraction of the host time."""
    import time

    import bench

    wl = workloads.WORKLOADS["llama8b-1k"]
    prob = bench.make_problem(wl, torch.device("cuda"), wl.base_seed, "tc")
    prob.step()
    torch.cuda.synchronize()
    want = _outputs(prob)
    n_ref = wl.n_ref
    calls = [
        ss.semshare_hash(prob.emb, prob.table, prob.hyp, prob.pos, codes=prob.codes, err_flag=prob.flag,
                         workspace=prob.hash_ws, prepare=True),
        ss.semshare_match_tc(prob.codes[n_ref:], prob.codes[:n_ref], idx=prob.idx, dist=prob.dist,
                             workspace=prob.tc_ws, err_flag=prob.flag, prepare=True),
        ss.semshare_gather_kv(prob.ref_k, prob.ref_v, prob.idx.view(1, -1), out_k=prob.out_k, out_v=prob.out_v,
                              err_flag=prob.flag, prepare=True),
    ]
    for stream in (None, torch.cuda.Stream()):
        _scramble(prob)
        torch.cuda.synchronize()
        if stream is None:
            for c in calls:
                c()
        else:
            stream.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(stream):
                for c in calls:
                    c(stream)
            torch.cuda.current_stream().wait_stream(stream)
        torch.cuda.synchronize()
        for a, b in zip(_outputs(prob), want):
            assert torch.equal(a, b)
    ss.check_flag(prob.flag, "prepared calls")
    assert calls[1]()[0] is prob.idx  # the outputs are returned
    # host time of a prepared call: enqueue-only, averaged
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(200):
        calls[2]()
    dt = (time.perf_counter() - t0) / 200
    torch.cuda.synchronize()
    assert dt < 1e-3
