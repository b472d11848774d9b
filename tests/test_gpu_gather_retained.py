"""Parity of semshare_gather_kv_retained (retention, Sec. 3.3.4 and App. A: each layer keeps
only its retained target tokens, packed in list order) with the oracle: bit-exact rows, rows past
a layer's count untouched, bad entries flagged and skipped."""
import numpy as np
import pytest

import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SENTINEL = -12345


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


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _run(ss, segs_k, segs_v, idx, ret, cap=None, flag=None):
    dev = segs_k[0].device
    L, H, _, hd = segs_k[0].shape
    offs = np.concatenate([[0], np.cumsum([len(r) for r in ret])]).astype(np.int64)
    flat = torch.from_numpy(np.concatenate(ret).astype(np.int32) if offs[-1] else np.zeros(1, np.int32)).to(dev)
    cap = max(len(r) for r in ret) if cap is None else cap
    out_k = torch.full((L, H, cap, hd), SENTINEL, dtype=torch.int16, device=dev).view(torch.bfloat16)
    out_v = torch.full((L, H, cap, hd), SENTINEL, dtype=torch.int16, device=dev).view(torch.bfloat16)
    ss.semshare_gather_kv_retained(segs_k, segs_v, torch.from_numpy(idx).to(dev), flat, offs, out_k=out_k,
                                   out_v=out_v, err_flag=flag)
    torch.cuda.synchronize()
    return out_k, out_v


def _expect(orc, segs_k, segs_v, idx, ret, cap):
    k = np.concatenate([_bits(s) for s in segs_k], axis=2)
    v = np.concatenate([_bits(s) for s in segs_v], axis=2)
    L, H, _, hd = k.shape
    ek = np.full((L, H, cap, hd), np.uint16(SENTINEL & 0xFFFF), dtype=np.uint16)
    ev = ek.copy()
    ek, ev, bad = orc.gather_kv_retained(k, v, idx, ret, cap=cap, out_k=ek, out_v=ev)
    return ek, ev, bad


@pytest.mark.parametrize("hd", [128, 64, 32, 256, 48])
def test_retained_parity(ss, orc, hd):
    g = np.random.default_rng(hd)
    L, H, N, T = 4, 2, 300, 200
    k = torch.randn((L, H, N, hd), device="cuda").to(torch.bfloat16)
    v = torch.randn((L, H, N, hd), device="cuda").to(torch.bfloat16)
    idx = g.integers(0, N, size=T).astype(np.int32)
    ret = workloads.retained_tokens(T, [200, 150, 64, 0], seed=hd)
    ret[2] = g.permutation(ret[2]).astype(np.int32)  # any order is allowed: packed in list order
    ok, ov = _run(ss, [k], [v], idx, ret, cap=210)
    ek, ev, bad = _expect(orc, [k], [v], idx, ret, 210)
    assert bad == 0
    assert np.array_equal(_bits(ok), ek) and np.array_equal(_bits(ov), ev)


def test_retained_pool_and_all_retained(ss, orc):
    g = np.random.default_rng(7)
    L, H, hd, T = 3, 4, 128, 333
    # segments share one layout: token slices of equal-capacity buffers
    segs = [(torch.randn((L, H, 256, hd), device="cuda").to(torch.bfloat16)[:, :, :n],
             torch.randn((L, H, 256, hd), device="cuda").to(torch.bfloat16)[:, :, :n]) for n in (100, 1, 250)]
    idx = g.integers(0, 351, size=T).astype(np.int32)
    ret = workloads.retained_tokens(T, [333, 200, 17], seed=1)
    ok, ov = _run(ss, [s[0] for s in segs], [s[1] for s in segs], idx, ret)
    ek, ev, bad = _expect(orc, [s[0] for s in segs], [s[1] for s in segs], idx, ret, 333)
    assert bad == 0 and np.array_equal(_bits(ok), ek) and np.array_equal(_bits(ov), ev)
    # every token retained in order = the plain rearrangement of one prompt
    full = [np.arange(T, dtype=np.int32)] * L
    ok2, ov2 = _run(ss, [s[0] for s in segs], [s[1] for s in segs], idx, full)
    pk, pv = ss.semshare_gather_kv([s[0] for s in segs], [s[1] for s in segs], torch.from_numpy(idx).cuda())
    torch.cuda.synchronize()
    assert torch.equal(ok2.view(torch.int16), pk[0].view(torch.int16))
    assert torch.equal(ov2.view(torch.int16), pv[0].view(torch.int16))


def test_retained_bad_entries_flagged(ss, orc):
    L, H, N, hd, T = 2, 2, 50, 64, 30
    k = torch.randn((L, H, N, hd), device="cuda").to(torch.bfloat16)
    v = torch.randn((L, H, N, hd), device="cuda").to(torch.bfloat16)
    idx = np.arange(T, dtype=np.int32)
    idx[4] = N + 3                                            # outside the reference
    ret = [np.array([0, 4, 7, 29], np.int32), np.array([30, -1, 2], np.int32)]  # outside the target
    flag = ss.new_err_flag()
    ok, ov = _run(ss, [k], [v], idx, ret, flag=flag)
    assert int(flag.item()) & ss.FLAG_INDEX
    ek, ev, bad = _expect(orc, [k], [v], idx, ret, 4)
    assert bad == 3
    assert np.array_equal(_bits(ok), ek) and np.array_equal(_bits(ov), ev)


def test_retained_empty(ss):
    k = torch.randn((2, 1, 10, 64), device="cuda").to(torch.bfloat16)
    ok, ov = ss.semshare_gather_kv_retained(k, k, torch.zeros(5, dtype=torch.int32, device="cuda"),
                                            torch.zeros(1, dtype=torch.int32, device="cuda"), [0, 0, 0])
    assert ok.shape == (2, 1, 0, 64)


def test_retained_workload_5k(ss, orc):
    """The 5k workload's reference cache, the match's indices, the synthetic schedule (0.8 on the
    first layer, then 0.98 per layer): sampled layers compared with the oracle."""
    wl = workloads.WORKLOADS["llama8b-5k"]
    dev = torch.device("cuda")
    k, v = workloads.kv_cache_device(wl, dev)
    g = np.random.default_rng(11)
    idx = g.integers(0, wl.n_ref, size=wl.n_tgt).astype(np.int32)
    counts = ss.retain_counts(wl.n_tgt, workloads.retain_alphas(wl.n_layers), workloads.RETAIN_DEN)
    ret = workloads.retained_tokens(wl.n_tgt, counts, seed=wl.base_seed)
    ok, ov = _run(ss, [k], [v], idx, ret)
    for l in (0, 1, 17, wl.n_layers - 1):
        ek, ev, bad = orc.gather_kv_retained(_bits(k[l:l + 1]), _bits(v[l:l + 1]), idx, [ret[l]], cap=counts[0])
        n = counts[l]
        assert bad == 0
        assert np.array_equal(_bits(ok[l, :, :n]), ek[0, :, :n]) and np.array_equal(_bits(ov[l, :, :n]), ev[0, :, :n])
    print(f"retained per layer: first {counts[0]}, last {counts[-1]}, mean {np.mean(counts):.0f} of {wl.n_tgt}")
