"""End-to-end parity of the whole path (hash -> match -> gather, through the C ABI) on the five
workloads at their full sizes.  The three small ones are compared with the oracle everywhere;
the batched (64 x 2048 targets) and pool (16 x 4096 references) ones run in full on the GPU
and are compared on sampled rows, targets and (prompt, layer, head) planes, each of which the
oracle recomputes from scratch."""
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


def _kv_bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _run_path(ss, wl, emb, pos, want_proj):
    """The step bench.py times: one hash launch over reference + target rows, one match,
    one gather.  Returns device results."""
    dev = torch.device("cuda")
    n_rows = emb.shape[0]
    e = emb_dev(emb, dev)
    p = torch.from_numpy(pos).to(dev)
    R = bf16_dev(workloads.hyperplanes(wl), dev)
    table = ss.semshare_rope_table(wl.d, 10000.0, device=dev)
    proj = torch.empty((n_rows, wl.nbits), dtype=torch.float32, device=dev) if want_proj else None
    flag = ss.new_err_flag(dev)
    codes = ss.semshare_hash(e, table, R, p, proj_out=proj, err_flag=flag)
    idx, dist = ss.semshare_match_tc(codes[wl.n_ref:], codes[: wl.n_ref], err_flag=flag)
    pidx, pdist = ss.semshare_match(codes[wl.n_ref:], codes[: wl.n_ref])
    torch.cuda.synchronize()
    assert torch.equal(idx, pidx) and torch.equal(dist, pdist), "tensor-core and popc matchers disagree"
    segs = [workloads.kv_cache_device(wl, dev, segment=s) for s in range(wl.n_seg)]
    out_k, out_v = ss.semshare_gather_kv([s[0] for s in segs], [s[1] for s in segs],
                                         idx.view(wl.n_batch, wl.n_tgt), err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, wl.name)
    return codes, proj, idx, dist, segs, out_k, out_v


@pytest.mark.parametrize("name", ["tiny", "llama8b-1k", "llama8b-5k"])
def test_small_workloads_everywhere(ss, orc, name):
    wl = workloads.WORKLOADS[name]
    emb, pos, src = workloads.prompt_rows(wl)
    codes, proj, idx, dist, segs, out_k, out_v = _run_path(ss, wl, emb, pos, want_proj=True)

    gc = codes_host(codes)
    oc, op = orc.hash_codes(emb, pos, workloads.hyperplanes(wl))
    band, total = check_hash(gc, proj.cpu().numpy(), oc, op)

    # the match is exact on identical codes: search the GPU's codes on both sides ...
    oi, od = orc.match(gc[wl.n_ref:], gc[: wl.n_ref])
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(dist.cpu().numpy(), od)
    # ... and the oracle's codes on both sides
    ti = torch.from_numpy(oc[wl.n_ref:].view(np.int32)).cuda()
    ri = torch.from_numpy(oc[: wl.n_ref].view(np.int32)).cuda()
    i2, d2 = ss.semshare_match(ti, ri)
    oi2, od2 = orc.match(oc[wl.n_ref:], oc[: wl.n_ref])
    np.testing.assert_array_equal(i2.cpu().numpy(), oi2)
    np.testing.assert_array_equal(d2.cpu().numpy(), od2)

    k, v = segs[0]
    ek, ev, bad = orc.gather_kv(_kv_bits(k), _kv_bits(v), oi)
    assert bad == 0
    assert np.array_equal(_kv_bits(out_k), ek) and np.array_equal(_kv_bits(out_v), ev)

    copied = src[0] >= 0
    recall = float((oi[copied] == src[0][copied]).mean())
    print(f"{name}: band bits {band}/{total}, recall of copied rows {recall:.3f}")


@pytest.mark.parametrize("name", ["batched-64x2048", "pool-16x4096"])
def test_large_workloads_sampled(ss, orc, name):
    wl = workloads.WORKLOADS[name]
    emb, pos, src = workloads.prompt_rows(wl)
    codes, proj, idx, dist, segs, out_k, out_v = _run_path(ss, wl, emb, pos, want_proj=True)
    g = np.random.default_rng(17)
    n_rows = emb.shape[0]

    rows = np.sort(np.concatenate([g.choice(n_rows, 384, replace=False), [0, wl.n_ref - 1, wl.n_ref, n_rows - 1]]))
    gc = codes_host(codes)
    oc, op = orc.hash_codes(emb[rows], pos[rows], workloads.hyperplanes(wl))
    check_hash(gc, proj.cpu().numpy(), oc, op, rows=rows)

    n_t = wl.n_batch * wl.n_tgt
    tsel = np.sort(g.choice(n_t, 512, replace=False))
    oi, od = orc.match(gc[wl.n_ref:][tsel], gc[: wl.n_ref])
    np.testing.assert_array_equal(idx.cpu().numpy()[tsel], oi)
    np.testing.assert_array_equal(dist.cpu().numpy()[tsel], od)

    idx_b = idx.view(wl.n_batch, wl.n_tgt).cpu().numpy()
    L, H, _ = wl.kv
    for _ in range(6):
        b, l, h = int(g.integers(wl.n_batch)), int(g.integers(L)), int(g.integers(H))
        seg_k = [_kv_bits(s[0][l:l + 1, h:h + 1]) for s in segs]
        seg_v = [_kv_bits(s[1][l:l + 1, h:h + 1]) for s in segs]
        ek, ev, bad = orc.gather_kv(seg_k, seg_v, idx_b[b])
        assert bad == 0
        assert np.array_equal(_kv_bits(out_k[b, l, h]), ek[0, 0, 0])
        assert np.array_equal(_kv_bits(out_v[b, l, h]), ev[0, 0, 0])
