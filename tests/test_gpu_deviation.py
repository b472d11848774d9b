"""Parity of semshare_kv_deviation (App. A.4) and semshare_select_hd (Insight 1) with the oracle.

Tolerance of the deviations, from the arithmetic: a bf16 - bf16 difference is exact in fp32;
each lane sums about H*hd/32 squares in order and a 5-level shuffle tree adds the lanes, a
relative error below (H*hd/32 + 5 + 1) * 2^-24 of the sum (2.3e-6 for H*hd = 1024); the square
root halves it.  Tested at 5e-6 relative.  The HD selection is an integer decision taken in the
kernel's fp32: it must equal the oracle's selection on the GPU's own deviations exactly, and may
differ from the selection on the oracle's fp64 deviations only by tokens inside that tolerance
band around the k-th value."""
import numpy as np
import pytest

import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

RTOL = 5e-6


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


def _host(t):
    t = t.detach().cpu().contiguous()
    return t.view(torch.int16).numpy().view(np.uint16) if t.dtype == torch.bfloat16 else t.numpy()


def _caches(shape, dtype, seed, device="cuda"):
    g = torch.Generator(device=device).manual_seed(seed)
    base = torch.randn(shape, generator=g, device=device)
    out = []
    for i in range(4):
        noise = torch.randn(shape, generator=g, device=device) * (0.05 if i >= 2 else 0.0)
        out.append((base + noise).to(dtype))
    # k_reused, v_reused (v = k scaled), k_recomp, v_recomp
    return out[0], (out[1] * 0.5).to(dtype), out[2], (out[3] * 0.5).to(dtype)


def _check_sigma(got, want):
    got = got.detach().cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=1e-30)


def _check_select(ss, orc, sig_gpu, sig_orc, k):
    idx, mask = ss.semshare_select_hd(sig_gpu, k, want_mask=True)
    torch.cuda.synchronize()
    idx, mask = idx.cpu().numpy(), mask.cpu().numpy()
    s = sig_gpu.cpu().numpy()
    np.testing.assert_array_equal(idx, orc.select_hd(s, k))   # same decision on the same values
    assert (mask.sum(axis=1) == k).all()
    for l in range(s.shape[0]):
        assert (mask[l][idx[l]] == 1).all()
        # against the fp64 deviations: only tokens within the tolerance band of the k-th value differ
        ref = orc.select_hd(sig_orc[l:l + 1], k)[0]
        diff = np.setxor1d(idx[l], ref)
        if len(diff) and k:
            kth = np.sort(sig_orc[l])[::-1][k - 1]
            assert np.all(np.abs(sig_orc[l][diff] - kth) <= 2 * RTOL * kth), (l, diff)
    return idx


@pytest.mark.parametrize("shape,dtype", [((1, 8, 5120, 128), torch.bfloat16), ((3, 2, 37, 64), torch.bfloat16),
                                         ((2, 1, 1, 8), torch.bfloat16), ((2, 3, 300, 4), torch.float32),
                                         ((1, 5, 1000, 96), torch.bfloat16)])
def test_deviation_parity(ss, orc, shape, dtype):
    k_re, v_re, k_rc, v_rc = _caches(shape, dtype, seed=sum(shape))
    sk, sv, skv = ss.semshare_kv_deviation(k_re, v_re, k_rc, v_rc, want_parts=True)
    torch.cuda.synchronize()
    ok, ov, okv = orc.kv_deviation(*(_host(t) for t in (k_re, v_re, k_rc, v_rc)))
    _check_sigma(sk, ok)
    _check_sigma(sv, ov)
    _check_sigma(skv, okv)
    # the same bits on a second call
    assert torch.equal(ss.semshare_kv_deviation(k_re, v_re, k_rc, v_rc), skv)
    T = shape[2]
    for k in sorted({0, 1, ss.hd_count(T), T}):
        _check_select(ss, orc, skv, okv, k)


def test_deviation_strided_views(ss, orc):
    """A batch slice of a gather-shaped [B][L][H][T][hd] output against a cache that is a
    T-slice of a longer one: both strided."""
    g = torch.Generator(device="cuda").manual_seed(4)
    big = torch.randn((3, 2, 4, 200, 64), generator=g, device="cuda").to(torch.bfloat16)
    other = torch.randn((2, 2, 4, 300, 64), generator=g, device="cuda").to(torch.bfloat16)
    k_re, v_re = big[1], big[2]
    k_rc, v_rc = other[0, :, :, 50:250], other[1, :, :, 50:250]
    skv = ss.semshare_kv_deviation(k_re, v_re, k_rc, v_rc)
    torch.cuda.synchronize()
    _, _, okv = orc.kv_deviation(*(_host(t) for t in (k_re, v_re, k_rc, v_rc)))
    _check_sigma(skv, okv)


def test_identical_caches_and_ties(ss, orc):
    k = torch.randn((2, 4, 777, 128), device="cuda").to(torch.bfloat16)
    v = torch.randn((2, 4, 777, 128), device="cuda").to(torch.bfloat16)
    skv = ss.semshare_kv_deviation(k, v, k, v)
    torch.cuda.synchronize()
    assert int(torch.count_nonzero(skv)) == 0
    idx = ss.semshare_select_hd(skv, 300)
    # all deviations equal: the lowest 300 token indices
    assert torch.equal(idx.cpu(), torch.arange(300, dtype=torch.int32).repeat(2, 1))


@pytest.mark.parametrize("T", [5120, 70000])
def test_select_staged_and_global(ss, orc, T):
    """n_tok small enough to stage the deviations in shared memory, and too large for it."""
    g = np.random.default_rng(T)
    s = g.random((2, T)).astype(np.float32)
    s[1, ::3] = 0.25  # a block of ties around the middle of the range
    sd = torch.from_numpy(s).cuda()
    for k in (1, ss.hd_count(T), T - 1):
        idx = ss.semshare_select_hd(sd, k)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(idx.cpu().numpy(), orc.select_hd(s, k))


def test_empty(ss):
    e = torch.empty((1, 2, 0, 64), dtype=torch.bfloat16, device="cuda")
    assert ss.semshare_kv_deviation(e, e, e, e).shape == (1, 0)
    s = torch.empty((3, 0), dtype=torch.float32, device="cuda")
    assert ss.semshare_select_hd(s, 0).shape == (3, 0)


def test_workload_layer0_after_gather(ss, orc):
    """The 5k workload: gather the reference cache by the match, compare its first layer with a
    synthetic recomputed first layer, select the HD tokens; compare with the oracle."""
    wl = workloads.WORKLOADS["llama8b-5k"]
    emb, pos, src = workloads.prompt_rows(wl)
    dev = torch.device("cuda")
    from gpu_helpers import bf16_dev, emb_dev

    codes = ss.semshare_hash(emb_dev(emb, dev), ss.semshare_rope_table(wl.d, device=dev),
                             bf16_dev(workloads.hyperplanes(wl), dev), torch.from_numpy(pos).to(dev))
    idx, _ = ss.semshare_match_tc(codes[wl.n_ref:], codes[:wl.n_ref])
    k_ref, v_ref = workloads.kv_cache_device(wl, dev)
    out_k, out_v = ss.semshare_gather_kv(k_ref, v_ref, idx)
    k_rc, v_rc = workloads.recomputed_kv_device(wl, dev, k_ref[:1], v_ref[:1], src[0])
    sk, sv, skv = ss.semshare_kv_deviation(out_k[0, :1], out_v[0, :1], k_rc, v_rc, want_parts=True)
    hd = ss.semshare_select_hd(skv)
    torch.cuda.synchronize()
    ok, ov, okv = orc.kv_deviation(*(_host(t) for t in (out_k[0, :1], out_v[0, :1], k_rc, v_rc)))
    _check_sigma(skv, okv)
    _check_select(ss, orc, skv, okv, ss.hd_count(wl.n_tgt))
    fresh = src[0] < 0
    frac = float(np.isin(np.nonzero(fresh)[0], hd.cpu().numpy()[0]).mean())
    print(f"HD tokens {hd.shape[1]} of {wl.n_tgt}; fresh tokens among them {frac:.3f}")


def _f32_specials():
    bits = np.array([0x7FC00000, 0xFFC00000, 0x7F800001, 0xFFBFFFFF,   # NaNs: both signs, several payloads
                     0x7F800000, 0xFF800000, 0x00000000, 0x80000000,   # +inf, -inf, +0, -0
                     0x3F800000, 0x3F800000, 0x40000000, 0xBF800000,   # 1, 1 (a tie), 2, -1
                     0x00000001, 0x7F7FFFFF], dtype=np.uint32)          # a subnormal, the largest float
    return bits.view(np.float32)


@pytest.mark.parametrize("T", [13, 600, 70000])
def test_select_nan_inf_signed_zero(ss, orc, T):
    """NaNs of both signs rank above +inf and tie with each other (lower token first), -0 ties
    with +0: element for element against the oracle's total order, on the staged (T <= ~57 K)
    and the global selection paths, at every k around the special values."""
    g = np.random.default_rng(T)
    pool = _f32_specials()
    s = pool[g.integers(0, len(pool), size=(3, T))].astype(np.float32)
    s[2] = g.random(T).astype(np.float32)
    s[2, g.integers(0, T, size=max(1, T // 50))] = pool[1]   # a few negative NaNs among ordinary values
    s[2, g.integers(0, T, size=max(1, T // 50))] = -0.0
    sd = torch.from_numpy(s).cuda()
    n_nan = int(np.isnan(s).sum(axis=1).max())
    ks = sorted({0, 1, 2, n_nan - 1, n_nan, n_nan + 1, (40 * T + 99) // 100, T - 1, T} & set(range(T + 1)))
    for k in ks:
        idx, mask = ss.semshare_select_hd(sd, k, want_mask=True)
        torch.cuda.synchronize()
        with np.errstate(invalid="ignore"):  # widening a signalling NaN raises the invalid flag
            want = orc.select_hd(s.astype(np.float64), k)
        np.testing.assert_array_equal(idx.cpu().numpy(), want, err_msg=f"T={T} k={k}")
        m = np.zeros((3, T), dtype=np.uint8)
        for l in range(3):
            m[l, want[l]] = 1
        np.testing.assert_array_equal(mask.cpu().numpy(), m)


def test_deviation_nan_inf_payloads(ss, orc):
    """K/V rows holding NaN and inf payloads: NaN and inf deviations land on the same tokens as the
    oracle's, the finite ones agree within the tolerance, and the selection ranks them the same."""
    shape = (2, 4, 333, 64)
    k_re, v_re, k_rc, v_rc = _caches(shape, torch.bfloat16, seed=91)
    kb = k_re.view(torch.int16)
    vb, vcb = v_re.view(torch.int16), v_rc.view(torch.int16)
    kb[0, 1, 7, 3] = 0x7FC1           # NaN in token 7 of layer 0
    kb[1, 0, 100, 0] = -128           # 0xFF80 = -inf against a finite recomputed value
    vb[0, 3, 200, 63] = -128          # -inf minus -inf: NaN
    vcb[0, 3, 200, 63] = -128
    kb[1, 2, 5, 9] = 0x7F80           # +inf
    kb[1, 2, 6, 9] = -63              # 0xFFC1: a NaN with the sign bit set
    sk, sv, skv = ss.semshare_kv_deviation(k_re, v_re, k_rc, v_rc, want_parts=True)
    torch.cuda.synchronize()
    ok, ov, okv = orc.kv_deviation(*(_host(t) for t in (k_re, v_re, k_rc, v_rc)))
    for got, want in ((sk, ok), (sv, ov), (skv, okv)):
        g = got.cpu().numpy().astype(np.float64)
        np.testing.assert_array_equal(np.isnan(g), np.isnan(want))
        np.testing.assert_array_equal(np.isinf(g), np.isinf(want))
        fin = np.isfinite(want)
        np.testing.assert_allclose(g[fin], want[fin], rtol=RTOL, atol=1e-30)
    assert np.isnan(okv[0, 7]) and np.isnan(okv[0, 200]) and np.isnan(okv[1, 6]) and np.isinf(okv[1, 100])
    for k in (1, 2, 3, 4, 133, 333):
        _check_select(ss, orc, skv, okv, k)
