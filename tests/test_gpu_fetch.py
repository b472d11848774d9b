"""Parity of semshare_fetch_rows (Sec. 3.2 loads the retrieved reference prompt's KV cache onto
the GPU; Sec. 3.3 reads only the rows the match selects) with the oracle: the selected rows are
copied bit for bit, every other row is left alone, bad indices are flagged and skipped, and the
rearrangement of the loaded copy is the rearrangement of the source."""
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


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _sentinel_like(t, cap):
    """A sentinel-filled device tensor with t's shape and strides (a token slice of capacity cap)."""
    L, H, n, hd = t.shape
    buf = torch.full((L, H, cap, hd), SENTINEL, dtype=torch.int16, device="cuda").view(t.dtype)
    out = buf[:, :, :n]
    assert out.stride() == t.stride()
    return out


def _pool(sizes, L, H, hd, cap, pinned=False, seed=0):
    torch.manual_seed(seed)
    ks, vs = [], []
    for n in sizes:
        k = torch.randn((L, H, cap, hd), device="cuda").to(torch.bfloat16)[:, :, :n]
        v = torch.randn((L, H, cap, hd), device="cuda").to(torch.bfloat16)[:, :, :n]
        if pinned:
            k = torch.empty((L, H, cap, hd), dtype=torch.bfloat16).pin_memory()[:, :, :n].copy_(k)
            v = torch.empty((L, H, cap, hd), dtype=torch.bfloat16).pin_memory()[:, :, :n].copy_(v)
        ks.append(k)
        vs.append(v)
    return ks, vs


def _check(ss, orc, ks, vs, idx, cap, flag=None):
    dk = [_sentinel_like(k, cap) for k in ks]
    dv = [_sentinel_like(v, cap) for v in vs]
    ss.semshare_fetch_rows(ks, vs, torch.from_numpy(idx).cuda(), dev_k=dk, dev_v=dv, err_flag=flag)
    torch.cuda.synchronize()
    hk = [_bits(k) for k in ks]
    hv = [_bits(v) for v in vs]
    ek = [np.full_like(a, np.uint16(SENTINEL & 0xFFFF)) for a in hk]
    ev = [np.full_like(a, np.uint16(SENTINEL & 0xFFFF)) for a in hv]
    ek, ev, bad = orc.fetch_rows(hk, hv, idx, ek, ev)
    for s in range(len(ks)):
        assert np.array_equal(_bits(dk[s]), ek[s]), f"K segment {s}"
        assert np.array_equal(_bits(dv[s]), ev[s]), f"V segment {s}"
    return dk, dv, bad


@pytest.mark.parametrize("hd", [128, 64, 256, 8])
def test_fetch_parity(ss, oracle_mod, hd):
    g = np.random.default_rng(hd)
    ks, vs = _pool([300], 4, 2, hd, 320, seed=hd)
    idx = g.integers(0, 300, size=500).astype(np.int32)  # repeats, ragged last row block
    _, _, bad = _check(ss, oracle_mod, ks, vs, idx, 320)
    assert bad == 0


@pytest.mark.parametrize("pinned", [False, True])
def test_fetch_pool_segments(ss, oracle_mod, pinned):
    g = np.random.default_rng(11)
    sizes = [130, 0, 64, 1, 257]
    ks, vs = _pool(sizes, 3, 4, 128, 260, pinned=pinned, seed=3)
    idx = g.integers(0, sum(sizes), size=(3, 200)).astype(np.int32)
    _, _, bad = _check(ss, oracle_mod, ks, vs, idx, 260)
    assert bad == 0


def test_fetch_then_gather_equals_gather(ss):
    g = np.random.default_rng(5)
    ks, vs = _pool([777, 1000], 8, 8, 128, 1024, seed=5)
    idx = torch.from_numpy(g.integers(0, 1777, size=(2, 900)).astype(np.int32)).cuda()
    dk, dv = ss.semshare_fetch_rows(ks, vs, idx)
    want_k, want_v = ss.semshare_gather_kv(ks, vs, idx)
    got_k, got_v = ss.semshare_gather_kv(dk, dv, idx)
    torch.cuda.synchronize()
    assert torch.equal(got_k.view(torch.int16), want_k.view(torch.int16))
    assert torch.equal(got_v.view(torch.int16), want_v.view(torch.int16))


def test_fetch_bad_indices_flagged(ss, oracle_mod):
    ks, vs = _pool([100, 60], 2, 2, 64, 128, seed=8)
    idx = np.array([5, -1, 160, 159, 2**31 - 1, 100, 5], dtype=np.int32)
    flag = ss.new_err_flag()
    _, _, bad = _check(ss, oracle_mod, ks, vs, idx, 128, flag=flag)
    assert bad == 3
    assert int(flag.item()) & ss.FLAG_INDEX


def test_fetch_empty_idx_writes_nothing(ss, oracle_mod):
    ks, vs = _pool([50], 2, 2, 64, 64, seed=9)
    _check(ss, oracle_mod, ks, vs, np.zeros(0, dtype=np.int32), 64)


def test_fetch_full_size_pinned(ss):
    """The llama8b-5k reference cache (32 layers x 8 KV heads x 5120 tokens x 128, bf16) in pinned
    host memory, with the workload's own match: fetch + gather equals the gather of the source."""
    wl = workloads.WORKLOADS["llama8b-5k"]
    L, H, hd = wl.kv
    g = np.random.default_rng(1)
    n_ref = wl.n_ref
    k = torch.empty((L, H, n_ref, hd), dtype=torch.bfloat16).pin_memory()
    v = torch.empty_like(k).pin_memory()
    k.view(torch.int16).copy_(torch.from_numpy(g.integers(-32768, 32767, size=k.shape, dtype=np.int16)))
    v.view(torch.int16).copy_(torch.from_numpy(g.integers(-32768, 32767, size=v.shape, dtype=np.int16)))
    # a skewed selection like the match's: 70% distinct rows
    idx = torch.from_numpy(np.sort(g.integers(0, n_ref, size=wl.n_tgt)).astype(np.int32)).cuda()
    dk, dv = ss.semshare_fetch_rows(k, v, idx)
    got_k, got_v = ss.semshare_gather_kv(dk, dv, idx)
    want_k, want_v = ss.semshare_gather_kv(k, v, idx)
    torch.cuda.synchronize()
    assert torch.equal(got_k.view(torch.int16), want_k.view(torch.int16))
    assert torch.equal(got_v.view(torch.int16), want_v.view(torch.int16))


def test_fetch_with_64_segments_and_f32_rows(ss, oracle_mod):
    """The most segments a pool may have (64, some empty), fp32 rows of 16 bytes (4 elements)."""
    g = np.random.default_rng(31)
    sizes = g.integers(0, 40, size=64)
    L, H, hd = 2, 3, 4
    cap = 48
    ks = [torch.randn((L, H, cap, hd), device="cuda")[:, :, :n] for n in sizes]
    vs = [torch.randn((L, H, cap, hd), device="cuda")[:, :, :n] for n in sizes]
    n_rows = int(sizes.sum())
    idx = g.integers(0, n_rows, size=700).astype(np.int32)
    dk = [torch.full((L, H, cap, hd), -7.0, device="cuda")[:, :, :n] for n in sizes]
    dv = [torch.full((L, H, cap, hd), -7.0, device="cuda")[:, :, :n] for n in sizes]
    ss.semshare_fetch_rows(ks, vs, torch.from_numpy(idx).cuda(), dev_k=dk, dev_v=dv)
    torch.cuda.synchronize()
    hk = [k.cpu().contiguous().numpy() for k in ks]
    hv = [v.cpu().contiguous().numpy() for v in vs]
    ek = [np.full_like(a, -7.0) for a in hk]
    ev = [np.full_like(a, -7.0) for a in hv]
    ek, ev, bad = oracle_mod.fetch_rows(hk, hv, idx, ek, ev)
    assert bad == 0
    for s in range(64):
        assert np.array_equal(dk[s].cpu().contiguous().numpy(), ek[s]), s
        assert np.array_equal(dv[s].cpu().contiguous().numpy(), ev[s]), s
