"""Parity of each CUDA kernel, called through the C ABI, against the CPU oracle on the same
seeded inputs: several tiles, ragged tails and the edge cases of each step."""
import math

import numpy as np
import pytest

import workloads
from gpu_helpers import bf16_dev, check_hash, codes_host, emb_dev, operand_flip_allowance

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


# ---- rotation table ------------------------------------------------------------------------

@pytest.mark.parametrize("d,base", [(4096, 10000.0), (512, 10000.0), (128, 500000.0), (4, (2 / math.pi) ** 2)])
def test_rope_table(ss, orc, d, base):
    t = ss.semshare_rope_table(d, base).cpu().numpy().view(np.uint64)
    for k in range(d // 2):
        turns = orc.theta(k, d, base) / (2 * math.pi)
        want = (turns - math.floor(turns)) * 2.0 ** 64
        got = float(t[k])
        err = min(abs(got - want), 2.0 ** 64 - abs(got - want))   # modulo one turn
        assert err <= 4e-15 * 2.0 ** 64 * max(turns, 1e-3), k


# ---- hash -----------------------------------------------------------------------------------

def _hash_case(ss, orc, n, d, nbits, dtype, pos_kind, pad=0, seed=0):
    wl = workloads.Workload("t", n_ref=n, n_tgt=1, d=d, emb_dtype=dtype, nbits=nbits, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=1234 + seed)
    emb = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    g = np.random.default_rng(seed)
    if pos_kind == "own":
        pos = np.arange(n, dtype=np.int32)
    elif pos_kind == "random":
        pos = g.integers(0, 8192, size=n).astype(np.int32)
    elif pos_kind == "large":
        pos = g.integers(0, 2 ** 31 - 1, size=n).astype(np.int32)
    else:
        pos = None
    dev_emb = emb_dev(emb)
    if pad:
        wide = torch.zeros((n, d + pad), dtype=dev_emb.dtype, device="cuda")
        wide[:, :d] = dev_emb
        dev_emb = wide[:, :d]
    table = ss.semshare_rope_table(d)
    proj = torch.full((n, nbits), float("nan"), dtype=torch.float32, device="cuda")
    flag = ss.new_err_flag()
    codes = ss.semshare_hash(dev_emb, table, bf16_dev(R), None if pos is None else torch.from_numpy(pos).cuda(),
                             proj_out=proj, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, "hash")
    oc, op = orc.hash_codes(emb, pos, R)
    return codes_host(codes), proj.cpu().numpy(), oc, op, emb, pos, R


@pytest.mark.parametrize(
    "n,d,nbits,dtype,pos_kind,pad",
    [
        (1000, 4096, 256, "bf16", "own", 0),      # 8 tiles, ragged tail of 104 rows
        (640, 4096, 128, "bf16", "random", 0),
        (300, 512, 64, "f32", "own", 0),          # the tiny workload's shape: fp32 rows
        (77, 1024, 32, "bf16", None, 0),          # one partial tile, positions 0..n-1
        (129, 512, 96, "bf16", "own", 64),        # strided rows, 3-word codes
        (1, 128, 160, "f32", "random", 0),
        (2000, 256, 224, "bf16", "large", 0),     # positions up to 2^31-1
        (385, 2048, 256, "f32", "large", 32),
        (1536, 1024, 192, "bf16", "own", 0),     # 192-bit codes: the slot count rounded to the RoPE groups
        (700, 512, 128, "f32", "random", 0),      # fp32 rows with 128-bit codes: two pipeline slots
        (300, 8192, 256, "bf16", "own", 0),       # wider rows than any workload: 128 K blocks per tile
        (257, 64, 64, "bf16", "random", 0),       # one K block per tile
    ],
)
def test_hash_parity(ss, orc, n, d, nbits, dtype, pos_kind, pad):
    gc, gp, oc, op, emb, pos, R = _hash_case(ss, orc, n, d, nbits, dtype, pos_kind, pad)
    if d >= 512:
        check_hash(gc, gp, oc, op)
    else:
        check_hash(gc, gp, oc, op, flips=operand_flip_allowance(orc, emb, pos, R))


def test_hash_scaling_and_negation_invariants(ss):
    wl = workloads.WORKLOADS["llama8b-1k"].scaled(n_ref=500)
    emb = workloads.reference_embeddings(wl)
    R = bf16_dev(workloads.hyperplanes(wl))
    table = ss.semshare_rope_table(wl.d)
    x = bf16_dev(emb)
    pos = torch.arange(500, dtype=torch.int32, device="cuda") * 7
    p1 = torch.empty((500, wl.nbits), device="cuda")
    p4 = torch.empty_like(p1)
    pn = torch.empty_like(p1)
    c1 = ss.semshare_hash(x, table, R, pos, proj_out=p1)
    c4 = ss.semshare_hash(x * 4, table, R, pos, proj_out=p4)
    cn = ss.semshare_hash(-x, table, R, pos, proj_out=pn)
    torch.cuda.synchronize()
    scale = p1.abs().amax(dim=1, keepdim=True)
    assert torch.equal(c1, c4)
    assert bool(((p4 - 4 * p1).abs() <= 1e-6 * 4 * scale).all())
    assert bool(((pn + p1).abs() <= 1e-6 * scale).all())
    # outside a thin band around zero the negated rows carry the complemented bits
    sure = (p1.abs() > 1e-5 * scale).cpu().numpy()
    from gpu_helpers import unpack_bits
    b1 = unpack_bits(codes_host(c1))
    bn = unpack_bits(codes_host(cn))
    assert ((b1 != bn) | ~sure).all()


def test_hash_empty_and_repeatable(ss):
    table = ss.semshare_rope_table(128)
    R = torch.zeros((64, 128), dtype=torch.bfloat16, device="cuda")
    x = torch.zeros((0, 128), dtype=torch.bfloat16, device="cuda")
    assert ss.semshare_hash(x, table, R).shape == (0, 2)
    x = torch.randn((300, 128), device="cuda").to(torch.bfloat16)
    R = torch.randn((64, 128), device="cuda").to(torch.bfloat16)
    a = ss.semshare_hash(x, table, R)
    b = ss.semshare_hash(x, table, R)
    assert torch.equal(a, b)


def test_hash_workspace_shared_across_sizes(ss):
    """One workspace serves calls of different sizes one after another: each call's codes and
    projections equal those of the same call on a fresh zero-filled workspace (the per-tile
    counters never land on an earlier call's partial sums)."""
    g = torch.Generator(device="cuda").manual_seed(3)
    cases = [(256, 512, 64), (10240, 4096, 256), (300, 4096, 256), (5000, 1024, 128), (70000, 128, 32),
             (1000, 4096, 96), (129, 64, 256)]
    big = max(ss.semshare_hash_workspace_size(n, d, nb) for n, d, nb in cases)
    shared = torch.zeros(big, dtype=torch.uint8, device="cuda")
    for n, d, nb in cases:
        x = torch.randn((n, d), generator=g, device="cuda").to(torch.bfloat16)
        R = torch.randn((nb, d), generator=g, device="cuda").to(torch.bfloat16)
        table = ss.semshare_rope_table(d)
        p1 = torch.empty((n, nb), dtype=torch.float32, device="cuda")
        p2 = torch.empty_like(p1)
        fresh = torch.zeros(ss.semshare_hash_workspace_size(n, d, nb), dtype=torch.uint8, device="cuda")
        a = ss.semshare_hash(x, table, R, proj_out=p1, workspace=shared)
        b = ss.semshare_hash(x, table, R, proj_out=p2, workspace=fresh)
        torch.cuda.synchronize()
        assert torch.equal(a, b) and torch.equal(p1, p2), (n, d, nb)


def test_hash_stream_k_split_tiles_are_deterministic(ss, orc):
    # 3 tiles x 64 K blocks over all SMs: every tile is shared by many CTAs
    gc1, gp1, oc, op, emb, pos, R = _hash_case(ss, orc, 300, 4096, 256, "bf16", "own", seed=5)
    gc2, gp2, _, _, _, _, _ = _hash_case(ss, orc, 300, 4096, 256, "bf16", "own", seed=5)
    assert np.array_equal(gc1, gc2) and np.array_equal(gp1, gp2)
    check_hash(gc1, gp1, oc, op)


# ---- match ----------------------------------------------------------------------------------

@pytest.mark.parametrize("nbits", [32, 64, 96, 128, 256])
@pytest.mark.parametrize("n_tgt,n_ref", [(1, 1), (513, 255), (3000, 1000), (700, 5000)])
def test_match_parity(ss, orc, nbits, n_tgt, n_ref):
    g = np.random.default_rng(nbits * 7 + n_ref)
    ref = workloads.random_codes(n_ref, nbits, seed=nbits + n_ref, stream=1)
    tgt = workloads.random_codes(n_tgt, nbits, seed=nbits + n_tgt, stream=2)
    k = n_tgt // 3
    if k:
        tgt[:k] = ref[g.integers(0, n_ref, size=k)]          # exact copies
        tgt[:k, 0] ^= np.uint32(1) << np.uint32(g.integers(0, 32))  # one bit off
    if n_ref > 4:
        ref[n_ref - 1] = ref[2]                               # duplicate: ties to the lower index
    ti = torch.from_numpy(tgt.view(np.int32)).cuda()
    ri = torch.from_numpy(ref.view(np.int32)).cuda()
    idx, dist = ss.semshare_match(ti, ri)
    oi, od = orc.match(tgt, ref)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(dist.cpu().numpy(), od)


@pytest.mark.parametrize("nbits", [32, 64, 96, 128, 160, 256])
@pytest.mark.parametrize("n_tgt,n_ref", [(1, 1), (513, 255), (3000, 1000), (700, 5000), (129, 257)])
def test_match_tc_parity(ss, orc, nbits, n_tgt, n_ref):
    g = np.random.default_rng(nbits * 11 + n_ref)
    ref = workloads.random_codes(n_ref, nbits, seed=nbits + n_ref, stream=3)
    tgt = workloads.random_codes(n_tgt, nbits, seed=nbits + n_tgt, stream=4)
    k = n_tgt // 3
    if k:
        tgt[:k] = ref[g.integers(0, n_ref, size=k)]
        tgt[:k, 0] ^= np.uint32(1) << np.uint32(g.integers(0, 32))
    if n_ref > 4:
        ref[n_ref - 1] = ref[2]
    ti = torch.from_numpy(tgt.view(np.int32)).cuda()
    ri = torch.from_numpy(ref.view(np.int32)).cuda()
    flag = ss.new_err_flag()
    idx, dist = ss.semshare_match_tc(ti, ri, err_flag=flag)
    pi, pd = ss.semshare_match(ti, ri)
    torch.cuda.synchronize()
    ss.check_flag(flag, "match_tc")
    oi, od = orc.match(tgt, ref)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(dist.cpu().numpy(), od)
    assert torch.equal(idx, pi) and torch.equal(dist, pd)


def test_match_tc_ties_and_all_equal(ss):
    c = torch.randint(-2 ** 31, 2 ** 31 - 1, (3000, 8), dtype=torch.int32, device="cuda")
    c[2999] = c[7]
    idx, dist = ss.semshare_match_tc(c, c)
    want = torch.arange(3000, dtype=torch.int32, device="cuda")
    want[2999] = 7
    assert torch.equal(idx, want) and int(dist.max()) == 0
    same = torch.full((600, 8), 5, dtype=torch.int32, device="cuda")
    idx2, d2 = ss.semshare_match_tc(c[:100].contiguous(), same)
    assert int(idx2.max()) == 0


def test_match_tc_workspace_reused_across_shapes(ss, orc):
    """One workspace, sized for the largest call and left dirty by each, serves calls of different
    shapes in turn: many target blocks and few reference blocks, one target block against many
    reference blocks, ragged last blocks, codes narrower than one 128-bit chunk.  Each result
    equals the xor/popc search (and the oracle where that is quick)."""
    shapes = [(40000, 600, 256), (50, 70000, 256), (3001, 2999, 128), (129, 257, 64), (40000, 600, 256)]
    need = max(ss.semshare_match_tc_workspace_size(t, r, b) for t, r, b in shapes)
    ws = torch.full((need,), 0x5A, dtype=torch.uint8, device="cuda")
    for i, (n_tgt, n_ref, nbits) in enumerate(shapes):
        ref = workloads.random_codes(n_ref, nbits, seed=90 + i, stream=3)
        tgt = workloads.random_codes(n_tgt, nbits, seed=90 + i, stream=4)
        tgt[: n_tgt // 4] = ref[np.arange(n_tgt // 4) % n_ref]
        ti = torch.from_numpy(tgt.view(np.int32)).cuda()
        ri = torch.from_numpy(ref.view(np.int32)).cuda()
        flag = ss.new_err_flag()
        idx, dist = ss.semshare_match_tc(ti, ri, workspace=ws, err_flag=flag)
        pi, pd = ss.semshare_match(ti, ri)
        torch.cuda.synchronize()
        ss.check_flag(flag, "match_tc")
        assert torch.equal(idx, pi) and torch.equal(dist, pd), (n_tgt, n_ref, nbits)
        if n_tgt * n_ref <= 10 ** 7:
            oi, od = orc.match(tgt, ref)
            np.testing.assert_array_equal(idx.cpu().numpy(), oi)
            np.testing.assert_array_equal(dist.cpu().numpy(), od)


def test_match_identity_ties_and_determinism(ss):
    c = torch.randint(-2 ** 31, 2 ** 31 - 1, (4000, 8), dtype=torch.int32, device="cuda")
    c[3999] = c[5]
    idx, dist = ss.semshare_match(c, c)
    want = torch.arange(4000, dtype=torch.int32, device="cuda")
    want[3999] = 5
    assert torch.equal(idx, want) and int(dist.max()) == 0
    same = torch.full((300, 4), 7, dtype=torch.int32, device="cuda")
    idx2, _ = ss.semshare_match(c[:, :4].contiguous(), same)
    assert int(idx2.max()) == 0
    a = ss.semshare_match(c[:1000], c[1000:])
    b = ss.semshare_match(c[:1000], c[1000:])
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])


# ---- gather ---------------------------------------------------------------------------------

def _rand_kv(shape, dtype=torch.bfloat16, seed=0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    if dtype == torch.float32:
        return torch.randn(shape, generator=g, device="cuda")
    return torch.randint(-2 ** 15, 2 ** 15, shape, generator=g, device="cuda", dtype=torch.int32).to(
        torch.int16).view(torch.bfloat16)


def _np_bits(t):
    return t.detach().cpu().contiguous().view(torch.uint8).numpy()


@pytest.mark.parametrize("L,H,hd,dtype", [(4, 2, 128, torch.bfloat16), (2, 4, 64, torch.bfloat16),
                                          (3, 1, 96, torch.bfloat16), (2, 2, 32, torch.float32),
                                          (1, 3, 256, torch.bfloat16), (2, 1, 8, torch.bfloat16)])
def test_gather_parity_single_reference(ss, orc, L, H, hd, dtype):
    n_ref, n_tgt = 333, 200
    k = _rand_kv((L, H, n_ref, hd), dtype, 1)
    v = _rand_kv((L, H, n_ref, hd), dtype, 2)
    idx = torch.randint(0, n_ref, (n_tgt,), dtype=torch.int32, device="cuda")
    idx[0], idx[-1] = 0, n_ref - 1
    flag = ss.new_err_flag()
    ok, ov = ss.semshare_gather_kv(k, v, idx, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, "gather")
    ek, ev, bad = orc.gather_kv(_np_bits(k).reshape(L, H, n_ref, -1), _np_bits(v).reshape(L, H, n_ref, -1),
                                idx.cpu().numpy())
    assert bad == 0
    assert np.array_equal(_np_bits(ok).reshape(ek.shape), ek)
    assert np.array_equal(_np_bits(ov).reshape(ev.shape), ev)


def test_gather_pool_batch_and_strided_output(ss, orc):
    L, H, hd, cap = 3, 2, 128, 300
    lens = [300, 17, 0, 129]
    kb = _rand_kv((len(lens), L, H, cap, hd), seed=3)
    vb = _rand_kv((len(lens), L, H, cap, hd), seed=4)
    seg_k = [kb[s, :, :, :n] for s, n in enumerate(lens)]
    seg_v = [vb[s, :, :, :n] for s, n in enumerate(lens)]
    total = sum(lens)
    B, T = 3, 150
    idx = torch.randint(0, total, (B, T), dtype=torch.int32, device="cuda")
    big_k = torch.zeros((B, L, H, T + 5, hd), dtype=torch.bfloat16, device="cuda")
    big_v = torch.zeros_like(big_k)
    ok, ov = ss.semshare_gather_kv(seg_k, seg_v, idx, out_k=big_k[:, :, :, 2:T + 2], out_v=big_v[:, :, :, 2:T + 2])
    torch.cuda.synchronize()
    np_k = [_np_bits(s).reshape(L, H, s.shape[2], hd * 2) for s in seg_k]
    np_v = [_np_bits(s).reshape(L, H, s.shape[2], hd * 2) for s in seg_v]
    ek, ev, bad = orc.gather_kv(np_k, np_v, idx.cpu().numpy())
    assert bad == 0
    assert np.array_equal(_np_bits(ok.contiguous()).reshape(ek.shape), ek)
    assert np.array_equal(_np_bits(ov.contiguous()).reshape(ev.shape), ev)
    assert int(big_k[:, :, :, :2].abs().sum()) == 0 and int(big_k[:, :, :, T + 2:].abs().sum()) == 0


@pytest.mark.parametrize("hd,dtype", [(32, torch.bfloat16), (96, torch.bfloat16), (128, torch.bfloat16),
                                      (256, torch.bfloat16), (128, torch.float32)])
def test_gather_several_prompts_every_row_size(ss, orc, hd, dtype):
    # several target prompts against one reference take the evict-first store path; row sizes of
    # 4, 12 (generic kernel), 16 and 32 chunks
    L, H, n_ref, B, T = 3, 2, 257, 4, 131
    k = _rand_kv((L, H, n_ref, hd), dtype, 21)
    v = _rand_kv((L, H, n_ref, hd), dtype, 22)
    idx = torch.randint(0, n_ref, (B, T), dtype=torch.int32, device="cuda")
    idx[1, :] = idx[0, :]  # two prompts selecting the same rows
    ok, ov = ss.semshare_gather_kv(k, v, idx)
    torch.cuda.synchronize()
    ek, ev, bad = orc.gather_kv(_np_bits(k).reshape(L, H, n_ref, -1), _np_bits(v).reshape(L, H, n_ref, -1),
                                idx.cpu().numpy())
    assert bad == 0
    assert np.array_equal(_np_bits(ok).reshape(ek.shape), ek)
    assert np.array_equal(_np_bits(ov).reshape(ev.shape), ev)


def test_gather_out_of_range_flags_and_skips(ss):
    k = _rand_kv((2, 2, 50, 64), seed=5)
    v = _rand_kv((2, 2, 50, 64), seed=6)
    idx = torch.tensor([3, 50, -1, 49, 1 << 30], dtype=torch.int32, device="cuda")
    out_k = torch.full((1, 2, 2, 5, 64), 1.5, dtype=torch.bfloat16, device="cuda")
    out_v = torch.full((1, 2, 2, 5, 64), 2.5, dtype=torch.bfloat16, device="cuda")
    flag = ss.new_err_flag()
    ss.semshare_gather_kv(k, v, idx, out_k=out_k, out_v=out_v, err_flag=flag)
    torch.cuda.synchronize()
    assert ss.flag_status(flag) == 4
    bits = lambda t: t.contiguous().view(torch.int16)  # noqa: E731  (random patterns include NaNs)
    assert torch.equal(bits(out_k[0, :, :, 0]), bits(k[:, :, 3])) and torch.equal(bits(out_v[0, :, :, 3]), bits(v[:, :, 49]))
    for t in (1, 2, 4):
        assert bool((out_k[0, :, :, t] == 1.5).all()) and bool((out_v[0, :, :, t] == 2.5).all())


def test_gather_preserves_special_bit_patterns(ss):
    pats = torch.tensor([0x7FC1, -1, -32768, 1, 0x7F80, -128, -32641, 0x7FA5], dtype=torch.int16)
    k = pats.repeat(1, 1, 8, 8).view(torch.bfloat16).cuda()   # [1][1][8][64]
    v = k.flip(-1).contiguous()
    idx = torch.arange(7, -1, -1, dtype=torch.int32, device="cuda")
    ok, ov = ss.semshare_gather_kv(k, v, idx)
    assert torch.equal(ok[0].view(torch.int16), k.flip(2).view(torch.int16))
    assert torch.equal(ov[0].view(torch.int16), v.flip(2).view(torch.int16))


# ---- failure detection: a pipeline wait that runs out ----------------------------------------

def test_wait_timeout_reports_status_and_context_survives(ss, orc, monkeypatch):
    # a 1 ns wait limit makes the pipelined kernels' waits run out: they must report
    # SEMSHARE_ETIMEOUT through the error word, return without trapping, and leave the CUDA
    # context usable (the next calls, with the default limit, give correct results)
    wl = workloads.WORKLOADS["llama8b-1k"]
    emb, pos, _ = workloads.prompt_rows(wl)
    e = emb_dev(emb)
    p = torch.from_numpy(pos).cuda()
    R = bf16_dev(workloads.hyperplanes(wl))
    table = ss.semshare_rope_table(wl.d)
    ws = torch.zeros(ss.semshare_hash_workspace_size(len(emb), wl.d, wl.nbits) + 256, dtype=torch.uint8,
                     device="cuda")
    codes = torch.empty((len(emb), wl.nbits // 32), dtype=torch.int32, device="cuda")
    monkeypatch.setenv("SEMSHARE_WAIT_LIMIT_NS", "1")
    for kernel in ("pair", "one"):  # the bf16 hash on SM pairs and on single SMs
        monkeypatch.setenv("SEMSHARE_HASH_KERNEL", kernel)
        ws.zero_()
        flag = ss.new_err_flag()
        ss.semshare_hash(e, table, R, p, codes=codes, workspace=ws, err_flag=flag)
        torch.cuda.synchronize()
        assert ss.flag_status(flag) == 5, kernel  # SEMSHARE_ETIMEOUT
    monkeypatch.delenv("SEMSHARE_HASH_KERNEL")
    tgt, ref = codes[wl.n_ref:], codes[: wl.n_ref]
    flag2 = ss.new_err_flag()
    ss.semshare_match_tc(tgt, ref, err_flag=flag2)
    torch.cuda.synchronize()
    assert ss.flag_status(flag2) == 5
    monkeypatch.delenv("SEMSHARE_WAIT_LIMIT_NS")
    # the context is intact: rerun with the default limit (the timed-out hash may have left
    # its workspace dirty, so it is zeroed first) and compare with the oracle
    ws.zero_()
    flag3 = ss.new_err_flag()
    proj = torch.empty((len(emb), wl.nbits), dtype=torch.float32, device="cuda")
    codes = ss.semshare_hash(e, table, R, p, codes=codes, proj_out=proj, workspace=ws, err_flag=flag3)
    idx, dist = ss.semshare_match_tc(codes[wl.n_ref:], codes[: wl.n_ref], err_flag=flag3)
    torch.cuda.synchronize()
    ss.check_flag(flag3, "after timeout")
    oc, op = orc.hash_codes(emb, pos, workloads.hyperplanes(wl))
    check_hash(codes_host(codes), proj.cpu().numpy(), oc, op)
    gc = codes_host(codes)
    oi, od = orc.match(gc[wl.n_ref:], gc[: wl.n_ref])
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)


def test_gather_from_pinned_host_cache(ss):
    """Reference segments in page-locked host memory: the kernel reads the selected rows across the
    host link in place; the result equals the gather from device copies bit for bit."""
    g = torch.Generator().manual_seed(5)
    segs = [(torch.randn((3, 2, n, 128), generator=g).to(torch.bfloat16).pin_memory(),
             torch.randn((3, 2, n, 128), generator=g).to(torch.bfloat16).pin_memory()) for n in (300, 300)]
    idx = torch.randint(0, 600, (2, 257), generator=g, dtype=torch.int32).cuda()
    flag = ss.new_err_flag()
    hk, hv = ss.semshare_gather_kv([s[0] for s in segs], [s[1] for s in segs], idx, err_flag=flag)
    dk, dv = ss.semshare_gather_kv([s[0].cuda() for s in segs], [s[1].cuda() for s in segs], idx)
    torch.cuda.synchronize()
    assert hk.is_cuda and int(flag.item()) == 0
    assert torch.equal(hk.view(torch.int16), dk.view(torch.int16)) and torch.equal(hv.view(torch.int16), dv.view(torch.int16))


@pytest.mark.gpu
def test_hamming_rate_probe_runs_and_is_plausible():
    """The word-operation probe (the xor/popc matcher's roofline denominator) runs on every SM and
    reports a rate between 1 and 100 T word-ops/s (the Programming Guide's table gives ~5 T)."""
    import bench

    rate = bench.measure_hamming_rate(torch.device("cuda"), iters=1 << 12, reps=3)
    assert 1e12 < rate < 1e14, rate
