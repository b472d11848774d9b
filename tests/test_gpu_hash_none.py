"""semshare_hash_ex with SEMSHARE_ROPE_NONE (no rotation: the retrieval codes of Sec. 3.2) against
the oracle's hash at position 0, where RoPE is the identity (Eq. 1 at m = 0): projections within
1e-3 of the row's largest |p|, codes bit-exact outside that band; and bit-identical to the
interleaved kernel given every position 0.  The pair call (plain and rotary codes in one launch)
equals the two calls, on every SM and, for the one-SM kernel, on odd numbers of CTAs."""
import numpy as np
import pytest

import workloads
from gpu_helpers import bf16_dev, check_hash, codes_host, emb_dev, unpack_bits

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ss():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_24832_gb300 as ss

    ss.load()
    return ss


@pytest.mark.parametrize("n,d,nbits,dtype", [(300, 4096, 256, "bf16"), (1000, 512, 64, "f32"), (129, 256, 128, "bf16"),
                                             (5000, 1024, 256, "bf16")])
def test_no_rotation(ss, oracle_mod, n, d, nbits, dtype):
    wl = workloads.Workload("t", n_ref=n, n_tgt=1, d=d, emb_dtype=dtype, nbits=nbits, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=4242 + n)
    emb = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    dev = torch.device("cuda")
    e = emb_dev(emb, dev)
    Rd = bf16_dev(R, dev)
    table = ss.semshare_rope_table(d, 10000.0, device=dev)
    proj = torch.empty((n, nbits), dtype=torch.float32, device=dev)
    flag = ss.new_err_flag(dev)
    codes = ss.semshare_hash(e, None, Rd, None, proj_out=proj, err_flag=flag, rope_layout="none")
    zeros = torch.zeros(n, dtype=torch.int32, device=dev)
    proj0 = torch.empty_like(proj)
    codes0 = ss.semshare_hash(e, table, Rd, zeros, proj_out=proj0, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, "hash none")
    assert torch.equal(codes, codes0) and torch.equal(proj, proj0)
    oc, op = oracle_mod.hash_codes(emb, np.zeros(n, dtype=np.int32), R)
    check_hash(codes_host(codes), proj.cpu().numpy(), oc, op)


@pytest.mark.parametrize("n,d,nbits,dtype,pos", [(4096, 4096, 256, "bf16", "own"), (300, 512, 64, "f32", "random"),
                                                 (77, 256, 128, "bf16", "none"), (5000, 1024, 256, "bf16", "random")])
def test_pair_equals_the_two_calls(ss, oracle_mod, n, d, nbits, dtype, pos):
    """semshare_hash_pair: the unrotated and the rotated codes of the same rows in one launch
    equal those of the two separate calls (ragged tails, fewer rows than a tile, fp32 rows).

    The launches split the K blocks between SMs differently (the pair call has twice the tiles),
    so the fp32 partial sums are added in a different order and a projection within a few ulps
    of zero may take the other sign.  Every differing bit must therefore lie inside the oracle's
    band (|p| < 1e-3 of the row's largest |p|), and there may be only a handful of them."""
    wl = workloads.Workload("t", n_ref=n, n_tgt=1, d=d, emb_dtype=dtype, nbits=nbits, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=99 + n)
    emb = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    dev = torch.device("cuda")
    e = emb_dev(emb, dev)
    Rd = bf16_dev(R, dev)
    table = ss.semshare_rope_table(d, 10000.0, device=dev)
    g = np.random.default_rng(n)
    pos_np = None if pos == "none" else (
        np.arange(n, dtype=np.int32) if pos == "own" else g.integers(0, 1 << 20, size=n).astype(np.int32))
    p = None if pos_np is None else torch.from_numpy(pos_np).to(dev)
    flag = ss.new_err_flag(dev)
    for _ in range(2):  # the shared workspace stays usable
        plain, rot = ss.semshare_hash_pair(e, table, Rd, p, err_flag=flag)
        want_plain = ss.semshare_hash(e, None, Rd, None, err_flag=flag, rope_layout="none")
        want_rot = ss.semshare_hash(e, table, Rd, p, err_flag=flag)
        torch.cuda.synchronize()
        ss.check_flag(flag, "hash pair")
        for got, want, positions in ((plain, want_plain, np.zeros(n, dtype=np.int32)), (rot, want_rot, pos_np)):
            diff = unpack_bits(codes_host(got)) != unpack_bits(codes_host(want))
            assert diff.sum() <= max(4, diff.size // 100000), int(diff.sum())
            rows = np.nonzero(diff.any(axis=1))[0]
            if len(rows):
                sub_pos = None if positions is None else positions[rows]
                if sub_pos is None:
                    sub_pos = rows.astype(np.int32)
                _, op = oracle_mod.hash_codes(emb[rows], sub_pos, R)
                band = np.abs(op) < 1e-3 * np.abs(op).max(axis=1, keepdims=True)
                assert (band | ~diff[rows]).all(), "a bit outside the band differs between the launches"


@pytest.mark.parametrize("ctas", ["1", "7", "33", "151"])
@pytest.mark.parametrize("n,d,nbits,dtype,pos", [(700, 512, 128, "f32", "random"), (3000, 1024, 256, "bf16", "own")])
def test_pair_call_on_one_sm_with_odd_grids(ss, oracle_mod, monkeypatch, ctas, n, d, nbits, dtype, pos):
    """The one-SM kernel's pair call on fewer CTAs than SMs (SEMSHARE_HASH_CTAS), odd counts among
    them: a CTA's range then runs from the last plain tiles into the first rotated ones, and the
    rotation table entries of its next stage are fetched across that boundary.  The same checks
    as the call on every SM."""
    monkeypatch.setenv("SEMSHARE_HASH_CTAS", ctas)
    monkeypatch.setenv("SEMSHARE_HASH_KERNEL", "one")
    test_pair_equals_the_two_calls(ss, oracle_mod, n, d, nbits, dtype, pos)
