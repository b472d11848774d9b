"""semshare_hash_ex with SEMSHARE_ROPE_NONE (no rotation: the retrieval codes of Sec. 3.2) against
the oracle's hash at position 0, where RoPE is the identity (Eq. 1 at m = 0): projections within
1e-3 of the row's largest |p|, codes bit-exact outside that band; and bit-identical to the
interleaved kernel given every position 0."""
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
def test_pair_equals_the_two_calls(ss, n, d, nbits, dtype, pos):
    """semshare_hash_pair: the unrotated and the rotated codes of the same rows in one launch,
    bit for bit those of the two separate calls (ragged tails, fewer rows than a tile, fp32 rows)."""
    wl = workloads.Workload("t", n_ref=n, n_tgt=1, d=d, emb_dtype=dtype, nbits=nbits, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=99 + n)
    emb = workloads.reference_embeddings(wl)
    dev = torch.device("cuda")
    e = emb_dev(emb, dev)
    Rd = bf16_dev(workloads.hyperplanes(wl), dev)
    table = ss.semshare_rope_table(d, 10000.0, device=dev)
    g = np.random.default_rng(n)
    p = None if pos == "none" else torch.from_numpy(
        np.arange(n, dtype=np.int32) if pos == "own" else g.integers(0, 1 << 20, size=n).astype(np.int32)).to(dev)
    flag = ss.new_err_flag(dev)
    for _ in range(2):  # the shared workspace stays usable
        plain, rot = ss.semshare_hash_pair(e, table, Rd, p, err_flag=flag)
        want_plain = ss.semshare_hash(e, None, Rd, None, err_flag=flag, rope_layout="none")
        want_rot = ss.semshare_hash(e, table, Rd, p, err_flag=flag)
        torch.cuda.synchronize()
        ss.check_flag(flag, "hash pair")
        assert torch.equal(plain, want_plain) and torch.equal(rot, want_rot)
