"""The bf16 hash on CTA pairs (hash_2sm.cu, forced with SEMSHARE_HASH_KERNEL=pair at these
sizes): the stream-K split over clusters must not change what is computed.  With the cluster
count lowered through SEMSHARE_HASH_CLUSTERS (1, odd counts that leave one cluster straddling
tiles, and counts above the tile count), the codes and projections must satisfy the oracle's
rules, and the pair call (plain + rotated codes in one launch) must equal the two separate calls
even when a cluster's range crosses from the plain into the rotated half."""
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


@pytest.fixture(autouse=True)
def _pair_kernel(monkeypatch):
    # these sizes are below the pair kernel's dispatch threshold: force it
    monkeypatch.setenv("SEMSHARE_HASH_KERNEL", "pair")


def _inputs(n, d, nbits, seed):
    wl = workloads.Workload("t", n_ref=n, n_tgt=1, d=d, emb_dtype="bf16", nbits=nbits, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=777 + seed)
    return workloads.reference_embeddings(wl), workloads.hyperplanes(wl)


@pytest.mark.parametrize("clusters", ["1", "3", "7", "37", "75"])
@pytest.mark.parametrize("n,d,nbits", [(1000, 4096, 256), (300, 1024, 128), (2600, 512, 64)])
def test_cluster_count_keeps_parity(ss, oracle_mod, monkeypatch, clusters, n, d, nbits):
    emb, R = _inputs(n, d, nbits, seed=n)
    pos = np.arange(n, dtype=np.int32) * 3 + 11
    e, Rd = emb_dev(emb), bf16_dev(R)
    table = ss.semshare_rope_table(d)
    p = torch.from_numpy(pos).cuda()
    monkeypatch.setenv("SEMSHARE_HASH_CLUSTERS", clusters)
    flag = ss.new_err_flag()
    proj = torch.full((n, nbits), float("nan"), dtype=torch.float32, device="cuda")
    codes = ss.semshare_hash(e, table, Rd, p, proj_out=proj, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, f"hash with {clusters} clusters")
    oc, op = oracle_mod.hash_codes(emb, pos, R)
    check_hash(codes_host(codes), proj.cpu().numpy(), oc, op)


@pytest.mark.parametrize("clusters", ["1", "5", "9"])
def test_pair_call_with_odd_cluster_counts(ss, oracle_mod, monkeypatch, clusters):
    """With 5 or 9 clusters over 2 x 4 pair tiles of 16 K blocks, one cluster's range runs from
    the last plain tile into the first rotated one."""
    n, d, nbits = 900, 1024, 256
    emb, R = _inputs(n, d, nbits, seed=5)
    e, Rd = emb_dev(emb), bf16_dev(R)
    table = ss.semshare_rope_table(d)
    pos = torch.arange(n, dtype=torch.int32, device="cuda")
    monkeypatch.setenv("SEMSHARE_HASH_CLUSTERS", clusters)
    flag = ss.new_err_flag()
    plain, rot = ss.semshare_hash_pair(e, table, Rd, pos, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, "hash pair")
    oc0, op0 = oracle_mod.hash_codes(emb, np.zeros(n, dtype=np.int32), R)
    oc1, op1 = oracle_mod.hash_codes(emb, np.arange(n, dtype=np.int32), R)
    check_hash(codes_host(plain), None, oc0, op0)
    check_hash(codes_host(rot), None, oc1, op1)


def test_positions_not_32_apart(ss, oracle_mod):
    """Rows whose positions are not 32 apart take the sincos of every row (no 32-step rotation),
    mixed with tiles whose positions are."""
    n, d, nbits = 777, 2048, 256
    emb, R = _inputs(n, d, nbits, seed=9)
    pos = np.arange(n, dtype=np.int32)
    pos[300:500] = np.random.default_rng(9).integers(0, 1 << 30, size=200)
    flag = ss.new_err_flag()
    proj = torch.empty((n, nbits), dtype=torch.float32, device="cuda")
    codes = ss.semshare_hash(emb_dev(emb), ss.semshare_rope_table(d), bf16_dev(R), torch.from_numpy(pos).cuda(),
                             proj_out=proj, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, "hash")
    oc, op = oracle_mod.hash_codes(emb, pos, R)
    check_hash(codes_host(codes), proj.cpu().numpy(), oc, op)


@pytest.mark.parametrize("n,d,nbits", [(2048, 4096, 128), (2432, 4096, 256), (600, 512, 64)])
def test_dispatch_either_kernel_keeps_parity(ss, oracle_mod, monkeypatch, n, d, nbits):
    # bf16 calls below 8 stages per SM pair go to the one-SM kernel; 2432 rows x 4096 is 10 pair
    # tiles x 64 K blocks = 640 stages, just above the threshold on 152 SMs.  Whichever kernel the
    # dispatch picks, and either one forced, the codes and projections follow the oracle's rules.
    emb, R = _inputs(n, d, nbits, seed=n + d)
    pos = np.arange(n, dtype=np.int32)
    oc, op = oracle_mod.hash_codes(emb, pos, R)
    table = ss.semshare_rope_table(d)
    for kernel in ("", "pair", "one"):
        if kernel:
            monkeypatch.setenv("SEMSHARE_HASH_KERNEL", kernel)
        else:
            monkeypatch.delenv("SEMSHARE_HASH_KERNEL", raising=False)
        proj = torch.empty((n, nbits), dtype=torch.float32, device="cuda")
        flag = ss.new_err_flag()
        codes = ss.semshare_hash(emb_dev(emb), table, bf16_dev(R), torch.from_numpy(pos).cuda(), proj_out=proj,
                                 err_flag=flag)
        torch.cuda.synchronize()
        assert int(flag.item()) == 0, kernel
        check_hash(codes_host(codes), proj.cpu().numpy(), oc, op)
