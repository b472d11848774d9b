"""Parity of semshare_hash_ex with the rotate-half pairing (pairs (k, k + d/2) turned by
m * theta_k) against the oracle's hash with layout="half", under the same rules as the
interleaved hash: projections within 1e-3 of the row's largest |p|, codes bit-exact outside
that band (plus the derived operand-rounding allowance where d < 512)."""
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


def _case(ss, orc, n, d, nbits, pos_kind, pad=0, seed=0):
    wl = workloads.Workload("t", n_ref=n, n_tgt=1, d=d, emb_dtype="bf16", nbits=nbits, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=777 + seed)
    emb = workloads.reference_embeddings(wl)
    R = workloads.hyperplanes(wl)
    g = np.random.default_rng(seed)
    pos = {"own": np.arange(n, dtype=np.int32), "large": g.integers(0, 2 ** 31 - 1, size=n).astype(np.int32),
           "random": g.integers(0, 8192, size=n).astype(np.int32)}[pos_kind]
    e = emb_dev(emb)
    if pad:
        wide = torch.zeros((n, d + pad), dtype=e.dtype, device="cuda")
        wide[:, :d] = e
        e = wide[:, :d]
    proj = torch.full((n, nbits), float("nan"), dtype=torch.float32, device="cuda")
    flag = ss.new_err_flag()
    codes = ss.semshare_hash(e, ss.semshare_rope_table(d), bf16_dev(R), torch.from_numpy(pos).cuda(), proj_out=proj,
                             err_flag=flag, rope_layout="half")
    torch.cuda.synchronize()
    ss.check_flag(flag, "hash half")
    oc, op = orc.hash_codes(emb, pos, R, layout="half")
    flips = operand_flip_allowance(orc, emb, pos, R, layout="half") if d < 512 else None
    return codes_host(codes), proj.cpu().numpy(), oc, op, flips


@pytest.mark.parametrize("n,d,nbits,pos_kind,pad", [
    (1000, 4096, 256, "own", 0),     # 8 tiles, ragged tail; 32 half-pairs of blocks
    (300, 128, 64, "large", 0),      # the smallest d: one block and its partner
    (129, 512, 96, "random", 64),    # strided rows, 3-word codes
    (5, 1024, 32, "own", 0),         # fewer rows than one tile
])
def test_hash_half_parity(ss, orc, n, d, nbits, pos_kind, pad):
    gc, gp, oc, op, flips = _case(ss, orc, n, d, nbits, pos_kind, pad)
    check_hash(gc, gp, oc, op, flips=flips)


def test_hash_half_differs_from_interleaved_and_is_deterministic(ss, orc):
    gc1, gp1, _, _, _ = _case(ss, orc, 700, 4096, 256, "own", seed=3)
    gc2, gp2, _, _, _ = _case(ss, orc, 700, 4096, 256, "own", seed=3)
    assert np.array_equal(gc1, gc2) and np.array_equal(gp1, gp2)
    wl = workloads.Workload("t", n_ref=700, n_tgt=1, d=4096, emb_dtype="bf16", nbits=256, kv=(1, 1, 8), reuse=0.5,
                            noise=0.1, recipe="perm", base_seed=777 + 3)
    inter = ss.semshare_hash(emb_dev(workloads.reference_embeddings(wl)), ss.semshare_rope_table(4096),
                             bf16_dev(workloads.hyperplanes(wl)))
    torch.cuda.synchronize()
    assert (codes_host(inter) != gc1).mean() > 0.1


def test_hash_half_unsupported_shapes(ss):
    table = ss.semshare_rope_table(192)
    R = torch.zeros((64, 192), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ss.SemshareError):  # d not a multiple of 128
        ss.semshare_hash(torch.zeros((4, 192), dtype=torch.bfloat16, device="cuda"), table, R, rope_layout="half")
    table = ss.semshare_rope_table(256)
    R = torch.zeros((64, 256), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ss.SemshareError):  # fp32 rows
        ss.semshare_hash(torch.zeros((4, 256), dtype=torch.float32, device="cuda"), table, R, rope_layout="half")


def test_hash_half_workload_5k(ss, orc):
    """The 5k workload's 10,240 rows hashed with the half pairing, compared everywhere."""
    wl = workloads.WORKLOADS["llama8b-5k"]
    emb, pos, _ = workloads.prompt_rows(wl)
    R = workloads.hyperplanes(wl)
    proj = torch.empty((len(emb), wl.nbits), dtype=torch.float32, device="cuda")
    codes = ss.semshare_hash(emb_dev(emb), ss.semshare_rope_table(wl.d), bf16_dev(R), torch.from_numpy(pos).cuda(),
                             proj_out=proj, rope_layout="half")
    torch.cuda.synchronize()
    oc, op = orc.hash_codes(emb, pos, R, layout="half")
    band, total = check_hash(codes_host(codes), proj.cpu().numpy(), oc, op)
    print(f"half pairing, 5k: band bits {band}/{total}")
