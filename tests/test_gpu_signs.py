"""The sign-row path: semshare_hash_signs writes the codes a second time as e4m3 +-1 rows, and
semshare_match_tc_signs searches those rows in one launch (Sec. 3.3: the most similar reference
token of each target token, ties to the lowest index).

Checks: the sign rows are exactly the expansion of the packed codes (0x38 for a set bit, 0xB8 for a
clear one, zero padding to the pitch) on both hash kernels (bf16 rows on SM pairs with and without
rotation, fp32 rows and rotate-half on one SM), including tiles finished by the stream-K close;
the codes equal semshare_hash's and pass the oracle's band rule; the match's idx/dist are
bit-exact against the oracle's exhaustive scan on the same codes, in the fused path (the last CTA
splits the keys) and the split-kernel path (more than 16384 targets), on several calls in a row
through one workspace, which every call leaves 0xFF-filled again."""
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


def expand(codes: np.ndarray, nbits: int, pitch: int) -> np.ndarray:
    """The sign rows of packed codes, written out bit by bit."""
    bits = np.unpackbits(np.ascontiguousarray(codes).view(np.uint8), axis=1, bitorder="little")[:, :nbits]
    rows = np.zeros((codes.shape[0], pitch), dtype=np.uint8)
    rows[:, :nbits] = np.where(bits == 1, 0x38, 0xB8)
    return rows


def _hash_inputs(n, d, nbits, dtype, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((n, d)).astype(np.float32)
    emb = torch.from_numpy(x).cuda()
    if dtype == "bf16":
        emb = emb.to(torch.bfloat16)
    hyp = torch.from_numpy(rng.standard_normal((nbits, d)).astype(np.float32)).cuda().to(torch.bfloat16)
    pos = torch.from_numpy(rng.integers(0, 1 << 20, n).astype(np.int32)).cuda()
    return emb, hyp, pos


@pytest.mark.parametrize(
    "n,d,nbits,dtype,layout,clusters",
    [
        (1000, 512, 64, "bf16", "interleaved", ""),      # pad bytes 64..127
        (1000, 512, 96, "bf16", "interleaved", "7"),     # odd cluster count: shared tiles closed
        (3000, 1024, 160, "bf16", "none", ""),           # pad bytes 160..255
        (2600, 4096, 256, "bf16", "interleaved", "5"),   # several contributors per tile
        (700, 512, 128, "fp32", "interleaved", ""),      # the one-SM kernel
        (900, 1024, 192, "bf16", "half", ""),            # rotate-half, one-SM kernel
    ],
)
def test_hash_signs_are_the_expanded_codes(ss, monkeypatch, n, d, nbits, dtype, layout, clusters):
    if clusters:
        monkeypatch.setenv("SEMSHARE_HASH_CLUSTERS", clusters)
        monkeypatch.setenv("SEMSHARE_HASH_KERNEL", "pair")  # below the pair kernel's dispatch threshold
    emb, hyp, pos = _hash_inputs(n, d, nbits, dtype, seed=n + nbits)
    table = ss.semshare_rope_table(d)
    flag = ss.new_err_flag()
    want = ss.semshare_hash(emb, table, hyp, pos, err_flag=flag, rope_layout=layout)
    pitch = ss.semshare_signs_pitch(nbits)
    signs = torch.full((n, pitch), 0x5A, dtype=torch.uint8, device="cuda")  # every byte must be written
    codes, signs = ss.semshare_hash_signs(emb, table, hyp, pos, signs=signs, err_flag=flag, rope_layout=layout)
    torch.cuda.synchronize()
    assert int(flag.item()) == 0
    c = codes_host(codes)
    assert np.array_equal(c, codes_host(want)), "codes differ from semshare_hash's"
    assert np.array_equal(signs.cpu().numpy(), expand(c, nbits, pitch))


def test_hash_signs_codes_follow_the_oracle(ss, oracle_mod):
    # the codes and projections written beside the sign rows obey the band rule against the
    # fp64 oracle (the 1k-token workload, every row)
    wl = workloads.WORKLOADS["llama8b-1k"]
    emb, pos, _ = workloads.prompt_rows(wl)
    hyp = workloads.hyperplanes(wl)
    table = ss.semshare_rope_table(wl.d)
    proj = torch.empty((len(emb), wl.nbits), dtype=torch.float32, device="cuda")
    codes, signs = ss.semshare_hash_signs(emb_dev(emb), table, bf16_dev(hyp), torch.from_numpy(pos).cuda(),
                                          proj_out=proj)
    torch.cuda.synchronize()
    c = codes_host(codes)
    oc, op = oracle_mod.hash_codes(emb, pos, hyp)
    check_hash(c, proj.cpu().numpy(), oc, op)
    assert np.array_equal(signs.cpu().numpy(), expand(c, wl.nbits, ss.semshare_signs_pitch(wl.nbits)))


def _signs_dev(codes, nbits, pitch):
    return torch.from_numpy(expand(codes, nbits, pitch)).cuda()


@pytest.mark.parametrize(
    "n_tgt,n_ref,nbits",
    [(1, 1, 32), (333, 300, 64), (1000, 5000, 256), (5120, 5120, 256), (129, 257, 96), (16384, 700, 160),
     (20000, 3000, 128), (16385, 513, 256)],
)
def test_match_tc_signs_parity(ss, oracle_mod, n_tgt, n_ref, nbits):
    pitch = ss.semshare_signs_pitch(nbits)
    tgt = workloads.random_codes(n_tgt, nbits, seed=n_tgt + nbits, stream=1)
    ref = workloads.random_codes(n_ref, nbits, seed=n_ref + nbits, stream=2)
    k = min(n_tgt, n_ref) // 3
    tgt[:k] = ref[n_ref - k:]          # exact matches: distance 0
    if n_ref > 4:
        ref[n_ref - 1] = ref[2]        # a duplicate row: the tie goes to row 2
    flag = ss.new_err_flag()
    idx, dist = ss.semshare_match_tc_signs(_signs_dev(tgt, nbits, pitch), _signs_dev(ref, nbits, pitch), nbits,
                                           err_flag=flag)
    torch.cuda.synchronize()
    assert int(flag.item()) == 0
    ei, ed = oracle_mod.match(tgt, ref, nbits)
    assert np.array_equal(idx.cpu().numpy(), ei)
    assert np.array_equal(dist.cpu().numpy(), ed)


def test_match_tc_signs_calls_in_a_row_leave_the_workspace_ready(ss, oracle_mod):
    # one workspace, sizes alternating between the fused path and the split-kernel path; each call
    # must find every key reset by the one before
    ws = torch.full((ss.semshare_match_tc_signs_workspace_size(20000),), 0xFF, dtype=torch.uint8, device="cuda")
    for i, (n_tgt, n_ref, nbits) in enumerate([(5000, 4000, 256), (300, 200, 64), (20000, 1000, 128),
                                               (4096, 4096, 256), (17, 3, 32)]):
        pitch = ss.semshare_signs_pitch(nbits)
        tgt = workloads.random_codes(n_tgt, nbits, seed=100 + i, stream=1)
        ref = workloads.random_codes(n_ref, nbits, seed=100 + i, stream=2)
        idx, dist = ss.semshare_match_tc_signs(_signs_dev(tgt, nbits, pitch), _signs_dev(ref, nbits, pitch), nbits,
                                               workspace=ws)
        torch.cuda.synchronize()
        ei, ed = oracle_mod.match(tgt, ref, nbits)
        assert np.array_equal(idx.cpu().numpy(), ei), f"call {i}"
        assert np.array_equal(dist.cpu().numpy(), ed), f"call {i}"
        assert bool((ws == 0xFF).all()), f"workspace not reset after call {i}"


def test_signs_step_on_the_5k_workload(ss, oracle_mod):
    # the bench's step: one hash of the reference and target rows with sign rows, the match on
    # slices of them, against the oracle's scan of the same codes and against semshare_match_tc
    wl = workloads.WORKLOADS["llama8b-5k"]
    emb, pos, _ = workloads.prompt_rows(wl)
    e, hyp = emb_dev(emb), bf16_dev(workloads.hyperplanes(wl))
    table = ss.semshare_rope_table(wl.d)
    codes, signs = ss.semshare_hash_signs(e, table, hyp, torch.from_numpy(pos).cuda())
    idx, dist = ss.semshare_match_tc_signs(signs[wl.n_ref:], signs[: wl.n_ref], wl.nbits)
    i2, d2 = ss.semshare_match_tc(codes[wl.n_ref:], codes[: wl.n_ref])
    torch.cuda.synchronize()
    c = codes_host(codes)
    ei, ed = oracle_mod.match(c[wl.n_ref:], c[: wl.n_ref], wl.nbits)
    assert np.array_equal(idx.cpu().numpy(), ei) and np.array_equal(dist.cpu().numpy(), ed)
    assert torch.equal(idx, i2) and torch.equal(dist, d2)
