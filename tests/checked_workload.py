"""Runs the library's pipelined calls on fixed seeded inputs and saves their outputs, for
tests/test_gpu_checked.py: that test runs this script once with the checked build
(SEMSHARE_CHECKED=1, every call's error word must stay 0) and compares the saved outputs with
the same calls made by the plain build.

    python tests/checked_workload.py OUT.npz"""
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads  # noqa: E402

import paper_2509_24832_gb300 as ss  # noqa: E402


def bf16(x: np.ndarray, dev) -> torch.Tensor:
    return torch.from_numpy(x.astype(np.float32)).to(dev).to(torch.bfloat16)


def run(dev) -> dict:
    """name -> numpy array; raises if an error word is not 0."""
    out = {}
    flags = []

    def flag():
        f = ss.new_err_flag(dev)
        flags.append(f)
        return f

    g = np.random.default_rng(2024)
    # the hash on SM pairs (bf16 rows): ragged tiles, stream-K shares at several cluster counts
    n, d, nbits = 2348, 1024, 256
    emb = bf16(g.standard_normal((n, d)), dev)
    hyp = bf16(g.standard_normal((nbits, d)), dev)
    pos = torch.from_numpy((np.arange(n) % 1500).astype(np.int32)).to(dev)
    table = ss.semshare_rope_table(d, device=dev)
    os.environ["SEMSHARE_HASH_KERNEL"] = "pair"  # a call this small would otherwise go to the one-SM kernel
    for cl in ("", "3", "37"):
        if cl:
            os.environ["SEMSHARE_HASH_CLUSTERS"] = cl
        else:
            os.environ.pop("SEMSHARE_HASH_CLUSTERS", None)
        ws = torch.zeros(ss.semshare_hash_workspace_size(n, d, nbits), dtype=torch.uint8, device=dev)
        out[f"hash2sm_{cl or 'all'}"] = ss.semshare_hash(emb, table, hyp, pos, workspace=ws, err_flag=flag())
    os.environ.pop("SEMSHARE_HASH_CLUSTERS", None)
    # the pair call (plain and rotary codes in one launch)
    cp, cr = ss.semshare_hash_pair(emb[:513].contiguous(), table, hyp, pos[:513].contiguous(), err_flag=flag())
    out["pair_plain"], out["pair_rotary"] = cp, cr
    os.environ.pop("SEMSHARE_HASH_KERNEL", None)
    # the one-SM kernel: fp32 rows, and the rotate-half pairing
    e32 = torch.from_numpy(g.standard_normal((700, 512)).astype(np.float32)).to(dev)
    h128 = bf16(g.standard_normal((128, 512)), dev)
    t512 = ss.semshare_rope_table(512, device=dev)
    out["hash_f32"] = ss.semshare_hash(e32, t512, h128, None, err_flag=flag())
    out["hash_half"] = ss.semshare_hash(bf16(g.standard_normal((1000, 512)), dev), t512, h128, None, err_flag=flag(),
                                        rope_layout="half")
    # the tensor-core search, retrieval and the selected match
    ref = torch.from_numpy(workloads.random_codes(2500, 256, seed=7, stream=1).view(np.int32)).to(dev)
    tgt = torch.from_numpy(workloads.random_codes(3000, 256, seed=7, stream=2).view(np.int32)).to(dev)
    tgt[:1000] = ref[:1000]
    idx, dist = ss.semshare_match_tc(tgt, ref, err_flag=flag())
    out["match_idx"], out["match_dist"] = idx, dist
    offs = [0, 400, 1100, 1600, 2500]
    r = ss.semshare_retrieve(tgt[:900].contiguous(), ref, offs, err_flag=flag())
    out["ret_mean"], out["ret_best"], out["ret_idx"] = r.mean_dist, r.best, r.idx
    si, sd = ss.semshare_match_tc_selected(tgt[:900].contiguous(), ref, offs, r.best, err_flag=flag())
    out["sel_idx"], out["sel_dist"] = si, sd
    # the sign rows of the hash and the one-launch search on them (its last CTA splits the keys)
    os.environ["SEMSHARE_HASH_KERNEL"] = "pair"
    sc, signs = ss.semshare_hash_signs(emb, table, hyp, pos, err_flag=flag())
    os.environ.pop("SEMSHARE_HASH_KERNEL", None)
    out["signs_codes"], out["signs"] = sc, signs
    si2, sd2 = ss.semshare_match_tc_signs(signs[1200:], signs[:1200], nbits, err_flag=flag())
    out["signs_idx"], out["signs_dist"] = si2, sd2
    torch.cuda.synchronize()
    for i, f in enumerate(flags):
        v = int(f.item()) & 0xFFFFFFFF
        if v:
            kernel, line = ss.check_record(v)
            raise RuntimeError(f"call {i}: error word {v:#x} (check kernel {kernel}, line {line})")
    return {k: v.cpu().numpy() for k, v in out.items()}


def main():
    dev = torch.device("cuda")
    ss.load()
    res = run(dev)
    if ss.semshare_checked_build():
        f = ss.new_err_flag(dev)
        ss.semshare_check_selftest(f)
        torch.cuda.synchronize()
        v = int(f.item()) & 0xFFFFFFFF
        kernel, line = ss.check_record(v)
        res["selftest"] = np.array([v & 0xFF, kernel, line], dtype=np.int64)
        res["checked"] = np.array([1])
    np.savez(sys.argv[1], **res)
    print("ok")


if __name__ == "__main__":
    main()
