"""Runs one library call on a workload's synthetic inputs, a few times, for profilers.

    python -m paper_2509_24832_gb300.kernel_runner --kernel hash|match|gather --workload NAME [--reps N]

Only the buffers that call needs are allocated (e.g. the 5k-token hash holds ~100 MB, the
5k-token gather ~1.4 GB), which keeps a profiler's capture small.  Inputs come from workloads.py;
the match and gather run on the codes and indices the library computes for that workload."""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads  # noqa: E402

import paper_2509_24832_gb300 as ss  # noqa: E402


def main(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--kernel", choices=["hash", "match", "match_tc", "gather"], required=True)
    p.add_argument("--workload", default="llama8b-5k", choices=sorted(workloads.WORKLOADS))
    p.add_argument("--reps", type=int, default=3)
    a = p.parse_args(argv)
    dev = torch.device("cuda")
    wl = workloads.WORKLOADS[a.workload]
    emb, pos, _ = workloads.prompt_rows(wl)
    e = torch.from_numpy(emb).to(dev) if emb.dtype == np.float32 else \
        torch.from_numpy(emb.view(np.int16)).to(dev).view(torch.bfloat16)
    pd = torch.from_numpy(pos).to(dev)
    R = torch.from_numpy(workloads.hyperplanes(wl).view(np.int16)).to(dev).view(torch.bfloat16)
    table = ss.semshare_rope_table(wl.d, 10000.0, device=dev)
    flag = ss.new_err_flag(dev)
    codes = ss.semshare_hash(e, table, R, pd, err_flag=flag)
    if a.kernel == "hash":
        for _ in range(a.reps):
            ss.semshare_hash(e, table, R, pd, codes=codes, err_flag=flag)
    else:
        tc, rc = codes[wl.n_ref:], codes[: wl.n_ref]
        idx, dist = ss.semshare_match(tc, rc)
        if a.kernel == "match":
            for _ in range(a.reps):
                ss.semshare_match(tc, rc, idx=idx, dist=dist)
        elif a.kernel == "match_tc":
            for _ in range(a.reps):
                ss.semshare_match_tc(tc, rc, idx=idx, dist=dist, err_flag=flag)
        else:
            del e
            segs = [workloads.kv_cache_device(wl, dev, segment=s) for s in range(wl.n_seg)]
            L, H, hd = wl.kv
            out_k = torch.empty((wl.n_batch, L, H, wl.n_tgt, hd), dtype=torch.bfloat16, device=dev)
            out_v = torch.empty_like(out_k)
            for _ in range(a.reps):
                ss.semshare_gather_kv([s[0] for s in segs], [s[1] for s in segs], idx.view(wl.n_batch, wl.n_tgt),
                                      out_k=out_k, out_v=out_v, err_flag=flag)
    torch.cuda.synchronize()
    ss.check_flag(flag, a.kernel)
    print(f"{a.kernel} on {wl.name}: {a.reps} launches ok")


if __name__ == "__main__":
    main()
