"""Runs one library call on a workload's synthetic inputs, a few times, for profilers.

    python kernel_runner.py --kernel hash|match|match_tc|gather|retrieve
        --workload NAME [--reps N]

Only the buffers that call needs are allocated (e.g. the 5k-token hash holds ~100 MB, the
5k-token gather ~1.4 GB), which keeps a profiler's capture small.  Inputs come from workloads.py;
the match and gather run on the codes and indices the library computes for that workload.  On
a retrieval workload the calls follow the retrieval step: `retrieve` searches the plain codes of
the stored prompts, `match_tc` matches the target against the winner's rotary codes and
`gather` moves the winner's K/V rows (only the winner's cache is allocated)."""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads  # noqa: E402

import paper_2509_24832_gb300 as ss  # noqa: E402

ALL = {**workloads.WORKLOADS, **workloads.RETRIEVAL_WORKLOADS}


def _retrieval(a, wl, e, pd, R, table, flag, dev):
    n_pool = wl.n_ref
    offs = [m * wl.seg_len for m in range(wl.n_seg + 1)]
    plain = ss.semshare_hash(e, None, R, None, err_flag=flag, rope_layout="none")
    ws = torch.empty(ss.semshare_retrieve_workspace_size(wl.n_tgt, n_pool, wl.n_seg, wl.nbits), dtype=torch.uint8,
                     device=dev)
    reps = a.reps if a.kernel == "retrieve" else 1
    for _ in range(reps):
        res = ss.semshare_retrieve(plain[n_pool:], plain[:n_pool], offs, workspace=ws, err_flag=flag,
                                   want_match=False)
    if a.kernel == "retrieve":
        return
    m = int(res.best.item())
    codes = ss.semshare_hash(e, table, R, pd, err_flag=flag)
    del plain
    tc, rc = codes[n_pool:], codes[offs[m]:offs[m + 1]]
    idx = torch.empty(wl.n_tgt, dtype=torch.int32, device=dev)
    dist = torch.empty_like(idx)
    reps = a.reps if a.kernel == "match_tc" else 1
    for _ in range(reps):
        ss.semshare_match_tc(tc, rc, idx=idx, dist=dist, err_flag=flag)
    if a.kernel != "gather":
        return
    del e, codes
    k, v = workloads.kv_cache_device(wl, dev, segment=m)
    L, H, hd = wl.kv
    out_k = torch.empty((1, L, H, wl.n_tgt, hd), dtype=torch.bfloat16, device=dev)
    out_v = torch.empty_like(out_k)
    for _ in range(a.reps):
        ss.semshare_gather_kv([k], [v], idx.view(1, wl.n_tgt), out_k=out_k, out_v=out_v, err_flag=flag)


def main(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--kernel", choices=["hash", "match", "match_tc", "gather", "gather_retained", "retrieve",
                                        "deviation", "select", "fetch"], required=True)
    p.add_argument("--workload", default="llama8b-5k", choices=sorted(ALL))
    p.add_argument("--reps", type=int, default=3)
    a = p.parse_args(argv)
    dev = torch.device("cuda")
    wl = ALL[a.workload]
    emb, pos, src = workloads.prompt_rows(wl)
    e = torch.from_numpy(emb).to(dev) if emb.dtype == np.float32 else \
        torch.from_numpy(emb.view(np.int16)).to(dev).view(torch.bfloat16)
    pd = torch.from_numpy(pos).to(dev)
    R = torch.from_numpy(workloads.hyperplanes(wl).view(np.int16)).to(dev).view(torch.bfloat16)
    table = ss.semshare_rope_table(wl.d, 10000.0, device=dev)
    flag = ss.new_err_flag(dev)
    if wl.recipe == "retrieve":
        if a.kernel not in ("retrieve", "match_tc", "gather"):
            raise SystemExit("a retrieval workload runs retrieve, match_tc or gather")
        _retrieval(a, wl, e, pd, R, table, flag, dev)
    elif a.kernel == "retrieve":
        raise SystemExit("retrieve needs a retrieval workload")
    else:
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
            elif a.kernel == "gather_retained":
                # the synthetic retention schedule of bench.py --retain (one prompt)
                del e
                k, v = workloads.kv_cache_device(wl, dev)
                counts = ss.retain_counts(wl.n_tgt, workloads.retain_alphas(wl.n_layers), workloads.RETAIN_DEN)
                ret = workloads.retained_tokens(wl.n_tgt, counts, wl.base_seed)
                flat = torch.from_numpy(np.concatenate(ret)).to(dev)
                offs = [0] + list(np.cumsum(counts))
                out_k = torch.empty((wl.n_layers, wl.n_heads, counts[0], wl.head_dim), dtype=torch.bfloat16,
                                    device=dev)
                out_v = torch.empty_like(out_k)
                for _ in range(a.reps):
                    ss.semshare_gather_kv_retained(k, v, idx, flat, offs, out_k=out_k, out_v=out_v, err_flag=flag)
            elif a.kernel == "fetch":
                # the selected rows from a reference cache in pinned host memory into HBM
                del e
                segs = [workloads.kv_cache_device(wl, dev, segment=s) for s in range(wl.n_seg)]
                hk = [s[0].cpu().pin_memory() for s in segs]
                hv = [s[1].cpu().pin_memory() for s in segs]
                dk = [s[0] for s in segs]
                dv = [s[1] for s in segs]
                for _ in range(a.reps):
                    ss.semshare_fetch_rows(hk, hv, idx, dev_k=dk, dev_v=dv, err_flag=flag)
            elif a.kernel == "gather":
                del e
                segs = [workloads.kv_cache_device(wl, dev, segment=s) for s in range(wl.n_seg)]
                L, H, hd = wl.kv
                out_k = torch.empty((wl.n_batch, L, H, wl.n_tgt, hd), dtype=torch.bfloat16, device=dev)
                out_v = torch.empty_like(out_k)
                for _ in range(a.reps):
                    ss.semshare_gather_kv([s[0] for s in segs], [s[1] for s in segs],
                                          idx.view(wl.n_batch, wl.n_tgt), out_k=out_k, out_v=out_v, err_flag=flag)
            else:
                # first layer only: gather it, compare with a synthetic recomputed first layer
                del e
                segs = [workloads.kv_cache_device(wl, dev, segment=s) for s in range(wl.n_seg)]
                k0 = torch.cat([s[0][:1] for s in segs], dim=2)
                v0 = torch.cat([s[1][:1] for s in segs], dim=2)
                del segs
                _, H, _, hd = k0.shape
                out_k = torch.empty((wl.n_batch, 1, H, wl.n_tgt, hd), dtype=torch.bfloat16, device=dev)
                out_v = torch.empty_like(out_k)
                ss.semshare_gather_kv(k0, v0, idx.view(wl.n_batch, wl.n_tgt), out_k=out_k, out_v=out_v,
                                      err_flag=flag)
                rc = [workloads.recomputed_kv_device(wl, dev, k0, v0, src[b], seed=wl.base_seed + b)
                      for b in range(wl.n_batch)]
                rc_k = torch.stack([r[0][0] for r in rc])
                rc_v = torch.stack([r[1][0] for r in rc])
                sigma = ss.semshare_kv_deviation(out_k[:, 0], out_v[:, 0], rc_k, rc_v)
                reps = a.reps if a.kernel == "deviation" else 1
                for _ in range(reps - 1):
                    ss.semshare_kv_deviation(out_k[:, 0], out_v[:, 0], rc_k, rc_v, sigma_kv=sigma)
                if a.kernel == "select":
                    for _ in range(a.reps):
                        ss.semshare_select_hd(sigma)
    torch.cuda.synchronize()
    ss.check_flag(flag, a.kernel)
    print(f"{a.kernel} on {wl.name}: {a.reps} launches ok")


if __name__ == "__main__":
    main()
