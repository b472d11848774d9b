"""Times semshare_hash beside its operand stream alone, on one workload's rows.

    python -m paper_2509_24832_gb300.operand_stream [--workload llama8b-5k] [--reps 20]

semshare_probe_operand_stream moves the hash kernel's operand blocks (the 128 x 64 embedding
block and the nbits x 64 hyperplane block of every (tile, K block) iteration, one CTA per SM,
the same TMA boxes) through shared memory with no rotation and no MMA, so its launch time is the
floor that the operand traffic alone sets for the hash kernel.  Both are timed with CUDA events
after each of two L2 flushes:

  write   a 512 MB buffer is written, as bench.py does between steps; L2 is then full of dirty
          lines, which the next kernel's reads must write back to DRAM as they evict them
  clean   the same write, then a 256 MB buffer is read; L2 then holds only clean lines

Prints one line per (flush, case) and a JSON summary.  Rows are the workload's rows rounded
down to a multiple of 128 (the probe's unit); embeddings are seeded N(0,1) rows in bf16."""
from __future__ import annotations

import argparse
import json
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
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--workload", default="llama8b-5k", choices=sorted(workloads.WORKLOADS))
    p.add_argument("--reps", type=int, default=20)
    a = p.parse_args(argv)
    wl = workloads.WORKLOADS[a.workload]
    if wl.emb_dtype != "bf16":
        raise SystemExit("the probe streams bf16 rows; pick a workload with bf16 embeddings")
    dev = torch.device("cuda")
    rows = (wl.n_ref + wl.n_batch * wl.n_tgt) // 128 * 128
    g = torch.Generator(device=dev)
    g.manual_seed(wl.base_seed)
    emb = torch.randn((rows, wl.d), device=dev, generator=g).to(torch.bfloat16)
    hyp = torch.from_numpy(workloads.hyperplanes(wl).view(np.int16)).to(dev).view(torch.bfloat16)
    pos = (torch.arange(rows, dtype=torch.int32, device=dev) % wl.n_ref).contiguous()
    table = ss.semshare_rope_table(wl.d, 10000.0, device=dev)
    codes = torch.empty((rows, wl.nbits // 32), dtype=torch.int32, device=dev)
    ws = torch.zeros(max(256, ss.semshare_hash_workspace_size(rows, wl.d, wl.nbits)), dtype=torch.uint8, device=dev)
    flag = ss.new_err_flag(dev)
    write_buf = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    read_buf = torch.ones(64 << 20, dtype=torch.float32, device=dev)

    cases = {
        "embedding blocks, 4 slots": lambda: ss.semshare_probe_operand_stream(emb, None, 4, 0, flag),
        "embedding blocks, 12 slots": lambda: ss.semshare_probe_operand_stream(emb, None, 12, 0, flag),
        "embedding + hyperplane blocks, 4 slots, prefetch 8": lambda: ss.semshare_probe_operand_stream(
            emb, hyp, 4, 8, flag),
        "semshare_hash": lambda: ss.semshare_hash(emb, table, hyp, pos, codes=codes, workspace=ws, err_flag=flag),
    }
    out = {"workload": a.workload, "rows": rows, "d": wl.d, "nbits": wl.nbits,
           "operand_bytes": rows * wl.d * 2, "us": {}}
    for flush in ("write", "clean"):
        for name, fn in cases.items():
            ts = []
            for r in range(a.reps + 3):
                write_buf.zero_()
                if flush == "clean":
                    read_buf.sum()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                fn()
                e1.record()
                e1.synchronize()
                if r >= 3:
                    ts.append(e0.elapsed_time(e1) * 1e3)
            ss.check_flag(flag, name)
            us = float(np.median(ts))
            out["us"][f"{flush}: {name}"] = us
            print(f"{flush:5s} flush  {name:52s} {us:8.1f} us  {rows * wl.d * 2 / us / 1e3:7.0f} GB/s of embedding rows",
                  flush=True)
    print(json.dumps(out))


if __name__ == "__main__":
    main()
