#!/usr/bin/env python
"""Throughput of SemShareKV's fuzzy token-matching path on GB300: target tokens matched and
gathered per second.

One step = the whole path over one synthetic matching problem resident in HBM:
  semshare_hash      RoPE + LSH codes of the reference and target rows (one launch)
  semshare_match     Hamming nearest reference token of every target token
  semshare_gather_kv reference K/V rows rearranged into the target's order, all layers/heads
value = target tokens of all ranks / max over ranks of the mean device time of a step.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl gb300|reference]

With N > 1 it runs under torch.distributed.run, one rank per GPU; every rank solves its own
independent problem (different seed): weak scaling with no collective in the data path.
`--impl reference` times the CPU oracle (the plain fp64 restatement of the paper, test
infrastructure) on bounded samples of the same workload instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "target tokens matched+gathered/sec at 5k tokens"
DEFAULT_WORKLOAD = "llama8b-5k"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20
LAUNCHES_PER_STEP = 5  # hash 1, match 3 (tc: expand + key reset, search, split; popc: key init, search, split), gather 1

# DRAM bytes per launch from ncu captures (dram__bytes_read.sum + dram__bytes_write.sum),
# valid only while the kernel source has the recorded sha256 prefix.
NCU_TRAFFIC = {
    "gather": {"file": "gather.cu", "sha": "e03583daf19419cb", "bytes_per_launch": 1092.8e6, "targets": 5120},
    "hash": {"file": "hash.cu", "sha": "7cf51b07f7d5874d", "bytes_per_launch": 92.63e6, "targets": 5120},
    "match": {"file": "match.cu", "sha": "69ac4b7ce5b193e4", "bytes_per_launch": 0.3845e6, "targets": 5120},
    "match_tc": {"file": "match_tc.cu", "sha": "3bcc238fb9cfe314", "bytes_per_launch": 2.712e6, "targets": 5120},
}


def parse_args(argv=None):
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(workloads.WORKLOADS))
    p.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    p.add_argument("--matcher", default="tc", choices=["tc", "popc"],
                   help="Hamming search: tensor-core GEMM (semshare_match_tc) or xor/popc (semshare_match)")
    p.add_argument("--e2e-steps", type=int, default=20)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-clocks", action="store_true")
    return p.parse_args(argv)


# ---- multi-rank plumbing (weak scaling, no data-path collective) ------------------------------

def dist_info():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def reduce_max(value: float, device=None) -> float:
    """Max of a per-rank float over all ranks (identity without a process group)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(device=None):
    import torch.distributed as dist

    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        if device is not None and dist.get_backend() == "nccl":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# ---- algorithmic work per step (roofline numerators) -----------------------------------------

def work(wl: workloads.Workload) -> dict:
    rows = wl.n_ref + wl.n_batch * wl.n_tgt
    esz = 4 if wl.emb_dtype == "f32" else 2
    L, H, hd = wl.kv
    n_t = wl.n_batch * wl.n_tgt
    return {
        "hash_flops": 2.0 * rows * wl.d * wl.nbits,
        "hash_bytes": rows * wl.d * esz + rows * wl.nbits / 8 + rows * 4 + wl.nbits * wl.d * 2,
        "match_wordops": float(n_t) * wl.n_ref * (wl.nbits // 32),
        "match_bytes": (n_t + wl.n_ref) * wl.nbits / 8 + n_t * 8,
        "gather_bytes": 2.0 * 2.0 * n_t * L * H * hd * 2,  # K and V, read + write
        "targets": n_t,
        "rows": rows,
    }


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return {k: float(pk[k]) for k in FALLBACK_PEAKS}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def popc_peak_wordops(sm_mhz: float, sms: int) -> float:
    """Word-op ceiling of the xor/popc/add Hamming loop: 16 population counts per clock per SM
    (the CUDA C++ Programming Guide's throughput table for compute capability 10.x); one
    word-op needs one popc, the xor and add issue on other pipes."""
    return 16.0 * sms * sm_mhz * 1e6


def kernel_sha(name: str) -> str:
    p = os.path.join(ROOT, "paper_2509_24832_gb300", "csrc", name)
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


# ---- clocks -------------------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.proc = None
        self.gpu_id = gpu_id

    def __enter__(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100"]
        if self.gpu_id:
            cmd += ["-i", self.gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()
        return False

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---- the GPU arm --------------------------------------------------------------------------------

class Problem:
    """Device buffers of one matching problem and the three library calls of a step."""

    def __init__(self, wl: workloads.Workload, device, seed: int, matcher: str = "tc"):
        import torch

        import paper_2509_24832_gb300 as ss

        self.ss, self.wl, self.dev, self.matcher = ss, wl, device, matcher
        emb, pos, _ = workloads.prompt_rows(wl, seed=seed)
        self.host_emb, self.host_pos = emb, pos
        if wl.emb_dtype == "f32":
            self.emb = torch.from_numpy(emb).to(device)
        else:
            self.emb = torch.from_numpy(emb.view(np.int16)).to(device).view(torch.bfloat16)
        self.pos = torch.from_numpy(pos).to(device)
        R = workloads.hyperplanes(wl, seed=seed)
        self.hyp = torch.from_numpy(R.view(np.int16)).to(device).view(torch.bfloat16)
        self.table = ss.semshare_rope_table(wl.d, 10000.0, device=device)
        rows = emb.shape[0]
        w = wl.nbits // 32
        n_t = wl.n_batch * wl.n_tgt
        self.codes = torch.empty((rows, w), dtype=torch.int32, device=device)
        self.idx = torch.empty(n_t, dtype=torch.int32, device=device)
        self.dist = torch.empty(n_t, dtype=torch.int32, device=device)
        self.ws = torch.empty(ss.semshare_match_workspace_size(n_t), dtype=torch.uint8, device=device)
        self.tc_ws = torch.empty(max(256, ss.semshare_match_tc_workspace_size(n_t, wl.n_ref, wl.nbits)),
                                 dtype=torch.uint8, device=device)
        self.hash_ws = torch.zeros(max(256, ss.semshare_hash_workspace_size(rows, wl.d, wl.nbits)), dtype=torch.uint8,
                                   device=device)
        segs = [workloads.kv_cache_device(wl, device, seed=seed, segment=s) for s in range(wl.n_seg)]
        self.ref_k = [s[0] for s in segs]
        self.ref_v = [s[1] for s in segs]
        L, H, hd = wl.kv
        self.out_k = torch.empty((wl.n_batch, L, H, wl.n_tgt, hd), dtype=torch.bfloat16, device=device)
        self.out_v = torch.empty_like(self.out_k)
        self.flag = ss.new_err_flag(device)

    def hash(self):
        self.ss.semshare_hash(self.emb, self.table, self.hyp, self.pos, codes=self.codes, err_flag=self.flag,
                              workspace=self.hash_ws)

    def match(self):
        n_ref = self.wl.n_ref
        if self.matcher == "tc":
            self.ss.semshare_match_tc(self.codes[n_ref:], self.codes[:n_ref], idx=self.idx, dist=self.dist,
                                      workspace=self.tc_ws, err_flag=self.flag)
        else:
            self.ss.semshare_match(self.codes[n_ref:], self.codes[:n_ref], idx=self.idx, dist=self.dist,
                                   workspace=self.ws)

    def gather(self):
        self.ss.semshare_gather_kv(self.ref_k, self.ref_v, self.idx.view(self.wl.n_batch, self.wl.n_tgt),
                                   out_k=self.out_k, out_v=self.out_v, err_flag=self.flag)

    def step(self, ev=None):
        if ev:
            ev[0].record()
        self.hash()
        if ev:
            ev[1].record()
        self.match()
        if ev:
            ev[2].record()
        self.gather()
        if ev:
            ev[3].record()


def run_gpu_arm(args, rank, world, local_rank):
    import torch

    import paper_2509_24832_gb300 as ss

    ss.load()
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    wl = workloads.WORKLOADS[args.workload]
    seed = wl.base_seed + 7919 * rank
    prob = Problem(wl, device, seed, args.matcher)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

    for _ in range(max(args.warmup, 3)):
        prob.step()
    torch.cuda.synchronize()
    ss.check_flag(prob.flag, "warm-up")

    K = args.steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
    except Exception:
        gpu_id = None
    sampler = ClockSampler(None if args.no_clocks else gpu_id)
    if args.no_clocks:
        sampler.proc = None
    barrier(device)
    torch.cuda.synchronize()
    with (sampler if not args.no_clocks else _Null()):
        t_wall0 = time.perf_counter()
        for k in range(K):
            flush.zero_()  # evict the previous step's lines from the 129 MB L2 (untimed gap)
            prob.step(evs[k])
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall0
    barrier(device)
    ss.check_flag(prob.flag, "timed steps")

    st = np.array([[evs[k][0].elapsed_time(evs[k][1]), evs[k][1].elapsed_time(evs[k][2]),
                    evs[k][2].elapsed_time(evs[k][3])] for k in range(K)])
    ms_local = float(st.sum(axis=1).mean())
    ms_step = reduce_max(ms_local, device)
    stage_ms = {n: reduce_max(float(st[:, i].mean()), device) for i, n in enumerate(["hash", "match", "gather"])}
    W = work(wl)
    value = world * W["targets"] / (ms_step * 1e-3)

    peaks, peak_src = load_peaks()
    props = torch.cuda.get_device_properties(device)
    clocks = sampler.summary() if not args.no_clocks else None
    sm_mhz = (clocks or {}).get("sm_mhz") or 2070.0
    stages = {
        "hash": {"ms": stage_ms["hash"], "tflops": W["hash_flops"] / (stage_ms["hash"] * 1e-3) / 1e12,
                 "gbs": W["hash_bytes"] / (stage_ms["hash"] * 1e-3) / 1e9},
        "match": {"ms": stage_ms["match"], "gwordops": W["match_wordops"] / (stage_ms["match"] * 1e-3) / 1e9},
        "gather": {"ms": stage_ms["gather"], "gbs": W["gather_bytes"] / (stage_ms["gather"] * 1e-3) / 1e9},
    }
    stages["hash"]["frac_tensor"] = stages["hash"]["tflops"] / peaks["bf16_tflops"]
    stages["hash"]["frac_hbm"] = stages["hash"]["gbs"] / peaks["hbm_gbs"]
    popc_peak = popc_peak_wordops(sm_mhz, props.multi_processor_count)
    stages["match"]["matcher"] = args.matcher
    if args.matcher == "popc":
        stages["match"]["frac_popc"] = stages["match"]["gwordops"] * 1e9 / popc_peak
    else:
        # the GEMM over padded code bits: 2 * n_t * n_ref * kpad fp8 flops; fp8 peak = 2 x bf16 (nominal ratio)
        kpad = ((wl.nbits + 127) // 128) * 128
        fl = 2.0 * W["targets"] * wl.n_ref * kpad
        stages["match"]["tflops_fp8"] = fl / (stage_ms["match"] * 1e-3) / 1e12
        stages["match"]["frac_fp8_tensor"] = stages["match"]["tflops_fp8"] / (2.0 * peaks["bf16_tflops"])
    stages["gather"]["frac_hbm"] = stages["gather"]["gbs"] / peaks["hbm_gbs"]

    dominant = max(stage_ms, key=stage_ms.get)
    if dominant == "gather":
        roof = {"kernel": "kv_gather_kernel", "bound": "hbm", "achieved": stages["gather"]["gbs"],
                "peak": peaks["hbm_gbs"], "unit": "GB/s"}
        tr = NCU_TRAFFIC.get("gather")
    elif dominant == "hash":
        roof = {"kernel": "lsh_hash_kernel", "bound": "tensor", "achieved": stages["hash"]["tflops"],
                "peak": peaks["bf16_tflops"], "unit": "TFLOP/s"}
        tr = NCU_TRAFFIC.get("hash")
    elif args.matcher == "popc":
        roof = {"kernel": "hamming_nn_kernel", "bound": "alu", "achieved": stages["match"]["gwordops"],
                "peak": popc_peak / 1e9, "unit": "Gwordop/s"}
        tr = NCU_TRAFFIC.get("match")
    else:
        roof = {"kernel": "hamming_tc_kernel", "bound": "tensor", "achieved": stages["match"]["tflops_fp8"],
                "peak": 2.0 * peaks["bf16_tflops"], "unit": "TFLOP/s"}
        tr = NCU_TRAFFIC.get("match_tc")
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"
    if tr and tr.get("sha") == kernel_sha(tr["file"]):
        roof["traffic"] = tr["bytes_per_launch"] * (W["targets"] / tr["targets"])
    else:
        roof["traffic"] = None

    e2e = run_e2e(args, prob, device)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, prob)

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if wl.emb_dtype == "bf16" else "f32",
        "data": "synthetic (seeded; see workloads.py)",
        "config": {"workload": wl.name, "n_ref": wl.n_ref, "n_tgt": wl.n_tgt, "n_batch": wl.n_batch,
                   "n_seg": wl.n_seg, "d": wl.d, "nbits": wl.nbits, "kv": list(wl.kv),
                   "parallelism": f"replicas x{world}", "l2": "flushed before every step (256 MB write)",
                   "matcher": args.matcher},
        "roofline": roof, "stages": stages, "e2e": e2e, "cpu_baseline": cpu,
        "gpu_launches": LAUNCHES_PER_STEP * K, "clocks": clocks, "wall_s_timed": reduce_max(t_wall, device),
        "impl": "gb300",
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


class _Null:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False


def run_e2e(args, prob: Problem, device):
    """Same metric through the public API with host buffers: every step copies its inputs
    (embedding rows, positions, the reference K/V cache) from pinned host memory, runs the
    three calls and reads the match result (idx, dist) back."""
    import torch

    wl = prob.wl
    h_emb = prob.emb.cpu().pin_memory()
    h_pos = prob.pos.cpu().pin_memory()
    h_k = [t.cpu().pin_memory() for t in prob.ref_k]
    h_v = [t.cpu().pin_memory() for t in prob.ref_v]
    h_idx = torch.empty_like(prob.idx, device="cpu").pin_memory()
    h_dist = torch.empty_like(prob.dist, device="cpu").pin_memory()
    h2d = h_emb.numel() * h_emb.element_size() + h_pos.numel() * 4 + \
        sum(t.numel() * t.element_size() for t in h_k + h_v)
    d2h = (h_idx.numel() + h_dist.numel()) * 4

    def one():
        prob.emb.copy_(h_emb, non_blocking=True)
        prob.pos.copy_(h_pos, non_blocking=True)
        for d, h in zip(prob.ref_k + prob.ref_v, h_k + h_v):
            d.copy_(h, non_blocking=True)
        prob.step()
        h_idx.copy_(prob.idx, non_blocking=True)
        h_dist.copy_(prob.dist, non_blocking=True)

    for _ in range(3):
        one()
    torch.cuda.synchronize()
    n = max(1, args.e2e_steps)
    times = []
    for _ in range(n):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        one()
        b.record()
        b.synchronize()
        _ = int(h_idx[0])  # the host reads the result
        times.append(a.elapsed_time(b))
    ms = reduce_max(float(np.mean(times)), device)
    _, world, _ = dist_info()
    return {"value": world * wl.n_batch * wl.n_tgt / (ms * 1e-3), "unit": "tokens/s", "ms_per_step": ms,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)}


# ---- CPU oracle (baseline leg and reference arm) -----------------------------------------------

def _oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np, tsel):
    """The oracle's whole path for the target tokens `tsel` of prompt 0: hash them plus an
    equal share of reference rows, match them against every reference code, gather their K/V
    rows.  Returns seconds."""
    n_t = len(tsel)
    share = max(1, int(round(n_t * wl.n_ref / (wl.n_batch * wl.n_tgt))))
    t0 = time.perf_counter()
    oracle.hash_codes(emb[:share], pos[:share], R)  # the reference rows' share of hashing
    tc, _ = oracle.hash_codes(emb[wl.n_ref + tsel], pos[wl.n_ref + tsel], R)
    idx, _ = oracle.match(tc, ref_codes)
    oracle.gather_kv(k_np, v_np, idx)
    return time.perf_counter() - t0


def _oracle_inputs(oracle, wl, emb, pos, R, k_dev=None, v_dev=None):
    ref_codes, _ = oracle.hash_codes(emb[: wl.n_ref], pos[: wl.n_ref], R)
    if k_dev is not None:
        k_np = [t.cpu().view(__import__("torch").int16).numpy().view(np.uint16) for t in k_dev]
        v_np = [t.cpu().view(__import__("torch").int16).numpy().view(np.uint16) for t in v_dev]
    else:
        k_np, v_np = [], []
        for s in range(wl.n_seg):
            k, v = workloads.kv_cache(wl, segment=s)
            k_np.append(k)
            v_np.append(v)
    return ref_codes, k_np, v_np


def cpu_baseline(wl, prob):
    """The oracle as it stands on the host cores: one bounded sample of the workload."""
    import oracle

    oracle.build()
    emb, pos = prob.host_emb, prob.host_pos
    R = prob.hyp.cpu().view(__import__("torch").int16).numpy().view(np.uint16)
    ref_codes, k_np, v_np = _oracle_inputs(oracle, wl, emb, pos, R, prob.ref_k, prob.ref_v)
    n_s = min(wl.n_tgt, 5120)
    tsel = np.arange(n_s)
    secs = _oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np, tsel)
    return {"value": n_s / secs, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{n_s} target tokens of prompt 0 (hash of them + {n_s * wl.n_ref // (wl.n_batch * wl.n_tgt)} "
                      f"reference rows, match against all {wl.n_ref} reference codes, gather of their "
                      f"{wl.n_layers}x{wl.n_heads} K/V rows); seconds={secs:.2f}"}


def run_reference_arm(args, rank, world):
    if rank != 0:
        return
    import oracle

    oracle.build()
    wl = workloads.WORKLOADS[args.workload]
    emb, pos, _ = workloads.prompt_rows(wl, batches=[0])
    R = workloads.hyperplanes(wl)
    ref_codes, k_np, v_np = _oracle_inputs(oracle, wl, emb, pos, R)
    per_step = 64
    g = np.random.default_rng(wl.base_seed)
    for _ in range(max(args.warmup, 3)):
        _oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np, np.sort(g.choice(wl.n_tgt, per_step, False)))
    secs = []
    for _ in range(args.steps):
        secs.append(_oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np,
                                   np.sort(g.choice(wl.n_tgt, per_step, False))))
    ms = 1e3 * float(np.mean(secs))
    value = per_step / (ms * 1e-3)
    sample = (f"per step {per_step} random target tokens of prompt 0: hash of them plus their share of reference "
              f"rows, match against all {wl.n_ref} reference codes, gather of their K/V rows")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded; see workloads.py)",
        "config": {"workload": wl.name, "n_ref": wl.n_ref, "n_tgt": wl.n_tgt, "n_batch": wl.n_batch,
                   "n_seg": wl.n_seg, "d": wl.d, "nbits": wl.nbits, "kv": list(wl.kv)},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main(argv=None):
    args = parse_args(argv)
    rank, world, local_rank = dist_info()
    if world > 1:
        import torch.distributed as dist

        if args.impl == "reference":
            if rank != 0:
                return 0
            world_eff = world
            run_reference_arm(args, 0, world_eff)
            return 0
        import torch

        torch.cuda.set_device(local_rank)
        dist.init_process_group(backend="nccl")
    if args.impl == "reference":
        run_reference_arm(args, rank, world)
    else:
        run_gpu_arm(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
