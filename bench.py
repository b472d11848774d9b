#!/usr/bin/env python
"""Throughput of SemShareKV's fuzzy token-matching path on GB300: target tokens matched and
gathered per second.

One step = the whole path over one synthetic matching problem resident in HBM:
  semshare_hash      RoPE + LSH codes of the reference and target rows (one launch)
  semshare_match     Hamming nearest reference token of every target token
  semshare_gather_kv reference K/V rows rearranged into the target's order, all layers/heads
value = target tokens of all ranks / max over ranks of the mean device time of a step.

`--workload retrieve-16x4096` times the path with reference retrieval in front (Sec. 3.2):
16 stored prompts whose codes were computed when they were stored; per step the target is
hashed without rotary encoding, the most similar stored prompt is retrieved
(semshare_retrieve), the target is hashed with it, matched against the winner's codes
(semshare_match_tc_selected reads the choice on the device) and the winner's K/V rows are
gathered -- all enqueued back to back, with no host round trip.

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
METRIC_RETRIEVE = "target tokens retrieved+matched+gathered/sec"
DEFAULT_WORKLOAD = "llama8b-5k"
ALL_WORKLOADS = {**workloads.WORKLOADS, **workloads.RETRIEVAL_WORKLOADS}
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 512 << 20
NVTX = [False]  # --nvtx: stage ranges on the timeline


def nvtx_push(name: str):
    if NVTX[0]:
        import torch

        torch.cuda.nvtx.range_push(name)


def nvtx_pop():
    if NVTX[0]:
        import torch

        torch.cuda.nvtx.range_pop()

# DRAM bytes per launch from ncu captures (dram__bytes_read.sum + dram__bytes_write.sum) on a
# workload, valid only for that workload and while the kernel source has the recorded sha256
# prefix (the traffic depends on the index pattern, e.g. how often a gathered row repeats).
NCU_TRAFFIC = {
    ("gather", "llama8b-5k"): {"file": "gather.cu", "sha": "8b2db284dbc5f706", "bytes_per_launch": 1079.6e6},
    ("gather_retained", "llama8b-5k"): {"file": "gather.cu", "sha": "8b2db284dbc5f706", "bytes_per_launch": 661.7e6},
    ("hash", "llama8b-5k"): {"file": "hash_2sm.cu", "sha": "2996a1dfad32b843", "bytes_per_launch": 87.13e6},
    ("match_tc", "llama8b-5k"): {"file": "match_tc.cu", "sha": "e1ef461ac0e1f77d", "bytes_per_launch": 2.72e6},
    ("retrieve", "retrieve-16x4096"): {"file": "match_tc.cu", "sha": "e1ef461ac0e1f77d", "bytes_per_launch": 18.41e6},
}


def parse_args(argv=None):
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(ALL_WORKLOADS))
    p.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    p.add_argument("--matcher", default="tc", choices=["tc", "signs", "popc"],
                   help="Hamming search: tensor-core GEMM from the packed codes (semshare_match_tc: expansion, "
                        "search, key split), the same search on the sign rows the hash writes beside the codes "
                        "(semshare_hash_signs + semshare_match_tc_signs, one launch) or xor/popc (semshare_match)")
    p.add_argument("--e2e-steps", type=int, default=20)
    p.add_argument("--rope", default="interleaved", choices=["interleaved", "half"],
                   help="rotary pairing: (2k, 2k+1) as Eq. 1 prints it, or (k, k + d/2)")
    p.add_argument("--retain", action="store_true",
                   help="gather only each layer's retained tokens (Sec. 3.3.4; synthetic schedule: 0.8 on the "
                        "first layer, then 0.98 per layer; one-prompt workloads)")
    p.add_argument("--hd", action="store_true",
                   help="append the first layer's KV deviation against a (synthetic) recomputed first layer "
                        "and the HD-token selection (App. A.4, Insight 1) to the step")
    p.add_argument("--graph", action="store_true",
                   help="capture one step in a CUDA graph and replay it for the timed steps (the host "
                        "enqueues one graph instead of the library calls)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-clocks", action="store_true")
    p.add_argument("--nvtx", action="store_true",
                   help="name each stage of a step with an NVTX range (for a profiler's timeline)")
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
    if wl.recipe == "retrieve":
        return work_retrieve(wl)
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
        # first layer of every target prompt: reused and recomputed K and V read, 3 floats out
        "deviation_bytes": 4.0 * n_t * H * hd * 2 + 3.0 * 4 * n_t,
        "select_bytes": 4.0 * n_t + 4.0 * ((n_t * 40 + 99) // 100),
        "targets": n_t,
        "rows": rows,
    }


def work_retrieve(wl: workloads.Workload) -> dict:
    """Retrieval step: the target rows hashed twice in one launch (plain and rotary codes), the
    retrieval GEMM over the whole pool, the match against one member, the gather of one member's
    rows."""
    n_t = wl.n_tgt
    esz = 4 if wl.emb_dtype == "f32" else 2
    L, H, hd = wl.kv
    kpad = ((wl.nbits + 127) // 128) * 128
    return {
        "hash_flops": 2.0 * 2.0 * n_t * wl.d * wl.nbits,
        "hash_bytes": n_t * wl.d * esz + 2 * n_t * wl.nbits / 8 + n_t * 4 + wl.nbits * wl.d * 2,
        "retrieve_flops": 2.0 * n_t * wl.n_ref * kpad,
        "match_wordops": float(n_t) * wl.seg_len * (wl.nbits // 32),
        "match_flops": 2.0 * n_t * wl.seg_len * kpad,
        "gather_bytes": 2.0 * 2.0 * n_t * L * H * hd * 2,
        "targets": n_t,
        "rows": n_t,
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
    """Word-op ceiling of the xor/popc/add Hamming loop from the CUDA C++ Programming Guide's
    throughput table (16 population counts per clock per SM for compute capability 10.x); one
    word-op needs one popc, the xor and add issue on other pipes.  A cross-check for the measured
    rate below."""
    return 16.0 * sms * sm_mhz * 1e6


PROBE_CHAINS = 8  # SEMSHARE_PROBE_CHAINS (include/semshare_probe.h): word operations per thread and iteration


def load_probe():
    """libsemshare_probe.so (measurement support, built beside libsemshare.so by build.py)."""
    import ctypes

    from paper_2509_24832_gb300 import build

    if not os.path.exists(build.PROBE_LIB):
        raise RuntimeError(f"{build.PROBE_LIB} is missing: build the library first")
    lib = ctypes.CDLL(build.PROBE_LIB)
    lib.semshare_probe_hamming_threads.argtypes = []
    lib.semshare_probe_hamming_threads.restype = ctypes.c_int64
    lib.semshare_probe_hamming_rate.argtypes = [ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]
    lib.semshare_probe_hamming_rate.restype = ctypes.c_int
    return lib


def measure_hamming_rate(device, iters: int = 1 << 14, reps: int = 5) -> float:
    """Sustained xor/popc/add word-ops per second of this GPU (semshare_probe_hamming_rate:
    independent chains in registers, every SM fully occupied), best of `reps` launches timed
    with CUDA events after a warm-up launch."""
    import torch

    probe = load_probe()
    threads = int(probe.semshare_probe_hamming_threads())
    if threads <= 0:
        raise RuntimeError("semshare_probe_hamming_threads failed")
    sink = torch.empty(threads, dtype=torch.int32, device=device)

    def launch():
        st = probe.semshare_probe_hamming_rate(iters, sink.data_ptr(), sink.numel(),
                                               torch.cuda.current_stream(device).cuda_stream)
        if st != 0:
            raise RuntimeError(f"semshare_probe_hamming_rate: status {st}")

    ops = threads * iters * PROBE_CHAINS
    launch()
    torch.cuda.synchronize()
    best = float("inf")
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        launch()
        b.record()
        b.synchronize()
        best = min(best, a.elapsed_time(b) * 1e-3)
    return ops / best


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

    STAGES = ("hash", "match", "gather")

    def __init__(self, wl: workloads.Workload, device, seed: int, matcher: str = "tc", with_hd: bool = False,
                 with_retain: bool = False):
        import torch

        import paper_2509_24832_gb300 as ss

        self.ss, self.wl, self.dev, self.matcher = ss, wl, device, matcher
        self.rope_layout = "interleaved"
        emb, pos, src = workloads.prompt_rows(wl, seed=seed)
        self.host_emb, self.host_pos, self.src = emb, pos, src
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
        # matcher "signs": the hash also writes the sign rows, which the one-launch search reads; its
        # workspace starts 0xFF-filled and every call leaves it so
        self.signs = torch.empty((rows, ss.semshare_signs_pitch(wl.nbits)), dtype=torch.uint8, device=device) \
            if matcher == "signs" else None
        self.signs_ws = torch.full((max(512, ss.semshare_match_tc_signs_workspace_size(n_t)),), 0xFF,
                                   dtype=torch.uint8, device=device) if matcher == "signs" else None
        # library launches per step: hash 1; match: signs 1 (2 above the fused split's target count),
        # tc 3 (expansion + key reset, search, key split), popc 3 (key init, search, split); gather 1
        self.LAUNCHES_PER_STEP = 2 + ({"signs": 1 if n_t <= ss.MATCH_SIGNS_FUSED_MAX_TARGETS else 2}.get(matcher, 3))
        self.hash_ws = torch.zeros(max(256, ss.semshare_hash_workspace_size(rows, wl.d, wl.nbits)), dtype=torch.uint8,
                                   device=device)
        segs = [workloads.kv_cache_device(wl, device, seed=seed, segment=s) for s in range(wl.n_seg)]
        self.ref_k = [s[0] for s in segs]
        self.ref_v = [s[1] for s in segs]
        L, H, hd = wl.kv
        self.out_k = torch.empty((wl.n_batch, L, H, wl.n_tgt, hd), dtype=torch.bfloat16, device=device)
        self.out_v = torch.empty_like(self.out_k)
        self.flag = ss.new_err_flag(device)
        self.retain = with_retain
        # e2e fetch mode: layer groups whose gathers overlap the next group's copy (plain gather only)
        self.fetch_groups = E2E_LAYER_GROUPS if not with_retain and L >= E2E_LAYER_GROUPS else 1
        if with_retain:
            if wl.n_batch != 1 or with_hd:
                raise ValueError("--retain takes a one-prompt workload and no --hd")
            self.counts = ss.retain_counts(wl.n_tgt, workloads.retain_alphas(L), workloads.RETAIN_DEN)
            ret = workloads.retained_tokens(wl.n_tgt, self.counts, seed)
            self.ret = torch.from_numpy(np.concatenate(ret)).to(device)
            self.ret_off = [0] + list(np.cumsum(self.counts))
            self.out_k = torch.empty((L, H, self.counts[0], hd), dtype=torch.bfloat16, device=device)
            self.out_v = torch.empty_like(self.out_k)
        self.hd = with_hd
        if with_hd:
            # a synthetic recomputed first layer per target prompt, [B][H][T][hd] (the layer-0 view
            # of the gathered cache has the same shape, batch standing in for the layer index)
            ks, vs = [], []
            k0 = torch.cat([t[:1] for t in self.ref_k], dim=2)  # first layer of every member: global rows
            v0 = torch.cat([t[:1] for t in self.ref_v], dim=2)
            for b in range(wl.n_batch):
                k_rc, v_rc = workloads.recomputed_kv_device(wl, device, k0, v0, src[b], seed=seed + b)
                ks.append(k_rc[0])
                vs.append(v_rc[0])
            self.rc_k, self.rc_v = torch.stack(ks), torch.stack(vs)
            del ks, vs, k0, v0
            self.sigma = torch.empty((wl.n_batch, wl.n_tgt), dtype=torch.float32, device=device)
            self.hd_k = ss.hd_count(wl.n_tgt)
            self.hd_idx = torch.empty((wl.n_batch, self.hd_k), dtype=torch.int32, device=device)
            self.STAGES = Problem.STAGES + ("deviation", "select")
            self.LAUNCHES_PER_STEP += 2

    def deviation(self):
        self.ss.semshare_kv_deviation(self.out_k[:, 0], self.out_v[:, 0], self.rc_k, self.rc_v, sigma_kv=self.sigma)

    def select(self):
        self.ss.semshare_select_hd(self.sigma, self.hd_k, hd_idx=self.hd_idx)

    def hash(self):
        self.hash_rows(self.emb, self.pos, self.codes, self.signs, self.hash_ws)

    def hash_rows(self, emb, pos, codes, signs, ws):
        """The hash of some rows (all of them, or only the target's), with the sign rows when the
        matcher reads them."""
        if signs is not None:
            self.ss.semshare_hash_signs(emb, self.table, self.hyp, pos, codes=codes, signs=signs, err_flag=self.flag,
                                        workspace=ws, rope_layout=self.rope_layout)
        else:
            self.ss.semshare_hash(emb, self.table, self.hyp, pos, codes=codes, err_flag=self.flag, workspace=ws,
                                  rope_layout=self.rope_layout)

    def match(self):
        n_ref = self.wl.n_ref
        if self.matcher == "signs":
            self.ss.semshare_match_tc_signs(self.signs[n_ref:], self.signs[:n_ref], self.wl.nbits, idx=self.idx,
                                            dist=self.dist, workspace=self.signs_ws, err_flag=self.flag)
        elif self.matcher == "tc":
            self.ss.semshare_match_tc(self.codes[n_ref:], self.codes[:n_ref], idx=self.idx, dist=self.dist,
                                      workspace=self.tc_ws, err_flag=self.flag)
        else:
            self.ss.semshare_match(self.codes[n_ref:], self.codes[:n_ref], idx=self.idx, dist=self.dist,
                                   workspace=self.ws)

    def gather(self, src_k=None, src_v=None):
        src_k = self.ref_k if src_k is None else src_k
        src_v = self.ref_v if src_v is None else src_v
        if self.retain:
            self.ss.semshare_gather_kv_retained(src_k, src_v, self.idx, self.ret, self.ret_off,
                                                out_k=self.out_k, out_v=self.out_v, err_flag=self.flag)
            return
        self.ss.semshare_gather_kv(src_k, src_v, self.idx.view(self.wl.n_batch, self.wl.n_tgt),
                                   out_k=self.out_k, out_v=self.out_v, err_flag=self.flag)

    def step(self, ev=None):
        stages = [self.hash, self.match, self.gather] + ([self.deviation, self.select] if self.hd else [])
        if ev:
            ev[0].record()
        for i, (name, fn) in enumerate(zip(self.STAGES, stages)):
            nvtx_push(name)
            fn()
            nvtx_pop()
            if ev:
                ev[i + 1].record()

    def unique_rows(self) -> int:
        """Distinct reference rows the current match selects (over every target prompt)."""
        return int(np.unique(self.idx.cpu().numpy()).size)

    def e2e_plan(self, mode: str = "fetch", ref_cached: bool = False):
        """(one, h2d, d2h, read): a step through the public API with host buffers.  The
        embedding rows and positions are copied in from pinned host memory (with ref_cached only the
        target's: the reference codes were computed once when the reference was stored, reading M
        of the paper, and stay on the device); the reference K/V cache
        stays in pinned host memory, and the gather's rows reach it one of three ways (`mode`):
          fetch     semshare_fetch_rows copies each row the match selects into HBM once, then the
                    gather runs on HBM;
          inplace   the gather reads every selected row across the host link, repeats included;
          copy_all  the whole cache is copied in first, then gathered from HBM;
          kv_resident  the stored cache stays in HBM (no K/V crosses the link).
        The match result (idx, dist) is copied back."""
        import torch

        n_ref = self.wl.n_ref
        emb_d, pos_d = (self.emb[n_ref:], self.pos[n_ref:]) if ref_cached else (self.emb, self.pos)
        h_emb = emb_d.cpu().pin_memory()
        h_pos = pos_d.cpu().pin_memory()
        if ref_cached:
            tgt_codes = self.codes[n_ref:]
            tgt_ws = torch.zeros(max(256, self.ss.semshare_hash_workspace_size(emb_d.shape[0], self.wl.d,
                                                                                 self.wl.nbits)),
                                 dtype=torch.uint8, device=self.dev)
            self.hash()  # the reference codes, once (store time)

            tgt_signs = None if self.signs is None else self.signs[n_ref:]

            def hash_step():
                self.hash_rows(emb_d, pos_d, tgt_codes, tgt_signs, tgt_ws)
        else:
            hash_step = self.hash
        resident = mode == "kv_resident"
        h_k = [] if resident else [t.cpu().pin_memory() for t in self.ref_k]
        h_v = [] if resident else [t.cpu().pin_memory() for t in self.ref_v]
        h_idx = torch.empty_like(self.idx, device="cpu").pin_memory()
        h_dist = torch.empty_like(self.dist, device="cpu").pin_memory()
        kv_bytes = self.e2e_kv_bytes()[mode]
        h2d = h_emb.numel() * h_emb.element_size() + h_pos.numel() * 4 + kv_bytes
        d2h = (h_idx.numel() + h_dist.numel()) * 4
        ss = self.ss
        fetch_ws = torch.empty(max(16, ss.semshare_fetch_workspace_size(self.wl.n_ref)), dtype=torch.uint8,
                               device=self.dev)
        src_k, src_v = (h_k, h_v) if mode == "inplace" else (self.ref_k, self.ref_v)

        # fetch: layer groups in turn -- the rows of group g cross the host link while group g-1 is
        # gathered on HBM from a second stream (the copy kernel leaves room on the SMs for it)
        L = self.wl.n_layers
        groups = [(g * L // E2E_LAYER_GROUPS, (g + 1) * L // E2E_LAYER_GROUPS) for g in range(E2E_LAYER_GROUPS)]
        pipelined = self.fetch_groups > 1
        side = torch.cuda.Stream(self.dev)
        idx2 = self.idx.view(self.wl.n_batch, self.wl.n_tgt)

        def fetch_gather_by_layers():
            main = torch.cuda.current_stream(self.dev)
            side.wait_stream(main)
            for l0, l1 in groups:
                ss.semshare_fetch_rows([t[l0:l1] for t in h_k], [t[l0:l1] for t in h_v], self.idx,
                                       dev_k=[t[l0:l1] for t in self.ref_k], dev_v=[t[l0:l1] for t in self.ref_v],
                                       workspace=fetch_ws, err_flag=self.flag)
                side.wait_stream(main)
                with torch.cuda.stream(side):
                    ss.semshare_gather_kv([t[l0:l1] for t in self.ref_k], [t[l0:l1] for t in self.ref_v], idx2,
                                          out_k=self.out_k[:, l0:l1], out_v=self.out_v[:, l0:l1], err_flag=self.flag)
            main.wait_stream(side)

        def one():
            emb_d.copy_(h_emb, non_blocking=True)
            pos_d.copy_(h_pos, non_blocking=True)
            if mode == "copy_all":
                for d, h in zip(self.ref_k + self.ref_v, h_k + h_v):
                    d.copy_(h, non_blocking=True)
            hash_step()
            self.match()
            if mode == "fetch" and pipelined:
                fetch_gather_by_layers()
            else:
                if mode == "fetch":
                    ss.semshare_fetch_rows(h_k, h_v, self.idx, dev_k=self.ref_k, dev_v=self.ref_v,
                                           workspace=fetch_ws, err_flag=self.flag)
                self.gather(src_k, src_v)
            if self.hd:
                self.deviation()
                self.select()
            h_idx.copy_(self.idx, non_blocking=True)
            h_dist.copy_(self.dist, non_blocking=True)

        return one, h2d, d2h, lambda: int(h_idx[0])

    def e2e_kv_bytes(self) -> dict:
        """K/V bytes crossing the host link per step in each e2e mode."""
        wl = self.wl
        L, H, hd = wl.kv
        row = hd * 2 * 2  # a K and a V row, bf16
        gathered = float(sum(self.counts)) * H if self.retain else float(wl.n_batch * wl.n_tgt) * L * H
        return {"inplace": gathered * row, "fetch": float(self.unique_rows()) * L * H * row,
                "copy_all": float(sum(t.numel() * t.element_size() for t in self.ref_k + self.ref_v)),
                "kv_resident": 0.0}


class RetrieveProblem:
    """Reference retrieval in front of the path (Sec. 3.2).  The stored prompts' codes -- plain
    for retrieval, rotary-encoded for matching -- are computed once when they are stored; a step
    handles one new target prompt:
      hash        codes of the target rows without rotation (for retrieval, which precedes RoPE)
                  and with it (Sec. 3.3.1), in one launch (semshare_hash_pair)
      retrieve    similarity to every stored prompt, the best one (semshare_retrieve)
      match       1-NN against the winner's rotary codes (the choice is read on the device)
      gather      the winner's K/V rows in the target's order (pool rows over every member)"""

    STAGES = ("hash", "retrieve", "match", "gather")
    # hash pair 1, retrieve 3 (expand + key reset, search, per-candidate reduction),
    # selected match 3 (expand, search, split), gather 1
    LAUNCHES_PER_STEP = 8

    def __init__(self, wl: workloads.Workload, device, seed: int, matcher: str = "tc"):
        import torch

        import paper_2509_24832_gb300 as ss

        if matcher not in ("signs", "tc"):
            raise ValueError("the retrieval step uses the tensor-core matcher")
        self.ss, self.wl, self.dev, self.matcher = ss, wl, device, matcher
        emb, pos, _ = workloads.prompt_rows(wl, seed=seed)
        self.host_emb, self.host_pos = emb, pos
        n_pool, n_t, w = wl.n_ref, wl.n_tgt, wl.nbits // 32

        def dev_rows(a):
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(device).view(torch.bfloat16)

        R = workloads.hyperplanes(wl, seed=seed)
        self.hyp = torch.from_numpy(R.view(np.int16)).to(device).view(torch.bfloat16)
        self.table = ss.semshare_rope_table(wl.d, 10000.0, device=device)
        self.flag = ss.new_err_flag(device)
        self.offsets = [m * wl.seg_len for m in range(wl.n_seg + 1)]
        # store time: every stored prompt's codes, plain and rotary (its own positions)
        pool = dev_rows(emb[:n_pool])
        self.pool_rcodes = ss.semshare_hash(pool, None, self.hyp, None, rope_layout="none")
        self.pool_codes = ss.semshare_hash(pool, self.table, self.hyp, torch.from_numpy(pos[:n_pool]).to(device))
        del pool
        self.emb = dev_rows(emb[n_pool:])
        self.pos = torch.from_numpy(pos[n_pool:]).to(device)
        self.t_rcodes = torch.empty((n_t, w), dtype=torch.int32, device=device)
        self.codes = torch.empty((n_t, w), dtype=torch.int32, device=device)
        self.hash_ws = torch.zeros(max(256, ss.semshare_hash_pair_workspace_size(n_t, wl.d, wl.nbits)),
                                   dtype=torch.uint8, device=device)
        self.ret_ws = torch.empty(ss.semshare_retrieve_workspace_size(n_t, n_pool, wl.n_seg, wl.nbits),
                                  dtype=torch.uint8, device=device)
        self.choice = choice = torch.zeros(2, dtype=torch.int32, device=device)  # best, applies
        self.ret = ss.Retrieval(torch.empty(wl.n_seg, dtype=torch.float64, device=device),
                                torch.empty(wl.n_seg, dtype=torch.float64, device=device),
                                choice[:1], choice[1:], None, None)
        self.h_choice = torch.zeros(2, dtype=torch.int32).pin_memory()
        self.idx = torch.empty(n_t, dtype=torch.int32, device=device)
        self.dist = torch.empty(n_t, dtype=torch.int32, device=device)
        self.tc_ws = torch.empty(ss.semshare_match_tc_selected_workspace_size(n_t, self.offsets, wl.nbits),
                                 dtype=torch.uint8, device=device)
        segs = [workloads.kv_cache_device(wl, device, seed=seed, segment=m) for m in range(wl.n_seg)]
        self.ref_k = [m[0] for m in segs]
        self.ref_v = [m[1] for m in segs]
        L, H, hd = wl.kv
        self.out_k = torch.empty((1, L, H, n_t, hd), dtype=torch.bfloat16, device=device)
        self.out_v = torch.empty_like(self.out_k)
        self.load_winner = None  # e2e (copy_all): brings the winner's whole cache in from host memory
        self.fetch_gather = None  # e2e (fetch): brings the selected rows in and gathers them, layer group by group
        self.fetch_groups = E2E_LAYER_GROUPS if L >= E2E_LAYER_GROUPS else 1
        self.gather_src = None   # e2e (inplace): the stored caches in pinned host memory, read in place

    @property
    def winner(self) -> int:
        """The retrieved candidate of the last step (read after the stream has synchronised)."""
        return int(self.h_choice[0])

    def step(self, ev=None):
        """One target prompt, enqueued back to back: the retrieval's choice stays on the device
        and the selected match and the gather read it there (no host round trip)."""
        ss, wl = self.ss, self.wl
        if ev:
            ev[0].record()
        nvtx_push("hash")
        ss.semshare_hash_pair(self.emb, self.table, self.hyp, self.pos, codes_plain=self.t_rcodes,
                              codes_rotary=self.codes, err_flag=self.flag, workspace=self.hash_ws)
        nvtx_pop()
        if ev:
            ev[1].record()
        nvtx_push("retrieve")
        ss.semshare_retrieve(self.t_rcodes, self.pool_rcodes, self.offsets, workspace=self.ret_ws,
                             err_flag=self.flag, out=self.ret)
        nvtx_pop()
        if ev:
            ev[2].record()
        nvtx_push("match")
        ss.semshare_match_tc_selected(self.codes, self.pool_codes, self.offsets, self.ret.best, idx=self.idx,
                                      dist=self.dist, workspace=self.tc_ws, err_flag=self.flag)
        nvtx_pop()
        nvtx_push("gather")
        if self.fetch_gather is not None:
            # e2e fetch mode: the rows come in from host memory and are gathered, in layer groups
            self.fetch_gather()
        else:
            if self.load_winner is not None:
                self.load_winner()
            if ev:
                ev[3].record()
            src_k, src_v = (self.ref_k, self.ref_v) if self.gather_src is None else self.gather_src
            ss.semshare_gather_kv(src_k, src_v, self.idx.view(1, wl.n_tgt), out_k=self.out_k, out_v=self.out_v,
                                  err_flag=self.flag)
        nvtx_pop()
        if ev:
            ev[4].record()
        self.h_choice.copy_(self.choice, non_blocking=True)  # best, applies

    def unique_rows(self) -> int:
        return int(np.unique(self.idx.cpu().numpy()).size)

    def e2e_kv_bytes(self) -> dict:
        L, H, hd = self.wl.kv
        row = hd * 2 * 2
        return {"inplace": float(self.wl.n_tgt) * L * H * row, "fetch": float(self.unique_rows()) * L * H * row,
                "copy_all": float(self.ref_k[0].numel() * self.ref_k[0].element_size() * 2)}

    def e2e_plan(self, mode: str = "fetch"):
        """(one, h2d, d2h, read): the target's embedding rows and positions copied in; the stored
        prompts' K/V caches stay in pinned host memory and the gather's rows reach it one of three
        ways (`mode`): fetch -- semshare_fetch_rows copies each row the match selects (pool rows of
        the winner, known only on the device) into HBM once; inplace -- the gather reads them across
        the host link, repeats included; copy_all -- the host reads the winner and its whole cache is
        copied in first (Sec. 3.2 loads the retrieved prompt onto the GPU with its KV cache).  The
        winner and the match result (idx, dist) are copied back."""
        import torch

        h_emb = self.emb.cpu().pin_memory()
        h_pos = self.pos.cpu().pin_memory()
        h_k = [t.cpu().pin_memory() for t in self.ref_k]
        h_v = [t.cpu().pin_memory() for t in self.ref_v]
        h_idx = torch.empty_like(self.idx, device="cpu").pin_memory()
        h_dist = torch.empty_like(self.dist, device="cpu").pin_memory()
        kv_bytes = self.e2e_kv_bytes()[mode]
        h2d = h_emb.numel() * h_emb.element_size() + h_pos.numel() * 4 + kv_bytes
        d2h = (h_idx.numel() + h_dist.numel()) * 4 + self.h_choice.numel() * 4
        ss = self.ss
        fetch_ws = torch.empty(max(16, ss.semshare_fetch_workspace_size(self.wl.n_ref)), dtype=torch.uint8,
                               device=self.dev)
        h_best = torch.zeros(1, dtype=torch.int32).pin_memory()

        L = self.wl.n_layers
        groups = [(g * L // self.fetch_groups, (g + 1) * L // self.fetch_groups) for g in range(self.fetch_groups)]
        side = torch.cuda.Stream(self.dev)
        idx2 = self.idx.view(1, self.wl.n_tgt)

        def load():
            # the copy engines need the winner's address: the host waits for the retrieval
            h_best.copy_(self.ret.best)
            m = int(h_best[0])
            self.ref_k[m].copy_(h_k[m], non_blocking=True)
            self.ref_v[m].copy_(h_v[m], non_blocking=True)

        def fetch_gather():
            # pool rows of whichever candidate won, found on the device; group g's gather (second
            # stream) overlaps group g+1's copy across the host link
            main = torch.cuda.current_stream(self.dev)
            for l0, l1 in groups:
                ss.semshare_fetch_rows([t[l0:l1] for t in h_k], [t[l0:l1] for t in h_v], self.idx,
                                       dev_k=[t[l0:l1] for t in self.ref_k], dev_v=[t[l0:l1] for t in self.ref_v],
                                       workspace=fetch_ws, err_flag=self.flag)
                side.wait_stream(main)
                with torch.cuda.stream(side):
                    ss.semshare_gather_kv([t[l0:l1] for t in self.ref_k], [t[l0:l1] for t in self.ref_v], idx2,
                                          out_k=self.out_k[:, l0:l1], out_v=self.out_v[:, l0:l1], err_flag=self.flag)
            main.wait_stream(side)

        def one():
            self.emb.copy_(h_emb, non_blocking=True)
            self.pos.copy_(h_pos, non_blocking=True)
            if mode == "inplace":
                self.gather_src = (h_k, h_v)
            elif mode == "copy_all":
                self.load_winner = load
            else:
                self.fetch_gather = fetch_gather
            try:
                self.step()
            finally:
                self.load_winner = None
                self.gather_src = None
                self.fetch_gather = None
            h_idx.copy_(self.idx, non_blocking=True)
            h_dist.copy_(self.dist, non_blocking=True)

        return one, h2d, d2h, lambda: int(h_idx[0])


def make_problem(wl, device, seed, matcher, with_hd=False, with_retain=False):
    if wl.recipe == "retrieve":
        if with_hd or with_retain:
            raise ValueError("--hd and --retain apply to the matching workloads")
        return RetrieveProblem(wl, device, seed, matcher)
    return Problem(wl, device, seed, matcher, with_hd=with_hd, with_retain=with_retain)


def stage_report(wl, W, stage_ms, peaks, popc_peak, matcher):
    """Per-stage throughput and fraction of the relevant peak."""
    kpad = ((wl.nbits + 127) // 128) * 128
    fp8_peak = 2.0 * peaks["bf16_tflops"]  # fp8 dense = 2 x bf16 (nominal ratio)
    out = {}
    for name, ms in stage_ms.items():
        sec = ms * 1e-3
        r = {"ms": ms}
        if name in ("hash", "hash_plain"):
            r["tflops"] = W["hash_flops"] / sec / 1e12
            r["gbs"] = W["hash_bytes"] / sec / 1e9
            r["frac_tensor"] = r["tflops"] / peaks["bf16_tflops"]
            r["frac_hbm"] = r["gbs"] / peaks["hbm_gbs"]
        elif name == "retrieve":
            r["tflops_fp8"] = W["retrieve_flops"] / sec / 1e12
            r["frac_fp8_tensor"] = r["tflops_fp8"] / fp8_peak
        elif name == "match":
            r["gwordops"] = W["match_wordops"] / sec / 1e9
            r["matcher"] = matcher
            if matcher == "popc":
                r["frac_popc"] = r["gwordops"] * 1e9 / popc_peak
            else:
                fl = W.get("match_flops", 2.0 * W["targets"] * wl.n_ref * kpad)
                r["tflops_fp8"] = fl / sec / 1e12
                r["frac_fp8_tensor"] = r["tflops_fp8"] / fp8_peak
        elif name == "gather":
            r["gbs"] = W["gather_bytes"] / sec / 1e9
            r["frac_hbm"] = r["gbs"] / peaks["hbm_gbs"]
        elif name in ("deviation", "select"):
            r["gbs"] = W[name + "_bytes"] / sec / 1e9
            r["frac_hbm"] = r["gbs"] / peaks["hbm_gbs"]
        out[name] = r
    return out


def roofline_for(dominant, stages, peaks, matcher, workload):
    if dominant == "gather":
        return {"kernel": "kv_gather_kernel", "bound": "hbm", "achieved": stages["gather"]["gbs"],
                "peak": peaks["hbm_gbs"], "unit": "GB/s"}, NCU_TRAFFIC.get(("gather", workload))
    if dominant in ("hash", "hash_plain"):
        # bf16 rows with the interleaved pairing (or none) run on SM pairs; fp32 rows and rotate-half
        # on the one-SM kernel
        return {"kernel": "lsh_hash_2sm_kernel / lsh_hash_kernel", "bound": "tensor", "achieved": stages[dominant]["tflops"],
                "peak": peaks["bf16_tflops"], "unit": "TFLOP/s"}, NCU_TRAFFIC.get(("hash", workload))
    if dominant == "retrieve":
        return {"kernel": "hamming_tc_kernel<256> (segmented)", "bound": "tensor",
                "achieved": stages["retrieve"]["tflops_fp8"], "peak": 2.0 * peaks["bf16_tflops"],
                "unit": "TFLOP/s"}, NCU_TRAFFIC.get(("retrieve", workload))
    if matcher == "popc":
        return {"kernel": "hamming_nn_kernel", "bound": "alu", "achieved": stages["match"]["gwordops"],
                "peak": stages["match"]["gwordops"] / stages["match"]["frac_popc"], "unit": "Gwordop/s"}, \
            NCU_TRAFFIC.get(("match", workload))
    return {"kernel": "hamming_tc_kernel", "bound": "tensor", "achieved": stages["match"]["tflops_fp8"],
            "peak": 2.0 * peaks["bf16_tflops"], "unit": "TFLOP/s"}, NCU_TRAFFIC.get(("match_tc", workload))


def run_gpu_arm(args, rank, world, local_rank):
    import torch

    import paper_2509_24832_gb300 as ss

    ss.load()
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    wl = ALL_WORKLOADS[args.workload]
    seed = wl.base_seed + 7919 * rank
    prob = make_problem(wl, device, seed, args.matcher, with_hd=args.hd, with_retain=args.retain)
    if args.rope != "interleaved":
        if not isinstance(prob, Problem):
            raise ValueError("--rope applies to the matching workloads")
        prob.rope_layout = args.rope
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)
    n_ev = len(prob.STAGES) + 1

    for _ in range(max(args.warmup, 3)):
        prob.step()
    torch.cuda.synchronize()
    ss.check_flag(prob.flag, "warm-up")
    run_step = prob.step
    if args.graph:
        # every library call only enqueues kernels on the current stream: the step records into one
        # graph (programmatic-dependency edges between the kernels)
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream(device)
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            prob.step()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        with torch.cuda.graph(graph, capture_error_mode="thread_local"):
            prob.step()
        for _ in range(3):
            graph.replay()
        torch.cuda.synchronize()
        ss.check_flag(prob.flag, "graph warm-up")
        run_step = graph.replay

    K = args.steps
    # timed steps: one event pair per step (events between kernels would keep a kernel from being
    # scheduled while the previous one drains); the per-stage split comes from a second pass below
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
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
            evs[k][0].record()
            run_step()
            evs[k][1].record()
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall0
    barrier(device)
    ss.check_flag(prob.flag, "timed steps")
    ms_local = float(evs_total(evs))
    ms_median = reduce_max(float(np.median([e[0].elapsed_time(e[-1]) for e in evs])), device)

    # per-stage split: a second pass with events between the stages
    Ks = min(K, 200)
    sevs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ev)] for _ in range(Ks)]
    torch.cuda.synchronize()
    for k in range(Ks):
        flush.zero_()
        prob.step(sevs[k])
    torch.cuda.synchronize()
    ss.check_flag(prob.flag, "stage pass")
    st = np.array([[sevs[k][i].elapsed_time(sevs[k][i + 1]) for i in range(n_ev - 1)] for k in range(Ks)])
    ms_step = reduce_max(ms_local, device)
    stage_ms = {n: reduce_max(float(st[:, i].mean()), device) for i, n in enumerate(prob.STAGES)}
    W = work(wl)
    if getattr(prob, "retain", False):
        L, H, hd = wl.kv
        W["gather_bytes"] = 2.0 * 2.0 * float(sum(prob.counts)) * H * hd * 2
    value = world * W["targets"] / (ms_step * 1e-3)

    peaks, peak_src = load_peaks()
    props = torch.cuda.get_device_properties(device)
    clocks = sampler.summary() if not args.no_clocks else None
    sm_mhz = (clocks or {}).get("sm_mhz") or 2070.0
    popc_table = popc_peak_wordops(sm_mhz, props.multi_processor_count)
    popc_peak = measure_hamming_rate(device) if args.matcher == "popc" else popc_table
    stages = stage_report(wl, W, stage_ms, peaks, popc_peak, args.matcher)
    if args.matcher == "popc":
        stages["match"]["popc_peak"] = {"measured_wordops_per_s": popc_peak, "table_wordops_per_s": popc_table,
                                        "source": "semshare_probe_hamming_rate (measured); table: 16 popc/clk/SM "
                                                  "at the sampled SM clock, cross-check"}

    dominant = max(stage_ms, key=stage_ms.get)
    roof, tr = roofline_for(dominant, stages, peaks, args.matcher, wl.name)
    if getattr(prob, "retain", False) and dominant == "gather":
        roof["kernel"] = "kv_gather_kernel (retained rows)"
        tr = NCU_TRAFFIC.get(("gather_retained", wl.name))
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else "fallback"
    roof["traffic"] = tr["bytes_per_launch"] if tr and tr.get("sha") == kernel_sha(tr["file"]) else None
    if roof["traffic"] and roof["unit"] == "GB/s":
        # the DRAM bytes ncu counts per launch over the same duration: repeats served by L2 are in
        # "achieved" (algorithmic bytes) but not here
        roof["frac_dram"] = roof["traffic"] / (stage_ms[dominant] * 1e-3) / 1e9 / roof["peak"]

    # e2e: the reference K/V cache lives in pinned host memory and its rows reach the gather one of
    # three ways (Problem.e2e_plan).  A cost model of the step's K/V movement -- host-link bytes at
    # the measured link rate plus HBM bytes at the measured copy rate (fetch and copy_all write the rows to
    # HBM and the gather then reads and writes them again; inplace only writes the gathered rows; a
    # fetch in layer groups overlaps the two) -- predicts the best mode; all three are measured.
    link = measure_link_peak(device)
    kv_bytes = prob.e2e_kv_bytes()
    model_mode = e2e_mode(kv_bytes, peaks["hbm_gbs"], getattr(prob, "fetch_groups", 1), link["gbs"])
    # every e2e mode must give the rearranged cache of the device-resident step, bit for bit
    want = (prob.out_k.clone(), prob.out_v.clone(), prob.idx.clone())
    runs = {m: run_e2e(args, prob, device, m, want, link["gbs"]) for m in E2E_KV}
    resident = run_e2e(args, prob, device, "kv_resident", want, link["gbs"]) if isinstance(prob, Problem) else None
    # all three are complete paths through the public API; the headline is the mode the cost model
    # picks before anything is measured (the fastest measured is recorded beside it)
    fastest = min(runs, key=lambda m: runs[m]["ms_per_step"])
    e2e = dict(runs[model_mode], chosen_by="cost model (link bytes at the measured link rate, HBM bytes at the "
                                          "measured copy rate)", fastest_measured=fastest, link=link)
    e2e_alt = {m: r for m, r in runs.items() if m != model_mode}
    if resident is not None:
        # the GB300 layout: stored caches resident in HBM (a 5k-token cache is 671 MB of 288 GB), so
        # a request moves only its embedding rows in and its match result out
        e2e_alt["kv_resident"] = resident
    if isinstance(prob, Problem) and args.rope == "interleaved":
        # reading M: the reference's codes computed when it was stored; only the target's rows cross
        e2e_alt["ref_codes_cached"] = run_e2e(args, prob, device, model_mode, want, link["gbs"], ref_cached=True)
    del want
    ref_cached = run_ref_codes_cached(args, prob, device, flush) if isinstance(prob, Problem) else None
    parity = parity_diagnostics(prob) if isinstance(prob, Problem) and rank == 0 else None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, prob)

    config = {"workload": wl.name, "n_ref": wl.n_ref, "n_tgt": wl.n_tgt, "n_batch": wl.n_batch,
              "n_seg": wl.n_seg, "d": wl.d, "nbits": wl.nbits, "kv": list(wl.kv),
              "parallelism": f"replicas x{world}", "l2": "flushed before every step (512 MB write)",
              "matcher": args.matcher, "launch": "CUDA graph replay" if args.graph else "eager library calls"}
    if args.rope != "interleaved":
        config["rope"] = "pairs (k, k + d/2)"
    if args.retain:
        config["retain"] = (f"per-layer retained tokens, first {prob.counts[0]}, last {prob.counts[-1]}, "
                            f"{sum(prob.counts)} rows of {wl.n_layers * wl.n_tgt} (0.8, then 0.98 per layer)")
    if args.hd:
        config["hd"] = (f"first-layer KV deviation against a synthetic recomputed first layer, "
                        f"top {workloads_hd_percent()}% tokens per prompt")
    if isinstance(prob, RetrieveProblem):
        config["retrieved"] = prob.winner
        config["stored_codes"] = "computed when the prompts were stored (outside the timed region)"
    line = {
        "metric": METRIC_RETRIEVE if isinstance(prob, RetrieveProblem) else METRIC, "value": value,
        "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if wl.emb_dtype == "bf16" else "f32",
        "data": "synthetic (seeded; see workloads.py)",
        "config": config,
        "e2e_alt": e2e_alt,
        "ms_per_step_median": ms_median,
        "stages_ms_sum": float(sum(stage_ms.values())),
        "roofline": roof, "stages": stages, "e2e": e2e, "cpu_baseline": cpu, "ref_codes_cached": ref_cached,
        "parity": parity,
        "gpu_launches": prob.LAUNCHES_PER_STEP * K, "clocks": clocks, "wall_s_timed": reduce_max(t_wall, device),
        "impl": "gb300",
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


PARITY_SAMPLE_ROWS = 128  # reference and target rows the oracle re-hashes for the bench's parity record


def parity_diagnostics(prob) -> dict:
    """Parity record of the timed workload (outside the timed region): the oracle re-hashes a seeded
    sample of the step's rows and the GPU's codes are compared bit by bit (mismatches outside the
    band must be 0; band bits are the ones the tolerance exempts), against codes of the unrounded
    fp64 projection too (how often the bf16 operand contract changes a sign: a diagnostic); and the
    recall of the generator's ground-truth source rows by the match (targets built from a reference
    row whose nearest reference row, by code distance, is that row)."""
    import oracle

    oracle.build()
    wl = prob.wl
    g = np.random.default_rng(wl.base_seed + 17)
    rows_all = prob.host_emb.shape[0]
    half = PARITY_SAMPLE_ROWS // 2
    rows = np.sort(np.concatenate([g.choice(wl.n_ref, min(half, wl.n_ref), replace=False),
                                   wl.n_ref + g.choice(rows_all - wl.n_ref, min(half, rows_all - wl.n_ref),
                                                       replace=False)]))
    emb = prob.host_emb[rows]
    pos = prob.host_pos[rows]
    R = prob.hyp.cpu().view(__import__("torch").int16).numpy().view(np.uint16)
    layout = "half" if prob.rope_layout == "half" else "interleaved"
    oc, op = oracle.hash_codes(emb, pos, R, layout=layout)
    uc, _ = oracle.hash_codes(emb, pos, R, layout=layout, round_operand=False)
    gc = prob.codes.cpu().numpy().view(np.uint32)[rows]

    def bits(c):
        return np.unpackbits(np.ascontiguousarray(c).view(np.uint8), axis=1, bitorder="little").astype(bool)

    band = np.abs(op) < 1e-3 * np.abs(op).max(axis=1, keepdims=True)
    gb, ob, ub = bits(gc), bits(oc), bits(uc)
    out = {"rows_sampled": int(len(rows)), "bits_sampled": int(gb.size),
           "band_bits": int(band.sum()),
           "mismatches_outside_band": int(((gb != ob) & ~band).sum()),
           "mismatches_inside_band": int(((gb != ob) & band).sum()),
           "agreement_with_unrounded_fp64": float((gb == ub).mean()),
           "oracle": "oracle.hash_codes (fp64, bf16 operand contract) on the sampled rows"}
    idx = prob.idx.cpu().numpy().reshape(wl.n_batch, wl.n_tgt)
    src = np.asarray(prob.src).reshape(wl.n_batch, wl.n_tgt)
    reused = src >= 0
    out["recall_of_source_rows"] = float((idx[reused] == src[reused]).mean()) if reused.any() else None
    out["reused_targets"] = int(reused.sum())
    return out


def run_ref_codes_cached(args, prob, device, flush):
    """The step with the reference prompt's codes computed once beforehand (they depend only on
    the reference and its own positions), so each step hashes only the target rows; reported
    beside the main number, which hashes both (§3.2 applies RoPE to both prompts per request)."""
    import torch

    wl, ss = prob.wl, prob.ss
    if wl.n_ref == 0 or args.rope != "interleaved":
        return None
    tgt_emb, tgt_pos = prob.emb[wl.n_ref:], prob.pos[wl.n_ref:]
    tgt_codes = prob.codes[wl.n_ref:]
    ws = torch.zeros(max(256, ss.semshare_hash_workspace_size(tgt_emb.shape[0], wl.d, wl.nbits)),
                     dtype=torch.uint8, device=device)
    prob.hash()  # the reference codes, once

    tgt_signs = None if prob.signs is None else prob.signs[wl.n_ref:]

    def step():
        prob.hash_rows(tgt_emb, tgt_pos, tgt_codes, tgt_signs, ws)
        prob.match()
        prob.gather()
        if prob.hd:
            prob.deviation()
            prob.select()

    for _ in range(3):
        step()
    n = min(args.steps, 200)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    torch.cuda.synchronize()
    for a, b in evs:
        flush.zero_()
        a.record()
        step()
        b.record()
    torch.cuda.synchronize()
    ss.check_flag(prob.flag, "reference codes cached")
    ms = reduce_max(float(np.mean([a.elapsed_time(b) for a, b in evs])), device)
    _, world, _ = dist_info()
    return {"value": world * wl.n_batch * wl.n_tgt / (ms * 1e-3), "unit": "tokens/s", "ms_per_step": ms,
            "steps": n, "note": "reference codes hashed once before timing; each step hashes the target rows only"}


def workloads_hd_percent():
    import paper_2509_24832_gb300 as ss

    return ss.HD_PERCENT


def evs_total(evs):
    """Mean device time of a step: first to last event of each step."""
    return float(np.mean([e[0].elapsed_time(e[-1]) for e in evs]))


class _Null:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False


E2E_LAYER_GROUPS = 4  # fetch mode: layer groups whose fetch and gather overlap

def measure_link_peak(device, nbytes: int = 1 << 30, reps: int = 5) -> dict:
    """Host -> HBM rate of the link the e2e path uses: one cudaMemcpyAsync of a 1 GiB pinned buffer,
    best of `reps`, CUDA events on the current stream; plus where the pinned pages can live (the
    NUMA nodes of this host and the one the GPU is attached to)."""
    import glob

    import torch

    h = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    d = torch.empty(nbytes, dtype=torch.uint8, device=device)
    d.copy_(h, non_blocking=True)
    torch.cuda.synchronize()
    best = float("inf")
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        d.copy_(h, non_blocking=True)
        b.record()
        b.synchronize()
        best = min(best, a.elapsed_time(b))
    del h, d
    nodes = sorted(glob.glob("/sys/devices/system/node/node[0-9]*"))
    gpu_node = None
    try:
        props = torch.cuda.get_device_properties(device)
        bus = f"{props.pci_domain_id:04x}:{props.pci_bus_id:02x}:{props.pci_device_id:02x}.0"
        with open(f"/sys/bus/pci/devices/{bus}/numa_node") as f:
            gpu_node = int(f.read().strip())
    except Exception:
        gpu_node = None
    return {"gbs": nbytes / (best * 1e-3) / 1e9, "bytes": nbytes, "method": "cudaMemcpyAsync of a pinned "
            "buffer, best of %d, CUDA events" % reps, "numa_nodes": len(nodes), "gpu_numa_node": gpu_node,
            "placement": "pinned with the default policy" + (" (one NUMA node: the GPU's own)" if len(nodes) == 1
                                                               else "")}


def e2e_mode(kv_bytes: dict, hbm_gbs: float, fetch_groups: int = 1, link_gbs: float = 211.0) -> str:
    """The e2e mode with the least estimated K/V movement time; ties go to the bulk copy.  With
    fetch_groups > 1 the fetch runs in that many layer groups whose HBM gathers overlap the next
    group's host-link copy: max of the two times plus one group's share of the smaller."""
    gathered = kv_bytes["inplace"]
    hbm = {"inplace": gathered, "fetch": kv_bytes["fetch"] + 2 * gathered,
           "copy_all": kv_bytes["copy_all"] + 2 * gathered}
    order = ("copy_all", "fetch", "inplace")
    link_s = {m: kv_bytes[m] / (link_gbs * 1e9) for m in order}
    hbm_s = {m: hbm[m] / (hbm_gbs * 1e9) for m in order}
    cost = {m: link_s[m] + hbm_s[m] for m in order}
    if fetch_groups > 1:
        a, b = link_s["fetch"], hbm_s["fetch"]
        cost["fetch"] = max(a, b) + min(a, b) / fetch_groups
    return min(order, key=lambda m: (round(cost[m], 7), order.index(m)))


E2E_KV = {
    "fetch": "reference cache in pinned host memory; semshare_fetch_rows copies each selected row into HBM "
             "once, then the gather runs on HBM (in 4 layer groups, each group's gather on a second stream "
             "overlapping the next group's copy; one group with retention)",
    "inplace": "reference cache in pinned host memory; the gather reads the selected rows in place "
               "(h2d counts every selected row; repeats may be served by L2)",
    "copy_all": "reference cache copied to HBM every step, then gathered",
}
E2E_KV_RESIDENT = {
    "kv_resident": "reference cache resident in HBM (stored there, not per request); only the embedding rows "
                   "cross the host link",
}


def run_e2e(args, prob, device, mode: str = "fetch", want=None, link_gbs=None, ref_cached: bool = False):
    """Same metric through the public API with host buffers (the problem's e2e_plan says which
    inputs are copied in and which results are read back every step)."""
    import torch

    wl = prob.wl
    one, h2d, d2h, read = prob.e2e_plan(mode, ref_cached=True) if ref_cached else prob.e2e_plan(mode)
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
        _ = read()  # the host reads the result
        times.append(a.elapsed_time(b))
    if want is not None:
        got = (prob.out_k, prob.out_v, prob.idx)
        if not all(torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a,
                               b.view(torch.int16) if b.dtype == torch.bfloat16 else b) for a, b in zip(got, want)):
            raise RuntimeError(f"e2e mode {mode}: the result differs from the device-resident step")
    ms = reduce_max(float(np.mean(times)), device)
    _, world, _ = dist_info()
    out = {"value": world * wl.n_batch * wl.n_tgt / (ms * 1e-3), "unit": "tokens/s", "ms_per_step": ms,
           "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "mode": mode,
           "kv": {**E2E_KV, **E2E_KV_RESIDENT}[mode]}
    if link_gbs:
        ach = h2d / (ms * 1e-3) / 1e9
        out["roofline"] = {"bound": "host_link", "achieved": ach, "peak": link_gbs, "unit": "GB/s",
                           "frac": ach / link_gbs, "peak_source": "measured in this run (1 GiB pinned H2D copy)"}
    return out


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


def _oracle_retrieve_setup(oracle, wl, emb, pos, R):
    """Store time for the oracle: every stored prompt's plain and rotary codes."""
    n_pool = wl.n_ref
    rcodes, _ = oracle.hash_codes(emb[:n_pool], np.zeros(n_pool, dtype=np.int32), R)
    codes, _ = oracle.hash_codes(emb[:n_pool], pos[:n_pool], R)
    return {"rcodes": rcodes, "codes": codes, "offsets": [m * wl.seg_len for m in range(wl.n_seg + 1)]}


def _oracle_retrieve_sample(oracle, wl, emb, pos, R, ctx, kv_of, tsel):
    """The oracle's retrieval step for the target tokens `tsel`: their plain codes, the
    similarity to every stored prompt and the winner, their rotary codes, the match against the
    winner's codes, the gather of the winner's K/V rows.  Returns (seconds, winner)."""
    rows = wl.n_ref + tsel
    t0 = time.perf_counter()
    tr, _ = oracle.hash_codes(emb[rows], np.zeros(len(tsel), dtype=np.int32), R)
    _, _, best, _ = oracle.retrieve(tr, ctx["rcodes"], ctx["offsets"], wl.nbits)
    tc, _ = oracle.hash_codes(emb[rows], pos[rows], R)
    o = ctx["offsets"]
    idx, _ = oracle.match(tc, ctx["codes"][o[best]:o[best + 1]])
    k, v = kv_of(best)
    oracle.gather_kv(k, v, idx)
    return time.perf_counter() - t0, best


def _kv_from_device(prob):
    import torch

    cache = {}

    def kv_of(m):
        if m not in cache:
            cache.clear()
            cache[m] = (prob.ref_k[m].cpu().view(torch.int16).numpy().view(np.uint16),
                        prob.ref_v[m].cpu().view(torch.int16).numpy().view(np.uint16))
        return cache[m]

    return kv_of


def _kv_from_host(wl):
    cache = {}

    def kv_of(m):
        if m not in cache:
            cache.clear()
            cache[m] = workloads.kv_cache(wl, segment=m)
        return cache[m]

    return kv_of


CPU_BASELINE_SECONDS = 10.0


def cpu_baseline(wl, prob):
    """The oracle as it stands on the host cores: one bounded sample of the workload."""
    import oracle

    oracle.build()
    if wl.recipe == "retrieve":
        emb, pos = prob.host_emb, prob.host_pos
        R = prob.hyp.cpu().view(__import__("torch").int16).numpy().view(np.uint16)
        ctx = _oracle_retrieve_setup(oracle, wl, emb, pos, R)
        n_s = wl.n_tgt
        kv_of = _kv_from_device(prob)
        reps, secs = 0, 0.0
        while reps == 0 or secs < CPU_BASELINE_SECONDS:
            dt, best = _oracle_retrieve_sample(oracle, wl, emb, pos, R, ctx, kv_of, np.arange(n_s))
            secs += dt
            reps += 1
        return {"value": reps * n_s / secs, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
                "sample": f"all {n_s} target tokens: plain codes, similarity to the {wl.n_seg} stored prompts "
                          f"({wl.n_ref} stored codes, computed beforehand as on the GPU), rotary codes, match "
                          f"against the winner ({best}), gather of its {wl.n_layers}x{wl.n_heads} K/V rows, "
                          f"{reps} times; seconds={secs:.2f}"}
    emb, pos = prob.host_emb, prob.host_pos
    R = prob.hyp.cpu().view(__import__("torch").int16).numpy().view(np.uint16)
    ref_codes, k_np, v_np = _oracle_inputs(oracle, wl, emb, pos, R, prob.ref_k, prob.ref_v)
    n_s = min(wl.n_tgt, 5120)
    tsel = np.arange(n_s)
    # repeat the sample until about CPU_BASELINE_SECONDS of oracle work have run (at least once)
    reps, secs = 0, 0.0
    while reps == 0 or secs < CPU_BASELINE_SECONDS:
        secs += _oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np, tsel)
        reps += 1
    out = {"value": reps * n_s / secs, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
           "sample": f"{n_s} target tokens of prompt 0 (hash of them + {n_s * wl.n_ref // (wl.n_batch * wl.n_tgt)} "
                     f"reference rows, match against all {wl.n_ref} reference codes, gather of their "
                     f"{wl.n_layers}x{wl.n_heads} K/V rows), {reps} times; seconds={secs:.2f}"}
    out["single_thread"] = cpu_baseline_single_thread(oracle, wl, emb, pos, R, ref_codes, k_np, v_np)
    return out


CPU_SINGLE_THREAD_SECONDS = 4.0


def cpu_baseline_single_thread(oracle, wl, emb, pos, R, ref_codes, k_np, v_np) -> dict:
    """The same oracle sample on one host thread (a smaller slice of target tokens, repeated for
    about CPU_SINGLE_THREAD_SECONDS)."""
    n_s = min(wl.n_tgt, 256)
    tsel = np.arange(n_s)
    prev = oracle.set_threads(1)
    try:
        reps, secs = 0, 0.0
        while reps == 0 or secs < CPU_SINGLE_THREAD_SECONDS:
            secs += _oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np, tsel)
            reps += 1
    finally:
        oracle.set_threads(prev)
    return {"value": reps * n_s / secs, "unit": "tokens/s", "cores": 1,
            "sample": f"{n_s} target tokens of prompt 0 with their share of reference rows, {reps} times; "
                      f"seconds={secs:.2f}"}


REFERENCE_ARM_SECONDS = 120.0


def run_reference_arm(args, rank, world):
    if rank != 0:
        return
    import oracle

    oracle.build()
    wl = ALL_WORKLOADS[args.workload]
    emb, pos, _ = workloads.prompt_rows(wl, batches=[0])
    R = workloads.hyperplanes(wl)
    g = np.random.default_rng(wl.base_seed)
    if wl.recipe == "retrieve":
        ctx = _oracle_retrieve_setup(oracle, wl, emb, pos, R)
        kv_of = _kv_from_host(wl)

        def sample_step(tsel):
            return _oracle_retrieve_sample(oracle, wl, emb, pos, R, ctx, kv_of, tsel)[0]

        what = (f"plain codes, similarity to the {wl.n_seg} stored prompts ({wl.n_ref} stored codes computed "
                f"beforehand), rotary codes, match against the winner, gather of its K/V rows")
    else:
        ref_codes, k_np, v_np = _oracle_inputs(oracle, wl, emb, pos, R)

        def sample_step(tsel):
            return _oracle_sample(oracle, wl, emb, pos, R, ref_codes, k_np, v_np, tsel)

        what = (f"hash of them plus their share of reference rows, match against all {wl.n_ref} reference "
                f"codes, gather of their {wl.n_layers}x{wl.n_heads} K/V rows")
    # A step is the same kind of slice the GPU arm's cpu_baseline leg times: as many target tokens
    # as the run's K + W steps can afford in about REFERENCE_ARM_SECONDS (all of the prompt's, at
    # the driver's step counts), at least 1024 so that every host core has rows to work on.
    t_tok = sample_step(np.arange(min(wl.n_tgt, 1024))) / min(wl.n_tgt, 1024)  # calibration
    n_steps = args.steps + max(args.warmup, 3)
    per_step = int(min(wl.n_tgt, max(1024, REFERENCE_ARM_SECONDS / n_steps / max(t_tok, 1e-9))))
    per_step = min(wl.n_tgt, 1 << int(np.floor(np.log2(per_step)))) if per_step < wl.n_tgt else per_step
    sample = f"per step {per_step} of the prompt's {wl.n_tgt} target tokens (a seeded random choice): {what}"
    for _ in range(max(args.warmup, 3)):
        sample_step(np.sort(g.choice(wl.n_tgt, per_step, False)))
    secs = []
    for _ in range(args.steps):
        secs.append(sample_step(np.sort(g.choice(wl.n_tgt, per_step, False))))
    ms = 1e3 * float(np.mean(secs))
    value = per_step / (ms * 1e-3)
    line = {
        "impl": "reference", "metric": METRIC_RETRIEVE if wl.recipe == "retrieve" else METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
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
    NVTX[0] = args.nvtx
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
