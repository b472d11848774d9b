"""bench.py's host-side arithmetic on CPU: the algorithmic work per step that every roofline
fraction divides by (the per-unit figures of the scope table: 2*rows*d*nbits flops for the
projection, N_t*N_r*(nbits/32) word-ops for the search, 2*2*N_t*L*H*hd*2 bytes for the gather),
the e2e cost model's choice of how the reference cache reaches the gather, and the DRAM traffic
table's rule that a recorded count only stands for the kernel source it was taken on."""
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402


@pytest.mark.parametrize("name,flops,wordops,gbytes", [
    # 10,240 rows of 4096 -> 256 bits; 5120 x 5120 x 8 words; 5120 targets x 32 x 8 x 128 bf16
    ("llama8b-5k", 21_474_836_480, 209_715_200, 1_342_177_280),
    # 64 x 2048 + 4096 = 135,168 rows; 131,072 x 4096 x 8 words; 131,072 targets
    ("batched-64x2048", 283_467_841_536, 4_294_967_296, 34_359_738_368),
    # 16 x 4096 + 4096 = 69,632 rows; 4096 x 65,536 x 8 words; 4096 targets
    ("pool-16x4096", 146_028_888_064, 2_147_483_648, 1_073_741_824),
    # 1024 + 1024 rows, 128 bits; 1024 x 1024 x 4 words
    ("llama8b-1k", 2.0 * 2048 * 4096 * 128, 1024 * 1024 * 4, 2 * 2 * 1024 * 32 * 8 * 128 * 2),
])
def test_algorithmic_work_per_step(name, flops, wordops, gbytes):
    w = bench.work(bench.ALL_WORKLOADS[name])
    assert w["hash_flops"] == pytest.approx(flops, rel=0, abs=0.5)
    assert w["match_wordops"] == pytest.approx(wordops, rel=0, abs=0.5)
    assert w["gather_bytes"] == pytest.approx(gbytes, rel=0, abs=0.5)


def test_roofline_fraction_is_achieved_over_peak():
    wl = bench.ALL_WORKLOADS["llama8b-5k"]
    w = bench.work(wl)
    peaks = {"hbm_gbs": 1000.0, "bf16_tflops": 100.0}
    st = bench.stage_report(wl, w, {"hash": 1.0, "gather": 2.0}, peaks, 1.0, "tc")
    assert st["gather"]["gbs"] == pytest.approx(w["gather_bytes"] / 2e-3 / 1e9)
    assert st["gather"]["frac_hbm"] == pytest.approx(st["gather"]["gbs"] / 1000.0)
    assert st["hash"]["tflops"] == pytest.approx(w["hash_flops"] / 1e-3 / 1e12)
    assert st["hash"]["frac_tensor"] == pytest.approx(st["hash"]["tflops"] / 100.0)


HBM = 6686.8


def test_e2e_model_prefers_the_fetch_when_rows_repeat():
    # the 5k step: 3569 distinct selected rows (468 MB) against 671 MB gathered and a 671 MB cache
    kv = {"inplace": 671e6, "fetch": 468e6, "copy_all": 671e6}
    assert bench.e2e_mode(kv, HBM, fetch_groups=4) == "fetch"
    assert bench.e2e_mode(kv, HBM, fetch_groups=1) == "fetch"


def test_e2e_model_with_every_row_distinct():
    # each selected row once (pool, retrieval): in sequence the in-place read moves the fewest
    # bytes through HBM; overlapped in layer groups the fetch's HBM time mostly hides
    x = 537e6
    kv = {"inplace": x, "fetch": x, "copy_all": 16 * x}
    assert bench.e2e_mode(kv, HBM, fetch_groups=1) == "inplace"
    assert bench.e2e_mode(kv, HBM, fetch_groups=4) == "fetch"


def test_e2e_model_with_many_prompts_sharing_one_cache():
    # 64 prompts gather 17.2 GB from one 537 MB cache: reading in place would cross the link 64
    # times; fetch and bulk copy move the cache once, and a tie goes to the bulk copy
    cache, gathered = 537e6, 17.18e9
    kv = {"inplace": gathered, "fetch": cache, "copy_all": cache}
    assert bench.e2e_mode(kv, HBM, fetch_groups=1) == "copy_all"
    assert bench.e2e_mode(kv, HBM, fetch_groups=4) == "fetch"


def test_traffic_entries_name_their_kernel_source():
    for (kernel, workload), tr in bench.NCU_TRAFFIC.items():
        assert workload in bench.ALL_WORKLOADS, workload
        assert os.path.exists(os.path.join(bench.ROOT, "paper_2509_24832_gb300", "csrc", tr["file"]))
        assert len(tr["sha"]) == 16 and tr["bytes_per_launch"] > 0
    # a recorded count stands only while the source hashes to the recorded prefix
    sha = bench.kernel_sha("gather.cu")
    assert len(sha) == 16 and all(c in "0123456789abcdef" for c in sha)
