"""Host-side bookkeeping of bench.py (no GPU): the algorithmic bytes of a decode
step, the DRAM traffic taken from a committed ncu summary only while the
kernel source it was measured on is unchanged, the roofline peak, and the
whole-job throughput."""
import json
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402
from paper_2607_29591_gb300 import workloads as wl  # noqa: E402


def test_algorithmic_bytes_count_rows_and_residual_log_counts():
    n_main = np.array([1000, 900, 1024], np.int32)
    n_res = np.array([24, 100, 0], np.int32)
    want = (1024 + 1000 + 1024) * 512 + (24 + 100) * 4
    assert bench.algorithmic_bytes(n_main, n_res) == want
    # a 32-layer 32K cache at b = 1024: 1 GiB of rows plus the log-counts
    U = 32 * 8 * 8
    nm = np.full(U, 1000, np.int32)
    nr = np.full(U, 24, np.int32)
    assert bench.algorithmic_bytes(nm, nr) == U * 1024 * 512 + U * 24 * 4


def _write_profile(path, bpu, digest):
    with open(path, "w") as f:
        f.write(f"# summary\n\ndram_bytes_per_unit: {bpu}\nkernel_source_sha256_16: {digest}\n")


def test_profiled_traffic_only_for_the_source_it_was_measured_on(tmp_path):
    src = tmp_path / "kernel.cu"
    src.write_text("__global__ void k() {}\n")
    prof = tmp_path / "profile.md"
    digest = bench.kernel_hash([str(src)])
    _write_profile(prof, 541179.5, digest)
    assert bench.profiled_traffic(2048, str(prof), [str(src)]) == int(541179.5 * 2048)
    src.write_text("__global__ void k() { /* changed */ }\n")      # kernel edited since
    assert bench.profiled_traffic(2048, str(prof), [str(src)]) is None
    assert bench.profiled_traffic(2048, str(tmp_path / "missing.md"), [str(src)]) is None


def test_committed_profiles_name_the_kernels_they_summarise():
    """Each committed decode summary carries a per-unit figure and a source
    digest in the form bench.py reads."""
    for prof in (bench.PROFILE, bench.PROFILE_LAYER):
        text = open(prof).read()
        assert "dram_bytes_per_unit:" in text and "kernel_source_sha256_16:" in text
        assert "--clock-control none" in text


def test_peak_comes_from_the_measured_file_or_the_stated_fallback():
    peak, kind = bench.measured_peak_gbs()
    path = os.path.join(bench.ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        assert kind == "measured" and peak == float(json.load(open(path))["hbm_gbs"])
    else:
        assert (peak, kind) == (6800.0, "fallback")


def test_whole_job_throughput_over_the_slowest_rank():
    assert bench.aggregate(per_rank_units=8 * 200, max_seconds=0.032, world=1) == 50000.0
    assert bench.aggregate(per_rank_units=8 * 200, max_seconds=0.032, world=4) == 200000.0


def test_construction_flops_follow_the_stage_formulas():
    w = wl.WORKLOADS["llama8b_32l_32k_b8"]
    f = bench.construction_flops(w)
    d, s, b, G, U = 128, 32768, 1024, 4, 32 * 8 * 8
    assert f["scores"] == 2 * 24 * G * s * d * U
    assert f["validation_targets"] == 4 * 8 * G * s * d * U
    rs = [51, 102, 153, 204]
    assert f["lloyd"] == sum(2 * 4 * (s - b + r) * r * d for r in rs) * U
