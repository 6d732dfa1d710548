"""bench.py reports the GEMM family's DRAM traffic only for the kernel source
the ncu counters were taken on: any other k_gemm.cu yields no traffic figure
(null in the roofline object) instead of a stale one."""
import os
import shutil
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_traffic_follows_the_profiled_source(tmp_path):
    src = os.path.join(ROOT, "paper_2511_22533_gb300", "csrc", "k_gemm.cu")
    copy = tmp_path / "k_gemm.cu"
    shutil.copyfile(src, copy)
    live = bench.gemm_traffic(str(copy))
    # the recorded figure belongs to exactly one source text
    if live is not None:
        assert live["dram_bytes_per_launch"] > 0
        assert live["profile"].startswith("profiles/") and os.path.exists(os.path.join(ROOT, live["profile"]))
    with open(copy, "ab") as f:
        f.write(b"\n// any change\n")
    assert bench.gemm_traffic(str(copy)) is None
    assert bench.gemm_traffic(str(tmp_path / "missing.cu")) is None


def test_recorded_traffic_is_within_the_operand_bytes():
    # the capture showed no operand re-read: DRAM bytes per launch within a
    # few percent of the algorithmic operand bytes
    t = bench.GEMM_TRAFFIC
    assert 1.0 <= t["dram_bytes_per_launch"] / t["algorithmic_bytes_per_launch"] < 1.05
