"""Host-side logic of bench.py: the DRAM traffic it reports for the GEMM kernel
comes from the committed ncu summary only for the kernel source, weight set,
matrix count and launch mode that summary was captured on."""

import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _profile():
    vals = {}
    with open(bench.PROFILE_FILE) as f:
        for line in f:
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                vals[k.strip()] = v.strip()
    return vals


def test_traffic_only_for_the_captured_case():
    vals = _profile()
    fresh = vals["source_sha256"] == bench.tc_source_hash()
    wl, n = vals["workload"], int(vals["matrices"])
    got = bench.tc_traffic(wl, n, vals["launch_mode"] == "per-phase")
    if fresh:
        assert got == pytest.approx(float(vals["dram_bytes_per_launch_scaled"]))
    else:
        assert got is None
    # any other set, count or launch mode: no figure
    assert bench.tc_traffic("resnet18", n, True) is None
    assert bench.tc_traffic(wl, n // 2, True) is None
    assert bench.tc_traffic(wl, n, vals["launch_mode"] != "per-phase") is None


def test_traffic_scaling_is_consistent():
    vals = _profile()
    sub = float(vals["dram_bytes_per_launch_subset"])
    scale = float(vals["scale_subset_to_vit_l16"])
    assert float(vals["dram_bytes_per_launch_scaled"]) == pytest.approx(sub * scale, rel=1e-3)
