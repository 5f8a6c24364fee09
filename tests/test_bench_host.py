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
    got = bench.tc_traffic(wl, n, vals["launch_mode"] == "per-phase", vals["compute"])
    if fresh:
        assert got == pytest.approx(float(vals["dram_bytes_per_launch_scaled"]))
    else:
        assert got is None
    # any other set, count, launch mode or operand mode: no figure
    pp = vals["launch_mode"] == "per-phase"
    assert bench.tc_traffic("resnet18", n, pp, vals["compute"]) is None
    assert bench.tc_traffic(wl, n // 2, pp, vals["compute"]) is None
    assert bench.tc_traffic(wl, n, not pp, vals["compute"]) is None
    assert bench.tc_traffic(wl, n, pp, "bf16_split") is None


def test_traffic_scaling_is_consistent():
    vals = _profile()
    sub = float(vals["dram_bytes_per_launch_subset"])
    scale = float(vals["scale_subset_to_vit_l16"])
    assert float(vals["dram_bytes_per_launch_scaled"]) == pytest.approx(sub * scale, rel=1e-3)


def test_reference_arm_prints_the_contract_line():
    """bench.py --impl reference (the fp64 oracle on the host cores) prints one
    JSON line with the contract's keys, its own cpu_baseline and an e2e object
    with no host<->device bytes."""
    import json
    import subprocess
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "cfg1",
                          "--steps", "1", "--warmup", "3"], capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["steps"] == 1
    assert line["value"] > 0 and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["e2e"]["value"] == line["value"] and line["e2e"]["unit"] == line["unit"]


def test_clock_sampler_summary(tmp_path):
    """The clock record of a bench line: the median SM clock of the loaded
    half of the samples, the throttle reasons seen, and the power draw."""
    sampler = bench.ClockSampler(0)
    sampler.path = str(tmp_path / "clocks.csv")
    with open(sampler.path, "w") as f:
        f.write("0, 1980, 2070, 1385.21, 0x4, Not Active, Not Active, Not Active, Active\n"
                "0, 2070, 2070, 950.00, 0x0, Not Active, Not Active, Not Active, Not Active\n"
                "0, 2010, 2070, [N/A], 0x0, Not Active, Not Active, Not Active, Not Active\n")

    class _Done:
        def terminate(self):
            pass

        def wait(self, timeout=None):
            pass

    sampler.proc = _Done()
    sampler.out = open(os.devnull, "w")
    rec = sampler.stop()
    assert rec["sm_mhz"] == 2040.0 and rec["sm_max_mhz"] == 2070.0 and rec["samples"] == 3
    assert rec["reasons"] == ["sw_power_cap"]
    assert rec["power_w_median"] == pytest.approx((1385.21 + 950.0) / 2) and rec["power_w_max"] == 1385.21


def test_code_hash_ignores_comments_only():
    """The traffic figure is keyed on the kernel's code: comments and
    whitespace do not change it, a changed token does."""
    src = "int f(int x) {  // the /* inner */ comment\n  return x + 1; /* block\n comment */ }\n"
    assert bench.code_only(src) == bench.code_only("int f(int x) {\n return x + 1; }")
    assert bench.code_only(src) != bench.code_only("int f(int x) { return x + 2; }")
