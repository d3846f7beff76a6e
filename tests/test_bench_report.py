"""Host logic of the benchmark report: the source digest that decides whether
the committed ncu traffic figures still describe the kernels, and the
per-kernel roofline bookkeeping.  CPU only."""
import importlib.util
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    argv, sys.argv = sys.argv, ["bench.py"]
    try:
        spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
        mod = importlib.util.module_from_spec(spec)
        spec.loader.exec_module(mod)
    finally:
        sys.argv = argv
    return mod


def test_code_only_drops_comments_and_layout(bench):
    a = 'int f(int x) {  // one\n  return x + 1; /* two\n lines */ }\n'
    b = 'int f(int x)\n{\n  return x + 1;\n}'
    assert bench._code_only(a) == bench._code_only(b)
    # a code change is seen
    assert bench._code_only(a) != bench._code_only(a.replace("+ 1", "+ 2"))
    # comment markers inside string and character literals are code
    s = 'asm("mov.u32 %0, 1; // not a comment");'
    assert bench._code_only(s) == s
    assert bench._code_only("char c = '/'; // x") == "char c = '/';"


def test_committed_traffic_is_reported_only_for_its_sources(bench):
    # the bench reports the committed ncu traffic while the kernel code is the
    # one it was taken on, and nothing (null) once the kernels have changed
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
        d = json.load(f)
    names = ("tsg_umma", "rowstats_umma", "row_bias", "colsum_umma", "css_umma", "css_phi", "gather",
             "select_gate_topk")
    for name in names:
        assert d["kernels"][name]["dram_bytes_per_launch_full"] > 0
    current = d["src_digest"] == bench.src_digest()
    for name in names:
        got = bench.traffic_for(name)
        assert got == (d["kernels"][name]["dram_bytes_per_launch_full"] if current else None)


def test_kernel_roofline_units(bench):
    peaks = {"hbm": 6783.5, "bf16": 1910.3, "bf16_sus": 1704.3, "sm_mhz": 2070.0}
    t = 1e-3
    r = bench.kernel_roofline("tsg_umma", t, 28, 10720, peaks)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert abs(r["achieved"] - bench.tsg_flops_per_layer() * 28 / t / 1e12) < 1e-6
    for name in ("rowstats_umma", "row_bias", "colsum_umma", "css_umma", "css_phi", "gather", "select_gate_topk"):
        r = bench.kernel_roofline(name, t, 28, 10720, peaks)
        assert r["bound"] == "hbm" and r["unit"] == "GB/s" and 0 < r["frac"]
    # the row-bias pass moves a fraction of a key pass
    assert (bench.kernel_roofline("row_bias", t, 1, 10720, peaks)["achieved"]
            < 0.01 * bench.kernel_roofline("rowstats_umma", t, 1, 10720, peaks)["achieved"])
