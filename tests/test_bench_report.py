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
    # the bench reports a kernel's committed ncu traffic while the code of
    # the units it is built from is the code the counters were taken on, and
    # nothing (null) once they have changed
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
        d = json.load(f)
    assert set(d["kernels"]) == set(bench.KERNEL_UNITS)
    for name, e in d["kernels"].items():
        assert e["dram_bytes_per_launch_full"] > 0
        current = e["src_digest"] == bench.kernel_digest(name)
        assert bench.traffic_for(name) == (e["dram_bytes_per_launch_full"] if current else None)


def test_kernel_digest_follows_its_own_units(bench):
    # a code change in one translation unit stales the counters of the
    # kernels built from it and of no other; a comment change stales none
    def edited(unit, old, new):
        def read(name):
            text = bench._read_csrc(name)
            if name == unit:
                assert old in text
                text = text.replace(old, new, 1)
            return text
        return read

    base = {k: bench.kernel_digest(k) for k in bench.KERNEL_UNITS}
    code = edited("select.cu", "k_gather(", "k_gather2(")
    for k in bench.KERNEL_UNITS:
        changed = bench.kernel_digest(k, code) != base[k]
        assert changed == ("select.cu" in bench.KERNEL_UNITS[k]), k
    code = edited("umma.cu", "k_css_phi(", "k_css_phi2(")
    for k in bench.KERNEL_UNITS:
        changed = bench.kernel_digest(k, code) != base[k]
        assert changed == ("umma.cu" in bench.KERNEL_UNITS[k]), k
    shared = edited("common.cuh", "struct FrameTable", "struct FrameTable2")
    assert all(bench.kernel_digest(k, shared) != base[k] for k in bench.KERNEL_UNITS)
    comment = edited("select.cu", "k_gather(", "k_gather(/* a comment */")
    assert all(bench.kernel_digest(k, comment) == base[k] for k in bench.KERNEL_UNITS)


def test_src_digest_reads_source_files_only(bench, tmp_path, monkeypatch):
    # whatever else lands beside the sources (a cache folder of a Python
    # helper, an editor's backup) neither breaks nor changes the digest
    (tmp_path / "a.cu").write_text("int a;\n")
    (tmp_path / "b.cuh").write_text("int b;\n")
    monkeypatch.setattr(bench, "CSRC", str(tmp_path))
    read = lambda name: (tmp_path / name).read_text()
    base = bench.src_digest(read)
    (tmp_path / "__pycache__").mkdir()
    (tmp_path / "notes.txt").write_text("x")
    (tmp_path / "a.cu~").write_text("int z;\n")
    assert bench.src_digest(read) == base
    (tmp_path / "c.cu").write_text("int c;\n")
    assert bench.src_digest(read) != base


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


def test_reference_arm_line(bench):
    # `bench.py --impl reference` times the oracle on the host and prints one
    # JSON line in the bench's own metric, unit and workload
    import subprocess
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "0"], cwd=ROOT, capture_output=True, text=True,
                         timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["metric"].startswith("KV tokens compressed/sec") and d["unit"] == "tokens/s/layer"
    assert d["config"]["layers"] == 28 and d["config"]["n_tokens"] == 53600
    # the same workload description as the GPU arm's line
    assert d["config"] == bench.bench_config(28, 10720, 1)
    # the timing claimed is the timing measured: steps x ms_per_step is the
    # measured time of the timed samples, and the value is extrapolated from it
    assert d["steps"] == 1 and d["extrapolated"] is True
    assert abs(d["steps"] * d["ms_per_step"] - 1e3 * d["measured_s"]) <= 1.0
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    import oracle
    assert cb["cores"] == oracle.host_threads()
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_reference_arm_two_ranks_one_line():
    # under torchrun rank 0 alone times the oracle and prints the line; the
    # other rank exits 0 without work
    import socket
    import subprocess
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    out = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
