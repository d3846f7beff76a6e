#!/usr/bin/env python
"""Benchmark of the ST-Lite per-layer KV-cache compression pass on GB300.

Workload (one "step"): the 28-layer, 50-step GUI trajectory at UI-TARS-1.5-7B
head shape -- 50 frames of 32x32 patches + 48 text tokens per step
(N = 53,600 tokens), 28 query / 4 KV heads, head_dim 128, bf16, window
w = 32, flat budget beta = 20% (B = 10,720 per head and layer).  A step runs
the whole pass (window score, TSG, CSS, top-B, compaction) on all 28 layers.
Synthetic seeded inputs (``synth.trajectory_50``); the 28 layers' K/V
(3.07 GB) exceed the 129 MB L2, so every layer is read cold.

Metric: KV tokens compressed per second per layer = N * layers / step time.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl stlite|reference]

Under torchrun each rank compresses its own trajectory (weak scaling, no
data-path collective); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time
from concurrent.futures import ThreadPoolExecutor

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "KV tokens compressed/sec per layer at beta=20%"
UNIT = "tokens/s/layer"
LAYERS = 28
N_TOK, N_STEPS, GH, GW, N_TEXT = 53600, 50, 32, 32, 48
HQ, HKV, D, W, BETA = 28, 4, 128, 32, 0.2
WORKLOAD = "traj50_32x32+48text_28layers_bf16_beta0.2"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="stlite", choices=["stlite", "reference"])
    ap.add_argument("--layers", type=int, default=LAYERS)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode", action="store_true", help="skip the decode-over-the-cache measurement")
    ap.add_argument("--no-variants", action="store_true", help="skip the ablation-variant step times")
    ap.add_argument("--no-trajectory", action="store_true", help="skip the per-step trajectory sweep")
    ap.add_argument("--prompt-rows", type=int, default=0,
                    help="--workload mean_attention: prompt query rows (0 = the whole cache)")
    ap.add_argument("--workload", default="traj50",
                    choices=["traj50", "uitars", "small_backbone", "long_horizon", "mean_attention"],
                    help="traj50 (default): the 28-layer, 50-step trajectory of the contract line; the others time "
                         "the remaining configurations (one JSON line of their own)")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d["bf16_tflops_sustained"],
                    sm_mhz=d.get("sm_max_mhz", 2070.0), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, sm_mhz=2070.0, source="fallback")


# --------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling (every 100 ms) of SM clock and throttle reasons."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.gpu = gpu_index
        self.p = None

    def start(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        time.sleep(0.3)

    def stop(self):
        if self.p is None:
            return dict(sm_mhz=None, sm_max_mhz=None, reasons=["nvidia-smi unavailable"], samples=0)
        time.sleep(0.15)
        self.p.terminate()
        self.p.wait()
        self.f.flush()
        with open(self.f.name) as f:
            rows = [r.strip().split(", ") for r in f if r.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx = float(r[2])
            except ValueError:
                continue
            for nm, v in zip(names, r[5:9]):
                if v.strip() == "Active":
                    reasons.add(nm)
        return dict(sm_mhz=statistics.median(sm) if sm else None, sm_max_mhz=mx, reasons=sorted(reasons),
                    samples=len(sm))


# ------------------------------------------------------------------- workload

def gen_layers(layers: int, seed: int):
    from paper_2603_00188_gb300 import synth
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        return list(ex.map(lambda l: synth.trajectory_50(l, seed=seed), range(layers)))


def alg_bytes_per_layer(budget: int) -> float:
    """Read K once, read the kept V rows, write the kept K and V rows."""
    s = N_TOK * HKV * D * 2
    kept = budget * HKV * D * 2
    return s + kept + 2 * kept


def tsg_flops_per_layer() -> float:
    n_hist = (N_STEPS - 1) * GH * GW
    return 2.0 * n_hist * GH * GW * D * HKV


def score_flops_per_layer() -> float:
    return 2 * (2.0 * W * (HQ // HKV) * N_TOK * D * HKV)


def exps_per_layer() -> float:
    return 2.0 * W * (HQ // HKV) * N_TOK * HKV


def mufu_peak_texp(peaks) -> float:
    """ex2 throughput of the SM's special-function units: 32 results per
    clock per SM on GB300 (ncu counts one xu warp-instruction per SM-clock
    as its peak), 152 SMs, at the maximum SM clock."""
    return 152 * 32 * peaks["sm_mhz"] * 1e6 / 1e12


def kernel_roofline(name: str, t_launch: float, layers: int, budget: int, peaks) -> dict:
    """Roofline of one launch of `name` (which covers `layers` layers):
    algorithmic work per layer x layers / measured launch time, against the
    bound that limits it.  Algorithmic bytes count each operand once (what a
    perfectly fused kernel must move), not the intermediates this design
    writes."""
    tok_head = N_TOK * HKV
    kbytes = tok_head * D * 2                      # every key once, bf16
    kept = budget * HKV * D * 2                    # kept rows of K (or V)
    if name.startswith("tsg"):
        work = tsg_flops_per_layer()
        ach = work * layers / t_launch / 1e12
        return dict(bound="tensor", achieved=ach, peak=peaks["bf16"], unit="TFLOP/s", frac=ach / peaks["bf16"],
                    frac_of_sustained=ach / peaks["bf16_sus"],
                    work="2*N_hist*N_cur*d*H_kv = %.4g FLOP per layer x %d layers" % (work, layers))
    if name.startswith(("rowstats", "colsum", "css_umma")):
        # every key once; colsum and CSS also write one fp32 value per token and head
        out = 0 if name.startswith("rowstats") else tok_head * 4
        work = kbytes + out
        ach = work * layers / t_launch / 1e9
        d = dict(bound="hbm", achieved=ach, peak=peaks["hbm"], unit="GB/s", frac=ach / peaks["hbm"],
                 work="%.4g bytes per layer (keys once%s) x %d layers"
                      % (work, ", fp32 output per token and head" if out else "", layers))
        if name.startswith(("rowstats", "colsum")):
            ex = exps_per_layer() / 2 * layers / t_launch / 1e12
            d["mufu"] = dict(achieved=ex, peak=mufu_peak_texp(peaks), unit="Texp/s",
                             frac=ex / mufu_peak_texp(peaks))
        return d
    if name.startswith("row_bias"):
        # window-score pass 1's split partials in, one bias per query row out;
        # the split count follows the library's rule for this shape (one
        # layer's splits fill one wave of 152 SMs, every split non-empty)
        rows = HKV * W * (HQ // HKV)
        tiles = (N_TOK + 255) // 256
        target = min(tiles, (152 + HKV - 1) // HKV)
        per_t = max(2, (tiles + target - 1) // target)
        nsplit = (tiles + per_t - 1) // per_t
        work = rows * nsplit * 8 + rows * 4
    elif name.startswith("css_phi"):
        work = tok_head * (5 * 4 + 4)              # five dot products in, Phi out
    elif name.startswith("css_box"):
        work = kbytes + tok_head * 8               # every key once; Phi and 1/|k| out
    elif name.startswith("select"):
        work = tok_head * 3 * 4 + budget * HKV * 4  # A, Phi, rho in; indices out
    elif name.startswith("gather"):
        work = 4 * kept + budget * HKV * 4         # kept K, V rows in and out; indices
    else:
        work = kbytes
    ach = work * layers / t_launch / 1e9
    return dict(bound="hbm", achieved=ach, peak=peaks["hbm"], unit="GB/s", frac=ach / peaks["hbm"],
                work="%.4g bytes per layer x %d layers" % (work, layers))


# --------------------------------------------------------------- oracle arm

def bench_config(layers: int, budget: int, world: int) -> dict:
    """The workload description both arms print (same keys and values)."""
    return dict(workload=WORKLOAD, layers=layers, n_tokens=N_TOK, frames=N_STEPS, grid="%dx%d" % (GH, GW),
                text_per_step=N_TEXT, q_heads=HQ, kv_heads=HKV, head_dim=D, window=W, beta=BETA,
                budget=budget, l2="inputs larger than L2 (%.2f GB K/V per step)" %
                (2 * layers * N_TOK * HKV * D * 2 / 1e9),
                timing=("CUDA graph of one step (one stlite_compress_layers call: window score and Phi on the "
                        "call's second stream, joined before the selection), replayed"),
                parallelism="dp%d" % world)


def bf16_inputs(wl):
    """The workload's q and k as the bf16 values the GPU arm computes on,
    exactly converted to float64 for the oracle."""
    import torch
    q = torch.from_numpy(wl.q).to(torch.bfloat16).to(torch.float64).numpy()
    k = torch.from_numpy(wl.k).to(torch.bfloat16).to(torch.float64).numpy()
    return q, k


def oracle_sample(wl, pool_stride: int = 16, q_heads: int = HQ // HKV):
    """Times the oracle single-threaded on KV head 0 of one layer: the
    window score of `q_heads` of the head's G query heads, CSS, the TSG
    threshold and gate, integrated score and top-B in full, and rho on every
    pool_stride-th historical token.  Returns the seconds extrapolated to the
    whole layer (all query heads, every historical token, all KV heads), the
    measured seconds, and a description of the sample."""
    import oracle
    G = HQ // HKV
    q64, k64 = bf16_inputs(wl)
    off, gh, gw = wl.frames
    b = oracle.budget(wl.n, wl.beta)
    kh = np.ascontiguousarray(k64[:, :1])
    qh = np.ascontiguousarray(q64[:, :q_heads])
    t0 = time.perf_counter()
    a = oracle.abase(qh, kh)
    t1 = time.perf_counter()
    phi = oracle.css_phi(kh, wl.frames)
    t2 = time.perf_counter()
    pool = oracle.pool_tokens(wl.frames)
    sample = pool[::pool_stride]
    rho = oracle.tsg_rho(kh, wl.frames, tokens=sample)
    t3 = time.perf_counter()
    rho[0, pool] = np.nan_to_num(rho[0, pool], nan=0.5)   # unsampled tokens: placeholder values
    tau, gate, _ = oracle.tsg_gate(rho, wl.frames, b)
    s = oracle.combine(a, phi, gate, wl.frames)
    oracle.topk(s, b)
    t4 = time.perf_counter()
    per_head = (t1 - t0) * (G / q_heads) + (t2 - t1) + (t3 - t2) * (len(pool) / len(sample)) + (t4 - t3)
    note = ("oracle on 1 thread, KV head 0 of one layer: window score of %d/%d query heads, CSS, gate and top-B "
            "in full, rho on 1/%d of the %d historical tokens; extrapolated to all query heads, all historical "
            "tokens and %d KV heads" % (q_heads, G, pool_stride, len(pool), HKV))
    return per_head * HKV, t4 - t0, note


def oracle_layer(wl, threads: int, pool_stride: int = 1):
    """Times the oracle on one whole layer (all KV heads and query heads) on
    `threads` host threads: window score, CSS, rho on every pool_stride-th
    historical token (all of them at stride 1), threshold, gate, integrated
    score and top-B.  Returns the seconds for the whole layer (rho's time
    scaled by the pool fraction when strided), the measured seconds, and a
    description."""
    import oracle
    q64, k64 = bf16_inputs(wl)
    b = oracle.budget(wl.n, wl.beta)
    t0 = time.perf_counter()
    a = oracle.abase(q64, k64, threads=threads)
    t1 = time.perf_counter()
    phi = oracle.css_phi(k64, wl.frames, threads=threads)
    t2 = time.perf_counter()
    pool = oracle.pool_tokens(wl.frames)
    sample = pool[::pool_stride]
    rho = oracle.tsg_rho(k64, wl.frames, threads=threads, tokens=sample)
    t3 = time.perf_counter()
    if pool_stride > 1:
        rho[:, pool] = np.nan_to_num(rho[:, pool], nan=0.5)   # unsampled tokens: placeholder values
    tau, gate, _ = oracle.tsg_gate(rho, wl.frames, b)
    s = oracle.combine(a, phi, gate, wl.frames)
    oracle.topk(s, b)
    t4 = time.perf_counter()
    est = (t1 - t0) + (t2 - t1) + (t3 - t2) * (len(pool) / len(sample)) + (t4 - t3)
    if pool_stride == 1:
        note = ("oracle on %d threads, one whole layer (all %d KV heads and %d query heads, rho of all %d "
                "historical tokens), nothing extrapolated" % (threads, HKV, HQ, len(pool)))
    else:
        note = ("oracle on %d threads, one layer (all %d KV heads and %d query heads) with rho on 1/%d of the %d "
                "historical tokens; rho's time scaled to the whole pool" % (threads, HKV, HQ, pool_stride,
                                                                         len(pool)))
    return est, t4 - t0, note


def run_reference(args):
    """The reference arm: the oracle, as it stands, on the host cores.  Each
    step is one bounded sample of the workload (one layer with rho on 1/16 of
    the pool, all host threads); the line reports the seconds really
    measured per step and the throughput extrapolated from them."""
    world, rank, _ = dist_env()
    if rank != 0:   # under torchrun rank 0 alone times the oracle; the others exit 0
        return
    sys.stdout.flush()
    import oracle
    oracle.build()
    threads = oracle.host_threads()
    wls = gen_layers(2, seed=0)
    stride = 16
    vals, measured = [], []
    note = ""
    for step in range(args.warmup + args.steps):
        t_layer, t_raw, note = oracle_layer(wls[step % len(wls)], threads, pool_stride=stride)
        if step >= args.warmup:
            vals.append(N_TOK / t_layer)
            measured.append(t_raw)
    value = statistics.mean(vals)
    ms_step = 1e3 * statistics.mean(measured)
    budget = oracle.budget(N_TOK, BETA)
    line = dict(impl="reference", metric=METRIC, value=value, unit=UNIT, n_gpus=args.gpus, steps=args.steps,
                warmup=args.warmup, ms_per_step=ms_step, higher_is_better=True, scaling="weak", vs_baseline=None,
                dtype="f64", data="synthetic", config=bench_config(LAYERS, budget, max(world, args.gpus)),
                extrapolated=True, measured_s=round(sum(measured), 3),
                step_note="each step is one bounded sample (%s); value = N / the layer time extrapolated from "
                          "it, ms_per_step = the sample's measured time" % note,
                cpu_baseline=dict(value=value, unit=UNIT, cores=threads, kind="oracle", sample=note,
                                  measured_s=round(sum(measured), 3)),
                e2e=dict(value=value, unit=UNIT, h2d_bytes_per_step=0, d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------- GPU arm

def _code_only(text: str) -> str:
    """C/C++/CUDA source without its comments (string and character literals
    kept) and with every run of white space made one blank, so that editing
    a comment or reflowing lines does not mark counters as stale."""
    out, i, n = [], 0, len(text)
    while i < n:
        if text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
        elif text[i] in "\"'":
            q, j = text[i], i + 1
            while j < n and text[j] != q:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        else:
            out.append(text[i])
            i += 1
    return " ".join("".join(out).split())


CSRC = os.path.join(ROOT, "paper_2603_00188_gb300", "csrc")

# The translation units each step kernel is built from, on top of the shared
# headers and the host planning in api.cu (frame tables, workspace plan):
# a code change there changes what the kernel does, a change elsewhere does
# not.  The row-bias pass also depends on umma.cu, whose launcher picks the
# number of row-statistics splits it merges.
KERNEL_UNITS = {
    "tsg_umma": ("umma.cu",),
    "rowstats_umma": ("umma.cu",),
    "colsum_umma": ("umma.cu",),
    "css_umma": ("umma.cu",),
    "css_phi": ("umma.cu",),
    "row_bias": ("simt.cu", "umma.cu"),
    "select_gate_topk": ("select.cu",),
    "gather": ("select.cu",),
}
SHARED_UNITS = ("api.cu", "common.cuh", "kernels.cuh", "ptx.cuh")


def _digest(names, read):
    h = hashlib.sha256()
    for name in sorted(names):
        h.update(name.encode() + _code_only(read(name)).encode())
    return h.hexdigest()[:16]


def _read_csrc(name):
    with open(os.path.join(CSRC, name), encoding="utf-8") as f:
        return f.read()


def src_digest(read=_read_csrc):
    """Digest of all kernel sources (comments excluded)."""
    return _digest([n for n in os.listdir(CSRC) if n.endswith((".cu", ".cuh", ".h"))], read)


def kernel_digest(kernel: str, read=_read_csrc):
    """Digest of the sources (comments excluded) that `kernel` is built from:
    the committed ncu counters of that kernel must have been taken on them."""
    return _digest(KERNEL_UNITS[kernel] + SHARED_UNITS, read)


def traffic_for(kernel: str):
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, if it
    was taken on the kernel's current sources."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get("kernels", {}).get(kernel)
    if e is None:
        return None
    want = e.get("src_digest")
    if want is None:
        return e.get("dram_bytes_per_launch_full") if d.get("src_digest") == src_digest() else None
    return e.get("dram_bytes_per_launch_full") if want == kernel_digest(kernel) else None


# ------------------------------------------------------- critical hit rate

def gpu_critical_hit_rate(stlite, q_probe, k, idx_keep, stream=None):
    """Per KV head, the share of a probe query's B most-attended tokens that
    the compressed cache kept: the probe's window score over every cached key
    (Eq. 2 with the probe as the only window row, stlite_score) and its Top_B
    (stlite_select_topk with no gate and no CSS: S = A) run in the library's
    kernels; only the set intersection is a torch op."""
    import torch
    n, hkv = k.shape[0], k.shape[1]
    b = idx_keep.shape[1]
    none = ([], [], [])
    prm = stlite.make_params(1.0, k_override=b, alpha=0.0, tsg_enable=0, css_enable=0)
    sh = stlite.make_shape(q_probe, k)
    ws = stlite.workspace(sh, none, prm, device=k.device)
    a = torch.empty((hkv, n), dtype=torch.float32, device=k.device)
    top = torch.empty((hkv, b), dtype=torch.int32, device=k.device)
    stlite.stlite_score(q_probe, k, a, ws, stream)
    stlite.stlite_select_topk(q_probe, k, none, prm, a, None, None, b, top, None, ws, stream)
    return torch.stack([torch.isin(idx_keep[h], top[h]).sum() for h in range(hkv)]).double() / b


# ------------------------------------------------------------ multi-rank glue

def dist_env():
    """(world, rank, local_rank) from the torchrun environment (1, 0, 0 alone)."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(ms: float, device, world: int) -> float:
    """The slowest rank's time: every rank processed its own units, so the job
    took as long as its slowest rank."""
    if world == 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, layers: int, ms: float) -> float:
    """Whole-job tokens per second per layer: every rank compresses its own
    trajectory of `layers` layers of N_TOK tokens (weak scaling)."""
    return world * N_TOK * layers / (ms * 1e-3)


def run_gpu(args):
    import torch
    import torch.distributed as dist

    world, rank, local = dist_env()
    if world > 1:
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2603_00188_gb300 import build as pkg_build
    if rank == 0:
        pkg_build.build()
    if world > 1:
        dist.barrier()
    from paper_2603_00188_gb300 import stlite

    def barrier():
        if world > 1:
            dist.barrier()

    peaks = load_peaks()
    L = args.layers
    wls = gen_layers(L, seed=rank)
    fs = stlite.FrameSpec(*wls[0].frames)
    host = []
    for wl in wls:
        host.append(tuple(torch.from_numpy(x).to(torch.bfloat16).pin_memory() for x in (wl.q, wl.k, wl.v)))
    qs = [h[0].to(dev) for h in host]
    ks = [h[1].to(dev) for h in host]
    vs = [h[2].to(dev) for h in host]
    prm = stlite.make_params(BETA)
    sh = stlite.make_shape(qs[0], ks[0])
    budget = stlite.stlite_budget(N_TOK, BETA)
    ws_layer = stlite.stlite_workspace_size(sh, fs, prm)
    ws = torch.zeros(L * ws_layer, dtype=torch.uint8, device=dev)
    kos = [torch.empty((budget, HKV, D), dtype=torch.bfloat16, device=dev) for _ in range(L)]
    vos = [torch.empty_like(kos[0]) for _ in range(L)]
    idxs = [torch.empty((HKV, budget), dtype=torch.int32, device=dev) for _ in range(L)]
    layer_io = [(qs[l], ks[l], vs[l], kos[l], vos[l], idxs[l]) for l in range(L)]
    stream = torch.cuda.Stream(device=dev)

    def step(st=None):
        # all layers in one call: every stage is one launch over the 28 layers
        stlite.stlite_compress_layers(layer_io, fs, prm, ws, st)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step(stream)
    stream.synchronize()
    assert stlite.stlite_device_status(ws, stream) == stlite.STLITE_OK

    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step(stream)
    # ---- timed region: K graph replays of the full 28-layer step.  The clock
    # sampler runs from one second of untimed replays (steady clocks) to the end.
    clocks = ClockSampler(local)
    clocks.start()
    t_warm = time.perf_counter()
    with torch.cuda.stream(stream):
        while True:
            for _ in range(max(3, args.warmup)):
                graph.replay()
            stream.synchronize()
            if time.perf_counter() - t_warm > 1.0:
                break
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            graph.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1) / args.steps
    ms = max_over_ranks(ms, dev, world)
    assert stlite.stlite_device_status(ws, stream) == stlite.STLITE_OK
    value = job_throughput(world, L, ms)

    # ---- per-kernel device time (CUDA events around each launch, eager replay)
    stlite.stlite_timing_read()
    stlite.stlite_timing_enable(True)
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            step(stream)
    stream.synchronize()
    stlite.stlite_timing_enable(False)
    ktimes = stlite.stlite_timing_read()
    per_step_launches = sum(c for c, _ in ktimes.values()) // args.steps
    kernels = {k: dict(launches_per_step=c // args.steps, ms_per_launch=t / c, share=None)
               for k, (c, t) in ktimes.items()}
    tot = sum(t for _, t in ktimes.values())
    for k, (c, t) in ktimes.items():
        kernels[k]["share"] = t / tot
    dom = max(ktimes, key=lambda k: ktimes[k][1])
    for k, (c, t) in ktimes.items():
        kernels[k]["roofline"] = kernel_roofline(k, t / c * 1e-3, L, budget, peaks)
        kernels[k]["roofline"]["traffic"] = traffic_for(k) if L == LAYERS else None
    roof = dict(kernels[dom]["roofline"], kernel=dom)
    roof["traffic"] = traffic_for(dom) if L == LAYERS else None
    roof["peak_source"] = peaks["source"] + (" burst" if roof["unit"] == "TFLOP/s" else "")

    # ---- the paper's ablation variants on the same workload: step time of
    # the whole pass (one graph per variant) and the kernels each one changes
    variants = None
    if not args.no_variants:
        variants = {}
        rng = np.random.default_rng(2603)
        mass = 1.0 + 0.013 * rng.standard_normal(L)   # near-uniform layer mass (cross-layer CV about 1.3 %)
        h_budgets = stlite.stlite_hierarchical_budgets(list(mass), L * budget, N_TOK)
        h_out = [(torch.empty((b, HKV, D), dtype=torch.bfloat16, device=dev),
                  torch.empty((b, HKV, D), dtype=torch.bfloat16, device=dev),
                  torch.empty((HKV, b), dtype=torch.int32, device=dev)) for b in h_budgets]
        h_io = [(qs[l], ks[l], vs[l]) + h_out[l] for l in range(L)]
        cases = [("tsg_dot", dict(tsg_metric=stlite.STLITE_TSG_DOT)),
                 ("tsg_neg_l2", dict(tsg_metric=stlite.STLITE_TSG_NEG_L2)),
                 ("fixed_tau_0.85", dict(fixed_tau=0.85)),
                 ("uniform_base", dict(base_scorer=stlite.STLITE_BASE_UNIFORM)),
                 ("abase_max", dict(abase_norm=stlite.STLITE_ABASE_MAX)),
                 ("css_3x3_box", None), ("css_5x5", dict(css_size=5)), ("css_7x7", dict(css_size=7)),
                 ("css_9x9", dict(css_size=9)), ("hierarchical_budgets", dict())]
        for name, kw in cases:
            if name == "css_3x3_box":
                # the method's CSS on the box-sum kernel instead of the tensor cores (staged entry)
                phi_b = torch.empty((HKV, N_TOK), dtype=torch.float32, device=dev)

                def vstep(st=None):
                    for l in range(L):
                        stlite.stlite_spatial_saliency_size(qs[l], ks[l], fs, 3, phi_b, ws, st)
            elif name == "hierarchical_budgets":
                def vstep(st=None):
                    stlite.stlite_compress_layers_budgets(h_io, fs, prm, h_budgets, ws, st)
            else:
                prm_v = stlite.make_params(BETA, **kw)

                def vstep(st=None, prm_v=prm_v):
                    stlite.stlite_compress_layers(layer_io, fs, prm_v, ws, st)
            with torch.cuda.stream(stream):
                for _ in range(2):
                    vstep(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                vstep(stream)
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            reps = max(5, min(20, args.steps))
            with torch.cuda.stream(stream):
                for _ in range(2):
                    g.replay()
                a0.record(stream)
                for _ in range(reps):
                    g.replay()
                a1.record(stream)
            torch.cuda.synchronize()
            assert stlite.stlite_device_status(ws, stream) == stlite.STLITE_OK
            stlite.stlite_timing_read()
            stlite.stlite_timing_enable(True)
            with torch.cuda.stream(stream):
                vstep(stream)
            stream.synchronize()
            stlite.stlite_timing_enable(False)
            vk = stlite.stlite_timing_read()
            entry = dict(ms_per_step=a0.elapsed_time(a1) / reps,
                         kernels_ms={k: t / c for k, (c, t) in vk.items()})
            if "css_box" in vk:
                # the staged entry launches once per layer, the fused pass once for all layers
                c, t = vk["css_box"]
                entry["css_box_roofline"] = kernel_roofline("css_box", t / c * 1e-3,
                                                            1 if name == "css_3x3_box" else L, budget, peaks)
            if name == "hierarchical_budgets":
                entry["budgets_min_max"] = [min(h_budgets), max(h_budgets)]
            variants[name] = entry
        # the prompt-wide bases (Mean Attention, full attention): every one of
        # the N prompt positions' query rows votes (causal), the work of the
        # prompt's attention twice, so one layer (layer 0) is timed: prompt
        # score, CSS, gate, Eq. 9 and Top-B on that base, compaction
        gq = torch.Generator().manual_seed(2604)
        q_prompt = torch.randn((N_TOK, HQ, D), generator=gq).to(torch.bfloat16).to(dev)
        shp = stlite.prompt_shape(q_prompt, ks[0])
        ws_p = torch.zeros(stlite.stlite_prompt_workspace_size(shp, N_TOK), dtype=torch.uint8, device=dev)
        a_p = torch.empty((HKV, N_TOK), dtype=torch.float32, device=dev)
        phi_p, rho_p = torch.empty_like(a_p), torch.empty_like(a_p)
        tau_p = torch.empty((HKV,), dtype=torch.float32, device=dev)
        gate_p = torch.empty((HKV, N_TOK), dtype=torch.uint8, device=dev)
        for name, base in (("mean_attention_base", stlite.STLITE_PROMPT_MEAN),
                           ("full_attention_base", stlite.STLITE_PROMPT_FULL)):
            def pstep(st=None, base=base):
                stlite.stlite_prompt_score(q_prompt, ks[0], base, a_p, ws_p, st)
                stlite.stlite_spatial_saliency(qs[0], ks[0], fs, phi_p, ws, st)
                stlite.stlite_gate_frames(qs[0], ks[0], fs, budget, rho_p, tau_p, gate_p, ws, st)
                stlite.stlite_select_topk(qs[0], ks[0], fs, prm, a_p, phi_p, gate_p, budget, idxs[0], None, ws, st)
                stlite.stlite_compact(qs[0], ks[0], vs[0], budget, idxs[0], kos[0], vos[0], st)
            with torch.cuda.stream(stream):
                pstep(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                pstep(stream)
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            reps = 5
            with torch.cuda.stream(stream):
                g.replay()
                a0.record(stream)
                for _ in range(reps):
                    g.replay()
                a1.record(stream)
            torch.cuda.synchronize()
            assert stlite.stlite_device_status(ws_p, stream) == stlite.STLITE_OK
            stlite.stlite_timing_read()
            stlite.stlite_timing_enable(True)
            with torch.cuda.stream(stream):
                pstep(stream)
            stream.synchronize()
            stlite.stlite_timing_enable(False)
            vk = stlite.stlite_timing_read()
            pass_flop = 2.0 * (N_TOK * (N_TOK + 1) / 2) * D * HQ   # one causal QK^T over the prompt
            entry = dict(ms_per_layer=a0.elapsed_time(a1) / reps, layers_timed=1, prompt_rows=N_TOK,
                         kernels_ms={k: t / c for k, (c, t) in vk.items()})
            for kname in ("prompt_rowstats", "prompt_colsum"):
                if kname in vk:
                    c, t = vk[kname]
                    ach = pass_flop / (t / c * 1e-3) / 1e12
                    entry[kname + "_roofline"] = dict(bound="tensor", achieved=ach, peak=peaks["bf16"],
                                                      unit="TFLOP/s", frac=ach / peaks["bf16"],
                                                      work="2*(N(N+1)/2)*d*Hq = %.4g FLOP (causal half)" %
                                                           pass_flop)
            variants[name] = entry
        del q_prompt, ws_p
        # the variants overwrote the shared workspace's per-layer results; the
        # published method's outputs are recomputed for what follows
        with torch.cuda.stream(stream):
            step(stream)
        stream.synchronize()

    # ---- per-step use across the trajectory: at agent step t the prompt holds
    # frames 0..t-1 (t * 1072 tokens), and all 28 layers are compressed once
    # the step's prefill is done; one graph per step length
    trajectory = None
    if not args.no_trajectory:
        trajectory = []
        step_tok = GH * GW + N_TEXT
        for t in (1, 2, 5, 10, 20, 30, 40, 50):
            n_t = t * step_tok
            fr = wls[0].frames
            fs_t = stlite.FrameSpec(fr[0][:t], fr[1][:t], fr[2][:t])
            b_t = stlite.stlite_budget(n_t, BETA)
            prm_t = stlite.make_params(BETA)
            sh_t = stlite.make_shape(qs[0], ks[0][:n_t])
            assert stlite.stlite_workspace_size(sh_t, fs_t, prm_t) <= ws_layer
            ix_t = torch.empty((L, HKV, b_t), dtype=torch.int32, device=dev)
            io_t = [(qs[l], ks[l][:n_t], vs[l][:n_t], kos[l][:b_t], vos[l][:b_t], ix_t[l]) for l in range(L)]

            def tstep(st=None, io_t=io_t, fs_t=fs_t, prm_t=prm_t):
                stlite.stlite_compress_layers(io_t, fs_t, prm_t, ws, st)
            with torch.cuda.stream(stream):
                for _ in range(2):
                    tstep(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                tstep(stream)
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            reps = max(5, min(20, args.steps))
            with torch.cuda.stream(stream):
                for _ in range(2):
                    g.replay()
                a0.record(stream)
                for _ in range(reps):
                    g.replay()
                a1.record(stream)
            torch.cuda.synchronize()
            assert stlite.stlite_device_status(ws, stream) == stlite.STLITE_OK
            t_ms = a0.elapsed_time(a1) / reps
            trajectory.append(dict(frames=t, n_tokens=n_t, budget=b_t, ms_per_step=t_ms,
                                   value=n_t * L / (t_ms * 1e-3), unit=UNIT))
        with torch.cuda.stream(stream):
            step(stream)
        stream.synchronize()

    # ---- consumer: one decode step (a query row per layer) over the full and
    # the compressed caches of all layers, each step one CUDA graph
    decode = None
    if not args.no_decode:
        probes = [qs[l][-1:].contiguous() for l in range(L)]    # the last window row as the next query
        dsh = stlite.make_shape(probes[0], ks[0])
        dws = torch.zeros(max(stlite.stlite_decode_workspace_size(dsh),
                              stlite.stlite_decode_layers_workspace_size(dsh, L)), dtype=torch.uint8, device=dev)
        douts = [torch.empty((1, HQ, D), dtype=torch.float32, device=dev) for _ in range(L)]

        def decode_ms(kk, vv, batched=True):
            # batched: one stlite_decode_attention_layers call for all layers;
            # else one stlite_decode_attention call per layer
            io = [(probes[l], kk[l], vv[l], douts[l]) for l in range(L)]

            def one():
                if batched:
                    stlite.stlite_decode_attention_layers(io, dws, stream)
                else:
                    for l in range(L):
                        stlite.stlite_decode_attention(probes[l], kk[l], vv[l], douts[l], dws, stream)
            with torch.cuda.stream(stream):
                for _ in range(3):
                    one()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                one()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            reps = max(10, args.steps)
            with torch.cuda.stream(stream):
                for _ in range(3):
                    g.replay()
                a.record(stream)
                for _ in range(reps):
                    g.replay()
                b.record(stream)
            torch.cuda.synchronize()
            return a.elapsed_time(b) / reps

        t_full = decode_ms(ks, vs)
        t_comp = decode_ms(kos, vos)
        t_full_1 = decode_ms(ks, vs, batched=False)
        t_comp_1 = decode_ms(kos, vos, batched=False)
        assert stlite.stlite_device_status(dws, stream) == stlite.STLITE_OK
        # critical hit rate of the same probe rows: mean over layers and KV heads
        chr_ = torch.stack([gpu_critical_hit_rate(stlite, probes[l], ks[l], idxs[l], stream) for l in range(L)])
        row = HKV * D * 2 * 2   # one cached token's key and value rows, bf16
        decode = dict(layers=L, cache_rows_full=N_TOK, cache_rows_compressed=budget,
                      full_us_per_step=t_full * 1e3, compressed_us_per_step=t_comp * 1e3,
                      speedup=t_full / t_comp,
                      full_gbs=N_TOK * row * L / (t_full * 1e-3) / 1e9,
                      compressed_gbs=budget * row * L / (t_comp * 1e-3) / 1e9,
                      peak_gbs=peaks["hbm"],
                      critical_hit_rate=float(chr_.mean()), critical_hit_rate_min=float(chr_.min()),
                      per_layer_calls=dict(full_us_per_step=t_full_1 * 1e3, compressed_us_per_step=t_comp_1 * 1e3),
                      note="one query row per layer (the last window row) attends over every cached row (keys and "
                           "values read once), all layers in one stlite_decode_attention_layers call "
                           "(per_layer_calls: one stlite_decode_attention call per layer); full = N rows, "
                           "compressed = the B kept rows; critical hit rate = share of that probe's B "
                           "most-attended tokens kept (synthetic inputs)")

    # ---- end to end: host (pinned) inputs -> device -> compress -> host outputs.
    # Q and K of every layer are copied to the device (every stage reads all
    # keys); V stays in page-locked host memory, from which the compaction
    # reads only the kept rows.  Device inputs and outputs are double-buffered
    # so that step s+1's copies overlap step s's compression and read-back.
    e2e = None
    if not args.no_e2e:
        GRP = 4  # layers per batched call, so that compression overlaps the copies
        sets = []
        for b in range(2):
            dq = qs if b == 0 else [torch.empty_like(t) for t in qs]
            dk = ks if b == 0 else [torch.empty_like(t) for t in ks]
            dko = kos if b == 0 else [torch.empty_like(t) for t in kos]
            dvo = vos if b == 0 else [torch.empty_like(t) for t in vos]
            dix = idxs if b == 0 else [torch.empty_like(t) for t in idxs]
            io = [(dq[l], dk[l], host[l][2], dko[l], dvo[l], dix[l]) for l in range(L)]
            h_out = [(torch.empty(kos[0].shape, dtype=torch.bfloat16).pin_memory(),
                      torch.empty(vos[0].shape, dtype=torch.bfloat16).pin_memory(),
                      torch.empty(idxs[0].shape, dtype=torch.int32).pin_memory()) for _ in range(L)]
            sets.append(dict(q=dq, k=dk, ko=dko, vo=dvo, ix=dix, io=io, h_out=h_out,
                             ws=torch.zeros(L * ws_layer, dtype=torch.uint8, device=dev),
                             ev_in=[torch.cuda.Event() for _ in range(L)],
                             ev_done=[torch.cuda.Event() for _ in range(L)],
                             ev_free=torch.cuda.Event()))
        cp_in, cp_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
        kept_v = budget * HKV * D * 2
        bi = sum(host[l][0].numel() * 2 + host[l][1].numel() * 2 + kept_v for l in range(L))
        bo = sum(t.numel() * t.element_size() for t in sets[0]["h_out"][0]) * L

        def e2e_step(it):
            S = sets[it % 2]
            if it >= 2:
                cp_in.wait_event(S["ev_free"])   # step it-2 has read this set and copied its outputs back
            with torch.cuda.stream(cp_in):
                for l in range(L):
                    S["q"][l].copy_(host[l][0], non_blocking=True)
                    S["k"][l].copy_(host[l][1], non_blocking=True)
                    S["ev_in"][l].record(cp_in)
            for g0 in range(0, L, GRP):
                g1 = min(L, g0 + GRP)
                stream.wait_event(S["ev_in"][g1 - 1])
                stlite.stlite_compress_layers(S["io"][g0:g1], fs, prm, S["ws"][g0 * ws_layer:g1 * ws_layer],
                                              stream)
                S["ev_done"][g0].record(stream)
                cp_out.wait_event(S["ev_done"][g0])
                with torch.cuda.stream(cp_out):
                    for l in range(g0, g1):
                        S["h_out"][l][0].copy_(S["ko"][l], non_blocking=True)
                        S["h_out"][l][1].copy_(S["vo"][l], non_blocking=True)
                        S["h_out"][l][2].copy_(S["ix"][l], non_blocking=True)
            S["ev_free"].record(cp_out)

        for it in range(max(2, args.warmup)):
            e2e_step(it)
        torch.cuda.synchronize()
        barrier()
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(cp_in)
        stream.wait_stream(cp_in)
        cp_out.wait_stream(cp_in)
        # the end of every step (its last read-back), for the spread of the
        # intervals between steps: the host link sees other traffic of the
        # machine, and a step or two that stall for tens of ms raise the mean
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        for it in range(args.steps):
            e2e_step(it)
            ends[it].record(cp_out)
        stream.wait_stream(cp_out)
        stream.wait_stream(cp_in)
        f1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ms_e2e = f0.elapsed_time(f1) / args.steps
        gaps = sorted(ends[i - 1].elapsed_time(ends[i]) for i in range(1, args.steps))
        ms_e2e = max_over_ranks(ms_e2e, dev, world)
        # the host copies hold the device results of the last step
        last = sets[(args.steps - 1) % 2]
        for l in (0, L - 1):
            assert torch.equal(last["h_out"][l][2], idxs[l].cpu())
            assert torch.equal(last["h_out"][l][1], vos[l].cpu())
        # the host link alone, measured on the same buffers: the step's input
        # bytes host -> device (q, k and as many bytes of v as the kept rows)
        # and its output bytes device -> host, each direction alone and both
        # at once (the floor of a step that moves them)
        S = sets[0]
        hv = [host[l][2].view(-1)[:kept_v // 2] for l in range(L)]
        dv = torch.empty(kept_v // 2, dtype=torch.bfloat16, device=dev)

        def h2d():
            with torch.cuda.stream(cp_in):
                for l in range(L):
                    S["q"][l].copy_(host[l][0], non_blocking=True)
                    S["k"][l].copy_(host[l][1], non_blocking=True)
                    dv.copy_(hv[l], non_blocking=True)

        def d2h():
            with torch.cuda.stream(cp_out):
                for l in range(L):
                    S["h_out"][l][0].copy_(S["ko"][l], non_blocking=True)
                    S["h_out"][l][1].copy_(S["vo"][l], non_blocking=True)
                    S["h_out"][l][2].copy_(S["ix"][l], non_blocking=True)

        def link_ms(fns, reps=3):
            best = None
            for _ in range(reps):
                torch.cuda.synchronize()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(cp_in)
                cp_out.wait_stream(cp_in)
                for fn in fns:
                    fn()
                cp_in.wait_stream(cp_out)
                e1.record(cp_in)
                torch.cuda.synchronize()
                t = e0.elapsed_time(e1)
                best = t if best is None else min(best, t)
            return best

        t_in, t_out, t_both = link_ms([h2d]), link_ms([d2h]), link_ms([h2d, d2h])
        link = dict(h2d_gbs=bi / (t_in * 1e-3) / 1e9, d2h_gbs=bo / (t_out * 1e-3) / 1e9,
                    h2d_ms=t_in, d2h_ms=t_out, both_directions_ms=t_both,
                    floor_ms=t_both, e2e_over_floor=ms_e2e / t_both,
                    note="cudaMemcpyAsync of the step's bytes from and to page-locked host memory, best of 3; "
                         "floor = both directions at once")
        spread = dict(min=gaps[0], median=statistics.median(gaps), max=gaps[-1],
                      note="ms between the ends of consecutive steps (last read-back), rank 0") if gaps else None
        e2e = dict(value=job_throughput(world, L, ms_e2e), unit=UNIT, h2d_bytes_per_step=bi,
                   d2h_bytes_per_step=bo, ms_per_step=ms_e2e, step_interval_ms=spread, host_link=link,
                   note="q and k copied host -> device by torch (cudaMemcpyAsync on a copy stream) before the "
                        "library call; v read by the compaction kernel in place from page-locked host memory "
                        "(kept rows only); k_out, v_out, idx copied back by torch")

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        threads = oracle.host_threads()
        # all host threads: one whole layer, nothing extrapolated
        t_all, t_all_raw, note_all = oracle_layer(wls[0], threads, pool_stride=1)
        # one thread: a sample of one KV head, extrapolated to the layer
        t_one, t_one_raw, note_one = oracle_sample(wls[0], pool_stride=16)
        cpu = dict(value=N_TOK / t_all, unit=UNIT, cores=threads, kind="oracle", sample=note_all,
                   measured_s=round(t_all_raw, 2),
                   single_core=dict(value=N_TOK / t_one, unit=UNIT, cores=1, sample=note_one,
                                    measured_s=round(t_one_raw, 2), extrapolated=True))

    if rank == 0:
        line = dict(metric=METRIC, value=value, unit=UNIT, n_gpus=world, steps=args.steps, warmup=args.warmup,
                    ms_per_step=ms, higher_is_better=True, scaling="weak", vs_baseline=None, dtype="bf16",
                    data="synthetic",
                    config=bench_config(L, budget, world),
                    hbm=dict(achieved_gbs=alg_bytes_per_layer(budget) * L / (ms * 1e-3) / 1e9,
                             peak_gbs=peaks["hbm"],
                             frac=alg_bytes_per_layer(budget) * L / (ms * 1e-3) / 1e9 / peaks["hbm"],
                             bytes_per_layer=alg_bytes_per_layer(budget)),
                    tensor=dict(achieved_tflops=(tsg_flops_per_layer() + score_flops_per_layer()) * L / (ms * 1e-3) / 1e12,
                                peak_tflops=peaks["bf16"]),
                    roofline=roof, kernels=kernels, gpu_launches=per_step_launches * args.steps,
                    clocks=dict(sm_mhz=clk["sm_mhz"], sm_max_mhz=clk["sm_max_mhz"], reasons=clk["reasons"],
                                samples=clk["samples"]),
                    e2e=e2e, cpu_baseline=cpu, decode=decode, variants=variants, trajectory=trajectory)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_workload(args):
    """The other configurations, timed through the same API on one GPU: a
    1-layer UI-TARS-shaped cache at beta 10-40 %, the batch-8 smaller-backbone
    shape (28 layers, one packed varlen call per layer) at beta 10 and 40 %,
    and the long-horizon cache (1 layer and 28 layers) at beta 10 %.  One graph
    per case; L2 is flushed between timed replays by inputs larger than L2
    where they are (the 1-layer cases are not, and say so)."""
    import torch
    from paper_2603_00188_gb300 import build as pkg_build
    from paper_2603_00188_gb300 import stlite, synth
    pkg_build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks = load_peaks()
    stream = torch.cuda.Stream(device=dev)

    def bf16(x):
        return torch.from_numpy(x).to(torch.bfloat16).to(dev)

    def timed(step, reps):
        with torch.cuda.stream(stream):
            for _ in range(max(3, args.warmup)):
                step(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step(stream)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            for _ in range(3):
                g.replay()
            a.record(stream)
            for _ in range(reps):
                g.replay()
            b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / reps
        stlite.stlite_timing_read()
        stlite.stlite_timing_enable(True)
        with torch.cuda.stream(stream):
            step(stream)
        stream.synchronize()
        stlite.stlite_timing_enable(False)
        kt = stlite.stlite_timing_read()
        # per kernel: ms per step (all of the step's launches) and launches
        return ms, {k: dict(ms_per_step=t, launches=c) for k, (c, t) in kt.items()}

    def tsg_tflops(wls, layers, kernels):
        # 2 N_hist N_cur d Hkv per layer and sequence, over the TSG launches
        flop = 0.0
        for wl in wls:
            gh, gw = wl.frames[1], wl.frames[2]
            cur = int(gh[-1] * gw[-1])
            hist = int((gh[:-1] * gw[:-1]).sum())
            flop += 2.0 * hist * cur * D * wl.k.shape[1]
        flop *= layers
        t = sum(v["ms_per_step"] for k, v in kernels.items() if k.startswith("tsg")) * 1e-3
        ach = flop / t / 1e12 if t > 0 else 0.0
        return dict(bound="tensor", achieved=ach, peak=peaks["bf16"], unit="TFLOP/s", frac=ach / peaks["bf16"],
                    peak_source=peaks["source"] + " burst")

    reps = max(5, min(20, args.steps))
    runs = []
    if args.workload == "uitars":
        for beta in (0.1, 0.2, 0.3, 0.4):
            wl = synth.uitars_layer(beta=beta)
            q, k, v = bf16(wl.q), bf16(wl.k), bf16(wl.v)
            fs = stlite.FrameSpec(*wl.frames)
            prm = stlite.make_params(beta)
            sh = stlite.make_shape(q, k)
            b = stlite.stlite_budget(wl.n, beta)
            ws = torch.zeros(stlite.stlite_workspace_size(sh, fs, prm), dtype=torch.uint8, device=dev)
            ko = torch.empty((b, sh.n_kv_heads, D), dtype=torch.bfloat16, device=dev)
            vo, ix = torch.empty_like(ko), torch.empty((sh.n_kv_heads, b), dtype=torch.int32, device=dev)

            def step(st, q=q, k=k, v=v, fs=fs, prm=prm, ko=ko, vo=vo, ix=ix, ws=ws):
                stlite.stlite_compress_layer(q, k, v, fs, prm, ko, vo, ix, ws, st)
            ms, kern = timed(step, reps)
            runs.append(dict(beta=beta, layers=1, n_tokens=wl.n, budget=b, ms_per_step=ms,
                             value=wl.n / (ms * 1e-3), kernels=kern, tsg_roofline=tsg_tflops([wl], 1, kern),
                             l2="one layer's K/V (24 MB) fits in L2: replays may hit L2"))
    elif args.workload == "small_backbone":
        L, S = LAYERS, 8
        # one packed batch of 8 sequences per layer (the data does not depend
        # on beta, only the budgets do)
        layers = []
        for l in range(L):
            wls = [synth.small_backbone_seq(s, layer=l) for s in range(S)]
            cu = np.concatenate([[0], np.cumsum([wl.n for wl in wls])]).astype(np.int32)
            layers.append((wls, cu, torch.stack([bf16(wl.q) for wl in wls]), torch.cat([bf16(wl.k) for wl in wls]),
                           torch.cat([bf16(wl.v) for wl in wls])))
        for beta in (0.1, 0.4):
            prm = stlite.make_params(beta)
            per_layer = []
            for (wls, cu, q, k, v) in layers:
                tot = sum(stlite.stlite_budget(wl.n, beta) for wl in wls)
                ko = torch.empty((tot, k.shape[1], D), dtype=torch.bfloat16, device=dev)
                per_layer.append((wls, cu, q, k, v, ko, torch.empty_like(ko),
                                  torch.empty((k.shape[1] * tot,), dtype=torch.int32, device=dev)))
            wsb = max(stlite.stlite_workspace_size_varlen(stlite.make_shape(pl[2][0], pl[3]), pl[1],
                                                          [wl.frames for wl in pl[0]], prm) for pl in per_layer)
            ws = torch.zeros(wsb, dtype=torch.uint8, device=dev)

            def step(st, per_layer=per_layer, prm=prm, ws=ws):
                for (wls, cu, q, k, v, ko, vo, ix) in per_layer:
                    stlite.stlite_compress_varlen(q, k, v, cu, [wl.frames for wl in wls], prm, ko, vo, ix, ws, st)
            ms, kern = timed(step, reps)
            ntok = sum(int(pl[1][-1]) for pl in per_layer)
            runs.append(dict(beta=beta, layers=L, sequences=S, api="stlite_compress_varlen per layer",
                             n_tokens_per_layer=ntok // L, ms_per_step=ms,
                             value=ntok / (ms * 1e-3), kernels=kern,
                             tsg_roofline=tsg_tflops([wl for pl in per_layer for wl in pl[0]], 1, kern),
                             l2="inputs larger than L2 (%.2f GB K/V per step)" % (
                                 2 * sum(pl[3].numel() for pl in per_layer) * 2 / 1e9)))
            del ws
            # the same step as one stlite_compress_varlen_layers call: every
            # sequence's 28 layers in one launch per step
            frames_l = [wl.frames for wl in per_layer[0][0]]
            wsz = max(stlite.stlite_workspace_size_varlen(stlite.make_shape(pl[2][0], pl[3]), pl[1],
                                                          [wl.frames for wl in pl[0]], prm) for pl in per_layer)
            ws3 = torch.zeros(L * wsz, dtype=torch.uint8, device=dev)
            lay3 = [pl[2:] for pl in per_layer]

            def step3(st, lay3=lay3, cu=per_layer[0][1], frames_l=frames_l, prm=prm, ws3=ws3):
                stlite.stlite_compress_varlen_layers(lay3, cu, frames_l, prm, ws3, st)
            ms3, kern3 = timed(step3, reps)
            runs.append(dict(beta=beta, layers=L, sequences=S, api="stlite_compress_varlen_layers",
                             n_tokens_per_layer=ntok // L, ms_per_step=ms3, value=ntok / (ms3 * 1e-3), kernels=kern3,
                             tsg_roofline=tsg_tflops([wl for pl in per_layer for wl in pl[0]], 1, kern3)))
            del ws3
            # the same step as one stlite_compress_layers call per sequence
            # (its 28 layers share the sequence's frame layout): every stage
            # is one launch over the 28 layers
            seq_io, seq_ws = [], []
            for s_ in range(S):
                wl_s = [per_layer[l][0][s_] for l in range(L)]
                fr = wl_s[0].frames
                ios = []
                for l in range(L):
                    wls, cu, q, k, v, ko, vo, ix = per_layer[l]
                    a0, a1 = int(cu[s_]), int(cu[s_ + 1])
                    b0 = sum(stlite.stlite_budget(int(cu[i + 1] - cu[i]), beta) for i in range(s_))
                    b_s = stlite.stlite_budget(a1 - a0, beta)
                    ios.append((q[s_], k[a0:a1], v[a0:a1], ko[b0:b0 + b_s], vo[b0:b0 + b_s],
                                torch.empty((k.shape[1], b_s), dtype=torch.int32, device=dev)))
                sh_s = stlite.make_shape(ios[0][0], ios[0][1])
                seq_ws.append(torch.zeros(L * stlite.stlite_workspace_size(sh_s, stlite.FrameSpec(*fr), prm),
                                          dtype=torch.uint8, device=dev))
                seq_io.append((ios, stlite.FrameSpec(*fr)))

            def step2(st, seq_io=seq_io, seq_ws=seq_ws, prm=prm):
                for (ios, fs_s), ws_s in zip(seq_io, seq_ws):
                    stlite.stlite_compress_layers(ios, fs_s, prm, ws_s, st)
            ms2, kern2 = timed(step2, reps)
            runs.append(dict(beta=beta, layers=L, sequences=S, api="stlite_compress_layers per sequence",
                             n_tokens_per_layer=ntok // L, ms_per_step=ms2, value=ntok / (ms2 * 1e-3), kernels=kern2,
                             tsg_roofline=tsg_tflops([wl for pl in per_layer for wl in pl[0]], 1, kern2)))
            del per_layer, seq_io, seq_ws
            torch.cuda.empty_cache()
    elif args.workload == "mean_attention":
        # the prompt-wide bases of the base-scoring ablation on one layer of
        # the 50-step trajectory: every prompt position's query rows vote
        wl = synth.trajectory_50(0)
        k = bf16(wl.k)
        n_prompt = args.prompt_rows if args.prompt_rows > 0 else wl.n
        gq = torch.Generator().manual_seed(2604)
        qp = torch.randn((n_prompt, HQ, D), generator=gq).to(torch.bfloat16).to(dev)
        shp = stlite.prompt_shape(qp, k)
        ws = torch.zeros(stlite.stlite_prompt_workspace_size(shp, n_prompt), dtype=torch.uint8, device=dev)
        a = torch.empty((HKV, wl.n), dtype=torch.float32, device=dev)
        n0 = wl.n - n_prompt
        pass_flop = 2.0 * (n_prompt * n0 + n_prompt * (n_prompt + 1) / 2) * D * HQ   # causal QK^T of the rows
        for name, base in (("mean_attention", stlite.STLITE_PROMPT_MEAN), ("full_attention", stlite.STLITE_PROMPT_FULL)):
            def step(st, base=base):
                stlite.stlite_prompt_score(qp, k, base, a, ws, st)
            ms, kern = timed(step, max(3, min(10, args.steps)))
            roof = {}
            for kname in ("prompt_rowstats", "prompt_colsum"):
                if kname in kern:
                    ach = pass_flop / (kern[kname]["ms_per_step"] * 1e-3) / 1e12
                    roof[kname] = dict(bound="tensor", achieved=ach, peak=peaks["bf16"], unit="TFLOP/s",
                                       frac=ach / peaks["bf16"], peak_source=peaks["source"] + " burst")
            runs.append(dict(base=name, layers=1, n_tokens=wl.n, prompt_rows=n_prompt, ms_per_step=ms,
                             value=wl.n / (ms * 1e-3), kernels=kern, roofline=roof,
                             work="2*(causal pairs)*d*Hq = %.4g FLOP per pass" % pass_flop))
    else:  # long_horizon
        distinct = [synth.long_horizon(l) for l in range(4)]
        for L in (1, LAYERS):
            # layer l holds a copy of distinct layer l % 4 (its own buffers)
            q4, k4, v4 = [bf16(wl.q) for wl in distinct], [bf16(wl.k) for wl in distinct], [bf16(wl.v) for wl in distinct]
            qs = [q4[l % 4] for l in range(L)]
            ks = [k4[l % 4] if L == 1 else k4[l % 4].clone() for l in range(L)]
            vs = [v4[l % 4] if L == 1 else v4[l % 4].clone() for l in range(L)]
            wl0 = distinct[0]
            fs = stlite.FrameSpec(*wl0.frames)
            prm = stlite.make_params(wl0.beta)
            sh = stlite.make_shape(qs[0], ks[0])
            b = stlite.stlite_budget(wl0.n, wl0.beta)
            ws = torch.zeros(L * stlite.stlite_workspace_size(sh, fs, prm), dtype=torch.uint8, device=dev)
            io = []
            for l in range(L):
                ko = torch.empty((b, sh.n_kv_heads, D), dtype=torch.bfloat16, device=dev)
                io.append((qs[l], ks[l], vs[l], ko, torch.empty_like(ko),
                           torch.empty((sh.n_kv_heads, b), dtype=torch.int32, device=dev)))

            def step(st, io=io, fs=fs, prm=prm, ws=ws):
                stlite.stlite_compress_layers(io, fs, prm, ws, st)
            ms, kern = timed(step, reps)
            runs.append(dict(beta=wl0.beta, layers=L, n_tokens=wl0.n, budget=b, ms_per_step=ms,
                             value=wl0.n * L / (ms * 1e-3), kernels=kern, tsg_roofline=tsg_tflops([wl0], L, kern),
                             data="synthetic; 4 distinct layers, repeated" if L > 4 else "synthetic",
                             l2=("inputs larger than L2 (%.2f GB K/V per step)" % (2 * L * ks[0].numel() * 2 / 1e9))))
            del io, ws, ks, vs
            torch.cuda.empty_cache()
    line = dict(workload=args.workload, metric=METRIC, unit=UNIT, higher_is_better=True, dtype="bf16",
                data="synthetic", n_gpus=1, runs=runs)
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.workload != "traj50":
        run_workload(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
