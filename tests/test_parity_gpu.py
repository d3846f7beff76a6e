"""GPU vs oracle parity, stage by stage and end to end, through the C ABI.

Workloads: the seeded synthetic trajectories of ``synth`` at sizes the fp64
oracle finishes in seconds (several 128-token tiles, ragged tails: 36x36
frames = 10.1 row tiles and a 1296-column current frame = 2.53 chunks of
512; w*G = 448, 224 and 96 query rows), the fp32 tiny reference, and edge
cases.  Full-size configurations are checked in test_full_size_gpu.py.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_00188_gb300 import synth
from parity import (A_FLOOR, A_RTOL, CACHE, COS_ATOL, a_bound, assert_within, check_kept_sets, cos_bound,
                    exact64, gate_flip_tokens, pool_mask, to_device, visual_mask)

pytestmark = pytest.mark.gpu

WORKLOADS = {
    "tiny_ref_fp32": lambda: synth.tiny_ref(),
    "uitars_3f": lambda: synth.scaled("uitars", 3),
    "traj50_4f": lambda: synth.scaled("traj50", 4),
    "small_3f": lambda: synth.scaled("small", 3, beta=0.4),
    "long_3f": lambda: synth.scaled("long", 3, beta=0.1),
}
THREADS = 8


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


def load(name):
    def make():
        wl = WORKLOADS[name]()
        q, k, v = to_device(wl)
        q64, k64 = exact64(q), exact64(k)
        b = oracle.budget(wl.n, wl.beta)
        ref = oracle.compress_layer(q64, k64, wl.frames, beta=wl.beta, threads=THREADS)
        return wl, q64, k64, b, ref
    wl, q64, k64, b, ref = CACHE.get(name, make)
    q, k, v = to_device(wl)
    return wl, (q, k, v), q64, k64, b, ref


def s_tol(x):
    return A_RTOL * abs(x) + A_FLOOR + COS_ATOL * 2


@pytest.mark.parametrize("name", list(WORKLOADS))
def test_score(st, name):
    wl, (q, k, v), q64, k64, b, ref = load(name)
    sh = st.make_shape(q, k)
    ws = st.workspace(sh, wl.frames)
    a = torch.empty((sh.n_kv_heads, sh.n_tokens), dtype=torch.float32, device="cuda")
    st.stlite_score(q, k, a, ws)
    torch.cuda.synchronize()
    ag = a.cpu().numpy()
    for h in range(sh.n_kv_heads):
        assert_within(ag[h], ref["a"][h], a_bound(ref["a"][h]), "A_base head %d" % h)
    np.testing.assert_allclose(ag.astype(np.float64).sum(1), wl.q.shape[0], rtol=1e-4)
    assert st.stlite_device_status(ws) == st.STLITE_OK


@pytest.mark.parametrize("name", list(WORKLOADS))
def test_css(st, name):
    wl, (q, k, v), q64, k64, b, ref = load(name)
    sh = st.make_shape(q, k)
    ws = st.workspace(sh, wl.frames)
    phi = torch.empty((sh.n_kv_heads, sh.n_tokens), dtype=torch.float32, device="cuda")
    st.stlite_spatial_saliency(q, k, wl.frames, phi, ws)
    torch.cuda.synchronize()
    pg = phi.cpu().numpy()
    vis = visual_mask(wl.n, wl.frames)
    assert np.isnan(pg[:, ~vis]).all()
    assert_within(pg[:, vis], ref["phi"][:, vis], cos_bound(ref["phi"][:, vis]), "Phi")


@pytest.mark.parametrize("name", list(WORKLOADS))
def test_gate(st, name):
    wl, (q, k, v), q64, k64, b, ref = load(name)
    sh = st.make_shape(q, k)
    ws = st.workspace(sh, wl.frames)
    H, n = sh.n_kv_heads, sh.n_tokens
    rho = torch.empty((H, n), dtype=torch.float32, device="cuda")
    tau = torch.empty((H,), dtype=torch.float32, device="cuda")
    gate = torch.empty((H, n), dtype=torch.uint8, device="cuda")
    st.stlite_gate_frames(q, k, wl.frames, b, rho, tau, gate, ws)
    torch.cuda.synchronize()
    rg, tg, gg = rho.cpu().numpy(), tau.cpu().numpy(), gate.cpu().numpy()
    pool = pool_mask(n, wl.frames)
    assert np.isnan(rg[:, ~pool]).all() and (gg[:, ~pool] == 1).all()
    assert_within(rg[:, pool], ref["rho"][:, pool], cos_bound(ref["rho"][:, pool]), "rho")
    # staged: the oracle's threshold and gate on the GPU's own rho are exact
    t2, g2, _ = oracle.tsg_gate(rg.astype(np.float64), wl.frames, b)
    np.testing.assert_array_equal(t2, tg.astype(np.float64))
    np.testing.assert_array_equal(g2, gg)
    # against the oracle's own rho: flips only at the threshold
    for h in range(H):
        assert abs(tg[h] - ref["tau"][h]) <= A_RTOL * abs(ref["tau"][h]) + COS_ATOL
        gate_flip_tokens(gg[h], ref["gate"][h], ref["rho"][h], ref["tau"][h])


@pytest.mark.parametrize("name", list(WORKLOADS))
def test_select_and_compact(st, name):
    wl, (q, k, v), q64, k64, b, ref = load(name)
    sh = st.make_shape(q, k)
    prm = st.make_params(wl.beta)
    ws = st.workspace(sh, wl.frames, prm)
    H, n = sh.n_kv_heads, sh.n_tokens
    a = torch.empty((H, n), dtype=torch.float32, device="cuda")
    phi = torch.empty_like(a)
    rho = torch.empty_like(a)
    tau = torch.empty((H,), dtype=torch.float32, device="cuda")
    gate = torch.empty((H, n), dtype=torch.uint8, device="cuda")
    st.stlite_score(q, k, a, ws)
    st.stlite_spatial_saliency(q, k, wl.frames, phi, ws)
    st.stlite_gate_frames(q, k, wl.frames, b, rho, tau, gate, ws)
    idx = torch.empty((H, b), dtype=torch.int32, device="cuda")
    score = torch.empty_like(a)
    st.stlite_select_topk(q, k, wl.frames, prm, a, phi, gate, b, idx, score, ws)
    ko = torch.empty((b, H, sh.head_dim), dtype=k.dtype, device="cuda")
    vo = torch.empty_like(ko)
    st.stlite_compact(q, k, v, b, idx, ko, vo)
    torch.cuda.synchronize()
    ig, sg = idx.cpu().numpy(), score.cpu().numpy()
    # S from the GPU's own stage outputs, recomputed by the oracle
    s2 = oracle.combine(a.cpu().numpy(), phi.cpu().numpy(), gate.cpu().numpy(), wl.frames)
    assert_within(sg, s2, A_RTOL * np.abs(s2) + 2 * COS_ATOL, "S")
    # staged exactness: oracle top-B on the GPU's S equals the GPU's idx
    np.testing.assert_array_equal(oracle.topk(sg.astype(np.float64), b), ig)
    # compaction is a bit copy
    raw = torch.int16 if k.dtype == torch.bfloat16 else torch.int32
    ko2, vo2 = oracle.gather(k.view(raw).cpu().numpy(), v.view(raw).cpu().numpy(), ig)
    np.testing.assert_array_equal(ko.view(raw).cpu().numpy(), ko2)
    np.testing.assert_array_equal(vo.view(raw).cpu().numpy(), vo2)


@pytest.mark.parametrize("name", list(WORKLOADS))
def test_end_to_end(st, name):
    wl, (q, k, v), q64, k64, b, ref = load(name)
    ko, vo, idx = st.compress_layer(q, k, v, wl.frames, beta=wl.beta)
    torch.cuda.synchronize()
    ig = idx.cpu().numpy()
    H = k.shape[1]
    assert ig.shape == (H, b)
    # fused call == staged calls (same kernels, deterministic)
    sh = st.make_shape(q, k)
    prm = st.make_params(wl.beta)
    ws = st.workspace(sh, wl.frames, prm)
    a = torch.empty((H, wl.n), dtype=torch.float32, device="cuda")
    phi, rho = torch.empty_like(a), torch.empty_like(a)
    tau = torch.empty((H,), dtype=torch.float32, device="cuda")
    gate = torch.empty((H, wl.n), dtype=torch.uint8, device="cuda")
    st.stlite_score(q, k, a, ws)
    st.stlite_spatial_saliency(q, k, wl.frames, phi, ws)
    st.stlite_gate_frames(q, k, wl.frames, b, rho, tau, gate, ws)
    idx2 = torch.empty_like(idx)
    st.stlite_select_topk(q, k, wl.frames, prm, a, phi, gate, b, idx2, None, ws)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(idx2.cpu().numpy(), ig)
    # against the oracle: kept sets equal up to threshold swaps and gate flips
    gg = gate.cpu().numpy()
    for h in range(H):
        flips = gate_flip_tokens(gg[h], ref["gate"][h], ref["rho"][h], ref["tau"][h])
        check_kept_sets(ig[h], ref["idx"][h], ref["s"][h], b, s_tol, allowed_extra=flips)
    raw = torch.int16 if k.dtype == torch.bfloat16 else torch.int32
    ko2, vo2 = oracle.gather(k.view(raw).cpu().numpy(), v.view(raw).cpu().numpy(), ig)
    np.testing.assert_array_equal(ko.view(raw).cpu().numpy(), ko2)
    np.testing.assert_array_equal(vo.view(raw).cpu().numpy(), vo2)


# ------------------------------------------------------------------ edge cases

def _run_edge(st, wl, beta, k_override=0, tsg=1, css=1, alpha=1.0, **variant):
    """variant: tsg_metric / fixed_tau / base_scorer, the same names for the
    library and the oracle."""
    q, k, v = to_device(wl)
    q64, k64 = exact64(q), exact64(k)
    ko, vo, idx = st.compress_layer(q, k, v, wl.frames, beta=beta, k_override=k_override, tsg_enable=tsg,
                                    css_enable=css, alpha=alpha, **variant)
    torch.cuda.synchronize()
    ref = oracle.compress_layer(q64, k64, wl.frames, beta=beta, k_override=k_override, tsg_enable=tsg,
                                css_enable=css, alpha=alpha, threads=THREADS, **variant)
    ig = idx.cpu().numpy()
    b = ref["budget"]
    assert ig.shape[1] == b
    for h in range(k.shape[1]):
        flips = set()
        if tsg and len(wl.frames[0]) >= 2:
            flips = set(np.nonzero(np.abs(ref["rho"][h] - ref["tau"][h]) <= 1e-3 * abs(ref["tau"][h]) + COS_ATOL)[0].tolist())
        check_kept_sets(ig[h], ref["idx"][h], ref["s"][h], b, s_tol, allowed_extra=flips)
    raw = torch.int16 if k.dtype == torch.bfloat16 else torch.int32
    ko2, _ = oracle.gather(k.view(raw).cpu().numpy(), v.view(raw).cpu().numpy(), ig)
    np.testing.assert_array_equal(ko.view(raw).cpu().numpy(), ko2)
    return ig, ref


def test_edge_single_frame(st):
    wl = synth.trajectory(n_steps=1, gh=20, gw=30, n_text=17, seed=(700,))
    _run_edge(st, wl, 0.2)


def test_edge_no_frames_text_only(st):
    wl = synth.trajectory(n_steps=1, gh=2, gw=2, n_text=301, seed=(701,))
    wl.offset, wl.grid_h, wl.grid_w = (np.zeros(0, np.int32),) * 3
    ig, ref = _run_edge(st, wl, 0.3)
    # text only: S = A_base, so top-B of the window score
    for h in range(ig.shape[0]):
        np.testing.assert_array_equal(ig[h], ref["idx"][h])


def test_edge_beta_one_and_override(st):
    wl = synth.scaled("traj50", 2)
    ig, _ = _run_edge(st, wl, 1.0)
    assert (ig == np.arange(wl.n)[None, :]).all()
    _run_edge(st, wl, 0.2, k_override=wl.n - 3)
    _run_edge(st, wl, 0.2, k_override=1)


def test_edge_flags(st):
    wl = synth.scaled("small", 2)
    _run_edge(st, wl, 0.25, tsg=0)
    _run_edge(st, wl, 0.25, css=0)
    _run_edge(st, wl, 0.25, tsg=0, css=0)
    _run_edge(st, wl, 0.25, alpha=0.5)


def test_edge_ragged_small(st):
    # N not a multiple of anything, 1x1 and 1xW grids, frames separated by text
    rng = np.random.default_rng(5)
    n, hq, hkv, w = 997, 12, 2, 7
    q = rng.standard_normal((w, hq, 128), dtype=np.float32)
    k = rng.standard_normal((n, hkv, 128), dtype=np.float32)
    k[400:500] = k[600:700] + 0.01 * rng.standard_normal((100, hkv, 128), dtype=np.float32)
    v = rng.standard_normal((n, hkv, 128), dtype=np.float32)
    wl = synth.Workload("ragged", q, k, v, np.array([3, 10, 41, 400, 600], np.int32),
                        np.array([1, 1, 7, 10, 10], np.int32), np.array([1, 13, 9, 10, 10], np.int32), beta=0.15)
    _run_edge(st, wl, 0.15)
    wl.dtype = "f32"
    _run_edge(st, wl, 0.15)


def test_edge_exact_duplicate_ties(st):
    # exact duplicate frames: equal rho at the threshold and equal S (ties by index)
    wl = synth.scaled("long", 4, beta=0.1)
    _run_edge(st, wl, 0.1)


def test_repeat_deterministic(st):
    wl = synth.scaled("uitars", 2)
    q, k, v = to_device(wl)
    outs = [st.compress_layer(q, k, v, wl.frames, beta=0.2) for _ in range(3)]
    torch.cuda.synchronize()
    for o in outs[1:]:
        for x, y in zip(o, outs[0]):
            assert torch.equal(x, y)


# ------------------------------------------------------------ batched layers

def _batched_vs_single(st, wls):
    dev = [to_device(wl) for wl in wls]
    wl0 = wls[0]
    sh = st.make_shape(dev[0][0], dev[0][1])
    prm = st.make_params(wl0.beta)
    b = st.stlite_budget(wl0.n, wl0.beta)
    H = sh.n_kv_heads
    single = [st.compress_layer(q, k, v, wl0.frames, beta=wl0.beta) for (q, k, v) in dev]
    outs = []
    for (q, k, v) in dev:
        ko = torch.empty((b, H, 128), dtype=k.dtype, device="cuda")
        outs.append((q, k, v, ko, torch.empty_like(ko), torch.empty((H, b), dtype=torch.int32, device="cuda")))
    ws = torch.zeros(len(wls) * st.stlite_workspace_size(sh, wl0.frames, prm), dtype=torch.uint8, device="cuda")
    assert st.stlite_compress_layers(outs, wl0.frames, prm, ws) == b
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    for (ko1, vo1, i1), (_, _, _, ko2, vo2, i2) in zip(single, outs):
        assert torch.equal(i1, i2)
        assert torch.equal(ko1, ko2) and torch.equal(vo1, vo2)


def test_compress_layers_equals_single_bf16(st):
    _batched_vs_single(st, [synth.scaled("traj50", 3, seed=s) for s in range(3)])


def test_compress_layers_equals_single_fp32(st):
    _batched_vs_single(st, [synth.tiny_ref(seed=s) for s in range(2)])


def test_compress_layers_more_than_one_launch(st):
    # 34 layers: two launches of up to 32 layers each
    wls = [synth.trajectory(n_steps=3, gh=5, gw=7, n_text=4, hq=8, hkv=2, w=4, beta=0.3, seed=(800, s))
           for s in range(34)]
    _batched_vs_single(st, wls)


# ------------------------------------------- per-layer (hierarchical) budgets

def _budgets_vs_single(st, wls, budgets, oracle_layers=()):
    """stlite_compress_layers_budgets: layer l equals a single-layer call with
    k_override = budgets[l] (bit-exact), and the layers in oracle_layers
    match the oracle's kept sets."""
    dev = [to_device(wl) for wl in wls]
    wl0 = wls[0]
    sh = st.make_shape(dev[0][0], dev[0][1])
    prm = st.make_params(wl0.beta)
    H = sh.n_kv_heads
    outs = []
    for (q, k, v), b in zip(dev, budgets):
        ko = torch.empty((b, H, 128), dtype=k.dtype, device="cuda")
        outs.append((q, k, v, ko, torch.empty_like(ko), torch.empty((H, b), dtype=torch.int32, device="cuda")))
    ws = torch.zeros(len(wls) * st.stlite_workspace_size(sh, wl0.frames, prm), dtype=torch.uint8, device="cuda")
    st.stlite_compress_layers_budgets(outs, wl0.frames, prm, budgets, ws)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    for l, ((q, k, v), b, (_, _, _, ko2, vo2, i2)) in enumerate(zip(dev, budgets, outs)):
        ko1, vo1, i1 = st.compress_layer(q, k, v, wl0.frames, beta=wl0.beta, k_override=b)
        torch.cuda.synchronize()
        assert torch.equal(i1, i2), l
        assert torch.equal(ko1, ko2) and torch.equal(vo1, vo2), l
    for l in oracle_layers:
        ig, ref = _run_edge(st, wls[l], wl0.beta, k_override=budgets[l])
        np.testing.assert_array_equal(ig, outs[l][5].cpu().numpy())


def test_hierarchical_budgets_from_window_mass(st):
    # S^(l) = the window score's mass on the prefix keys (all heads), the
    # budgets B^(l) = S^(l) / sum S * B_total with B_total = L * floor(beta N)
    wls = [synth.scaled("traj50", 3, seed=s) for s in range(4)]
    n, w = wls[0].n, wls[0].q.shape[0]
    mass = []
    for wl in wls:
        q, k, _ = to_device(wl)
        mass.append(float(oracle.abase(exact64(q), exact64(k), threads=THREADS)[:, :n - w].sum()))
    total = len(wls) * oracle.budget(n, wls[0].beta)
    budgets = st.stlite_hierarchical_budgets(mass, total, n)
    assert budgets == oracle.hierarchical_budgets(mass, total, n)
    assert sum(budgets) == total
    _budgets_vs_single(st, wls, budgets, oracle_layers=(0, len(wls) - 1))


def test_per_layer_budgets_extremes_two_launches(st):
    # 34 layers (two launches), budgets from 1 to N in a pyramid
    wls = [synth.trajectory(n_steps=3, gh=5, gw=7, n_text=4, hq=8, hkv=2, w=4, beta=0.3, seed=(810, s))
           for s in range(34)]
    n = wls[0].n
    budgets = [max(1, min(n, int(round(n * (1.0 - l / 33.0))))) for l in range(34)]
    budgets[5], budgets[20] = 1, n
    _budgets_vs_single(st, wls, budgets, oracle_layers=(0, 5, 20, 33))


# ------------------------------------------------- values in page-locked host memory

def test_host_resident_values(st):
    """v may live in page-locked host memory (only the kept rows are read):
    the outputs equal those of a device-resident v, for the single-layer and
    the batched entry, bf16 and fp32."""
    for wls in ([synth.scaled("traj50", 3, seed=s) for s in range(2)], [synth.tiny_ref(seed=5)]):
        wl0 = wls[0]
        dev = [to_device(wl) for wl in wls]
        ref = [st.compress_layer(q, k, v, wl0.frames, beta=wl0.beta) for (q, k, v) in dev]
        hv = [v.cpu().pin_memory() for (_, _, v) in dev]
        torch.cuda.synchronize()
        one = [st.compress_layer(q, k, v_h, wl0.frames, beta=wl0.beta) for (q, k, _), v_h in zip(dev, hv)]
        sh = st.make_shape(dev[0][0], dev[0][1])
        prm = st.make_params(wl0.beta)
        b = st.stlite_budget(wl0.n, wl0.beta)
        H = sh.n_kv_heads
        outs = []
        for (q, k, _), v_h in zip(dev, hv):
            ko = torch.empty((b, H, sh.head_dim), dtype=k.dtype, device="cuda")
            outs.append((q, k, v_h, ko, torch.empty_like(ko), torch.empty((H, b), dtype=torch.int32, device="cuda")))
        ws = torch.zeros(len(wls) * st.stlite_workspace_size(sh, wl0.frames, prm), dtype=torch.uint8,
                         device="cuda")
        assert st.stlite_compress_layers(outs, wl0.frames, prm, ws) == b
        torch.cuda.synchronize()
        assert st.stlite_device_status(ws) == st.STLITE_OK
        for (k1, v1, i1), (k2, v2, i2), (_, _, _, k3, v3, i3) in zip(ref, one, outs):
            assert torch.equal(i1, i2) and torch.equal(i1, i3)
            assert torch.equal(k1, k2) and torch.equal(k1, k3)
            assert torch.equal(v1, v2) and torch.equal(v1, v3)


# ------------------------------------------------------- packed batch of sequences

def _varlen_vs_single(st, wls):
    dev = [to_device(wl) for wl in wls]
    cu = np.concatenate([[0], np.cumsum([wl.n for wl in wls])]).astype(np.int32)
    q = torch.stack([d[0] for d in dev])
    k = torch.cat([d[1] for d in dev])
    v = torch.cat([d[2] for d in dev])
    beta = wls[0].beta
    prm = st.make_params(beta)
    budgets = [st.stlite_budget(wl.n, beta) for wl in wls]
    H, D = k.shape[1], k.shape[2]
    tot = sum(budgets)
    ko = torch.empty((tot, H, D), dtype=k.dtype, device="cuda")
    vo = torch.empty_like(ko)
    ix = torch.empty((H * tot,), dtype=torch.int32, device="cuda")
    sh = st.make_shape(dev[0][0], k)
    ws = torch.zeros(st.stlite_workspace_size_varlen(sh, cu, [wl.frames for wl in wls], prm), dtype=torch.uint8,
                     device="cuda")
    cb = st.stlite_compress_varlen(q, k, v, cu, [wl.frames for wl in wls], prm, ko, vo, ix, ws)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    assert list(cb) == list(np.concatenate([[0], np.cumsum(budgets)]))
    for s, (wl, (qs, ks, vs)) in enumerate(zip(wls, dev)):
        k1, v1, i1 = st.compress_layer(qs, ks, vs, wl.frames, beta=beta)
        b0, b1 = cb[s], cb[s + 1]
        assert torch.equal(ix[H * b0:H * b1].view(H, b1 - b0), i1)
        assert torch.equal(ko[b0:b1], k1) and torch.equal(vo[b0:b1], v1)
    return cb


def test_varlen_small_backbone_batch(st):
    # the batch-8 smaller-backbone configuration: 12-20 frames of 24x42 per sequence
    _varlen_vs_single(st, [synth.small_backbone_seq(s, beta=0.1) for s in range(8)])


def test_varlen_ragged_fp32_and_oracle(st):
    # three sequences of different frame layouts (fp32), one of them a single frame;
    # the packed call equals per-sequence calls, and those match the oracle
    wls = [synth.trajectory(n_steps=3, gh=5, gw=7, n_text=4, hq=8, hkv=2, w=4, beta=0.3, seed=(900, 0),
                            dtype="f32"),
           synth.trajectory(n_steps=1, gh=6, gw=3, n_text=9, hq=8, hkv=2, w=4, beta=0.3, seed=(900, 1),
                            dtype="f32"),
           synth.trajectory(n_steps=4, gh=3, gw=9, n_text=2, hq=8, hkv=2, w=4, beta=0.3, seed=(900, 2),
                            dtype="f32")]
    _varlen_vs_single(st, wls)
    for wl in wls:
        _run_edge(st, wl, wl.beta)


def test_text_permutation_equivariance(st):
    # Reordering the text tokens reorders the GPU's kept set the same way
    # (up to swaps at the B-th score, where fp32 sums in a different key order
    # may round differently).
    wl = synth.scaled("traj50", 3)
    q, k, v = to_device(wl)
    off, gh, gw = wl.frames
    vis = visual_mask(wl.n, wl.frames)
    text = np.nonzero(~vis)[0]
    perm = np.arange(wl.n)
    perm[text] = text[::-1]
    pt = torch.from_numpy(perm).cuda()
    _, _, ia = st.compress_layer(q, k, v, wl.frames, beta=wl.beta)
    _, _, ib = st.compress_layer(q, k[pt].contiguous(), v[pt].contiguous(), wl.frames, beta=wl.beta)
    torch.cuda.synchronize()
    ref = oracle.compress_layer(exact64(q), exact64(k), wl.frames, beta=wl.beta, threads=THREADS)
    ia, ib = ia.cpu().numpy(), ib.cpu().numpy()
    b = ref["budget"]
    for h in range(k.shape[1]):
        flips = set(np.nonzero(np.abs(ref["rho"][h] - ref["tau"][h]) <= 1e-3 * abs(ref["tau"][h]) + COS_ATOL)[0].tolist())
        check_kept_sets(np.sort(perm[ib[h]]), ia[h], ref["s"][h], b, s_tol, allowed_extra=flips)


# ------------------------------------------------------------ critical hit rate

def test_critical_hit_rate(st):
    import bench
    # consistency: alpha = 0, TSG off, the probe as the only window row -> the
    # kept set is exactly the probe's Top_B, so the GPU's rate is 1
    wl = synth.trajectory(n_steps=3, gh=8, gw=9, n_text=5, hq=8, hkv=2, w=1, beta=0.25, seed=(950,))
    q, k, v = to_device(wl)
    _, _, idx = st.compress_layer(q, k, v, wl.frames, beta=wl.beta, tsg_enable=0, css_enable=0, alpha=0.0)
    assert torch.equal(bench.gpu_critical_hit_rate(st, q, k, idx), torch.ones(2, dtype=torch.float64, device="cuda"))
    # the full method on a 4-frame trajectory: the GPU's rate against the
    # oracle's (both kept sets and both top sets may differ by swaps at their
    # thresholds; each swap moves the rate by at most 1/B)
    wl = synth.scaled("traj50", 4)
    q, k, v = to_device(wl)
    _, _, idx = st.compress_layer(q, k, v, wl.frames, beta=wl.beta)
    probe = q[-1:].contiguous()
    got = bench.gpu_critical_hit_rate(st, probe, k, idx).cpu().numpy()
    ref_keep = oracle.compress_layer(exact64(q), exact64(k), wl.frames, beta=wl.beta, threads=THREADS)["idx"]
    ref = oracle.critical_hit_rate(ref_keep, exact64(probe), exact64(k))
    assert np.all(np.abs(got - ref) <= 4.0 / idx.shape[1]), (got, ref)


# ----------------------------------------------------- the paper's ablation variants

@pytest.mark.parametrize("name", ["uitars_3f", "tiny_ref_fp32"])
@pytest.mark.parametrize("metric", [1, 2])
def test_variant_tsg_metric(st, name, metric):
    # TSG similarity: dot product (1) and negative squared L2 distance (2)
    wl = WORKLOADS[name]()
    _run_edge(st, wl, wl.beta, tsg_metric=metric)


@pytest.mark.parametrize("name", ["traj50_4f", "tiny_ref_fp32"])
def test_variant_fixed_threshold(st, name):
    # fixed-threshold control: gate every pool token with cosine above 0.85
    wl = WORKLOADS[name]()
    ig, ref = _run_edge(st, wl, wl.beta, fixed_tau=0.85)
    assert (ref["tau"] == 0.85).all()


@pytest.mark.parametrize("name", ["small_3f", "tiny_ref_fp32"])
def test_variant_uniform_base(st, name):
    # uniform base prior: A = w/N for every token (the score passes are skipped)
    wl = WORKLOADS[name]()
    _run_edge(st, wl, wl.beta, base_scorer=1)


@pytest.mark.parametrize("size", [3, 5, 7, 9])
@pytest.mark.parametrize("name", ["uitars_3f", "traj50_4f", "tiny_ref_fp32"])
def test_css_size_phi(st, name, size):
    # CSS over the size x size neighbourhood (box-sum kernel), element by
    # element against the oracle; uitars has 64-column grids
    wl = WORKLOADS[name]()
    q, k, v = to_device(wl)
    sh = st.make_shape(q, k)
    ws = st.workspace(sh, wl.frames)
    phi = torch.empty((sh.n_kv_heads, sh.n_tokens), dtype=torch.float32, device="cuda")
    st.stlite_spatial_saliency_size(q, k, wl.frames, size, phi, ws)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    ref = oracle.css_phi(exact64(k), wl.frames, threads=THREADS, size=size)
    pg = phi.cpu().numpy()
    vis = visual_mask(wl.n, wl.frames)
    assert np.isnan(pg[:, ~vis]).all()
    assert_within(pg[:, vis], ref[:, vis], cos_bound(ref[:, vis]), "Phi")


def test_css_size_ragged_grids(st):
    # 1x1, 1xW, Hx1 and odd grids separated by text, fp32 and bf16
    rng = np.random.default_rng(44)
    n, hq, hkv, w = 700, 8, 2, 5
    q = rng.standard_normal((w, hq, 128), dtype=np.float32)
    k = rng.standard_normal((n, hkv, 128), dtype=np.float32)
    k[300:340] = k[200:240] + 0.05 * rng.standard_normal((40, hkv, 128), dtype=np.float32)
    v = rng.standard_normal((n, hkv, 128), dtype=np.float32)
    frames = (np.array([2, 5, 40, 200, 300, 400], np.int32), np.array([1, 1, 23, 5, 5, 17], np.int32),
              np.array([1, 30, 1, 8, 8, 17], np.int32))
    wl = synth.Workload("ragged_css", q, k, v, *frames, beta=0.2)
    for dtype in ("bf16", "f32"):
        wl.dtype = dtype
        qd, kd, _ = to_device(wl)
        ws = st.workspace(st.make_shape(qd, kd), wl.frames)
        for size in (3, 5, 9):
            phi = torch.empty((hkv, n), dtype=torch.float32, device="cuda")
            st.stlite_spatial_saliency_size(qd, kd, wl.frames, size, phi, ws)
            torch.cuda.synchronize()
            ref = oracle.css_phi(exact64(kd), wl.frames, size=size)
            vis = visual_mask(n, wl.frames)
            assert_within(phi.cpu().numpy()[:, vis], ref[:, vis], cos_bound(ref[:, vis]), "Phi")


@pytest.mark.parametrize("size", [5, 9])
@pytest.mark.parametrize("name", ["traj50_4f", "tiny_ref_fp32"])
def test_variant_css_size(st, name, size):
    # the neighbourhood-size ablation end to end
    wl = WORKLOADS[name]()
    _run_edge(st, wl, wl.beta, css_size=size)


@pytest.mark.parametrize("name", ["traj50_4f", "small_3f", "tiny_ref_fp32"])
def test_variant_abase_max(st, name):
    # A_base divided by its per-head maximum before Eq. 9
    wl = WORKLOADS[name]()
    _run_edge(st, wl, wl.beta, abase_norm=1)
    _run_edge(st, wl, wl.beta, abase_norm=1, base_scorer=1)


# ----------------------------------------------------------- kernel boundaries

def test_edge_grid_width_limits(st):
    # 127 columns: the widest grid of the tensor-core CSS band (256 key rows);
    # 128 columns: the CUDA-core CSS; both against the oracle, bf16 and fp32
    for gw, seed in ((127, 960), (128, 961), (200, 962)):
        wl = synth.trajectory(n_steps=3, gh=3, gw=gw, n_text=5, hq=8, hkv=2, w=4, beta=0.2, seed=(seed,))
        _run_edge(st, wl, 0.2)
        wl.dtype = "f32"
        _run_edge(st, wl, 0.2)


def test_edge_query_rows_512(st):
    # R = w G = 512 query rows per KV head, the largest the score passes take
    wl = synth.trajectory(n_steps=3, gh=6, gw=7, n_text=9, hq=8, hkv=1, w=64, beta=0.25, seed=(963,))
    _run_edge(st, wl, 0.25)


def test_edge_query_rows_ragged_second_half(st):
    # R = 33 x 9 = 297: pass 1 runs two CTAs per key split, the second with
    # 41 valid rows in its first M-tile and none in its second; pass 2 runs
    # two column halves of 160 whose last epilogue group has no columns
    wl = synth.trajectory(n_steps=3, gh=5, gw=6, n_text=7, hq=9, hkv=1, w=33, beta=0.25, seed=(967,))
    _run_edge(st, wl, 0.25)
    # R = 129 x 2 = 258: two rows past the one-CTA limit
    wl = synth.trajectory(n_steps=2, gh=4, gw=5, n_text=3, hq=2, hkv=1, w=129, beta=0.3, seed=(968,))
    _run_edge(st, wl, 0.3)


def test_edge_one_query_head_per_group(st):
    # G = 1: every query head has its own KV head
    wl = synth.trajectory(n_steps=3, gh=5, gw=9, n_text=3, hq=4, hkv=4, w=16, beta=0.3, seed=(964,))
    _run_edge(st, wl, 0.3)


def test_edge_tiny_caches(st):
    # one cached token (text only) and a one-token budget
    rng = np.random.default_rng(965)
    for n in (1, 2, 3):
        q = rng.standard_normal((2, 4, 128), dtype=np.float32)
        k = rng.standard_normal((n, 2, 128), dtype=np.float32)
        v = rng.standard_normal((n, 2, 128), dtype=np.float32)
        wl = synth.Workload("tiny%d" % n, q, k, v, np.zeros(0, np.int32), np.zeros(0, np.int32),
                            np.zeros(0, np.int32), beta=0.5)
        ig, ref = _run_edge(st, wl, 0.5)
        assert ig.shape[1] == max(1, n // 2)
    wl = synth.trajectory(n_steps=2, gh=2, gw=3, n_text=2, hq=4, hkv=2, w=2, beta=0.2, seed=(966,))
    _run_edge(st, wl, 0.2, k_override=1)


@pytest.mark.parametrize("beta", [0.1, 0.4])
def test_varlen_layers_equals_per_layer(st, beta):
    # a packed batch over several layers in one call equals one packed call
    # per layer, bit for bit (4 sequences of the batch-8 shape, 3 layers;
    # at beta = 10 % some sequences' index blocks start on odd offsets)
    S, L = 4, 3
    layers = []
    for l in range(L):
        wls = [synth.small_backbone_seq(s, layer=l, beta=beta) for s in range(S)]
        dev = [to_device(wl) for wl in wls]
        layers.append((wls, dev))
    wls0 = layers[0][0]
    cu = np.concatenate([[0], np.cumsum([wl.n for wl in wls0])]).astype(np.int32)
    frames = [wl.frames for wl in wls0]
    prm = st.make_params(beta)
    tot = sum(st.stlite_budget(wl.n, beta) for wl in wls0)
    packed, single = [], []
    for wls, dev in layers:
        q = torch.stack([d[0] for d in dev])
        k = torch.cat([d[1] for d in dev])
        v = torch.cat([d[2] for d in dev])
        H = k.shape[1]
        mk = lambda: (torch.empty((tot, H, 128), dtype=k.dtype, device="cuda"),
                      torch.empty((tot, H, 128), dtype=k.dtype, device="cuda"),
                      torch.empty((H * tot,), dtype=torch.int32, device="cuda"))
        packed.append((q, k, v) + mk())
        single.append((q, k, v) + mk())
    if beta == 0.1:
        assert any(st.stlite_budget(wl.n, beta) % 2 for wl in wls0)
    sh = st.make_shape(packed[0][0][0], packed[0][1])
    wsz = st.stlite_workspace_size_varlen(sh, cu, frames, prm)
    ws = torch.zeros(L * wsz, dtype=torch.uint8, device="cuda")
    cb = st.stlite_compress_varlen_layers(packed, cu, frames, prm, ws)
    ws1 = torch.zeros(wsz, dtype=torch.uint8, device="cuda")
    for (q, k, v, ko, vo, ix) in single:
        cb1 = st.stlite_compress_varlen(q, k, v, cu, frames, prm, ko, vo, ix, ws1)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    assert list(cb) == list(cb1)
    for a, b in zip(packed, single):
        for x, y in zip(a[3:], b[3:]):
            assert torch.equal(x, y)
