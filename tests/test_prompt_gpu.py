"""Prompt-wide base scores (the base-scoring ablation's Mean Attention and
full-attention bases) through the C ABI against the fp64 oracle: every
element of A within the window score's tolerance, for prompts covering the
whole cache and its last n_prompt positions (ragged m-tiles and chunks),
group sizes 7, 6 and 1, Gaussian and heavy-tailed keys, bf16 caches (tensor
cores) and fp32 caches (CUDA cores); the row-mass
invariant; bit-identical repeated calls; and the kept set of the method run
on this base (Eq. 9 with A replaced, then Top-B) against the oracle's.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_00188_gb300 import synth
from parity import (A_FLOOR, A_RTOL, CACHE, COS_ATOL, a_bound, assert_within, check_kept_sets, exact64, to_device)

pytestmark = pytest.mark.gpu

CASES = {
    # name: (workload, n_prompt or None for the whole cache)
    "traj50_4f_all": (lambda: synth.scaled("traj50", 4), None),
    "traj50_4f_last1000": (lambda: synth.scaled("traj50", 4), 1000),
    "small_3f_all": (lambda: synth.scaled("small", 3, beta=0.4), None),
    "long_2f_last777": (lambda: synth.scaled("long", 2, beta=0.1), 777),
    "g1_ragged": (lambda: synth.trajectory(n_steps=3, gh=7, gw=9, n_text=5, hq=2, hkv=2, w=4, beta=0.3,
                                           seed=(77,)), None),
    "last_7": (lambda: synth.scaled("small", 2, beta=0.4), 7),
    "last_1": (lambda: synth.scaled("traj50", 2), 1),
    # fp32 caches (CUDA-core passes): the tiny reference, whole and partial prompts
    "fp32_tiny_all": (lambda: synth.tiny_ref(), None),
    "fp32_tiny_last333": (lambda: synth.tiny_ref(), 333),
}


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


def prompt_rows(wl, q_all, n_prompt):
    """The prompt's query rows: the window queries stand in for the last w
    positions, and earlier positions take query rows drawn like them."""
    n = wl.n
    npr = n if n_prompt is None else n_prompt
    rng = np.random.default_rng(4242 + n + npr)
    qp = rng.standard_normal((npr, q_all.shape[1], q_all.shape[2])).astype(np.float32)
    w = min(npr, q_all.shape[0])
    qp[npr - w:] = q_all[q_all.shape[0] - w:]
    dt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    return torch.from_numpy(qp).to(dt).cuda()


def load(name):
    make, n_prompt = CASES[name]

    def run():
        wl = make()
        q, k, v = to_device(wl)
        qp = prompt_rows(wl, wl.q, n_prompt)
        t = oracle.host_threads()
        full = oracle.prompt_abase(exact64(qp), exact64(k), oracle.PROMPT_FULL, threads=t)
        mean = oracle.prompt_abase(exact64(qp), exact64(k), oracle.PROMPT_MEAN, threads=t)
        return wl, qp.cpu(), full, mean
    wl, qp, full, mean = CACHE.get("prompt_" + name, run)
    q, k, v = to_device(wl)
    return wl, qp.cuda(), k, v, full, mean


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("base", ["full", "mean"])
def test_prompt_score(st, name, base):
    wl, qp, k, v, full, mean = load(name)
    mode = st.STLITE_PROMPT_FULL if base == "full" else st.STLITE_PROMPT_MEAN
    ora = full if base == "full" else mean
    a, ws = st.prompt_score(qp, k, mode)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    ag = a.cpu().numpy()
    for h in range(k.shape[1]):
        assert_within(ag[h], ora[h], a_bound(ora[h]), "%s base head %d" % (base, h))
    if base == "full":
        # every prompt row's probabilities sum to one
        np.testing.assert_allclose(ag.astype(np.float64).sum(1), qp.shape[0], rtol=1e-4)
    # a second call gives the same bits
    a2, _ = st.prompt_score(qp, k, mode)
    torch.cuda.synchronize()
    assert torch.equal(a, a2)


@pytest.mark.parametrize("name", ["traj50_4f_all", "small_3f_all", "long_2f_last777", "fp32_tiny_all"])
def test_method_on_prompt_base(st, name):
    """Eq. 9 and Top-B with the Mean Attention base in place of the window
    score (CSS and TSG unchanged): kept sets against the oracle's pipeline."""
    wl, qp, k, v, full, mean = load(name)
    a, _ = st.prompt_score(qp, k, st.STLITE_PROMPT_MEAN)
    q = torch.from_numpy(wl.q).to(k.dtype).cuda()
    sh = st.make_shape(q, k)
    prm = st.make_params(wl.beta)
    ws = st.workspace(sh, wl.frames, prm)
    H, n = k.shape[1], wl.n
    b = oracle.budget(n, wl.beta)
    phi, rho = torch.empty_like(a), torch.empty_like(a)
    tau = torch.empty((H,), dtype=torch.float32, device="cuda")
    gate = torch.empty((H, n), dtype=torch.uint8, device="cuda")
    st.stlite_spatial_saliency(q, k, wl.frames, phi, ws)
    st.stlite_gate_frames(q, k, wl.frames, b, rho, tau, gate, ws)
    idx = torch.empty((H, b), dtype=torch.int32, device="cuda")
    st.stlite_select_topk(q, k, wl.frames, prm, a, phi, gate, b, idx, None, ws)
    torch.cuda.synchronize()
    k64 = exact64(k)
    phi_o = oracle.css_phi(k64, wl.frames)
    rho_o = oracle.tsg_rho(k64, wl.frames, threads=oracle.host_threads())
    tau_o, gate_o, _ = oracle.tsg_gate(rho_o, wl.frames, b)
    s_o = oracle.combine(mean, phi_o, gate_o, wl.frames)
    idx_o = oracle.topk(s_o, b)
    ig = idx.cpu().numpy()

    def s_tol(x):
        return A_RTOL * abs(x) + A_FLOOR + COS_ATOL * 2
    for h in range(H):
        flips = set(np.nonzero(np.abs(rho_o[h] - tau_o[h]) <= A_RTOL * abs(tau_o[h]) + COS_ATOL)[0].tolist())
        check_kept_sets(ig[h], idx_o[h], s_o[h], b, s_tol, allowed_extra=flips)


def test_prompt_rejects(st):
    """Groups of more than 128 query heads and prompts longer than the cache
    are refused on the host."""
    kb = torch.zeros((64, 1, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(st.StliteError) as e:
        st.prompt_score(torch.zeros((64, 256, 128), dtype=torch.bfloat16, device="cuda"), kb)
    assert e.value.status == st.STLITE_EUNSUPPORTED
    with pytest.raises(st.StliteError) as e:
        st.prompt_score(torch.zeros((65, 4, 128), dtype=torch.bfloat16, device="cuda"), kb)
    assert e.value.status == st.STLITE_EINVAL


def test_prompt_full_size_bench_layer(st):
    """The bench's full-size case: layer 0 of the 50-step trajectory (N =
    53,600) with the whole prompt voting.  The oracle cannot redo 10 TFLOP,
    so: every row's mass is one (sum_j C_j = N per head); the Mean Attention
    base times the rows that see a key equals the full base; and the last 64
    keys, which only the last 64 prompt rows can see, equal the oracle's
    scores of those 64 rows exactly as defined (same rows, same keys)."""
    wl = synth.trajectory_50(0)
    k = torch.from_numpy(wl.k).to(torch.bfloat16).cuda()
    qp = prompt_rows(wl, wl.q, None)
    n, H = wl.n, k.shape[1]
    full, _ = st.prompt_score(qp, k, st.STLITE_PROMPT_FULL)
    mean, ws = st.prompt_score(qp, k, st.STLITE_PROMPT_MEAN)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    f, m = full.cpu().numpy().astype(np.float64), mean.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(f.sum(1), n, rtol=1e-4)
    count = np.minimum(n, n - np.arange(n)).astype(np.float64)
    np.testing.assert_allclose(m * count, f, rtol=2e-6, atol=0)
    tail = 64
    ora = oracle.prompt_abase(exact64(qp[n - tail:]), exact64(k), oracle.PROMPT_FULL, threads=oracle.host_threads())
    for h in range(H):
        assert_within(f[h, n - tail:], ora[h, n - tail:], a_bound(ora[h, n - tail:]), "full base, last keys, head %d" % h)
