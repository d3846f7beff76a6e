"""Full-size configurations through the C ABI, checked where the fp64 oracle
can follow: sampled per-token values (Phi, rho), the window-score invariant
sum_j A = w (and the full oracle A where it finishes in seconds), and exact
staged parity of everything downstream of the scores (tau/gate on the GPU's
rho, Eq. 9 and Top-B on the GPU's stage outputs, compaction byte copies).
The fused call is the one bench.py times.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_00188_gb300 import synth
from parity import (A_RTOL, COS_ATOL, a_bound, assert_within, cos_bound, exact64, pool_mask, to_device,
                    visual_mask)

pytestmark = pytest.mark.gpu

CONFIGS = {
    "uitars_b10": (lambda: synth.uitars_layer(beta=0.1), True),
    "uitars_b20": (lambda: synth.uitars_layer(beta=0.2), True),
    "uitars_b30": (lambda: synth.uitars_layer(beta=0.3), False),
    "uitars_b40": (lambda: synth.uitars_layer(beta=0.4), False),
    "traj50_l0": (lambda: synth.trajectory_50(0), True),
    "traj50_l27": (lambda: synth.trajectory_50(27), False),
    "small_s0_b10": (lambda: synth.small_backbone_seq(0, beta=0.1), True),
    "small_s5_b40": (lambda: synth.small_backbone_seq(5, beta=0.4), True),
    "long_l0": (lambda: synth.long_horizon(0), False),
    # the frame-table limit: 256 frames (2x3 grids, one text token after each)
    "max_frames_256": (lambda: synth.trajectory(n_steps=256, gh=2, gw=3, n_text=1, hq=4, hkv=2, w=4, beta=0.3,
                                                n_boxes=(1, 2), box_hw=((1, 1), (2, 2)), seed=(990,)), True),
    # the largest cache the selection holds on chip: 393,216 tokens
    # (256 frames of 32x48, one KV head)
    "max_tokens_393216": (lambda: synth.trajectory(n_steps=256, gh=32, gw=48, n_text=0, hq=2, hkv=1, w=2,
                                                   beta=0.1, seed=(991,)), False),
}


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


@pytest.mark.parametrize("name", list(CONFIGS))
def test_full_size(st, name):
    make, full_abase = CONFIGS[name]
    wl = make()
    q, k, v = to_device(wl)
    H, n, w = k.shape[1], wl.n, wl.q.shape[0]
    b = oracle.budget(n, wl.beta)
    # fused call, as timed by bench.py
    ko, vo, idx = st.compress_layer(q, k, v, wl.frames, beta=wl.beta)
    # staged calls on the same inputs
    sh = st.make_shape(q, k)
    prm = st.make_params(wl.beta)
    ws = st.workspace(sh, wl.frames, prm)
    a = torch.empty((H, n), dtype=torch.float32, device="cuda")
    phi, rho, score = torch.empty_like(a), torch.empty_like(a), torch.empty_like(a)
    tau = torch.empty((H,), dtype=torch.float32, device="cuda")
    gate = torch.empty((H, n), dtype=torch.uint8, device="cuda")
    st.stlite_score(q, k, a, ws)
    st.stlite_spatial_saliency(q, k, wl.frames, phi, ws)
    st.stlite_gate_frames(q, k, wl.frames, b, rho, tau, gate, ws)
    idx2 = torch.empty_like(idx)
    st.stlite_select_topk(q, k, wl.frames, prm, a, phi, gate, b, idx2, score, ws)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    ig = idx.cpu().numpy()
    np.testing.assert_array_equal(idx2.cpu().numpy(), ig)
    ag, pg, rg, tg, gg, sg = (x.cpu().numpy() for x in (a, phi, rho, tau, gate, score))
    k64 = exact64(k)
    rng = np.random.default_rng(1234)

    # window score: invariant, and the full oracle where affordable
    np.testing.assert_allclose(ag.astype(np.float64).sum(1), w, rtol=1e-4)
    if full_abase:
        a_ora = oracle.abase(exact64(q), k64, threads=8)
        for h in range(H):
            assert_within(ag[h], a_ora[h], a_bound(a_ora[h]), "A_base head %d" % h)

    # CSS and TSG: sampled tokens against the oracle one by one
    off, gh, gw = wl.frames
    vis = np.nonzero(visual_mask(n, wl.frames))[0]
    pool = np.nonzero(pool_mask(n, wl.frames))[0]
    assert np.isnan(pg[:, ~visual_mask(n, wl.frames)]).all()
    for h in range(H):
        for j in rng.choice(vis, 400, replace=False):
            f = int(np.searchsorted(off, j, side="right") - 1)
            loc = j - off[f]
            o = oracle.css_phi_token(k64, h, int(off[f]), int(gh[f]), int(gw[f]), int(loc // gw[f]), int(loc % gw[f]))
            assert abs(pg[h, j] - o) <= A_RTOL * abs(o) + COS_ATOL, ("Phi", h, j, pg[h, j], o)
        for i in rng.choice(pool, 150, replace=False):
            o = oracle.tsg_rho_token(k64, h, int(i), wl.frames)
            assert abs(rg[h, i] - o) <= A_RTOL * abs(o) + COS_ATOL, ("rho", h, i, rg[h, i], o)

    # threshold and gate: exact on the GPU's rho
    t2, g2, _ = oracle.tsg_gate(rg.astype(np.float64), wl.frames, b)
    np.testing.assert_array_equal(t2, tg.astype(np.float64))
    np.testing.assert_array_equal(g2, gg)
    # integrated score from the GPU's stage outputs, and exact Top-B on it
    s2 = oracle.combine(ag, pg, gg, wl.frames)
    assert_within(sg, s2, A_RTOL * np.abs(s2) + 2 * COS_ATOL, "S")
    np.testing.assert_array_equal(oracle.topk(sg.astype(np.float64), b), ig)
    for h in range(H):
        assert len(np.unique(ig[h])) == b and (np.diff(ig[h]) > 0).all()
    # compaction: byte copies
    ko2, vo2 = oracle.gather(k.view(torch.int16).cpu().numpy(), v.view(torch.int16).cpu().numpy(), ig)
    np.testing.assert_array_equal(ko.view(torch.int16).cpu().numpy(), ko2)
    np.testing.assert_array_equal(vo.view(torch.int16).cpu().numpy(), vo2)
