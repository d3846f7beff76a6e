"""Full-size configurations through the C ABI against the whole fp64 oracle.

For every configuration the oracle computes A_base of every token, Phi of
every visual token and rho of every pool token (its work spread over the
host's cores by query head and by runs of pool tokens), then the threshold,
gate, integrated score and Top-B of Algorithm 1.  The GPU's fused call (the
one bench.py times) and its staged calls are compared with it under the
matching rules: every score element within tolerance, gate flips only at
the threshold, kept sets equal up to swaps at the B-th score or at gate
flips, compacted rows bit-exact, and exact staged parity downstream of the
scores (tau/gate on the GPU's rho, Eq. 9 and Top-B on the GPU's stage
outputs, compaction byte copies).  Nothing is sampled.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_00188_gb300 import synth
from parity import (A_FLOOR, A_RTOL, COS_ATOL, a_bound, assert_within, check_kept_sets, cos_bound, exact64,
                    gate_flip_tokens, pool_mask, to_device, visual_mask)

pytestmark = pytest.mark.gpu

# name: (inputs key, generator); configurations that differ only in beta
# share their inputs and so their oracle scores
CONFIGS = {
    "uitars_b10": ("uitars", lambda: synth.uitars_layer(beta=0.1)),
    "uitars_b20": ("uitars", lambda: synth.uitars_layer(beta=0.2)),
    "uitars_b30": ("uitars", lambda: synth.uitars_layer(beta=0.3)),
    "uitars_b40": ("uitars", lambda: synth.uitars_layer(beta=0.4)),
    "traj50_l0": ("traj50_l0", lambda: synth.trajectory_50(0)),
    "traj50_l27": ("traj50_l27", lambda: synth.trajectory_50(27)),
    "small_s0_b10": ("small_s0_b10", lambda: synth.small_backbone_seq(0, beta=0.1)),
    "small_s5_b40": ("small_s5_b40", lambda: synth.small_backbone_seq(5, beta=0.4)),
    "long_l0": ("long_l0", lambda: synth.long_horizon(0)),
    "long_l27": ("long_l27", lambda: synth.long_horizon(27)),
    # the frame-table limit: 256 frames (2x3 grids, one text token after each)
    "max_frames_256": ("max_frames_256", lambda: synth.trajectory(
        n_steps=256, gh=2, gw=3, n_text=1, hq=4, hkv=2, w=4, beta=0.3, n_boxes=(1, 2),
        box_hw=((1, 1), (2, 2)), seed=(990,))),
    # the largest cache the selection holds on chip: 393,216 tokens
    # (256 frames of 32x48, one KV head)
    "max_tokens_393216": ("max_tokens_393216", lambda: synth.trajectory(
        n_steps=256, gh=32, gw=48, n_text=0, hq=2, hkv=1, w=2, beta=0.1, seed=(991,))),
}

_SCORES = {}


def oracle_scores(key, q64, k64, frames):
    """A_base, Phi and rho of every token (fp64), once per set of inputs."""
    if key not in _SCORES:
        _SCORES.clear()   # one set of full-size scores held at a time
        t = oracle.host_threads()
        _SCORES[key] = (oracle.abase(q64, k64, threads=t), oracle.css_phi(k64, frames, threads=t),
                        oracle.tsg_rho(k64, frames, threads=t))
    return _SCORES[key]


def s_tol(x):
    return A_RTOL * abs(x) + A_FLOOR + COS_ATOL * 2


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
    key, make = CONFIGS[name]
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

    # the whole oracle pipeline on the same (bf16-exact) inputs
    a_o, phi_o, rho_o = oracle_scores(key, exact64(q), exact64(k), wl.frames)
    tau_o, gate_o, _ = oracle.tsg_gate(rho_o, wl.frames, b)
    s_o = oracle.combine(a_o, phi_o, gate_o, wl.frames)
    idx_o = oracle.topk(s_o, b)

    # every score element
    np.testing.assert_allclose(ag.astype(np.float64).sum(1), w, rtol=1e-4)
    for h in range(H):
        assert_within(ag[h], a_o[h], a_bound(a_o[h]), "A_base head %d" % h)
    vis, pool = visual_mask(n, wl.frames), pool_mask(n, wl.frames)
    assert np.isnan(pg[:, ~vis]).all()
    assert_within(pg[:, vis], phi_o[:, vis], cos_bound(phi_o[:, vis]), "Phi")
    assert np.isnan(rg[:, ~pool]).all() and (gg[:, ~pool] == 1).all()
    assert_within(rg[:, pool], rho_o[:, pool], cos_bound(rho_o[:, pool]), "rho")

    # threshold and gate: exact on the GPU's rho; against the oracle's own
    # rho, flips only at the threshold
    t2, g2, _ = oracle.tsg_gate(rg.astype(np.float64), wl.frames, b)
    np.testing.assert_array_equal(t2, tg.astype(np.float64))
    np.testing.assert_array_equal(g2, gg)
    flips = []
    for h in range(H):
        if pool.any():
            assert abs(tg[h] - tau_o[h]) <= A_RTOL * abs(tau_o[h]) + COS_ATOL, (h, tg[h], tau_o[h])
        flips.append(gate_flip_tokens(gg[h], gate_o[h], rho_o[h], tau_o[h]))

    # integrated score: from the GPU's stage outputs (staged), and against the
    # oracle's wherever the gates agree
    s2 = oracle.combine(ag, pg, gg, wl.frames)
    assert_within(sg, s2, A_RTOL * np.abs(s2) + 2 * COS_ATOL, "S (staged)")
    same = gg == gate_o
    assert_within(sg[same], s_o[same], A_RTOL * np.abs(s_o[same]) + A_FLOOR * np.abs(s_o).max() + 2 * COS_ATOL,
                  "S")
    np.testing.assert_array_equal(oracle.topk(sg.astype(np.float64), b), ig)

    # kept sets against the whole oracle pipeline
    for h in range(H):
        assert len(np.unique(ig[h])) == b and (np.diff(ig[h]) > 0).all()
        check_kept_sets(ig[h], idx_o[h], s_o[h], b, s_tol, allowed_extra=flips[h])
    # compaction: byte copies
    ko2, vo2 = oracle.gather(k.view(torch.int16).cpu().numpy(), v.view(torch.int16).cpu().numpy(), ig)
    np.testing.assert_array_equal(ko.view(torch.int16).cpu().numpy(), ko2)
    np.testing.assert_array_equal(vo.view(torch.int16).cpu().numpy(), vo2)
