"""Pins for the CPU oracle: closed forms, invariants, hand-derived fixtures and
brute force on tiny inputs (none of them re-types the oracle's own formula).

Each test names the paper passage it pins: Eq. 2 (window score), Eqs. 4-5
(CSS), Eqs. 6-8 (TSG), Eq. 9 (integrated score), Sec. 2.1 (budget, top-B) and
Algorithm 1 (whole procedure).
"""
import itertools
import math
import os

import numpy as np
import pytest

import oracle
from paper_2603_00188_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def frames_of(*spans):
    """spans: (offset, gh, gw) per frame."""
    off = np.array([s[0] for s in spans], np.int32)
    gh = np.array([s[1] for s in spans], np.int32)
    gw = np.array([s[2] for s in spans], np.int32)
    return off, gh, gw


# ------------------------------------------------------------------ budget

@pytest.mark.parametrize("n,beta,expect", [
    (1152, 0.2, 230), (23680, 0.1, 2368), (23680, 0.2, 4736), (23680, 0.3, 7104),
    (23680, 0.4, 9472), (53600, 0.2, 10720), (132800, 0.1, 13280), (10, 1.0, 10),
    (10, 0.01, 1), (7, 0.5, 3),
])
def test_budget_floor(n, beta, expect):
    # Sec. 2.1: B = floor(beta * L); integer values worked by hand.
    assert oracle.budget(n, beta) == expect


def test_budget_override():
    assert oracle.budget(1152, 0.2, 231) == 231    # ceil(0.2 * 1152) via override
    assert oracle.budget(10, 0.2, 50) == 10


# ------------------------------------------------------- window score, Eq. 2

def test_abase_closed_form_single_head():
    # w = 1, G = 1, q = e_0 and k_j = sqrt(d) * x_j * e_0, so q.k_j / sqrt(d) = x_j
    # and A_j = exp(x_j) / sum exp(x).  Catches a missing or wrong 1/sqrt(d).
    d, n = 16, 7
    x = np.array([0.3, -1.2, 2.0, 0.0, 0.7, -0.4, 1.1])
    q = np.zeros((1, 1, d)); q[0, 0, 0] = 1.0
    k = np.zeros((n, 1, d)); k[:, 0, 0] = math.sqrt(d) * x
    a = oracle.abase(q, k)
    z = sum(math.exp(t) for t in x)
    np.testing.assert_allclose(a[0], [math.exp(t) / z for t in x], rtol=1e-13)


def test_abase_equal_keys_uniform():
    # All keys identical: every softmax row is uniform, so A_j = w / N.
    rng = np.random.default_rng(1)
    w, hq, hkv, d, n = 5, 6, 2, 8, 11
    q = rng.standard_normal((w, hq, d))
    k = np.repeat(rng.standard_normal((1, hkv, d)), n, axis=0)
    a = oracle.abase(q, k)
    np.testing.assert_allclose(a, np.full((hkv, n), w / n), rtol=1e-12)


def test_abase_sums_to_window():
    # Each softmax row sums to 1; w rows summed, G heads averaged -> sum_j A = w.
    rng = np.random.default_rng(2)
    w, hq, hkv, d, n = 4, 6, 3, 16, 40
    a = oracle.abase(rng.standard_normal((w, hq, d)) * 2, rng.standard_normal((n, hkv, d)))
    np.testing.assert_allclose(a.sum(axis=1), np.full(hkv, w), rtol=1e-12)
    assert (a > 0).all()


def test_abase_gqa_grouping():
    # Query head g belongs to KV head g // G: perturbing query head 2 (G=2)
    # moves A of KV head 1 only.
    rng = np.random.default_rng(3)
    w, hq, hkv, d, n = 3, 4, 2, 8, 9
    q = rng.standard_normal((w, hq, d)); k = rng.standard_normal((n, hkv, d))
    a0 = oracle.abase(q, k)
    q2 = q.copy(); q2[:, 2] += rng.standard_normal((w, d))
    a1 = oracle.abase(q2, k)
    np.testing.assert_array_equal(a0[0], a1[0])
    assert np.abs(a0[1] - a1[1]).max() > 1e-3


def test_abase_gqa_mean_closed_form():
    # G = 2 query heads with logits x (head 0) and y (head 1), w = 1:
    # A = (softmax(x) + softmax(y)) / 2, built from hand-chosen logits.
    d = 4
    x = np.array([0.5, -0.5, 1.5]); y = np.array([2.0, 0.0, -1.0])
    q = np.zeros((1, 2, d)); q[0, 0, 0] = 1.0; q[0, 1, 1] = 1.0
    k = np.zeros((3, 1, d)); k[:, 0, 0] = 2 * x; k[:, 0, 1] = 2 * y   # sqrt(4) = 2
    sx = np.exp(x) / np.exp(x).sum(); sy = np.exp(y) / np.exp(y).sum()
    np.testing.assert_allclose(oracle.abase(q, k)[0], (sx + sy) / 2, rtol=1e-13)


def test_abase_library_softmax():
    # Special case that reduces to a library routine: torch.softmax in float64.
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(4)
    w, hq, hkv, d, n = 6, 4, 1, 32, 50
    q = rng.standard_normal((w, hq, d)); k = rng.standard_normal((n, hkv, d)) * 1.5
    logits = torch.einsum("rgd,nd->rgn", torch.from_numpy(q), torch.from_numpy(k[:, 0])) / math.sqrt(d)
    ref = torch.softmax(logits, dim=-1).sum(dim=0).mean(dim=0).numpy()
    np.testing.assert_allclose(oracle.abase(q, k)[0], ref, rtol=1e-12)


# ------------------------------------------------------------- CSS, Eqs. 4-5

def _read_fixture(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                rows.append(line)
    return rows


def _closed(expr):
    return float(eval(expr, {"sqrt": math.sqrt, "__builtins__": {}}))


def test_css_handworked_fixture():
    rows = _read_fixture("css_handworked_2x3.txt")
    k = np.zeros((6, 1, 2)); expect = np.zeros(6)
    for r in rows:
        parts = r.split()
        u, v = int(parts[1]), int(parts[2])
        k[u * 3 + v, 0] = [float(parts[3]), float(parts[4])]
        expect[u * 3 + v] = _closed(" ".join(parts[5:]))
    phi = oracle.css_phi(k, frames_of((0, 2, 3)))
    np.testing.assert_allclose(phi[0], expect, rtol=0, atol=1e-14)


def test_css_checkerboard_fixture():
    rows = _read_fixture("css_checkerboard_3x4.txt")
    expect = np.array([[_closed(t) for t in r.split()] for r in rows])
    gh, gw, d = 3, 4, 5
    k = np.zeros((gh * gw, 1, d))
    for u in range(gh):
        for v in range(gw):
            k[u * gw + v, 0, 0] = (-1) ** (u + v)
    phi = oracle.css_phi(k, frames_of((0, gh, gw)))
    np.testing.assert_allclose(phi[0].reshape(gh, gw), expect, atol=1e-14)


def test_css_equal_keys_zero():
    rng = np.random.default_rng(5)
    k = np.repeat(rng.standard_normal((1, 2, 16)), 30, axis=0)
    phi = oracle.css_phi(k, frames_of((0, 5, 6)))
    np.testing.assert_allclose(phi, 0.0, atol=1e-14)


def test_css_orthonormal_one():
    # Distinct basis vectors: every cosine 0 -> Phi = 1 everywhere.
    gh, gw = 4, 5
    k = np.eye(gh * gw)[:, None, :] * np.arange(1, gh * gw + 1)[:, None, None]  # magnitudes differ
    phi = oracle.css_phi(k, frames_of((0, gh, gw)))
    np.testing.assert_allclose(phi[0], 1.0, atol=1e-15)


def test_css_planted_rectangle_closed_form():
    # Identical keys r on a 2x3 rectangle, distinct basis vectors elsewhere:
    # rectangle cell Phi = 1 - (#rectangle neighbours)/|N|, background Phi = 1.
    gh, gw, d = 6, 7, 64
    k = np.eye(d)[: gh * gw][:, None, :].copy()
    r = np.zeros(d); r[-1] = 2.5
    rect = [(u, v) for u in range(2, 4) for v in range(3, 6)]
    for (u, v) in rect:
        k[u * gw + v, 0] = r
    phi = oracle.css_phi(k, frames_of((0, gh, gw)))[0].reshape(gh, gw)
    for u in range(gh):
        for v in range(gw):
            nb = [(u + a, v + b) for a in (-1, 0, 1) for b in (-1, 0, 1)
                  if (a or b) and 0 <= u + a < gh and 0 <= v + b < gw]
            if (u, v) in rect:
                expect = 1 - sum((p in rect) for p in nb) / len(nb)
            else:
                expect = 1.0
            assert abs(phi[u, v] - expect) < 1e-14, (u, v)


def test_css_edge_cases_and_frame_isolation():
    rng = np.random.default_rng(6)
    # 1x1 grid: no neighbour -> Phi = 0; text tokens -> NaN.
    k = rng.standard_normal((10, 1, 8))
    fr = frames_of((0, 1, 1), (3, 2, 2))
    phi = oracle.css_phi(k, fr)[0]
    assert phi[0] == 0.0
    assert np.isnan(phi[[1, 2, 7, 8, 9]]).all()
    # 1xW grid: each cell sees only its left/right neighbours.
    k2 = np.zeros((3, 1, 2)); k2[:, 0] = [[1, 0], [1, 1], [0, 1]]
    p2 = oracle.css_phi(k2, frames_of((0, 1, 3)))[0]
    s = 1 / math.sqrt(2)
    np.testing.assert_allclose(p2, [1 - s, 1 - s, 1 - s], atol=1e-15)
    # frames do not see each other: changing frame 1 leaves frame 0 alone
    k3 = k.copy(); k3[3:7] = rng.standard_normal((4, 1, 8))
    np.testing.assert_array_equal(oracle.css_phi(k3, fr)[0][:3], phi[:3])


def test_css_magnitude_invariance():
    rng = np.random.default_rng(7)
    k = rng.standard_normal((24, 2, 16))
    fr = frames_of((0, 4, 6))
    scale = rng.uniform(0.1, 10, size=(24, 2, 1))
    np.testing.assert_allclose(oracle.css_phi(k * scale, fr), oracle.css_phi(k, fr), atol=1e-13)


def test_css_zero_vector():
    # Reading: norms clamp at 1e-8, so a zero key has cosine 0 with every neighbour.
    k = np.ones((4, 1, 3)); k[0] = 0.0
    phi = oracle.css_phi(k, frames_of((0, 2, 2)))[0]
    assert phi[0] == 1.0
    np.testing.assert_allclose(phi[1:], 1 - 2 / 3, atol=1e-15)


# ------------------------------------------------------------- TSG, Eqs. 6-8

def test_rho_angles_closed_form():
    # 2-D keys at angles; rho_i = max_j cos(theta_i - phi_j) by trigonometry.
    rng = np.random.default_rng(8)
    th = rng.uniform(-math.pi, math.pi, 6)     # historical frame, 2x3
    ph = rng.uniform(-math.pi, math.pi, 4)     # current frame, 2x2
    mags = rng.uniform(0.5, 3, 10)
    ang = np.concatenate([th, ph])
    k = np.stack([np.cos(ang), np.sin(ang)], -1)[:, None, :] * mags[:, None, None]
    fr = frames_of((0, 2, 3), (6, 2, 2))
    rho = oracle.tsg_rho(k, fr)[0]
    expect = [max(math.cos(t - p) for p in ph) for t in th]
    np.testing.assert_allclose(rho[:6], expect, atol=1e-14)
    assert np.isnan(rho[6:]).all()


def test_rho_duplicate_and_orthogonal():
    rng = np.random.default_rng(9)
    d = 32
    cur = rng.standard_normal((4, 1, d))
    ortho = np.eye(d)[8:12][:, None, :]           # orthogonal to the current frame below
    cur_o = np.eye(d)[:4][:, None, :] * 3
    # frame 0 = copy of current (rho = 1); frame 1 orthogonal (rho = 0)
    k = np.concatenate([cur, np.zeros((1, 1, d)), cur, np.zeros((1, 1, d))])
    fr = frames_of((0, 2, 2), (5, 2, 2))
    np.testing.assert_allclose(oracle.tsg_rho(k, fr)[0][:4], 1.0, atol=1e-14)
    k2 = np.concatenate([ortho, cur_o])
    fr2 = frames_of((0, 2, 2), (4, 2, 2))
    np.testing.assert_allclose(oracle.tsg_rho(k2, fr2)[0][:4], 0.0, atol=1e-15)


def test_rho_single_frame_and_scale():
    rng = np.random.default_rng(10)
    k = rng.standard_normal((20, 2, 8))
    assert np.isnan(oracle.tsg_rho(k, frames_of((2, 3, 3)))).all()   # F = 1: empty pool
    fr = frames_of((0, 2, 3), (6, 1, 4), (12, 2, 2))
    r1 = oracle.tsg_rho(k, fr)
    r2 = oracle.tsg_rho(k * 7.5, fr)
    np.testing.assert_allclose(r1, r2, atol=1e-14)
    # pool = frames 0 and 1 only; text and current frame are NaN
    pool = np.zeros(20, bool); pool[0:6] = True; pool[6:10] = True
    assert np.isfinite(r1[:, pool]).all() and np.isnan(r1[:, ~pool]).all()


def test_tau_rank_property():
    # tau is the min(B, |pool|)-th smallest pool value:
    # #{rho < tau} < m <= #{rho <= tau}; gate = [rho <= tau] on the pool only.
    rng = np.random.default_rng(11)
    fr = frames_of((0, 3, 4), (14, 2, 5), (30, 2, 2))
    n = 36
    rho = np.full((2, n), np.nan)
    pool = np.r_[0:12, 14:24]
    rho[:, pool] = np.round(rng.uniform(0, 1, (2, pool.size)), 1)   # many ties
    for b in (1, 5, 13, 22, 40):
        tau, gate, psz = oracle.tsg_gate(rho, fr, b)
        assert psz == 22
        m = min(b, 22)
        for h in range(2):
            vals = rho[h, pool]
            assert (vals < tau[h]).sum() < m <= (vals <= tau[h]).sum()
            assert tau[h] in vals
            expect = np.ones(n, np.uint8); expect[pool] = vals <= tau[h]
            np.testing.assert_array_equal(gate[h], expect)
        if b >= 22:
            assert (gate == 1).all()   # B >= |pool| admits the whole pool


def test_gate_disabled_or_empty_pool():
    rho = np.random.default_rng(12).uniform(size=(1, 10))
    tau, gate, _ = oracle.tsg_gate(rho, frames_of((0, 2, 2), (5, 1, 2)), 1, tsg_enable=0)
    assert np.isnan(tau).all() and (gate == 1).all()
    tau, gate, psz = oracle.tsg_gate(np.full((1, 10), np.nan), frames_of((2, 2, 2)), 3)
    assert psz == 0 and np.isnan(tau).all() and (gate == 1).all()


# ------------------------------------------------------- integrated score, Eq. 9

def test_combine_cases():
    fr = frames_of((0, 1, 3), (4, 1, 2))      # tokens 3, 6, 7 are text
    a = np.array([[0.1, 0.2, 0.3, 0.4, 0.5, 0.6, 0.7, 0.8]])
    phi = np.array([[1.0, 0.5, 0.25, np.nan, 2.0, 0.0, np.nan, np.nan]])
    gate = np.array([[1, 0, 1, 1, 1, 1, 1, 1]], np.uint8)
    s = oracle.combine(a, phi, gate, fr, alpha=1.0)
    np.testing.assert_allclose(s[0], [1.1, 0.0, 0.55, 0.4, 2.5, 0.6, 0.7, 0.8], atol=1e-15)
    s2 = oracle.combine(a, phi, gate, fr, alpha=0.5)
    np.testing.assert_allclose(s2[0], [0.6, 0.0, 0.425, 0.4, 1.5, 0.6, 0.7, 0.8], atol=1e-15)
    s3 = oracle.combine(a, phi, gate, fr, alpha=1.0, css_enable=0)
    np.testing.assert_allclose(s3[0], [0.1, 0.0, 0.3, 0.4, 0.5, 0.6, 0.7, 0.8], atol=1e-15)


# ----------------------------------------------------------- top-B, Sec. 2.1

def _dominates(s, keep):
    """The kept set of size B: every kept token outranks every dropped one,
    where i outranks j iff s_i > s_j or (s_i == s_j and i < j)."""
    drop = [j for j in range(len(s)) if j not in keep]
    return all((s[i] > s[j]) or (s[i] == s[j] and i < j) for i in keep for j in drop)


@pytest.mark.parametrize("seed", range(6))
def test_topk_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    n = 8
    s = rng.integers(0, 4, size=(1, n)).astype(np.float64) / 2      # heavy ties
    for b in range(1, n + 1):
        got = oracle.topk(s, b)[0]
        valid = [c for c in itertools.combinations(range(n), b) if _dominates(s[0], set(c))]
        assert len(valid) == 1
        np.testing.assert_array_equal(got, valid[0])


def test_topk_invariants_large():
    rng = np.random.default_rng(13)
    s = rng.standard_normal((3, 5000)); s[:, ::7] = 0.25          # planted ties
    idx = oracle.topk(s, 1234)
    for h in range(3):
        row = idx[h]
        assert len(row) == 1234 and (np.diff(row) > 0).all() and row.min() >= 0 and row.max() < 5000
        thr = np.sort(s[h])[::-1][1233]
        assert (s[h, row] >= thr).all()
        assert (s[h][np.setdiff1d(np.arange(5000), row)] <= thr).all()


# --------------------------------------------------------------------- gather

def test_gather_bytes():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(14)
    k = torch.from_numpy(rng.standard_normal((50, 3, 128)).astype(np.float32)).to(torch.bfloat16)
    v = torch.from_numpy(rng.standard_normal((50, 3, 128)).astype(np.float32)).to(torch.bfloat16)
    kk, vv = k.view(torch.int16).numpy(), v.view(torch.int16).numpy()
    idx = np.sort(np.stack([rng.choice(50, 17, replace=False) for _ in range(3)]), axis=1).astype(np.int32)
    ko, vo = oracle.gather(kk, vv, idx)
    for h in range(3):
        np.testing.assert_array_equal(ko[:, h], kk[idx[h], h])
        np.testing.assert_array_equal(vo[:, h], vv[idx[h], h])


# ------------------------------------------------------- Algorithm 1, end to end

def _tiny_traj(seed=0, n_steps=4, gh=4, gw=5, nt=3, hq=4, hkv=2, d=16, w=3):
    return synth.trajectory(n_steps=n_steps, gh=gh, gw=gw, n_text=nt, hq=hq, hkv=hkv, d=d, w=w,
                            n_boxes=(1, 2), box_hw=((1, 1), (2, 2)), seed=(900, seed))


def test_end_to_end_beta_one_keeps_all():
    wl = _tiny_traj()
    out = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=1.0)
    assert out["budget"] == wl.n
    np.testing.assert_array_equal(out["idx"], np.tile(np.arange(wl.n), (2, 1)))


def test_end_to_end_single_frame_tsg_noop():
    # One frame: TSG has an empty pool and must not change anything (CSS only).
    wl = _tiny_traj(n_steps=1)
    a = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.3, tsg_enable=1)
    b = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.3, tsg_enable=0)
    np.testing.assert_array_equal(a["idx"], b["idx"])
    assert (a["gate"] == 1).all()


def test_end_to_end_snapkv_base():
    # alpha = 0 and TSG off: the retained set is top-B of A_base (library argsort).
    wl = _tiny_traj(seed=3)
    out = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.25, tsg_enable=0, css_enable=0)
    for h in range(2):
        order = np.lexsort((np.arange(wl.n), -out["a"][h]))   # S desc, index asc
        np.testing.assert_array_equal(out["idx"][h], np.sort(order[: out["budget"]]))


def test_end_to_end_exact_budget_and_gate_invariants():
    wl = _tiny_traj(seed=4, n_steps=5)
    out = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.2)
    b = out["budget"]
    off, gh, gw = wl.frames
    cur = np.arange(off[-1], off[-1] + gh[-1] * gw[-1])
    for h in range(2):
        assert len(np.unique(out["idx"][h])) == b
        assert (out["gate"][h][cur] == 1).all()
        assert out["gate"][h].sum() - (wl.n - out["pool"]) >= min(b, out["pool"])


def test_tiny_ref_duplicate_frame_gated():
    # Frame 3 (current) = frame 2 + N(0, 0.01^2): frame 2's rho is ~1 and the
    # m = 230 lowest-rho pool tokens come from frames 0-1, so TSG gates all of frame 2.
    wl = synth.tiny_ref()
    b = oracle.budget(wl.n, 0.2)
    rho = oracle.tsg_rho(wl.k, wl.frames, threads=4)
    tau, gate, pool = oracle.tsg_gate(rho, wl.frames, b)
    assert pool == 768 and b == 230
    f2 = np.arange(2 * 288, 2 * 288 + 256)
    assert (rho[:, f2] > 0.99).all()
    assert (gate[:, f2] == 0).all()
    assert (tau < 0.6).all()


def test_salient_rectangle_kept():
    # CSS purpose (Sec. 3.1): on a uniform background a small element with
    # different keys has Phi ~ 1 on its cells and ring, ~0 elsewhere, so at a
    # budget just above the element+ring size all element cells are kept.
    rng = np.random.default_rng(15)
    gh, gw, d, hq, hkv, w = 8, 8, 32, 2, 1, 2
    base = rng.standard_normal(d)
    k = np.tile(base, (gh * gw, 1)) + 1e-3 * rng.standard_normal((gh * gw, d))
    elem = [(3, 3), (3, 4)]
    other = rng.standard_normal(d)
    for (u, v) in elem:
        k[u * gw + v] = other
    k = k[:, None, :]
    q = rng.standard_normal((w, hq, d)) * 0.1
    out = oracle.compress_layer(q, k, frames_of((0, gh, gw)), beta=0.25)   # B = 16
    kept = set(out["idx"][0].tolist())
    assert all(u * gw + v in kept for (u, v) in elem)


def _text_reversal(n, frames):
    """Permutation that reverses the order of the text tokens (positions
    outside every frame) and leaves every visual token in place: new
    position p holds old token perm[p]."""
    off, gh, gw = frames
    vis = np.zeros(n, bool)
    for o, a, b in zip(off, gh, gw):
        vis[o:o + a * b] = True
    text = np.nonzero(~vis)[0]
    perm = np.arange(n)
    perm[text] = text[::-1]
    return perm


def test_end_to_end_text_permutation_equivariance():
    # Nothing in Algorithm 1 depends on where a text token sits (no positional
    # term; CSS and TSG only see visual tokens): reordering the text tokens
    # reorders A_base and S the same way, leaves Phi, rho and tau unchanged,
    # and maps the kept set through the permutation.
    wl = _tiny_traj(seed=6, n_steps=4, nt=5)
    perm = _text_reversal(wl.n, wl.frames)
    assert (perm != np.arange(wl.n)).any()
    a = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.3)
    b = oracle.compress_layer(wl.q, wl.k[perm], wl.frames, beta=0.3)
    np.testing.assert_allclose(b["a"], a["a"][:, perm], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(b["s"], a["s"][:, perm], rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(b["phi"], a["phi"][:, perm])
    np.testing.assert_array_equal(b["gate"], a["gate"][:, perm])
    np.testing.assert_array_equal(np.isnan(b["rho"]), np.isnan(a["rho"]))
    np.testing.assert_array_equal(b["tau"], a["tau"])
    inv = np.argsort(perm)
    for h in range(2):
        np.testing.assert_array_equal(b["idx"][h], np.sort(inv[a["idx"][h]]))


# ------------------------------------------- consumer: decode over the cache

def test_decode_single_and_equal_keys():
    rng = np.random.default_rng(21)
    d, hq, hkv = 8, 4, 2
    q = rng.standard_normal((2, hq, d))
    v = rng.standard_normal((5, hkv, d))
    # one cached token: the output is its value row, whatever the query
    out = oracle.decode_attention(q, rng.standard_normal((1, hkv, d)), v[:1])
    for g in range(hq):
        np.testing.assert_allclose(out[:, g], np.broadcast_to(v[0, g // 2], (2, d)), rtol=0, atol=1e-15)
    # equal keys: uniform weights, the output is the mean value row of the head
    k = np.tile(rng.standard_normal((1, hkv, d)), (5, 1, 1))
    out = oracle.decode_attention(q, k, v)
    for g in range(hq):
        np.testing.assert_allclose(out[:, g], np.broadcast_to(v[:, g // 2].mean(0), (2, d)), rtol=1e-13,
                                   atol=1e-15)


def test_decode_dominant_key_and_weights_sum_to_one():
    rng = np.random.default_rng(22)
    d, hq, hkv, n = 16, 2, 1, 7
    q = rng.standard_normal((1, hq, d))
    k = rng.standard_normal((n, hkv, d)) * 0.01
    k[3, 0] = 100.0 * q[0, 0] / np.linalg.norm(q[0, 0])   # dominates head 0's softmax
    v = rng.standard_normal((n, hkv, d))
    out = oracle.decode_attention(q, k, v)
    np.testing.assert_allclose(out[0, 0], v[3, 0], rtol=0, atol=1e-12)
    # constant value rows: convex weights return the constant exactly (up to rounding)
    out = oracle.decode_attention(q, k, np.full((n, hkv, d), 2.5))
    np.testing.assert_allclose(out, 2.5, rtol=1e-14)


def test_decode_library_attention():
    # the textbook case against the library routine (fp64 CPU scaled-dot-product attention)
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(23)
    w, hq, hkv, n, d = 3, 6, 2, 40, 32
    q, k, v = rng.standard_normal((w, hq, d)), rng.standard_normal((n, hkv, d)), rng.standard_normal((n, hkv, d))
    out = oracle.decode_attention(q, k, v)
    G = hq // hkv
    tq = torch.from_numpy(q).permute(1, 0, 2)                                     # [hq][w][d]
    tk = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(G, 0)              # [hq][n][d]
    tv = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(G, 0)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-14)


def test_critical_hit_rate_cases():
    wl = _tiny_traj(seed=8, n_steps=3, w=1)
    # kept set = Top_B of the probe's own attention (alpha = 0, TSG off, the
    # probe as the only window row): every critical token is kept
    out = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.3, tsg_enable=0, css_enable=0)
    np.testing.assert_array_equal(oracle.critical_hit_rate(out["idx"], wl.q, wl.k), 1.0)
    # beta = 1 keeps everything
    out = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=1.0)
    np.testing.assert_array_equal(oracle.critical_hit_rate(out["idx"], wl.q, wl.k), 1.0)
    # the complement of the critical set scores 0
    b = oracle.budget(wl.n, 0.3)
    a = oracle.abase(wl.q, wl.k)
    top = oracle.topk(a, b)
    rest = np.stack([np.setdiff1d(np.arange(wl.n), top[h])[:b] for h in range(a.shape[0])])
    np.testing.assert_array_equal(oracle.critical_hit_rate(rest, wl.q, wl.k), 0.0)


# ------------------------------------------------------ ablation variants

def _two_frame_keys(hist, cur, d=16):
    """Keys of two 1 x n frames (historical then current) in R^d from short
    explicit vectors (zero-padded); one KV head."""
    rows = [np.pad(np.asarray(v, float), (0, d - len(v))) for v in list(hist) + list(cur)]
    k = np.asarray(rows)[:, None, :]
    frames = frames_of((0, 1, len(hist)), (len(hist), 1, len(cur)))
    return k, frames


def test_rho_dot_and_neg_l2_closed_form():
    k, fr = _two_frame_keys(hist=[[3, 0], [0, 2], [1, 1]], cur=[[2, 0], [0, 1], [4, 0]])
    dot = oracle.tsg_rho(k, fr, metric=oracle.TSG_DOT)[0]
    l2 = oracle.tsg_rho(k, fr, metric=oracle.TSG_NEG_L2)[0]
    # dot: max(6, 0, 12) = 12; max(0, 2, 0) = 2; max(2, 1, 4) = 4
    np.testing.assert_array_equal(dot[:3], [12.0, 2.0, 4.0])
    # -|a-b|^2: (3,0) vs (2,0),(0,1),(4,0): 1, 10, 1 -> -1; (0,2): 8, 1, 20 -> -1; (1,1): 2, 1, 10 -> -1
    np.testing.assert_array_equal(l2[:3], [-1.0, -1.0, -1.0])
    assert np.isnan(dot[3:]).all() and np.isnan(l2[3:]).all()
    # homogeneity: scaling every key by c scales both by c^2 (cosine is invariant)
    np.testing.assert_allclose(oracle.tsg_rho(2.5 * k, fr, metric=oracle.TSG_DOT)[0][:3], 6.25 * dot[:3])
    np.testing.assert_allclose(oracle.tsg_rho(2.5 * k, fr, metric=oracle.TSG_NEG_L2)[0][:3], 6.25 * l2[:3])


def test_rho_neg_l2_duplicate_is_zero():
    wl = _tiny_traj(seed=9, n_steps=3)
    k = wl.k.copy()
    off, gh, gw = wl.frames
    P = gh[0] * gw[0]
    k[off[-1]:off[-1] + P] = k[off[0]:off[0] + P]          # current frame = a copy of frame 0
    rho = oracle.tsg_rho(k, wl.frames, metric=oracle.TSG_NEG_L2)
    np.testing.assert_array_equal(rho[:, off[0]:off[0] + P], 0.0)
    assert (rho[:, off[1]:off[1] + P] < 0).all()


def test_fixed_threshold_gate():
    wl = _tiny_traj(seed=10, n_steps=4)
    rho = oracle.tsg_rho(wl.k, wl.frames)
    pool = np.isfinite(rho[0])
    for t in (0.85, -2.0, 2.0):
        tau, gate, _ = oracle.tsg_gate(rho, wl.frames, 5, fixed_tau=t)
        np.testing.assert_array_equal(tau, t)
        for h in range(rho.shape[0]):
            np.testing.assert_array_equal(gate[h][pool], (rho[h][pool] <= t).astype(np.uint8))
            assert (gate[h][~pool] == 1).all()
    # a threshold below every rho closes the whole pool; one above admits it all
    _, g_lo, _ = oracle.tsg_gate(rho, wl.frames, 5, fixed_tau=-2.0)
    _, g_hi, _ = oracle.tsg_gate(rho, wl.frames, 5, fixed_tau=2.0)
    assert (g_lo[:, pool] == 0).all() and (g_hi[:, pool] == 1).all()


def test_uniform_base_prior():
    wl = _tiny_traj(seed=11, n_steps=3)
    out = oracle.compress_layer(wl.q, wl.k, wl.frames, beta=0.3, tsg_enable=0, css_enable=0,
                                base_scorer=oracle.BASE_UNIFORM)
    # every S equal: Top_B is the first B indices (ties by lower index)
    b = out["budget"]
    np.testing.assert_array_equal(out["a"], wl.q.shape[0] / wl.n)
    np.testing.assert_array_equal(out["idx"], np.tile(np.arange(b), (2, 1)))


# ------------------------------------------- hierarchical per-layer budgets

def test_hierarchical_uniform_mass_is_flat():
    # equal S^(l): every layer gets B_total / L (the flat allocation of
    # Sec. 3.3); a remainder goes one token each to the lowest layers
    assert oracle.hierarchical_budgets([2.5] * 28, 28 * 4718, 23592) == [4718] * 28
    assert oracle.hierarchical_budgets([1.0] * 4, 10, 100) == [3, 3, 2, 2]


def test_hierarchical_exact_proportions():
    # shares that are whole numbers come back unchanged
    assert oracle.hierarchical_budgets([1.0, 2.0, 3.0, 4.0], 100, 1000) == [10, 20, 30, 40]
    assert oracle.hierarchical_budgets([3.0, 1.0], 8, 100) == [6, 2]
    # scale invariance of B = S / sum S * B_total
    assert oracle.hierarchical_budgets([0.3, 0.6, 0.9, 1.2], 100, 1000) == [10, 20, 30, 40]


def _cost(b, share):
    return sum((x - s) ** 2 for x, s in zip(b, share))


@pytest.mark.parametrize("seed", range(40))
def test_hierarchical_brute_force_nearest(seed):
    # tiny problems: the oracle's budgets reach the least squared distance to
    # the real shares over every integer vector in [1, N]^L adding to B_total
    rng = np.random.default_rng(1000 + seed)
    n_layers = int(rng.integers(1, 5))
    n_tokens = int(rng.integers(1, 7))
    mass = list(rng.lognormal(0.0, 1.5 if seed % 2 else 0.2, n_layers))
    total = int(rng.integers(n_layers, n_layers * n_tokens + 1))
    b = oracle.hierarchical_budgets(mass, total, n_tokens)
    share = [m / math.fsum(mass) * total for m in mass]
    assert sum(b) == total and all(1 <= x <= n_tokens for x in b)
    best = min(_cost(c, share) for c in itertools.product(range(1, n_tokens + 1), repeat=n_layers)
               if sum(c) == total)
    assert _cost(b, share) <= best + 1e-9


def test_hierarchical_largest_remainder_when_unclamped():
    # away from the [1, N] bounds every budget is the floor or the ceiling of
    # its share, and the ceilings go to the largest fractional parts
    rng = np.random.default_rng(77)
    for _ in range(50):
        n_layers = int(rng.integers(2, 29))
        mass = list(1.0 + 0.05 * rng.standard_normal(n_layers))
        total = int(rng.integers(100 * n_layers, 1000 * n_layers))
        b = oracle.hierarchical_budgets(mass, total, 10 ** 6)
        share = [m / math.fsum(mass) * total for m in mass]
        frac = [s - math.floor(s) for s in share]
        up = [l for l in range(n_layers) if b[l] == math.floor(share[l]) + 1]
        down = [l for l in range(n_layers) if b[l] == math.floor(share[l])]
        assert len(up) + len(down) == n_layers
        if up and down:
            assert min(frac[l] for l in up) >= max(frac[l] for l in down) - 1e-12


def test_hierarchical_deviation_bound():
    # F2 proposition: the budget deviation ratio D = (max B - min B) / mean B
    # equals (max S - min S) / mean S for real budgets and is at most
    # sqrt(2L) CV_S; with L = 28 and CV_S = 1.3 % the bound is 9.7 %.
    # Whole-token budgets move each share by less than one token.
    assert abs(math.sqrt(56) * 0.013 - 0.097) < 5e-4
    rng = np.random.default_rng(12)
    n_layers, n_tokens = 28, 393216
    total = int(0.2 * n_tokens) * n_layers
    for cv in (0.013, 0.05, 0.3):
        mass = 1.0 + cv * rng.standard_normal(n_layers)
        mu = mass.mean()
        cv_s = mass.std() / mu
        b = np.array(oracle.hierarchical_budgets(list(mass), total, n_tokens), dtype=np.float64)
        d_real = (mass.max() - mass.min()) / mu
        d_int = (b.max() - b.min()) / (total / n_layers)
        assert d_real <= math.sqrt(2 * n_layers) * cv_s + 1e-12
        assert abs(d_int - d_real) <= 2.0 / (total / n_layers) + 1e-9


# ------------------------------------- CSS neighbourhood size (5x5 .. 9x9)

def _alt_sum(lo, hi):
    # sum of (-1)^t for t in [lo, hi]
    return sum((-1) ** t for t in range(lo, hi + 1))


@pytest.mark.parametrize("size", [3, 5, 7, 9])
def test_css_size_checkerboard_closed_form(size):
    # keys +-e by the checkerboard: cos = (-1)^(du + dv), so the neighbour sum
    # factorises into two alternating sums over the in-grid offsets, minus
    # the cell itself
    gh, gw, r = 11, 13, size // 2
    k = np.zeros((gh * gw, 1, 4))
    for u in range(gh):
        for v in range(gw):
            k[u * gw + v, 0, 2] = (-1) ** (u + v)
    phi = oracle.css_phi(k, frames_of((0, gh, gw)), size=size)[0].reshape(gh, gw)
    for u in range(gh):
        for v in range(gw):
            du0, du1 = -min(r, u), min(r, gh - 1 - u)
            dv0, dv1 = -min(r, v), min(r, gw - 1 - v)
            cnt = (du1 - du0 + 1) * (dv1 - dv0 + 1) - 1
            expect = 1 - (_alt_sum(du0, du1) * _alt_sum(dv0, dv1) - 1) / cnt
            assert abs(phi[u, v] - expect) < 1e-13, (size, u, v)


@pytest.mark.parametrize("size", [5, 7, 9])
def test_css_size_equal_orthonormal_and_rectangle(size):
    rng = np.random.default_rng(size)
    # equal keys: Phi = 0; distinct basis vectors: Phi = 1
    k = np.repeat(rng.standard_normal((1, 2, 16)), 42, axis=0)
    np.testing.assert_allclose(oracle.css_phi(k, frames_of((0, 6, 7)), size=size), 0.0, atol=1e-13)
    gh, gw, d = 6, 9, 64
    k = np.eye(d)[: gh * gw][:, None, :] * rng.uniform(0.5, 3.0, size=(gh * gw, 1, 1))
    np.testing.assert_allclose(oracle.css_phi(k, frames_of((0, gh, gw)), size=size), 1.0, atol=1e-14)
    # planted 3x4 rectangle of one key on the orthonormal background:
    # Phi = 1 - (#rectangle cells in the window, self excluded) / |N|
    r = np.zeros(d); r[-1] = 1.7
    rect = [(u, v) for u in range(1, 4) for v in range(2, 6)]
    for (u, v) in rect:
        k[u * gw + v, 0] = r
    phi = oracle.css_phi(k, frames_of((0, gh, gw)), size=size)[0].reshape(gh, gw)
    rad = size // 2
    for u in range(gh):
        for v in range(gw):
            nb = [(u + a, v + b) for a in range(-rad, rad + 1) for b in range(-rad, rad + 1)
                  if (a or b) and 0 <= u + a < gh and 0 <= v + b < gw]
            expect = 1 - sum((p in rect) for p in nb) / len(nb) if (u, v) in rect else 1.0
            assert abs(phi[u, v] - expect) < 1e-14, (size, u, v)


def test_css_size_edges():
    rng = np.random.default_rng(9)
    k = rng.standard_normal((20, 1, 8))
    # 1x1 grid: no neighbour at any size
    for size in (5, 9):
        assert oracle.css_phi(k, frames_of((4, 1, 1)), size=size)[0][4] == 0.0
    # a 1x4 strip with a 9x9 kernel: every other cell of the strip is a neighbour
    k2 = np.zeros((4, 1, 2)); k2[:, 0] = [[1, 0], [0, 1], [1, 1], [1, -1]]
    p = oracle.css_phi(k2, frames_of((0, 1, 4)), size=9)[0]
    s = 1 / math.sqrt(2)
    np.testing.assert_allclose(p, [1 - (0 + s + s) / 3, 1 - (0 + s - s) / 3, 1 - (s + s + 0) / 3,
                                   1 - (s - s + 0) / 3], atol=1e-15)
    # size 3 through the size argument is the method's Moore neighbourhood
    np.testing.assert_array_equal(oracle.css_phi(k, frames_of((0, 4, 5)), size=3),
                                  oracle.css_phi(k, frames_of((0, 4, 5))))


# ------------------------------------------------ A_base scaled by its maximum

def test_abase_max_normalisation():
    wl = _tiny_traj(seed=3)
    q, k, fr = wl.q, wl.k, wl.frames
    ref = oracle.compress_layer(q, k, fr, beta=0.3)
    nrm = oracle.compress_layer(q, k, fr, beta=0.3, abase_norm=oracle.ABASE_MAX)
    # every head's largest A becomes exactly 1, the order of A is unchanged
    np.testing.assert_array_equal(nrm["a"].max(axis=1), 1.0)
    for h in range(k.shape[1]):
        np.testing.assert_array_equal(np.argsort(nrm["a"][h], kind="stable"), np.argsort(ref["a"][h], kind="stable"))
    # without CSS and TSG, S = A: a positive scale leaves the kept set alone
    a = oracle.compress_layer(q, k, fr, beta=0.3, tsg_enable=0, css_enable=0)
    b = oracle.compress_layer(q, k, fr, beta=0.3, tsg_enable=0, css_enable=0, abase_norm=oracle.ABASE_MAX)
    np.testing.assert_array_equal(a["idx"], b["idx"])
    # equal keys: A is uniform, so A / max A = 1 and S = 1 for every token
    # (CSS and TSG off): the first B tokens by index
    kk = np.repeat(k[:1], k.shape[0], axis=0)
    u = oracle.compress_layer(q, kk, fr, beta=0.3, tsg_enable=0, css_enable=0, abase_norm=oracle.ABASE_MAX)
    np.testing.assert_array_equal(u["s"], 1.0)
    np.testing.assert_array_equal(u["idx"], np.tile(np.arange(u["budget"]), (k.shape[1], 1)))


# ------------------------------------------- task splits of the oracle drivers

@pytest.mark.parametrize("threads", [1, 3])
def test_abase_task_split_matches_single_pass(threads):
    # Eq. 2 (reading R1): the per-query-head partials summed per group equal
    # the group accumulated in one pass, whatever the thread count; the two
    # differ only in the order of the fp64 additions.
    wl = synth.scaled("long", 2, beta=0.1)
    q, k = wl.q[:, :8].astype(np.float64), wl.k[:2000, :1].astype(np.float64)
    a1 = oracle.abase(q, k, threads=threads)
    a2 = oracle.abase_per_head(q, k)
    np.testing.assert_allclose(a1, a2, rtol=1e-12, atol=0)
    np.testing.assert_allclose(a1.sum(1), q.shape[0], rtol=1e-12)


@pytest.mark.parametrize("threads,chunk", [(1, 2048), (4, 97), (3, 1)])
def test_rho_task_split_matches_single_pass(threads, chunk):
    # Eq. 6: the pool cut into token runs (ragged last run, one-token runs)
    # gives exactly the per-head pass's values, NaN outside the pool.
    wl = synth.scaled("traj50", 3)
    k = wl.k.astype(np.float64)
    r1 = oracle.tsg_rho(k, wl.frames, threads=threads, chunk=chunk)
    r2 = oracle.tsg_rho_per_head(k, wl.frames)
    np.testing.assert_array_equal(np.isnan(r1), np.isnan(r2))
    np.testing.assert_array_equal(r1[~np.isnan(r1)], r2[~np.isnan(r2)])
    for metric in (oracle.TSG_DOT, oracle.TSG_NEG_L2):
        np.testing.assert_array_equal(
            np.nan_to_num(oracle.tsg_rho(k, wl.frames, threads=threads, chunk=chunk, metric=metric), nan=7.0),
            np.nan_to_num(oracle.tsg_rho_per_head(k, wl.frames, metric=metric), nan=7.0))


# ------------------------------- prompt-wide base scores (base-scoring ablation)

@pytest.mark.parametrize("n,n_q", [(9, 9), (12, 5), (7, 1)])
def test_prompt_equal_keys_harmonic(n, n_q):
    # Mean Attention / full-attention bases (appendix on the base scoring
    # function), causal reading R18: with every key equal, prompt row r (at
    # position p = n - n_q + r) spreads 1/(p+1) over keys 0..p, so the full
    # base is C_j = sum_{p >= max(j, n - n_q)} 1/(p + 1) (harmonic numbers)
    # and the mean base divides by the rows that see j.  A flipped mask or a
    # missing 1/G would change both.
    rng = np.random.default_rng(5)
    d, hq, hkv = 8, 4, 2
    q = rng.standard_normal((n_q, hq, d))
    k = np.ones((n, hkv, d))
    full = oracle.prompt_abase(q, k, oracle.PROMPT_FULL)
    mean = oracle.prompt_abase(q, k, oracle.PROMPT_MEAN)
    for j in range(n):
        c = sum(1.0 / (p + 1) for p in range(max(j, n - n_q), n))
        cnt = min(n_q, n - j)
        np.testing.assert_allclose(full[:, j], c, rtol=1e-13)
        np.testing.assert_allclose(mean[:, j], c / cnt, rtol=1e-13)


def test_prompt_single_row_is_textbook_softmax():
    # n_q = 1: the last position sees every key, so the full base is one
    # softmax row: q = e_0, k_j = sqrt(d) x_j e_0 gives softmax(x).
    d, n = 16, 6
    x = np.array([0.5, -2.0, 1.5, 0.25, -0.75, 3.0])
    q = np.zeros((1, 1, d)); q[0, 0, 0] = 1.0
    k = np.zeros((n, 1, d)); k[:, 0, 0] = math.sqrt(d) * x
    z = sum(math.exp(t) for t in x)
    want = [math.exp(t) / z for t in x]
    np.testing.assert_allclose(oracle.prompt_abase(q, k, oracle.PROMPT_FULL)[0], want, rtol=1e-13)
    np.testing.assert_allclose(oracle.prompt_abase(q, k, oracle.PROMPT_MEAN)[0], want, rtol=1e-13)


def test_prompt_dominant_key_sees_only_later_rows():
    # a key with an overwhelming logit takes all the mass of every row at or
    # after its position and none of the rows before it (causality): its full
    # base is the number of rows that see it and its mean base is 1.
    d, n = 8, 10
    q = np.zeros((n, 1, d)); q[:, 0, 0] = 1.0
    k = np.zeros((n, 1, d)); k[:, 0, 1] = 1.0
    js = 4
    k[js, 0, 0] = 400.0 * math.sqrt(d)
    full = oracle.prompt_abase(q, k, oracle.PROMPT_FULL)[0]
    mean = oracle.prompt_abase(q, k, oracle.PROMPT_MEAN)[0]
    np.testing.assert_allclose(full[js], n - js, rtol=1e-12)
    np.testing.assert_allclose(mean[js], 1.0, rtol=1e-12)
    # rows before js see keys 0..p uniformly (all logits 0 there)
    for j in range(js):
        np.testing.assert_allclose(full[j], sum(1.0 / (p + 1) for p in range(j, js)), rtol=1e-12)
    np.testing.assert_allclose(full[js + 1:], 0.0, atol=1e-100)


def test_prompt_mass_and_library_softmax():
    # every prompt row's probabilities sum to one (sum_j C_j = n_q), and the
    # full base equals torch's softmax over causally masked logits, summed
    # over rows and averaged over the group's query heads
    import torch
    rng = np.random.default_rng(11)
    n, n_q, hq, hkv, d = 40, 23, 6, 2, 16
    q = rng.standard_normal((n_q, hq, d))
    k = rng.standard_normal((n, hkv, d))
    full = oracle.prompt_abase(q, k, oracle.PROMPT_FULL, threads=3)
    mean = oracle.prompt_abase(q, k, oracle.PROMPT_MEAN)
    np.testing.assert_allclose(full.sum(1), n_q, rtol=1e-12)
    cnt = np.minimum(n_q, n - np.arange(n))
    np.testing.assert_allclose((mean * cnt).sum(1), n_q, rtol=1e-12)
    G = hq // hkv
    qt, kt = torch.from_numpy(q), torch.from_numpy(k)
    pos = torch.arange(n - n_q, n)[:, None]
    mask = torch.arange(n)[None, :] > pos                      # [n_q, n]
    for h in range(hkv):
        acc = torch.zeros(n, dtype=torch.float64)
        for g in range(h * G, (h + 1) * G):
            logits = qt[:, g] @ kt[:, h].T / math.sqrt(d)
            acc += torch.softmax(logits.masked_fill(mask, float("-inf")), dim=1).sum(0)
        np.testing.assert_allclose(full[h], (acc / G).numpy(), rtol=1e-12, atol=1e-15)


def test_prompt_gqa_grouping():
    # only the owning KV head's keys move its scores
    rng = np.random.default_rng(2)
    n, hq, hkv, d = 15, 6, 3, 8
    q = rng.standard_normal((n, hq, d))
    k = rng.standard_normal((n, hkv, d))
    a = oracle.prompt_abase(q, k, oracle.PROMPT_MEAN)
    k2 = k.copy()
    k2[:, 1] = rng.standard_normal((n, d))
    b = oracle.prompt_abase(q, k2, oracle.PROMPT_MEAN)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[2], b[2])
    assert not np.allclose(a[1], b[1])
