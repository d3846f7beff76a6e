"""C-ABI library checks that need no GPU: the library builds and loads, it
exports every symbol ``include/stlite.h`` declares, and the host-side
validation rejects malformed calls before anything is enqueued."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2603_00188_gb300 import build as pkg_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def st():
    pkg_build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


@pytest.fixture(scope="module")
def good():
    """A 16-byte-aligned address the rejection tests pass where a tensor is
    expected: a real 32 MiB device allocation (larger than any buffer these
    shapes describe) when a CUDA device is present, so that no unmapped
    address could reach a kernel even if a host check regressed; without a
    device, where nothing can launch, a stand-in value."""
    import torch
    if torch.cuda.is_available():
        buf = torch.zeros(32 << 20, dtype=torch.uint8, device="cuda")
        yield buf.data_ptr()
        del buf
    else:
        yield 0x10000


def header_functions():
    text = open(os.path.join(ROOT, "include", "stlite.h")).read()
    return sorted(set(re.findall(r"STLITE_API\s+[\w\s\*]+?\b(stlite_\w+)\s*\(", text)))


def test_exports_match_header(st):
    declared = header_functions()
    assert len(declared) >= 10
    assert sorted(st.EXPORTED) == declared
    lib = ctypes.CDLL(st._LIB_PATH)
    for name in declared:
        assert hasattr(lib, name), name


@pytest.mark.parametrize("n,beta,ko", [(1152, 0.2, 0), (23680, 0.1, 0), (23680, 0.3, 0), (53600, 0.2, 0),
                                       (132800, 0.1, 0), (10, 1.0, 0), (10, 0.01, 0), (1152, 0.2, 231),
                                       (5, 0.2, 99), (7, 0.5, 0)])
def test_budget_matches_oracle(st, n, beta, ko):
    assert st.stlite_budget(n, beta, ko) == oracle.budget(n, beta, ko)


def test_budget_rejects(st):
    assert st.stlite_budget(0, 0.2, 0) == -1
    assert st.stlite_budget(10, 0.0, 0) == -1
    assert st.stlite_budget(10, 1.5, 0) == -1


def test_status_strings(st):
    for s in range(6):
        assert st._lib.stlite_status_string(s)
    assert st._lib.stlite_status_string(1).decode() == "invalid argument"


def _shape(st, n=100, hq=4, hkv=2, d=128, w=4, dt=0):
    return st.Shape(n, hq, hkv, d, w, dt)


def test_workspace_size_and_validation(st):
    fr = st.FrameSpec([0, 30], [4, 5], [5, 6])
    assert st.stlite_workspace_size(_shape(st), fr) > 0
    bad = [
        (_shape(st, hq=5), fr, st.STLITE_EINVAL),                 # Hq % Hkv
        (_shape(st, d=64), fr, st.STLITE_EUNSUPPORTED),           # head_dim
        (_shape(st, w=0), fr, st.STLITE_EINVAL),
        (_shape(st, w=300), fr, st.STLITE_EUNSUPPORTED),
        (_shape(st, dt=7), fr, st.STLITE_EINVAL),
        (_shape(st), st.FrameSpec([0, 10], [4, 5], [5, 6]), st.STLITE_EINVAL),   # overlap
        (_shape(st), st.FrameSpec([30, 0], [4, 5], [5, 6]), st.STLITE_EINVAL),   # unsorted
        (_shape(st), st.FrameSpec([0, 90], [4, 5], [5, 6]), st.STLITE_EINVAL),   # past N
        (_shape(st), st.FrameSpec([0], [0], [5]), st.STLITE_EINVAL),             # empty grid
        (_shape(st), st.FrameSpec(np.zeros(257), np.ones(257), np.ones(257)), st.STLITE_EUNSUPPORTED),
    ]
    for sh, f, code in bad:
        with pytest.raises(st.StliteError) as e:
            st.stlite_workspace_size(sh, f)
        assert e.value.status == code


def test_entry_points_reject_before_launch(st, good):
    """Malformed pointers and sizes are refused on the host (no GPU needed)."""
    lib = st._lib
    sh = _shape(st)
    fr = st.FrameSpec([0, 30], [4, 5], [5, 6])
    prm = st.make_params(0.2)
    need = st.stlite_workspace_size(sh, fr, prm)
    P = ctypes.c_void_p
    mis = P(good + 8)          # not 16-byte aligned
    good = P(good)
    assert lib.stlite_score(ctypes.byref(sh), None, good, good, good, need, None) == st.STLITE_EINVAL
    assert lib.stlite_score(ctypes.byref(sh), mis, good, good, good, need, None) == st.STLITE_EINVAL
    # stlite_score takes no frames: its workspace is the frame-less size
    need_score = st.stlite_workspace_size(sh, st.FrameSpec([], [], []), prm)
    assert lib.stlite_score(ctypes.byref(sh), good, good, good, good, need_score - 1, None) == st.STLITE_EWORKSPACE
    assert lib.stlite_gate_frames(ctypes.byref(sh), ctypes.byref(fr.c), good, 0, good, good, good, good,
                                  need, None) == st.STLITE_EINVAL
    bad_prm = st.make_params(beta=0.0)
    assert lib.stlite_compress_layer(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(bad_prm), good, good,
                                     good, good, good, good, None, good, need, None) == st.STLITE_EINVAL
    neg_alpha = st.make_params(alpha=-1.0)
    assert lib.stlite_select_topk(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(neg_alpha), good, good,
                                  None, 5, good, None, good, need, None) == st.STLITE_EINVAL
    assert lib.stlite_compact(ctypes.byref(sh), 0, good, good, good, good, good, None) == st.STLITE_EINVAL
    assert lib.stlite_compact(ctypes.byref(sh), 101, good, good, good, good, good, None) == st.STLITE_EINVAL
    assert lib.stlite_device_status(None, None, None) == st.STLITE_EINVAL


def test_varlen_validation(st):
    """stlite_compress_varlen / stlite_workspace_size_varlen reject malformed
    packed batches on the host (no GPU needed)."""
    sh = _shape(st, n=300, hq=4, hkv=2, w=4)
    fr = [st.FrameSpec([0], [5], [8]), st.FrameSpec([10], [4], [6]), st.FrameSpec([], [], [])]
    prm = st.make_params(0.2)
    ok = st.stlite_workspace_size_varlen(sh, [0, 100, 200, 300], fr, prm)
    assert ok > 0
    # the largest sequence sets the size
    assert ok == max(st.stlite_workspace_size(_shape(st, n=100, hq=4, hkv=2, w=4), f, prm) for f in fr)
    for cu in ([0, 100, 200, 299], [1, 100, 200, 300], [0, 100, 100, 300], [0, 200, 100, 300]):
        with pytest.raises(st.StliteError):
            st.stlite_workspace_size_varlen(sh, cu, fr, prm)
    # a frame outside its own sequence
    bad = [st.FrameSpec([0], [10], [11]), fr[1], fr[2]]
    with pytest.raises(st.StliteError):
        st.stlite_workspace_size_varlen(sh, [0, 100, 200, 300], bad, prm)


def _mass_cases():
    rng = np.random.default_rng(31)
    cases = [([1.0, 2.0, 3.0, 4.0], 100, 1000), ([1.0] * 28, 28 * 4718, 23592), ([5.0, 1.0, 1.0], 10, 4),
             ([1e-9, 1.0, 1.0, 1e-9], 9, 5), ([1.0] * 3, 7, 3), ([100.0, 1.0], 2, 1)]
    for _ in range(200):
        n_layers = int(rng.integers(1, 33))
        n_tokens = int(rng.integers(1, 2000))
        kind = rng.integers(0, 3)
        if kind == 0:  # near-uniform: the paper's GUI regime (CV about 1%)
            mass = 1.0 + 0.013 * rng.standard_normal(n_layers)
        elif kind == 1:  # pyramid-shaped, shallow layers heavier
            mass = np.linspace(3.0, 0.5, n_layers) * rng.uniform(0.9, 1.1, n_layers)
        else:  # heavy-tailed: forces clamping at 1 and at N
            mass = rng.lognormal(0.0, 3.0, n_layers)
        total = int(rng.integers(n_layers, n_layers * n_tokens + 1))
        cases.append((list(mass), total, n_tokens))
    return cases


def test_hierarchical_budgets_match_oracle(st):
    """The host helper reaches the oracle's integer budgets exactly."""
    for mass, total, n_tokens in _mass_cases():
        got = st.stlite_hierarchical_budgets(mass, total, n_tokens)
        assert got == oracle.hierarchical_budgets(mass, total, n_tokens), (mass, total, n_tokens)
        assert sum(got) == total and min(got) >= 1 and max(got) <= n_tokens


def test_hierarchical_budgets_reject(st):
    for mass, total, n_tokens in [([], 4, 10), ([1.0, 0.0], 4, 10), ([1.0, -1.0], 4, 10),
                                  ([1.0, float("nan")], 4, 10), ([1.0, float("inf")], 4, 10),
                                  ([1.0, 1.0], 1, 10), ([1.0, 1.0], 21, 10), ([1.0], 1, 0),
                                  ([1e308, 1e308], 4, 10)]:
        with pytest.raises(st.StliteError):
            st.stlite_hierarchical_budgets(mass, total, n_tokens)


def test_compress_layers_budgets_reject_before_launch(st, good):
    """Per-layer budgets outside [1, N] and NULL arrays are refused on the host."""
    lib = st._lib
    sh = _shape(st)
    fr = st.FrameSpec([0, 30], [4, 5], [5, 6])
    prm = st.make_params(0.2)
    need = st.stlite_workspace_size(sh, fr, prm)
    lay = (st.LayerIO * 2)(st.LayerIO(*([good] * 6)), st.LayerIO(*([good] * 6)))
    P = ctypes.c_void_p
    for bud in ([20, 0], [20, 101], [-1, 20]):
        arr = (ctypes.c_int32 * 2)(*bud)
        assert lib.stlite_compress_layers_budgets(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(prm), 2, lay,
                                                  arr, P(good), 2 * need, None) == st.STLITE_EINVAL
    arr = (ctypes.c_int32 * 2)(20, 30)
    assert lib.stlite_compress_layers_budgets(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(prm), 2, lay,
                                              None, P(good), 2 * need, None) == st.STLITE_EINVAL
    assert lib.stlite_compress_layers_budgets(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(prm), 2, lay,
                                              arr, P(good), 2 * need - 1, None) == st.STLITE_EWORKSPACE
    bad = (st.LayerIO * 2)(st.LayerIO(*([good] * 6)), st.LayerIO(*([good] * 5 + [good + 8])))
    assert lib.stlite_compress_layers_budgets(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(prm), 2, bad,
                                              arr, P(good), 2 * need, None) == st.STLITE_EINVAL


def test_variant_params_validation(st, good):
    """CSS sizes other than 0/3/5/7/9 and unknown A_base scalings are refused
    on the host, in the fused and in the staged entry points."""
    lib = st._lib
    sh = _shape(st)
    fr = st.FrameSpec([0, 30], [4, 5], [5, 6])
    need = st.stlite_workspace_size(sh, fr, st.make_params(0.2))
    good = ctypes.c_void_p(good)
    for kw in (dict(css_size=4), dict(css_size=11), dict(css_size=-3), dict(abase_norm=2), dict(abase_norm=-1)):
        prm = st.make_params(0.2, **kw)
        assert lib.stlite_compress_layer(ctypes.byref(sh), ctypes.byref(fr.c), ctypes.byref(prm), good, good, good,
                                         good, good, good, None, good, need, None) == st.STLITE_EINVAL, kw
    for size in (0, 1, 4, 11):
        assert lib.stlite_spatial_saliency_size(ctypes.byref(sh), ctypes.byref(fr.c), good, size, good, good, need,
                                                None) == st.STLITE_EINVAL
    assert lib.stlite_spatial_saliency_size(ctypes.byref(sh), ctypes.byref(fr.c), good, 5, good, good, need - 1,
                                            None) == st.STLITE_EWORKSPACE
    for size in (0, 3, 5, 7, 9):
        assert st.stlite_workspace_size(sh, fr, st.make_params(0.2, css_size=size, abase_norm=1)) == need


def test_varlen_layers_validation(st, good):
    """stlite_compress_varlen_layers refuses a short workspace and malformed
    layer arrays on the host."""
    lib = st._lib
    sh = _shape(st, n=300, hq=4, hkv=2, w=4)
    fr = [st.FrameSpec([0], [5], [8]), st.FrameSpec([10], [4], [6]), st.FrameSpec([], [], [])]
    prm = st.make_params(0.2)
    need = st.stlite_workspace_size_varlen(sh, [0, 100, 200, 300], fr, prm)
    cu, specs, arr = st._varlen_args([0, 100, 200, 300], fr)
    ip = ctypes.POINTER(ctypes.c_int32)
    lay = (st.LayerIO * 2)(st.LayerIO(*([good] * 6)), st.LayerIO(*([good] * 6)))
    call = lambda layers, n, ws_bytes: lib.stlite_compress_varlen_layers(
        ctypes.byref(sh), 3, cu.ctypes.data_as(ip), arr, ctypes.byref(prm), n, layers, None,
        ctypes.c_void_p(good), ws_bytes, None)
    assert call(lay, 2, 2 * need - 1) == st.STLITE_EWORKSPACE
    assert call(None, 2, 2 * need) == st.STLITE_EINVAL
    assert call(lay, 0, 2 * need) == st.STLITE_EINVAL
    bad = (st.LayerIO * 2)(st.LayerIO(*([good] * 6)), st.LayerIO(*([good] * 5 + [0])))
    assert call(bad, 2, 2 * need) == st.STLITE_EINVAL


NOALLOC_SCRATCH = 2 << 20


def _noalloc_need(hkv, r, splits):
    return 256 + hkv * splits * r * 8 + hkv * r * 4


@pytest.mark.parametrize("n,hq,hkv,w,dt", [
    (53600, 28, 4, 32, 0), (132800, 28, 4, 64, 0), (20960, 12, 2, 16, 0), (1152, 28, 4, 32, 1),
    (5000, 400, 400, 1, 1), (5000, 400, 400, 1, 0), (100000, 64, 64, 8, 1), (100000, 64, 64, 8, 0),
    (100000, 256, 16, 32, 1), (100000, 256, 16, 32, 0), (300, 8, 1, 64, 1), (64, 4096, 1024, 128, 0),
    (64, 4096, 1024, 128, 1), (5000, 1024, 1024, 1, 1), (100000, 1024, 512, 1, 0)])
def test_noalloc_scratch_bound(st, n, hq, hkv, w, dt):
    """The no-workspace window score's capacity rule, checked on the host: a
    shape whose scratch fits in the fixed 2 MiB even with the documented
    largest split count, S = max(4, 4 ceil(304 / Hkv)), passes the capacity
    check (and then fails only on the NULL pointers given here); a shape that
    does not fit even with one split is refused as unsupported.  Nothing can
    launch: the pointers are NULL."""
    sh = st.Shape(n, hq, hkv, 128, w, dt)
    r = w * (hq // hkv)
    s_max = max(4, 4 * (-(-304 // hkv)))
    got = st._lib.stlite_score_noalloc(ctypes.byref(sh), None, None, None, None)
    if _noalloc_need(hkv, r, s_max) <= NOALLOC_SCRATCH:
        assert got == st.STLITE_EINVAL
    elif _noalloc_need(hkv, r, 1) > NOALLOC_SCRATCH:
        assert got == st.STLITE_EUNSUPPORTED
    else:
        assert got in (st.STLITE_EINVAL, st.STLITE_EUNSUPPORTED)


def test_noalloc_shape_limits_match_score(st):
    """stlite_score_noalloc applies the same shape limits as stlite_score
    (both refuse before looking at any pointer)."""
    for sh, code in [(st.Shape(100, 5, 2, 128, 4, 0), st.STLITE_EINVAL),
                     (st.Shape(100, 4, 2, 64, 4, 0), st.STLITE_EUNSUPPORTED),
                     (st.Shape(100, 4, 2, 128, 300, 0), st.STLITE_EUNSUPPORTED),
                     (st.Shape(100, 4 * 5000, 5000, 128, 1, 1), st.STLITE_EUNSUPPORTED),
                     (st.Shape(1 << 29, 4, 4, 128, 1, 1), st.STLITE_EUNSUPPORTED),
                     (st.Shape(0, 4, 2, 128, 4, 0), st.STLITE_EINVAL)]:
        assert st._lib.stlite_score_noalloc(ctypes.byref(sh), None, None, None, None) == code
        assert st._lib.stlite_score(ctypes.byref(sh), None, None, None, None, 0, None) == code


def test_device_status_without_scratch_argument(st, good):
    """stlite_device_status(NULL, ...) reads the no-workspace scratch; a NULL
    status pointer or a misaligned workspace is refused on the host."""
    lib = st._lib
    assert lib.stlite_device_status(None, None, None) == st.STLITE_EINVAL
    status = ctypes.c_int32(0)
    assert lib.stlite_device_status(ctypes.c_void_p(good + 8), None, ctypes.byref(status)) == st.STLITE_EINVAL


def test_selftest_validation_on_host(st, good):
    """The failure-path diagnostic refuses a NULL or misaligned error word and
    limits outside 1 us .. 2 s before launching anything."""
    lib = st._lib
    assert lib.stlite_selftest_wait_timeout(None, 10_000_000, None) == st.STLITE_EINVAL
    assert lib.stlite_selftest_wait_timeout(ctypes.c_void_p(good + 8), 10_000_000, None) == st.STLITE_EINVAL
    for limit in (0, 999, 2_000_000_001):
        assert lib.stlite_selftest_wait_timeout(ctypes.c_void_p(good), limit, None) == st.STLITE_EINVAL
