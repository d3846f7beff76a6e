"""ST-Lite reference oracle -- TEST INFRASTRUCTURE ONLY.

Thin ctypes wrapper around ``stlite_oracle.c``: a plain, slow, fp64 CPU
restatement of the ST-Lite compression procedure (Algorithm 1 of arXiv
2603.00188; Eqs. 2, 4-9).  Only the test suite, the package smoke check and
the benchmark's CPU-baseline leg may import this module.  It shares no code
with the CUDA library and never imports it.

Arrays: ``q`` [w, Hq, d] and ``k`` [N, Hkv, d] as float64 (exact copies of the
bf16/fp32 inputs).  Frames are three int32 arrays (offset, grid_h, grid_w);
the last frame is the current frame.  Per-head results are [Hkv, N].

Every function here is pinned by ``tests/test_oracle_pins.py`` to closed
forms, invariants, hand-computed fixtures (``tests/golden/``) and brute force.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "stlite_oracle.c")
_SO = os.path.join(_HERE, "libstlite_oracle.so")
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int32)
_bp = ctypes.POINTER(ctypes.c_uint8)
_i32 = ctypes.c_int32


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain -O2, IEEE semantics kept)."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_SO)
        lib.orc_budget.restype = _i32
        lib.orc_budget.argtypes = [_i32, ctypes.c_double, _i32]
        lib.orc_abase.restype = None
        lib.orc_abase.argtypes = [_dp, _dp, _i32, _i32, _i32, _i32, _i32, _i32, _dp]
        lib.orc_abase_qhead.restype = None
        lib.orc_abase_qhead.argtypes = [_dp, _dp, _i32, _i32, _i32, _i32, _i32, _i32, _dp]
        lib.orc_prompt_qhead.restype = None
        lib.orc_prompt_qhead.argtypes = [_dp, _dp, _i32, _i32, _i32, _i32, _i32, _i32, _dp]
        lib.orc_tsg_rho_tokens.restype = None
        lib.orc_tsg_rho_tokens.argtypes = [_dp, _i32, _i32, _i32, _ip, _i32, _i32, _i32, _i32, _dp]
        lib.orc_css_phi_token.restype = ctypes.c_double
        lib.orc_css_phi_token.argtypes = [_dp, _i32, _i32, _i32, _i32, _i32, _i32, _i32, _i32, _i32]
        lib.orc_css_phi.restype = None
        lib.orc_css_phi.argtypes = [_dp, _i32, _i32, _i32, _i32, _i32, _ip, _ip, _ip, _i32, _dp]
        lib.orc_tsg_rho_token.restype = ctypes.c_double
        lib.orc_tsg_rho_token.argtypes = [_dp, _i32, _i32, _i32, _i32, _i32, _i32, _i32]
        lib.orc_tsg_rho.restype = None
        lib.orc_tsg_rho.argtypes = [_dp, _i32, _i32, _i32, _i32, _i32, _ip, _ip, _ip, _i32, _dp]
        lib.orc_tsg_gate.restype = _i32
        lib.orc_tsg_gate.argtypes = [_dp, _i32, _i32, _ip, _ip, _ip, _i32, _i32, _i32, ctypes.c_double, _dp, _bp]
        lib.orc_combine.restype = None
        lib.orc_combine.argtypes = [_dp, _dp, _bp, _i32, _i32, _ip, _ip, _ip, ctypes.c_double, _i32, _dp]
        lib.orc_topk.restype = None
        lib.orc_topk.argtypes = [_dp, _i32, _i32, _ip]
        lib.orc_gather.restype = None
        lib.orc_gather.argtypes = [_bp, _bp, _i32, _i32, _i32, _i32, _ip, _i32, _bp, _bp]
        lib.orc_decode_row.argtypes = [_dp, _dp, _dp, _i32, _i32, _i32, _i32, _i32, _i32, _dp]
        _lib = lib
    return _lib


def _d(a):
    return a.ctypes.data_as(_dp)


def _c64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _frames(frames):
    off, gh, gw = (np.ascontiguousarray(x, dtype=np.int32) for x in frames)
    assert off.shape == gh.shape == gw.shape
    return off, gh, gw


def _per_head(fn, hkv, threads):
    _run_tasks(fn, list(range(hkv)), threads)


def _run_tasks(fn, tasks, threads):
    """Runs fn on every task, on `threads` threads (the C calls release the
    GIL); each task writes its own slice of the output, so the result does
    not depend on the thread count."""
    if threads and threads > 1 and len(tasks) > 1:
        with ThreadPoolExecutor(max_workers=min(threads, len(tasks))) as ex:
            list(ex.map(fn, tasks))
    else:
        for t in tasks:
            fn(t)


def host_threads() -> int:
    """Threads this process may run on (its CPU affinity)."""
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


def budget(n: int, beta: float, k_override: int = 0) -> int:
    """B = floor(beta * N) (Sec. 2.1), >= 1; k_override > 0 replaces it."""
    return int(_load().orc_budget(int(n), float(beta), int(k_override)))


def hierarchical_budgets(layer_mass, total_budget: int, n_tokens: int) -> list:
    """Hierarchical allocation of the F2 proposition (appendix "Failure Mode
    Derivations"): layer l gets the real share B^(l) = S^(l) / sum S * B_total.
    Budgets must be whole tokens in [1, N] adding up to B_total; the reading
    taken is the integer vector nearest to the shares in squared distance
    (ties to the lower layer), found by single-token moves from the clamped
    floors, which is exact for a separable convex objective."""
    mass = [float(x) for x in layer_mass]
    n_layers = len(mass)
    tot = 0.0
    for m in mass:  # left to right, no compensated summation
        tot += m
    share = [m / tot * float(total_budget) for m in mass]
    b = [min(max(int(np.floor(x)), 1), int(n_tokens)) for x in share]
    while sum(b) < total_budget:
        room = [l for l in range(n_layers) if b[l] < n_tokens]
        l = max(room, key=lambda i: share[i] - b[i])
        b[l] += 1
    while sum(b) > total_budget:
        room = [l for l in range(n_layers) if b[l] > 1]
        l = max(room, key=lambda i: b[i] - share[i])
        b[l] -= 1
    return b


def abase(q, k, threads: int = 1) -> np.ndarray:
    """Eq. 2 window score per KV head (mean over the G query heads of a group):
    each query head's sum over the window rows of its softmax rows is one
    task (``orc_abase_qhead``), and A[h] = (1/G) * the sum of its group's
    partials in query-head order."""
    lib = _load()
    q, k = _c64(q), _c64(k)
    w, hq, d = q.shape
    n, hkv, d2 = k.shape
    assert d == d2 and hq % hkv == 0
    G = hq // hkv
    part = np.zeros((hq, n), dtype=np.float64)

    def run(g):
        lib.orc_abase_qhead(_d(q), _d(k), n, w, hq, hkv, d, g, part[g].ctypes.data_as(_dp))

    _run_tasks(run, list(range(hq)), threads)
    out = np.zeros((hkv, n), dtype=np.float64)
    for h in range(hkv):
        for g in range(h * G, (h + 1) * G):
            out[h] += part[g]
        out[h] /= G
    return out


def abase_per_head(q, k) -> np.ndarray:
    """Eq. 2 computed head by head in one pass (``orc_abase``: the G query
    heads and w rows of a group accumulated into A directly); the same
    quantity as ``abase``, kept as a cross-check of its task split."""
    lib = _load()
    q, k = _c64(q), _c64(k)
    w, hq, d = q.shape
    n, hkv, d2 = k.shape
    out = np.zeros((hkv, n), dtype=np.float64)
    for h in range(hkv):
        lib.orc_abase(_d(q), _d(k), n, w, hq, hkv, d, h, out[h].ctypes.data_as(_dp))
    return out


PROMPT_FULL, PROMPT_MEAN = 0, 1


def prompt_abase(q_prompt, k, mode: int = PROMPT_MEAN, threads: int = 1) -> np.ndarray:
    """Prompt-wide base scores of the base-scoring ablation (appendix
    "Sensitivity to the Base Attention Scoring Function").  q_prompt
    [n_q, Hq, d] are the query rows of the last n_q cached positions, each
    attending causally (keys up to its own position).  PROMPT_FULL (the
    full-attention "snapshot" base): A[h][j] = (1/G) sum over the group's query
    heads and every prompt row of its softmax probability of key j.
    PROMPT_MEAN (Mean Attention, 1D average pooling over the prompt): the same
    sum divided by the number of prompt rows that attend to j."""
    lib = _load()
    q, k = _c64(q_prompt), _c64(k)
    n_q, hq, d = q.shape
    n, hkv, d2 = k.shape
    assert d == d2 and hq % hkv == 0 and 1 <= n_q <= n
    G = hq // hkv
    part = np.zeros((hq, n), dtype=np.float64)

    def run(g):
        lib.orc_prompt_qhead(_d(q), _d(k), n, n_q, hq, hkv, d, g, part[g].ctypes.data_as(_dp))

    _run_tasks(run, list(range(hq)), threads)
    out = np.zeros((hkv, n), dtype=np.float64)
    for h in range(hkv):
        for g in range(h * G, (h + 1) * G):
            out[h] += part[g]
        out[h] /= G
    if mode == PROMPT_MEAN:
        j = np.arange(n)
        count = np.minimum(n_q, n - j).astype(np.float64)   # rows r with n - n_q + r >= j
        out /= count[None, :]
    return out


def css_phi(k, frames, threads: int = 1, size: int = 3) -> np.ndarray:
    """Eqs. 4-5: Phi = 1 - mean neighbour cosine over the in-grid cells of the
    size x size neighbourhood (3: the Moore neighbourhood of the method; 5, 7,
    9: the neighbourhood-size ablation); NaN for text tokens."""
    assert size in (3, 5, 7, 9)
    lib = _load()
    k = _c64(k)
    n, hkv, d = k.shape
    off, gh, gw = _frames(frames)
    out = np.zeros((hkv, n), dtype=np.float64)

    def run(h):
        lib.orc_css_phi(_d(k), n, hkv, d, h, len(off), off.ctypes.data_as(_ip),
                        gh.ctypes.data_as(_ip), gw.ctypes.data_as(_ip), size // 2, out[h].ctypes.data_as(_dp))

    _per_head(run, hkv, threads)
    return out


def css_phi_token(k, h: int, off: int, gh: int, gw: int, u: int, v: int, size: int = 3) -> float:
    """Phi of the single visual token (u, v) of the frame at ``off``."""
    assert size in (3, 5, 7, 9)
    k = _c64(k)
    n, hkv, d = k.shape
    return float(_load().orc_css_phi_token(_d(k), hkv, d, h, off, gh, gw, u, v, size // 2))


TSG_COSINE, TSG_DOT, TSG_NEG_L2 = 0, 1, 2


def pool_tokens(frames) -> np.ndarray:
    """The historical pool T_pool: the visual tokens of frames 0..F-2, ascending."""
    off, gh, gw = _frames(frames)
    if len(off) < 2:
        return np.zeros(0, np.int32)
    return np.concatenate([np.arange(o, o + a * b, dtype=np.int32) for o, a, b in
                           zip(off[:-1], gh[:-1], gw[:-1])])


def tsg_rho(k, frames, threads: int = 1, metric: int = TSG_COSINE, chunk: int = 2048,
            tokens=None) -> np.ndarray:
    """Eq. 6: rho_i = max similarity to the current frame (cosine; or, for the
    similarity-metric ablation, dot product / negative squared L2 distance);
    NaN outside the pool.  The pool (visual tokens of frames 0..F-2) is cut
    into runs of `chunk` tokens per KV head, one task each
    (``orc_tsg_rho_tokens``), so that every host core can take part.
    ``tokens`` (a subset of the pool) restricts the computation to those
    tokens; every other entry is NaN."""
    lib = _load()
    k = _c64(k)
    n, hkv, d = k.shape
    off, gh, gw = _frames(frames)
    out = np.full((hkv, n), np.nan, dtype=np.float64)
    if len(off) < 2:
        return out
    pool = pool_tokens(frames)
    if tokens is not None:
        tokens = np.asarray(tokens, dtype=np.int32)
        assert np.isin(tokens, pool).all(), "tokens outside the historical pool"
        pool = tokens
    cur_off, cur_len = int(off[-1]), int(gh[-1] * gw[-1])
    tasks = [(h, c) for h in range(hkv) for c in range(0, len(pool), chunk)]

    def run(t):
        h, c = t
        tok = np.ascontiguousarray(pool[c:c + chunk])
        vals = np.zeros(len(tok), dtype=np.float64)
        lib.orc_tsg_rho_tokens(_d(k), hkv, d, h, tok.ctypes.data_as(_ip), len(tok), cur_off, cur_len,
                               int(metric), vals.ctypes.data_as(_dp))
        out[h, tok] = vals

    _run_tasks(run, tasks, threads)
    return out


def tsg_rho_per_head(k, frames, metric: int = TSG_COSINE) -> np.ndarray:
    """Eq. 6 in one pass per KV head over the frames (``orc_tsg_rho``); the
    same quantity as ``tsg_rho``, kept as a cross-check of its task split."""
    lib = _load()
    k = _c64(k)
    n, hkv, d = k.shape
    off, gh, gw = _frames(frames)
    out = np.zeros((hkv, n), dtype=np.float64)
    for h in range(hkv):
        lib.orc_tsg_rho(_d(k), n, hkv, d, h, len(off), off.ctypes.data_as(_ip),
                        gh.ctypes.data_as(_ip), gw.ctypes.data_as(_ip), int(metric), out[h].ctypes.data_as(_dp))
    return out


def tsg_rho_token(k, h: int, i: int, frames, metric: int = TSG_COSINE) -> float:
    """rho of the single token i against the current (last) frame."""
    k = _c64(k)
    n, hkv, d = k.shape
    off, gh, gw = _frames(frames)
    return float(_load().orc_tsg_rho_token(_d(k), hkv, d, h, i, int(off[-1]), int(gh[-1] * gw[-1]), int(metric)))


def tsg_gate(rho, frames, budget_b: int, tsg_enable: int = 1, fixed_tau=None):
    """Eqs. 7-8: tau = min(B,|pool|)-th smallest rho; M = [rho <= tau].  With
    fixed_tau (the fixed-threshold control) tau is that constant instead.

    Returns (tau [Hkv], gate [Hkv, N] uint8, pool_size)."""
    lib = _load()
    rho = _c64(rho)
    hkv, n = rho.shape
    off, gh, gw = _frames(frames)
    tau = np.zeros(hkv, dtype=np.float64)
    gate = np.zeros((hkv, n), dtype=np.uint8)
    pool = 0
    for h in range(hkv):
        t = ctypes.c_double()
        pool = lib.orc_tsg_gate(rho[h].ctypes.data_as(_dp), n, len(off), off.ctypes.data_as(_ip),
                                gh.ctypes.data_as(_ip), gw.ctypes.data_as(_ip), int(budget_b),
                                int(tsg_enable), 0 if fixed_tau is None else 1,
                                0.0 if fixed_tau is None else float(fixed_tau), ctypes.byref(t),
                                gate[h].ctypes.data_as(_bp))
        tau[h] = t.value
    return tau, gate, int(pool)


def combine(a, phi, gate, frames, alpha: float = 1.0, css_enable: int = 1) -> np.ndarray:
    """Eq. 9: S = A (text); S = M * (A + alpha * Phi) (visual)."""
    lib = _load()
    a, phi = _c64(a), _c64(phi)
    gate = np.ascontiguousarray(gate, dtype=np.uint8)
    hkv, n = a.shape
    off, gh, gw = _frames(frames)
    out = np.zeros((hkv, n), dtype=np.float64)
    for h in range(hkv):
        lib.orc_combine(a[h].ctypes.data_as(_dp), phi[h].ctypes.data_as(_dp), gate[h].ctypes.data_as(_bp),
                        n, len(off), off.ctypes.data_as(_ip), gh.ctypes.data_as(_ip),
                        gw.ctypes.data_as(_ip), float(alpha), int(css_enable), out[h].ctypes.data_as(_dp))
    return out


def topk(s, budget_b: int) -> np.ndarray:
    """Top-B by (S desc, index asc), returned in ascending index order: [Hkv, B]."""
    lib = _load()
    s = _c64(s)
    hkv, n = s.shape
    b = min(int(budget_b), n)
    out = np.zeros((hkv, b), dtype=np.int32)
    for h in range(hkv):
        lib.orc_topk(s[h].ctypes.data_as(_dp), n, int(budget_b), out[h].ctypes.data_as(_ip))
    return out


def gather(k, v, idx):
    """K'[r,h,:] = K[idx[h,r],h,:] (and V), byte-exact for any element type."""
    lib = _load()
    k = np.ascontiguousarray(k)
    v = np.ascontiguousarray(v)
    assert k.shape == v.shape and k.dtype == v.dtype
    n, hkv, d = k.shape
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    b = idx.shape[1]
    ko = np.zeros((b, hkv, d), dtype=k.dtype)
    vo = np.zeros((b, hkv, d), dtype=v.dtype)
    kb, vb = k.view(np.uint8), v.view(np.uint8)
    for h in range(hkv):
        lib.orc_gather(kb.ctypes.data_as(_bp), vb.ctypes.data_as(_bp), hkv, d, k.itemsize, h,
                       idx[h].ctypes.data_as(_ip), b, ko.view(np.uint8).ctypes.data_as(_bp),
                       vo.view(np.uint8).ctypes.data_as(_bp))
    return ko, vo


BASE_WINDOW, BASE_UNIFORM = 0, 1
ABASE_RAW, ABASE_MAX = 0, 1


def normalise_max(a) -> np.ndarray:
    """A divided by its maximum over the tokens, per head (rows whose maximum
    is not positive are left as they are): the reading of A_base's scale that
    the paper's reported A_base magnitudes suggest."""
    a = np.asarray(a, dtype=np.float64)
    out = a.copy()
    for h in range(a.shape[0]):
        m = a[h].max()
        if m > 0:
            out[h] = a[h] / m
    return out


def compress_layer(q, k, frames, beta: float = 0.2, k_override: int = 0, alpha: float = 1.0,
                   tsg_enable: int = 1, css_enable: int = 1, threads: int = 1, tsg_metric: int = TSG_COSINE,
                   fixed_tau=None, base_scorer: int = BASE_WINDOW, abase_norm: int = ABASE_RAW,
                   css_size: int = 3) -> dict:
    """Algorithm 1 for one layer: every stage in the paper's order.  The
    keyword variants are the paper's ablations: TSG similarity metric, a fixed
    gate threshold, and the uniform base prior (A = w/N for every token, the
    same total as the window score); abase_norm = ABASE_MAX divides A by its
    per-head maximum before Eq. 9; css_size is the CSS neighbourhood k x k."""
    n = k.shape[0]
    w = q.shape[0]
    b = budget(n, beta, k_override)
    if base_scorer == BASE_UNIFORM:
        a = np.full((k.shape[1], n), w / n, dtype=np.float64)
    else:
        a = abase(q, k, threads)
    if abase_norm == ABASE_MAX:
        a = normalise_max(a)
    phi = css_phi(k, frames, threads, size=css_size)
    if tsg_enable:
        rho = tsg_rho(k, frames, threads, metric=tsg_metric)
    else:
        rho = np.full_like(a, np.nan)
    tau, gate, pool = tsg_gate(rho, frames, b, tsg_enable, fixed_tau=fixed_tau)
    s = combine(a, phi, gate, frames, alpha, css_enable)
    idx = topk(s, b)
    return dict(budget=b, a=a, phi=phi, rho=rho, tau=tau, gate=gate, pool=pool, s=s, idx=idx)


def decode_attention(q, k, v) -> np.ndarray:
    """Attention of every query row over the whole cache (the decoder's use of
    the compressed cache): out[r][g] = sum_j softmax_j(q_{r,g}.k_{j,g/G}/sqrt(d))
    v_{j,g/G}.  q [w][Hq][d], k and v [n][Hkv][d]; returns [w][Hq][d] float64."""
    lib = _load()
    q, k, v = _c64(q), _c64(k), _c64(v)
    w, hq, d = q.shape
    n, hkv, d2 = k.shape
    assert d == d2 and v.shape == k.shape and hq % hkv == 0
    out = np.zeros((w, hq, d), dtype=np.float64)
    for r in range(w):
        for g in range(hq):
            lib.orc_decode_row(_d(q), _d(k), _d(v), n, hq, hkv, d, r, g, out[r, g].ctypes.data_as(_dp))
    return out


def critical_hit_rate(idx_keep, q_probe, k) -> np.ndarray:
    """Share of the probe query's B most-attended tokens (per KV head: its
    window score with the probe as the only window row, Eq. 2 with w = 1)
    that the compressed cache kept: |I_keep & Top_B(A_probe)| / B."""
    idx_keep = np.asarray(idx_keep)
    hkv, b = idx_keep.shape
    a = abase(q_probe, k)
    out = np.zeros(hkv, dtype=np.float64)
    for h in range(hkv):
        top = topk(a[h:h + 1], b)[0]
        out[h] = len(np.intersect1d(top, idx_keep[h])) / b
    return out
