"""Shared helpers of the GPU parity tests: moving a synthetic workload to the
device, its exact float64 image for the oracle, and the matching rules.

Matching rules (GPU vs fp64 oracle):
* window score A: |g - o| <= 1e-3 |o| + 1e-7 max|o|  (fp32 softmax; the floor
  absorbs fp32 underflow of vanishing probabilities);
* cosine quantities Phi, rho: |g - o| <= 1e-3 |o| + COS_ATOL.  COS_ATOL = 2e-5
  bounds the fp32 error of a 128-term dot product of normalised vectors
  (d * 2^-24 ~ 7.6e-6) plus the two rounded reciprocal norms, so values near
  zero (Phi of uniform patches) are compared absolutely;
* integrated score S: sum of the two rules above;
* gate: a token may differ only if its oracle rho lies within the rho
  tolerance of the oracle threshold tau;
* kept sets: identical except swaps of tokens whose oracle score lies within
  the S tolerance of the oracle's B-th score, or whose gate flipped as above;
* compacted rows: bit-exact.
"""
import numpy as np
import torch

import oracle

COS_ATOL = 2e-5
A_RTOL = 1e-3
A_FLOOR = 1e-7


def to_device(wl):
    dt = torch.float32 if wl.dtype == "f32" else torch.bfloat16
    q = torch.from_numpy(wl.q).to(dt).cuda()
    k = torch.from_numpy(wl.k).to(dt).cuda()
    v = torch.from_numpy(wl.v).to(dt).cuda()
    return q, k, v


def exact64(t):
    return t.detach().cpu().to(torch.float64).numpy()


def a_bound(ora):
    return A_RTOL * np.abs(ora) + A_FLOOR * np.nanmax(np.abs(ora))


def cos_bound(ora):
    return A_RTOL * np.abs(ora) + COS_ATOL


def assert_within(gpu, ora, bound, what):
    gpu = np.asarray(gpu, dtype=np.float64)
    ora = np.asarray(ora, dtype=np.float64)
    err = np.abs(gpu - ora)
    bad = ~(err <= bound)
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError("%s: %d/%d outside tolerance; first at %s gpu=%r oracle=%r bound=%r"
                             % (what, int(bad.sum()), bad.size, tuple(i), gpu[tuple(i)], ora[tuple(i)],
                                np.broadcast_to(bound, ora.shape)[tuple(i)]))


def visual_mask(n, frames):
    off, gh, gw = frames
    m = np.zeros(n, bool)
    for o, a, b in zip(off, gh, gw):
        m[o:o + a * b] = True
    return m


def pool_mask(n, frames):
    off, gh, gw = frames
    m = np.zeros(n, bool)
    for o, a, b in list(zip(off, gh, gw))[:-1]:
        m[o:o + a * b] = True
    return m


def check_kept_sets(idx_gpu, idx_ora, s_ora, budget, s_tol, allowed_extra=None):
    """Kept-set rule for one head; returns the number of swapped pairs."""
    g, o = set(idx_gpu.tolist()), set(idx_ora.tolist())
    assert len(idx_gpu) == budget and len(g) == budget
    assert (np.diff(idx_gpu) > 0).all()
    only_g, only_o = g - o, o - g
    assert len(only_g) == len(only_o)
    if not only_g:
        return 0
    thr = np.sort(s_ora)[::-1][budget - 1]
    tol = s_tol(thr)
    for t in only_g | only_o:
        if allowed_extra is not None and t in allowed_extra:
            continue
        assert abs(s_ora[t] - thr) <= tol, ("kept-set swap away from the threshold", t, s_ora[t], thr, tol)
    return len(only_g)


def gate_flip_tokens(gate_gpu, gate_ora, rho_ora, tau_ora):
    """Tokens whose gate differs; each must sit at the oracle threshold."""
    flips = np.nonzero(gate_gpu != gate_ora)[0]
    for t in flips:
        assert abs(rho_ora[t] - tau_ora) <= A_RTOL * abs(tau_ora) + COS_ATOL, (t, rho_ora[t], tau_ora)
    return set(flips.tolist())


class OracleCache:
    """Oracle results per workload name (each computed once per session)."""

    def __init__(self):
        self._d = {}

    def get(self, key, fn):
        if key not in self._d:
            self._d[key] = fn()
        return self._d[key]


CACHE = OracleCache()
