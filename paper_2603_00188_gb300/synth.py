"""Seeded synthetic GUI-trajectory KV caches (input generation only).

This module draws the inputs that both the CUDA path and the test oracle
consume.  It contains none of the compression arithmetic: it only lays out a
trajectory of screenshot frames and text spans and fills keys, values and
window queries with seeded random numbers.

Layout of one trajectory (one layer, one sequence): for each step the frame's
``gh x gw`` patch-grid tokens (row-major) come first, then ``n_text`` text
tokens (action / instruction tokens).  The last frame is the current frame.

Value recipe (shapes follow the UI-TARS-1.5-7B / Qwen2.5-VL GQA layout the
paper evaluates: 28 query heads over 4 KV heads, head_dim 128):

* K background: frame 0 ~ N(0, 1); frame f = frame f-1 + N(0, drift^2)
  (inter-frame redundancy).  A near-duplicate frame uses sigma = dup_sigma and
  also copies the previous frame's planted boxes.  ``dup_exact_runs`` instead
  makes runs of exact copies (long-horizon tie stress).
* Planted UI boxes: rectangles of patches whose keys are
  ``box_scale * q_hat + N(0, box_noise^2)``, q_hat = unit mean window query of
  the KV head's query group (an element the window attends to).
* Text tokens, values and queries ~ N(0, 1) (or Student-t nu=3 if
  ``heavy_tail``).

Everything is float32 on the host; callers round to bf16 with torch.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

BASE_SEED = 0x5714E


@dataclass
class Workload:
    name: str
    q: np.ndarray          # [w, Hq, d] float32
    k: np.ndarray          # [N, Hkv, d] float32
    v: np.ndarray          # [N, Hkv, d] float32
    offset: np.ndarray     # [F] int32
    grid_h: np.ndarray     # [F] int32
    grid_w: np.ndarray     # [F] int32
    beta: float = 0.2
    dtype: str = "bf16"    # "bf16" or "f32"
    meta: dict = field(default_factory=dict)

    @property
    def frames(self):
        return (self.offset, self.grid_h, self.grid_w)

    @property
    def n(self) -> int:
        return int(self.k.shape[0])

    @property
    def shape(self):
        w, hq, d = self.q.shape
        return dict(n_tokens=self.n, n_q_heads=hq, n_kv_heads=self.k.shape[1], head_dim=d, window=w)


def _rng(*key) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([BASE_SEED, *key])))


def _draw(rng, shape, heavy_tail: bool):
    if heavy_tail:
        z = rng.standard_normal(shape, dtype=np.float32)
        chi = rng.chisquare(3.0, size=shape).astype(np.float32)
        return z / np.sqrt(chi / np.float32(3.0))
    return rng.standard_normal(shape, dtype=np.float32)


def _unit_mean_query(q: np.ndarray, hkv: int) -> np.ndarray:
    """Unit-norm mean of each KV head's group of window queries: [Hkv, d]."""
    w, hq, d = q.shape
    g = hq // hkv
    m = q.reshape(w, hkv, g, d).mean(axis=(0, 2))
    return m / np.maximum(np.linalg.norm(m, axis=-1, keepdims=True), 1e-12)


def trajectory(*, n_steps: int, gh: int, gw: int, n_text: int, hq: int = 28, hkv: int = 4,
               d: int = 128, w: int = 32, drift: float = 0.1, dup_frac: float = 0.3,
               dup_sigma: float = 0.01, dup_exact_runs: tuple | None = None,
               n_boxes: tuple = (5, 20), box_hw: tuple = ((2, 2), (4, 8)),
               box_scale: float = 3.0, box_noise: float = 0.1, heavy_tail: bool = False,
               beta: float = 0.2, dtype: str = "bf16", seed: tuple = (0,), name: str = "") -> Workload:
    """One layer of one sequence of a synthetic GUI trajectory (see module doc)."""
    rng = _rng(*seed)
    P = gh * gw
    step = P + n_text
    n = n_steps * step
    q = _draw(rng, (w, hq, d), False)
    qhat = _unit_mean_query(q, hkv)

    # which frames are near-duplicates of their predecessor
    dup = np.zeros(n_steps, dtype=bool)
    if dup_exact_runs is not None:
        # at each fresh frame, with probability dup_frac start a run of
        # lo..hi identical frames (the fresh one plus its copies)
        lo, hi = dup_exact_runs
        f = 0
        while f < n_steps:
            if rng.random() < dup_frac:
                run = int(rng.integers(lo, hi + 1))
                dup[f + 1:f + run] = True
                f += run
            else:
                f += 1
    elif n_steps > 1:
        n_dup = int(round(dup_frac * (n_steps - 1)))
        dup[1 + rng.permutation(n_steps - 1)[:n_dup]] = True

    k = np.empty((n, hkv, d), dtype=np.float32)
    bg = _draw(rng, (P, hkv, d), heavy_tail)
    prev = None
    for f in range(n_steps):
        off = f * step
        if f > 0 and dup[f]:
            if dup_exact_runs is not None:
                frame = prev.copy()
            else:
                frame = prev + dup_sigma * rng.standard_normal((P, hkv, d), dtype=np.float32)
        else:
            if f > 0:
                bg = bg + drift * rng.standard_normal((P, hkv, d), dtype=np.float32)
            frame = bg.copy()
            nb = int(rng.integers(n_boxes[0], n_boxes[1] + 1))
            for _ in range(nb):
                bh = int(rng.integers(box_hw[0][0], box_hw[1][0] + 1))
                bw = int(rng.integers(box_hw[0][1], box_hw[1][1] + 1))
                bh, bw = min(bh, gh), min(bw, gw)
                u0 = int(rng.integers(0, gh - bh + 1))
                v0 = int(rng.integers(0, gw - bw + 1))
                cells = (np.arange(u0, u0 + bh)[:, None] * gw + np.arange(v0, v0 + bw)[None, :]).ravel()
                noise = box_noise * rng.standard_normal((cells.size, hkv, d), dtype=np.float32)
                frame[cells] = box_scale * qhat[None, :, :] + noise
        k[off:off + P] = frame
        k[off + P:off + step] = _draw(rng, (n_text, hkv, d), heavy_tail)
        prev = frame
    v = _draw(rng, (n, hkv, d), heavy_tail)
    offset = (np.arange(n_steps, dtype=np.int32) * step).astype(np.int32)
    return Workload(name=name, q=q, k=k, v=v, offset=offset,
                    grid_h=np.full(n_steps, gh, np.int32), grid_w=np.full(n_steps, gw, np.int32),
                    beta=beta, dtype=dtype, meta=dict(dup=dup.tolist(), step=step))


# --------------------------------------------------------------------------
# The five workload configurations (UI-TARS-1.5-7B-shaped caches).

def tiny_ref(seed: int = 0) -> Workload:
    """1 layer, 4 KV / 28 Q heads, d=128, fp32; 4 frames of 16x16 + 32 text
    tokens (N=1152); w=32, beta=20%.  Frame 3 (current) is frame 2 +
    N(0, 0.01^2) in full; two 2x3 rectangles per frame carry keys 3 * q_hat
    (frame 3's are the noisy copies of frame 2's)."""
    rng = _rng(1, seed)
    hq, hkv, d, w, gh, gw, nt, F = 28, 4, 128, 32, 16, 16, 32, 4
    P, step = gh * gw, gh * gw + nt
    n = F * step
    q = rng.standard_normal((w, hq, d), dtype=np.float32)
    qhat = _unit_mean_query(q, hkv)
    k = rng.standard_normal((n, hkv, d), dtype=np.float32)
    v = rng.standard_normal((n, hkv, d), dtype=np.float32)

    def plant(off):
        for _ in range(2):
            u0 = int(rng.integers(0, gh - 2 + 1))
            v0 = int(rng.integers(0, gw - 3 + 1))
            cells = off + (np.arange(u0, u0 + 2)[:, None] * gw + np.arange(v0, v0 + 3)[None, :]).ravel()
            k[cells] = 3.0 * qhat[None]

    for f in range(3):
        plant(f * step)
    # frame 3 is frame 2 plus noise, its two rectangles included
    k[3 * step:3 * step + P] = k[2 * step:2 * step + P] + 0.01 * rng.standard_normal((P, hkv, d), dtype=np.float32)
    offset = (np.arange(F, dtype=np.int32) * step).astype(np.int32)
    return Workload(name="tiny_ref_fp32", q=q, k=k, v=v, offset=offset,
                    grid_h=np.full(F, gh, np.int32), grid_w=np.full(F, gw, np.int32),
                    beta=0.2, dtype="f32", meta=dict(step=step))


def uitars_layer(beta: float = 0.2, seed: int = 0) -> Workload:
    """1 layer at full UI-TARS-1.5-7B shape: 10 frames of 36x64 + 64 text
    tokens (N=23680), w=32, bf16."""
    return trajectory(n_steps=10, gh=36, gw=64, n_text=64, beta=beta, seed=(2, seed),
                      name="uitars_1layer_10x36x64")


def trajectory_50(layer: int, seed: int = 0) -> Workload:
    """One layer of the 28-layer, 50-step trajectory: 50 frames of 32x32 + 48
    text tokens (N=53600), w=32, beta=20%, bf16."""
    return trajectory(n_steps=50, gh=32, gw=32, n_text=48, beta=0.2, seed=(3, seed, layer),
                      name="traj50_32x32")


def small_backbone_seq(seq: int, layer: int = 0, beta: float = 0.1, seed: int = 0) -> Workload:
    """One sequence of the batch-8 smaller-backbone shape: 12 Q / 2 KV heads,
    12-20 frames of 24x42 + 40 text tokens, w=16, bf16."""
    r = _rng(4, seed, seq, 999)
    n_steps = int(r.integers(12, 21))
    return trajectory(n_steps=n_steps, gh=24, gw=42, n_text=40, hq=12, hkv=2, w=16, beta=beta,
                      seed=(4, seed, seq, layer), name="small_backbone_24x42")


def long_horizon(layer: int = 0, seed: int = 0) -> Workload:
    """Long-horizon stress: 100 frames of 36x36 + 32 text tokens (N=132800),
    w=64, beta=10%; runs of 2-5 exact duplicate frames (about half of all
    frames are copies of their predecessor),
    1x2-patch micro-elements, Student-t (nu=3) keys and values."""
    return trajectory(n_steps=100, gh=36, gw=36, n_text=32, w=64, beta=0.1, dup_frac=0.4,
                      dup_exact_runs=(2, 5), n_boxes=(5, 20), box_hw=((1, 2), (1, 2)),
                      heavy_tail=True, seed=(5, seed, layer), name="long_horizon_100x36x36")


def scaled(base: str, n_steps: int, seed: int = 0, **kw) -> Workload:
    """A shorter trajectory with the value recipe of a named configuration
    (used where the oracle must finish in seconds)."""
    if base == "uitars":
        return trajectory(n_steps=n_steps, gh=36, gw=64, n_text=64, seed=(12, seed, n_steps),
                          name="uitars_scaled", **kw)
    if base == "traj50":
        return trajectory(n_steps=n_steps, gh=32, gw=32, n_text=48, seed=(13, seed, n_steps),
                          name="traj50_scaled", **kw)
    if base == "small":
        return trajectory(n_steps=n_steps, gh=24, gw=42, n_text=40, hq=12, hkv=2, w=16,
                          seed=(14, seed, n_steps), name="small_scaled", **kw)
    if base == "long":
        return trajectory(n_steps=n_steps, gh=36, gw=36, n_text=32, w=64, dup_frac=0.4,
                          dup_exact_runs=(2, 5), box_hw=((1, 2), (1, 2)), heavy_tail=True,
                          seed=(15, seed, n_steps), name="long_scaled", **kw)
    raise ValueError(base)
