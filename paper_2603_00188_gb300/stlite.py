"""Python binding of libstlite.so (ctypes; argument marshalling only).

Every function here has the name of the C entry point it calls (declared in
``include/stlite.h``) and forwards torch CUDA tensors as raw device pointers
on the current torch stream.  No computation happens in Python: if the
library is not built this module raises at import time.

    from paper_2603_00188_gb300 import stlite
    k_out, v_out, idx = stlite.compress_layer(q, k, v, frames, beta=0.2)
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libstlite.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError("libstlite.so is not built (run paper_2603_00188_gb300.build.build()): %s" % _LIB_PATH)
_lib = ctypes.CDLL(_LIB_PATH)

STLITE_OK, STLITE_EINVAL, STLITE_EUNSUPPORTED, STLITE_EWORKSPACE, STLITE_ECUDA, STLITE_ETIMEOUT = range(6)
STLITE_BF16, STLITE_F32 = 0, 1
MAX_FRAMES = 256
EXPORTED = ("stlite_budget", "stlite_workspace_size", "stlite_score", "stlite_gate_frames",
            "stlite_spatial_saliency", "stlite_select_topk", "stlite_compact",
            "stlite_compress_layer", "stlite_device_status", "stlite_timing_enable", "stlite_timing_read",
            "stlite_status_string", "stlite_score_noalloc", "stlite_compress_layers", "stlite_compress_varlen",
            "stlite_workspace_size_varlen", "stlite_decode_attention", "stlite_decode_workspace_size",
            "stlite_compress_layers_budgets", "stlite_hierarchical_budgets", "stlite_spatial_saliency_size",
            "stlite_compress_varlen_layers", "stlite_prompt_score", "stlite_prompt_workspace_size",
            "stlite_decode_attention_layers", "stlite_decode_layers_workspace_size",
            "stlite_selftest_wait_timeout")


class Shape(ctypes.Structure):
    _fields_ = [("n_tokens", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("window", ctypes.c_int32), ("dtype", ctypes.c_int32)]


class Frames(ctypes.Structure):
    _fields_ = [("n_frames", ctypes.c_int32), ("offset", ctypes.POINTER(ctypes.c_int32)),
                ("grid_h", ctypes.POINTER(ctypes.c_int32)), ("grid_w", ctypes.POINTER(ctypes.c_int32))]


class Params(ctypes.Structure):
    _fields_ = [("beta", ctypes.c_double), ("k_override", ctypes.c_int32), ("alpha", ctypes.c_float),
                ("tsg_enable", ctypes.c_int32), ("css_enable", ctypes.c_int32), ("tsg_metric", ctypes.c_int32),
                ("tsg_fixed", ctypes.c_int32), ("tsg_fixed_tau", ctypes.c_float), ("base_scorer", ctypes.c_int32),
                ("abase_norm", ctypes.c_int32), ("css_size", ctypes.c_int32)]


STLITE_TSG_COSINE, STLITE_TSG_DOT, STLITE_TSG_NEG_L2 = 0, 1, 2
STLITE_BASE_WINDOW, STLITE_BASE_UNIFORM = 0, 1
STLITE_ABASE_RAW, STLITE_ABASE_MAX = 0, 1
STLITE_PROMPT_FULL, STLITE_PROMPT_MEAN = 0, 1


class LayerIO(ctypes.Structure):
    _fields_ = [("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("k_out", ctypes.c_void_p), ("v_out", ctypes.c_void_p), ("idx_out", ctypes.c_void_p)]


class DecodeIO(ctypes.Structure):
    _fields_ = [("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("out", ctypes.c_void_p)]


class KernelTime(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int32), ("total_ms", ctypes.c_double)]


_P = ctypes.c_void_p
_S = ctypes.c_int32
_sig = {
    "stlite_budget": (ctypes.c_int32, [ctypes.c_int32, ctypes.c_double, ctypes.c_int32]),
    "stlite_workspace_size": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), ctypes.POINTER(Params),
                                   ctypes.POINTER(ctypes.c_size_t)]),
    "stlite_score": (_S, [ctypes.POINTER(Shape), _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "stlite_gate_frames": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), _P, ctypes.c_int32, _P, _P, _P,
                                _P, ctypes.c_size_t, _P]),
    "stlite_spatial_saliency": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), _P, _P, _P,
                                     ctypes.c_size_t, _P]),
    "stlite_select_topk": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), ctypes.POINTER(Params), _P, _P,
                                _P, ctypes.c_int32, _P, _P, _P, ctypes.c_size_t, _P]),
    "stlite_compact": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, _P, _P, _P, _P, _P, _P]),
    "stlite_compress_layer": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), ctypes.POINTER(Params), _P,
                                   _P, _P, _P, _P, _P, ctypes.POINTER(ctypes.c_int32), _P, ctypes.c_size_t, _P]),
    "stlite_device_status": (_S, [_P, _P, ctypes.POINTER(ctypes.c_int32)]),
    "stlite_timing_enable": (_S, [ctypes.c_int32]),
    "stlite_timing_read": (_S, [ctypes.POINTER(KernelTime), ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)]),
    "stlite_status_string": (ctypes.c_char_p, [ctypes.c_int32]),
    "stlite_score_noalloc": (_S, [ctypes.POINTER(Shape), _P, _P, _P, _P]),
    "stlite_compress_layers": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), ctypes.POINTER(Params),
                                    ctypes.c_int32, ctypes.POINTER(LayerIO), ctypes.POINTER(ctypes.c_int32), _P,
                                    ctypes.c_size_t, _P]),
    "stlite_compress_varlen": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, ctypes.POINTER(ctypes.c_int32),
                                    ctypes.POINTER(Frames), ctypes.POINTER(Params), _P, _P, _P, _P, _P, _P,
                                    ctypes.POINTER(ctypes.c_int32), _P, ctypes.c_size_t, _P]),
    "stlite_workspace_size_varlen": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, ctypes.POINTER(ctypes.c_int32),
                                          ctypes.POINTER(Frames), ctypes.POINTER(Params),
                                          ctypes.POINTER(ctypes.c_size_t)]),
    "stlite_decode_attention": (_S, [ctypes.POINTER(Shape), _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "stlite_decode_workspace_size": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(ctypes.c_size_t)]),
    "stlite_compress_layers_budgets": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), ctypes.POINTER(Params),
                                            ctypes.c_int32, ctypes.POINTER(LayerIO), ctypes.POINTER(ctypes.c_int32),
                                            _P, ctypes.c_size_t, _P]),
    "stlite_spatial_saliency_size": (_S, [ctypes.POINTER(Shape), ctypes.POINTER(Frames), _P, ctypes.c_int32, _P, _P,
                                          ctypes.c_size_t, _P]),
    "stlite_compress_varlen_layers": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, ctypes.POINTER(ctypes.c_int32),
                                           ctypes.POINTER(Frames), ctypes.POINTER(Params), ctypes.c_int32,
                                           ctypes.POINTER(LayerIO), ctypes.POINTER(ctypes.c_int32), _P,
                                           ctypes.c_size_t, _P]),
    "stlite_hierarchical_budgets": (_S, [ctypes.c_int32, ctypes.POINTER(ctypes.c_double), ctypes.c_int64,
                                         ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)]),
    "stlite_prompt_score": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, ctypes.c_int32, _P, _P, _P, _P,
                                 ctypes.c_size_t, _P]),
    "stlite_prompt_workspace_size": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]),
    "stlite_selftest_wait_timeout": (_S, [_P, ctypes.c_int64, _P]),
    "stlite_decode_attention_layers": (_S, [ctypes.POINTER(Shape), ctypes.c_int32, ctypes.POINTER(DecodeIO), _P,
                                            ctypes.c_size_t, _P]),
    "stlite_decode_layers_workspace_size": (_S, [ctypes.POINTER(Shape), ctypes.c_int32,
                                                 ctypes.POINTER(ctypes.c_size_t)]),
}
for _name, (_res, _args) in _sig.items():
    _f = getattr(_lib, _name)
    _f.restype = _res
    _f.argtypes = _args


class StliteError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s (%d)" % (where, _lib.stlite_status_string(status).decode(), status))


def _check(status: int, where: str):
    if status != STLITE_OK:
        raise StliteError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def make_shape(q, k) -> Shape:
    w, hq, d = q.shape
    n, hkv, d2 = k.shape
    if d != d2:
        raise ValueError("q and k head_dim differ")
    dt = {torch.bfloat16: STLITE_BF16, torch.float32: STLITE_F32}[k.dtype]
    return Shape(n, hq, hkv, d, w, dt)


class FrameSpec:
    """Host frame descriptor (offset, grid_h, grid_w), kept alive with its ctypes view."""

    def __init__(self, offset, grid_h, grid_w):
        self.offset = np.ascontiguousarray(offset, dtype=np.int32)
        self.grid_h = np.ascontiguousarray(grid_h, dtype=np.int32)
        self.grid_w = np.ascontiguousarray(grid_w, dtype=np.int32)
        ip = ctypes.POINTER(ctypes.c_int32)
        self.c = Frames(len(self.offset), self.offset.ctypes.data_as(ip), self.grid_h.ctypes.data_as(ip),
                        self.grid_w.ctypes.data_as(ip))


def _frames(frames) -> FrameSpec:
    if isinstance(frames, FrameSpec):
        return frames
    return FrameSpec(*frames)


def make_params(beta=0.2, k_override=0, alpha=1.0, tsg_enable=1, css_enable=1, tsg_metric=STLITE_TSG_COSINE,
                fixed_tau=None, base_scorer=STLITE_BASE_WINDOW, abase_norm=STLITE_ABASE_RAW, css_size=3) -> Params:
    """Parameters of the pass; the keywords after css_enable select the
    paper's ablation variants (TSG similarity metric, a fixed gate threshold,
    the uniform base prior, A_base divided by its maximum, the CSS
    neighbourhood size) and default to the method as published."""
    return Params(float(beta), int(k_override), float(alpha), int(tsg_enable), int(css_enable), int(tsg_metric),
                  0 if fixed_tau is None else 1, 0.0 if fixed_tau is None else float(fixed_tau), int(base_scorer),
                  int(abase_norm), int(css_size))


# ----------------------------------------------------------------- entries

def stlite_budget(n_tokens: int, beta: float, k_override: int = 0) -> int:
    return int(_lib.stlite_budget(int(n_tokens), float(beta), int(k_override)))


def stlite_workspace_size(shape: Shape, frames, params: Params | None = None) -> int:
    fs = _frames(frames)
    out = ctypes.c_size_t()
    _check(_lib.stlite_workspace_size(ctypes.byref(shape), ctypes.byref(fs.c),
                                      ctypes.byref(params) if params is not None else None,
                                      ctypes.byref(out)), "stlite_workspace_size")
    return int(out.value)


def workspace(shape: Shape, frames, params: Params | None = None, device="cuda"):
    """Zero-filled workspace tensor of the size the library asks for."""
    return torch.zeros(stlite_workspace_size(shape, frames, params), dtype=torch.uint8, device=device)


def stlite_score(q, k, a_base, ws, stream=None):
    sh = make_shape(q, k)
    _check(_lib.stlite_score(ctypes.byref(sh), _ptr(q), _ptr(k), _ptr(a_base), _ptr(ws), ws.numel(),
                             _stream(stream)), "stlite_score")


def stlite_gate_frames(q, k, frames, budget, rho, tau, gate, ws, stream=None):
    sh = make_shape(q, k)
    fs = _frames(frames)
    _check(_lib.stlite_gate_frames(ctypes.byref(sh), ctypes.byref(fs.c), _ptr(k), int(budget), _ptr(rho),
                                   _ptr(tau), _ptr(gate), _ptr(ws), ws.numel(), _stream(stream)),
           "stlite_gate_frames")


def stlite_spatial_saliency(q, k, frames, phi, ws, stream=None):
    sh = make_shape(q, k)
    fs = _frames(frames)
    _check(_lib.stlite_spatial_saliency(ctypes.byref(sh), ctypes.byref(fs.c), _ptr(k), _ptr(phi), _ptr(ws),
                                        ws.numel(), _stream(stream)), "stlite_spatial_saliency")


def stlite_spatial_saliency_size(q, k, frames, size, phi, ws, stream=None):
    sh = make_shape(q, k)
    fs = _frames(frames)
    _check(_lib.stlite_spatial_saliency_size(ctypes.byref(sh), ctypes.byref(fs.c), _ptr(k), int(size), _ptr(phi),
                                             _ptr(ws), ws.numel(), _stream(stream)), "stlite_spatial_saliency_size")


def stlite_select_topk(q, k, frames, params, a_base, phi, gate, budget, idx, score_out, ws, stream=None):
    sh = make_shape(q, k)
    fs = _frames(frames)
    _check(_lib.stlite_select_topk(ctypes.byref(sh), ctypes.byref(fs.c), ctypes.byref(params), _ptr(a_base),
                                   _ptr(phi), _ptr(gate), int(budget), _ptr(idx), _ptr(score_out), _ptr(ws),
                                   ws.numel(), _stream(stream)), "stlite_select_topk")


def stlite_compact(q, k, v, budget, idx, k_out, v_out, stream=None):
    sh = make_shape(q, k)
    _check(_lib.stlite_compact(ctypes.byref(sh), int(budget), _ptr(idx), _ptr(k), _ptr(v), _ptr(k_out),
                               _ptr(v_out), _stream(stream)), "stlite_compact")


def stlite_compress_layer(q, k, v, frames, params, k_out, v_out, idx_out, ws, stream=None) -> int:
    sh = make_shape(q, k)
    fs = _frames(frames)
    b = ctypes.c_int32(0)
    _check(_lib.stlite_compress_layer(ctypes.byref(sh), ctypes.byref(fs.c), ctypes.byref(params), _ptr(q),
                                      _ptr(k), _ptr(v), _ptr(k_out), _ptr(v_out), _ptr(idx_out),
                                      ctypes.byref(b), _ptr(ws), ws.numel(), _stream(stream)),
           "stlite_compress_layer")
    return int(b.value)


def stlite_compress_layers(layers, frames, params, ws, stream=None) -> int:
    """layers: list of (q, k, v, k_out, v_out, idx_out) device tensors, one
    tuple per layer (same shapes); ws: n_layers * stlite_workspace_size bytes."""
    q0, k0 = layers[0][0], layers[0][1]
    sh = make_shape(q0, k0)
    fs = _frames(frames)
    arr = (LayerIO * len(layers))(*[LayerIO(*(t.data_ptr() for t in lay)) for lay in layers])
    b = ctypes.c_int32(0)
    _check(_lib.stlite_compress_layers(ctypes.byref(sh), ctypes.byref(fs.c), ctypes.byref(params), len(layers),
                                       arr, ctypes.byref(b), _ptr(ws), ws.numel(), _stream(stream)),
           "stlite_compress_layers")
    return int(b.value)


def stlite_compress_layers_budgets(layers, frames, params, budgets, ws, stream=None):
    """As stlite_compress_layers with layer l keeping budgets[l] tokens per
    KV head (k_out / v_out of layer l: [budgets[l]][Hkv][d], idx_out:
    [Hkv][budgets[l]])."""
    q0, k0 = layers[0][0], layers[0][1]
    sh = make_shape(q0, k0)
    fs = _frames(frames)
    arr = (LayerIO * len(layers))(*[LayerIO(*(t.data_ptr() for t in lay)) for lay in layers])
    bud = (ctypes.c_int32 * len(layers))(*[int(b) for b in budgets])
    _check(_lib.stlite_compress_layers_budgets(ctypes.byref(sh), ctypes.byref(fs.c), ctypes.byref(params),
                                               len(layers), arr, bud, _ptr(ws), ws.numel(), _stream(stream)),
           "stlite_compress_layers_budgets")


def stlite_hierarchical_budgets(layer_mass, total_budget: int, n_tokens: int) -> list:
    """B^(l) = S^(l) / sum S * B_total as integers adding up to B_total
    (floor plus largest remainder, clamped to [1, n_tokens])."""
    n = len(layer_mass)
    mass = (ctypes.c_double * n)(*[float(x) for x in layer_mass])
    out = (ctypes.c_int32 * n)()
    _check(_lib.stlite_hierarchical_budgets(n, mass, int(total_budget), int(n_tokens), out),
           "stlite_hierarchical_budgets")
    return list(out)


def _varlen_args(cu_seqlens, frames_list):
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    specs = [_frames(f) for f in frames_list]
    arr = (Frames * len(specs))(*[f.c for f in specs])
    return cu, specs, arr


def stlite_workspace_size_varlen(shape: Shape, cu_seqlens, frames_list, params: Params | None = None) -> int:
    cu, specs, arr = _varlen_args(cu_seqlens, frames_list)
    out = ctypes.c_size_t()
    _check(_lib.stlite_workspace_size_varlen(ctypes.byref(shape), len(specs),
                                             cu.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), arr,
                                             ctypes.byref(params) if params is not None else None,
                                             ctypes.byref(out)), "stlite_workspace_size_varlen")
    return int(out.value)


def stlite_compress_varlen(q, k, v, cu_seqlens, frames_list, params, k_out, v_out, idx_out, ws, stream=None):
    """Packed batch of sequences (one layer): q [n_seqs][w][Hq][d], k/v packed
    [N][Hkv][d], cu_seqlens (n_seqs + 1 offsets), one frame descriptor per
    sequence (offsets relative to the sequence).  Returns the budget prefix
    sums (n_seqs + 1)."""
    n_seqs = len(frames_list)
    sh = make_shape(q[0] if q.dim() == 4 else q, k)
    cu, specs, arr = _varlen_args(cu_seqlens, frames_list)
    cb = np.zeros(n_seqs + 1, dtype=np.int32)
    ip = ctypes.POINTER(ctypes.c_int32)
    _check(_lib.stlite_compress_varlen(ctypes.byref(sh), n_seqs, cu.ctypes.data_as(ip), arr, ctypes.byref(params),
                                       _ptr(q), _ptr(k), _ptr(v), _ptr(k_out), _ptr(v_out), _ptr(idx_out),
                                       cb.ctypes.data_as(ip), _ptr(ws), ws.numel(), _stream(stream)),
           "stlite_compress_varlen")
    return cb


def stlite_compress_varlen_layers(layers, cu_seqlens, frames_list, params, ws, stream=None):
    """stlite_compress_varlen over several layers of one packed batch: layers
    is a list of (q, k, v, k_out, v_out, idx_out) per layer, each in the
    packed layouts of stlite_compress_varlen; ws: n_layers times
    stlite_workspace_size_varlen bytes.  Returns the budget prefix sums."""
    n_seqs = len(frames_list)
    q0, k0 = layers[0][0], layers[0][1]
    sh = make_shape(q0[0] if q0.dim() == 4 else q0, k0)
    cu, specs, arr = _varlen_args(cu_seqlens, frames_list)
    lio = (LayerIO * len(layers))(*[LayerIO(*(t.data_ptr() for t in lay)) for lay in layers])
    cb = np.zeros(n_seqs + 1, dtype=np.int32)
    ip = ctypes.POINTER(ctypes.c_int32)
    _check(_lib.stlite_compress_varlen_layers(ctypes.byref(sh), n_seqs, cu.ctypes.data_as(ip), arr,
                                              ctypes.byref(params), len(layers), lio, cb.ctypes.data_as(ip),
                                              _ptr(ws), ws.numel(), _stream(stream)),
           "stlite_compress_varlen_layers")
    return cb


def stlite_decode_workspace_size(shape: Shape) -> int:
    out = ctypes.c_size_t()
    _check(_lib.stlite_decode_workspace_size(ctypes.byref(shape), ctypes.byref(out)), "stlite_decode_workspace_size")
    return int(out.value)


def stlite_decode_attention(q, k, v, out, ws, stream=None):
    """Attention of the query rows q [w][Hq][d] over the cache k, v [n][Hkv][d]
    (full or compacted) into out [w][Hq][d] float32."""
    sh = make_shape(q, k)
    _check(_lib.stlite_decode_attention(ctypes.byref(sh), _ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(ws),
                                        ws.numel(), _stream(stream)), "stlite_decode_attention")


def decode_attention(q, k, v, stream=None):
    """Allocates the output and the workspace and runs stlite_decode_attention."""
    sh = make_shape(q, k)
    ws = torch.zeros(stlite_decode_workspace_size(sh), dtype=torch.uint8, device=k.device)
    out = torch.empty(q.shape, dtype=torch.float32, device=k.device)
    stlite_decode_attention(q, k, v, out, ws, stream)
    return out


def prompt_shape(q_prompt, k) -> Shape:
    """Shape of a prompt-wide score call: the window field is unused (1)."""
    n_q, hq, d = q_prompt.shape
    n, hkv, d2 = k.shape
    if d != d2:
        raise ValueError("q and k head_dim differ")
    dt = {torch.bfloat16: STLITE_BF16, torch.float32: STLITE_F32}[k.dtype]
    return Shape(n, hq, hkv, d, 1, dt)


def stlite_prompt_workspace_size(shape: Shape, n_prompt: int) -> int:
    out = ctypes.c_size_t()
    _check(_lib.stlite_prompt_workspace_size(ctypes.byref(shape), int(n_prompt), ctypes.byref(out)),
           "stlite_prompt_workspace_size")
    return int(out.value)


def stlite_prompt_score(q_prompt, k, base, a_base, ws, stream=None):
    """Prompt-wide base scores (STLITE_PROMPT_FULL / STLITE_PROMPT_MEAN) of
    the n_prompt = q_prompt.shape[0] rows of the last positions."""
    sh = prompt_shape(q_prompt, k)
    _check(_lib.stlite_prompt_score(ctypes.byref(sh), int(q_prompt.shape[0]), int(base), _ptr(q_prompt), _ptr(k),
                                    _ptr(a_base), _ptr(ws), ws.numel(), _stream(stream)), "stlite_prompt_score")


def prompt_score(q_prompt, k, base=STLITE_PROMPT_MEAN, stream=None):
    """Allocates the output and a workspace and runs stlite_prompt_score."""
    sh = prompt_shape(q_prompt, k)
    ws = torch.zeros(stlite_prompt_workspace_size(sh, q_prompt.shape[0]), dtype=torch.uint8, device=k.device)
    a = torch.empty((sh.n_kv_heads, sh.n_tokens), dtype=torch.float32, device=k.device)
    stlite_prompt_score(q_prompt, k, base, a, ws, stream)
    return a, ws


def stlite_decode_layers_workspace_size(shape: Shape, n_layers: int) -> int:
    out = ctypes.c_size_t()
    _check(_lib.stlite_decode_layers_workspace_size(ctypes.byref(shape), int(n_layers), ctypes.byref(out)),
           "stlite_decode_layers_workspace_size")
    return int(out.value)


def stlite_decode_attention_layers(layers, ws, stream=None):
    """layers: list of (q, k, v, out) device tensors, one tuple per layer
    (same shapes)."""
    sh = make_shape(layers[0][0], layers[0][1])
    arr = (DecodeIO * len(layers))(*[DecodeIO(*(t.data_ptr() for t in lay)) for lay in layers])
    _check(_lib.stlite_decode_attention_layers(ctypes.byref(sh), len(layers), arr, _ptr(ws), ws.numel(),
                                               _stream(stream)), "stlite_decode_attention_layers")


def decode_attention_layers(qs, ks, vs, stream=None):
    """Allocates the outputs and the workspace and runs
    stlite_decode_attention_layers over the layers' (q, k, v)."""
    sh = make_shape(qs[0], ks[0])
    ws = torch.zeros(stlite_decode_layers_workspace_size(sh, len(qs)), dtype=torch.uint8, device=ks[0].device)
    outs = [torch.empty(q.shape, dtype=torch.float32, device=ks[0].device) for q in qs]
    stlite_decode_attention_layers(list(zip(qs, ks, vs, outs)), ws, stream)
    return outs, ws


def stlite_selftest_wait_timeout(ws, limit_ns: int, stream=None):
    """Runs the failure-path diagnostic: a bounded wait that runs out after
    limit_ns and records STLITE_ETIMEOUT in ws's error word."""
    _check(_lib.stlite_selftest_wait_timeout(_ptr(ws), int(limit_ns), _stream(stream)),
           "stlite_selftest_wait_timeout")


def stlite_device_status(ws, stream=None) -> int:
    """Reads and clears a workspace's device error word; ws=None reads the
    error word of stlite_score_noalloc's fixed scratch on the current device."""
    st = ctypes.c_int32(0)
    _check(_lib.stlite_device_status(_ptr(ws), _stream(stream), ctypes.byref(st)), "stlite_device_status")
    return int(st.value)


def stlite_score_noalloc(q, k, a_base, stream=None):
    """Window score without a workspace (for callers that cannot allocate
    device memory); see include/stlite.h."""
    sh = make_shape(q, k)
    _check(_lib.stlite_score_noalloc(ctypes.byref(sh), _ptr(q), _ptr(k), _ptr(a_base), _stream(stream)),
           "stlite_score_noalloc")


def stlite_timing_enable(on: bool = True):
    _check(_lib.stlite_timing_enable(1 if on else 0), "stlite_timing_enable")


def stlite_timing_read() -> dict:
    """{kernel name: (launches, total device ms)} since the last read."""
    cap = 64
    buf = (KernelTime * cap)()
    cnt = ctypes.c_int32(0)
    _check(_lib.stlite_timing_read(buf, cap, ctypes.byref(cnt)), "stlite_timing_read")
    return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].total_ms)) for i in range(min(cnt.value, cap))}


# ------------------------------------------------------- convenience layer

def compress_layer(q, k, v, frames, beta=0.2, k_override=0, alpha=1.0, tsg_enable=1, css_enable=1,
                   ws=None, stream=None, tsg_metric=STLITE_TSG_COSINE, fixed_tau=None, base_scorer=STLITE_BASE_WINDOW,
                   abase_norm=STLITE_ABASE_RAW, css_size=3):
    """Allocates outputs (and a workspace if none is given) and runs
    stlite_compress_layer.  Returns (k_out, v_out, idx)."""
    fs = _frames(frames)
    params = make_params(beta, k_override, alpha, tsg_enable, css_enable, tsg_metric, fixed_tau, base_scorer,
                         abase_norm, css_size)
    sh = make_shape(q, k)
    b = stlite_budget(sh.n_tokens, beta, k_override)
    if b < 1:
        raise StliteError(STLITE_EINVAL, "stlite_budget")
    if ws is None:
        ws = workspace(sh, fs, params, device=k.device)
    k_out = torch.empty((b, sh.n_kv_heads, sh.head_dim), dtype=k.dtype, device=k.device)
    v_out = torch.empty_like(k_out)
    idx = torch.empty((sh.n_kv_heads, b), dtype=torch.int32, device=k.device)
    stlite_compress_layer(q, k, v, fs, params, k_out, v_out, idx, ws, stream)
    return k_out, v_out, idx
