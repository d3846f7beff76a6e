"""The window score without a workspace, for callers that cannot allocate
device memory (allocator callbacks, processes whose device memory another
runtime has fully reserved): its scratch is a fixed device array inside the
library.  Checked through the C ABI against stlite_score, the entry point
that takes a workspace, on two calls in a row; its error word is read back
through stlite_device_status(NULL); and a child process checks that a call in
a second CUDA context (where the library's module, and so the array, is
loaded anew) and a later call back in the first one both match.  This file
is collected last.
"""
import ctypes
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from paper_2603_00188_gb300 import synth
from parity import a_bound, assert_within, to_device

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


@pytest.mark.parametrize("make", [lambda: synth.scaled("traj50", 3), lambda: synth.tiny_ref()],
                         ids=["bf16_traj50_3f", "fp32_tiny_ref"])
def test_score_without_workspace_matches(st, make):
    wl = make()
    q, k, v = to_device(wl)
    sh = st.make_shape(q, k)
    ws = st.workspace(sh, wl.frames)
    ref = torch.empty((sh.n_kv_heads, sh.n_tokens), dtype=torch.float32, device="cuda")
    st.stlite_score(q, k, ref, ws)
    torch.cuda.synchronize()
    r = ref.cpu().numpy()
    for call in range(2):
        out = torch.full_like(ref, float("nan"))
        status = st._lib.stlite_score_noalloc(ctypes.byref(sh), ctypes.c_void_p(q.data_ptr()),
                                              ctypes.c_void_p(k.data_ptr()), ctypes.c_void_p(out.data_ptr()),
                                              ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert status == st.STLITE_OK
        torch.cuda.synchronize()
        # the fixed scratch's error word: no bounded wait ran out
        assert st.stlite_device_status(None) == st.STLITE_OK
        g = out.cpu().numpy()
        for h in range(sh.n_kv_heads):
            assert_within(g[h], r[h], a_bound(r[h]), "A_base (call %d, head %d)" % (call, h))


def test_rejects_beyond_fixed_scratch(st):
    # 1024 KV heads with 512 query rows each need more than the fixed 2 MiB;
    # the buffers are real allocations of the stated shape
    sh = st.Shape(64, 1024 * 4, 1024, 128, 128, st.STLITE_BF16)
    q = torch.zeros((128, 1024 * 4, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((64, 1024, 128), dtype=torch.bfloat16, device="cuda")
    a = torch.zeros((1024, 64), dtype=torch.float32, device="cuda")
    P = ctypes.c_void_p
    assert st._lib.stlite_score_noalloc(ctypes.byref(sh), P(q.data_ptr()), P(k.data_ptr()), P(a.data_ptr()),
                                        None) == st.STLITE_EUNSUPPORTED


_CHILD = r'''
import ctypes, sys
import numpy as np
sys.path.insert(0, ROOT)
from paper_2603_00188_gb300 import stlite as st

cu = ctypes.CDLL("libcuda.so.1")
def ok(r, what):
    assert r == 0, (what, r)
ok(cu.cuInit(0), "cuInit")
dev = ctypes.c_int(0)
ok(cu.cuDeviceGet(ctypes.byref(dev), 0), "cuDeviceGet")
primary = ctypes.c_void_p()
ok(cu.cuDevicePrimaryCtxRetain(ctypes.byref(primary), dev), "retain")
ok(cu.cuCtxSetCurrent(primary), "set primary")

rng = np.random.default_rng(7)
n, hq, hkv, w = 3000, 8, 2, 16
q32 = rng.standard_normal((w, hq, 128)).astype(np.float32)
k32 = rng.standard_normal((n, hkv, 128)).astype(np.float32)
# bf16 bit patterns: values chosen as the upper halves of the fp32 ones
q16 = (q32.view(np.uint32) >> 16).astype(np.uint16)
k16 = (k32.view(np.uint32) >> 16).astype(np.uint16)
fr = st.Frames(0, None, None, None)
cu.cuMemAlloc_v2.argtypes = [ctypes.POINTER(ctypes.c_uint64), ctypes.c_size_t]
cu.cuMemcpyHtoD_v2.argtypes = [ctypes.c_uint64, ctypes.c_void_p, ctypes.c_size_t]
cu.cuMemcpyDtoH_v2.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_size_t]
cu.cuMemsetD8_v2.argtypes = [ctypes.c_uint64, ctypes.c_ubyte, ctypes.c_size_t]
cu.cuMemFree_v2.argtypes = [ctypes.c_uint64]

def run(label, dtype):
    """stlite_score (workspace) and stlite_score_noalloc on buffers of the current context."""
    q, k = (q16, k16) if dtype == st.STLITE_BF16 else (q32, k32)
    sh = st.Shape(n, hq, hkv, 128, w, dtype)
    need = ctypes.c_size_t(0)
    ok(st._lib.stlite_workspace_size(ctypes.byref(sh), ctypes.byref(fr), None, ctypes.byref(need)), "ws size")
    bufs = {}
    for name, nbytes in (("q", q.nbytes), ("k", k.nbytes), ("ref", hkv * n * 4), ("out", hkv * n * 4),
                         ("ws", need.value)):
        p = ctypes.c_uint64(0)
        ok(cu.cuMemAlloc_v2(ctypes.byref(p), nbytes), "alloc " + name)
        bufs[name] = p.value
    ok(cu.cuMemsetD8_v2(bufs["ws"], 0, need.value), "memset ws")
    ok(cu.cuMemcpyHtoD_v2(bufs["q"], q.ctypes.data, q.nbytes), "h2d q")
    ok(cu.cuMemcpyHtoD_v2(bufs["k"], k.ctypes.data, k.nbytes), "h2d k")
    P = ctypes.c_void_p
    ok(st._lib.stlite_score(ctypes.byref(sh), P(bufs["q"]), P(bufs["k"]), P(bufs["ref"]), P(bufs["ws"]),
                            need.value, None), "stlite_score " + label)
    ok(st._lib.stlite_score_noalloc(ctypes.byref(sh), P(bufs["q"]), P(bufs["k"]), P(bufs["out"]), None),
       "stlite_score_noalloc " + label)
    ok(cu.cuCtxSynchronize(), "sync " + label)
    status = ctypes.c_int32(-1)
    ok(st._lib.stlite_device_status(None, None, ctypes.byref(status)), "status " + label)
    assert status.value == 0, (label, status.value)
    ref = np.empty((hkv, n), np.float32)
    out = np.empty((hkv, n), np.float32)
    ok(cu.cuMemcpyDtoH_v2(ref.ctypes.data, bufs["ref"], ref.nbytes), "d2h ref")
    ok(cu.cuMemcpyDtoH_v2(out.ctypes.data, bufs["out"], out.nbytes), "d2h out")
    for p in bufs.values():
        ok(cu.cuMemFree_v2(p), "free")
    err = np.abs(out.astype(np.float64) - ref)
    assert (err <= 1e-3 * np.abs(ref) + 1e-7 * np.abs(ref).max()).all(), (label, float(err.max()))

for dt in (st.STLITE_BF16, st.STLITE_F32):
    run("primary context", dt)
second = ctypes.c_void_p()
ok(cu.cuCtxCreate_v2(ctypes.byref(second), 0, dev), "create")   # made current
for dt in (st.STLITE_BF16, st.STLITE_F32):
    run("second context", dt)
ok(cu.cuCtxDestroy_v2(second), "destroy")
ok(cu.cuCtxSetCurrent(primary), "back to primary")
for dt in (st.STLITE_BF16, st.STLITE_F32):
    run("primary context again", dt)
print("CONTEXTS_OK")
'''


def test_second_context_resolves_its_own_scratch(st):
    """The array lives in the library's module, which each CUDA context loads
    anew: a call in a newly created context must use that context's copy, and
    a later call back in the first context the first one's.  Both calls are
    compared with stlite_score on the same buffers (a child process, so that
    this process's CUDA state is not touched)."""
    code = "ROOT = %r\n" % ROOT + _CHILD
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and "CONTEXTS_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
