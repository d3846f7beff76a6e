"""The window score without a workspace, for callers that cannot allocate
device memory (allocator callbacks, processes whose device memory another
runtime has fully reserved): its scratch is a fixed device array inside the
library.  Checked through the C ABI against stlite_score, the entry point
that takes a workspace, on two calls in a row.  This file is collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2603_00188_gb300 import synth
from parity import a_bound, assert_within, to_device

pytestmark = pytest.mark.gpu


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
        g = out.cpu().numpy()
        for h in range(sh.n_kv_heads):
            assert_within(g[h], r[h], a_bound(r[h]), "A_base (call %d, head %d)" % (call, h))


def test_rejects_beyond_fixed_scratch(st):
    # 1024 KV heads with 512 query rows each need more than the fixed 2 MiB
    sh = st.Shape(64, 1024 * 4, 1024, 128, 128, st.STLITE_BF16)
    p = ctypes.c_void_p(0x10000)
    assert st._lib.stlite_score_noalloc(ctypes.byref(sh), p, p, p, None) == st.STLITE_EUNSUPPORTED
