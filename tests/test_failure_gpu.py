"""The failure path of the kernels' bounded waits, exercised without faulting
or hanging the GPU: a diagnostic kernel waits, through the library's own
bounded wait, on a barrier that nothing completes.  The wait must give up
after its limit, the host must read STLITE_ETIMEOUT from the error word (once:
the read clears it), and the context must stay usable: a compression on the
same device afterwards runs clean and gives the same result as before."""
import time

import numpy as np
import pytest
import torch

from paper_2603_00188_gb300 import synth
from parity import to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


def test_bounded_wait_runs_out_and_reports(st):
    wl = synth.scaled("traj50", 3)
    q, k, v = to_device(wl)
    ko0, vo0, idx0 = st.compress_layer(q, k, v, wl.frames, beta=wl.beta)
    torch.cuda.synchronize()
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    assert st.stlite_device_status(ws) == st.STLITE_OK
    limit_ns = 20_000_000   # 20 ms
    t0 = time.perf_counter()
    st.stlite_selftest_wait_timeout(ws, limit_ns)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert elapsed >= limit_ns * 1e-9 * 0.9          # it did wait for its limit
    assert elapsed < 10.0                             # and it ended by itself
    assert st.stlite_device_status(ws) == st.STLITE_ETIMEOUT
    assert st.stlite_device_status(ws) == st.STLITE_OK   # the read cleared it
    # the context is still usable: the same compression, bit for bit, clean
    prm = st.make_params(wl.beta)
    ws2 = st.workspace(st.make_shape(q, k), wl.frames, prm)
    ko1, vo1, idx1 = st.compress_layer(q, k, v, wl.frames, beta=wl.beta, ws=ws2)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws2) == st.STLITE_OK
    assert torch.equal(idx0, idx1) and torch.equal(ko0.view(torch.int16), ko1.view(torch.int16))


def test_selftest_rejects_on_host(st):
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    for limit in (0, 999, 3_000_000_000):
        with pytest.raises(st.StliteError):
            st.stlite_selftest_wait_timeout(ws, limit)
