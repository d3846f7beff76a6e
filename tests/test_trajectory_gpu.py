"""Per-step use across a trajectory: at agent step t the prompt holds frames
0..t-1 of the 50-step trajectory (t * 1,072 tokens), and all 28 layers are
compressed in one stlite_compress_layers call on the first t * 1,072 tokens
of each layer's cache, the last of the t frames being the current one
(Algorithm 1 run once per prefill, as the efficiency study's per-length
latency table does).  These are the calls bench.py's trajectory sweep
times.  Each layer's result is compared with the fp64 oracle under the
matching rules (kept sets equal up to swaps at the B-th score or at gate
flips; compacted rows bit-exact) and with the single-layer call bit for bit.
"""
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
from paper_2603_00188_gb300 import synth
from parity import A_FLOOR, A_RTOL, COS_ATOL, check_kept_sets, exact64

pytestmark = pytest.mark.gpu

LAYERS = 28
STEP_TOKENS = 32 * 32 + 48
BETA = 0.2


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


@pytest.fixture(scope="module")
def cache(st):
    with ThreadPoolExecutor(max_workers=8) as ex:
        wls = list(ex.map(synth.trajectory_50, range(LAYERS)))
    qs = [torch.from_numpy(wl.q).to(torch.bfloat16).cuda() for wl in wls]
    ks = [torch.from_numpy(wl.k).to(torch.bfloat16).cuda() for wl in wls]
    vs = [torch.from_numpy(wl.v).to(torch.bfloat16).cuda() for wl in wls]
    return wls[0].frames, qs, ks, vs


@pytest.mark.parametrize("t", [1, 2, 5, 50])
def test_prefix_step(st, cache, t):
    frames, qs, ks, vs = cache
    n_t = t * STEP_TOKENS
    fs = st.FrameSpec(frames[0][:t], frames[1][:t], frames[2][:t])
    fr_t = (fs.offset, fs.grid_h, fs.grid_w)
    prm = st.make_params(BETA)
    sh = st.make_shape(qs[0], ks[0][:n_t])
    b = st.stlite_budget(n_t, BETA)
    hkv, d = ks[0].shape[1], ks[0].shape[2]
    ws = torch.zeros(LAYERS * st.stlite_workspace_size(sh, fs, prm), dtype=torch.uint8, device="cuda")
    kos = torch.empty((LAYERS, b, hkv, d), dtype=torch.bfloat16, device="cuda")
    vos = torch.empty_like(kos)
    ixs = torch.empty((LAYERS, hkv, b), dtype=torch.int32, device="cuda")
    io = [(qs[l], ks[l][:n_t], vs[l][:n_t], kos[l], vos[l], ixs[l]) for l in range(LAYERS)]
    assert st.stlite_compress_layers(io, fs, prm, ws) == b
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    ig = ixs.cpu().numpy()

    # every layer equals the single-layer call on the same prefix, bit for bit
    for l in range(LAYERS):
        ko1, vo1, ix1 = st.compress_layer(qs[l], ks[l][:n_t], vs[l][:n_t], fs, beta=BETA)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(ix1.cpu().numpy(), ig[l])
        assert torch.equal(ko1.view(torch.int16), kos[l].view(torch.int16))
        assert torch.equal(vo1.view(torch.int16), vos[l].view(torch.int16))

    # against the oracle: every layer for the short prefixes, three layers of
    # the full 50-frame prompt (whose single layers the full-size tests cover)
    check = range(LAYERS) if t <= 5 else (0, 13, 27)
    threads = oracle.host_threads()
    for l in check:
        k64 = exact64(ks[l][:n_t])
        ref = oracle.compress_layer(exact64(qs[l]), k64, fr_t, beta=BETA, threads=threads)
        assert ref["budget"] == b
        for h in range(hkv):
            flips = set()
            if t >= 2:
                flips = set(np.nonzero(np.abs(ref["rho"][h] - ref["tau"][h])
                                       <= A_RTOL * abs(ref["tau"][h]) + COS_ATOL)[0].tolist())
            check_kept_sets(ig[l, h], ref["idx"][h], ref["s"][h], b, s_tol, allowed_extra=flips)
        ko2, vo2 = oracle.gather(ks[l][:n_t].view(torch.int16).cpu().numpy(),
                                 vs[l][:n_t].view(torch.int16).cpu().numpy(), ig[l])
        np.testing.assert_array_equal(kos[l].view(torch.int16).cpu().numpy(), ko2)
        np.testing.assert_array_equal(vos[l].view(torch.int16).cpu().numpy(), vo2)
