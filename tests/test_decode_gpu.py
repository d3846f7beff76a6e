"""Decode attention over a full and a compressed cache (the consumer of the
compressed cache) through the C ABI, against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_00188_gb300 import synth
from parity import exact64, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


def _close(got, ref, v64):
    # fp32 scores and sums: |g - o| <= 1e-3 |o| + 2e-4 max|v| (the output is a
    # convex combination of value rows, so max|v| bounds it)
    tol = 1e-3 * np.abs(ref) + 2e-4 * np.abs(v64).max()
    bad = np.abs(got - ref) > tol
    assert not bad.any(), ("decode mismatch", int(bad.sum()), float(np.abs(got - ref).max()))


@pytest.mark.parametrize("w,hq,hkv,n,dtype", [(1, 28, 4, 1000, torch.bfloat16), (3, 28, 4, 257, torch.bfloat16),
                                              (2, 16, 1, 33, torch.bfloat16), (1, 4, 4, 1, torch.bfloat16),
                                              (1, 28, 4, 20000, torch.bfloat16), (2, 6, 2, 130, torch.bfloat16),
                                              (2, 12, 2, 513, torch.float32), (1, 8, 2, 31, torch.float32)])
def test_decode_matches_oracle(st, w, hq, hkv, n, dtype):
    g = torch.Generator().manual_seed(n * 7 + hq)
    q = torch.randn((w, hq, 128), generator=g).to(dtype).cuda()
    k = torch.randn((n, hkv, 128), generator=g).to(dtype).cuda()
    v = torch.randn((n, hkv, 128), generator=g).to(dtype).cuda()
    sh = st.make_shape(q, k)
    ws = torch.zeros(st.stlite_decode_workspace_size(sh), dtype=torch.uint8, device="cuda")
    out = torch.empty((w, hq, 128), dtype=torch.float32, device="cuda")
    st.stlite_decode_attention(q, k, v, out, ws)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    ref = oracle.decode_attention(exact64(q), exact64(k), exact64(v))
    _close(out.cpu().numpy().astype(np.float64), ref, exact64(v))


def test_decode_workspace_reused(st):
    # one workspace serves many calls, eager and in a replayed graph, and
    # every call equals a call on a fresh workspace, bit for bit
    g = torch.Generator().manual_seed(977)
    w, hq, hkv, n = 2, 28, 4, 3000
    k = torch.randn((n, hkv, 128), generator=g).to(torch.bfloat16).cuda()
    v = torch.randn((n, hkv, 128), generator=g).to(torch.bfloat16).cuda()
    qs = [torch.randn((w, hq, 128), generator=g).to(torch.bfloat16).cuda() for _ in range(3)]
    sh = st.make_shape(qs[0], k)
    nbytes = st.stlite_decode_workspace_size(sh)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    outs = []
    for q in qs + qs:
        out = torch.empty((w, hq, 128), dtype=torch.float32, device="cuda")
        st.stlite_decode_attention(q, k, v, out, ws)
        outs.append(out)
    torch.cuda.synchronize()
    for i, q in enumerate(qs):
        fresh = torch.empty((w, hq, 128), dtype=torch.float32, device="cuda")
        st.stlite_decode_attention(q, k, v, fresh, torch.zeros(nbytes, dtype=torch.uint8, device="cuda"))
        torch.cuda.synchronize()
        assert torch.equal(outs[i], fresh) and torch.equal(outs[i + 3], fresh)
    out = torch.empty((w, hq, 128), dtype=torch.float32, device="cuda")
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        st.stlite_decode_attention(qs[1], k, v, out, ws, stream=stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        st.stlite_decode_attention(qs[1], k, v, out, ws, stream=stream)
    for _ in range(4):
        out.zero_()
        graph.replay()
    torch.cuda.synchronize()
    assert torch.equal(out, outs[1])
    assert st.stlite_device_status(ws) == st.STLITE_OK


def test_decode_over_compressed_cache(st):
    # compress one layer, then decode a probe row over the compacted rows
    wl = synth.scaled("traj50", 4)
    q, k, v = to_device(wl)
    ko, vo, idx = st.compress_layer(q, k, v, wl.frames, beta=wl.beta)
    probe = q[-1:].contiguous()                      # the last window row as the next query
    full = st.decode_attention(probe, k, v)
    comp = st.decode_attention(probe, ko, vo)
    torch.cuda.synchronize()
    _close(comp.cpu().numpy().astype(np.float64),
           oracle.decode_attention(exact64(probe), exact64(ko), exact64(vo)), exact64(vo))
    _close(full.cpu().numpy().astype(np.float64),
           oracle.decode_attention(exact64(probe), exact64(k), exact64(v)), exact64(v))
    assert ko.shape[0] == idx.shape[1] < k.shape[0]


def test_decode_rejects(st):
    q = torch.zeros((1, 32, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((10, 1, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(st.StliteError):
        st.decode_attention(q, k, k)                  # 32 query heads per KV head > 16


@pytest.mark.parametrize("layers,w,hq,hkv,n,dtype", [(28, 1, 28, 4, 3000, torch.bfloat16),
                                                      (5, 2, 12, 2, 1001, torch.bfloat16),
                                                      (34, 1, 8, 2, 300, torch.bfloat16),
                                                      (3, 1, 16, 1, 77, torch.bfloat16),
                                                      (4, 2, 12, 2, 513, torch.float32)])
def test_decode_layers_match_oracle(st, layers, w, hq, hkv, n, dtype):
    """The layer-batched decode (one launch pair per batch of up to 32
    layers; 34 layers take two) against the oracle layer by layer, and
    against the single-layer call within fp32 rounding."""
    g = torch.Generator().manual_seed(layers * 131 + n)
    qs = [torch.randn((w, hq, 128), generator=g).to(dtype).cuda() for _ in range(layers)]
    ks = [torch.randn((n, hkv, 128), generator=g).to(dtype).cuda() for _ in range(layers)]
    vs = [torch.randn((n, hkv, 128), generator=g).to(dtype).cuda() for _ in range(layers)]
    outs, ws = st.decode_attention_layers(qs, ks, vs)
    torch.cuda.synchronize()
    assert st.stlite_device_status(ws) == st.STLITE_OK
    for l in sorted({0, layers // 2, layers - 1}):
        ref = oracle.decode_attention(exact64(qs[l]), exact64(ks[l]), exact64(vs[l]))
        _close(outs[l].cpu().numpy().astype(np.float64), ref, exact64(vs[l]))
    for l in range(layers):
        one = st.decode_attention(qs[l], ks[l], vs[l])
        torch.cuda.synchronize()
        _close(outs[l].cpu().numpy().astype(np.float64), one.cpu().numpy().astype(np.float64), exact64(vs[l]))


def test_decode_layers_in_graph(st):
    """The batched call replays in a CUDA graph with the same bits."""
    g = torch.Generator().manual_seed(5)
    qs = [torch.randn((1, 28, 128), generator=g).to(torch.bfloat16).cuda() for _ in range(6)]
    ks = [torch.randn((2000, 4, 128), generator=g).to(torch.bfloat16).cuda() for _ in range(6)]
    vs = [torch.randn((2000, 4, 128), generator=g).to(torch.bfloat16).cuda() for _ in range(6)]
    outs, ws = st.decode_attention_layers(qs, ks, vs)
    torch.cuda.synchronize()
    ref = [o.clone() for o in outs]
    stream = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    io = list(zip(qs, ks, vs, outs))
    with torch.cuda.stream(stream):
        st.stlite_decode_attention_layers(io, ws, stream)
    stream.synchronize()
    with torch.cuda.graph(graph, stream=stream):
        st.stlite_decode_attention_layers(io, ws, stream)
    for o in outs:
        o.zero_()
    graph.replay()
    torch.cuda.synchronize()
    for o, r in zip(outs, ref):
        assert torch.equal(o, r)
