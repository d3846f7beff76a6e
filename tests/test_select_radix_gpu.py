"""The exact Top-B of the selection kernel on score distributions aimed at
each branch of its radix select, through stlite_select_topk.

With no frames, TSG and CSS off, every token is text and S = A_base (Eq. 9
with alpha = 0), so the kept set must equal the Top-B of the given scores by
(S descending, index ascending), index for index.  The distributions are
chosen so that the select ends in each of its ways: a bin that holds exactly
the keys still needed after two or three 8-bit passes (the early stop),
bins whose keys tie at the threshold (all four passes and the tie count),
scores one unit in the last place apart, every score equal, and signed
zeros next to negative and positive scores (-0.0 and +0.0 compare equal).
Sizes cover one CTA per problem, clusters, a ragged N and budgets of one,
about a third of N and all of N.
"""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def st():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2603_00188_gb300 import build
    build.build()
    from paper_2603_00188_gb300 import stlite
    return stlite


def _ulps(base, n, rng):
    """n float32 values base, base + 1 ulp, ..., shuffled."""
    b = np.array([base], dtype=np.float32).view(np.uint32)[0]
    v = (b + np.arange(n, dtype=np.uint32)).view(np.float32)
    return rng.permutation(v)


def scores(kind, h, n, seed):
    rng = np.random.default_rng(seed)
    out = np.empty((h, n), dtype=np.float32)
    for i in range(h):
        if kind == "normal":
            x = rng.standard_normal(n).astype(np.float32)
        elif kind == "ulps":
            x = _ulps(0.3 + 0.01 * i, n, rng)
        elif kind == "few_ulps_with_ties":
            # values within 16 ulps of each other: every key shares its top
            # 24 bits, so the last pass decides among large tie groups
            b = np.array([0.7], dtype=np.float32).view(np.uint32)[0]
            x = (b + rng.integers(0, 16, n).astype(np.uint32)).view(np.float32)
        elif kind == "four_values":
            x = rng.choice(np.array([0.25, 0.5, 1.0, 2.0], dtype=np.float32), n)
        elif kind == "all_equal":
            x = np.full(n, 0.125, dtype=np.float32)
        elif kind == "signed_zeros":
            x = rng.choice(np.array([-0.0, 0.0, -1.5, 3.0, -1e-30, 1e-30], dtype=np.float32), n)
        else:
            raise ValueError(kind)
        out[i] = x
    return out


KINDS = ["normal", "ulps", "few_ulps_with_ties", "four_values", "all_equal", "signed_zeros"]


@pytest.mark.parametrize("n,h", [(2048, 2), (5001, 2), (53600, 4)])
@pytest.mark.parametrize("kind", KINDS)
def test_topk_matches_exact_order(st, kind, n, h):
    q = torch.zeros((1, h, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((n, h, 128), dtype=torch.bfloat16, device="cuda")
    none = ([], [], [])
    a = scores(kind, h, n, seed=1000 + n + len(kind))
    a_d = torch.from_numpy(a).cuda()
    for b in sorted({1, n // 3 + 1, n}):
        prm = st.make_params(1.0, k_override=b, alpha=0.0, tsg_enable=0, css_enable=0)
        sh = st.make_shape(q, k)
        ws = st.workspace(sh, none, prm)
        idx = torch.empty((h, b), dtype=torch.int32, device="cuda")
        score = torch.empty_like(a_d)
        st.stlite_select_topk(q, k, none, prm, a_d, None, None, b, idx, score, ws)
        torch.cuda.synchronize()
        s = score.cpu().numpy()
        # S = A (text tokens; -0.0 folded onto +0.0)
        np.testing.assert_array_equal(s, a + np.float32(0.0))
        np.testing.assert_array_equal(idx.cpu().numpy(), oracle.topk(a.astype(np.float64), b),
                                      err_msg="%s n=%d b=%d" % (kind, n, b))
