"""Pins of the oracle's one-output-at-a-time functions (conv_fwd_at, conv_dgrad_at,
conv_wgrad_at, sq_at, rq_at), which check tensors too large for the full loops at sampled
positions.  Each is pinned against torch's fp64 convolution and its two gradients (exact on
these integer inputs) and against the exact-rational quantizer definitions of Eq. (ScaleQ)
and Eqs. (SQ),(SR), independently of the full-tensor oracle functions."""
from fractions import Fraction as Fr

import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import synthetic as S

CASES = [
    O.Conv(2, 9, 11, 16, 8, 3, 3, 1, 1, 1, 1),
    O.Conv(2, 9, 9, 8, 12, 3, 3, 2, 1, 1, 1),      # stride 2, odd extent
    O.Conv(1, 13, 13, 8, 8, 3, 3, 1, 6, 6, 1),     # atrous, most taps outside
    O.Conv(1, 8, 8, 12, 6, 1, 1, 2, 0, 1, 3),      # 1x1 stride 2, groups
    O.Conv(2, 12, 10, 3, 5, 7, 7, 2, 3, 1, 1),     # stem-like
]


def _t(a):
    return torch.from_numpy(np.asarray(a, np.float64))


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_sampled_conv_matches_torch_fp64(ci):
    cv = CASES[ci]
    g = S.rng(300 + ci)
    p, q = cv.pq
    x = S.int8_uniform(g, (cv.n, cv.h, cv.w, cv.c))
    w = S.int8_uniform(g, (cv.k, cv.r, cv.s, cv.c // cv.groups))
    e = S.int8_uniform(g, (cv.n, p, q, cv.k))
    xt, wt, et = (_t(a).permute(0, 3, 1, 2) for a in (x, w, e))
    kw = dict(stride=cv.stride, padding=cv.pad, dilation=cv.dil, groups=cv.groups)
    y = torch.nn.functional.conv2d(xt, wt, **kw).permute(0, 2, 3, 1).numpy().astype(np.int64)
    dx = torch.nn.grad.conv2d_input(xt.shape, wt, et, **kw).permute(0, 2, 3, 1).numpy()
    dw = torch.nn.grad.conv2d_weight(xt, wt.shape, et, **kw).permute(0, 2, 3, 1).numpy()
    for fn, a, b, want in ((O.conv_fwd_at, x, w, y), (O.conv_dgrad_at, e, w, dx),
                           (O.conv_wgrad_at, e, x, dw)):
        want = want.astype(np.int64).ravel()
        # every index (so a wrong decomposition of the flat index cannot hide) in a
        # shuffled order, plus repeats
        idx = np.concatenate([g.permutation(want.size), g.integers(0, want.size, 50)])
        assert np.array_equal(fn(cv, a, b, idx), want[idx]), fn.__name__


def _rhu(v: Fr) -> int:
    return (v + Fr(1, 2)).__floor__()


def test_sq_at_matches_exact_rationals():
    g = S.rng(41)
    for k in (8, 16):
        for relu in (False, True):
            for M in (1, 127, 12345, 2 ** 33 + 5):
                q = g.integers(-M, M + 1, 400)
                qm = np.maximum(q, 0) if relu else q
                lim = 2 ** (k - 1) - 1
                want = [max(-lim, min(lim, _rhu(Fr(int(v), M) * 2 ** (k - 1)))) for v in qm]
                got, s = O.sq_at(q, M, 0.375, k, relu)
                assert got.tolist() == want
                assert s == 0.375 * M * 2.0 ** (1 - k)
    got, s = O.sq_at([5, -5], 0, 0.5, 8)
    assert got.tolist() == [0, 0] and s == 0.5 * 2.0 ** -7


def test_rq_at_definition_and_counter():
    """y = q 2^(k-1)/M rounds up exactly when the element's Philox word u satisfies
    u/2^32 < frac(y); an exact y never rounds; the counter is the element's flat index."""
    g = S.rng(42)
    M, k = 1000003, 8
    q = g.integers(-M, M + 1, 500)
    q[:3] = [M, -M, 0]
    idx = g.integers(0, 10 ** 9, 500)
    got, s = O.rq_at(q, idx, M, 0.5, k, 1, seed=9, layer=4, step=2)
    for v, i, c in zip(q.tolist(), idx.tolist(), got.tolist()):
        y = Fr(v * 2 ** (k - 1), M)
        f = y.__floor__()
        u = O.rq_uniform(9, 4, 2, 0, i)
        want = f + (1 if Fr(u, 2 ** 32) < y - f else 0)
        assert c == max(-127, min(127, want))
    assert got[:3].tolist() == [127, -127, 0]
    assert s == 0.5 * M * 2.0 ** -7
    _, s2 = O.rq_at(q, idx, M, 0.5, k, 2, seed=9, layer=4, step=2)
    assert s2 == 2.0 ** -7


def test_sampled_quantizers_agree_with_full_tensor_ones():
    g = S.rng(43)
    q = g.integers(-2 ** 30, 2 ** 30, 3000)
    M = int(np.abs(q).max())
    full, s_full = O.rq_int(q, 0.25, 8, 1, 5, 6, 7)
    idx = g.permutation(q.size)[:700]
    part, s_part = O.rq_at(q[idx], idx, M, 0.25, 8, 1, 5, 6, 7)
    assert np.array_equal(part, full[idx]) and s_part == s_full
    fs, ss = O.sq_int(q, 0.25, 8, True)
    ps, sps = O.sq_at(q[idx], max(0, int(q.max())), 0.25, 8, True)
    assert np.array_equal(ps, fs[idx]) and sps == ss
