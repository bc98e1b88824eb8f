"""Pins of the CPU oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: every expected value comes from
an independent route (exact rational arithmetic with ``fractions``, numpy /
torch library routines, closed forms, invariants, or values the paper fixes).
"""
from fractions import Fraction as Fr
import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import synthetic as S


def rhu_exact(v: Fr) -> int:
    """floor(v + 1/2) on an exact rational (Eq. (UQ))."""
    return math.floor(v + Fr(1, 2))


def clip(c, k):
    lim = 2 ** (k - 1) - 1
    return max(-lim, min(lim, c))


# ----------------------------------------------------------------- UQ (P1, P2)

@pytest.mark.parametrize("k", [2, 4, 8, 16, 24])
def test_uq_special_values(k):
    d = 2.0 ** (1 - k)
    x = np.array([0.0, 1.0, -1.0, d / 2, -d / 2, 3 * d / 2, -3 * d / 2, 5.0, -5.0, 1 - d,
                  -(1 - d)], np.float32)
    lim = 2 ** (k - 1) - 1
    want = [0, lim, -lim, 1, 0, min(2, lim), -1, lim, -lim, lim, -lim]
    assert O.uq(x, k).tolist() == want


def _near_ties(g, k, n):
    """Floats at, and one ulp either side of, the rounding ties (j + 1/2) * Delta."""
    d = 2.0 ** (1 - k)
    j = g.integers(-(2 ** (k - 1)) - 2, 2 ** (k - 1) + 2, size=n)
    t = ((j + 0.5) * d).astype(np.float32)
    return np.concatenate([t, np.nextafter(t, np.float32(np.inf)),
                           np.nextafter(t, np.float32(-np.inf))])


@pytest.mark.parametrize("k", [4, 8, 16, 24])
def test_uq_matches_exact_rationals(k):
    g = S.rng(k)
    x = np.concatenate([S.float_uniform(g, 3000, -1.2, 1.2), _near_ties(g, k, 1000),
                        np.array([np.float32(0.49999997) * 2.0 ** (1 - k)], np.float32),
                        (g.standard_normal(500) * 1e-30).astype(np.float32)])
    got = O.uq(x, k)
    want = [clip(rhu_exact(Fr(float(v)) * 2 ** (k - 1)), k) for v in x]
    assert got.tolist() == want


@pytest.mark.parametrize("k", [8, 16])
def test_uq2_is_twice_uq_of_half(k):
    g = S.rng(100 + k)
    x = np.concatenate([S.float_uniform(g, 3000, -2.5, 2.5), _near_ties(g, k, 500) * 2])
    got = O.uq2(x, k)
    want = [clip(rhu_exact(Fr(float(v)) / 2 * 2 ** (k - 1)), k) for v in x]
    assert got.tolist() == want
    # value grid: 2 * UQ(x/2) has step 2^(2-k), range +-2(1 - Delta)
    assert np.abs(got).max() <= 2 ** (k - 1) - 1


@pytest.mark.parametrize("k", [4, 8, 16])
def test_uq_idempotent_and_in_range(k):
    g = S.rng(7 * k)
    x = S.float_uniform(g, 20000, -3, 3)
    c = O.uq(x, k)
    assert np.abs(c).max() <= 2 ** (k - 1) - 1
    v = (c.astype(np.float64) * 2.0 ** (1 - k)).astype(np.float32)
    assert np.array_equal(O.uq(v, k), c)


# ----------------------------------------------------------------- SQ (P3, A4)

def sq_exact_int(q, k, relu=False):
    q = [max(0, int(v)) if relu else int(v) for v in q]
    M = max(abs(v) for v in q)
    if M == 0:
        return [0] * len(q)
    return [clip(rhu_exact(Fr(v, M) * 2 ** (k - 1)), k) for v in q]


@pytest.mark.parametrize("k", [4, 8, 16])
@pytest.mark.parametrize("relu", [False, True])
def test_sq_int_matches_exact_rationals(k, relu):
    g = S.rng(11 + k + relu)
    for M in (1, 3, 127, 1000, 2 ** 20 + 7, 404644352):
        q = g.integers(-M, M + 1, size=600)
        q[0] = M
        got, s = O.sq_int(q, 0.25, k, relu)
        assert got.tolist() == sq_exact_int(q, k, relu)
        Mq = max(0, int(q.max())) if relu else int(np.abs(q).max())
        assert s == 0.25 * Mq * 2.0 ** (1 - k)


def test_sq_max_element_maps_to_top_code():
    # the largest element lands on floor(2^(k-1) + 1/2) = 2^(k-1), clipped to 2^(k-1)-1
    c, _ = O.sq_int([5, -3, 0, 17], 1.0, 8)
    assert c[3] == 127
    c, _ = O.sq_int([5, -3, 0, -17], 1.0, 8)
    assert c[3] == -127
    c, s = O.sq_int([0, 0, 0], 0.5, 8)
    assert c.tolist() == [0, 0, 0] and s == 0.5 * 2 ** -7


def test_sq_not_idempotent():
    # Scale quantization rescales by 128/127 after the top code is clipped,
    # so applying SQ8 to an SQ8 output moves code 64 to 65.
    c, _ = O.sq_int([127, 64, -5], 1.0, 8)
    assert c.tolist() == [127, 65, -5]


@pytest.mark.parametrize("k", [8, 16])
def test_sq_float_matches_exact_rationals(k):
    g = S.rng(3 + k)
    x = np.concatenate([S.float_uniform(g, 2000, -3, 3), np.float32([2.75, -1.0, 0.0])])
    S_ = np.float32(np.abs(x).max())
    # plant exact ties: x/S * 2^(k-1) = j + 1/2
    j = g.integers(-(2 ** (k - 1)), 2 ** (k - 1) - 1, size=200)
    ties = ((j + 0.5) / 2 ** (k - 1) * float(S_)).astype(np.float32)
    x = np.concatenate([x, ties])
    got, s = O.sq_float(x, k)
    Sx = Fr(float(np.abs(x).max()))
    want = [clip(rhu_exact(Fr(float(v)) / Sx * 2 ** (k - 1)), k) for v in x]
    assert got.tolist() == want
    assert s == float(np.abs(x).max()) * 2.0 ** (1 - k)


# ----------------------------------------------------------------- RQ (P4)

def test_philox_matches_numpy():
    g = S.rng(5)
    for _ in range(20):
        ctr = g.integers(0, 2 ** 63, size=4, dtype=np.uint64)
        key = g.integers(0, 2 ** 63, size=2, dtype=np.uint64)
        if ctr[0] == 0:
            continue
        # numpy's Philox advances word 0 of its counter before producing a block
        prev = ctr.copy()
        prev[0] -= np.uint64(1)
        want = np.random.Philox(key=key, counter=prev).random_raw(4)
        assert O.philox(ctr, key).tolist() == want.tolist()
    # published known-answer vector of Philox4x64-10 (zero counter and key)
    assert [hex(int(v)) for v in O.philox([0, 0, 0, 0], [0, 0])] == [
        "0x16554d9eca36314c", "0xdb20fe9d672d0fdc", "0xd7e772cee186176b", "0x7e68b68aec7ba23b"]


def test_rq_exact_values_never_round():
    # q * 2^(k-1) / M integral -> the stochastic rounding has nothing to round
    M = 2 ** 10
    q = np.arange(-M, M + 1, 8, dtype=np.int64)
    for step in range(5):
        c, s = O.rq_int(q, 1.0, 8, 2, seed=9, layer=3, step=step)
        assert c.tolist() == [clip(int(v) * 2 ** 7 // M, 8) for v in q]
        assert s == 2.0 ** -7


def test_rq_unbiased():
    # E[Round(y)] = y (Eq. (SR)); y = q * 128 / M with a fractional part
    M = 1000
    q = np.array([1, 3, 7, 333, -333, -1, 990, -990, 500], np.int64)
    q = np.concatenate([q, [M]])
    n = 4000
    acc = np.zeros(q.size)
    for step in range(n):
        c, _ = O.rq_int(q, 1.0, 8, 2, seed=1, layer=0, step=step)
        acc += c
    mean = acc / n
    y = q * 128 / M
    y_clip = np.clip(y, -127, 127)
    frac = y - np.floor(y)
    sd = np.sqrt(frac * (1 - frac) / n) + 1e-12
    ok = np.abs(mean[:-1] - y[:-1]) <= 5 * sd[:-1] + 1e-9
    assert ok.all(), (mean, y)
    assert mean[-1] == y_clip[-1]  # the max element: 128 clipped to 127 every time


def test_rq_gq1_gq2_scales():
    q = np.array([-40, 10, 0, 80], np.int64)
    _, s1 = O.rq_int(q, 0.5, 8, 1, 0, 0, 0)
    _, s2 = O.rq_int(q, 0.5, 8, 2, 0, 0, 0)
    assert s1 == 0.5 * 80 * 2 ** -7   # Eq. (GQ1): Scale(G) kept
    assert s2 == 2 ** -7              # Eq. (GQ2): magnitude dropped


def test_rq_probability_matches_fraction():
    # for one element, over many steps the fraction of round-ups is rem/M
    M, q = 7, 3  # y = 3*128/7 = 54.857..., rem/M = 6/7
    qs = np.array([q, M], np.int64)
    ups = 0
    n = 20000
    for step in range(n):
        c, _ = O.rq_int(qs, 1.0, 8, 2, seed=77, layer=1, step=step)
        ups += int(c[0] == 55)
        assert c[0] in (54, 55)
    p = 6 / 7
    assert abs(ups / n - p) < 5 * math.sqrt(p * (1 - p) / n)


# ----------------------------------------------------------------- weights, update (P11)

def test_master_to_forward_weights():
    g = S.rng(21)
    m = O.uq(S.he_weights(g, 5000, 9), 24)
    m[:4] = [2 ** 15, -(2 ** 15), 2 ** 23 - 1, -(2 ** 23 - 1)]
    got = O.requant_master(m)
    want = [clip(rhu_exact(Fr(int(v), 2 ** 16)), 8) for v in m]
    assert got.tolist() == want
    assert got[:4].tolist() == [1, 0, 127, -127]


def test_update_gq2_shift_identity_and_clip():
    g = S.rng(22)
    m = O.uq(S.he_weights(g, 4000, 64), 24)
    gc = S.int8_uniform(g, 4000).astype(np.int32)
    for e in (6, 10, 16):
        m2, wq = O.update(m, gc, 2.0 ** -7, e)
        # GQ2: G_q = c * 2^-7, lr = 2^-e -> Delta W code = c * 2^(16-e) exactly
        want = np.clip(m.astype(np.int64) - gc.astype(np.int64) * 2 ** (16 - e),
                       -(2 ** 23 - 1), 2 ** 23 - 1)
        assert np.array_equal(m2, want)
        assert np.array_equal(wq, O.requant_master(want))
    m = np.array([2 ** 23 - 5, -(2 ** 23 - 5)], np.int32)
    m2, _ = O.update(m, np.array([-127, 127], np.int32), 2.0 ** -7, 0)
    assert m2.tolist() == [2 ** 23 - 1, -(2 ** 23 - 1)]


def test_update_gq1_rounds_half_up():
    # G_q * lr * 2^23 = c * s * 2^(23-e); pick s so the product sits on ties
    m = np.zeros(4, np.int32)
    c = np.array([1, -1, 3, -3], np.int32)
    m2, _ = O.update(m, c, 2.0 ** -24, 0)   # 2^-24 * 2^23 = 1/2 per unit
    assert m2.tolist() == [-1, 0, -2, 1]    # dW = rhu(0.5)=1, rhu(-0.5)=0, rhu(1.5)=2, rhu(-1.5)=-1


# ----------------------------------------------------------------- conv (P5, P6)

CONV_CASES = [
    O.Conv(2, 7, 9, 16, 8, 3, 3, 1, 1, 1, 1),
    O.Conv(1, 9, 8, 8, 12, 3, 3, 2, 1, 1, 1),
    O.Conv(2, 11, 10, 8, 8, 3, 3, 1, 2, 2, 1),
    O.Conv(1, 8, 8, 12, 6, 1, 1, 1, 0, 1, 3),
    O.Conv(1, 10, 10, 6, 4, 5, 5, 2, 2, 1, 2),
    O.Conv(1, 13, 13, 4, 4, 3, 3, 1, 6, 6, 1),   # atrous, mostly padding
    O.Conv(2, 6, 6, 3, 5, 7, 7, 2, 3, 1, 1),     # stem-like, C=3
]


def _conv_inputs(cv, seed):
    g = S.rng(seed)
    p, q = cv.pq
    x = S.int8_uniform(g, (cv.n, cv.h, cv.w, cv.c))
    w = S.int8_uniform(g, (cv.k, cv.r, cv.s, cv.c // cv.groups))
    e = S.int8_uniform(g, (cv.n, p, q, cv.k))
    return x, w, e


def _torch(a):
    return torch.from_numpy(np.asarray(a, np.float64))


@pytest.mark.parametrize("ci", range(len(CONV_CASES)))
def test_conv_matches_torch_fp64(ci):
    cv = CONV_CASES[ci]
    x, w, e = _conv_inputs(cv, ci)
    xt = _torch(x).permute(0, 3, 1, 2)
    wt = _torch(w).permute(0, 3, 1, 2)
    y = torch.nn.functional.conv2d(xt, wt, stride=cv.stride, padding=cv.pad, dilation=cv.dil,
                                   groups=cv.groups).permute(0, 2, 3, 1).numpy()
    assert np.array_equal(O.conv_fwd(cv, x, w), y.astype(np.int64))
    et = _torch(e).permute(0, 3, 1, 2)
    dx = torch.nn.grad.conv2d_input(xt.shape, wt, et, stride=cv.stride, padding=cv.pad,
                                    dilation=cv.dil, groups=cv.groups).permute(0, 2, 3, 1).numpy()
    assert np.array_equal(O.conv_dgrad(cv, e, w), dx.astype(np.int64))
    dw = torch.nn.grad.conv2d_weight(xt, wt.shape, et, stride=cv.stride, padding=cv.pad,
                                     dilation=cv.dil, groups=cv.groups).permute(0, 2, 3, 1).numpy()
    assert np.array_equal(O.conv_wgrad(cv, e, x), dw.astype(np.int64))


@pytest.mark.parametrize("ci", range(len(CONV_CASES)))
def test_conv_adjoint_identities(ci):
    cv = CONV_CASES[ci]
    x, w, e = _conv_inputs(cv, 50 + ci)
    y = O.conv_fwd(cv, x, w)
    dx = O.conv_dgrad(cv, e, w)
    dw = O.conv_wgrad(cv, e, x)
    a = int((y.astype(np.int64) * e.astype(np.int64)).sum())
    b = int((x.astype(np.int64) * dx.astype(np.int64)).sum())
    c = int((w.astype(np.int64) * dw).sum())
    assert a == b == c


def test_conv_1x1_is_integer_gemm():
    cv = O.Conv(3, 5, 7, 24, 10, 1, 1)
    x, w, _ = _conv_inputs(cv, 9)
    y = O.conv_fwd(cv, x, w)
    want = x.reshape(-1, 24).astype(np.int64) @ w.reshape(10, 24).astype(np.int64).T
    assert np.array_equal(y.reshape(-1, 10), want)


def test_conv_brute_force_tiny():
    cv = O.Conv(1, 3, 4, 2, 2, 2, 3, 1, 1, 2, 1)
    x, w, _ = _conv_inputs(cv, 13)
    p, q = cv.pq
    y = O.conv_fwd(cv, x, w)
    for pp in range(p):
        for qq in range(q):
            for k in range(2):
                s = 0
                for r in range(2):
                    for t in range(3):
                        h, ww = pp + 2 * r - 1, qq + 2 * t - 1
                        if 0 <= h < 3 and 0 <= ww < 4:
                            s += sum(int(x[0, h, ww, c]) * int(w[k, r, t, c]) for c in range(2))
                assert y[0, pp, qq, k] == s


def test_int32_accumulation_bound_largest_layer():
    # fc6 of FCN-VGG16: C*R*S = 512*7*7 = 25088; all-(+-127) operands stay below 2^31
    cv = O.Conv(1, 7, 7, 512, 2, 7, 7)
    x = np.full((1, 7, 7, 512), 127, np.int8)
    w = np.full((2, 7, 7, 512), 127, np.int8)
    w[1] = -127
    y = O.conv_fwd(cv, x, w)
    assert y.reshape(-1).tolist() == [25088 * 16129, -25088 * 16129]
    assert 25088 * 16129 < 2 ** 31


def test_wgrad_exceeds_int32_and_is_exact():
    cv = O.Conv(1, 512, 512, 1, 1, 1, 1)
    x = np.full((1, 512, 512, 1), 127, np.int8)
    e = np.full((1, 512, 512, 1), -127, np.int8)
    dw = O.conv_wgrad(cv, e, x)
    assert int(dw.reshape(-1)[0]) == -262144 * 16129 and 262144 * 16129 > 2 ** 31


# ----------------------------------------------------------------- L1BN forward (P7, P8, P9)

def float_l1bn(x, eps):
    """Eqs. (BN2),(BN4),(BN5) in fp64, per channel of x[m, C]."""
    mu = x.mean(axis=0)
    sig = np.abs(x - mu).mean(axis=0)
    return (x - mu) / (sig + eps), mu, sig


def _bn_case(seed, m=600, C=12, spread=3000, offset=500):
    g = S.rng(seed)
    acc = (g.standard_normal((m, C)) * spread + g.integers(-offset, offset + 1, C)).astype(np.int32)
    gam, bet = S.bn_gamma_beta_codes(g, C)
    return acc, gam, bet


def test_float_l1bn_identities():
    acc, _, _ = _bn_case(1)
    x = acc * 2.0 ** -14
    eps = 2.0 ** -14
    xh, mu, sig = float_l1bn(x, eps)
    assert np.allclose((x - mu).sum(axis=0), 0, atol=1e-9)
    assert np.allclose(np.abs(xh).mean(axis=0), sig / (sig + eps), rtol=1e-12)


def test_bn_sigma_and_mu_codes_exact():
    # mu_q, sigma_q codes against exact rationals of Eqs. (BN2),(BN5) + the QBN block
    acc, gam, bet = _bn_case(2)
    s_acc = 2.0 ** -13
    r = O.bn_fwd(acc, s_acc, gam, bet)
    m = acc.shape[0]
    for c in range(acc.shape[1]):
        col = [int(v) for v in acc[:, c]]
        mu = Fr(sum(col), m) * Fr(s_acc)
        sig = sum(abs(Fr(v) * Fr(s_acc) - mu) for v in col) / m
        # fp64 evaluation of mu, sigma may differ from exact only far below the grid
        assert abs(r.c_mu[c] - clip(rhu_exact(mu * 2 ** 14), 16)) <= 0
        assert abs(r.c_sigma[c] - clip(rhu_exact(sig * 2 ** 14), 16)) <= 0


@pytest.mark.parametrize("seed", [3, 4, 5])
def test_int_l1bn_within_bound_of_float_l1bn(seed):
    acc, gam, bet = _bn_case(seed)
    s_acc = 2.0 ** -12
    r = O.bn_fwd(acc, s_acc, gam, bet)
    eps = 2.0 ** -14
    x = acc * s_acc
    xh_f, mu, sig = float_l1bn(x, eps)
    den_q = (r.c_sigma + 1) * 2.0 ** -14
    # |xhat_int - xhat_float| <= 2^-15 (1 + |xhat|) / (sigma_q + eps) (mu_q, sigma_q half
    # steps) + half an X step; the clip of Eq. (UQ) at 1 - Delta costs the top code a
    # whole step (the element at Scale lands on 2^(k-1) and is clipped to 2^(k-1) - 1).
    step = np.where(np.abs(r.X) == 2 ** 15 - 1, 1.0, 0.5)
    bound = 2.0 ** -15 * (1 + np.abs(xh_f)) / den_q + r.s_xhat * (step + 2 ** -8) + 1e-12
    err = np.abs(r.X * r.s_xhat - xh_f)
    assert (err <= bound).all(), err.max()
    gq = gam * 2.0 ** -6
    bq = bet * 2.0 ** -6
    y_f = gq * xh_f + bq
    y_i = gq * (r.X * r.s_xhat) + bq
    assert (np.abs(y_i - y_f) <= np.abs(gq) * bound + 1e-12).all()


@pytest.mark.parametrize("seed", [6, 7])
def test_int_l1bn_fixed_point_vs_exact_rationals(seed):
    # X and A of the oracle vs SQ evaluated with exact rationals (same mu_q,
    # sigma_q codes and s_acc): at most one code apart, and rarely.
    acc, gam, bet = _bn_case(seed, m=300, C=8)
    s_acc = 2.0 ** -11 * 3
    r = O.bn_fwd(acc, s_acc, gam, bet)
    C = acc.shape[1]
    sa = Fr(s_acc)
    muq = [Fr(int(c), 2 ** 14) for c in r.c_mu]
    den = [Fr(int(c) + 1, 2 ** 14) for c in r.c_sigma]
    xh = [[(int(acc[i, c]) * sa - muq[c]) / den[c] for c in range(C)] for i in range(acc.shape[0])]
    M = max(abs(v) for row in xh for v in row)
    X = np.array([[clip(rhu_exact(v / M * 2 ** 15), 16) for v in row] for row in xh])
    dX = np.abs(X - r.X)
    assert dX.max() <= 1 and (dX > 0).mean() < 1e-3
    # A from the oracle's X with exact rationals
    sX = Fr(r.s_xhat)
    y = [[Fr(int(gam[c]), 64) * int(r.X[i, c]) * sX + Fr(int(bet[c]), 64) for c in range(C)]
         for i in range(acc.shape[0])]
    My = max(max(v, 0) for row in y for v in row)
    A = np.array([[max(0, min(127, rhu_exact(max(v, 0) / My * 128))) for v in row] for row in y])
    dA = np.abs(A - r.A)
    assert dA.max() <= 1 and (dA > 0).mean() < 1e-3
    assert r.A.max() == 127 and r.A.min() >= 0


def test_bn_degenerate_constant_channel():
    # a channel with all-equal accumulators: sigma_B = 0, sigma_q = 0, xhat = (x - mu_q)/eps
    acc = np.zeros((50, 2), np.int32)
    acc[:, 1] = np.arange(50) - 25
    r = O.bn_fwd(acc, 2.0 ** -10, [64, 64], [0, 0])
    assert r.c_sigma[0] == 0 and r.c_mu[0] == 0
    assert (r.X[:, 0] == 0).all()


def test_u128_to_double_correctly_rounded():
    g = S.rng(31)
    vals = [2 ** 64, 2 ** 64 + 1, 2 ** 100 + 2 ** 47, 2 ** 100 + 2 ** 47 + 1, 2 ** 77 - 1,
            (2 ** 53 + 1) * 2 ** 40, (2 ** 53 + 3) * 2 ** 40]
    vals += [int(g.integers(0, 2 ** 62)) * int(g.integers(0, 2 ** 40)) for _ in range(200)]
    for v in vals:
        assert O.u128_to_double(v) == float(v)


# ----------------------------------------------------------------- L1BN backward (P10)

def float_l1bn_bwd(g, xh, den):
    """d x_i = (1/den)[g_i - mean g - mean(g xhat)(sgn_i - mean sgn)] per channel."""
    sg = np.sign(xh)
    return (g - g.mean(0) - (g * xh).mean(0) * (sg - sg.mean(0))) / den


def test_l1bn_backward_formula_finite_differences():
    g = S.rng(40)
    m, C = 40, 3
    x = g.standard_normal((m, C))
    eps = 1e-3
    up = g.standard_normal((m, C))

    def loss(xx):
        xh, _, _ = float_l1bn(xx, eps)
        return (xh * up).sum()

    xh, mu, sig = float_l1bn(x, eps)
    ana = float_l1bn_bwd(up, xh, sig + eps)
    num = np.zeros_like(x)
    h = 1e-6
    for i in range(m):
        for c in range(C):
            xp = x.copy(); xp[i, c] += h
            xm = x.copy(); xm[i, c] -= h
            num[i, c] = (loss(xp) - loss(xm)) / (2 * h)
    assert np.allclose(ana, num, rtol=1e-5, atol=1e-6)
    assert np.allclose(ana.sum(0), 0, atol=1e-9)   # the mean is removed: sum_i dL/dx_i = 0


@pytest.mark.parametrize("k_e2", [16, 8])
def test_bn_backward_vs_float_formula(k_e2):
    acc, gam, bet = _bn_case(41, m=500, C=6)
    s_acc = 2.0 ** -12
    r = O.bn_fwd(acc, s_acc, gam, bet)
    g = S.rng(42)
    eA = S.int8_uniform(g, acc.shape)
    s_e = 2.0 ** -20
    E, s_E, dg, db = O.bn_bwd(eA, s_e, r.A, r.X, r.s_xhat, gam, r.c_sigma, k_e2=k_e2)
    ey = np.where(r.A > 0, eA.astype(np.int64), 0)
    assert np.array_equal(db, ey.sum(0))
    assert np.array_equal(dg, (ey * r.X.astype(np.int64)).sum(0))
    # E2 = SQ_{k_e2}(gamma_q e_y) with exact rationals
    z = ey * gam[None, :].astype(np.int64)
    E2 = np.array(sq_exact_int(z.reshape(-1), k_e2)).reshape(z.shape)
    s_e2 = s_e * 2.0 ** -6 * np.abs(z).max() * 2.0 ** (1 - k_e2)
    den = (r.c_sigma + 1) * 2.0 ** -14
    dx = float_l1bn_bwd(E2 * s_e2, r.X * r.s_xhat, den)
    M = np.abs(dx).max()
    want = np.clip(np.floor(dx / M * 128 + 0.5), -127, 127)
    d = np.abs(want - E)
    assert d.max() <= 1 and (d > 0).mean() < 2e-3
    assert abs(s_E - M * 2 ** -7) <= 1e-12 * M


def test_relu_bwd_mask():
    eA = np.array([5, -3, 7, 0, -9], np.int8)
    A = np.array([1, 0, 127, 3, 0], np.int8)
    assert O.relu_bwd(eA, A).tolist() == [5, 0, 7, 0, 0]


def test_image_input_quantization_exact():
    g = S.rng(60)
    img = S.images_u8(g, 2, 5, 7)
    img[0, 0, 0, 0] = 200
    img = np.minimum(img, 200).astype(np.uint8)
    codes, s = O.quantize_image_u8(img, 4)
    P = int(img.max())
    want = [clip(rhu_exact(Fr(int(p), 255) / Fr(P, 255) * 128), 8) for p in img.reshape(-1)]
    assert codes[..., :3].reshape(-1).tolist() == want
    assert (codes[..., 3] == 0).all()
    assert s == P / 255 * 2 ** -7


# ----------------------------------------------------------------- network glue

def test_maxpool_matches_torch_and_routes_first_max():
    g = S.rng(70)
    x = S.int8_uniform(g, (2, 9, 8, 5), -5, 5)   # many ties
    for k, s, p in ((2, 2, 0), (3, 2, 1)):
        y, a = O.maxpool_fwd(x, k, s, p)
        t = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
        want = torch.nn.functional.max_pool2d(t, k, s, p).permute(0, 2, 3, 1).numpy()
        assert np.array_equal(y, want.astype(np.int8))
        e = S.int8_uniform(g, y.shape)
        ex = O.maxpool_bwd(e, a, x.shape, k, s, p)
        # the routed error sums to the output error (every window has a maximum)
        assert ex.sum(dtype=np.int64) == e.sum(dtype=np.int64)
        # first maximum in scan order (ties): check a few windows by hand
        for (b, i, j, c) in [(0, 0, 0, 0), (1, 1, 2, 3), (0, 3, 3, 4)]:
            win = [(r, q) for r in range(k) for q in range(k)
                   if 0 <= i * s + r - p < 9 and 0 <= j * s + q - p < 8]
            vals = [x[b, i * s + r - p, j * s + q - p, c] for r, q in win]
            r, q = win[int(np.argmax(vals))]
            assert a[b, i, j, c] == r * k + q


@pytest.mark.parametrize("k,s,p", [(2, 2, 0), (3, 2, 1), (3, 1, 1), (2, 3, 0), (3, 3, 1)])
def test_maxpool_backward_matches_autograd_without_ties(k, s, p):
    """Distinct values in every channel plane, so each window has one maximum: the routed
    errors (summed where windows overlap) are torch's max_pool2d gradient."""
    g = S.rng(72 + 10 * k + s)
    n, h, w, c = 2, 7, 6, 3
    x = np.empty((n, h, w, c), np.int8)
    for b in range(n):
        for ch in range(c):
            x[b, :, :, ch] = g.permutation(np.arange(-127, 128))[:h * w].reshape(h, w)
    y, a = O.maxpool_fwd(x, k, s, p)
    t = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2).requires_grad_(True)
    ty = torch.nn.functional.max_pool2d(t, k, s, p)
    assert np.array_equal(y, ty.detach().permute(0, 2, 3, 1).numpy().astype(np.int8))
    e = S.int8_uniform(g, y.shape)
    ty.backward(torch.from_numpy(e.astype(np.float64)).permute(0, 3, 1, 2))
    want = t.grad.permute(0, 2, 3, 1).numpy()
    assert np.array_equal(O.maxpool_bwd(e, a, x.shape, k, s, p), want.astype(np.int32))


def test_mse_grad_exact_rationals():
    g = S.rng(71)
    z = S.int8_uniform(g, (2, 7, 5, 6))
    lab = g.integers(0, 6, size=(2, 7, 5)).astype(np.uint8)
    lab[0, 0, 0] = 255     # no target at this pixel
    s_z = 3.0 * 2.0 ** -9
    E, s = O.mse_grad(z, s_z, lab)
    sz = Fr(s_z)
    vals = [[(int(z[idx + (c,)]) * sz - (1 if lab[idx] == c else 0)) for c in range(6)]
            for idx in np.ndindex(2, 7, 5)]
    M = max(abs(v) for row in vals for v in row)
    want = np.array([[clip(rhu_exact(v / M * 128), 8) for v in row] for row in vals])
    d = np.abs(want - E.reshape(-1, 6))
    assert d.max() <= 1 and (d > 0).mean() < 1e-3
    assert s == float(M) * 2 ** -7


def test_dgrad_exceeds_int32_and_is_exact():
    # 3x3 image, 7x7 kernel, pad 3: every one of the 9 output pixels reaches every
    # input pixel, so dx = 9 * k * 127^2 in closed form (beyond 2^31 for k = 20000)
    cv = O.Conv(1, 3, 3, 2, 20000, 7, 7, 1, 3)
    e = np.full((1, 3, 3, 20000), 127, np.int8)
    w = np.full((20000, 7, 7, 2), 127, np.int8)
    w[..., 1] = -127
    dx = O.conv_dgrad(cv, e, w)
    assert (dx[..., 0] == 9 * 20000 * 16129).all() and (dx[..., 1] == -9 * 20000 * 16129).all()
