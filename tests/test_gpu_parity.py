"""Parity of the CUDA path (through the C ABI) with the CPU oracle, element by element.

Integer outputs must be bit-exact; fp64 scale outputs must be equal (0 ULP): both
sides evaluate the same fixed-order fp64 steps.  Inputs come from the seeded
generators only.  Sizes span several tiles and a ragged tail.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import iq
from paper_2011_14504_gb300 import synthetic as S

pytestmark = pytest.mark.gpu

DEV = "cuda"


def dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(DEV)


def dscal(v=0.0):
    return torch.tensor([v], dtype=torch.float64, device=DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


# ----------------------------------------------------------------- quantizers

@pytest.mark.parametrize("k", [8, 16, 24])
@pytest.mark.parametrize("mode", [iq.IQ_MODE_UQ, iq.IQ_MODE_UQ2])
def test_uq_bitpattern_sweep(k, mode):
    # a strided sweep over all 2^32 fp32 bit patterns (finite ones), plus near-ties
    bits = np.arange(0, 2 ** 32, 9973, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    x = x[np.isfinite(x)]
    d = 2.0 ** (1 - k)
    j = np.arange(-(2 ** min(k - 1, 12)), 2 ** min(k - 1, 12))
    t = ((j + 0.5) * d * (2 if mode == iq.IQ_MODE_UQ2 else 1)).astype(np.float32)
    x = np.concatenate([x, t, np.nextafter(t, np.float32(1e30)), np.nextafter(t, np.float32(-1e30))])
    out = torch.empty(x.size, dtype=torch.int32, device=DEV)
    s = dscal()
    iq.iq_quantize(dev(x), k, mode, out, s)
    want = O.uq(x, k) if mode == iq.IQ_MODE_UQ else O.uq2(x, k)
    assert np.array_equal(host(out), want)
    assert host(s)[0] == 2.0 ** ((1 if mode == iq.IQ_MODE_UQ else 2) - k)


@pytest.mark.parametrize("k,dtype", [(8, torch.int8), (16, torch.int16)])
def test_sq_float(k, dtype):
    g = S.rng(1)
    x = np.concatenate([S.float_uniform(g, 100003, -3, 3), np.float32([3.5, -0.0])])
    out = torch.empty(x.size, dtype=dtype, device=DEV)
    s = dscal()
    iq.iq_quantize(dev(x), k, iq.IQ_MODE_SQ, out, s)
    want, ws = O.sq_float(x, k)
    assert np.array_equal(host(out).astype(np.int32), want)
    assert host(s)[0] == ws


def test_sq_float_all_zero_and_empty():
    x = np.zeros(1000, np.float32)
    out = torch.empty(1000, dtype=torch.int8, device=DEV)
    s = dscal()
    iq.iq_quantize(dev(x), 8, iq.IQ_MODE_SQ, out, s)
    assert (host(out) == 0).all() and host(s)[0] == 2.0 ** -7
    e = torch.empty(0, dtype=torch.float32, device=DEV)
    iq.iq_quantize(e, 8, iq.IQ_MODE_SQ, torch.empty(0, dtype=torch.int8, device=DEV), s)
    assert host(s)[0] == 2.0 ** -7


def test_image_input():
    g = S.rng(2)
    img = S.images_u8(g, 2, 37, 41)
    codes = torch.empty((2, 37, 41, 4), dtype=torch.int8, device=DEV)
    s = dscal()
    iq.iq_quantize_image_u8(dev(img), False, 4, codes, s)
    want, ws = O.quantize_image_u8(img, 4)
    assert np.array_equal(host(codes), want) and host(s)[0] == ws
    # NCHW input gives the same codes
    codes2 = torch.empty_like(codes)
    iq.iq_quantize_image_u8(dev(np.ascontiguousarray(img.transpose(0, 3, 1, 2))), True, 4, codes2, s)
    assert np.array_equal(host(codes2), want)


@pytest.mark.parametrize("relu", [False, True])
def test_requantize_sq_int32(relu):
    g = S.rng(3)
    q = g.integers(-404644352, 404644353, size=77777).astype(np.int32)
    out = torch.empty(q.size, dtype=torch.int8, device=DEV)
    so = dscal()
    iq.iq_requantize(dev(q), dscal(2.0 ** -20), 8, iq.IQ_MODE_SQ_RELU if relu else iq.IQ_MODE_SQ,
                     out, so)
    want, ws = O.sq_int(q, 2.0 ** -20, 8, relu)
    assert np.array_equal(host(out).astype(np.int32), want)
    assert host(so)[0] == ws


@pytest.mark.parametrize("relu", [False, True])
@pytest.mark.parametrize("M", [128, 129, 255, 256 * 1000, 2 ** 30 + 3, 2 ** 31])
def test_requantize_sq_int32_vector_path(relu, M):
    # the 4-wide int32 -> int8 kernel (n % 4 == 0, aligned), across its 32-bit branch (M > 128)
    # and the 64-bit one (M <= 128): random values, both extremes, and exact half-step ties
    g = S.rng(M % 1000 + relu)
    vals = [-M, M - 1 if M == 2 ** 31 else M, 0, 1, -1]
    if M % 256 == 0:
        vals += [(2 * k + 1) * M // 256 - M for k in range(0, 256, 5)]
    q = np.concatenate([np.array(vals, np.int64),
                        g.integers(-M, min(M, 2 ** 31 - 1) + 1, size=4000)])
    q = q[: len(q) // 4 * 4].astype(np.int32)
    assert np.abs(q.astype(np.int64)).max() == M
    out = torch.empty(q.size, dtype=torch.int8, device=DEV)
    so = dscal()
    iq.iq_requantize(dev(q), dscal(2.0 ** -20), 8, iq.IQ_MODE_SQ_RELU if relu else iq.IQ_MODE_SQ,
                     out, so)
    want, ws = O.sq_int(q, 2.0 ** -20, 8, relu)
    assert np.array_equal(host(out).astype(np.int32), want)
    assert host(so)[0] == ws


@pytest.mark.parametrize("relu,M", [(True, 2 ** 31), (False, 1000), (False, 100), (True, 3 * 2 ** 20)])
def test_requantize_sq_int32_large(relu, M):
    # a tensor of 573 k elements (the grid-stride loops wrap several times): both extremes,
    # ties spread over the whole tensor, and every branch
    g = S.rng(M % 997 + 3 * relu)
    n = 5 * 16384 * 7 + 12
    q = g.integers(-M, min(M, 2 ** 31 - 1) + 1, size=n).astype(np.int64)
    q[g.integers(n, size=64)] = -M
    q[g.integers(n, size=1)] = M - 1 if M == 2 ** 31 else M
    if M % 256 == 0:
        ties = np.array([(2 * k + 1) * M // 256 - M for k in range(256)], np.int64)
        q[g.integers(n, size=ties.size)] = ties
    q = q.astype(np.int32)
    out = torch.empty(n, dtype=torch.int8, device=DEV)
    so = dscal()
    iq.iq_requantize(dev(q), dscal(2.0 ** -20), 8, iq.IQ_MODE_SQ_RELU if relu else iq.IQ_MODE_SQ,
                     out, so)
    want, ws = O.sq_int(q, 2.0 ** -20, 8, relu)
    assert np.array_equal(host(out).astype(np.int32), want)
    assert host(so)[0] == ws


@pytest.mark.parametrize("relu", [False, True])
@pytest.mark.parametrize("M", [2 ** 31, 2 ** 31 - 1, 2 ** 30 + 3, 3 * 2 ** 20 + 7, 1000])
def test_requantize_sq_int32_code_boundaries(relu, M):
    """Values one unit below, at and above every code boundary of SQ8 (the smallest u = v + M
    with floor(128 u / M + 1/2) >= k, for every k): the 4-wide kernel's fp32 evaluation cannot
    tell these apart at large M, so its exact fallback decides them."""
    ks = np.arange(1, 256, dtype=np.int64)
    u_k = ((2 * ks - 1) * M + 255) // 256          # ceil((2k - 1) M / 256)
    u = np.concatenate([u_k - 1, u_k, u_k + 1, [0, 2 * M]])
    u = np.clip(u, 0, 2 * M)
    v = u - M
    v = v[(v >= -(2 ** 31)) & (v <= 2 ** 31 - 1)]
    g = S.rng(M % 1009 + relu)
    v = np.concatenate([v, [-M if M <= 2 ** 31 else -(2 ** 31)]])
    v = v[g.permutation(v.size)]
    v = v[: v.size // 4 * 4].astype(np.int32)
    if np.abs(v.astype(np.int64)).max() != M:           # the tensor's maximum must be M
        v[0] = np.int32(-M if M <= 2 ** 31 else 0)
    out = torch.empty(v.size, dtype=torch.int8, device=DEV)
    so = dscal()
    iq.iq_requantize(dev(v), dscal(2.0 ** -20), 8, iq.IQ_MODE_SQ_RELU if relu else iq.IQ_MODE_SQ,
                     out, so)
    want, ws = O.sq_int(v, 2.0 ** -20, 8, relu)
    assert np.array_equal(host(out).astype(np.int32), want)
    assert host(so)[0] == ws


def test_rq_epoch_changes_only_the_draws():
    # the epoch is the fourth Philox counter word: 0 reproduces the oracle; another value gives
    # other draws of the same stochastic rounding (every code within one of the exact value)
    g = S.rng(91)
    q = g.integers(-(2 ** 40), 2 ** 40, size=50000).astype(np.int64)
    out = torch.empty(q.size, dtype=torch.int8, device=DEV)
    so = dscal()
    want, _ = O.rq_int(q, 1e-9, 8, 1, 77, 3, 5)
    try:
        iq.iq_requantize(dev(q), dscal(1e-9), 8, iq.IQ_MODE_RQ_GQ1, out, so, seed=77, layer=3,
                         step=5)
        assert np.array_equal(host(out).astype(np.int32), want)
        iq.iq_rq_epoch_set(7)
        iq.iq_requantize(dev(q), dscal(1e-9), 8, iq.IQ_MODE_RQ_GQ1, out, so, seed=77, layer=3,
                         step=5)
        got = host(out).astype(np.int32)
        assert np.abs(got - want).max() <= 1 and (got != want).mean() > 0.2
        iq.iq_rq_epoch_advance()
        iq.iq_requantize(dev(q), dscal(1e-9), 8, iq.IQ_MODE_RQ_GQ1, out, so, seed=77, layer=3,
                         step=5)
        got8 = host(out).astype(np.int32)
        assert np.abs(got8 - want).max() <= 1 and (got8 != got).mean() > 0.2
    finally:
        iq.iq_rq_epoch_set(0)
    iq.iq_requantize(dev(q), dscal(1e-9), 8, iq.IQ_MODE_RQ_GQ1, out, so, seed=77, layer=3, step=5)
    assert np.array_equal(host(out).astype(np.int32), want)


@pytest.mark.parametrize("mode,gq", [(iq.IQ_MODE_RQ_GQ1, 1), (iq.IQ_MODE_RQ_GQ2, 2)])
def test_requantize_rq_int64(mode, gq):
    g = S.rng(4)
    q = (g.standard_normal(50001) * 3e9).astype(np.int64)
    for step in (0, 7):
        out = torch.empty(q.size, dtype=torch.int8, device=DEV)
        so = dscal()
        iq.iq_requantize(dev(q), dscal(1.5e-9), 8, mode, out, so, seed=1234, layer=5, step=step,
                         tag=2)
        want, ws = O.rq_int(q, 1.5e-9, 8, gq, 1234, 5, step, 2)
        assert np.array_equal(host(out).astype(np.int32), want)
        assert host(so)[0] == ws


def test_weight_requant_and_update():
    g = S.rng(5)
    m = O.uq(S.he_weights(g, 100001, 576), 24)
    wq = torch.empty(m.size, dtype=torch.int8, device=DEV)
    md = dev(m)
    iq.iq_weight_requant(md, wq)
    assert np.array_equal(host(wq).astype(np.int32), O.requant_master(m))
    gc = S.int8_uniform(g, m.size)
    for s_g, e, x2 in ((2.0 ** -7, 10, False), (3.3e-5, 4, False), (1.7e-3, 6, True)):
        md = dev(m)
        iq.iq_update(md, wq, dev(gc), dscal(s_g), e, x2=x2)
        wm, wwq = O.update(m, gc.astype(np.int32), s_g, e, x2=x2)
        assert np.array_equal(host(md), wm)
        assert np.array_equal(host(wq).astype(np.int32), wwq)


def test_relu_bwd():
    g = S.rng(6)
    ea = S.int8_uniform(g, 100003)
    a = S.int8_uniform(g, 100003, -3, 127)
    e = torch.empty(ea.size, dtype=torch.int8, device=DEV)
    iq.iq_relu_bwd(dev(ea), dev(a), e)
    assert np.array_equal(host(e), O.relu_bwd(ea, a))


# ----------------------------------------------------------------- convolution

CONV_CASES = [
    # n, h, w, c, k, r, s, stride, pad, dil, groups
    (1, 32, 32, 64, 64, 3, 3, 1, 1, 1, 1),      # the single-layer workload
    (2, 13, 11, 16, 24, 3, 3, 1, 1, 1, 1),      # ragged M and N tiles
    (1, 17, 19, 32, 40, 3, 3, 2, 1, 1, 1),      # stride 2
    (2, 15, 15, 16, 16, 3, 3, 1, 4, 4, 1),      # atrous
    (1, 9, 9, 24, 12, 1, 1, 1, 0, 1, 1),        # 1x1
    (1, 10, 12, 12, 8, 3, 3, 1, 1, 1, 4),       # grouped, C/G = 3 (byte path)
    (2, 20, 20, 4, 16, 7, 7, 2, 3, 1, 1),       # stem-like, C padded to 4
    (1, 7, 7, 256, 32, 7, 7, 1, 3, 1, 1),       # fc6-like, CRS = 12544
    (1, 65, 3, 8, 8, 3, 3, 1, 12, 12, 1),       # ASPP-like rate beyond the map
]


def _conv_case(ci, seed):
    n, h, w, c, k, r, s, st, pd, dl, gr = CONV_CASES[ci]
    cv = O.Conv(n, h, w, c, k, r, s, st, pd, dl, gr)
    d = iq.conv_desc(n, h, w, c, k, r, s, st, pd, dl, gr)
    g = S.rng(seed)
    p, q = cv.pq
    x = S.int8_uniform(g, (n, h, w, c))
    wm = O.uq(S.he_weights(g, (k, r, s, c // gr), c // gr * r * s), 24)
    wq = O.requant_master(wm).astype(np.int8)
    e = S.int8_uniform(g, (n, p, q, k))
    return cv, d, x, wq, e


@pytest.mark.parametrize("ci", range(len(CONV_CASES)))
@pytest.mark.parametrize("relu", [True, False])
def test_conv_fwd_no_bn(ci, relu):
    cv, d, x, w, _ = _conv_case(ci, 10 + ci)
    p, q = cv.pq
    a = torch.empty((cv.n, p, q, cv.k), dtype=torch.int8, device=DEV)
    acc = torch.empty((cv.n, p, q, cv.k), dtype=torch.int32, device=DEV)
    s_a = dscal()
    s_x = 2.0 ** -7 * 0.37
    iq.iq_conv_fwd(d, dev(x), dscal(s_x), dev(w), a, s_a, relu=relu, acc_out=acc)
    want_acc = O.conv_fwd(cv, x, w)
    assert np.array_equal(host(acc), want_acc)
    want_a, want_s = O.sq_int(want_acc, s_x * 2.0 ** -7, 8, relu)
    assert np.array_equal(host(a).astype(np.int32), want_a)
    assert host(s_a)[0] == want_s


@pytest.mark.parametrize("ci", range(len(CONV_CASES)))
def test_conv_dgrad(ci):
    cv, d, x, w, e = _conv_case(ci, 30 + ci)
    dx = torch.empty((cv.n, cv.h, cv.w, cv.c), dtype=torch.int8, device=DEV)
    acc = torch.empty((cv.n, cv.h, cv.w, cv.c), dtype=torch.int32, device=DEV)
    s_dx = dscal()
    s_e = 3.1e-6
    iq.iq_conv_dgrad(d, dev(e), dscal(s_e), dev(w), dx, s_dx, acc_out=acc)
    want_acc = O.conv_dgrad(cv, e, w)
    assert np.array_equal(host(acc), want_acc)
    want, ws = O.sq_int(want_acc, s_e * 2.0 ** -7, 8)
    assert np.array_equal(host(dx).astype(np.int32), want)
    assert host(s_dx)[0] == ws


@pytest.mark.parametrize("ci", range(len(CONV_CASES)))
@pytest.mark.parametrize("gq", [1, 2])
def test_conv_wgrad(ci, gq):
    cv, d, x, w, e = _conv_case(ci, 50 + ci)
    gco = torch.empty(w.shape, dtype=torch.int8, device=DEV)
    gacc = torch.empty(w.shape, dtype=torch.int64, device=DEV)
    s_g = dscal()
    s_e, s_x = 3.1e-6, 0.02
    iq.iq_conv_wgrad(d, dev(e), dscal(s_e), dev(x), dscal(s_x), gco, s_g, gq_mode=gq, seed=99,
                     layer=ci, step=3, g_acc_out=gacc)
    want_acc = O.conv_wgrad(cv, e, x)
    assert np.array_equal(host(gacc), want_acc)
    want, ws = O.rq_int(want_acc, s_e * s_x, 8, gq, 99, ci, 3, 0)
    assert np.array_equal(host(gco).astype(np.int32), want)
    assert host(s_g)[0] == ws


# ----------------------------------------------------------------- L1BN

def _bn_ref(acc, s_acc, gam, bet, k_e2=16):
    return O.bn_fwd(acc, s_acc, gam, bet)


@pytest.mark.parametrize("m,C,spread,offset", [(1024, 64, 3000, 500), (777, 32, 20, 40000),
                                               (300, 1032, 1e6, 1e6), (64, 2048, 5e5, 0)])
def test_bn_int_fwd(m, C, spread, offset):
    g = S.rng(int(m + C))
    acc = (g.standard_normal((m, C)) * spread + g.integers(-offset, offset + 1, C)).astype(np.int32)
    gam, bet = S.bn_gamma_beta_codes(g, C)
    s_acc = 2.0 ** -14 * 1.7
    X = torch.empty((m, C), dtype=torch.int16, device=DEV)
    A = torch.empty((m, C), dtype=torch.int8, device=DEV)
    codes = torch.empty(2 * C, dtype=torch.int32, device=DEV)
    scal = torch.empty(iq.IQ_BN_SCALES, dtype=torch.float64, device=DEV)
    fixed = torch.empty(4 * C + 2, dtype=torch.int64, device=DEV)
    s_a = dscal()
    iq.iq_bn_int_fwd(dev(acc), dscal(s_acc), dev(gam), dev(bet), A, s_a, xhat=X, bn_codes=codes,
                     bn_scales=scal, bn_fixed=fixed)
    r = O.bn_fwd(acc, s_acc, gam, bet)
    fx = host(fixed)
    assert np.array_equal(host(codes), np.concatenate([r.c_mu, r.c_sigma]))
    assert np.array_equal(fx[:C], r.F) and np.array_equal(fx[C:2 * C], r.B)
    assert np.array_equal(fx[2 * C:3 * C], r.G) and np.array_equal(fx[3 * C:4 * C], r.H)
    assert fx[4 * C] == r.p_x and fx[4 * C + 1] == r.p_a
    sc = host(scal)
    assert sc[iq.IQ_BN_S_XHAT] == r.s_xhat and sc[iq.IQ_BN_M_XHAT] == r.m_xhat
    assert sc[iq.IQ_BN_M_Y] == r.m_y and sc[iq.IQ_BN_S_A] == r.s_a and host(s_a)[0] == r.s_a
    assert np.array_equal(host(X), r.X)
    assert np.array_equal(host(A), r.A)


def test_conv_fwd_bn_single_layer_workload():
    # N=1, C=K=64, 32x32, 3x3 s1 p1, L1BN + ReLU + Q_A (the single-layer case)
    cv, d, x, w, _ = _conv_case(0, 70)
    g = S.rng(71)
    gam, bet = S.bn_gamma_beta_codes(g, 64)
    s_x = 2.0 ** -7
    A = torch.empty((1, 32, 32, 64), dtype=torch.int8, device=DEV)
    X = torch.empty((1, 32, 32, 64), dtype=torch.int16, device=DEV)
    codes = torch.empty(128, dtype=torch.int32, device=DEV)
    scal = torch.empty(iq.IQ_BN_SCALES, dtype=torch.float64, device=DEV)
    s_a = dscal()
    iq.iq_conv_fwd(d, dev(x), dscal(s_x), dev(w), A, s_a, gamma=dev(gam), beta=dev(bet),
                   bits=iq.bn_bits(), use_bn=True, xhat=X, bn_codes=codes, bn_scales=scal)
    acc = O.conv_fwd(cv, x, w)
    r = O.bn_fwd(acc.reshape(-1, 64), s_x * 2.0 ** -7, gam, bet)
    assert np.array_equal(host(X).reshape(-1, 64), r.X)
    assert np.array_equal(host(A).reshape(-1, 64), r.A)
    assert host(s_a)[0] == r.s_a


@pytest.mark.parametrize("k_e2", [16, 8])
@pytest.mark.parametrize("m,C", [(1024, 64), (333, 1028), (200, 2048)])
def test_bn_int_bwd(m, C, k_e2):
    g = S.rng(m * 7 + C + k_e2)
    acc = (g.standard_normal((m, C)) * 4000 + g.integers(-300, 301, C)).astype(np.int32)
    gam, bet = S.bn_gamma_beta_codes(g, C)
    s_acc = 2.0 ** -14
    r = O.bn_fwd(acc, s_acc, gam, bet)
    ea = S.int8_uniform(g, (m, C))
    s_e = 2.0 ** -21 * 1.3
    E, s_E, dg, db = O.bn_bwd(ea, s_e, r.A, r.X, r.s_xhat, gam, r.c_sigma, k_e2=k_e2)
    codes = dev(np.concatenate([r.c_mu, r.c_sigma]))
    scal = np.zeros(iq.IQ_BN_SCALES)
    scal[iq.IQ_BN_S_XHAT] = r.s_xhat
    e_out = torch.empty((m, C), dtype=torch.int8, device=DEV)
    s_out = dscal()
    dgam = torch.empty(C, dtype=torch.int64, device=DEV)
    dbet = torch.empty(C, dtype=torch.int64, device=DEV)
    iq.iq_bn_int_bwd(dev(ea), dscal(s_e), dev(r.A), dev(r.X), dev(gam), codes, dev(scal), e_out,
                     s_out, dgamma=dgam, dbeta=dbet, k_e2=k_e2)
    assert np.array_equal(host(dgam), dg) and np.array_equal(host(dbet), db)
    assert np.array_equal(host(e_out), E)
    assert host(s_out)[0] == s_E


# ----------------------------------------------------------------- tensor-core path specifics

TC_CASES = [
    # n, h, w, c, k, r, s, stride, pad, dil: shapes the tcgen05 kernel takes
    (2, 16, 16, 512, 256, 3, 3, 1, 1, 1),   # 5 fp32 chunks, 2 N tiles, 4 M tiles
    (1, 29, 31, 128, 144, 3, 3, 1, 2, 2),   # ragged M and N, dilation 2
    (3, 9, 10, 64, 80, 1, 1, 1, 0, 1),      # 1x1, ragged
    (1, 33, 33, 256, 64, 3, 3, 2, 1, 1),    # stride 2 (data gradient on CUDA cores)
    (4, 40, 40, 64, 64, 3, 3, 1, 1, 1),     # weight gradient split over 100 k-blocks
    (2, 24, 20, 64, 150, 1, 1, 1, 0, 1),    # 150 output channels (padded error rows)
    (2, 31, 29, 4, 64, 3, 3, 1, 1, 1),      # 4 input channels (fp16 im2col forward)
    (1, 35, 35, 4, 64, 7, 7, 2, 3, 1),      # stem: 7x7 stride 2 over 4 channels
    (2, 17, 15, 128, 96, 3, 3, 1, 2, 2),    # dilation 2, rectangle tiles with waste
    # channel-major kernel (at most 128 output channels, 256-pixel rectangles)
    (1, 64, 64, 64, 64, 3, 3, 1, 1, 1),     # conv1_2 shape: forward and data gradient
    (2, 50, 48, 64, 72, 3, 3, 1, 1, 1),     # ragged channels (72) and 16 x 16 rectangles
    (1, 64, 64, 128, 128, 3, 3, 2, 1, 1),   # stride 2, 128 output channels
    (1, 32, 40, 64, 128, 3, 3, 1, 1, 1),    # 128 output channels, data gradient to 64
    (2, 128, 160, 64, 64, 3, 3, 1, 1, 1),   # 160 tiles: persistent CTAs run two tiles
]


@pytest.mark.parametrize("ci", range(len(TC_CASES)))
def test_conv_fwd_tc_shapes(ci):
    n, h, w, c, k, r, s, st, pd, dl = TC_CASES[ci]
    cv = O.Conv(n, h, w, c, k, r, s, st, pd, dl)
    d = iq.conv_desc(n, h, w, c, k, r, s, st, pd, dl)
    g = S.rng(90 + ci)
    x = S.int8_uniform(g, (n, h, w, c))
    wq = O.requant_master(O.uq(S.he_weights(g, (k, r, s, c), c * r * s), 24)).astype(np.int8)
    p, q = cv.pq
    a = torch.empty((n, p, q, k), dtype=torch.int8, device=DEV)
    acc = torch.empty((n, p, q, k), dtype=torch.int32, device=DEV)
    s_a = dscal()
    iq.iq_conv_fwd(d, dev(x), dscal(0.01), dev(wq), a, s_a, relu=True, acc_out=acc)
    want = O.conv_fwd(cv, x, wq)
    assert np.array_equal(host(acc), want)
    wa, ws_ = O.sq_int(want, 0.01 * 2.0 ** -7, 8, True)
    assert np.array_equal(host(a).astype(np.int32), wa) and host(s_a)[0] == ws_
    # data and weight gradients of the same shape
    e = S.int8_uniform(g, (n, p, q, k))
    dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    dacc = torch.empty((n, h, w, c), dtype=torch.int32, device=DEV)
    s_dx = dscal()
    iq.iq_conv_dgrad(d, dev(e), dscal(2e-5), dev(wq), dx, s_dx, acc_out=dacc)
    want_d = O.conv_dgrad(cv, e, wq)
    assert np.array_equal(host(dacc), want_d)
    wd, wds = O.sq_int(want_d, 2e-5 * 2.0 ** -7, 8)
    assert np.array_equal(host(dx).astype(np.int32), wd) and host(s_dx)[0] == wds
    gq = torch.empty(wq.shape, dtype=torch.int8, device=DEV)
    gacc = torch.empty(wq.shape, dtype=torch.int64, device=DEV)
    s_g = dscal()
    iq.iq_conv_wgrad(d, dev(e), dscal(2e-5), dev(x), dscal(0.01), gq, s_g, gq_mode=1, seed=4,
                     layer=ci, step=1, g_acc_out=gacc)
    want_g = O.conv_wgrad(cv, e, x)
    assert np.array_equal(host(gacc), want_g)
    wg, wgs = O.rq_int(want_g, 2e-5 * 0.01, 8, 1, 4, ci, 1, 0)
    assert np.array_equal(host(gq).astype(np.int32), wg) and host(s_g)[0] == wgs


def test_conv_dgrad_int64_slices_one_launch():
    # an fc6-like data gradient, (k/groups) r s 127^2 >= 2^31: two reduction slices of 2048
    # channels run as tiles of one all-TMA launch, int64 sums
    n, h, w, c, k = 1, 16, 16, 64, 4096
    cv = O.Conv(n, h, w, c, k, 7, 7, 1, 3)
    d = iq.conv_desc(n, h, w, c, k, 7, 7, 1, 3)
    g = S.rng(501)
    e = np.full((n, h, w, k), 127, np.int8)
    e[0, :, :, g.integers(0, k, 300)] = -127
    wq = np.full((k, 7, 7, c), 127, np.int8)
    wq[:, :, :, 5] = -127
    dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    s_dx = dscal()
    iq.iq_conv_dgrad(d, dev(e), dscal(1e-4), dev(wq), dx, s_dx)
    want_acc = O.conv_dgrad(cv, e, wq)
    assert np.abs(want_acc).max() > 2 ** 31
    want, ws_ = O.sq_int(want_acc, 1e-4 * 2.0 ** -7, 8)
    assert np.array_equal(host(dx).astype(np.int32), want) and host(s_dx)[0] == ws_


@pytest.mark.parametrize("ci", [0, 4, 9, 11])
def test_conv_fp16_carriers_reused(ci):
    # the forward writes the fp16 copy of x, the data gradient that of e, and the weight
    # gradient reads both instead of converting: every output still equals the oracle's
    n, h, w, c, k, r, s, st, pd, dl = TC_CASES[ci]
    cv = O.Conv(n, h, w, c, k, r, s, st, pd, dl)
    d = iq.conv_desc(n, h, w, c, k, r, s, st, pd, dl)
    g = S.rng(400 + ci)
    x = S.int8_uniform(g, (n, h, w, c))
    wq = O.requant_master(O.uq(S.he_weights(g, (k, r, s, c), c * r * s), 24)).astype(np.int8)
    p, q = cv.pq
    x16 = torch.full((n * h * w * c,), float("nan"), dtype=torch.float16, device=DEV)
    e16 = torch.full((n * p * q * k,), float("nan"), dtype=torch.float16, device=DEV)
    acc = torch.empty((n, p, q, k), dtype=torch.int32, device=DEV)
    iq.iq_conv_fwd(d, dev(x), dscal(0.01), dev(wq), torch.empty((n, p, q, k), dtype=torch.int8,
                   device=DEV), dscal(), relu=True, acc_out=acc, x_f16=x16)
    assert np.array_equal(host(acc), O.conv_fwd(cv, x, wq))
    assert np.array_equal(host(x16).astype(np.int64), x.reshape(-1).astype(np.int64))
    e = S.int8_uniform(g, (n, p, q, k))
    if st == 1:
        dacc = torch.empty((n, h, w, c), dtype=torch.int32, device=DEV)
        iq.iq_conv_dgrad(d, dev(e), dscal(1e-3), dev(wq), torch.empty((n, h, w, c),
                         dtype=torch.int8, device=DEV), dscal(), acc_out=dacc, e_f16=e16)
        assert np.array_equal(host(dacc), O.conv_dgrad(cv, e, wq))
    else:
        e16.copy_(dev(e).view(-1).to(torch.float16))
    assert np.array_equal(host(e16).astype(np.int64), e.reshape(-1).astype(np.int64))
    gacc = torch.empty(wq.shape, dtype=torch.int64, device=DEV)
    iq.iq_conv_wgrad(d, dev(e), dscal(1e-3), dev(x), dscal(0.01), torch.empty(wq.shape,
                     dtype=torch.int8, device=DEV), dscal(), gq_mode=1, seed=1, layer=ci, step=0,
                     g_acc_out=gacc, e_f16=e16, x_f16=x16)
    want_g = O.conv_wgrad(cv, e, x)
    assert np.array_equal(host(gacc), want_g)
    # without the int64 copy (a single split requantizes its int32 sums directly)
    gq = torch.empty(wq.shape, dtype=torch.int8, device=DEV)
    s_g = dscal()
    iq.iq_conv_wgrad(d, dev(e), dscal(1e-3), dev(x), dscal(0.01), gq, s_g, gq_mode=1, seed=1,
                     layer=ci, step=0, e_f16=e16, x_f16=x16)
    wg, wgs = O.rq_int(want_g, 1e-3 * 0.01, 8, 1, 1, ci, 0, 0)
    assert np.array_equal(host(gq).astype(np.int32), wg) and host(s_g)[0] == wgs


@pytest.mark.parametrize("sign,h,k", [(1, 6, 128), (-1, 6, 128), (1, 16, 64), (-1, 16, 64)])
def test_conv_fwd_adversarial_full_scale(sign, h, k):
    # all codes at +-127: every fp32 chunk holds 1024 * 127^2 = 16,516,096 < 2^24 and
    # the int32 total is 4608 * 127^2 for interior pixels (16 x 16 x 64: channel-major kernel)
    n, w, c = 1, h, 512
    cv = O.Conv(n, h, w, c, k, 3, 3, 1, 1)
    d = iq.conv_desc(n, h, w, c, k, 3, 3, 1, 1)
    x = np.full((n, h, w, c), 127, np.int8)
    wq = np.full((k, 3, 3, c), 127 * sign, np.int8)
    a = torch.empty((n, h, w, k), dtype=torch.int8, device=DEV)
    acc = torch.empty((n, h, w, k), dtype=torch.int32, device=DEV)
    iq.iq_conv_fwd(d, dev(x), dscal(1.0), dev(wq), a, dscal(), relu=False, acc_out=acc)
    got = host(acc)
    assert np.array_equal(got, O.conv_fwd(cv, x, wq))
    assert got[0, 2, 2, 0] == sign * 4608 * 16129


# ----------------------------------------------------------------- network glue

@pytest.mark.parametrize("k,s,p,c", [(2, 2, 0, 24), (3, 2, 1, 24), (3, 2, 1, 6), (2, 2, 0, 64),
                                     (3, 2, 1, 64), (3, 1, 1, 8), (2, 3, 0, 8), (3, 3, 1, 16),
                                     (2, 2, 0, 6)])
def test_maxpool(k, s, p, c):
    g = S.rng(k * 10 + s)
    x = S.int8_uniform(g, (2, 37, 30, c), -9, 9)
    y_o, a_o = O.maxpool_fwd(x, k, s, p)
    y = torch.empty(y_o.shape, dtype=torch.int8, device=DEV)
    a = torch.empty(y_o.shape, dtype=torch.uint8, device=DEV)
    iq.iq_maxpool_fwd(dev(x), k, s, p, y, a)
    assert np.array_equal(host(y), y_o) and np.array_equal(host(a), a_o)
    e = S.int8_uniform(g, y_o.shape)
    ex = torch.empty(x.shape, dtype=torch.int8, device=DEV)
    s_ex = dscal()
    iq.iq_maxpool_bwd(dev(e), dscal(0.5), a, x.shape, k, s, p, ex, s_ex)
    sums = O.maxpool_bwd(e, a_o, x.shape, k, s, p)
    if k <= s:
        assert np.array_equal(host(ex).astype(np.int32), sums) and host(s_ex)[0] == 0.5
    else:
        want, ws_ = O.sq_int(sums, 0.5, 8)
        assert np.array_equal(host(ex).astype(np.int32), want) and host(s_ex)[0] == ws_


@pytest.mark.parametrize("n,h,c,R,st,pd", [(1, 2, 150, 64, 32, 16), (2, 3, 21, 16, 8, 4),
                                           (2, 5, 150, 64, 32, 16), (1, 3, 40, 64, 32, 16),
                                           (2, 4, 150, 64, 32, 16), (1, 8, 21, 64, 32, 16)])
def test_upsample_fwd_bwd_wgrad(n, h, c, R, st, pd):
    g = S.rng(c + R)
    H = (h - 1) * st - 2 * pd + R
    cv = O.Conv(n, H, H, c, c, R, R, st, pd, 1, c)      # the strided conv it is the adjoint of
    assert cv.pq == (h, h)
    x = S.int8_uniform(g, (n, h, h, c))
    w = S.int8_uniform(g, (c, R, R, 1))
    out = torch.empty((n, H, H, c), dtype=torch.int8, device=DEV)
    acc = torch.empty((n, H, H, c), dtype=torch.int32, device=DEV)
    s_out = dscal()
    iq.iq_upsample_fwd(dev(x), dscal(0.03), dev(w), R, st, pd, out, s_out, acc_out=acc)
    want_acc = O.conv_dgrad(cv, x, w)
    assert np.array_equal(host(acc), want_acc)
    want, ws_ = O.sq_int(want_acc, 0.03 * 2.0 ** -7, 8)
    assert np.array_equal(host(out).astype(np.int32), want) and host(s_out)[0] == ws_
    E = S.int8_uniform(g, (n, H, H, c))
    ex = torch.empty((n, h, h, c), dtype=torch.int8, device=DEV)
    eacc = torch.empty((n, h, h, c), dtype=torch.int32, device=DEV)
    s_ex = dscal()
    iq.iq_upsample_bwd(dev(E), dscal(1e-3), dev(w), (n, h, h, c), R, st, pd, ex, s_ex, acc_out=eacc)
    want_e = O.conv_fwd(cv, E, w)
    assert np.array_equal(host(eacc), want_e)
    want, ws_ = O.sq_int(want_e, 1e-3 * 2.0 ** -7, 8)
    assert np.array_equal(host(ex).astype(np.int32), want) and host(s_ex)[0] == ws_
    gq = torch.empty((c, R, R), dtype=torch.int8, device=DEV)
    gacc = torch.empty((c, R, R), dtype=torch.int64, device=DEV)
    s_g = dscal()
    iq.iq_upsample_wgrad(dev(x), dscal(0.03), dev(E), dscal(1e-3), R, st, pd, gq, s_g, gq_mode=2,
                         seed=5, layer=19, step=2, g_acc_out=gacc)
    want_g = O.conv_wgrad(cv, x, E).reshape(c, R, R)
    assert np.array_equal(host(gacc), want_g)
    want, ws_ = O.rq_int(want_g, 0.03 * 1e-3, 8, 2, 5, 19, 2, 0)
    assert np.array_equal(host(gq).astype(np.int32), want) and host(s_g)[0] == ws_


def test_upsample_fcn_shape_extremes():
    """Every sum at +-4 * 127^2: the largest SQ numerator of the decoder's 32-bit path."""
    n, h, c = 2, 3, 150
    H = 32 * h
    cv = O.Conv(n, H, H, c, c, 64, 64, 32, 16, 1, c)
    x = np.full((n, h, h, c), 127, np.int8)
    x[1] = -127
    w = np.full((c, 64, 64, 1), -127, np.int8)
    out = torch.empty((n, H, H, c), dtype=torch.int8, device=DEV)
    s_out = dscal()
    iq.iq_upsample_fwd(dev(x), dscal(0.5), dev(w), 64, 32, 16, out, s_out)
    want, ws_ = O.sq_int(O.conv_dgrad(cv, x, w), 0.5 * 2.0 ** -7, 8)
    assert np.array_equal(host(out).astype(np.int32), want) and host(s_out)[0] == ws_


@pytest.mark.parametrize("offset", [0, 1])
def test_mse_grad_alignment(offset):
    g = S.rng(78)
    z = S.int8_uniform(g, (1, 16, 8, 150))
    lab = S.labels_voronoi(g, 1, 16, 8, 150, sites=5)
    zbuf = torch.empty(z.size + 16, dtype=torch.int8, device=DEV)
    zbuf[offset:offset + z.size].copy_(dev(z).view(-1))
    ebuf = torch.empty(z.size + 16, dtype=torch.int8, device=DEV)
    s_e = dscal()
    zt = zbuf[offset:offset + z.size].view(z.shape)
    et = ebuf[offset:offset + z.size].view(z.shape)
    iq.iq_mse_grad(zt, dscal(0.05), dev(lab), et, s_e)
    want, ws_ = O.mse_grad(z, 0.05, lab)
    assert np.array_equal(host(et), want) and host(s_e)[0] == ws_


@pytest.mark.parametrize("c", [150, 21, 16, 5])
def test_mse_grad(c):
    g = S.rng(77 + c)
    z = S.int8_uniform(g, (2, 33, 17, c))
    lab = S.labels_voronoi(g, 2, 33, 17, c, sites=8)
    E = torch.empty(z.shape, dtype=torch.int8, device=DEV)
    s_e = dscal()
    iq.iq_mse_grad(dev(z), dscal(0.0123), dev(lab), E, s_e)
    want, ws_ = O.mse_grad(z, 0.0123, lab)
    assert np.array_equal(host(E), want) and host(s_e)[0] == ws_


def test_conv_dgrad_int64_reduction():
    # (k/groups) r s = 20000 * 49 products: sums beyond int32 range, accumulated in int64
    n, h, w, c, k = 1, 3, 3, 8, 20000
    cv = O.Conv(n, h, w, c, k, 7, 7, 1, 3)
    d = iq.conv_desc(n, h, w, c, k, 7, 7, 1, 3)
    e = np.full((n, h, w, k), 127, np.int8)
    wq = np.full((k, 7, 7, c), 127, np.int8)
    wq[:, :, :, 1] = -127
    dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    s_dx = dscal()
    iq.iq_conv_dgrad(d, dev(e), dscal(1e-4), dev(wq), dx, s_dx)
    want_acc = O.conv_dgrad(cv, e, wq)
    assert np.abs(want_acc).max() > 2 ** 31
    want, ws_ = O.sq_int(want_acc, 1e-4 * 2.0 ** -7, 8)
    assert np.array_equal(host(dx).astype(np.int32), want) and host(s_dx)[0] == ws_
    with pytest.raises(iq.IqError):
        iq.iq_conv_dgrad(d, dev(e), dscal(1e-4), dev(wq), dx, s_dx,
                         acc_out=torch.empty((n, h, w, c), dtype=torch.int32, device=DEV))


def test_kernel_timing_brackets_the_conv_kernels():
    # one forward, data-gradient and weight-gradient call of a 3x3 layer: each operation's
    # main kernel bracketed once, with the layer's algorithmic MACs
    n, h, c, k = 2, 32, 64, 128
    d = iq.conv_desc(n, h, h, c, k, 3, 3, 1, 1)
    g = S.rng(77)
    x = dev(S.int8_uniform(g, (n, h, h, c)))
    wq = dev(S.int8_uniform(g, (k, 3, 3, c)))
    e = dev(S.int8_uniform(g, (n, h, h, k)))
    a = torch.empty((n, h, h, k), dtype=torch.int8, device=DEV)
    dx = torch.empty((n, h, h, c), dtype=torch.int8, device=DEV)
    gw = torch.empty((k, 3, 3, c), dtype=torch.int8, device=DEV)
    iq.iq_kernel_timing_begin()
    iq.iq_conv_fwd(d, x, dscal(0.01), wq, a, dscal(0.0), relu=True)
    iq.iq_conv_dgrad(d, e, dscal(0.01), wq, dx, dscal(0.0))
    iq.iq_conv_wgrad(d, e, dscal(0.01), x, dscal(0.01), gw, dscal(0.0), gq_mode=2)
    rows = iq.iq_kernel_timing_end()
    dense = float(n * h * h * k * 9 * c)
    inb = float(n * k * c * (3 * h - 2) ** 2)      # taps that read inside the 32 x 32 input
    conv = [r for r in rows if r["op"] != 0]
    ops = {r["op"]: r for r in conv}
    assert sorted(ops) == [1, 2, 3] and len(conv) == 3
    for r in conv:
        assert r["launches"] == 1 and r["macs"] == inb and r["dense_macs"] == dense
        assert r["ms"] > 0 and r["bytes"] == 0
    assert ops[1]["kernel"] in (iq.IQ_KERNEL_CONV_PIXEL_MAJOR, iq.IQ_KERNEL_CONV_CHANNEL_MAJOR)
    assert ops[2]["kernel"] in (iq.IQ_KERNEL_CONV_PIXEL_MAJOR, iq.IQ_KERNEL_CONV_CHANNEL_MAJOR)
    assert ops[3]["kernel"] == iq.IQ_KERNEL_CONV_WGRAD
    # the bandwidth passes around them: the SQ codes of the forward and data-gradient sums,
    # each tagged with its int32 read and int8 write
    bw = {r["kernel"]: r for r in rows if r["op"] == 0}
    sq = bw[iq.IQ_KERNEL_SQ_CODES]
    assert sq["launches"] == 2 and sq["bytes"] == 5.0 * n * h * h * (k + c)
    assert iq.iq_kernel_timing_end() == []      # stopped: nothing recorded since


# ----------------------------------------------------------------- routing of the conv kernels

ROUTES = [
    # (n, h, w, c, k, r, stride, pad, dil), operation, kernels its call launches
    ((1, 7, 7, 256, 32, 7, 1, 3, 1), "fwd", {iq.IQ_KERNEL_CONV_CPASYNC}),
    ((16, 1, 1, 2048, 256, 1, 1, 0, 1), "dgrad", {iq.IQ_KERNEL_CONV_CPASYNC}),
    ((1, 13, 11, 16, 24, 3, 1, 1, 1), "fwd", {iq.IQ_KERNEL_CONV_GATHER}),
    ((3, 9, 10, 64, 80, 1, 1, 0, 1), "dgrad", {iq.IQ_KERNEL_CONV_GATHER}),
    ((1, 32, 40, 64, 128, 3, 1, 1, 1), "fwd", {iq.IQ_KERNEL_CONV_CHANNEL_MAJOR}),
    ((2, 16, 16, 512, 256, 3, 1, 1, 1), "dgrad", {iq.IQ_KERNEL_CONV_PIXEL_MAJOR}),
    ((2, 16, 16, 512, 256, 3, 1, 1, 1), "wgrad", {iq.IQ_KERNEL_CONV_WGRAD}),
    ((2, 31, 29, 4, 64, 3, 1, 1, 1), "dgrad", {iq.IQ_KERNEL_CONV_SIMT}),
]


@pytest.mark.parametrize("ri", range(len(ROUTES)))
def test_conv_kernel_routing(ri):
    """Which kernel a call runs on, read from the library's kernel timing, and its result
    against the oracle: every fallback of the tensor-core path (the cp.async-fed and the
    register-gather kernels, the channel-major kernel) and the CUDA-core kernel is reached by
    a shape of its own, so each one's parity is shown rather than assumed."""
    (n, h, w, c, k, r, st, pd, dl), op, want = ROUTES[ri]
    cv = O.Conv(n, h, w, c, k, r, r, st, pd, dl)
    d = iq.conv_desc(n, h, w, c, k, r, r, st, pd, dl)
    p, q = cv.pq
    g = S.rng(1200 + ri)
    x = S.int8_uniform(g, (n, h, w, c))
    wq = O.requant_master(O.uq(S.he_weights(g, (k, r, r, c), c * r * r), 24)).astype(np.int8)
    e = S.int8_uniform(g, (n, p, q, k))
    iq.iq_kernel_timing_begin()
    if op == "fwd":
        acc = torch.empty((n, p, q, k), dtype=torch.int32, device=DEV)
        a = torch.empty((n, p, q, k), dtype=torch.int8, device=DEV)
        iq.iq_conv_fwd(d, dev(x), dscal(0.02), dev(wq), a, dscal(), relu=True, acc_out=acc)
        got, ref = acc, O.conv_fwd(cv, x, wq)
    elif op == "dgrad":
        acc = torch.empty((n, h, w, c), dtype=torch.int32, device=DEV)
        dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
        iq.iq_conv_dgrad(d, dev(e), dscal(1e-5), dev(wq), dx, dscal(), acc_out=acc)
        got, ref = acc, O.conv_dgrad(cv, e, wq)
    else:
        gacc = torch.empty(wq.shape, dtype=torch.int64, device=DEV)
        gq = torch.empty(wq.shape, dtype=torch.int8, device=DEV)
        iq.iq_conv_wgrad(d, dev(e), dscal(1e-5), dev(x), dscal(0.02), gq, dscal(), gq_mode=1,
                         g_acc_out=gacc)
        got, ref = gacc, O.conv_wgrad(cv, e, x)
    torch.cuda.synchronize()
    ran = {t["kernel"] for t in iq.iq_kernel_timing_end() if t["kernel"] in iq.CONV_KERNELS}
    assert ran == want, (ROUTES[ri], ran)
    assert np.array_equal(host(got), ref)


def test_bounded_wait_gives_up_and_reports():
    """The bounded mbarrier wait of the tensor-core kernels, on a barrier nothing arrives on
    (iq_wait_selftest): it gives up after its limit, the sticky status reports code 5 once
    (IQ_ERR_TIMEOUT) and is cleared, and the context stays usable: a tensor-core convolution
    afterwards is exact."""
    import ctypes as C
    iq.iq_wait_selftest(1 << 20)
    code = C.c_int32(0)
    rc = iq.load().iq_device_status(C.byref(code), None)
    assert rc == iq.IQ_ERR_TIMEOUT and code.value == 5
    assert iq.iq_device_status() == 0
    cv, d, x, w, _ = _conv_case(0, 77)
    p, q = cv.pq
    acc = torch.empty((cv.n, p, q, cv.k), dtype=torch.int32, device=DEV)
    a = torch.empty((cv.n, p, q, cv.k), dtype=torch.int8, device=DEV)
    iq.iq_conv_fwd(d, dev(x), dscal(0.01), dev(w), a, dscal(), relu=True, acc_out=acc)
    assert np.array_equal(host(acc), O.conv_fwd(cv, x, w))
    with pytest.raises(iq.IqError):
        iq.iq_wait_selftest(-1)
