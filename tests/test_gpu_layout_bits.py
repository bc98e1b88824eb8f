"""GPU parity of the convolution entry points beyond the paper's default setting, through the
C ABI, bit-exact against the oracle:

  * NCHW activations / errors with KCRS filters (the layout flag of iq_conv_desc): forward
    with and without integer L1BN, data gradient and weight gradient, compared with the
    oracle's NHWC results transposed;
  * 4-bit weights and activations, the k_W = k_A = 4 rows of the paper's Table 1: W_q =
    UQ(W_m, 4) (Eq. (WQ1)), accumulator scale s_x 2^-3, Q_A = SQ(., 4) (Eq. (AQ1)) without
    and with L1BN, the data gradient's 8-bit Q_E on the 2^-3 weight step, and the update
    regenerating 4-bit weight codes from the 24-bit masters (Eq. (UQ2)).
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import iq
from paper_2011_14504_gb300 import synthetic as S

pytestmark = pytest.mark.gpu

DEV = "cuda"


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def sc(v=0.0):
    return torch.tensor([v], dtype=torch.float64, device=DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def nchw(a):
    return np.ascontiguousarray(np.moveaxis(a, -1, 1))


def kcrs(w):
    return np.ascontiguousarray(np.moveaxis(w, -1, 1))


LAYOUT_CASES = [
    # n, h, w, c, k, r, stride, pad, dil, bn
    (2, 13, 11, 64, 64, 3, 1, 1, 1, True),      # tensor-core shapes
    (1, 17, 19, 32, 40, 3, 2, 1, 1, False),     # stride 2, ragged
    (2, 9, 9, 24, 12, 1, 1, 0, 1, False),       # 1x1, output channels padded to 16
    (1, 15, 15, 16, 128, 3, 1, 4, 4, True),     # atrous
]


@pytest.mark.parametrize("ci", range(len(LAYOUT_CASES)))
def test_nchw_layer_matches_nhwc_oracle(ci):
    n, h, w, c, k, r, st, pd, dl, bn = LAYOUT_CASES[ci]
    cv = O.Conv(n, h, w, c, k, r, r, st, pd, dl)
    d = iq.conv_desc(n, h, w, c, k, r, r, st, pd, dl, layout=iq.IQ_LAYOUT_NCHW)
    p, q = cv.pq
    g = S.rng(700 + ci)
    x = S.int8_uniform(g, (n, h, w, c))
    wq = O.requant_master(O.uq(S.he_weights(g, (k, r, r, c), c * r * r), 24)).astype(np.int8)
    e = S.int8_uniform(g, (n, p, q, k))
    s_x, s_e = 0.0123, 4.1e-6
    acc = O.conv_fwd(cv, x, wq)
    # forward
    a = torch.empty((n, k, p, q), dtype=torch.int8, device=DEV)
    accd = torch.empty((n, k, p, q), dtype=torch.int32, device=DEV)
    s_a = sc()
    if bn:
        gam, bet = S.bn_gamma_beta_codes(g, k)
        X = torch.empty((n, k, p, q), dtype=torch.int16, device=DEV)
        iq.iq_conv_fwd(d, dev(nchw(x)), sc(s_x), dev(kcrs(wq)), a, s_a, dev(gam), dev(bet),
                       use_bn=True, relu=True, xhat=X, acc_out=accd)
        r_ = O.bn_fwd(acc.reshape(-1, k), s_x * 2.0 ** -7, gam, bet)
        assert np.array_equal(host(a), nchw(r_.A.reshape(n, p, q, k)))
        assert np.array_equal(host(X), nchw(r_.X.reshape(n, p, q, k)))
        assert s_a.item() == r_.s_a
    else:
        iq.iq_conv_fwd(d, dev(nchw(x)), sc(s_x), dev(kcrs(wq)), a, s_a, relu=True, acc_out=accd)
        want, s_want = O.sq_int(acc, s_x * 2.0 ** -7, 8, True)
        assert np.array_equal(host(a).astype(np.int32), nchw(want))
        assert s_a.item() == s_want
    assert np.array_equal(host(accd), nchw(acc))
    # data gradient
    dx = torch.empty((n, c, h, w), dtype=torch.int8, device=DEV)
    dacc = torch.empty((n, c, h, w), dtype=torch.int32, device=DEV)
    s_dx = sc()
    iq.iq_conv_dgrad(d, dev(nchw(e)), sc(s_e), dev(kcrs(wq)), dx, s_dx, acc_out=dacc)
    dwant = O.conv_dgrad(cv, e, wq)
    assert np.array_equal(host(dacc), nchw(dwant))
    cw, sw = O.sq_int(dwant, s_e * 2.0 ** -7, 8)
    assert np.array_equal(host(dx).astype(np.int32), nchw(cw)) and s_dx.item() == sw
    # weight gradient (codes and sums in the KCRS filter layout)
    gq = torch.empty((k, c, r, r), dtype=torch.int8, device=DEV)
    gacc = torch.empty((k, c, r, r), dtype=torch.int64, device=DEV)
    s_g = sc()
    iq.iq_conv_wgrad(d, dev(nchw(e)), sc(s_e), dev(nchw(x)), sc(s_x), gq, s_g, gq_mode=1, seed=3,
                     layer=ci, step=2, g_acc_out=gacc)
    G = O.conv_wgrad(cv, e, x)
    assert np.array_equal(host(gacc), kcrs(G))
    gw, gs = O.rq_int(G, s_e * s_x, 8, 1, 3, ci, 2)
    assert np.array_equal(host(gq).astype(np.int32), kcrs(gw)) and s_g.item() == gs


BITS_CASES = [
    # n, h, w, c, k, r, stride, pad, bn
    (2, 16, 16, 64, 64, 3, 1, 1, False),
    (1, 20, 18, 128, 96, 3, 1, 1, True),
    (2, 9, 9, 64, 32, 1, 1, 0, True),
]


@pytest.mark.parametrize("ci", range(len(BITS_CASES)))
def test_four_bit_layer_matches_oracle(ci):
    n, h, w, c, k, r, st, pd, bn = BITS_CASES[ci]
    kw = ka = 4
    cv = O.Conv(n, h, w, c, k, r, r, st, pd)
    d = iq.conv_desc(n, h, w, c, k, r, r, st, pd, k_w=kw, k_a=ka)
    p, q = cv.pq
    g = S.rng(800 + ci)
    # 4-bit activation codes in [0, 7] (a ReLU output under SQ(., 4)), errors at 8 bits
    x = np.maximum(g.integers(-7, 8, size=(n, h, w, c)), 0).astype(np.int8)
    master = O.uq(S.he_weights(g, (k, r, r, c), c * r * r), 24)
    wq = O.requant_master(master, 24, kw).astype(np.int8)
    assert np.abs(wq).max() <= 7
    e = S.int8_uniform(g, (n, p, q, k))
    s_x, s_e = 0.21, 2.0e-6
    s_acc = s_x * 2.0 ** (1 - kw)
    acc = O.conv_fwd(cv, x, wq)
    a = torch.empty((n, p, q, k), dtype=torch.int8, device=DEV)
    s_a = sc()
    if bn:
        gam, bet = S.bn_gamma_beta_codes(g, k)
        X = torch.empty((n, p, q, k), dtype=torch.int16, device=DEV)
        iq.iq_conv_fwd(d, dev(x), sc(s_x), dev(wq), a, s_a, dev(gam), dev(bet), use_bn=True,
                       relu=True, xhat=X)
        r_ = O.bn_fwd(acc.reshape(-1, k), s_acc, gam, bet, k_a=ka)
        assert np.array_equal(host(a).reshape(-1, k), r_.A)
        assert np.array_equal(host(X).reshape(-1, k), r_.X)
        assert s_a.item() == r_.s_a
        assert host(a).max() <= 7
        # the bits argument must agree with the descriptor's k_a
        with pytest.raises(iq.IqError):
            iq.iq_conv_fwd(d, dev(x), sc(s_x), dev(wq), a, s_a, dev(gam), dev(bet),
                           bits=iq.bn_bits(k_a=8), use_bn=True, relu=True)
    else:
        iq.iq_conv_fwd(d, dev(x), sc(s_x), dev(wq), a, s_a, relu=True)
        want, s_want = O.sq_int(acc, s_acc, ka, True)
        assert np.array_equal(host(a).astype(np.int32), want)
        assert s_a.item() == s_want
    dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    s_dx = sc()
    iq.iq_conv_dgrad(d, dev(e), sc(s_e), dev(wq), dx, s_dx)
    cw, sw = O.sq_int(O.conv_dgrad(cv, e, wq), s_e * 2.0 ** (1 - kw), 8)
    assert np.array_equal(host(dx).astype(np.int32), cw) and s_dx.item() == sw
    gq = torch.empty(wq.shape, dtype=torch.int8, device=DEV)
    s_g = sc()
    iq.iq_conv_wgrad(d, dev(e), sc(s_e), dev(x), sc(s_x), gq, s_g, gq_mode=1, seed=7, layer=ci,
                     step=1)
    gw, gs = O.rq_int(O.conv_wgrad(cv, e, x), s_e * s_x, 8, 1, 7, ci, 1)
    assert np.array_equal(host(gq).astype(np.int32), gw) and s_g.item() == gs
    # the update regenerates 4-bit forward codes from the 24-bit masters
    dm = dev(master.astype(np.int32))
    dwq = torch.empty(wq.shape, dtype=torch.int8, device=DEV)
    iq.iq_update(dm, dwq, gq, s_g, 6, k_w=kw)
    m2, w2 = O.update(master, gw, gs, 6, k_u=24, k_w=kw)
    assert np.array_equal(host(dm), m2)
    assert np.array_equal(host(dwq).astype(np.int32), w2)


def test_shared_input_carrier_ready_flag():
    """Two layers on one input (a block's first conv and its projection shortcut, the ASPP
    branches): the first forward writes the input's fp16 copy, the second reads it as it is
    (IQ_CONV_X_F16_READY); every forward and the weight gradients that read the same copy
    match the oracle."""
    n, h, w, c = 2, 33, 31, 128
    g = S.rng(911)
    x = S.int8_uniform(g, (n, h, w, c))
    x16 = torch.empty(x.size, dtype=torch.float16, device=DEV)
    xd = dev(x)
    s_x = 0.017
    for i, (k, r, pd, dl, bn, flags) in enumerate([(256, 1, 0, 1, True, 0),
                                                   (128, 3, 2, 2, True, iq.IQ_CONV_X_F16_READY),
                                                   (64, 3, 1, 1, False, iq.IQ_CONV_X_F16_READY)]):
        cv = O.Conv(n, h, w, c, k, r, r, 1, pd, dl)
        d = iq.conv_desc(n, h, w, c, k, r, r, 1, pd, dl, flags=flags)
        p, q = cv.pq
        wq = O.requant_master(O.uq(S.he_weights(g, (k, r, r, c), c * r * r), 24)).astype(np.int8)
        acc = O.conv_fwd(cv, x, wq)
        a = torch.empty((n, p, q, k), dtype=torch.int8, device=DEV)
        accd = torch.empty((n, p, q, k), dtype=torch.int32, device=DEV)
        s_a = sc()
        if bn:
            gam, bet = S.bn_gamma_beta_codes(g, k)
            iq.iq_conv_fwd(d, xd, sc(s_x), dev(wq), a, s_a, dev(gam), dev(bet), use_bn=True,
                           relu=True, acc_out=accd, x_f16=x16)
            r_ = O.bn_fwd(acc.reshape(-1, k), s_x * 2.0 ** -7, gam, bet)
            assert np.array_equal(host(a).reshape(-1, k), r_.A)
        else:
            iq.iq_conv_fwd(d, xd, sc(s_x), dev(wq), a, s_a, relu=True, acc_out=accd, x_f16=x16)
        assert np.array_equal(host(accd), acc), i
        # the weight gradient of this layer reads the same copy
        e = S.int8_uniform(g, (n, p, q, k))
        gacc = torch.empty((k, r, r, c), dtype=torch.int64, device=DEV)
        gq = torch.empty((k, r, r, c), dtype=torch.int8, device=DEV)
        iq.iq_conv_wgrad(d, dev(e), sc(1e-6), xd, sc(s_x), gq, sc(), gq_mode=1, seed=1, layer=i,
                         step=0, g_acc_out=gacc, x_f16=x16)
        assert np.array_equal(host(gacc), O.conv_wgrad(cv, e, x)), i


def _f16_codes(t16):
    """The int8 codes an fp16 copy holds (every int8 code is exact in fp16)."""
    torch.cuda.synchronize()
    v = t16.float().cpu().numpy()
    assert np.array_equal(v, np.round(v)) and np.abs(v).max() <= 127
    return v.astype(np.int8)


@pytest.mark.parametrize("bn,k_a", [(True, 0), (False, 0), (False, 4)])
def test_output_carrier_of_the_forward(bn, k_a):
    """a_f16: the requantization pass (the L1BN one, or the SQ one at 8 and at 4 bits) writes
    the fp16 copy of the output codes; a second layer reads it under IQ_CONV_X_F16_READY and
    matches the oracle."""
    n, h, w, c, k = 2, 19, 23, 64, 128
    g = S.rng(930 + 2 * bn + k_a)
    x = S.int8_uniform(g, (n, h, w, c))
    cv = O.Conv(n, h, w, c, k, 3, 3, 1, 1, 1)
    d = iq.conv_desc(n, h, w, c, k, 3, 3, 1, 1, k_a=k_a)
    wq = O.requant_master(O.uq(S.he_weights(g, (k, 3, 3, c), c * 9), 24)).astype(np.int8)
    a = torch.empty((n, h, w, k), dtype=torch.int8, device=DEV)
    a16 = torch.empty(a.numel(), dtype=torch.float16, device=DEV)
    s_a = sc()
    acc = O.conv_fwd(cv, x, wq)
    if bn:
        gam, bet = S.bn_gamma_beta_codes(g, k)
        iq.iq_conv_fwd(d, dev(x), sc(0.02), dev(wq), a, s_a, dev(gam), dev(bet), use_bn=True,
                       relu=True, a_f16=a16)
        want = O.bn_fwd(acc.reshape(-1, k), 0.02 * 2.0 ** -7, gam, bet).A.reshape(n, h, w, k)
    else:
        iq.iq_conv_fwd(d, dev(x), sc(0.02), dev(wq), a, s_a, relu=True, a_f16=a16)
        want, _ = O.sq_int(acc, 0.02 * 2.0 ** -7, 4 if k_a else 8, True)
    assert np.array_equal(host(a).astype(np.int32), want.astype(np.int32))
    assert np.array_equal(_f16_codes(a16).reshape(n, h, w, k), host(a))
    # the next layer reads the copy as it is
    k2 = 64
    cv2 = O.Conv(n, h, w, k, k2, 1, 1, 1, 0, 1)
    d2 = iq.conv_desc(n, h, w, k, k2, 1, 1, 1, 0, flags=iq.IQ_CONV_X_F16_READY)
    w2 = O.requant_master(O.uq(S.he_weights(g, (k2, 1, 1, k), k), 24)).astype(np.int8)
    acc2 = torch.empty((n, h, w, k2), dtype=torch.int32, device=DEV)
    iq.iq_conv_fwd(d2, a, s_a, dev(w2), torch.empty((n, h, w, k2), dtype=torch.int8, device=DEV),
                   sc(), relu=True, acc_out=acc2, x_f16=a16)
    assert np.array_equal(host(acc2), O.conv_fwd(cv2, host(a), w2))


def test_carriers_of_pool_relu_and_bn_backward():
    """y_f16 of the max pool, e_f16 of the ReLU backward and of the L1BN backward (the
    streamed tiles at 256 channels, the histogram path at 48) hold the fp16 copies of the
    codes they write; a data gradient reads the error copy under IQ_CONV_E_F16_READY."""
    g = S.rng(951)
    n, h, w, c = 2, 20, 22, 64
    x = S.int8_uniform(g, (n, h, w, c))
    y = torch.empty((n, h // 2, w // 2, c), dtype=torch.int8, device=DEV)
    arg = torch.empty_like(y, dtype=torch.uint8)
    y16 = torch.empty(y.numel(), dtype=torch.float16, device=DEV)
    iq.iq_maxpool_fwd(dev(x), 2, 2, 0, y, arg, y_f16=y16)
    yo, _ = O.maxpool_fwd(x, 2, 2, 0)
    assert np.array_equal(host(y), yo)
    assert np.array_equal(_f16_codes(y16).reshape(y.shape), yo)
    ea = S.int8_uniform(g, (n, h, w, c))
    e = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    e16 = torch.empty(e.numel(), dtype=torch.float16, device=DEV)
    iq.iq_relu_bwd(dev(ea), dev(x), e, e_f16=e16)
    assert np.array_equal(host(e), O.relu_bwd(ea, x))
    assert np.array_equal(_f16_codes(e16).reshape(e.shape), host(e))
    for C in (256, 48):
        m = 777
        acc = (g.standard_normal((m, C)) * 3000).astype(np.int32)
        gam, bet = S.bn_gamma_beta_codes(g, C)
        r = O.bn_fwd(acc, 2.0 ** -14, gam, bet)
        eA = S.int8_uniform(g, (m, C))
        want = O.bn_bwd(eA, 3e-6, r.A, r.X, r.s_xhat, gam, r.c_sigma)[0]
        codes = dev(np.concatenate([r.c_mu, r.c_sigma]))
        scal = torch.zeros(iq.IQ_BN_SCALES, dtype=torch.float64, device=DEV)
        scal[iq.IQ_BN_S_XHAT] = r.s_xhat
        eo = torch.empty((m, C), dtype=torch.int8, device=DEV)
        eo16 = torch.empty(eo.numel(), dtype=torch.float16, device=DEV)
        iq.iq_bn_int_bwd(dev(eA), sc(3e-6), dev(r.A), dev(r.X), dev(gam), codes, scal, eo, sc(),
                         e_f16=eo16)
        assert np.array_equal(host(eo), want), C
        assert np.array_equal(_f16_codes(eo16).reshape(m, C), want), C
    # a data gradient over an error copy written beforehand
    k = 64
    cv = O.Conv(n, h, w, c, k, 3, 3, 1, 1, 1)
    wq = O.requant_master(O.uq(S.he_weights(g, (k, 3, 3, c), c * 9), 24)).astype(np.int8)
    ee = S.int8_uniform(g, (n, h, w, k))
    ee16 = torch.empty(ee.size, dtype=torch.float16, device=DEV)
    iq.iq_relu_bwd(dev(ee), dev(np.full_like(ee, 1)), torch.empty_like(dev(ee)), e_f16=ee16)
    d = iq.conv_desc(n, h, w, c, k, 3, 3, 1, 1, flags=iq.IQ_CONV_E_F16_READY)
    dacc = torch.empty((n, h, w, c), dtype=torch.int32, device=DEV)
    dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    iq.iq_conv_dgrad(d, dev(ee), sc(1e-5), dev(wq), dx, sc(), acc_out=dacc, e_f16=ee16)
    assert np.array_equal(host(dacc), O.conv_dgrad(cv, ee, wq))


@pytest.mark.parametrize("case", ["tensor", "stride2", "int64"])
def test_dgrad_with_relu_mask_and_copy(case):
    """dx_mask / dx_f16: the data gradient's Q_E codes zeroed where the mask codes are not
    positive (the ReLU backward of the layer below, which iq_relu_bwd would apply next) and
    their fp16 copy, on the 4-wide SQ8 pass (tensor-core data gradient, stride-2 phases) and
    after the int64-sum form; the scale is the unmasked tensor's."""
    g = S.rng({"tensor": 971, "stride2": 972, "int64": 973}[case])
    if case == "tensor":
        n, h, w, c, k, r, st, pd = 2, 21, 19, 64, 128, 3, 1, 1
    elif case == "stride2":
        n, h, w, c, k, r, st, pd = 2, 18, 20, 64, 128, 3, 2, 1
    else:
        n, h, w, c, k, r, st, pd = 1, 8, 8, 64, 2720, 7, 1, 3    # (k r s) 127^2 >= 2^31
    cv = O.Conv(n, h, w, c, k, r, r, st, pd, 1)
    d = iq.conv_desc(n, h, w, c, k, r, r, st, pd)
    p, q = cv.pq
    if case == "int64":
        e = np.full((n, p, q, k), 127, np.int8)
        wq = np.full((k, r, r, c), 127, np.int8)
        wq[:, :, :, 3] = -127
    else:
        e = S.int8_uniform(g, (n, p, q, k))
        wq = O.requant_master(O.uq(S.he_weights(g, (k, r, r, c), c * r * r), 24)).astype(np.int8)
    mask = S.int8_uniform(g, (n, h, w, c))            # codes of either sign, zeros among them
    dx = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    dx16 = torch.full((dx.numel(),), float("nan"), dtype=torch.float16, device=DEV)
    s_dx = sc()
    iq.iq_conv_dgrad(d, dev(e), sc(1e-4), dev(wq), dx, s_dx, dx_mask=dev(mask), dx_f16=dx16)
    acc = O.conv_dgrad(cv, e, wq)
    codes, s_want = O.sq_int(acc, 1e-4 * 2.0 ** -7, 8)
    want = O.relu_bwd(codes.astype(np.int8), mask)
    assert np.array_equal(host(dx), want)
    assert s_dx.item() == s_want
    assert np.array_equal(_f16_codes(dx16).reshape(dx.shape), want)
