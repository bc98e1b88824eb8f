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
