"""GPU parity of the inference forward with frozen statistics, through the C ABI.

A calibration call of iq_conv_fwd exports its output map (frozen_out): with L1BN the
fixed-point F, B, G, H and the shifts P_x, P_a of Sec. 3.2.2's maps, without it the maximum M
that Q_A = SQ(ReLU(acc), 8) divides by.  These must equal the oracle's for the calibration
batch.  iq_conv_fwd_frozen then applies them to later batches -- one of them with activations
far beyond the calibration range -- and its X and A codes must equal the oracle's frozen maps
(or_bn_apply_fixed; SQ with the frozen M) on the accumulators of those batches."""
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


CASES = [
    # n, h, w, c, k, r, pad, dil, bn, relu: the all-TMA kernel (k > 128), the channel-major
    # kernel (k <= 128), an atrous 3x3, a 1x1 without BN and the 150-class padded score layer
    (2, 17, 15, 256, 256, 3, 1, 1, True, True),
    (2, 20, 20, 64, 64, 3, 1, 1, True, True),
    (1, 21, 21, 128, 192, 3, 4, 4, True, True),
    (2, 16, 16, 128, 256, 1, 0, 1, False, True),
    (4, 8, 8, 512, 150, 1, 0, 1, False, False),
]


def _acts(g, shape, hi=127):
    return np.maximum(g.integers(-hi, hi + 1, size=shape), 0).astype(np.int8)


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_frozen_forward_matches_oracle(ci):
    n, h, w, c, k, r, pd, dl, bn, relu = CASES[ci]
    cv = O.Conv(n, h, w, c, k, r, r, 1, pd, dl)
    d = iq.conv_desc(n, h, w, c, k, r, r, 1, pd, dl)
    p, q = cv.pq
    g = S.rng(900 + ci)
    wq = O.requant_master(O.uq(S.he_weights(g, (k, r, r, c), c * r * r), 24)).astype(np.int8)
    s_x = 0.02
    x0 = _acts(g, (n, h, w, c), 60)                 # calibration batch: codes up to 60
    acc0 = O.conv_fwd(cv, x0, wq)
    a = torch.empty((n, p, q, k), dtype=torch.int8, device=DEV)
    X = torch.empty((n, p, q, k), dtype=torch.int16, device=DEV) if bn else None
    s_a = sc()
    if bn:
        gam, bet = S.bn_gamma_beta_codes(g, k)
        fz = torch.empty(4 * k + 2, dtype=torch.int64, device=DEV)
        iq.iq_conv_fwd(d, dev(x0), sc(s_x), dev(wq), a, s_a, dev(gam), dev(bet), use_bn=True,
                       relu=True, xhat=X, frozen_out=fz)
        r0 = O.bn_fwd(acc0.reshape(-1, k), s_x * 2.0 ** -7, gam, bet)
        want = np.concatenate([r0.F, r0.B, r0.G, r0.H, [r0.p_x, r0.p_a]]).astype(np.int64)
        assert np.array_equal(host(fz), want)
        assert np.array_equal(host(a).reshape(-1, k), r0.A)
    else:
        fz = torch.empty(1, dtype=torch.int64, device=DEV)
        iq.iq_conv_fwd(d, dev(x0), sc(s_x), dev(wq), a, s_a, relu=relu, frozen_out=fz)
        M = int((np.maximum(acc0, 0) if relu else np.abs(acc0)).max())
        assert int(host(fz)[0]) == M
    # later batches: the same range, and codes up to 127 (beyond the calibration's 60)
    for b, hi in ((0, 60), (1, 127)):
        x1 = _acts(g, (n, h, w, c), hi)
        acc1 = O.conv_fwd(cv, x1, wq)
        a1 = torch.empty((n, p, q, k), dtype=torch.int8, device=DEV)
        if bn:
            X1 = torch.empty((n, p, q, k), dtype=torch.int16, device=DEV)
            iq.iq_conv_fwd_frozen(d, dev(x1), dev(wq), fz, a1, use_bn=True, xhat=X1)
            Xw, Aw = O.bn_apply_fixed(acc1.reshape(-1, k), r0.F, r0.B, r0.G, r0.H, r0.p_x,
                                      r0.p_a)
            assert np.array_equal(host(X1).reshape(-1, k), Xw), b
            assert np.array_equal(host(a1).reshape(-1, k), Aw), b
        else:
            iq.iq_conv_fwd_frozen(d, dev(x1), dev(wq), fz, a1, relu=relu)
            Aw, _ = O.sq_at(acc1.ravel(), M, 1.0, 8, relu)
            assert np.array_equal(host(a1).ravel().astype(np.int32), Aw), b


def test_frozen_forward_nchw_and_argument_checks():
    n, h, w, c, k = 2, 12, 12, 64, 128
    cv = O.Conv(n, h, w, c, k, 3, 3, 1, 1)
    d = iq.conv_desc(n, h, w, c, k, 3, 3, 1, 1, layout=iq.IQ_LAYOUT_NCHW)
    p, q = cv.pq
    g = S.rng(950)
    wq = O.requant_master(O.uq(S.he_weights(g, (k, 3, 3, c), c * 9), 24)).astype(np.int8)
    x0, x1 = _acts(g, (n, h, w, c)), _acts(g, (n, h, w, c))
    gam, bet = S.bn_gamma_beta_codes(g, k)
    nchw = lambda t: np.ascontiguousarray(np.moveaxis(t, -1, 1))
    kcrs = nchw
    fz = torch.empty(4 * k + 2, dtype=torch.int64, device=DEV)
    a = torch.empty((n, k, p, q), dtype=torch.int8, device=DEV)
    iq.iq_conv_fwd(d, dev(nchw(x0)), sc(0.01), dev(kcrs(wq)), a, sc(), dev(gam), dev(bet),
                   use_bn=True, relu=True, frozen_out=fz)
    r0 = O.bn_fwd(O.conv_fwd(cv, x0, wq).reshape(-1, k), 0.01 * 2.0 ** -7, gam, bet)
    iq.iq_conv_fwd_frozen(d, dev(nchw(x1)), dev(kcrs(wq)), fz, a, use_bn=True)
    _, Aw = O.bn_apply_fixed(O.conv_fwd(cv, x1, wq).reshape(-1, k), r0.F, r0.B, r0.G, r0.H,
                             r0.p_x, r0.p_a)
    assert np.array_equal(host(a), nchw(Aw.reshape(n, p, q, k)))
    # X codes exist only with batch norm; the constants are required
    dn = iq.conv_desc(n, h, w, c, k, 3, 3, 1, 1)
    with pytest.raises(iq.IqError):
        iq.iq_conv_fwd_frozen(dn, dev(x1), dev(wq), fz, a, use_bn=False,
                              xhat=torch.empty((n, p, q, k), dtype=torch.int16, device=DEV))
    with pytest.raises(iq.IqError):
        iq.iq_conv_fwd_frozen(dn, dev(x1), dev(wq), None, a, use_bn=True)
