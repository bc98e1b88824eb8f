"""Pins of the oracle's DeepLab glue against what mathematics fixes (CPU only).

Covered: the quantized sum / concatenation (residual add, sum of errors, ASPP concat),
spatial sums (global average pooling and the backward of a broadcast), the x8
aligned-corner bilinear upsampling and its adjoint, the fp32 exponential of the softmax
head and the cross-entropy gradient.  Every expected value here comes from an independent
route: exact rationals (fractions), torch's fp64 interpolation, numpy fp64 softmax,
adjoint identities and brute force.
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle as O


def sq8_exact(vals):
    """Eq. (ScaleQ) with Scale = max|v| on exact rationals: rhu(v / M * 128), clipped."""
    M = max((abs(v) for v in vals), default=Fraction(0))
    if M == 0:
        return np.zeros(len(vals), np.int64), M
    out = []
    for v in vals:
        y = v / M * 128
        c = math.floor(y + Fraction(1, 2))
        out.append(max(-127, min(127, c)))
    return np.array(out, np.int64), M


# ---------------------------------------------------------------- combine

def test_combine_single_term_is_integer_sq():
    g = np.random.default_rng(1)
    v = g.integers(-127, 128, size=(2, 5, 8), dtype=np.int8)
    s = 0.0123
    out, so = O.combine([O.CombineTerm(v, s)], 2, 5, 8)
    codes, M = sq8_exact([Fraction(int(a)) for a in v.ravel()])
    assert np.array_equal(out.astype(np.int64), codes)
    assert so == pytest.approx(s * float(M) / 128, rel=2.0 ** -45)


def test_combine_equal_scales_is_sq_of_integer_sum():
    g = np.random.default_rng(2)
    a = g.integers(-127, 128, size=(1, 7, 6), dtype=np.int8)
    b = g.integers(-127, 128, size=(1, 7, 6), dtype=np.int8)
    s = 2.0 ** -9 * 3
    out, so = O.combine([O.CombineTerm(a, s), O.CombineTerm(b, s)], 1, 7, 6, relu=True)
    tot = [Fraction(max(0, int(x) + int(y))) for x, y in zip(a.ravel(), b.ravel())]
    codes, M = sq8_exact(tot)
    assert np.array_equal(out.astype(np.int64), codes)
    assert so == pytest.approx(s * float(M) / 128, rel=2.0 ** -45)


def test_combine_bn_affine_and_residual_matches_rationals():
    """ReLU(gamma_q xhat + beta_q + shortcut): the residual add of a bottleneck."""
    g = np.random.default_rng(3)
    n, hw, c = 2, 9, 12
    X = g.integers(-32767, 32768, size=(n, hw, c), dtype=np.int16)
    sc = g.integers(0, 128, size=(n, hw, c), dtype=np.int8)
    gam = g.integers(-127, 128, size=c).astype(np.int32)
    bet = g.integers(-127, 128, size=c).astype(np.int32)
    s_x, s_sc = 2.0 ** -15 * 5.5, 0.0371
    out, so = O.combine([O.CombineTerm(X, s_x, gamma=gam, beta=bet), O.CombineTerm(sc, s_sc)],
                        n, hw, c, relu=True)
    vals = []
    Fs, Fss = Fraction(s_x), Fraction(s_sc)
    for i in range(n * hw):
        for ch in range(c):
            y = (Fraction(int(gam[ch]), 64) * Fraction(int(X.reshape(-1, c)[i, ch])) * Fs
                 + Fraction(int(bet[ch]), 64) + Fraction(int(sc.reshape(-1, c)[i, ch])) * Fss)
            vals.append(max(Fraction(0), y))
    codes, M = sq8_exact(vals)
    d = np.abs(out.astype(np.int64) - codes)
    assert d.max() <= 1 and np.count_nonzero(d) <= 1
    assert so == pytest.approx(float(M) / 128, rel=2.0 ** -40)


def test_combine_concat_with_broadcast_term():
    g = np.random.default_rng(4)
    n, hw = 2, 6
    a = g.integers(0, 128, size=(n, hw, 4), dtype=np.int8)
    b = g.integers(0, 128, size=(n, hw, 3), dtype=np.int8)
    p = g.integers(0, 128, size=(n, 5), dtype=np.int8)
    sa, sb, sp = 0.02, 0.5, 0.003
    out, so = O.combine([O.CombineTerm(a, sa, 0), O.CombineTerm(b, sb, 4),
                         O.CombineTerm(p, sp, 7, bcast=True)], n, hw, 12, concat=True)
    vals = []
    for i in range(n):
        for q in range(hw):
            vals += [Fraction(int(v)) * Fraction(sa) for v in a[i, q]]
            vals += [Fraction(int(v)) * Fraction(sb) for v in b[i, q]]
            vals += [Fraction(int(v)) * Fraction(sp) for v in p[i]]
    codes, M = sq8_exact(vals)
    assert np.array_equal(out.astype(np.int64), codes)
    assert so == pytest.approx(float(M) / 128, rel=2.0 ** -40)


def test_combine_all_zero():
    z = np.zeros((1, 4, 8), np.int8)
    out, so = O.combine([O.CombineTerm(z, 0.5)], 1, 4, 8)
    assert not out.any() and so > 0


# ---------------------------------------------------------------- spatial sums

@pytest.mark.parametrize("mean", [True, False])
def test_spatial_sum_matches_rationals(mean):
    g = np.random.default_rng(5)
    x = g.integers(-127, 128, size=(3, 5, 7, 10), dtype=np.int8)
    s = 0.0077
    out, so = O.spatial_sum(x, s, mean, c_offset=2, c=6)
    vals = []
    for i in range(3):
        for ch in range(6):
            t = Fraction(int(x[i, :, :, 2 + ch].astype(np.int64).sum())) * Fraction(s)
            vals.append(t / 35 if mean else t)
    codes, M = sq8_exact(vals)
    assert np.array_equal(out.ravel().astype(np.int64), codes)
    assert so == pytest.approx(float(M) / 128, rel=2.0 ** -45)


# ---------------------------------------------------------------- bilinear x f

def interp_matrix(h, f):
    """1-D linear interpolation with aligned corners, times f: U[I, i] = f - |I - f i|."""
    H = (h - 1) * f + 1
    U = np.zeros((H, h), np.int64)
    for I in range(H):
        for i in range(h):
            U[I, i] = max(0, f - abs(I - f * i))
    return U


@pytest.mark.parametrize("f,h,w", [(8, 3, 4), (2, 5, 5), (4, 1, 3)])
def test_bilinear_up_matches_torch_align_corners(f, h, w):
    g = np.random.default_rng(6)
    x = g.integers(-127, 128, size=(2, h, w, 3), dtype=np.int8)
    out, so, acc = O.bilinear_up(x, 0.01, f)
    H, W = (h - 1) * f + 1, (w - 1) * f + 1
    t = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
    ref = torch.nn.functional.interpolate(t, size=(H, W), mode="bilinear", align_corners=True)
    ref = (ref * (f * f)).permute(0, 2, 3, 1).numpy()
    assert np.array_equal(acc.astype(np.float64), ref)
    codes, M = sq8_exact([Fraction(int(v)) for v in acc.ravel()])
    assert np.array_equal(out.ravel().astype(np.int64), codes)
    assert so == pytest.approx(0.01 * float(M) / (f * f) / 128, rel=2.0 ** -45)


def test_bilinear_up_constant_and_identity():
    x = np.full((1, 4, 5, 2), 37, np.int8)
    out, so, acc = O.bilinear_up(x, 0.25, 8)
    assert (out == 127).all() and so == pytest.approx(0.25 * 37 / 127 * (127 / 128), rel=1e-15)
    y = np.random.default_rng(7).integers(-127, 128, size=(1, 3, 3, 4), dtype=np.int8)
    o1, s1, a1 = O.bilinear_up(y, 1.0, 1)
    assert np.array_equal(a1, y.astype(np.int32))


def test_bilinear_up_bwd_is_the_adjoint():
    g = np.random.default_rng(8)
    f, h, w = 8, 3, 4
    x = g.integers(-127, 128, size=(2, h, w, 3), dtype=np.int8)
    e = g.integers(-127, 128, size=(2, (h - 1) * f + 1, (w - 1) * f + 1, 3), dtype=np.int8)
    _, _, afwd = O.bilinear_up(x, 1.0, f)
    eb, sb, abwd = O.bilinear_up_bwd(e, 0.5, f, x.shape)
    lhs = int((afwd.astype(np.int64) * e.astype(np.int64)).sum())
    rhs = int((x.astype(np.int64) * abwd).sum())
    assert lhs == rhs
    Uh, Uw = interp_matrix(h, f), interp_matrix(w, f)
    ref = np.einsum("Ii,nIJc,Jj->nijc", Uh, e.astype(np.int64), Uw)
    assert np.array_equal(abwd, ref)
    codes, M = sq8_exact([Fraction(int(v)) for v in abwd.ravel()])
    assert np.array_equal(eb.ravel().astype(np.int64), codes)
    assert sb == pytest.approx(0.5 * float(M) / 64 / 128, rel=2.0 ** -45)


# ---------------------------------------------------------------- softmax head

def test_exp_f32_accuracy_and_special_values():
    g = np.random.default_rng(9)
    t = np.concatenate([g.uniform(-87.0, 0.0, 400000), g.uniform(-1.0, 0.0, 100000),
                        -np.arange(0, 87.01, 0.125)]).astype(np.float32)
    y = O.exp_f32(t).astype(np.float64)
    ref = np.exp(t.astype(np.float64))
    rel = np.abs(y - ref) / ref
    # <= 2 units in the last place of the fp32 result (2^-22 relative bounds 2 ulp)
    assert rel.max() < 2.0 ** -22, rel.max()
    assert O.exp_f32(np.array([0.0], np.float32))[0] == 1.0
    assert (O.exp_f32(np.array([-87.5, -100.0, -np.inf], np.float32)) == 0).all()
    # t = -k ln 2 rounded to fp32 is a different number for every k: compare with the
    # exact exponential of that fp32 input at the range-reduction boundaries
    t = (-np.arange(1, 126) * math.log(2)).astype(np.float32)
    y = O.exp_f32(t).astype(np.float64)
    assert np.all(np.abs(y / np.exp(t.astype(np.float64)) - 1) < 2.0 ** -22)


def softmax_grad_fp64(z, s, lab, ignore=255):
    t = z.astype(np.float64) * s
    t = t - t.max(axis=-1, keepdims=True)
    p = np.exp(t)
    p = p / p.sum(axis=-1, keepdims=True)
    oh = np.zeros_like(p)
    valid = lab != ignore
    idx = np.nonzero(valid)
    oh[idx + (lab[valid].astype(np.int64),)] = 1.0
    gr = p - oh
    gr[~valid] = 0.0
    return gr, int(valid.sum())


def test_ce_grad_close_to_fp64_softmax():
    g = np.random.default_rng(10)
    z = g.integers(-127, 128, size=(3, 11, 13, 21), dtype=np.int8)
    lab = g.integers(0, 21, size=(3, 11, 13)).astype(np.uint8)
    lab[g.random(lab.shape) < 0.05] = 255
    s = 0.04
    E, se, nv = O.ce_grad(z, s, lab)
    gr, nv_ref = softmax_grad_fp64(z, s, lab)
    assert nv == nv_ref
    M = np.abs(gr).max()
    assert se == pytest.approx(M / 128 / nv, rel=1e-6)
    ref = np.clip(np.floor(gr / M * 128 + 0.5), -127, 127)
    d = np.abs(E.astype(np.float64) - ref)
    assert d.max() <= 1 and np.count_nonzero(d) <= 2e-3 * d.size
    assert not E[lab == 255].any()
    # per pixel the (unquantized) gradient sums to 0; codes within rounding of that
    sums = E.astype(np.int64).sum(-1)[lab != 255]
    assert np.abs(sums).max() <= 21


def test_ce_grad_two_classes_is_sigmoid_and_uniform_case():
    z = np.array([[[[10, -10]]]], np.int8)
    lab = np.array([[[0]]], np.uint8)
    E, se, nv = O.ce_grad(z, 0.1, lab)
    p0 = 1.0 / (1.0 + math.exp(-2.0))
    assert nv == 1 and list(E.ravel()) == [-127, 127]
    assert se == pytest.approx((1 - p0) / 128, rel=1e-6)
    zu = np.zeros((1, 2, 2, 4), np.int8)
    lab = np.array([[[0, 1], [2, 255]]], np.uint8)
    E, se, nv = O.ce_grad(zu, 1.0, lab)
    assert nv == 3 and (E[0, 1, 1] == 0).all()
    # p = 1/4 everywhere: g = -3/4 at the label, 1/4 elsewhere -> codes -127 and 43
    assert E[0, 0, 0, 0] == -127 and E[0, 0, 0, 1] == math.floor(128 / 3 + 0.5)
    all_ignored = np.full((1, 2, 2), 255, np.uint8)
    E, se, nv = O.ce_grad(zu, 1.0, all_ignored)
    assert nv == 0 and not E.any() and se == 2.0 ** -7
