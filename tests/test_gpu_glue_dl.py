"""GPU parity of the DeepLab glue calls against the oracle: every code bit-exact and every
scale equal as fp64 (0 ULP), on seeded inputs that span several blocks and ragged tails,
plus the full-size shapes of the DeepLabv3-ResNet50 head (65 -> 513, 21 classes)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import iq

pytestmark = pytest.mark.gpu

DEV = "cuda"


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def dscal(v):
    return torch.tensor([v], dtype=torch.float64, device=DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def scal():
    return torch.zeros(1, dtype=torch.float64, device=DEV)


# ---------------------------------------------------------------- combine

def dev_offset(a, elems):
    """A device copy of `a` that starts `elems` elements into a larger buffer (an address
    that is not 16-byte aligned when elems * itemsize is not a multiple of 16)."""
    flat = np.ascontiguousarray(a).ravel()
    buf = torch.zeros(flat.size + elems, dtype=dev(flat[:1]).dtype, device=DEV)
    buf[elems:] = dev(flat)
    return buf[elems:].view(a.shape)


def run_combine(specs, n, hw, c_out, concat, relu, misalign=False):
    """specs: list of (codes np, scale, c_offset, bcast, gamma np|None, beta np|None).
    misalign: operands 8 bytes past a 16-byte boundary."""
    keep, terms, oterms = [], [], []
    for codes, s, off, bc, gam, bet in specs:
        dc = dev_offset(codes, 8 // codes.itemsize) if misalign else dev(codes)
        ds = dscal(s)
        dg = dev(gam) if gam is not None else None
        db = dev(bet) if bet is not None else None
        keep += [dc, ds, dg, db]
        terms.append(iq.term(dc, ds, off, bc, dg, db))
        oterms.append(O.CombineTerm(codes, s, off, bc, gam, bet))
    out = torch.empty(n * hw * c_out, dtype=torch.int8, device=DEV)
    so = scal()
    # the fp16 copy of the output codes wherever its size allows one
    out16 = (torch.empty(out.numel(), dtype=torch.float16, device=DEV)
             if out.numel() % 16 == 0 else None)
    iq.iq_combine(terms, n, hw, c_out, out, so, concat=concat, relu=relu, out_f16=out16)
    ref, sref = O.combine(oterms, n, hw, c_out, concat=concat, relu=relu)
    assert np.array_equal(host(out), ref)
    assert host(so)[0] == sref
    if out16 is not None:
        assert np.array_equal(host(out16).astype(np.float32), ref.astype(np.float32))


def test_combine_residual_bn_affine_plus_shortcut():
    g = np.random.default_rng(11)
    n, hw, c = 2, 37 * 29, 96
    X = g.integers(-32767, 32768, size=(n, hw, c)).astype(np.int16)
    sc = g.integers(0, 128, size=(n, hw, c)).astype(np.int8)
    gam = g.integers(-100, 128, size=c).astype(np.int32)
    bet = g.integers(-127, 128, size=c).astype(np.int32)
    run_combine([(X, 2.0 ** -15 * 3.7, 0, False, gam, bet), (sc, 0.041, 0, False, None, None)],
                n, hw, c, False, True)


def test_combine_two_bn_branches_downsample():
    g = np.random.default_rng(12)
    n, hw, c = 3, 17 * 17, 64
    terms = []
    for k in range(2):
        X = g.integers(-32767, 32768, size=(n, hw, c)).astype(np.int16)
        gam = g.integers(-127, 128, size=c).astype(np.int32)
        bet = g.integers(-127, 128, size=c).astype(np.int32)
        terms.append((X, 2.0 ** -15 * (1.5 + k), 0, False, gam, bet))
    run_combine(terms, n, hw, c, False, True)


def test_combine_sum_of_errors_with_broadcast():
    """The error reaching the ASPP input: four branch errors plus the pooled one."""
    g = np.random.default_rng(13)
    n, hw, c = 2, 9 * 11, 40
    specs = [(g.integers(-127, 128, size=(n, hw, c)).astype(np.int8), s, 0, False, None, None)
             for s in (0.01, 0.3, 1e-4, 0.02)]
    specs.append((g.integers(-127, 128, size=(n, c)).astype(np.int8), 0.5 / hw, 0, True, None, None))
    run_combine(specs, n, hw, c, False, False)


def test_combine_sum_of_many_operands_all_channels():
    # three to six operands covering every channel (the shared-memory row kernel): int16
    # with the BN affine, int8, and a broadcast term, with and without ReLU
    g = np.random.default_rng(20)
    n, hw, c = 3, 33 * 31, 64
    X = g.integers(-32767, 32768, size=(n, hw, c)).astype(np.int16)
    gam = g.integers(-127, 128, size=c).astype(np.int32)
    bet = g.integers(-127, 128, size=c).astype(np.int32)
    specs = [(X, 2.0 ** -15 * 2.1, 0, False, gam, bet),
             (g.integers(-127, 128, size=(n, hw, c)).astype(np.int8), 0.03, 0, False, None, None),
             (g.integers(-127, 128, size=(n, c)).astype(np.int8), 0.2, 0, True, None, None)]
    run_combine(specs, n, hw, c, False, True)
    more = specs + [(g.integers(-127, 128, size=(n, hw, c)).astype(np.int8), s, 0, False, None,
                     None) for s in (0.5, 1e-3, 0.07)]
    run_combine(more, n, hw, c, False, False)


def test_combine_concat_aspp():
    g = np.random.default_rng(14)
    n, hw, cb = 2, 13 * 13, 32
    specs = [(g.integers(0, 128, size=(n, hw, cb)).astype(np.int8), 0.01 * (k + 1), k * cb, False,
              None, None) for k in range(4)]
    specs.append((g.integers(0, 128, size=(n, cb)).astype(np.int8), 0.07, 4 * cb, True, None, None))
    run_combine(specs, n, hw, 5 * cb, True, False)


@pytest.mark.parametrize("n,hw,c", [(3, 7 * 13, 36), (2, 65 * 65, 256)])
def test_combine_four_channel_groups(n, hw, c):
    # c_out a multiple of 4 (not of 8 in the first case) and an odd pixel count: the
    # 4-channel kernel, its pairs of pixels and its single-pixel tail; then a full-size
    # bottleneck join (65 x 65 x 256)
    g = np.random.default_rng(18 + c)
    X = g.integers(-32767, 32768, size=(n, hw, c)).astype(np.int16)
    sc = g.integers(-127, 128, size=(n, hw, c)).astype(np.int8)
    gam = g.integers(-127, 128, size=c).astype(np.int32)
    bet = g.integers(-127, 128, size=c).astype(np.int32)
    run_combine([(X, 2.0 ** -15 * 1.9, 0, False, gam, bet), (sc, 0.013, 0, False, None, None)],
                n, hw, c, False, True)
    run_combine([(sc, 0.02, 0, False, None, None), (X, 2.0 ** -15, 0, False, gam, bet)],
                n, hw, c, False, False)


@pytest.mark.parametrize("n,hw,c,kinds,relu", [
    (3, 37 * 41, 512, ("x16", "x16"), True),      # downsample join, ragged last chunk
    (2, 29 * 31, 128, ("i8", "x16"), True),       # identity first, 16 row lanes
    (2, 23 * 19, 2048, ("e8", "e8"), False),      # sum of two errors over two slabs
    (1, 11 * 13, 3072, ("x16", "i8"), False),     # three slabs of 1024 channels
    (4, 65 * 65, 1024, ("e8", "e8"), False),      # a full-size stage-3 error sum
])
def test_combine_streamed_two_operands(n, hw, c, kinds, relu):
    """Two operands covering every channel with at least 128 channels (the streamed passes):
    int16 codes with the BN affine, int8 codes of a shortcut, and plain int8 errors."""
    g = np.random.default_rng(31 + c + hw)
    specs = []
    for k, kind in enumerate(kinds):
        if kind == "x16":
            X = g.integers(-32767, 32768, size=(n, hw, c)).astype(np.int16)
            gam = g.integers(-127, 128, size=c).astype(np.int32)
            bet = g.integers(-127, 128, size=c).astype(np.int32)
            specs.append((X, 2.0 ** -15 * (1.7 + k), 0, False, gam, bet))
        else:
            lo = 0 if kind == "i8" else -127
            v = g.integers(lo, 128, size=(n, hw, c)).astype(np.int8)
            specs.append((v, 0.021 if k else 3e-5, 0, False, None, None))
    run_combine(specs, n, hw, c, False, relu)


def test_combine_streamed_exact_paths():
    """The streamed passes where fp32 cannot decide: codes of magnitude <= 3 far below the
    fixed-point bound (every element exact), constant codes (every element at the maximum),
    and a ReLU sum that is negative everywhere (every code 0)."""
    g = np.random.default_rng(41)
    n, hw, c = 2, 17 * 19, 256
    X = g.integers(-3, 4, size=(n, hw, c)).astype(np.int16)
    sc = g.integers(-127, 128, size=(n, hw, c)).astype(np.int8)
    gam = g.integers(-127, 128, size=c).astype(np.int32)
    run_combine([(X, 2.0 ** -15, 0, False, gam, np.zeros(c, np.int32)),
                 (sc, 2.0 ** -30, 0, False, None, None)], n, hw, c, False, False)
    run_combine([(np.full((n, hw, c), 77, np.int8), 0.013, 0, False, None, None),
                 (np.full((n, hw, c), -5, np.int8), 0.2, 0, False, None, None)], n, hw, c,
                False, False)
    neg = -np.abs(g.integers(1, 128, size=(n, hw, c))).astype(np.int8)
    run_combine([(neg, 0.01, 0, False, None, None), (neg, 0.02, 0, False, None, None)],
                n, hw, c, False, True)


def test_combine_unaligned_operands():
    """Operands whose codes start 8 bytes past a 16-byte boundary (4-byte loads of int8
    codes, 8-byte loads of int16 codes stay aligned): a two-operand residual join and a
    five-operand sum with a broadcast operand."""
    g = np.random.default_rng(21)
    n, hw, c = 2, 21 * 23, 64
    X = g.integers(-32767, 32768, size=(n, hw, c)).astype(np.int16)
    sc = g.integers(-127, 128, size=(n, hw, c)).astype(np.int8)
    gam = g.integers(-127, 128, size=c).astype(np.int32)
    bet = g.integers(-127, 128, size=c).astype(np.int32)
    run_combine([(X, 2.0 ** -15 * 1.3, 0, False, gam, bet), (sc, 0.017, 0, False, None, None)],
                n, hw, c, False, True, misalign=True)
    specs = [(g.integers(-127, 128, size=(n, hw, c)).astype(np.int8), s, 0, False, None, None)
             for s in (0.01, 0.3, 1e-4, 0.02)]
    specs.append((g.integers(-127, 128, size=(n, c)).astype(np.int8), 0.5 / hw, 0, True, None, None))
    run_combine(specs, n, hw, c, False, False, misalign=True)


def test_combine_small_values_and_negative_relu():
    # values far below the fixed-point bound (int16 codes in [-3, 3]): M < 2^37, so the
    # float estimate cannot decide and every element takes the exact form; then a ReLU join
    # whose sums are all negative (max 0, every code 0)
    g = np.random.default_rng(19)
    n, hw, c = 2, 23 * 19, 48
    X = g.integers(-3, 4, size=(n, hw, c)).astype(np.int16)
    sc = g.integers(-127, 128, size=(n, hw, c)).astype(np.int8)
    gam = g.integers(-127, 128, size=c).astype(np.int32)
    bet = np.zeros(c, np.int32)
    run_combine([(X, 2.0 ** -15, 0, False, gam, bet), (sc, 2.0 ** -30, 0, False, None, None)],
                n, hw, c, False, False)
    neg = -np.abs(g.integers(1, 128, size=(n, hw, c))).astype(np.int8)
    run_combine([(neg, 0.01, 0, False, None, None), (neg, 0.02, 0, False, None, None)],
                n, hw, c, False, True)


def test_combine_ties_at_the_maximum():
    """Every element at the tensor's largest magnitude (constant codes): the max pass must
    take the exact form for all of them; then a three-operand int8 sum over 64 channels
    and an odd pixel count (16 channels per thread, more than two operands per group)."""
    n, hw, c = 2, 13 * 11, 64
    run_combine([(np.full((n, hw, c), 77, np.int8), 0.013, 0, False, None, None),
                 (np.full((n, hw, c), -5, np.int8), 0.2, 0, False, None, None)], n, hw, c,
                False, False)
    run_combine([(np.full((n, hw, c), 127, np.int8), 1e-6, 0, False, None, None)], n, hw, c,
                False, True)
    g = np.random.default_rng(22)
    specs = [(g.integers(-127, 128, size=(n, hw, c)).astype(np.int8), s, 0, False, None, None)
             for s in (3e-7, 1.1e-6, 2e-9)]
    run_combine(specs, n, hw, c, False, False)


def test_combine_edge_cases():
    # all zero, a single pixel, a single channel
    run_combine([(np.zeros((1, 5, 8), np.int8), 0.5, 0, False, None, None)], 1, 5, 8, False, False)
    run_combine([(np.full((1, 1, 3), -127, np.int8), 0.5, 0, False, None, None),
                 (np.full((1, 1, 3), 127, np.int8), 0.25, 0, False, None, None)], 1, 1, 3, False,
                False)
    g = np.random.default_rng(15)
    run_combine([(g.integers(-127, 128, size=(4, 33, 1)).astype(np.int8), 3.0, 0, False, None,
                  None)], 4, 33, 1, False, True)


# ---------------------------------------------------------------- spatial sums, slices

@pytest.mark.parametrize("mean,n,h,w,ct,off,c", [(True, 2, 65, 65, 256, 0, 256),
                                                  (True, 3, 7, 5, 40, 0, 40),
                                                  (False, 2, 9, 9, 96, 64, 32),
                                                  (False, 1, 1, 1, 8, 3, 5)])
def test_spatial_sum(mean, n, h, w, ct, off, c):
    g = np.random.default_rng(16)
    x = g.integers(-127, 128, size=(n, h, w, ct)).astype(np.int8)
    out = torch.empty((n, c), dtype=torch.int8, device=DEV)
    so = scal()
    iq.iq_spatial_sum(dev(x), dscal(0.013), out, so, mean=mean, c_off=off, c=c)
    ref, sref = O.spatial_sum(x, 0.013, mean, c_offset=off, c=c)
    assert np.array_equal(host(out), ref) and host(so)[0] == sref


def test_avgpool_bwd_and_channel_slice():
    g = np.random.default_rng(17)
    e = g.integers(-127, 128, size=(3, 24)).astype(np.int8)
    ex = torch.empty((3, 35, 24), dtype=torch.int8, device=DEV)
    sx = scal()
    iq.iq_avgpool_bwd(dev(e), dscal(0.37), 35, sx, ex=ex)
    assert host(sx)[0] == 0.37 / 35
    assert np.array_equal(host(ex), np.broadcast_to(e[:, None, :], (3, 35, 24)))
    x = g.integers(-127, 128, size=(2, 5, 7, 48)).astype(np.int8)
    out = torch.empty((2, 5, 7, 20), dtype=torch.int8, device=DEV)
    iq.iq_channel_slice(dev(x), 17, 20, out)
    assert np.array_equal(host(out), x[..., 17:37])


# ---------------------------------------------------------------- bilinear, softmax head

@pytest.mark.parametrize("n,h,w,c,f", [(2, 9, 9, 21, 8), (1, 5, 7, 3, 4), (3, 4, 3, 5, 1),
                                       (2, 65, 65, 21, 8)])
def test_bilinear_up_fwd_bwd(n, h, w, c, f):
    g = np.random.default_rng(18)
    x = g.integers(-127, 128, size=(n, h, w, c)).astype(np.int8)
    H, W = (h - 1) * f + 1, (w - 1) * f + 1
    out = torch.empty((n, H, W, c), dtype=torch.int8, device=DEV)
    so = scal()
    iq.iq_bilinear_up_fwd(dev(x), dscal(0.02), f, out, so)
    ref, sref, _ = O.bilinear_up(x, 0.02, f)
    assert np.array_equal(host(out), ref) and host(so)[0] == sref
    e = g.integers(-127, 128, size=(n, H, W, c)).astype(np.int8)
    ex = torch.empty((n, h, w, c), dtype=torch.int8, device=DEV)
    sx = scal()
    iq.iq_bilinear_up_bwd(dev(e), dscal(0.003), f, (n, h, w, c), ex, sx)
    refb, srefb, _ = O.bilinear_up_bwd(e, 0.003, f, (n, h, w, c))
    assert np.array_equal(host(ex), refb) and host(sx)[0] == srefb


@pytest.mark.parametrize("n,h,w,c,s", [(2, 33, 35, 21, 0.05), (1, 7, 9, 150, 0.5),
                                       (2, 513, 513, 21, 0.03), (1, 3, 3, 2, 4.0)])
def test_ce_grad(n, h, w, c, s):
    g = np.random.default_rng(19)
    z = g.integers(-127, 128, size=(n, h, w, c)).astype(np.int8)
    lab = g.integers(0, c, size=(n, h, w)).astype(np.uint8)
    lab[g.random(lab.shape) < 0.05] = 255
    E = torch.empty_like(dev(z))
    se = scal()
    nv = torch.zeros(1, dtype=torch.int64, device=DEV)
    iq.iq_ce_grad(dev(z), dscal(s), dev(lab), E, se, n_valid=nv)
    ref, sref, nref = O.ce_grad(z, s, lab)
    assert host(nv)[0] == nref
    assert np.array_equal(host(E), ref) and host(se)[0] == sref


def test_ce_grad_all_ignored_and_saturated():
    z = np.zeros((1, 4, 4, 21), np.int8)
    lab = np.full((1, 4, 4), 255, np.uint8)
    E = torch.ones((1, 4, 4, 21), dtype=torch.int8, device=DEV)
    se = scal()
    iq.iq_ce_grad(dev(z), dscal(1.0), dev(lab), E, se)
    ref, sref, _ = O.ce_grad(z, 1.0, lab)
    assert not host(E).any() and host(se)[0] == sref
    # logits far apart: exp underflows to 0 for every class but the max
    z = np.full((1, 2, 2, 4), -127, np.int8)
    z[..., 1] = 127
    lab = np.array([[[0, 1], [1, 3]]], np.uint8)
    E2 = torch.empty((1, 2, 2, 4), dtype=torch.int8, device=DEV)
    iq.iq_ce_grad(dev(z), dscal(2.0), dev(lab), E2, se)
    ref, sref, _ = O.ce_grad(z, 2.0, lab)
    assert np.array_equal(host(E2), ref) and host(se)[0] == sref


# ---------------------------------------------------------------- BN parameter update

def test_bn_update_matches_oracle():
    g = np.random.default_rng(20)
    c = 300
    gm = g.integers(-(2 ** 23) + 1, 2 ** 23, size=c).astype(np.int32)
    bm = g.integers(-(2 ** 23) + 1, 2 ** 23, size=c).astype(np.int32)
    dgam = g.integers(-(2 ** 35), 2 ** 35, size=c).astype(np.int64)
    dbet = g.integers(-(2 ** 20), 2 ** 20, size=c).astype(np.int64)
    s_e, s_x = 0.0123, 2.0 ** -15 * 1.7
    bn_scales = np.zeros(8, np.float64)
    bn_scales[0] = s_x
    dgm, dbm = dev(gm), dev(bm)
    dg, db = torch.empty(c, dtype=torch.int32, device=DEV), torch.empty(c, dtype=torch.int32, device=DEV)
    seed, layer, step, lr = 5, 17, 3, 8
    iq.iq_bn_update(dgm, dbm, dg, db, dev(dgam), dev(dbet), dscal(s_e), dev(bn_scales), lr, seed,
                    layer, step)
    qg, sg = O.rq_int(dgam, s_e * s_x, 8, 1, seed, layer, step, tag=1)
    qb, sb = O.rq_int(dbet, s_e, 8, 1, seed, layer, step, tag=2)
    rgm, rg = O.update(gm, qg, sg, lr, x2=True)
    rbm, rb = O.update(bm, qb, sb, lr, x2=True)
    assert np.array_equal(host(dgm), rgm) and np.array_equal(host(dg), rg)
    assert np.array_equal(host(dbm), rbm) and np.array_equal(host(db), rb)
