"""Parity at the benchmark's full sizes.

Every class of convolution geometry in the two training steps (batch 16, 3 x 513 x 513
DeepLabv3-ResNet50 and 3 x 512 x 512 FCN-VGG16, full width) is called through the C ABI
exactly as the networks call it -- the same optional carrier buffers, so the same kernels
and tilings as the timed step -- on seeded synthetic inputs with the workloads' value
structure, and compared with the oracle:

  * forward (integer L1BN + ReLU + Q_A, or SQ of ReLU), Sec. 3.2;
  * the L1BN / ReLU backward, Eq. (EQ) and the derivative of Eqs. (BN4), (BN5);
  * the data gradient with Q_E = SQ(., 8), Eq. (EQ);
  * the weight gradient with the stochastic rounding of Eqs. (SQ), (SR), (GQ1) / (GQ2).

Where the oracle's loops finish in seconds the whole tensor is compared element by
element.  Otherwise the output is compared at positions the oracle evaluates one at a
time: a seeded random sample plus every element at the top code +-127.  The largest
magnitude of the tensor is among the latter, so the oracle's maximum over them fixes the
output scale, which is compared exactly, and the codes of the sample follow from it.

The joins, pools and loss heads at their full sizes are compared in full.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle as O
from paper_2011_14504_gb300 import iq
from paper_2011_14504_gb300 import synthetic as S
from paper_2011_14504_gb300.work import conv_macs, out_size

pytestmark = pytest.mark.gpu

DEV = "cuda"
N = 16
# the oracle's full loops run where one pass is at most this many multiply-accumulates
FULL_MACS = 160e9
SAMPLE = 3000


def dt(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def sc(v=0.0):
    return torch.tensor([v], dtype=torch.float64, device=DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


# ------------------------------------------------------------------ geometry of the steps

def deeplab_geometry():
    """name -> (ConvSpec, input height = width) of every DeepLab conv at 513 x 513."""
    sp = S.deeplabv3_r50_spec(21)
    out = {"stem": (sp.stem, 513)}
    sz = out_size(513, 7, 2, 3, 1)
    sz = out_size(sz, 3, 2, 1, 1)                   # the stem's max pool
    for b in sp.blocks:
        s1 = sz
        for cv in (b.conv1, b.conv2, b.conv3):
            out[cv.name] = (cv, s1)
            s1 = out_size(s1, cv.r, cv.stride, cv.pad, cv.dil)
        if b.down:
            out[b.down.name] = (b.down, sz)
        sz = s1
    for cv in list(sp.aspp) + [sp.project, sp.head, sp.cls]:
        out[cv.name] = (cv, sz)
    out[sp.pool_conv.name] = (sp.pool_conv, 1)
    return out


def fcn_geometry():
    """name -> (cin, cout, r, pad, relu, input size) of every FCN conv at 512 x 512."""
    out, hh = {}, 512
    for name, cin, cout, r, pad, relu in S.fcn_vgg16_channels(150):
        if name == "pool":
            hh //= 2
            continue
        out[name] = (cin, cout, r, pad, relu, hh)
    return out


# ------------------------------------------------------------------ inputs

def act_codes(g, shape):
    """Codes of a ReLU output after Q_A: about half zeros, the rest uniform, one 127."""
    v = np.maximum(g.integers(-127, 128, size=shape, dtype=np.int16), 0).astype(np.int8)
    v.flat[int(g.integers(v.size))] = 127
    return v


def err_codes(g, shape):
    """Error codes after Q_E: uniform on [-127, 127], one element at 127."""
    v = S.int8_uniform(g, shape)
    v.flat[int(g.integers(v.size))] = 127
    return v


def image_codes(g, n, h):
    img = S.images_u8(g, n, h, h)
    codes, s = O.quantize_image_u8(img, 4)
    return codes, s


def he_codes(g, k, r, c, fan_in):
    """W_q = UQ(UQ(W, 24), 8) of He-initialised weights (Eqs. (WQ0), (WQ1))."""
    return O.requant_master(O.uq(S.he_weights(g, (k, r, r, c), fan_in), 24)).astype(np.int8)


# ------------------------------------------------------------------ sampled comparison

def check_sq(got, s_got, values_at, s_in, relu, g, what):
    """Q = SQ(., 8) (of ReLU when relu) of a tensor the oracle evaluates one element at a
    time (values_at(flat indices) -> int64): the top-code elements fix M, a random sample
    and those elements are compared code by code, and the scale exactly."""
    flat = got.ravel().astype(np.int32)
    top = np.flatnonzero(flat == 127) if relu else np.flatnonzero(np.abs(flat) == 127)
    assert 0 < top.size <= 60000, (what, top.size)
    idx = np.unique(np.concatenate([top, g.integers(0, flat.size, SAMPLE)]))
    v = values_at(idx)
    at_top = np.isin(idx, top)
    M = int((np.maximum(v, 0) if relu else np.abs(v))[at_top].max())
    codes, s = O.sq_at(v, M, s_in, 8, relu)
    bad = np.flatnonzero(codes != flat[idx])
    assert bad.size == 0, (what, idx[bad[:5]], codes[bad[:5]], flat[idx[bad[:5]]])
    assert s_got == s, what


def check_rq(got, s_got, values_at, s_in, gq_mode, seed, layer, step, g, what):
    """G_q = RQ(G / Scale(G), 8) of a gradient the oracle evaluates one element at a time."""
    flat = got.ravel().astype(np.int32)
    top = np.flatnonzero(np.abs(flat) == 127)
    assert 0 < top.size <= 60000, (what, top.size)
    idx = np.unique(np.concatenate([top, g.integers(0, flat.size, SAMPLE)]))
    v = values_at(idx)
    M = int(np.abs(v[np.isin(idx, top)]).max())
    codes, s = O.rq_at(v, idx, M, s_in, 8, gq_mode, seed, layer, step)
    bad = np.flatnonzero(codes != flat[idx])
    assert bad.size == 0, (what, idx[bad[:5]], codes[bad[:5]], flat[idx[bad[:5]]])
    assert s_got == s, what


# ------------------------------------------------------------------ one layer, as the nets run it

class LayerRun:
    """One conv layer's forward, backward and weight gradient through the C ABI with the
    networks' arguments: fp16 input carrier when the input channels are a multiple of 64,
    error carrier when the output channels are."""

    def __init__(self, cv: O.Conv, bn: bool, relu: bool, x, s_x, wq, gamma=None, beta=None):
        self.cv, self.bn, self.relu = cv, bn, relu
        self.d = iq.conv_desc(cv.n, cv.h, cv.w, cv.c, cv.k, cv.r, cv.s, cv.stride, cv.pad,
                              cv.dil)
        p, q = iq.iq_conv_out_size(self.d)
        self.out = (cv.n, p, q, cv.k)
        self.x, self.s_x, self.wq = dt(x), sc(s_x), dt(wq)
        self.x16 = (torch.empty(self.x.numel(), dtype=torch.float16, device=DEV)
                    if cv.c % 64 == 0 and self.x.numel() % 16 == 0 else None)
        self.e16 = (torch.empty(max(16, int(np.prod(self.out))), dtype=torch.float16, device=DEV)
                    if cv.k % 64 == 0 else None)
        ws = iq.iq_conv_fwd_workspace_size(self.d, bn)
        ws = max(ws, iq.iq_conv_dgrad_workspace_size(self.d), iq.iq_conv_wgrad_workspace_size(self.d))
        if bn:
            ws = max(ws, iq.iq_bn_int_workspace_size(int(np.prod(self.out[:3])), cv.k))
            self.gamma, self.beta = dt(gamma.astype(np.int32)), dt(beta.astype(np.int32))
        self.ws = torch.empty(ws + 4096, dtype=torch.uint8, device=DEV)

    def forward(self):
        self.a = torch.empty(self.out, dtype=torch.int8, device=DEV)
        self.s_a = sc()
        if self.bn:
            self.X = torch.empty(self.out, dtype=torch.int16, device=DEV)
            self.codes = torch.empty(2 * self.cv.k, dtype=torch.int32, device=DEV)
            self.scales = torch.zeros(iq.IQ_BN_SCALES, dtype=torch.float64, device=DEV)
            iq.iq_conv_fwd(self.d, self.x, self.s_x, self.wq, self.a, self.s_a, self.gamma,
                           self.beta, use_bn=True, relu=True, xhat=self.X, bn_codes=self.codes,
                           bn_scales=self.scales, x_f16=self.x16, ws=self.ws)
        else:
            iq.iq_conv_fwd(self.d, self.x, self.s_x, self.wq, self.a, self.s_a, relu=self.relu,
                           x_f16=self.x16, ws=self.ws)

    def bn_backward(self, e_a, s_ea, a=None, X=None, codes=None, scales=None):
        c = self.cv.k
        self.e = torch.empty(self.out, dtype=torch.int8, device=DEV)
        self.s_e = sc()
        self.dgamma = torch.empty(c, dtype=torch.int64, device=DEV)
        self.dbeta = torch.empty(c, dtype=torch.int64, device=DEV)
        iq.iq_bn_int_bwd(dt(e_a), sc(s_ea), self.a if a is None else a,
                         self.X if X is None else X, self.gamma,
                         self.codes if codes is None else codes,
                         self.scales if scales is None else scales, self.e, self.s_e,
                         self.dgamma, self.dbeta, k_e2=16, ws=self.ws)

    def dgrad(self, e, s_e):
        cv = self.cv
        self.ex = torch.empty((cv.n, cv.h, cv.w, cv.c), dtype=torch.int8, device=DEV)
        self.s_ex = sc()
        iq.iq_conv_dgrad(self.d, e, s_e, self.wq, self.ex, self.s_ex, e_f16=self.e16, ws=self.ws)

    def wgrad(self, e, s_e, gq_mode, seed, layer, step, with_dx):
        self.g = torch.empty_like(self.wq)
        self.s_g = sc()
        iq.iq_conv_wgrad(self.d, e, s_e, self.x, self.s_x, self.g, self.s_g, gq_mode=gq_mode,
                         seed=seed, layer=layer, step=step,
                         e_f16=self.e16 if with_dx else None, x_f16=self.x16, ws=self.ws)


def _conv_check(run: LayerRun, x, wq, e_pre, s_e_pre, g, name, full_fwd, full_dgrad, has_dx,
                gq_mode, layer, e_a=None, s_ea=None):
    """Forward, backward and weight gradient of one layer against the oracle."""
    cv = run.cv
    s_acc = run.s_x.item() * 2.0 ** -7
    run.forward()
    # ---- forward
    if full_fwd:
        acc = O.conv_fwd(cv, x, wq)
        if run.bn:
            r = O.bn_fwd(acc.reshape(-1, cv.k), s_acc, host(run.gamma), host(run.beta))
            assert np.array_equal(host(run.a).reshape(-1, cv.k), r.A), name
            assert np.array_equal(host(run.X).reshape(-1, cv.k), r.X), name
            assert run.s_a.item() == r.s_a, name
            assert np.array_equal(host(run.codes), np.concatenate([r.c_mu, r.c_sigma])), name
            assert host(run.scales)[iq.IQ_BN_S_XHAT] == r.s_xhat, name
        else:
            want, s_want = O.sq_int(acc, s_acc, 8, run.relu)
            assert np.array_equal(host(run.a).astype(np.int32), want), name
            assert run.s_a.item() == s_want, name
    else:
        assert not run.bn
        check_sq(host(run.a), run.s_a.item(), lambda i: O.conv_fwd_at(cv, x, wq, i), s_acc,
                 run.relu, g, name + " forward")
    # ---- the error at the conv output
    if run.bn:
        assert full_fwd
        run.bn_backward(e_a, s_ea)
        E, s_E, dg, db = O.bn_bwd(e_a, s_ea, r.A, r.X, r.s_xhat, host(run.gamma), r.c_sigma,
                                  k_e2=16)
        assert np.array_equal(host(run.e), E), name
        assert run.s_e.item() == s_E, name
        assert np.array_equal(host(run.dgamma), dg) and np.array_equal(host(run.dbeta), db), name
        e_np, e_dev, s_e_dev = E, run.e, run.s_e
    else:
        e_np = e_pre
        e_dev, s_e_dev = dt(e_pre), sc(s_e_pre)
    s_e = s_e_dev.item()
    # ---- data gradient
    if has_dx:
        run.dgrad(e_dev, s_e_dev)
        s_in = s_e * 2.0 ** -7
        if full_dgrad:
            want, s_want = O.sq_int(O.conv_dgrad(cv, e_np, wq), s_in, 8)
            assert np.array_equal(host(run.ex).astype(np.int32), want), name
            assert run.s_ex.item() == s_want, name
        else:
            check_sq(host(run.ex), run.s_ex.item(), lambda i: O.conv_dgrad_at(cv, e_np, wq, i),
                     s_in, False, g, name + " data gradient")
    # ---- weight gradient
    seed, step = 11, 3
    run.wgrad(e_dev, s_e_dev, gq_mode, seed, layer, step, has_dx)
    check_rq(host(run.g), run.s_g.item(), lambda i: O.conv_wgrad_at(cv, e_np, x, i),
             s_e * run.s_x.item(), gq_mode, seed, layer, step, g, name + " weight gradient")


DEEPLAB_LAYERS = ["stem", "layer1.0.conv1", "layer1.0.conv2", "layer1.0.conv3", "layer1.0.down",
                  "layer2.0.conv1", "layer2.0.conv2", "layer2.0.down", "layer2.1.conv3",
                  "layer3.0.conv1", "layer3.1.conv2", "layer3.0.down", "layer4.0.conv1",
                  "layer4.1.conv2", "layer4.2.conv3", "aspp.b0", "aspp.b1", "aspp.b3",
                  "aspp.pool", "aspp.project", "head", "cls"]


@pytest.mark.parametrize("name", DEEPLAB_LAYERS)
def test_deeplab_layer_full_size(name):
    geo = deeplab_geometry()
    spec, hw = geo[name]
    lid = list(geo).index(name)
    g = S.rng(5000 + lid)
    cv = O.Conv(N, hw, hw, spec.cin, spec.cout, spec.r, spec.r, spec.stride, spec.pad, spec.dil)
    if name == "stem":
        x, s_x = image_codes(g, N, hw)
    else:
        x, s_x = act_codes(g, (N, hw, hw, spec.cin)), 0.0123
    fan_in = (3 if spec.cin == 4 else spec.cin) * spec.r * spec.r
    wq = he_codes(g, spec.cout, spec.r, spec.cin, fan_in)
    if spec.cin == 4:
        wq[..., 3] = 0
    macs = conv_macs(N, hw, hw, spec.cin, spec.cout, spec.r, spec.stride, spec.pad, spec.dil)[0]
    p, q = cv.pq
    e_a = err_codes(g, (N, p, q, spec.cout))
    s_ea = 3.0e-6
    if spec.bn:
        gam, bet = S.bn_gamma_beta_codes(g, spec.cout)
        run = LayerRun(cv, True, True, x, s_x, wq, gam, bet)
    else:
        run = LayerRun(cv, False, False, x, s_x, wq)
    _conv_check(run, x, wq, e_a, s_ea, g, name, full_fwd=spec.bn or macs <= FULL_MACS,
                full_dgrad=macs <= FULL_MACS, has_dx=name != "stem", gq_mode=1, layer=lid,
                e_a=e_a, s_ea=s_ea)


FCN_LAYERS = ["conv1", "conv2", "conv3", "conv5", "conv6", "conv8", "conv11", "conv13", "fc6",
              "fc7", "score"]


@pytest.mark.parametrize("name", FCN_LAYERS)
def test_fcn_layer_full_size(name):
    geo = fcn_geometry()
    cin, cout, r, pad, relu, hw = geo[name]
    lid = list(geo).index(name)
    g = S.rng(6000 + lid)
    cv = O.Conv(N, hw, hw, cin, cout, r, r, 1, pad, 1)
    if cin == 4:
        x, s_x = image_codes(g, N, hw)
    else:
        x, s_x = act_codes(g, (N, hw, hw, cin)), 0.0087
    wq = he_codes(g, cout, r, cin, (3 if cin == 4 else cin) * r * r)
    if cin == 4:
        wq[..., 3] = 0
    macs = conv_macs(N, hw, hw, cin, cout, r, 1, pad, 1)[0]
    # the error after the ReLU mask of this layer's own output is what reaches the convs;
    # a uniform error stands in for it (the mask is a separate call, tested elsewhere)
    e = err_codes(g, (N, hw, hw, cout))
    run = LayerRun(cv, False, relu, x, s_x, wq)
    _conv_check(run, x, wq, e, 1.7e-5, g, name, full_fwd=macs <= FULL_MACS,
                full_dgrad=macs <= FULL_MACS, has_dx=cin != 4, gq_mode=2, layer=lid)


# ------------------------------------------------------------------ joins, pools and heads

def test_deeplab_joins_full_size():
    """Residual add of a stage-1 block (129 x 129 x 256: BN affine of the X codes plus the
    projected shortcut), the ASPP concatenation with the broadcast pooled branch
    (65 x 65 x 1280), and the five-operand error sum at the ASPP input (65 x 65 x 2048)."""
    g = S.rng(7001)
    # residual add with ReLU
    hw, c = 129 * 129, 256
    X3 = g.integers(-32767, 32768, size=(N, hw, c), dtype=np.int16)
    Xd = g.integers(-32767, 32768, size=(N, hw, c), dtype=np.int16)
    g3, b3 = S.bn_gamma_beta_codes(g, c)
    gd, bd = S.bn_gamma_beta_codes(g, c)
    s3, sd = 2.5e-5, 3.1e-5
    terms_o = [O.CombineTerm(X3, s3, gamma=g3, beta=b3), O.CombineTerm(Xd, sd, gamma=gd, beta=bd)]
    want, s_want = O.combine(terms_o, N, hw, c, relu=True)
    tX3, tXd, sc3, scd = dt(X3), dt(Xd), sc(s3), sc(sd)
    tg3, tb3, tgd, tbd = (dt(v.astype(np.int32)) for v in (g3, b3, gd, bd))
    terms = [iq.term(tX3, sc3, gamma=tg3, beta=tb3), iq.term(tXd, scd, gamma=tgd, beta=tbd)]
    out = torch.empty((N, hw, c), dtype=torch.int8, device=DEV)
    s_out = sc()
    iq.iq_combine(terms, N, hw, c, out, s_out, relu=True)
    assert np.array_equal(host(out).ravel(), want) and s_out.item() == s_want
    # ASPP concatenation
    hw, a = 65 * 65, 256
    br = [act_codes(g, (N, hw, a)) for _ in range(4)]
    pooled = act_codes(g, (N, a))
    scales = [0.011, 0.013, 0.017, 0.019, 0.023]
    terms_o = [O.CombineTerm(b, s, k * a) for k, (b, s) in enumerate(zip(br, scales))]
    terms_o.append(O.CombineTerm(pooled, scales[4], 4 * a, bcast=True))
    want, s_want = O.combine(terms_o, N, hw, 5 * a, concat=True)
    keep = [dt(b) for b in br] + [dt(pooled)]
    ss = [sc(s) for s in scales]
    terms = [iq.term(keep[k], ss[k], k * a) for k in range(4)]
    terms.append(iq.term(keep[4], ss[4], 4 * a, bcast=True))
    out = torch.empty((N, hw, 5 * a), dtype=torch.int8, device=DEV)
    iq.iq_combine(terms, N, hw, 5 * a, out, s_out, concat=True)
    assert np.array_equal(host(out).ravel(), want) and s_out.item() == s_want
    # error sum at the ASPP input: four branch errors and the broadcast pooled error
    c = 2048
    errs = [err_codes(g, (N, hw, c)) for _ in range(4)]
    ep = err_codes(g, (N, c))
    scales = [1.1e-6, 0.9e-6, 1.3e-6, 0.7e-6, 2.0e-9]
    terms_o = [O.CombineTerm(e, s) for e, s in zip(errs, scales[:4])]
    terms_o.append(O.CombineTerm(ep, scales[4], bcast=True))
    want, s_want = O.combine(terms_o, N, hw, c)
    keep = [dt(e) for e in errs] + [dt(ep)]
    ss = [sc(s) for s in scales]
    terms = [iq.term(keep[k], ss[k]) for k in range(4)] + [iq.term(keep[4], ss[4], bcast=True)]
    out = torch.empty((N, hw, c), dtype=torch.int8, device=DEV)
    iq.iq_combine(terms, N, hw, c, out, s_out)
    assert np.array_equal(host(out).ravel(), want) and s_out.item() == s_want


def test_deeplab_stem_pool_and_head_full_size():
    """The stem's 3 x 3 stride-2 max pool (257 -> 129, 64 channels) forward and backward,
    the x8 bilinear upsampling of the logits (65 -> 513, 21 classes) forward and backward,
    and the cross-entropy gradient over 16 x 513 x 513 pixels with 5% ignored labels."""
    g = S.rng(7002)
    x = act_codes(g, (N, 257, 257, 64))
    y_want, arg_want = O.maxpool_fwd(x, 3, 2, 1)
    tx = dt(x)
    y = torch.empty(y_want.shape, dtype=torch.int8, device=DEV)
    arg = torch.empty(y_want.shape, dtype=torch.uint8, device=DEV)
    iq.iq_maxpool_fwd(tx, 3, 2, 1, y, arg)
    assert np.array_equal(host(y), y_want) and np.array_equal(host(arg), arg_want)
    e = err_codes(g, y_want.shape)
    ex_acc = O.maxpool_bwd(e, arg_want, x.shape, 3, 2, 1)
    want, s_want = O.sq_int(ex_acc, 2.0e-6, 8)
    ex = torch.empty(x.shape, dtype=torch.int8, device=DEV)
    s_ex = sc()
    iq.iq_maxpool_bwd(dt(e), sc(2.0e-6), arg, x.shape, 3, 2, 1, ex, s_ex)
    assert np.array_equal(host(ex).astype(np.int32), want) and s_ex.item() == s_want
    # x8 bilinear head
    logits = err_codes(g, (N, 65, 65, 21))
    z_want, s_z_want, _ = O.bilinear_up(logits, 0.04, 8)
    z = torch.empty(z_want.shape, dtype=torch.int8, device=DEV)
    s_z = sc()
    iq.iq_bilinear_up_fwd(dt(logits), sc(0.04), 8, z, s_z)
    assert np.array_equal(host(z), z_want) and s_z.item() == s_z_want
    E = err_codes(g, z_want.shape)
    eb_want, s_eb_want, _ = O.bilinear_up_bwd(E, 1.0e-7, 8, logits.shape)
    eb = torch.empty(logits.shape, dtype=torch.int8, device=DEV)
    s_eb = sc()
    iq.iq_bilinear_up_bwd(dt(E), sc(1.0e-7), 8, logits.shape, eb, s_eb)
    assert np.array_equal(host(eb), eb_want) and s_eb.item() == s_eb_want
    # cross-entropy gradient on the logits
    lab = S.labels_uniform_ignore(g, N, 513, 513, 21)
    Ew, s_Ew, nv_w = O.ce_grad(z_want, s_z_want, lab)
    Eg = torch.empty(z_want.shape, dtype=torch.int8, device=DEV)
    s_Eg = sc()
    nv = torch.zeros(1, dtype=torch.int64, device=DEV)
    iq.iq_ce_grad(z, s_z, dt(lab), Eg, s_Eg, n_valid=nv)
    assert np.array_equal(host(Eg), Ew) and s_Eg.item() == s_Ew and int(host(nv)[0]) == nv_w


def test_fcn_head_full_size():
    """The FCN decoder (per-class transposed conv k64 s32 p16, 16 x 16 -> 512 x 512, 150
    classes) forward, data gradient and weight gradient, the MSE gradient over the 629 M
    logits with Voronoi labels, and a 2 x 2 max pool of conv1_2 (512 -> 256, 64 channels)."""
    g = S.rng(7003)
    c, R, st, pd = 150, 64, 32, 16
    score = err_codes(g, (N, 16, 16, c))
    wup = O.requant_master(O.uq(S.bilinear_filters(c, R), 24)).astype(np.int8)
    s_score = 0.05
    tsc, tw = dt(score), dt(wup)
    # the oracle: a grouped stride-32 conv's adjoint is the transposed conv
    cvu = O.Conv(N, 512, 512, c, c, R, R, st, pd, 1, c)
    zacc = O.conv_dgrad(cvu, score, wup.reshape(c, R, R, 1))
    z_want, s_z_want = O.sq_int(zacc, s_score * 2.0 ** -7, 8)
    z = torch.empty((N, 512, 512, c), dtype=torch.int8, device=DEV)
    s_z = sc()
    iq.iq_upsample_fwd(tsc, sc(s_score), tw, R, st, pd, z, s_z)
    assert np.array_equal(host(z).astype(np.int32), z_want) and s_z.item() == s_z_want
    lab = S.labels_voronoi(g, N, 512, 512, c, sites=64)
    E_want, s_E_want = O.mse_grad(z_want.astype(np.int8), s_z_want, lab)
    E = torch.empty_like(z)
    s_E = sc()
    iq.iq_mse_grad(z, s_z, dt(lab), E, s_E)
    assert np.array_equal(host(E), E_want) and s_E.item() == s_E_want
    ex_want, s_ex_want = O.sq_int(O.conv_fwd(cvu, E_want, wup.reshape(c, R, R, 1)),
                                  s_E_want * 2.0 ** -7, 8)
    ex = torch.empty(score.shape, dtype=torch.int8, device=DEV)
    s_ex = sc()
    iq.iq_upsample_bwd(E, s_E, tw, score.shape, R, st, pd, ex, s_ex)
    assert np.array_equal(host(ex).astype(np.int32), ex_want) and s_ex.item() == s_ex_want
    gw = O.conv_wgrad(cvu, score, E_want).reshape(c, R, R)
    gq_want, s_g_want = O.rq_int(gw, s_score * s_E_want, 8, 2, 5, 15, 2)
    gq = torch.empty_like(tw)
    s_g = sc()
    iq.iq_upsample_wgrad(tsc, sc(s_score), E, s_E, R, st, pd, gq, s_g, gq_mode=2, seed=5, layer=15,
                         step=2)
    assert np.array_equal(host(gq).astype(np.int32), gq_want) and s_g.item() == s_g_want
    # 2 x 2 max pool after conv1_2
    x = act_codes(g, (N, 512, 512, 64))
    y_want, arg_want = O.maxpool_fwd(x, 2, 2, 0)
    y = torch.empty(y_want.shape, dtype=torch.int8, device=DEV)
    arg = torch.empty(y_want.shape, dtype=torch.uint8, device=DEV)
    iq.iq_maxpool_fwd(dt(x), 2, 2, 0, y, arg)
    assert np.array_equal(host(y), y_want) and np.array_equal(host(arg), arg_want)
