"""Pins of the oracle's network composition (oracle/fcn.py) by exact symmetries.

The layer functions are pinned one by one elsewhere; these tests fix how the FCN-VGG16
step composes them, with properties that hold for the correct dataflow and fail for a
dropped layer, a wrong index, a transposed axis or a pool / decoder misplacement:

- Horizontal flip.  Take every convolution kernel and the decoder filters mirror-symmetric
  (w[.., s, ..] = w[.., S-1-s, ..]).  Then each step commutes with flipping the image
  width:
  - the image quantizer and SQ_8 use global maxima;
  - the convolutions pad symmetrically;
  - 2 x 2 max pools on even widths map windows onto windows;
  - the 32x decoder (kernel 64, stride 32, padding 16) maps output column y to
    W - 1 - y;
  - the MSE error is elementwise.
  So the flipped image and labels give the flipped forward trace and error. The backward
  gives the mirrored raw weight gradients and the flipped errors down to the last pool
  (the pools' argmax ties and the stochastic rounding of G_q, indexed by element, are not
  symmetric and are not compared).
- Batch order.  Every scale is a maximum over the whole batch and every gradient a sum over
  it, so permuting three images cyclically permutes every activation and error and leaves
  the raw gradients unchanged.
"""
import numpy as np

from oracle.fcn import OracleFcn
from paper_2011_14504_gb300 import synthetic as S

CLASSES, WIDTH, SEED = 21, 0.125, 5


def _mirrored_weights():
    wts, up = S.fcn_vgg16_weights(SEED, CLASSES, WIDTH)
    wts = [0.5 * (w + w[:, :, ::-1, :]) for w in wts]        # KRSC: mirror the S axis
    up = 0.5 * (up + up[..., ::-1])
    return wts, up


def _inputs(n=2, h=64, w=64):
    g = S.rng(41)
    return S.images_u8(g, n, h, w), S.labels_voronoi(g, n, h, w, CLASSES, sites=6)


def _net(wts, up):
    return OracleFcn(S.fcn_vgg16_channels(CLASSES, WIDTH), wts, up, CLASSES, seed=SEED,
                     lr_log2=6)


def _fw(a):           # flip the width axis of an NHWC / NHW array
    return a[:, :, ::-1, ...]


def test_fcn_step_commutes_with_a_horizontal_flip():
    wts, up = _mirrored_weights()
    img, lab = _inputs()
    a, b = _net(wts, up), _net(wts, up)
    ta = a.forward(img)
    tb = b.forward(np.ascontiguousarray(_fw(img)))
    assert np.array_equal(tb["img"][0], _fw(ta["img"][0])) and tb["img"][1] == ta["img"][1]
    for la, lb in zip(ta["layers"], tb["layers"]):
        if la[0] == "pool":
            assert np.array_equal(lb[3], _fw(la[3]))
            continue
        assert np.array_equal(lb[6], _fw(la[6])), la[2]          # int32 accumulators
        assert np.array_equal(lb[7], _fw(la[7])) and lb[8] == la[8]
    za, zb = ta["up"], tb["up"]
    assert np.array_equal(zb[4], _fw(za[4])) and np.array_equal(zb[5], _fw(za[5]))
    assert zb[6] == za[6]
    oa = a.backward_update(ta, lab)
    ob = b.backward_update(tb, np.ascontiguousarray(_fw(lab)))
    assert np.array_equal(ob["E"][0], _fw(oa["E"][0])) and ob["E"][1] == oa["E"][1]
    assert np.array_equal(ob["e_score"][0], _fw(oa["e_score"][0]))
    assert np.array_equal(ob["up_g"][0], oa["up_g"][0][..., ::-1])  # decoder kernel mirrored
    # layers after the last pool: raw gradients mirrored, errors flipped
    chans = S.fcn_vgg16_channels(CLASSES, WIDTH)
    last_pool = max(i for i, c in enumerate(chans) if c[0] == "pool")
    tail = [sum(1 for c in chans[:i] if c[0] != "pool") for i in range(last_pool + 1, len(chans))]
    assert tail
    for li in tail:
        assert np.array_equal(ob["grads"][li][0], oa["grads"][li][0][:, :, ::-1, :]), li
        if li in oa.get("ex", {}):
            assert np.array_equal(ob["ex"][li][0], _fw(oa["ex"][li][0])), li
            assert ob["ex"][li][1] == oa["ex"][li][1]


def test_fcn_step_is_equivariant_to_the_batch_order():
    wts, up = S.fcn_vgg16_weights(SEED, CLASSES, WIDTH)
    img, lab = _inputs(n=3)
    swap = [1, 2, 0]        # a 3-cycle: no reversal or swap of the batch commutes with it
    a, b = _net(wts, up), _net(wts, up)
    ta = a.forward(img)
    tb = b.forward(np.ascontiguousarray(img[swap]))
    for la, lb in zip(ta["layers"], tb["layers"]):
        if la[0] == "conv":
            assert np.array_equal(lb[7], la[7][swap]) and lb[8] == la[8], la[2]
    assert np.array_equal(tb["up"][5], ta["up"][5][swap]) and tb["up"][6] == ta["up"][6]
    oa = a.backward_update(ta, lab)
    ob = b.backward_update(tb, np.ascontiguousarray(lab[swap]))
    assert np.array_equal(ob["E"][0], oa["E"][0][swap])
    assert np.array_equal(ob["up_g"][0], oa["up_g"][0])
    for li, (G, _, _) in oa["grads"].items():
        assert np.array_equal(ob["grads"][li][0], G), li
    for li, (ex, s) in oa.get("ex", {}).items():
        assert np.array_equal(ob["ex"][li][0], ex[swap]) and ob["ex"][li][1] == s, li


# ---------------------------------------------------------------- FCN8s decoder
# The x2 (kernel 4, stride 2, padding 1) and x8 (kernel 16, stride 8, padding 4) transposed
# convolutions map input column j to output columns 2j - 1 + t / 8j - 4 + t, so under a flip
# tap t becomes 3 - t / 15 - t: with mirror-symmetric filters they commute with the flip, as
# do the 1x1 score convolutions on the pools and the real-valued sums.

def _net8(wts, up, skips):
    return OracleFcn(S.fcn_vgg16_channels(CLASSES, WIDTH), wts, up, CLASSES, seed=SEED,
                     lr_log2=6, skips=skips)


def _mirrored_skips():
    w4, w3, up2, up8 = S.fcn8s_skip_weights(SEED, CLASSES, WIDTH)
    return w4, w3, 0.5 * (up2 + up2[..., ::-1]), 0.5 * (up8 + up8[..., ::-1])


def test_fcn8s_step_commutes_with_a_horizontal_flip():
    wts, up = _mirrored_weights()
    sk = _mirrored_skips()
    img, lab = _inputs()
    a, b = _net8(wts, up, sk), _net8(wts, up, sk)
    ta = a.forward(img)
    tb = b.forward(np.ascontiguousarray(_fw(img)))
    for key in ("up2a", "sp4", "up2b", "sp3", "up"):
        assert np.array_equal(tb[key][4], _fw(ta[key][4])), key     # int32 sums
        assert np.array_equal(tb[key][5], _fw(ta[key][5])) and tb[key][6] == ta[key][6], key
    for key in ("fuse4", "fuse3"):
        assert np.array_equal(tb[key][0], _fw(ta[key][0])) and tb[key][1] == ta[key][1], key
    oa = a.backward_update(ta, lab)
    ob = b.backward_update(tb, np.ascontiguousarray(_fw(lab)))
    assert np.array_equal(ob["E"][0], _fw(oa["E"][0]))
    for key in ("e_fuse3", "e_fuse4", "e_sp3", "e_sp4", "e_score"):
        assert np.array_equal(ob[key][0], _fw(oa[key][0])) and ob[key][1] == oa[key][1], key
    for key in ("up8_g", "up2b_g", "up2a_g"):
        assert np.array_equal(ob[key][0], oa[key][0][..., ::-1]), key    # kernels mirrored
    for key in ("sp3_g", "sp4_g"):
        assert np.array_equal(ob[key][0], oa[key][0]), key                # 1x1: sums
    # (the joined errors at the pools' outputs lie below pool5's argmax ties: not compared)


def test_fcn8s_step_is_equivariant_to_the_batch_order():
    wts, up = S.fcn_vgg16_weights(SEED, CLASSES, WIDTH)
    sk = S.fcn8s_skip_weights(SEED, CLASSES, WIDTH)
    img, lab = _inputs(n=3)
    swap = [1, 2, 0]
    a, b = _net8(wts, up, sk), _net8(wts, up, sk)
    ta = a.forward(img)
    tb = b.forward(np.ascontiguousarray(img[swap]))
    for key in ("up2a", "sp4", "up2b", "sp3", "up"):
        assert np.array_equal(tb[key][5], ta[key][5][swap]) and tb[key][6] == ta[key][6], key
    oa = a.backward_update(ta, lab)
    ob = b.backward_update(tb, np.ascontiguousarray(lab[swap]))
    for key in ("up8_g", "up2b_g", "up2a_g", "sp3_g", "sp4_g"):
        assert np.array_equal(ob[key][0], oa[key][0]), key
    for li, (G, _, _) in oa["grads"].items():
        assert np.array_equal(ob["grads"][li][0], G), li
    for k, (e, s) in oa["e_pool"].items():
        assert np.array_equal(ob["e_pool"][k][0], e[swap]) and ob["e_pool"][k][1] == s, k


# ---------------------------------------------------------------- DeepLabv3-ResNet50

def _deeplab(mirror, blocks=(1, 1, 2, 1), width=0.0625):
    from oracle.deeplab import OracleDeepLab
    sp = S.deeplabv3_r50_spec(21, width, blocks)
    w, gm, bm = S.deeplabv3_r50_init(6, sp)
    if mirror:
        w = [0.5 * (x + x[:, :, ::-1, :]) for x in w]
    return sp, (lambda: OracleDeepLab(sp, w, gm, bm, seed=6, lr_log2=6))


def _conv_records(tr):
    return {k: v for k, v in tr.items() if isinstance(v, dict) and "a" in v}


def test_deeplab_step_commutes_with_a_horizontal_flip():
    # 33 x 33: every stride-2 stage (stem, its 3 x 3 pool, stage 2) sees an odd width, so
    # output column x takes input column 2x on both sides of the flip; the dilated and ASPP
    # convolutions pad by their rates, BN statistics, the image pooling and the scales are
    # sums and maxima over the whole tensor, and the x8 bilinear maps 5 -> 33 corner to
    # corner.  The stem's pool backward (overlapping windows, argmax ties) is not compared.
    sp, mk = _deeplab(True)
    g = S.rng(43)
    img = S.images_u8(g, 1, 33, 33)
    lab = S.labels_uniform_ignore(g, 1, 33, 33, 21)
    a, b = mk(), mk()
    ta = a.forward(img)
    tb = b.forward(np.ascontiguousarray(_fw(img)))
    ra, rb = _conv_records(ta), _conv_records(tb)
    assert ra.keys() == rb.keys() and len(ra) > 10
    for name in ra:
        assert np.array_equal(rb[name]["a"], _fw(ra[name]["a"])), name
        assert rb[name]["s_a"] == ra[name]["s_a"], name
        if "X" in ra[name]:
            assert np.array_equal(rb[name]["X"], _fw(ra[name]["X"])), name
    for blk in sp.blocks:
        assert np.array_equal(tb[blk.name]["out"][0], _fw(ta[blk.name]["out"][0])), blk.name
        assert tb[blk.name]["out"][1] == ta[blk.name]["out"][1]
    assert np.array_equal(tb["cat"][0], _fw(ta["cat"][0])) and tb["cat"][1] == ta["cat"][1]
    assert np.array_equal(tb["z"][0], _fw(ta["z"][0])) and tb["z"][1] == ta["z"][1]
    oa = a.backward_update(ta, lab)
    ob = b.backward_update(tb, np.ascontiguousarray(_fw(lab)))
    assert np.array_equal(ob["E"][0], _fw(oa["E"][0])) and ob["E"][1] == oa["E"][1]
    assert np.array_equal(ob["e_cls"][0], _fw(oa["e_cls"][0]))
    for name, rec in ra.items():
        if name == sp.stem.name:
            continue
        shp = rec["a"].shape
        ea, eb = oa[name]["e"], ob[name]["e"]
        assert np.array_equal(eb[0].reshape(shp), _fw(ea[0].reshape(shp))), name
        assert eb[1] == ea[1], name
        if "ex" in oa[name]:
            xs = rec["x"].shape
            assert np.array_equal(ob[name]["ex"][0].reshape(xs),
                                  _fw(oa[name]["ex"][0].reshape(xs))), name
        if "dgb" in oa[name]:
            assert all(np.array_equal(p, q) for p, q in zip(ob[name]["dgb"], oa[name]["dgb"]))
    for blk in sp.blocks:
        assert np.array_equal(ob[blk.name][0], _fw(oa[blk.name][0])), blk.name


def test_deeplab_step_is_equivariant_to_the_batch_order():
    sp, mk = _deeplab(False)
    g = S.rng(44)
    img = S.images_u8(g, 3, 33, 33)
    lab = S.labels_uniform_ignore(g, 3, 33, 33, 21)
    cyc = [1, 2, 0]
    a, b = mk(), mk()
    ta = a.forward(img)
    tb = b.forward(np.ascontiguousarray(img[cyc]))
    for name, rec in _conv_records(ta).items():
        assert np.array_equal(tb[name]["a"], rec["a"][cyc]) and tb[name]["s_a"] == rec["s_a"], name
    assert np.array_equal(tb["z"][0], ta["z"][0][cyc]) and tb["z"][1] == ta["z"][1]
    oa = a.backward_update(ta, lab)
    ob = b.backward_update(tb, np.ascontiguousarray(lab[cyc]))
    assert np.array_equal(ob["E"][0], oa["E"][0][cyc])
    for name, rec in _conv_records(ta).items():
        shp = rec["a"].shape
        assert np.array_equal(ob[name]["e"][0].reshape(shp), oa[name]["e"][0].reshape(shp)[cyc]), name
        if "dgb" in oa[name]:
            assert all(np.array_equal(p, q) for p, q in zip(ob[name]["dgb"], oa[name]["dgb"]))
