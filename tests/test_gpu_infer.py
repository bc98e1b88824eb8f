"""Inference passes of both networks on the GPU against the oracle network.

The inference configurations run batch 8 with no backward buffers (train=False: no fp16
carrier copies kept for weight gradients, L1BN on the inference batch's statistics).  A
reduced width keeps the oracle in seconds; both sides start from the same fp32 weights
and gamma / beta codes and read identical image bytes, so every activation, X code, join,
the ASPP concatenation and the logits must agree bit for bit, over two batches in a row
(the second one reuses every buffer the first one wrote)."""
import numpy as np
import pytest
import torch

from oracle.deeplab import OracleDeepLab
from oracle.fcn import OracleFcn
from paper_2011_14504_gb300 import synthetic as S
from paper_2011_14504_gb300.deeplab import DeepLabV3R50
from paper_2011_14504_gb300.fcn import FcnVgg16

pytestmark = pytest.mark.gpu


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


@pytest.mark.parametrize("n,size,width,blocks", [(8, 33, 0.0625, (3, 4, 6, 3)),
                                                 (8, 65, 0.0625, (1, 1, 2, 1))])
def test_deeplab_inference_matches_oracle(n, size, width, blocks):
    seed = 6
    g = S.rng(300 + size)
    net = DeepLabV3R50(n, size, size, classes=21, width=width, seed=seed, train=False,
                       blocks=blocks)
    sp = S.deeplabv3_r50_spec(21, width, blocks)
    w, gm, bm = S.deeplabv3_r50_init(seed, sp)
    ora = OracleDeepLab(sp, w, gm, bm, seed=seed)
    for batch in range(2):
        img = S.images_u8(g, n, size, size)
        net.forward(torch.from_numpy(img).cuda())
        tr = ora.forward(img)
        for name, L in net.layers.items():
            rec = tr[name]
            assert np.array_equal(host(L.a), rec["a"]), (batch, name)
            assert host(L.s_a)[0] == rec["s_a"], (batch, name)
            if L.spec.bn:
                assert np.array_equal(host(L.X), rec["X"]), (batch, name)
        for blk in net.blocks:
            ref, s_ref = tr[blk["spec"].name]["out"]
            assert np.array_equal(host(blk["out"]), ref), (batch, blk["spec"].name)
            assert host(blk["s_out"])[0] == s_ref
        assert np.array_equal(host(net.cat), tr["cat"][0]) and host(net.s_cat)[0] == tr["cat"][1]
        assert np.array_equal(host(net.z), tr["z"][0]) and host(net.s_z)[0] == tr["z"][1]


@pytest.mark.parametrize("classes,width,h", [(150, 0.0625, 64), (21, 0.125, 96)])
def test_fcn_inference_matches_oracle(classes, width, h):
    n, seed = 8, 7
    g = S.rng(400 + classes)
    net = FcnVgg16(n, h, h, classes=classes, width=width, seed=seed, train=False)
    chans = S.fcn_vgg16_channels(classes, width)
    wts, up = S.fcn_vgg16_weights(seed, classes, width)
    ora = OracleFcn(chans, wts, up, classes, seed=seed)
    for batch in range(2):
        img = S.images_u8(g, n, h, h)
        net.forward(torch.from_numpy(img).cuda())
        tr = ora.forward(img)
        convs = [it for it in tr["layers"] if it[0] == "conv"]
        for L, it in zip(net.convs, convs):
            _, li, cv, x, s_x, wq, acc, a, s_a, relu = it
            assert np.array_equal(host(L.a), a), (batch, L.name)
            assert host(L.s_a)[0] == s_a, (batch, L.name)
        _, _, _, _, _, z, s_z = tr["up"]
        assert np.array_equal(host(net.z), z) and host(net.s_z)[0] == s_z
