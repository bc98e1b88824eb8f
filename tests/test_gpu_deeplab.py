"""DeepLabv3-ResNet50 training steps on the GPU against the oracle network, free-running.

A reduced-width network (the full block structure, channels x 1/8, at least 16) on
65 x 65 images (output stride 8: 9 x 9 features, logits upsampled x8 back to 65 x 65)
keeps the oracle in seconds.  Both sides start from the same fp32 weights and gamma /
beta codes and consume identical input bytes, so every intermediate -- activations, BN
codes, residual sums, the ASPP concatenation, logits, loss gradient, every layer's
errors and gradients, master weights and gamma / beta after the update -- must agree bit
for bit, step after step."""
import numpy as np
import pytest
import torch

from oracle.deeplab import OracleDeepLab
from paper_2011_14504_gb300 import synthetic as S
from paper_2011_14504_gb300.deeplab import DeepLabV3R50

pytestmark = pytest.mark.gpu


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


@pytest.mark.parametrize("n,size,width,blocks", [(2, 65, 0.125, (3, 4, 6, 3)),
                                                 (1, 33, 0.0625, (1, 1, 2, 1))])
def test_deeplab_train_steps_match_oracle(n, size, width, blocks):
    seed = 4
    g = S.rng(200 + size)
    net = DeepLabV3R50(n, size, size, classes=21, width=width, seed=seed, lr_log2=6,
                       blocks=blocks)
    sp = S.deeplabv3_r50_spec(21, width, blocks)
    w, gm, bm = S.deeplabv3_r50_init(seed, sp)
    ora = OracleDeepLab(sp, w, gm, bm, seed=seed, lr_log2=6)
    for step in range(2):
        img = S.images_u8(g, n, size, size)
        lab = S.labels_uniform_ignore(g, n, size, size, 21)
        net.train_step(torch.from_numpy(img).cuda(), torch.from_numpy(lab).cuda())
        tr = ora.forward(img)
        for name, L in net.layers.items():
            rec = tr[name]
            assert np.array_equal(host(L.a), rec["a"]), (step, name)
            assert host(L.s_a)[0] == rec["s_a"], (step, name)
            if L.spec.bn:
                assert np.array_equal(host(L.X), rec["X"]), (step, name)
        for blk in net.blocks:
            ref, s_ref = tr[blk["spec"].name]["out"]
            assert np.array_equal(host(blk["out"]), ref), (step, blk["spec"].name)
            assert host(blk["s_out"])[0] == s_ref
        assert np.array_equal(host(net.cat), tr["cat"][0]) and host(net.s_cat)[0] == tr["cat"][1]
        assert np.array_equal(host(net.z), tr["z"][0]) and host(net.s_z)[0] == tr["z"][1]
        out = ora.backward_update(tr, lab)
        assert np.array_equal(host(net.E), out["E"][0]) and host(net.s_E)[0] == out["E"][1]
        assert np.array_equal(host(net.e_cls), out["e_cls"][0])
        assert np.array_equal(host(net.e_c4), out["e_c4"][0].reshape(net.e_c4.shape))
        assert host(net.s_e_c4)[0] == out["e_c4"][1]
        for blk in net.blocks:
            ref, s_ref = out[blk["spec"].name]
            assert np.array_equal(host(blk["e_in"]), ref), (step, blk["spec"].name)
            assert host(blk["s_e_in"])[0] == s_ref
        assert np.array_equal(host(net.e_stem), out["e_stem"][0])
        for name, L in net.layers.items():
            r = out[name]
            gq, s_g = r["g"]
            assert np.array_equal(host(L.g), gq.astype(np.int8)), (step, name)
            assert host(L.s_g)[0] == s_g, (step, name)
            if L.spec.bn:
                dg, db = r["dgb"]
                assert np.array_equal(host(L.dgamma), dg) and np.array_equal(host(L.dbeta), db)
        for name, L in net.layers.items():
            i = L.lid
            assert np.array_equal(host(L.master), ora.masters[i]), (step, name)
            if L.spec.bn:
                assert np.array_equal(host(L.gm), ora.gm[i]), (step, name)
                assert np.array_equal(host(L.bm), ora.bm[i]), (step, name)
