"""FCN-VGG16 training steps on the GPU against the oracle network, free-running.

A reduced-width network (same layer structure, channels x 1/8) on 64 x 64 images keeps
the oracle in seconds; both sides start from the same fp32 initial weights and consume
identical input bytes, so every intermediate must agree bit for bit, step after step.
"""
import numpy as np
import pytest
import torch

import oracle as O
from oracle.fcn import OracleFcn
from paper_2011_14504_gb300 import synthetic as S
from paper_2011_14504_gb300.fcn import FcnVgg16, Pool

pytestmark = pytest.mark.gpu


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


@pytest.mark.parametrize("classes,width,n,h", [(21, 0.125, 2, 64), (150, 0.0625, 1, 64),
                                               (150, 0.0625, 1, 128)])
def test_fcn_train_steps_match_oracle(classes, width, n, h):
    w = h
    seed = 3
    g = S.rng(100 + classes)
    net = FcnVgg16(n, h, w, classes=classes, width=width, seed=seed, lr_log2=6)
    chans = S.fcn_vgg16_channels(classes, width)
    wts, up = S.fcn_vgg16_weights(seed, classes, width)
    ora = OracleFcn(chans, wts, up, classes, seed=seed, lr_log2=6)
    for step in range(2):
        img = S.images_u8(g, n, h, w)
        lab = S.labels_voronoi(g, n, h, w, classes, sites=6)
        net.train_step(torch.from_numpy(img).cuda(), torch.from_numpy(lab).cuda())
        tr = ora.forward(img)
        convs = [it for it in tr["layers"] if it[0] == "conv"]
        for L, it in zip(net.convs, convs):
            _, li, cv, x, s_x, wq, acc, a, s_a, relu = it
            assert np.array_equal(host(L.a), a), (step, L.name)
            assert host(L.s_a)[0] == s_a, (step, L.name)
        cvu, score, s_score, up_wq, zacc, z, s_z = tr["up"]
        assert np.array_equal(host(net.z), z) and host(net.s_z)[0] == s_z
        out = ora.backward_update(tr, lab)
        E, s_E = out["E"]
        assert np.array_equal(host(net.Ez), E) and host(net.s_Ez)[0] == s_E
        assert np.array_equal(host(net.e_score), out["e_score"][0])
        assert np.array_equal(host(net.up_g), out["up_g"][1])
        for L in net.convs:
            G, gq, s_g = out["grads"][L.layer_id]
            assert np.array_equal(host(L.g), gq.astype(np.int8)), (step, L.name)
            assert host(L.s_g)[0] == s_g
            if L.layer_id > 0:
                want = out["ex"][L.layer_id][0]
                if L.ex_masked:      # the ReLU backward of the conv below, fused (mask: x > 0;
                    # x is the conv below's output, checked against the oracle above)
                    want = O.relu_bwd(want, host(L.x))
                assert np.array_equal(host(L.ex), want), (step, L.name)
            assert np.array_equal(host(L.master), ora.masters[L.layer_id]), (step, L.name)
        assert np.array_equal(host(net.up_master), ora.up_master)


@pytest.mark.parametrize("classes,width,n,h,wd", [(21, 0.125, 2, 64, 0), (150, 0.0625, 1, 128, 17)])
def test_fcn8s_train_steps_match_oracle(classes, width, n, h, wd):
    """The FCN8s decoder (score convs on pool4 / pool3, x2, x2, x8 transposed convs, the two
    joins and the skips' errors joined at the pools), two free-running steps; one case with
    the decoupled L2 weight decay after every update."""
    w = h
    seed = 4
    g = S.rng(200 + classes)
    net = FcnVgg16(n, h, w, classes=classes, width=width, seed=seed, lr_log2=6, skips=True,
                   wd_shift=wd)
    chans = S.fcn_vgg16_channels(classes, width)
    wts, up = S.fcn_vgg16_weights(seed, classes, width)
    ora = OracleFcn(chans, wts, up, classes, seed=seed, lr_log2=6,
                    skips=S.fcn8s_skip_weights(seed, classes, width), wd_shift=wd)
    for step in range(2):
        img = S.images_u8(g, n, h, w)
        lab = S.labels_voronoi(g, n, h, w, classes, sites=6)
        net.train_step(torch.from_numpy(img).cuda(), torch.from_numpy(lab).cuda())
        tr = ora.forward(img)
        convs = [it for it in tr["layers"] if it[0] == "conv"]
        for L, it in zip(net.convs, convs):
            assert np.array_equal(host(L.a), it[7]), (step, L.name)
            assert host(L.s_a)[0] == it[8], (step, L.name)
        for U, key in ((net.up2a, "up2a"), (net.up2b, "up2b"), (net.up8, "up")):
            assert np.array_equal(host(U.z), tr[key][5]), (step, key)
            assert host(U.s_z)[0] == tr[key][6], (step, key)
        for L, key in ((net.sp4, "sp4"), (net.sp3, "sp3")):
            assert np.array_equal(host(L.a), tr[key][5]), (step, key)
            assert host(L.s_a)[0] == tr[key][6], (step, key)
        assert np.array_equal(host(net.fuse4), tr["fuse4"][0])
        assert host(net.s_fuse4)[0] == tr["fuse4"][1]
        assert np.array_equal(host(net.fuse3), tr["fuse3"][0])
        assert host(net.s_fuse3)[0] == tr["fuse3"][1]
        out = ora.backward_update(tr, lab)
        assert np.array_equal(host(net.Ez), out["E"][0])
        assert np.array_equal(host(net.up8.ex), out["e_fuse3"][0])
        assert host(net.up8.s_ex)[0] == out["e_fuse3"][1]
        assert np.array_equal(host(net.up2b.ex), out["e_fuse4"][0])
        assert np.array_equal(host(net.sp3.ex), out["e_sp3"][0])
        assert np.array_equal(host(net.sp4.ex), out["e_sp4"][0])
        assert np.array_equal(host(net.e_score), out["e_score"][0])
        for k in (2, 3):
            assert np.array_equal(host(net.ej[k][0]), out["e_pool"][k][0]), (step, k)
            assert host(net.ej[k][1])[0] == out["e_pool"][k][1], (step, k)
        for U, key in ((net.up8, "up8_g"), (net.up2b, "up2b_g"), (net.up2a, "up2a_g"),
                       (net.sp3, "sp3_g"), (net.sp4, "sp4_g")):
            assert np.array_equal(host(U.g), out[key][1].astype(np.int8)), (step, key)
            assert host(U.s_g)[0] == out[key][2], (step, key)
        for L in net.convs:
            G, gq, s_g = out["grads"][L.layer_id]
            assert np.array_equal(host(L.g), gq.astype(np.int8)), (step, L.name)
            if L.layer_id > 0:
                want = out["ex"][L.layer_id][0]
                if L.ex_masked:      # the ReLU backward of the conv below, fused (mask: x > 0;
                    # x is the conv below's output, checked against the oracle above)
                    want = O.relu_bwd(want, host(L.x))
                assert np.array_equal(host(L.ex), want), (step, L.name)
            assert np.array_equal(host(L.master), ora.masters[L.layer_id]), (step, L.name)
        for U, m in ((net.up8, ora.up8_master), (net.up2b, ora.up2b_master),
                     (net.up2a, ora.up2a_master), (net.sp4, ora.sp4_master),
                     (net.sp3, ora.sp3_master)):
            assert np.array_equal(host(U.master), m)
