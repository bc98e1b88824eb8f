"""The network topology that the GPU networks and the oracle networks both read
(paper_2011_14504_gb300/synthetic.py), pinned against the benchmark configurations' own
description of the two networks, and the multiply-accumulate counts against figures
worked out independently from that description.

A wrong stride, dilation or channel count in the shared spec would pass every parity test
(both sides would build the same wrong network), so it is checked here against the
configuration text: FCN-VGG16 with 13 3x3 convs (64-64-128-128-256x3-512x3-512x3) and 5 max
pools, fc6 / fc7 as 7x7 / 1x1 convs at 4096 channels and a 150-class 1x1 score layer;
DeepLabv3-ResNet50 with bottleneck stages [3, 4, 6, 3], output stride 8 with dilation 2 / 4
in the last two stages, ASPP of a 1x1 branch, 3x3 branches at rates 12 / 24 / 36 and an
image-pool branch, all 256 channels, and 21 classes (paper Sec. 2.1 and Sec. 5.1)."""
import bench
from paper_2011_14504_gb300 import synthetic as S
from paper_2011_14504_gb300.work import conv_macs, inbounds_pairs, out_size, transposed_macs


def test_fcn_vgg16_topology():
    layers = S.fcn_vgg16_channels(150, 1.0)
    convs = [L for L in layers if L[0] != "pool"]
    pools = [L for L in layers if L[0] == "pool"]
    assert len(pools) == 5
    vgg = [L for L in convs if L[0].startswith("conv")]
    assert [L[2] for L in vgg] == [64, 64, 128, 128, 256, 256, 256, 512, 512, 512, 512, 512, 512]
    assert all(L[3] == 3 and L[4] == 1 and L[5] for L in vgg)
    assert vgg[0][1] == 4            # RGB padded to 4 channels
    # a pool after conv2, conv4, conv7, conv10, conv13
    order = [L[0] for L in layers]
    for i in (2, 4, 7, 10, 13):
        assert order[order.index(f"conv{i}") + 1] == "pool"
    fc6, fc7, score = convs[-3:]
    assert fc6[0] == "fc6" and fc6[1:5] == (512, 4096, 7, 3) and fc6[5]
    assert fc7[0] == "fc7" and fc7[1:5] == (4096, 4096, 1, 0) and fc7[5]
    assert score[0] == "score" and score[1:5] == (4096, 150, 1, 0) and not score[5]
    # output stride 32: 16 x 16 score map at 512 x 512
    _, (hs, ws) = bench.fcn_layers(16, 512, 512, 150)
    assert (hs, ws) == (16, 16)


def test_deeplabv3_r50_topology():
    sp = S.deeplabv3_r50_spec(21, 1.0)
    assert sp.classes == 21 and sp.up == 8
    assert (sp.stem.cin, sp.stem.cout, sp.stem.r, sp.stem.stride, sp.stem.pad) == (4, 64, 7, 2, 3)
    stages = {}
    for b in sp.blocks:
        stages.setdefault(b.name.split(".")[0], []).append(b)
    assert [len(stages[k]) for k in ("layer1", "layer2", "layer3", "layer4")] == [3, 4, 6, 3]
    mids = {"layer1": 64, "layer2": 128, "layer3": 256, "layer4": 512}
    for name, blocks in stages.items():
        for i, b in enumerate(blocks):
            mid = mids[name]
            assert (b.conv1.r, b.conv1.cout) == (1, mid)
            assert (b.conv2.r, b.conv2.cin, b.conv2.cout) == (3, mid, mid)
            assert (b.conv3.r, b.conv3.cout) == (1, 4 * mid)
            assert b.conv2.pad == b.conv2.dil
            # stride 2 only in the first 3x3 of stage 2; stages 3 / 4 dilated 2 / 4 after
            # their first block (which keeps the previous stage's dilation)
            assert b.conv2.stride == (2 if (name == "layer2" and i == 0) else 1)
            want_dil = {"layer1": 1, "layer2": 1, "layer3": 2, "layer4": 4}[name]
            if i == 0:
                want_dil = {"layer1": 1, "layer2": 1, "layer3": 1, "layer4": 2}[name]
            assert b.conv2.dil == want_dil, (name, i)
            assert (b.down is not None) == (i == 0)
    assert len(sp.aspp) == 4
    assert sp.aspp[0].r == 1 and [a.dil for a in sp.aspp[1:]] == [12, 24, 36]
    assert all(a.r == 3 and a.pad == a.dil for a in sp.aspp[1:])
    assert all(a.cin == 2048 and a.cout == 256 for a in sp.aspp)
    assert (sp.pool_conv.cin, sp.pool_conv.cout, sp.pool_conv.r) == (2048, 256, 1)
    assert (sp.project.cin, sp.project.cout) == (5 * 256, 256)
    assert (sp.head.r, sp.head.cout) == (3, 256)
    assert (sp.cls.cout, sp.cls.r, sp.cls.bn) == (21, 1, False)
    # output stride 8: 65 x 65 features at 513 x 513 (stem /2, pool /2, stage 2 /2)
    layers = bench.deeplab_layers(sp, 16, 513)
    aspp_in = [L for L in layers if L[3] == 2048 and L[4] == 256 and L[1] > 1]
    assert len(aspp_in) == 4 and all(L[1] == 65 and L[2] == 65 for L in aspp_in)
    pooled = [L for L in layers if L[3] == 2048 and L[4] == 256 and L[1] == 1]
    assert len(pooled) == 1          # the image-pool branch's 1x1 conv on the pooled map
    # the stride-2 3x3 reads the 129 x 129 stage-1 map and writes 65 x 65
    s2 = [L for L in layers if L[6] == 2 and L[5] == 3]
    assert len(s2) == 1 and s2[0][1] == 129 and out_size(129, 3, 2, 1, 1) == 65


def test_inbounds_pair_counts_by_brute_force():
    for extent in (1, 5, 16, 33, 65):
        for taps, stride, dil, pad in ((3, 1, 1, 1), (7, 2, 1, 3), (3, 1, 36, 36),
                                       (3, 2, 1, 1), (1, 1, 1, 0), (3, 1, 12, 12)):
            out = out_size(extent, taps, stride, pad, dil)
            if out < 1:
                continue
            brute = sum(1 for o in range(out) for t in range(taps)
                        if 0 <= o * stride + t * dil - pad < extent)
            assert inbounds_pairs(extent, out, taps, stride, dil, pad) == brute


def test_step_macs_match_independent_figures():
    # dense figures from the configuration text, worked out by hand: FCN-VGG16 forward at
    # N=8, 512^2: 0.889 T MAC; DeepLabv3-R50 forward at N=8, 513^2: 1.349 T MAC
    fcn, (hs, ws) = bench.fcn_layers(8, 512, 512, 150)
    dec = transposed_macs(8, hs, ws, 150, 64, 32, 16)
    assert dec[1] == 8 * 512 * 512 * 150 * 4                  # 2 x 2 taps per output pixel
    assert dec[0] == 8 * 150 * (64 * 16 - 32) ** 2             # the border rows lose a tap
    inb, dense = bench.step_macs(fcn, False, dec)
    assert abs(dense / 0.889e12 - 1) < 2e-3
    sp = S.deeplabv3_r50_spec(21, 1.0)
    inb_d, dense_d = bench.step_macs(bench.deeplab_layers(sp, 8, 513), False)
    assert abs(dense_d / 1.349e12 - 1) < 2e-3
    # the ASPP rates 12 / 24 / 36 keep 77 / 57 / 40 % of their taps at 65 x 65
    for rate, keep in ((12, 0.77), (24, 0.57), (36, 0.40)):
        i, d = conv_macs(1, 65, 65, 2048, 256, 3, 1, rate, rate)
        assert abs(i / d - keep) < 0.01
    assert 0.83 < inb_d / dense_d < 0.84
    # a training step: forward + data gradient (not the first layer) + weight gradient
    t_inb, t_dense = bench.step_macs(bench.deeplab_layers(sp, 16, 513), True)
    assert abs(t_dense / 8.085e12 - 1) < 1e-3
