"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module only draws random numbers (numpy ``default_rng``); it holds none of
the method's arithmetic, so the CUDA path and the CPU oracle can both consume
identical bytes without sharing any computation.  The distributions follow the
paper's workloads (Sec. 5: 8-bit activations and errors, He-initialised
weights stored on the 24-bit master grid, BN gamma/beta codes near 1 and 0,
uint8 RGB images, per-pixel class labels with an ignore value).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np



def rng(seed: int) -> np.random.Generator:
    return np.random.default_rng(seed)


def int8_uniform(g: np.random.Generator, shape, lo: int = -127, hi: int = 127) -> np.ndarray:
    """Integer codes uniform on [lo, hi] (activations / errors of the single-layer case)."""
    return g.integers(lo, hi + 1, size=shape, dtype=np.int64).astype(np.int8)


def he_weights(g: np.random.Generator, shape, fan_in: int) -> np.ndarray:
    """He (MSRA) initialisation, N(0, sqrt(2/fan_in)), as fp32 real weights (the
    method's W_m = UQ(W, k_U), Eq. (WQ0), is applied by whoever consumes them)."""
    std = np.sqrt(2.0 / fan_in)
    return (g.standard_normal(size=shape) * std).astype(np.float32)


def bilinear_filters(classes: int, R: int) -> np.ndarray:
    """Bilinear upsampling filters, one R x R filter per class, fp32 [classes][R][R]
    (the FCN decoder initialisation)."""
    f = (R + 1) // 2
    center = f - 1 if R % 2 == 1 else f - 0.5
    k1 = 1 - np.abs(np.arange(R) - center) / f
    return np.broadcast_to(np.outer(k1, k1).astype(np.float32), (classes, R, R)).copy()


VGG16 = [64, 64, "P", 128, 128, "P", 256, 256, 256, "P", 512, 512, 512, "P", 512, 512, 512, "P"]


def fcn_vgg16_channels(classes: int = 150, width: float = 1.0):
    """(name, cin, cout, r, pad, relu) of the FCN-VGG16 convolutions in forward order; the
    3 RGB input channels are padded to 4.  width scales every hidden channel count."""
    def ch(c):
        return max(8, int(round(c * width)) // 8 * 8)
    out, cin, i = [], 4, 0
    for item in VGG16:
        if item == "P":
            out.append(("pool", cin, cin, 2, 0, False))
            continue
        i += 1
        out.append((f"conv{i}", cin, ch(item), 3, 1, True))
        cin = ch(item)
    out.append(("fc6", cin, ch(4096), 7, 3, True))
    out.append(("fc7", ch(4096), ch(4096), 1, 0, True))
    out.append(("score", ch(4096), classes, 1, 0, False))
    return out


def fcn_vgg16_weights(seed: int, classes: int = 150, width: float = 1.0):
    """fp32 initial weights of FCN-VGG16: He-initialised KRSC filters for every conv
    (channel 3 of the first layer, the RGB padding, is zero) and the bilinear decoder."""
    g = rng(seed)
    ws = []
    for name, cin, cout, r, pad, relu in fcn_vgg16_channels(classes, width):
        if name == "pool":
            continue
        fan_in = (3 if cin == 4 else cin) * r * r
        w = he_weights(g, (cout, r, r, cin), fan_in)
        if cin == 4:
            w[..., 3] = 0.0
        ws.append(w)
    return ws, bilinear_filters(classes, 64)


def fcn8s_skip_weights(seed: int, classes: int = 150, width: float = 1.0):
    """fp32 initial weights of the FCN8s decoder: He-initialised 1x1 score filters on pool4
    and pool3 (KRSC), bilinear x2 (kernel 4) and x8 (kernel 16) per-class filters."""
    g = rng(seed + 7919)
    convs = [c for c in fcn_vgg16_channels(classes, width) if c[0] != "pool"]
    c4, c3 = convs[9][2], convs[6][2]          # conv4_3 and conv3_3 outputs (pool4, pool3)
    w4 = he_weights(g, (classes, 1, 1, c4), c4)
    w3 = he_weights(g, (classes, 1, 1, c3), c3)
    return w4, w3, bilinear_filters(classes, 4), bilinear_filters(classes, 16)


def bn_gamma_beta_codes(g: np.random.Generator, channels: int):
    """BN gamma in [0.5, 1.5] and beta in [-0.5, 0.5] drawn as integer codes of the
    8-bit x2-scaled grid (value = code * 2^-6)."""
    gam = g.integers(32, 97, size=channels, dtype=np.int64).astype(np.int32)
    bet = g.integers(-32, 33, size=channels, dtype=np.int64).astype(np.int32)
    return gam, bet


def images_u8(g: np.random.Generator, n: int, h: int, w: int, c: int = 3) -> np.ndarray:
    """Synthetic RGB images, uint8 uniform on [0, 255], NHWC."""
    return g.integers(0, 256, size=(n, h, w, c), dtype=np.int64).astype(np.uint8)


def labels_uniform_ignore(g: np.random.Generator, n: int, h: int, w: int, classes: int,
                          ignore_frac: float = 0.05, ignore: int = 255) -> np.ndarray:
    """Labels uniform on {0..classes-1}; an i.i.d. Bernoulli fraction set to ``ignore``."""
    lab = g.integers(0, classes, size=(n, h, w), dtype=np.int64)
    lab[g.random(size=(n, h, w)) < ignore_frac] = ignore
    return lab.astype(np.uint8)


def labels_voronoi(g: np.random.Generator, n: int, h: int, w: int, classes: int,
                   sites: int = 64) -> np.ndarray:
    """Piecewise-constant label maps: ``sites`` uniform points per image with uniform
    classes; each pixel takes the class of its nearest site (ties -> lower index)."""
    out = np.empty((n, h, w), np.uint8)
    yy, xx = np.mgrid[0:h, 0:w]
    for i in range(n):
        sy = g.integers(0, h, size=sites)
        sx = g.integers(0, w, size=sites)
        cls = g.integers(0, classes, size=sites)
        best = np.full((h, w), np.iinfo(np.int64).max, np.int64)
        lab = np.zeros((h, w), np.int64)
        for j in range(sites):
            d = (yy - sy[j]) ** 2 + (xx - sx[j]) ** 2
            m = d < best
            best[m] = d[m]
            lab[m] = cls[j]
        out[i] = lab
    return out


def float_uniform(g: np.random.Generator, shape, lo: float = -1.0, hi: float = 1.0) -> np.ndarray:
    return g.uniform(lo, hi, size=shape).astype(np.float32)


# ---------------------------------------------------------------- DeepLabv3-ResNet50

@dataclass
class ConvSpec:
    """One convolution of the network: KRSC weights [cout][r][r][cin], square kernel."""
    name: str
    cin: int
    cout: int
    r: int
    stride: int = 1
    pad: int = 0
    dil: int = 1
    bn: bool = True


@dataclass
class Bottleneck:
    name: str
    conv1: ConvSpec
    conv2: ConvSpec
    conv3: ConvSpec
    down: ConvSpec = None          # 1x1 projection shortcut (first block of a stage)


@dataclass
class DeepLabSpec:
    classes: int
    stem: ConvSpec                 # 7x7 stride 2, then 3x3 stride 2 max pool (padding 1)
    blocks: list
    aspp: list                     # 1x1 branch and the three atrous 3x3 branches
    pool_conv: ConvSpec            # image-pooling branch: global mean -> 1x1 conv
    project: ConvSpec              # 1x1 over the concatenation
    head: ConvSpec                 # 3x3
    cls: ConvSpec                  # 1x1 classifier, no BN, no ReLU
    up: int = 8                    # bilinear factor, aligned corners

    def convs(self):
        """Every convolution in forward order (the layer ids of the RNG key)."""
        out = [self.stem]
        for b in self.blocks:
            out += [b.conv1, b.conv2, b.conv3] + ([b.down] if b.down else [])
        return out + list(self.aspp) + [self.pool_conv, self.project, self.head, self.cls]


def deeplabv3_r50_spec(classes: int = 21, width: float = 1.0, blocks=(3, 4, 6, 3),
                       rates=(12, 24, 36)) -> DeepLabSpec:
    """DeepLabv3 on ResNet-50 at output stride 8: stages of (3, 4, 6, 3) bottlenecks with
    stride 2 in the 3x3 convolution of stage 2's first block, stages 3 and 4 dilated (2 and
    4; the first block of each keeps the previous dilation), ASPP with a 1x1 branch, 3x3
    branches at rates 12/24/36 and an image-pooling branch (256 channels each), a 1x1
    projection, a 3x3 head and a 1x1 classifier.  width scales every channel count
    (multiples of 16, at least 16); the input has 4 channels (RGB padded)."""
    def ch(c):
        return max(16, int(round(c * width)) // 16 * 16)
    stem = ConvSpec("stem", 4, ch(64), 7, 2, 3)
    out_blocks, cin, dil = [], ch(64), 1
    for si, (nb, mid, stride, new_dil) in enumerate(zip(blocks, (64, 128, 256, 512),
                                                        (1, 2, 1, 1), (1, 1, 2, 4))):
        cout = ch(mid * 4)
        for bi in range(nb):
            d = dil if bi == 0 else new_dil
            s = stride if bi == 0 else 1
            nm = f"layer{si + 1}.{bi}"
            down = None
            if bi == 0 and (s != 1 or cin != cout):
                down = ConvSpec(nm + ".down", cin, cout, 1, s, 0)
            out_blocks.append(Bottleneck(
                nm, ConvSpec(nm + ".conv1", cin, ch(mid), 1),
                ConvSpec(nm + ".conv2", ch(mid), ch(mid), 3, s, d, d),
                ConvSpec(nm + ".conv3", ch(mid), cout, 1), down))
            cin = cout
        dil = new_dil
    a = ch(256)
    aspp = [ConvSpec("aspp.b0", cin, a, 1)] + [
        ConvSpec(f"aspp.b{i + 1}", cin, a, 3, 1, r, r) for i, r in enumerate(rates)]
    return DeepLabSpec(classes, stem, out_blocks, aspp, ConvSpec("aspp.pool", cin, a, 1),
                       ConvSpec("aspp.project", 5 * a, a, 1), ConvSpec("head", a, a, 3, 1, 1),
                       ConvSpec("cls", a, classes, 1, bn=False))


def deeplabv3_r50_init(seed: int, spec: DeepLabSpec):
    """Initial parameters: fp32 He weights per conv (input channel 3 of the stem, the RGB
    padding, zero), and per BN conv the gamma / beta master codes on the 24-bit x2-scaled
    grid (value m 2^-22), drawn as 8-bit codes (gamma in [0.5, 1.5], beta in [-0.5, 0.5])
    times 2^16 so that the 8-bit codes the forward uses are exactly the drawn ones."""
    g = rng(seed)
    ws, gms, bms = [], [], []
    for cv in spec.convs():
        fan_in = (3 if cv.cin == 4 else cv.cin) * cv.r * cv.r
        w = he_weights(g, (cv.cout, cv.r, cv.r, cv.cin), fan_in)
        if cv.cin == 4:
            w[..., 3] = 0.0
        ws.append(w)
        if cv.bn:
            gam, bet = bn_gamma_beta_codes(g, cv.cout)
            gms.append(gam.astype(np.int32) * np.int32(1 << 16))
            bms.append(bet.astype(np.int32) * np.int32(1 << 16))
        else:
            gms.append(None)
            bms.append(None)
    return ws, gms, bms
