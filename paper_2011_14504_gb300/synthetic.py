"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module only draws random numbers (numpy ``default_rng``); it holds none of
the method's arithmetic, so the CUDA path and the CPU oracle can both consume
identical bytes without sharing any computation.  The distributions follow the
paper's workloads (Sec. 5: 8-bit activations and errors, He-initialised
weights stored on the 24-bit master grid, BN gamma/beta codes near 1 and 0,
uint8 RGB images, per-pixel class labels with an ignore value).
"""
from __future__ import annotations

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
