"""Algorithmic work of a convolution pass, for throughput figures.

A pass (forward, data gradient or weight gradient: the same products in three
arrangements) performs, per output channel and input channel, one multiply-accumulate
for every (output pixel, tap) pair whose input pixel lies inside the image.  Taps that
read the zero padding do no work; counting them as well gives the dense figure
N P Q K R S C / groups.
"""
from __future__ import annotations


def inbounds_pairs(extent: int, out: int, taps: int, stride: int, dil: int, pad: int) -> int:
    """(output index, tap) pairs of one spatial dimension with o stride + t dil - pad
    inside [0, extent)."""
    n = 0
    for t in range(taps):
        lo = t * dil - pad                      # input index of output 0
        # outputs o with 0 <= lo + o stride < extent
        first = 0 if lo >= 0 else (-lo + stride - 1) // stride
        last = (extent - 1 - lo) // stride if extent - 1 - lo >= 0 else -1
        last = min(last, out - 1)
        if last >= first:
            n += last - first + 1
    return n


def out_size(extent: int, taps: int, stride: int, pad: int, dil: int) -> int:
    return (extent + 2 * pad - dil * (taps - 1) - 1) // stride + 1


def conv_macs(n: int, h: int, w: int, cin: int, cout: int, r: int, stride: int = 1,
              pad: int = 0, dil: int = 1, groups: int = 1):
    """(in-bounds, dense) multiply-accumulates of one pass of an r x r convolution."""
    p, q = out_size(h, r, stride, pad, dil), out_size(w, r, stride, pad, dil)
    cg = cin // groups
    dense = n * p * q * cout * r * r * cg
    inb = n * cout * cg * inbounds_pairs(h, p, r, stride, dil, pad) * \
        inbounds_pairs(w, q, r, stride, dil, pad)
    return inb, dense


def transposed_macs(n: int, h: int, w: int, c: int, R: int, stride: int, pad: int):
    """(in-bounds, dense) multiply-accumulates of a per-channel transposed convolution
    (kernel R, stride, padding) of an h x w input into (h-1) stride - 2 pad + R outputs:
    every (input pixel, tap) pair whose output lands inside counts; the dense figure
    counts ceil(R / stride)^2 taps for every output pixel."""
    H = (h - 1) * stride - 2 * pad + R
    W = (w - 1) * stride - 2 * pad + R

    def pairs(extent, out):
        k = 0
        for i in range(extent):
            for t in range(R):
                y = i * stride + t - pad
                k += 0 <= y < out
        return k
    per = -(-R // stride)
    return n * c * pairs(h, H) * pairs(w, W), n * c * H * W * per * per
