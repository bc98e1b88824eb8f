"""FCN-VGG16 on the iq C ABI: the quantized training step and inference pass.

Network (Sec. 2.1 / Sec. 5): the 13 VGG16 3x3 convolutions with 5 max pools, fc6 as a
7x7 convolution (padding 3) and fc7 as a 1x1 convolution (4096 channels), a 1x1
score layer over the classes, and a 32x per-class transposed-convolution decoder
(kernel 64, stride 32, padding 16, bilinear-initialised, trainable).  No BN (Sec. 5:
FCN uses GQ2 and the MSE loss).  With skips=True the decoder is the paper's FCN8s
(Sec. 2.1): 1x1 score convolutions on pool4 and pool3, x2, x2 and x8 per-class transposed
convolutions (kernels 4 / 4 / 16, bilinear-initialised, trainable), each skip joined by a
real-valued sum requantized with SQ(., 8) (iq_combine); in the backward a sum's error
reaches both operands unchanged, and a skip's error joins the main path's at its pool.

Dataflow per layer (Sec. 3.2-3.3): W_q = UQ(W_m, 8) from 24-bit master weights,
int32 convolution, A = Q_A(ReLU(acc)) = SQ(., 8); backward e = e_A [A > 0],
E_1 = SQ(dgrad, 8), G_q = RQ(G/Scale(G), 8) (Eq. (GQ2)), W_m -= UQ(G_q lr, 24).

Every step runs in the library's kernels; this module only allocates device memory
(torch tensors) and sequences the C ABI calls on one stream.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from . import iq
from . import synthetic as S
from .work import conv_macs, transposed_macs

UP_R, UP_STRIDE, UP_PAD = 64, 32, 16
UP2 = (4, 2, 1)          # FCN8s x2: kernel, stride, padding
UP8 = (16, 8, 4)         # FCN8s x8


@dataclass
class Conv:
    name: str
    desc: iq.ConvDesc
    cin: int
    cout: int
    r: int
    pad: int
    relu: bool
    layer_id: int
    master: torch.Tensor = None
    wq: torch.Tensor = None
    g: torch.Tensor = None
    s_g: torch.Tensor = None
    x: torch.Tensor = None        # input codes (NHWC)
    s_x: torch.Tensor = None
    a: torch.Tensor = None        # output codes
    s_a: torch.Tensor = None
    ea: torch.Tensor = None       # error of the output (E_1)
    s_ea: torch.Tensor = None
    e: torch.Tensor = None        # error after the ReLU mask
    ex: torch.Tensor = None       # error of the input (dgrad output)
    s_ex: torch.Tensor = None
    x16: torch.Tensor = None      # fp16 copy of x, read by the forward and the wgrad
    a16: torch.Tensor = None      # the next conv's x16 when that conv reads a: written here
    ex_masked: bool = False       # ex carries the ReLU mask of the conv below (x > 0)
    macs: int = 0                 # in-bounds multiply-accumulates of one pass
    macs_dense: int = 0           # every tap, the zero padding included


@dataclass
class Pool:
    x: torch.Tensor
    y: torch.Tensor
    arg: torch.Tensor
    y16: torch.Tensor = None      # the next conv's x16 when it reads y: written by the pool
    ey: torch.Tensor = None       # error of the pooled output
    s_ey: torch.Tensor = None
    ex: torch.Tensor = None       # error of the pool input
    s_ex: torch.Tensor = None


@dataclass
class Up:
    """A per-class transposed convolution of the decoder."""
    R: int
    stride: int
    pad: int
    layer_id: int
    x: torch.Tensor
    s_x: torch.Tensor
    master: torch.Tensor = None
    wq: torch.Tensor = None
    z: torch.Tensor = None
    s_z: torch.Tensor = None
    g: torch.Tensor = None
    s_g: torch.Tensor = None
    ex: torch.Tensor = None       # error of its input
    s_ex: torch.Tensor = None
    macs: int = 0
    macs_dense: int = 0


class FcnVgg16:
    """Preallocated FCN-VGG16 for a fixed batch shape.

    width scales every channel count (1.0 = the paper's network); tests use small widths."""

    def __init__(self, n: int, h: int, w: int, classes: int = 150, width: float = 1.0,
                 seed: int = 0, lr_log2: int = 10, device: str = "cuda", train: bool = True,
                 skips: bool = False, wd_shift: int = 0):
        assert h % 32 == 0 and w % 32 == 0, "the 32x decoder needs sizes divisible by 32"
        self.n, self.h, self.w, self.classes = n, h, w, classes
        self.dev = torch.device(device)
        self.lr_log2 = lr_log2
        self.train = train
        self.skips = skips
        self.wd_shift = wd_shift      # decoupled L2 weight decay, step 2^-wd_shift (0: none)
        self.step_count = 0
        self.seed = seed
        dev = self.dev

        def scal():
            return torch.zeros(1, dtype=torch.float64, device=dev)

        self.img_codes = torch.empty((n, h, w, 4), dtype=torch.int8, device=dev)
        self.s_img = scal()
        self.layers: list = []   # Conv and Pool in forward order
        self.convs: list = []
        weights, up_filters = S.fcn_vgg16_weights(seed, classes, width)
        cur, s_cur, hh, ww = self.img_codes, self.s_img, h, w
        lid = 0
        self.pools = []          # (Pool, scale of its codes) in forward order
        for name, cin, cout, r, pad, relu in S.fcn_vgg16_channels(classes, width):
            if name == "pool":
                y = torch.empty((n, hh // 2, ww // 2, cin), dtype=torch.int8, device=dev)
                arg = torch.empty_like(y, dtype=torch.uint8)
                self.layers.append(Pool(cur, y, arg))
                self.pools.append((self.layers[-1], s_cur))
                cur, hh, ww = y, hh // 2, ww // 2
                continue
            cur, s_cur = self._add_conv(name, cur, s_cur, cin, cout, r, pad, relu, lid, hh, ww,
                                        weights[lid])
            lid += 1
        self.score, self.s_score, self.score_hw = cur, s_cur, (hh, ww)
        self.skip_convs = []
        if skips:
            self._build_fcn8s(lid, seed, width)
            self._alloc_carriers()
            self._alloc_backward()
            self.ws = torch.empty(self._ws_bytes(), dtype=torch.uint8, device=dev)
            return
        # decoder: per-class transposed convolution, W_m = UQ(W, 24) (Eq. (WQ0))
        self.up_layer_id = lid
        self.up_master = self._master(up_filters)
        self.up_wq = torch.empty((classes, UP_R, UP_R), dtype=torch.int8, device=dev)
        iq.iq_weight_requant(self.up_master, self.up_wq)
        self.z = torch.empty((n, h, w, classes), dtype=torch.int8, device=dev)
        self.s_z = scal()
        if train:
            self.Ez = torch.empty_like(self.z)
            self.s_Ez = scal()
            self.up_g = torch.empty_like(self.up_wq)
            self.up_s_g = scal()
            self.e_score = torch.empty_like(self.score)
            self.s_e_score = scal()
        # the decoder: (in-bounds, dense) multiply-accumulates, <= 2 x 2 taps per output pixel
        self.up_macs, self.up_macs_dense = transposed_macs(n, self.score_hw[0],
                                                           self.score_hw[1], classes, UP_R,
                                                           UP_STRIDE, UP_PAD)
        self._alloc_carriers()
        self._alloc_backward()
        self.ws = torch.empty(self._ws_bytes(), dtype=torch.uint8, device=dev)

    def _build_fcn8s(self, L: int, seed: int, width: float):
        """The FCN8s decoder over the encoder just built; layer ids as in the oracle."""
        n, dev, c = self.n, self.dev, self.classes
        w4, w3, up2, up8 = S.fcn8s_skip_weights(seed, c, width)
        (P3, s3), (P4, s4) = self.pools[2], self.pools[3]
        self.sp4 = self._skip_conv("score_pool4", P4.y, s4, w4, L + 3)
        self.sp3 = self._skip_conv("score_pool3", P3.y, s3, w3, L + 4)
        self.up2a = self._up_layer(self.score, self.s_score, up2, UP2, L + 2)
        self.fuse4 = torch.empty_like(self.sp4.a)
        self.s_fuse4 = torch.zeros(1, dtype=torch.float64, device=dev)
        self.up2b = self._up_layer(self.fuse4, self.s_fuse4, up2, UP2, L + 1)
        self.fuse3 = torch.empty_like(self.sp3.a)
        self.s_fuse3 = torch.zeros(1, dtype=torch.float64, device=dev)
        self.up8 = self._up_layer(self.fuse3, self.s_fuse3, up8, UP8, L)
        self.ups = [self.up2a, self.up2b, self.up8]
        self.z, self.s_z = self.up8.z, self.up8.s_z
        if self.train:
            self.Ez = torch.empty_like(self.z)
            self.s_Ez = torch.zeros(1, dtype=torch.float64, device=dev)
            self.e_score = self.up2a.ex
            self.s_e_score = self.up2a.s_ex
            # the joined errors at the outputs of pool4 and pool3
            self.ej = {3: (torch.empty_like(P4.y), torch.zeros(1, dtype=torch.float64, device=dev)),
                       2: (torch.empty_like(P3.y), torch.zeros(1, dtype=torch.float64, device=dev))}
        self.up_macs = sum(u.macs for u in self.ups)
        self.up_macs_dense = sum(u.macs_dense for u in self.ups)

    def _skip_conv(self, name, x, s_x, w_fp32, lid):
        n, dev = self.n, self.dev
        _, hh, ww, cin = x.shape
        d = iq.conv_desc(n, hh, ww, cin, self.classes, 1, 1, 1, 0)
        L = Conv(name, d, cin, self.classes, 1, 0, False, lid)
        L.master = self._master(w_fp32)
        L.wq = torch.empty((self.classes, 1, 1, cin), dtype=torch.int8, device=dev)
        iq.iq_weight_requant(L.master, L.wq)
        L.x, L.s_x = x, s_x
        L.a = torch.empty((n, hh, ww, self.classes), dtype=torch.int8, device=dev)
        L.s_a = torch.zeros(1, dtype=torch.float64, device=dev)
        L.macs, L.macs_dense = conv_macs(n, hh, ww, cin, self.classes, 1, 1, 0)
        if self.train:
            L.g = torch.empty_like(L.wq)
            L.s_g = torch.zeros(1, dtype=torch.float64, device=dev)
            L.ex = torch.empty_like(x)
            L.s_ex = torch.zeros(1, dtype=torch.float64, device=dev)
        self.skip_convs.append(L)
        return L

    def _up_layer(self, x, s_x, w_fp32, geom, lid):
        R, stride, pad = geom
        n, dev = self.n, self.dev
        _, hh, ww, c = x.shape
        U = Up(R, stride, pad, lid, x, s_x)
        U.master = self._master(w_fp32)
        U.wq = torch.empty((c, R, R), dtype=torch.int8, device=dev)
        iq.iq_weight_requant(U.master, U.wq)
        H, W = (hh - 1) * stride - 2 * pad + R, (ww - 1) * stride - 2 * pad + R
        U.z = torch.empty((n, H, W, c), dtype=torch.int8, device=dev)
        U.s_z = torch.zeros(1, dtype=torch.float64, device=dev)
        U.macs, U.macs_dense = transposed_macs(n, hh, ww, c, R, stride, pad)
        if self.train:
            U.g = torch.empty_like(U.wq)
            U.s_g = torch.zeros(1, dtype=torch.float64, device=dev)
            U.ex = torch.empty_like(x)
            U.s_ex = torch.zeros(1, dtype=torch.float64, device=dev)
        return U

    def _master(self, w_fp32: np.ndarray) -> torch.Tensor:
        """Master weights W_m = UQ(W, 24) (Eq. (WQ0)) computed on the device."""
        w = torch.from_numpy(np.ascontiguousarray(w_fp32)).to(self.dev)
        m = torch.empty(w.shape, dtype=torch.int32, device=self.dev)
        iq.iq_quantize(w, 24, iq.IQ_MODE_UQ, m, torch.zeros(1, dtype=torch.float64,
                                                            device=self.dev))
        return m

    # ------------------------------------------------------------------ construction

    def _add_conv(self, name, x, s_x, cin, cout, r, pad, relu, lid, hh, ww, w_fp32):
        n, dev = self.n, self.dev
        d = iq.conv_desc(n, hh, ww, cin, cout, r, r, 1, pad)
        L = Conv(name, d, cin, cout, r, pad, relu, lid)
        L.master = self._master(w_fp32)
        L.wq = torch.empty((cout, r, r, cin), dtype=torch.int8, device=dev)
        iq.iq_weight_requant(L.master, L.wq)
        L.x, L.s_x = x, s_x
        L.a = torch.empty((n, hh, ww, cout), dtype=torch.int8, device=dev)
        L.s_a = torch.zeros(1, dtype=torch.float64, device=dev)
        # the first layer's fourth input channel is the zero RGB padding: no work
        L.macs, L.macs_dense = conv_macs(n, hh, ww, 3 if cin == 4 else cin, cout, r, 1, pad)
        self.layers.append(L)
        self.convs.append(L)
        return L.a, L.s_a

    def _alloc_backward(self):
        if not self.train:
            return
        dev = self.dev
        for L in self.convs:
            L.ea = torch.empty_like(L.a)
            L.s_ea = torch.zeros(1, dtype=torch.float64, device=dev)
            L.e = torch.empty_like(L.a)
            L.g = torch.empty_like(L.wq)
            L.s_g = torch.zeros(1, dtype=torch.float64, device=dev)
            if L.layer_id > 0:
                L.ex = torch.empty_like(L.x)
                L.s_ex = torch.zeros(1, dtype=torch.float64, device=dev)
        for P in self.layers:
            if isinstance(P, Pool):
                P.ex = torch.empty_like(P.x)
                P.s_ex = torch.zeros(1, dtype=torch.float64, device=dev)
        # fp16 error buffers: written with the errors by the ReLU backward of a layer or by
        # the data gradient of the conv above it, read by its data and weight gradients
        # (IQ_CONV_E_F16_READY)
        e16 = 0
        for L in self.convs:
            if L.cout % 64 == 0:
                e16 = max(e16, L.a.numel())
                if L.relu:
                    L.desc.flags |= iq.IQ_CONV_E_F16_READY
        # two of them: a data gradient writes the next layer's copy (with the ReLU mask
        # fused, below) while this layer's weight gradient still reads its own
        self.e16 = [torch.empty(max(e16, 16), dtype=torch.float16, device=dev) for _ in range(2)]

    def _alloc_carriers(self):
        """fp16 copies of the codes that the tensor-core kernels read: one per conv input,
        written by the item that produces the input (the previous conv's requantization or
        the pool) and read as it is by the conv's forward (IQ_CONV_X_F16_READY) and weight
        gradient."""
        prev = None
        for item in self.layers:
            if isinstance(item, Conv):
                L = item
                if L.cin % 64 == 0 and L.x.numel() % 16 == 0:
                    L.x16 = torch.empty(L.x.numel(), dtype=torch.float16, device=self.dev)
                    if isinstance(prev, Conv) and prev.a is L.x:
                        prev.a16 = L.x16
                        L.desc.flags |= iq.IQ_CONV_X_F16_READY
                    elif isinstance(prev, Pool) and prev.y is L.x:
                        prev.y16 = L.x16
                        L.desc.flags |= iq.IQ_CONV_X_F16_READY
            prev = item

    def _ws_bytes(self) -> int:
        b = iq.iq_quantize_workspace_size(self.img_codes.numel())
        for L in self.convs:
            b = max(b, iq.iq_conv_fwd_workspace_size(L.desc, False))
            if self.train:
                b = max(b, iq.iq_conv_dgrad_workspace_size(L.desc),
                        iq.iq_conv_wgrad_workspace_size(L.desc))
        if self.skips:
            for L in self.skip_convs:
                b = max(b, iq.iq_conv_fwd_workspace_size(L.desc, False))
                if self.train:
                    b = max(b, iq.iq_conv_dgrad_workspace_size(L.desc),
                            iq.iq_conv_wgrad_workspace_size(L.desc))
            for U in self.ups:
                _, hh, ww, c = U.x.shape
                b = max(b, iq.iq_upsample_workspace_size(self.n, hh, ww, c, U.R))
            b = max(b, iq.iq_combine_workspace_size(
                [iq.term(self.sp3.a, self.sp3.s_a), iq.term(self.sp3.a, self.sp3.s_a)]))
            return b + 4096
        hs, ws_ = self.score_hw
        b = max(b, iq.iq_upsample_workspace_size(self.n, hs, ws_, self.classes, UP_R))
        return b + 4096

    # ------------------------------------------------------------------ passes

    @property
    def macs_forward(self) -> int:
        """In-bounds multiply-accumulates of the inference pass."""
        return sum(L.macs for L in self.convs + self.skip_convs) + self.up_macs

    @property
    def macs_step(self) -> int:
        """In-bounds multiply-accumulates of a training step: forward, data gradient (not for
        the first layer) and weight gradient of every conv, the decoder included."""
        return self._step(lambda L: L.macs, self.up_macs)

    @property
    def macs_step_dense(self) -> int:
        return self._step(lambda L: L.macs_dense, self.up_macs_dense)

    @property
    def macs_forward_dense(self) -> int:
        return sum(L.macs_dense for L in self.convs + self.skip_convs) + self.up_macs_dense

    def _step(self, get, up) -> int:
        f = sum(get(L) for L in self.convs + self.skip_convs)
        dg = sum(get(L) for L in self.convs + self.skip_convs if L.layer_id > 0)
        return f + dg + f + 3 * up

    def forward(self, img_u8: torch.Tensor, stream=None):
        ws = self.ws
        iq.iq_quantize_image_u8(img_u8, False, 4, self.img_codes, self.s_img, ws=ws, stream=stream)
        for item in self.layers:
            if isinstance(item, Pool):
                iq.iq_maxpool_fwd(item.x, 2, 2, 0, item.y, item.arg, y_f16=item.y16,
                                  stream=stream)
                continue
            L = item
            iq.iq_conv_fwd(L.desc, L.x, L.s_x, L.wq, L.a, L.s_a, relu=L.relu, x_f16=L.x16,
                           a_f16=L.a16, ws=ws, stream=stream)
        if self.skips:
            self._forward_fcn8s(stream)
            return
        iq.iq_upsample_fwd(self.score, self.s_score, self.up_wq, UP_R, UP_STRIDE, UP_PAD, self.z,
                           self.s_z, ws=ws, stream=stream)

    def _up_fwd(self, U, stream):
        iq.iq_upsample_fwd(U.x, U.s_x, U.wq, U.R, U.stride, U.pad, U.z, U.s_z, ws=self.ws,
                           stream=stream)

    def _sum(self, a, s_a, b, s_b, out, s_out, stream):
        """out = SQ8 of the real-valued sum of two quantized tensors of one shape."""
        n, hh, ww, c = a.shape
        iq.iq_combine([iq.term(a, s_a), iq.term(b, s_b)], n, hh * ww, c, out, s_out, ws=self.ws,
                      stream=stream)

    def _forward_fcn8s(self, stream):
        ws = self.ws
        self._up_fwd(self.up2a, stream)
        for L in (self.sp4, self.sp3):
            iq.iq_conv_fwd(L.desc, L.x, L.s_x, L.wq, L.a, L.s_a, relu=False, ws=ws,
                           stream=stream)
        self._sum(self.up2a.z, self.up2a.s_z, self.sp4.a, self.sp4.s_a, self.fuse4, self.s_fuse4,
                  stream)
        self._up_fwd(self.up2b, stream)
        self._sum(self.up2b.z, self.up2b.s_z, self.sp3.a, self.sp3.s_a, self.fuse3, self.s_fuse3,
                  stream)
        self._up_fwd(self.up8, stream)

    def backward_update(self, labels: torch.Tensor, stream=None):
        assert self.train
        ws, step, seed, lr = self.ws, self.step_count, self.seed, self.lr_log2
        iq.iq_mse_grad(self.z, self.s_z, labels, self.Ez, self.s_Ez, ws=ws, stream=stream)
        extra = {}
        if self.skips:
            extra = self._backward_fcn8s(stream)
        else:
            iq.iq_upsample_wgrad(self.score, self.s_score, self.Ez, self.s_Ez, UP_R, UP_STRIDE,
                                 UP_PAD, self.up_g, self.up_s_g, gq_mode=2, seed=seed,
                                 layer=self.up_layer_id, step=step, ws=ws, stream=stream)
            iq.iq_upsample_bwd(self.Ez, self.s_Ez, self.up_wq, self.score.shape, UP_R, UP_STRIDE,
                               UP_PAD, self.e_score, self.s_e_score, ws=ws, stream=stream)
            self._update(self.up_master, self.up_wq, self.up_g, self.up_s_g, stream)
        # error arriving at the output of the current item, walking backwards
        err, s_err = self.e_score, self.s_e_score
        npool = len(self.pools)
        items = list(reversed(self.layers))
        masked, buf = False, 0        # err already carries the ReLU mask, in e16[buf]
        for idx, item in enumerate(items):
            if isinstance(item, Pool):
                npool -= 1
                if npool in extra:        # the skip's error joins the main path's
                    ej, s_ej = self.ej[npool]
                    self._sum(err, s_err, extra[npool][0], extra[npool][1], ej, s_ej, stream)
                    err, s_err = ej, s_ej
                iq.iq_maxpool_bwd(err, s_err, item.arg, item.x.shape, 2, 2, 0, item.ex, item.s_ex,
                                  ws=ws, stream=stream)
                err, s_err = item.ex, item.s_ex
                continue
            L = item
            e16 = self.e16[buf] if L.cout % 64 == 0 else None
            if masked:
                e = err                   # the conv above applied this layer's ReLU mask
            elif L.relu:
                # the errors and, for the data and weight gradients, their fp16 copy
                iq.iq_relu_bwd(err, L.a, L.e, e_f16=e16, stream=stream)
                e = L.e
            else:
                e = err
            # the conv below, when it feeds this one directly: its ReLU backward rides on
            # this data gradient (dx masked by the input codes, which are its output), with
            # the fp16 copy for its own gradients
            below = items[idx + 1] if idx + 1 < len(items) else None
            fuse = (L.layer_id > 0 and isinstance(below, Conv) and below.relu and
                    below.a is L.x and below.cout % 64 == 0)
            if L.layer_id > 0:
                iq.iq_conv_dgrad(L.desc, e, s_err, L.wq, L.ex, L.s_ex, e_f16=e16,
                                 dx_mask=L.x if fuse else None,
                                 dx_f16=self.e16[1 - buf] if fuse else None, ws=ws,
                                 stream=stream)
            iq.iq_conv_wgrad(L.desc, e, s_err, L.x, L.s_x, L.g, L.s_g, gq_mode=2, seed=seed,
                             layer=L.layer_id, step=step, e_f16=e16, x_f16=L.x16, ws=ws,
                             stream=stream)
            self._update(L.master, L.wq, L.g, L.s_g, stream)
            if L.layer_id > 0:
                err, s_err = L.ex, L.s_ex
            L.ex_masked = fuse
            masked = fuse
            if fuse:
                buf = 1 - buf
        self.step_count += 1

    def _update(self, master, wq, g, s_g, stream):
        """Eq. (UQ2) update, then the decoupled weight decay when enabled."""
        iq.iq_update(master, wq, g, s_g, self.lr_log2, stream=stream)
        if self.wd_shift:
            iq.iq_weight_decay(master, wq, self.wd_shift, stream=stream)

    def _up_bwd(self, U, E, s_E, stream):
        """Weight gradient (GQ2), data gradient into U.ex and the update of one decoder layer."""
        ws, step, seed, lr = self.ws, self.step_count, self.seed, self.lr_log2
        iq.iq_upsample_wgrad(U.x, U.s_x, E, s_E, U.R, U.stride, U.pad, U.g, U.s_g, gq_mode=2,
                             seed=seed, layer=U.layer_id, step=step, ws=ws, stream=stream)
        iq.iq_upsample_bwd(E, s_E, U.wq, U.x.shape, U.R, U.stride, U.pad, U.ex, U.s_ex, ws=ws,
                           stream=stream)
        self._update(U.master, U.wq, U.g, U.s_g, stream)

    def _skip_bwd(self, L, e, s_e, stream):
        ws, step, seed, lr = self.ws, self.step_count, self.seed, self.lr_log2
        iq.iq_conv_wgrad(L.desc, e, s_e, L.x, L.s_x, L.g, L.s_g, gq_mode=2, seed=seed,
                         layer=L.layer_id, step=step, ws=ws, stream=stream)
        iq.iq_conv_dgrad(L.desc, e, s_e, L.wq, L.ex, L.s_ex, ws=ws, stream=stream)
        self._update(L.master, L.wq, L.g, L.s_g, stream)

    def _backward_fcn8s(self, stream):
        """The decoder's backward in the oracle's order; returns the skips' errors at the
        outputs of pool3 (2) and pool4 (3).  A sum's error reaches both operands as it is."""
        self._up_bwd(self.up8, self.Ez, self.s_Ez, stream)
        e3, s3 = self.up8.ex, self.up8.s_ex
        self._skip_bwd(self.sp3, e3, s3, stream)
        self._up_bwd(self.up2b, e3, s3, stream)
        e4, s4 = self.up2b.ex, self.up2b.s_ex
        self._skip_bwd(self.sp4, e4, s4, stream)
        self._up_bwd(self.up2a, e4, s4, stream)
        return {2: (self.sp3.ex, self.sp3.s_ex), 3: (self.sp4.ex, self.sp4.s_ex)}

    def train_step(self, img_u8, labels, stream=None):
        self.forward(img_u8, stream)
        self.backward_update(labels, stream)
