"""DeepLabv3-ResNet50 on the iq C ABI: the quantized training step and inference pass.

Network (Sec. 5): ResNet-50 at output stride 8 (stages of 3/4/6/3 bottlenecks, stages 3
and 4 dilated), ASPP (1x1, three atrous 3x3 at rates 12/24/36, image pooling), a 1x1
projection, a 3x3 head, a 1x1 classifier and x8 bilinear upsampling with aligned corners
(65 -> 513); integer L1BN after every convolution but the classifier, GQ1 gradients and a
softmax cross-entropy loss on the quantized logits.

Dataflow per layer (Sec. 3.2-3.3): W_q = UQ(W_m, 8) from 24-bit master weights; int32
convolution fused with the quantized L1BN (X codes kept for backward) + ReLU + Q_A; the
bottleneck output SQ(ReLU(gamma_q X3 + beta_q + shortcut), 8) by iq_combine from the X
codes; backward through iq_bn_int_bwd (ReLU mask of the stored output codes),
E_1 = SQ(dgrad, 8), G_q = RQ(G/Scale(G), 8) (Eq. (GQ1)), W_m -= UQ(G_q lr, 24), and the
gamma / beta masters from their gradient sums (iq_bn_update).  Errors that reach one
tensor along several paths are summed in real units and requantized (iq_combine).

Every step runs in the library's kernels; this module only allocates device memory
(torch tensors) and sequences the C ABI calls on one stream.
"""
from __future__ import annotations

import numpy as np
import torch

from . import iq
from . import synthetic as S
from .work import conv_macs

K_E2 = 16


class Layer:
    """One convolution with its parameters and forward / backward buffers."""

    def __init__(self, net, spec: S.ConvSpec, lid: int, x, s_x, w_fp32, gm, bm):
        dev = net.dev
        self.spec, self.lid, self.x, self.s_x = spec, lid, x, s_x
        n, h, w, c = x.shape
        assert c == spec.cin
        self.desc = iq.conv_desc(n, h, w, spec.cin, spec.cout, spec.r, spec.r, spec.stride,
                                 spec.pad, spec.dil)
        p, q = iq.iq_conv_out_size(self.desc)
        self.out_shape = (n, p, q, spec.cout)
        self.x16 = None
        self.a16 = None        # the next layer's x16 when that layer reads a: written here
        self.master = net.master(w_fp32)
        self.wq = torch.empty((spec.cout, spec.r, spec.r, spec.cin), dtype=torch.int8, device=dev)
        iq.iq_weight_requant(self.master, self.wq)
        self.a = torch.empty(self.out_shape, dtype=torch.int8, device=dev)
        self.s_a = net.scal()
        # in-bounds and dense multiply-accumulates of one pass (the stem's fourth input
        # channel is the zero RGB padding: no work)
        self.macs, self.macs_dense = conv_macs(n, h, w, 3 if spec.cin == 4 else spec.cin,
                                               spec.cout, spec.r, spec.stride, spec.pad,
                                               spec.dil)
        if spec.bn:
            self.gm = torch.from_numpy(gm).to(dev)
            self.bm = torch.from_numpy(bm).to(dev)
            self.gamma = torch.empty(spec.cout, dtype=torch.int32, device=dev)
            self.beta = torch.empty(spec.cout, dtype=torch.int32, device=dev)
            g8 = torch.empty(spec.cout, dtype=torch.int8, device=dev)
            iq.iq_weight_requant(self.gm, g8)
            self.gamma.copy_(g8)
            iq.iq_weight_requant(self.bm, g8)
            self.beta.copy_(g8)
            self.X = torch.empty(self.out_shape, dtype=torch.int16, device=dev)
            self.bn_codes = torch.empty(2 * spec.cout, dtype=torch.int32, device=dev)
            self.bn_scales = torch.zeros(iq.IQ_BN_SCALES, dtype=torch.float64, device=dev)
        if net.train:
            self.e = torch.empty(self.out_shape, dtype=torch.int8, device=dev)
            self.s_e = net.scal()
            self.g = torch.empty_like(self.wq)
            self.s_g = net.scal()
            self.ex = torch.empty(x.shape, dtype=torch.int8, device=dev)
            self.s_ex = net.scal()
            if spec.bn:
                self.dgamma = torch.empty(spec.cout, dtype=torch.int64, device=dev)
                self.dbeta = torch.empty(spec.cout, dtype=torch.int64, device=dev)

    @property
    def s_X(self) -> int:
        """Device address of the X codes' scale (bn_scales[IQ_BN_S_XHAT])."""
        return self.bn_scales.data_ptr() + 8 * iq.IQ_BN_S_XHAT

    def ws_bytes(self, train: bool) -> int:
        b = iq.iq_conv_fwd_workspace_size(self.desc, self.spec.bn)
        if train:
            n, p, q, k = self.out_shape
            b = max(b, iq.iq_conv_dgrad_workspace_size(self.desc),
                    iq.iq_conv_wgrad_workspace_size(self.desc),
                    iq.iq_bn_int_workspace_size(n * p * q, k) if self.spec.bn else 0,
                    4096 + 2 * k + 256)
        return b

    def forward(self, ws, stream):
        if self.spec.bn:
            iq.iq_conv_fwd(self.desc, self.x, self.s_x, self.wq, self.a, self.s_a, self.gamma,
                           self.beta, use_bn=True, relu=True, xhat=self.X, bn_codes=self.bn_codes,
                           bn_scales=self.bn_scales, x_f16=self.x16, a_f16=self.a16, ws=ws,
                           stream=stream)
        else:
            iq.iq_conv_fwd(self.desc, self.x, self.s_x, self.wq, self.a, self.s_a, relu=False,
                           x_f16=self.x16, a_f16=self.a16, ws=ws, stream=stream)

    def backward(self, net, e_a, s_ea, mask=None, need_dx=True, stream=None):
        """From the error of the output codes (before the ReLU mask) to the error of the
        input, with the weight and gamma / beta updates of this layer."""
        ws, step, seed, lr = net.ws, net.step_count, net.seed, net.lr_log2
        e16 = net.e16 if need_dx and self.spec.cout % 64 == 0 else None
        if self.spec.bn:
            # the errors and their fp16 copy for this layer's data and weight gradients
            # (the descriptor carries IQ_CONV_E_F16_READY)
            iq.iq_bn_int_bwd(e_a, s_ea, self.a if mask is None else mask, self.X, self.gamma,
                             self.bn_codes, self.bn_scales, self.e, self.s_e, self.dgamma,
                             self.dbeta, k_e2=K_E2, e_f16=e16, ws=ws, stream=stream)
            e, s_e = self.e, self.s_e
        else:
            e, s_e = e_a, s_ea
        if need_dx:
            iq.iq_conv_dgrad(self.desc, e, s_e, self.wq, self.ex, self.s_ex, e_f16=e16, ws=ws,
                             stream=stream)
        iq.iq_conv_wgrad(self.desc, e, s_e, self.x, self.s_x, self.g, self.s_g, gq_mode=1,
                         seed=seed, layer=self.lid, step=step, e_f16=e16, x_f16=self.x16, ws=ws,
                         stream=stream)
        iq.iq_update(self.master, self.wq, self.g, self.s_g, lr, stream=stream)
        if self.spec.bn:
            iq.iq_bn_update(self.gm, self.bm, self.gamma, self.beta, self.dgamma, self.dbeta,
                            s_ea, self.bn_scales, lr, seed, self.lid, step, ws=ws, stream=stream)
        return self.ex, self.s_ex


class DeepLabV3R50:
    """Preallocated DeepLabv3-ResNet50 for a fixed batch shape (h, w = 8k + 1).

    width scales every channel count (1.0 = the paper's network); tests use small widths."""

    def __init__(self, n: int, h: int, w: int, classes: int = 21, width: float = 1.0,
                 seed: int = 0, lr_log2: int = 10, device: str = "cuda", train: bool = True,
                 blocks=(3, 4, 6, 3)):
        assert (h - 1) % 8 == 0 and (w - 1) % 8 == 0, "output stride 8 needs h, w = 8k + 1"
        self.n, self.h, self.w, self.classes = n, h, w, classes
        self.dev = torch.device(device)
        self.lr_log2, self.seed, self.train, self.step_count = lr_log2, seed, train, 0
        self.spec = sp = S.deeplabv3_r50_spec(classes, width, blocks)
        ws_fp32, gms, bms = S.deeplabv3_r50_init(seed, sp)
        specs = sp.convs()
        lid = {cv.name: i for i, cv in enumerate(specs)}
        dev = self.dev
        self.layers = {}

        def conv(cv, x, s_x):
            i = lid[cv.name]
            L = Layer(self, cv, i, x, s_x, ws_fp32[i], gms[i], bms[i])
            self.layers[cv.name] = L
            return L

        self.img = torch.empty((n, h, w, 4), dtype=torch.int8, device=dev)
        self.s_img = self.scal()
        self.stem = conv(sp.stem, self.img, self.s_img)
        _, hs, wsd, cs = self.stem.out_shape
        hp, wp = (hs + 2 - 3) // 2 + 1, (wsd + 2 - 3) // 2 + 1
        self.pool = torch.empty((n, hp, wp, cs), dtype=torch.int8, device=dev)
        self.pool_arg = torch.empty((n, hp, wp, cs), dtype=torch.uint8, device=dev)
        x, s = self.pool, self.stem.s_a
        self.blocks = []
        for b in sp.blocks:
            l1 = conv(b.conv1, x, s)
            l2 = conv(b.conv2, l1.a, l1.s_a)
            l3 = conv(b.conv3, l2.a, l2.s_a)
            ld = conv(b.down, x, s) if b.down else None
            out = torch.empty(l3.out_shape, dtype=torch.int8, device=dev)
            s_out = self.scal()
            blk = {"spec": b, "l1": l1, "l2": l2, "l3": l3, "down": ld, "x": x, "s_x": s,
                   "out": out, "s_out": s_out}
            if train:
                blk["e_sc"] = torch.empty(l3.out_shape, dtype=torch.int8, device=dev)
                blk["e_in"] = torch.empty(x.shape, dtype=torch.int8, device=dev)
                blk["s_e_in"] = self.scal()
            self.blocks.append(blk)
            x, s = out, s_out
        self.c4, self.s_c4 = x, s
        n_, hh, ww, c4 = x.shape
        self.hw4 = hh * ww
        self.aspp = [conv(cv, x, s) for cv in sp.aspp]
        a = sp.pool_conv.cout
        self.pooled = torch.empty((n, 1, 1, c4), dtype=torch.int8, device=dev)
        self.s_pooled = self.scal()
        self.pconv = conv(sp.pool_conv, self.pooled, self.s_pooled)
        nb = len(sp.aspp) + 1
        self.cat = torch.empty((n, hh, ww, nb * a), dtype=torch.int8, device=dev)
        self.s_cat = self.scal()
        self.project = conv(sp.project, self.cat, self.s_cat)
        self.head = conv(sp.head, self.project.a, self.project.s_a)
        self.cls = conv(sp.cls, self.head.a, self.head.s_a)
        self.z = torch.empty((n, h, w, classes), dtype=torch.int8, device=dev)
        self.s_z = self.scal()
        if train:
            self.E = torch.empty_like(self.z)
            self.s_E = self.scal()
            self.n_valid = torch.zeros(1, dtype=torch.int64, device=dev)
            self.e_cls = torch.empty(self.cls.out_shape, dtype=torch.int8, device=dev)
            self.s_e_cls = self.scal()
            self.e_branch = [torch.empty(L.out_shape, dtype=torch.int8, device=dev)
                             for L in self.aspp]
            self.e_pool = torch.empty((n, 1, 1, a), dtype=torch.int8, device=dev)
            self.s_e_pool = self.scal()
            self.s_e_pooled_px = self.scal()
            self.e_c4 = torch.empty_like(self.c4)
            self.s_e_c4 = self.scal()
            self.e_stem = torch.empty(self.stem.out_shape, dtype=torch.int8, device=dev)
            self.s_e_stem = self.scal()
        # fp16 copies of the codes the tensor-core kernels read: one per distinct conv input,
        # written by the layer whose output codes it is (a layer's requantization writes its
        # successor's copy: conv1 -> conv2 -> conv3 of a block, project -> head -> cls), by
        # the stem's max pool, by the join that produces it (block outputs, the ASPP
        # concatenation), or else by the forward of the first layer (in forward order) that
        # reads it; read as it is by the others (IQ_CONV_X_F16_READY: the ASPP
        # branches, a block's first conv and its projection shortcut) and by the weight
        # gradients.  One error buffer: written with the errors by a BN layer's backward,
        # read by its data and weight gradients (IQ_CONV_E_F16_READY)
        x16, e16 = {}, 0
        producer = {L.a.data_ptr(): L for L in self.layers.values()}
        joins = {blk["out"].data_ptr() for blk in self.blocks} | {self.cat.data_ptr()}
        self.pool16, self.join16 = None, {}
        for L in self.layers.values():
            if L.spec.cin % 64 == 0 and L.x.numel() % 16 == 0:
                key = L.x.data_ptr()
                if key not in x16:
                    x16[key] = torch.empty(L.x.numel(), dtype=torch.float16, device=dev)
                    P = producer.get(key)
                    if P is not None:
                        P.a16 = x16[key]
                        L.desc.flags |= iq.IQ_CONV_X_F16_READY
                    elif key == self.pool.data_ptr():
                        self.pool16 = x16[key]
                        L.desc.flags |= iq.IQ_CONV_X_F16_READY
                    elif key in joins:
                        self.join16[key] = x16[key]
                        L.desc.flags |= iq.IQ_CONV_X_F16_READY
                else:
                    L.desc.flags |= iq.IQ_CONV_X_F16_READY
                L.x16 = x16[key]
            if L.spec.cout % 64 == 0:
                e16 = max(e16, L.a.numel())
                if L.spec.bn:
                    L.desc.flags |= iq.IQ_CONV_E_F16_READY
        if train:
            self.e16 = torch.empty(max(e16, 16), dtype=torch.float16, device=dev)
        self.ws = torch.empty(self._ws_bytes(), dtype=torch.uint8, device=dev)

    # ------------------------------------------------------------------ helpers

    def scal(self):
        return torch.zeros(1, dtype=torch.float64, device=self.dev)

    def master(self, w_fp32: np.ndarray) -> torch.Tensor:
        """Master weights W_m = UQ(W, 24) (Eq. (WQ0)) computed on the device."""
        w = torch.from_numpy(np.ascontiguousarray(w_fp32)).to(self.dev)
        m = torch.empty(w.shape, dtype=torch.int32, device=self.dev)
        iq.iq_quantize(w, 24, iq.IQ_MODE_UQ, m, self.scal())
        return m

    def _res_terms(self, blk):
        l3, ld = blk["l3"], blk["down"]
        t = [iq.term(l3.X, l3.s_X, gamma=l3.gamma, beta=l3.beta)]
        if ld is not None:
            t.append(iq.term(ld.X, ld.s_X, gamma=ld.gamma, beta=ld.beta))
        else:
            t.append(iq.term(blk["x"], blk["s_x"]))
        return t

    def _cat_terms(self):
        a = self.spec.pool_conv.cout
        t = [iq.term(L.a, L.s_a, k * a) for k, L in enumerate(self.aspp)]
        t.append(iq.term(self.pconv.a, self.pconv.s_a, len(self.aspp) * a, bcast=True))
        return t

    def _ws_bytes(self) -> int:
        n = self.n
        b = iq.iq_quantize_workspace_size(self.img.numel())
        for L in self.layers.values():
            b = max(b, L.ws_bytes(self.train))
        for blk in self.blocks:
            b = max(b, iq.iq_combine_workspace_size(self._res_terms(blk)))
        b = max(b, iq.iq_combine_workspace_size(self._cat_terms()))
        # the sum of the errors reaching the ASPP input: one operand per branch
        err_terms = [iq.term(self.c4, self.s_c4)] * (len(self.aspp) + 1)
        b = max(b, iq.iq_combine_workspace_size(err_terms))
        b = max(b, iq.iq_spatial_sum_workspace_size(n, self.c4.shape[-1]))
        _, hc, wc, cc = self.cls.out_shape
        b = max(b, iq.iq_bilinear_workspace_size(n, hc, wc, cc), 4096)
        if self.train:
            b = max(b, self.stem.a.numel() * 4 + 4096)
        return b + 4096

    # ------------------------------------------------------------------ passes

    @property
    def macs_forward(self) -> int:
        """In-bounds multiply-accumulates of the inference pass."""
        return sum(L.macs for L in self.layers.values())

    @property
    def macs_step(self) -> int:
        """In-bounds multiply-accumulates of a training step: forward, data gradient (not for
        the stem) and weight gradient of every conv."""
        f = self.macs_forward
        return f + (f - self.stem.macs) + f

    @property
    def macs_forward_dense(self) -> int:
        return sum(L.macs_dense for L in self.layers.values())

    @property
    def macs_step_dense(self) -> int:
        f = self.macs_forward_dense
        return f + (f - self.stem.macs_dense) + f

    def forward(self, img_u8: torch.Tensor, stream=None):
        ws = self.ws
        n = self.n
        iq.iq_quantize_image_u8(img_u8, False, 4, self.img, self.s_img, ws=ws, stream=stream)
        self.stem.forward(ws, stream)
        iq.iq_maxpool_fwd(self.stem.a, 3, 2, 1, self.pool, self.pool_arg, y_f16=self.pool16,
                          stream=stream)
        for blk in self.blocks:
            for key in ("l1", "l2", "l3", "down"):
                if blk[key] is not None:
                    blk[key].forward(ws, stream)
            out = blk["out"]
            _, hh, ww, c = out.shape
            iq.iq_combine(self._res_terms(blk), n, hh * ww, c, out, blk["s_out"], relu=True,
                          out_f16=self.join16.get(out.data_ptr()), ws=ws, stream=stream)
        for L in self.aspp:
            L.forward(ws, stream)
        iq.iq_spatial_sum(self.c4, self.s_c4, self.pooled.view(n, -1), self.s_pooled, mean=True,
                          ws=ws, stream=stream)
        self.pconv.forward(ws, stream)
        iq.iq_combine(self._cat_terms(), n, self.hw4, self.cat.shape[-1], self.cat, self.s_cat,
                      out_f16=self.join16.get(self.cat.data_ptr()),
                      concat=True, ws=ws, stream=stream)
        for L in (self.project, self.head, self.cls):
            L.forward(ws, stream)
        iq.iq_bilinear_up_fwd(self.cls.a, self.cls.s_a, self.spec.up, self.z, self.s_z, ws=ws,
                              stream=stream)

    def backward_update(self, labels: torch.Tensor, stream=None):
        assert self.train
        ws, n = self.ws, self.n
        iq.iq_ce_grad(self.z, self.s_z, labels, self.E, self.s_E, n_valid=self.n_valid, ws=ws,
                      stream=stream)
        iq.iq_bilinear_up_bwd(self.E, self.s_E, self.spec.up, self.cls.out_shape, self.e_cls,
                              self.s_e_cls, ws=ws, stream=stream)
        e, s = self.cls.backward(self, self.e_cls, self.s_e_cls, stream=stream)
        e, s = self.head.backward(self, e, s, stream=stream)
        e_cat, s_cat = self.project.backward(self, e, s, stream=stream)
        a = self.spec.pool_conv.cout
        terms = []
        for k, L in enumerate(self.aspp):
            iq.iq_channel_slice(e_cat, k * a, a, self.e_branch[k], stream=stream)
            ex, sx = L.backward(self, self.e_branch[k], s_cat, stream=stream)
            terms.append(iq.term(ex, sx))
        iq.iq_spatial_sum(e_cat, s_cat, self.e_pool.view(n, a), self.s_e_pool, mean=False,
                          c_off=len(self.aspp) * a, c=a, ws=ws, stream=stream)
        ep, sp = self.pconv.backward(self, self.e_pool, self.s_e_pool, stream=stream)
        iq.iq_avgpool_bwd(ep.view(n, -1), sp, self.hw4, self.s_e_pooled_px, stream=stream)
        terms.append(iq.term(ep.view(n, -1), self.s_e_pooled_px, bcast=True))
        iq.iq_combine(terms, n, self.hw4, self.c4.shape[-1], self.e_c4, self.s_e_c4, ws=ws,
                      stream=stream)
        e, s = self.e_c4, self.s_e_c4
        for blk in reversed(self.blocks):
            out = blk["out"]
            l1, l2, l3, ld = blk["l1"], blk["l2"], blk["l3"], blk["down"]
            e2, s2 = l3.backward(self, e, s, mask=out, stream=stream)
            e1, s1 = l2.backward(self, e2, s2, stream=stream)
            e0, s0 = l1.backward(self, e1, s1, stream=stream)
            t = [iq.term(e0, s0)]
            if ld is not None:
                ed, sd = ld.backward(self, e, s, mask=out, stream=stream)
                t.append(iq.term(ed, sd))
            else:
                iq.iq_relu_bwd(e, out, blk["e_sc"], stream=stream)
                t.append(iq.term(blk["e_sc"], s))
            x = blk["x"]
            _, hh, ww, c = x.shape
            iq.iq_combine(t, n, hh * ww, c, blk["e_in"], blk["s_e_in"], ws=ws, stream=stream)
            e, s = blk["e_in"], blk["s_e_in"]
        iq.iq_maxpool_bwd(e, s, self.pool_arg, self.stem.a.shape, 3, 2, 1, self.e_stem,
                          self.s_e_stem, ws=ws, stream=stream)
        self.stem.backward(self, self.e_stem, self.s_e_stem, need_dx=False, stream=stream)
        self.step_count += 1

    def train_step(self, img_u8, labels, stream=None):
        self.forward(img_u8, stream)
        self.backward_update(labels, stream)
