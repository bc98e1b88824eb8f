"""FCN-VGG16 training step composed from the CPU oracle -- TEST INFRASTRUCTURE.

Only tests/, the smoke check and bench.py's cpu_baseline / reference legs use it.
It follows the paper's dataflow one step after the other (Sec. 3.2-3.3, Sec. 5 FCN:
no BN, GQ2, MSE loss), each step a call into iq_oracle.c:

  image -> Q_A (pixel/255, SQ 8)
  per conv: W_q = UQ(W_m, 8); acc = conv; A = SQ(ReLU(acc), 8) (score layer: SQ(acc, 8))
  pools: max on codes
  decoder: per-class transposed conv (the adjoint of a stride-32 grouped conv), SQ 8;
    or FCN8s (Sec. 2.1): 1x1 score convs on pool4 / pool3, x2, x2 and x8 per-class
    transposed convs (bilinear-initialised, trainable), each skip joined by a real-valued
    sum requantized with SQ 8
  loss: E = SQ(z s_z - onehot, 8)
  backward per conv: e = e_A [A > 0]; E_1 = SQ(dgrad, 8); G_q = RQ(G / Scale(G), 8) (GQ2);
  update W_m <- Clip(W_m - UQ(G_q lr, 24)).
"""
from __future__ import annotations

import numpy as np

from . import (CombineTerm, Conv, combine, conv_dgrad, conv_fwd, conv_wgrad, maxpool_bwd,
               maxpool_fwd, mse_grad, quantize_image_u8, relu_bwd, requant_master, rq_int,
               sq_int, update, uq, weight_decay)

UP_R, UP_STRIDE, UP_PAD = 64, 32, 16
# FCN8s: x2 (kernel 4, stride 2, padding 1) and x8 (kernel 16, stride 8, padding 4)
UP2 = (4, 2, 1)
UP8 = (16, 8, 4)


class OracleFcn:
    """State of the oracle network: master weights (k_U = 24 codes) per conv and decoder."""

    def __init__(self, channels, weights_fp32, up_fp32, classes: int, seed: int = 0,
                 lr_log2: int = 10, skips=None, wd_shift: int = 0):
        """skips: None for the 32x decoder, else the FCN8s initial weights (score_pool4,
        score_pool3 KRSC filters; x2 and x8 per-class filters)."""
        self.channels = channels
        self.masters = [uq(w, 24) for w in weights_fp32]            # Eq. (WQ0)
        self.up_master = uq(up_fp32, 24)
        self.classes = classes
        self.seed = seed
        self.lr_log2 = lr_log2
        self.step = 0
        self.wd_shift = wd_shift      # decoupled L2 weight decay, step 2^-wd_shift (0: none)
        self.skips = skips is not None
        if self.skips:
            w4, w3, up2, up8 = skips
            self.sp4_master, self.sp3_master = uq(w4, 24), uq(w3, 24)
            self.up2a_master, self.up2b_master = uq(up2, 24), uq(up2, 24)
            self.up8_master = uq(up8, 24)
        # layer ids of the decoder layers (the Philox key of their gradients' rounding)
        L = sum(1 for c in channels if c[0] != "pool")
        self.lid = {"up": L, "up8": L, "up2b": L + 1, "up2a": L + 2, "sp4": L + 3, "sp3": L + 4}

    def _upd(self, master, gq, s_g, lr):
        """Eq. (UQ2), then the decoupled weight decay when enabled: the new master."""
        m, _ = update(master, gq, s_g, lr)
        if self.wd_shift:
            m, _ = weight_decay(m, self.wd_shift)
        return m

    # ------------------------------------------------------------------ decoder pieces

    def _up(self, x, s, master, R, stride, pad):
        """Per-class transposed convolution (the adjoint of a grouped stride conv), SQ 8."""
        n, hh, ww, c = x.shape
        wq = requant_master(master, 24, 8).astype(np.int8)
        cvu = Conv(n, (hh - 1) * stride - 2 * pad + R, (ww - 1) * stride - 2 * pad + R, c, c,
                   R, R, stride, pad, 1, c)
        zacc = conv_dgrad(cvu, x, wq.reshape(c, R, R, 1))
        z, s_z = sq_int(zacc, s * 2.0 ** -7, 8)
        return (cvu, x, s, wq, zacc, z.astype(np.int8), s_z)

    def _up_bwd(self, up, E, s_E, layer):
        """Its raw and GQ2 weight gradient and its data gradient; returns (G, gq, s_g, e, s_e)."""
        cvu, x, s, wq, _, _, _ = up
        c, R = cvu.c, cvu.r
        G = conv_wgrad(cvu, x, E).reshape(c, R, R)
        gq, s_g = rq_int(G, s * s_E, 8, 2, self.seed, layer, self.step, 0)
        ex = conv_fwd(cvu, E, wq.reshape(c, R, R, 1))
        err, s_err = sq_int(ex, s_E * 2.0 ** -7, 8)
        return G, gq, s_g, err.astype(np.int8), s_err

    def _skip(self, x, s, master):
        """A 1x1 score conv on a pool output (no ReLU), SQ 8."""
        n, hh, ww, cin = x.shape
        wq = requant_master(master, 24, 8).astype(np.int8)
        cv = Conv(n, hh, ww, cin, self.classes, 1, 1, 1, 0)
        acc = conv_fwd(cv, x, wq)
        a, s_a = sq_int(acc, s * 2.0 ** -7, 8)
        return (cv, x, s, wq, acc, a.astype(np.int8), s_a)

    def _skip_bwd(self, sk, e, s_e, layer):
        cv, x, s, wq, _, _, _ = sk
        G = conv_wgrad(cv, e, x)
        gq, s_g = rq_int(G, s_e * s, 8, 2, self.seed, layer, self.step, 0)
        dx = conv_dgrad(cv, e, wq)
        ex, s_ex = sq_int(dx, s_e * 2.0 ** -7, 8)
        return G, gq, s_g, ex.astype(np.int8), s_ex

    @staticmethod
    def _sum(a, s_a, b, s_b):
        """Real-valued sum of two quantized tensors of one shape, then SQ 8."""
        n, hh, ww, c = a.shape
        z, s_z = combine([CombineTerm(a.reshape(n, hh * ww, c), s_a),
                          CombineTerm(b.reshape(n, hh * ww, c), s_b)], n, hh * ww, c)
        return z.reshape(n, hh, ww, c), s_z

    def forward(self, img_u8):
        """Returns the trace of every intermediate (dict), the logits codes and scale."""
        n, h, w, _ = img_u8.shape
        x, s = quantize_image_u8(img_u8, 4)
        tr = {"img": (x, s), "layers": []}
        hh, ww = h, w
        li = 0
        pools = []
        for name, cin, cout, r, pad, relu in self.channels:
            if name == "pool":
                y, arg = maxpool_fwd(x, 2, 2, 0)
                tr["layers"].append(("pool", x, s, y, arg))
                pools.append((y, s))
                x = y
                hh, ww = hh // 2, ww // 2
                continue
            wq = requant_master(self.masters[li], 24, 8).astype(np.int8)      # Eq. (WQ1)
            cv = Conv(n, hh, ww, cin, cout, r, r, 1, pad)
            acc = conv_fwd(cv, x, wq)
            a, s_a = sq_int(acc, s * 2.0 ** -7, 8, relu)                      # Eq. (AQ1)
            tr["layers"].append(("conv", li, cv, x, s, wq, acc, a.astype(np.int8), s_a, relu))
            x, s = a.astype(np.int8), s_a
            li += 1
        if not self.skips:
            tr["up"] = self._up(x, s, self.up_master, UP_R, UP_STRIDE, UP_PAD)
            return tr
        # FCN8s: score (1/32) -x2-> + score_pool4 (1/16) -x2-> + score_pool3 (1/8) -x8->
        tr["up2a"] = self._up(x, s, self.up2a_master, *UP2)
        tr["sp4"] = self._skip(*pools[3], self.sp4_master)
        tr["fuse4"] = self._sum(tr["up2a"][5], tr["up2a"][6], tr["sp4"][5], tr["sp4"][6])
        tr["up2b"] = self._up(*tr["fuse4"], self.up2b_master, *UP2)
        tr["sp3"] = self._skip(*pools[2], self.sp3_master)
        tr["fuse3"] = self._sum(tr["up2b"][5], tr["up2b"][6], tr["sp3"][5], tr["sp3"][6])
        tr["up"] = self._up(*tr["fuse3"], self.up8_master, *UP8)
        return tr

    def backward_update(self, tr, labels):
        seed, step, lr = self.seed, self.step, self.lr_log2
        z, s_z = tr["up"][5], tr["up"][6]
        E, s_E = mse_grad(z, s_z, labels)
        out = {"E": (E, s_E)}
        extra = {}      # pool index -> the skip branch's error at that pool's output
        if not self.skips:
            G, gq, s_g, err, s_err = self._up_bwd(tr["up"], E, s_E, self.lid["up"])
            out["up_g"] = (G, gq, s_g)
            self.up_master = self._upd(self.up_master, gq, s_g, lr)
        else:
            # a sum's error reaches both of its operands unchanged
            G, gq, s_g, e3, s3 = self._up_bwd(tr["up"], E, s_E, self.lid["up8"])
            out["up8_g"] = (G, gq, s_g)
            out["e_fuse3"] = (e3, s3)
            self.up8_master = self._upd(self.up8_master, gq, s_g, lr)
            G, gq, s_g, ep3, sp3 = self._skip_bwd(tr["sp3"], e3, s3, self.lid["sp3"])
            out["sp3_g"] = (G, gq, s_g)
            out["e_sp3"] = (ep3, sp3)
            self.sp3_master = self._upd(self.sp3_master, gq, s_g, lr)
            extra[2] = (ep3, sp3)
            G, gq, s_g, e4, s4 = self._up_bwd(tr["up2b"], e3, s3, self.lid["up2b"])
            out["up2b_g"] = (G, gq, s_g)
            out["e_fuse4"] = (e4, s4)
            self.up2b_master = self._upd(self.up2b_master, gq, s_g, lr)
            G, gq, s_g, ep4, sp4 = self._skip_bwd(tr["sp4"], e4, s4, self.lid["sp4"])
            out["sp4_g"] = (G, gq, s_g)
            out["e_sp4"] = (ep4, sp4)
            self.sp4_master = self._upd(self.sp4_master, gq, s_g, lr)
            extra[3] = (ep4, sp4)
            G, gq, s_g, err, s_err = self._up_bwd(tr["up2a"], e4, s4, self.lid["up2a"])
            out["up2a_g"] = (G, gq, s_g)
            self.up2a_master = self._upd(self.up2a_master, gq, s_g, lr)
        out["e_score"] = (err, s_err)
        out["grads"] = {}
        npool = sum(1 for it in tr["layers"] if it[0] == "pool")
        for item in reversed(tr["layers"]):
            if item[0] == "pool":
                npool -= 1
                if npool in extra:        # the skip's error joins the main path's
                    err, s_err = self._sum(err, s_err, *extra[npool])
                    out.setdefault("e_pool", {})[npool] = (err, s_err)
                _, x, s_x, y, arg = item
                sums = maxpool_bwd(err, arg, x.shape, 2, 2, 0)
                err = sums.astype(np.int8)           # non-overlapping: codes pass through
                continue
            _, li, cv, x, s_x, wq, acc, a, s_a, relu = item
            e = relu_bwd(err, a) if relu else err
            G = conv_wgrad(cv, e, x)
            gq, s_g = rq_int(G, s_err * s_x, 8, 2, seed, li, step, 0)
            out["grads"][li] = (G, gq, s_g)
            if li > 0:
                dx = conv_dgrad(cv, e, wq)
                nerr, ns = sq_int(dx, s_err * 2.0 ** -7, 8)
                out.setdefault("ex", {})[li] = (nerr.astype(np.int8), ns)
            self.masters[li] = self._upd(self.masters[li], gq, s_g, lr)
            if li > 0:
                err, s_err = nerr.astype(np.int8), ns
        self.step += 1
        return out
