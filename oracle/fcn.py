"""FCN-VGG16 training step composed from the CPU oracle -- TEST INFRASTRUCTURE.

Only tests/, the smoke check and bench.py's cpu_baseline / reference legs use it.
It follows the paper's dataflow one step after the other (Sec. 3.2-3.3, Sec. 5 FCN:
no BN, GQ2, MSE loss), each step a call into iq_oracle.c:

  image -> Q_A (pixel/255, SQ 8)
  per conv: W_q = UQ(W_m, 8); acc = conv; A = SQ(ReLU(acc), 8) (score layer: SQ(acc, 8))
  pools: max on codes
  decoder: per-class transposed conv (the adjoint of a stride-32 grouped conv), SQ 8
  loss: E = SQ(z s_z - onehot, 8)
  backward per conv: e = e_A [A > 0]; E_1 = SQ(dgrad, 8); G_q = RQ(G / Scale(G), 8) (GQ2);
  update W_m <- Clip(W_m - UQ(G_q lr, 24)).
"""
from __future__ import annotations

import numpy as np

from . import (Conv, conv_dgrad, conv_fwd, conv_wgrad, maxpool_bwd, maxpool_fwd, mse_grad,
               quantize_image_u8, relu_bwd, requant_master, rq_int, sq_int, update, uq)

UP_R, UP_STRIDE, UP_PAD = 64, 32, 16


class OracleFcn:
    """State of the oracle network: master weights (k_U = 24 codes) per conv and decoder."""

    def __init__(self, channels, weights_fp32, up_fp32, classes: int, seed: int = 0,
                 lr_log2: int = 10):
        self.channels = channels
        self.masters = [uq(w, 24) for w in weights_fp32]            # Eq. (WQ0)
        self.up_master = uq(up_fp32, 24)
        self.classes = classes
        self.seed = seed
        self.lr_log2 = lr_log2
        self.step = 0

    def forward(self, img_u8):
        """Returns the trace of every intermediate (dict), the logits codes and scale."""
        n, h, w, _ = img_u8.shape
        x, s = quantize_image_u8(img_u8, 4)
        tr = {"img": (x, s), "layers": []}
        hh, ww = h, w
        li = 0
        for name, cin, cout, r, pad, relu in self.channels:
            if name == "pool":
                y, arg = maxpool_fwd(x, 2, 2, 0)
                tr["layers"].append(("pool", x, s, y, arg))
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
        up_wq = requant_master(self.up_master, 24, 8).astype(np.int8)
        H = (hh - 1) * UP_STRIDE - 2 * UP_PAD + UP_R
        cvu = Conv(n, H, (ww - 1) * UP_STRIDE - 2 * UP_PAD + UP_R, self.classes, self.classes,
                   UP_R, UP_R, UP_STRIDE, UP_PAD, 1, self.classes)
        zacc = conv_dgrad(cvu, x, up_wq.reshape(self.classes, UP_R, UP_R, 1))
        z, s_z = sq_int(zacc, s * 2.0 ** -7, 8)
        tr["up"] = (cvu, x, s, up_wq, zacc, z.astype(np.int8), s_z)
        return tr

    def backward_update(self, tr, labels):
        seed, step, lr = self.seed, self.step, self.lr_log2
        cvu, score, s_score, up_wq, _, z, s_z = tr["up"]
        E, s_E = mse_grad(z, s_z, labels)
        out = {"E": (E, s_E)}
        up_layer = sum(1 for c in self.channels if c[0] != "pool")
        G = conv_wgrad(cvu, score, E).reshape(self.classes, UP_R, UP_R)
        gq, s_g = rq_int(G, s_score * s_E, 8, 2, seed, up_layer, step, 0)
        out["up_g"] = (G, gq, s_g)
        ex = conv_fwd(cvu, E, up_wq.reshape(self.classes, UP_R, UP_R, 1))
        err, s_err = sq_int(ex, s_E * 2.0 ** -7, 8)
        err = err.astype(np.int8)
        out["e_score"] = (err, s_err)
        self.up_master, _ = update(self.up_master, gq, s_g, lr)
        out["grads"] = {}
        for item in reversed(tr["layers"]):
            if item[0] == "pool":
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
            self.masters[li], _ = update(self.masters[li], gq, s_g, lr)
            if li > 0:
                err, s_err = nerr.astype(np.int8), ns
        self.step += 1
        return out
