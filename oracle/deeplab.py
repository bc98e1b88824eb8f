"""DeepLabv3-ResNet50 training step composed from the CPU oracle -- TEST INFRASTRUCTURE.

Only tests/, the smoke check and bench.py's cpu_baseline / reference legs use it.  It
follows the paper's dataflow (Sec. 3.2-3.3; Sec. 5: DeepLabv3 with integer BN, GQ1, and
a cross-entropy loss) one step after the other, each step a call into iq_oracle.c:

  image -> Q_A (pixel/255, SQ 8)
  per conv: W_q = UQ(W_m, 8); acc = conv; with BN: the quantized L1BN (X codes, A codes)
  bottleneck output: SQ(ReLU(gamma_q X3 + beta_q + shortcut), 8), the shortcut being the
      block input or gamma_q Xd + beta_q of the projection
  ASPP: four conv branches, global mean -> 1x1 conv (BN over the batch), concatenation
      in real units -> SQ 8, 1x1 projection; 3x3 head; 1x1 classifier (SQ 8, no ReLU)
  logits: bilinear x8 with aligned corners -> SQ 8;  loss: softmax CE gradient -> SQ 8
  backward: BN backward (ReLU mask of the stored output codes), E_1 = SQ(dgrad, 8),
      G_q = RQ(G / Scale(G), 8) (GQ1), W_m <- Clip(W_m - UQ(G_q lr, 24)); gamma / beta
      from their gradient sums with GQ1 on the x2 grid; errors that reach one tensor
      along several paths are summed in real units -> SQ 8.
"""
from __future__ import annotations

import numpy as np

from . import (CombineTerm, Conv, bilinear_up, bilinear_up_bwd, bn_bwd, bn_fwd, ce_grad,
               combine, conv_dgrad, conv_fwd, conv_wgrad, maxpool_bwd, maxpool_fwd,
               quantize_image_u8, relu_bwd, requant_master, rq_int, spatial_sum, sq_int, update,
               uq)

K_E2 = 16


class OracleDeepLab:
    """State of the oracle network: master weights (k_U = 24) and gamma / beta masters."""

    def __init__(self, spec, weights_fp32, gamma_masters, beta_masters, seed: int = 0,
                 lr_log2: int = 10):
        self.spec = spec
        self.convs = spec.convs()
        self.lid = {cv.name: i for i, cv in enumerate(self.convs)}
        self.masters = [uq(w, 24) for w in weights_fp32]                 # Eq. (WQ0)
        self.gm = [None if g is None else np.array(g, np.int32) for g in gamma_masters]
        self.bm = [None if b is None else np.array(b, np.int32) for b in beta_masters]
        self.seed, self.lr_log2, self.step = seed, lr_log2, 0

    # ---------------------------------------------------------------- forward

    def _conv(self, tr, cv, x, s_x):
        """One conv (+ L1BN + ReLU + Q_A); returns the layer record."""
        i = self.lid[cv.name]
        n, h, w, _ = x.shape
        wq = requant_master(self.masters[i], 24, 8).astype(np.int8)        # Eq. (WQ1)
        geo = Conv(n, h, w, cv.cin, cv.cout, cv.r, cv.r, cv.stride, cv.pad, cv.dil)
        acc = conv_fwd(geo, x, wq)
        rec = {"i": i, "cv": cv, "geo": geo, "x": x, "s_x": s_x, "wq": wq}
        if cv.bn:
            gam = requant_master(self.gm[i], 24, 8)
            bet = requant_master(self.bm[i], 24, 8)
            r = bn_fwd(acc, s_x * 2.0 ** -7, gam, bet)
            rec.update(a=r.A, s_a=r.s_a, X=r.X, s_X=r.s_xhat, c_sigma=r.c_sigma, gam=gam, bet=bet)
        else:
            a, s_a = sq_int(acc, s_x * 2.0 ** -7, 8)                       # Eq. (AQ1), no ReLU
            rec.update(a=a.astype(np.int8), s_a=s_a)
        tr[cv.name] = rec
        return rec

    def forward(self, img_u8):
        sp = self.spec
        tr = {}
        x, s = quantize_image_u8(img_u8, 4)
        tr["img"] = (x, s)
        st = self._conv(tr, sp.stem, x, s)
        y, arg = maxpool_fwd(st["a"], 3, 2, 1)
        tr["pool"] = (st["a"], y, arg)
        x, s = y, st["s_a"]
        for b in sp.blocks:
            r1 = self._conv(tr, b.conv1, x, s)
            r2 = self._conv(tr, b.conv2, r1["a"], r1["s_a"])
            r3 = self._conv(tr, b.conv3, r2["a"], r2["s_a"])
            n, hh, ww, c = r3["X"].shape
            terms = [CombineTerm(r3["X"].reshape(n, hh * ww, c), r3["s_X"], gamma=r3["gam"],
                                 beta=r3["bet"])]
            if b.down:
                rd = self._conv(tr, b.down, x, s)
                terms.append(CombineTerm(rd["X"].reshape(n, hh * ww, c), rd["s_X"],
                                         gamma=rd["gam"], beta=rd["bet"]))
            else:
                terms.append(CombineTerm(x.reshape(n, hh * ww, c), s))
            out, s_out = combine(terms, n, hh * ww, c, relu=True)
            tr[b.name] = {"in": (x, s), "out": (out.reshape(n, hh, ww, c), s_out)}
            x, s = out.reshape(n, hh, ww, c), s_out
        # ASPP
        n, hh, ww, c4 = x.shape
        tr["c4"] = (x, s)
        br = [self._conv(tr, cv, x, s) for cv in sp.aspp]
        pooled, s_p = spatial_sum(x, s, True)
        rp = self._conv(tr, sp.pool_conv, pooled.reshape(n, 1, 1, c4), s_p)
        a = sp.pool_conv.cout
        terms = [CombineTerm(r["a"].reshape(n, hh * ww, a), r["s_a"], k * a)
                 for k, r in enumerate(br)]
        terms.append(CombineTerm(rp["a"].reshape(n, a), rp["s_a"], len(br) * a, bcast=True))
        cat, s_cat = combine(terms, n, hh * ww, (len(br) + 1) * a, concat=True)
        cat = cat.reshape(n, hh, ww, (len(br) + 1) * a)
        tr["cat"] = (cat, s_cat)
        rj = self._conv(tr, sp.project, cat, s_cat)
        rh = self._conv(tr, sp.head, rj["a"], rj["s_a"])
        rc = self._conv(tr, sp.cls, rh["a"], rh["s_a"])
        z, s_z, _ = bilinear_up(rc["a"], rc["s_a"], sp.up)
        tr["z"] = (z, s_z)
        return tr

    # ---------------------------------------------------------------- backward

    def _bwd(self, out, rec, e, s_e, mask_a=None, need_dx=True):
        """Backward of one conv: BN (or nothing), wgrad + GQ1, dgrad + SQ 8, updates.
        mask_a: the codes whose positivity is the ReLU mask (default: the layer's own A)."""
        i, cv, geo = rec["i"], rec["cv"], rec["geo"]
        seed, step, lr = self.seed, self.step, self.lr_log2
        if cv.bn:
            A = rec["a"] if mask_a is None else mask_a
            ec, s_ec, dg, db = bn_bwd(e, s_e, A, rec["X"], rec["s_X"], rec["gam"], rec["c_sigma"],
                                      k_e2=K_E2)
        else:
            ec, s_ec = e, s_e
        G = conv_wgrad(geo, ec, rec["x"])
        gq, s_g = rq_int(G, s_ec * rec["s_x"], 8, 1, seed, i, step, 0)      # Eq. (GQ1)
        res = {"e": (ec, s_ec), "g": (gq, s_g)}
        if need_dx:
            dx = conv_dgrad(geo, ec, rec["wq"])
            ex, s_ex = sq_int(dx, s_ec * 2.0 ** -7, 8)
            res["ex"] = (ex.astype(np.int8).reshape(rec["x"].shape), s_ex)
        self.masters[i], _ = update(self.masters[i], gq, s_g, lr)
        if cv.bn:
            qg, sg = rq_int(dg, s_e * rec["s_X"], 8, 1, seed, i, step, 1)
            qb, sb = rq_int(db, s_e, 8, 1, seed, i, step, 2)
            self.gm[i], _ = update(self.gm[i], qg, sg, lr, x2=True)
            self.bm[i], _ = update(self.bm[i], qb, sb, lr, x2=True)
            res["dgb"] = (dg, db)
        out[cv.name] = res
        return res

    def backward_update(self, tr, labels):
        sp = self.spec
        out = {}
        z, s_z = tr["z"]
        E, s_E, nv = ce_grad(z, s_z, labels)
        out["E"] = (E, s_E)
        rc = tr[sp.cls.name]
        ecl, s_ecl, _ = bilinear_up_bwd(E, s_E, sp.up, rc["a"].shape)
        out["e_cls"] = (ecl, s_ecl)
        r = self._bwd(out, rc, ecl, s_ecl)
        r = self._bwd(out, tr[sp.head.name], *r["ex"])
        r = self._bwd(out, tr[sp.project.name], *r["ex"])
        ecat, s_ecat = r["ex"]
        x4, s4 = tr["c4"]
        n, hh, ww, c4 = x4.shape
        a = sp.pool_conv.cout
        errs = []
        for k, cv in enumerate(sp.aspp):
            eb = np.ascontiguousarray(ecat[..., k * a:(k + 1) * a])
            r = self._bwd(out, tr[cv.name], eb, s_ecat)
            errs.append(CombineTerm(r["ex"][0].reshape(n, hh * ww, c4), r["ex"][1]))
        ep, s_ep = spatial_sum(ecat, s_ecat, False, c_offset=len(sp.aspp) * a, c=a)
        r = self._bwd(out, tr[sp.pool_conv.name], ep.reshape(n, 1, 1, a), s_ep)
        epool, s_epool = r["ex"]
        errs.append(CombineTerm(epool.reshape(n, c4), s_epool / (hh * ww), bcast=True))
        e4, s_e4 = combine(errs, n, hh * ww, c4)
        out["e_c4"] = (e4, s_e4)
        e, s_e = e4.reshape(n, hh, ww, c4), s_e4
        for b in reversed(sp.blocks):
            blk = tr[b.name]
            A_out = blk["out"][0]
            x, s_x = blk["in"]
            r3 = self._bwd(out, tr[b.conv3.name], e, s_e, mask_a=A_out)
            r2 = self._bwd(out, tr[b.conv2.name], *r3["ex"])
            r1 = self._bwd(out, tr[b.conv1.name], *r2["ex"])
            nb, hb, wb, cb = x.shape
            terms = [CombineTerm(r1["ex"][0].reshape(nb, hb * wb, cb), r1["ex"][1])]
            if b.down:
                rd = self._bwd(out, tr[b.down.name], e, s_e, mask_a=A_out)
                terms.append(CombineTerm(rd["ex"][0].reshape(nb, hb * wb, cb), rd["ex"][1]))
            else:
                terms.append(CombineTerm(relu_bwd(e, A_out).reshape(nb, hb * wb, cb), s_e))
            ein, s_ein = combine(terms, nb, hb * wb, cb)
            out[b.name] = (ein.reshape(nb, hb, wb, cb), s_ein)
            e, s_e = ein.reshape(nb, hb, wb, cb), s_ein
        st_a, y, arg = tr["pool"]
        sums = maxpool_bwd(e, arg, st_a.shape, 3, 2, 1)
        ep, s_ep = sq_int(sums, s_e, 8)
        out["e_stem"] = (ep.astype(np.int8), s_ep)
        self._bwd(out, tr[sp.stem.name], ep.astype(np.int8), s_ep, need_dx=False)
        self.step += 1
        return out
