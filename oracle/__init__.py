"""CPU oracle for the integer quantized convolution layer -- TEST INFRASTRUCTURE.

This package is the plain, slow definition that the CUDA library is checked
against.  Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline``
/ ``--impl reference`` legs of ``bench.py`` may import it; the product path
never does.  It shares no code with the CUDA sources: the arithmetic lives in
``iq_oracle.c`` (plain C, exact integers, fp64 scale metadata in a fixed
operation order) and this module only marshals numpy arrays through ctypes.

Paper: "Training and Inference for Integer-Based Semantic Segmentation
Network", arXiv 2011.14504.  Each wrapper names the section/equation its C
function follows.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "iq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile iq_oracle.c with gcc (no FMA contraction, OpenMP for the
    integer convolution loops, whose results do not depend on order)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fopenmp",
                               "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        _declare(_lib)
    return _lib


class ConvDesc(C.Structure):
    _fields_ = [(n, C.c_int32) for n in
                ("n", "h", "w", "c", "k", "r", "s", "stride_h", "stride_w", "pad_h", "pad_w",
                 "dil_h", "dil_w", "groups", "p", "q")]


class BnBits(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("k_mu", "k_sigma", "k_xhat", "k_gamma", "k_beta", "k_a")]


class BnOut(C.Structure):
    _fields_ = [("s_xhat", C.c_double), ("s_a", C.c_double), ("m_xhat", C.c_double),
                ("m_y", C.c_double), ("p_x", C.c_int32), ("p_a", C.c_int32)]


class Term(C.Structure):
    _fields_ = [("codes", C.c_void_p), ("is16", C.c_int32), ("c", C.c_int32),
                ("c_offset", C.c_int32), ("bcast", C.c_int32), ("scale", C.c_double),
                ("gamma", C.c_void_p), ("beta", C.c_void_p), ("k_gamma", C.c_int32),
                ("k_beta", C.c_int32)]


_P = C.c_void_p
_I64 = C.c_int64
_I32 = C.c_int
_D = C.c_double
_U64 = C.c_uint64


def _declare(L):
    L.or_uq_f32.argtypes = [_P, _I64, _I32, _P]
    L.or_uq2_f32.argtypes = [_P, _I64, _I32, _P]
    L.or_sq_f32.argtypes = [_P, _I64, _I32, _P]
    L.or_sq_f32.restype = _D
    L.or_sq_int64.argtypes = [_P, _I64, _D, _I32, _I32, _P]
    L.or_sq_int64.restype = _D
    L.or_sq_int32.argtypes = [_P, _I64, _D, _I32, _I32, _P]
    L.or_sq_int32.restype = _D
    L.or_philox4x64_10.argtypes = [_P, _P, _P]
    L.or_rq_uniform.argtypes = [_U64, _U64, _U64, _U64, _U64]
    L.or_rq_uniform.restype = C.c_uint32
    L.or_rq_int64.argtypes = [_P, _I64, _D, _I32, _I32, _U64, _U64, _U64, _U64, _P]
    L.or_rq_int64.restype = _D
    L.or_requant_master.argtypes = [_P, _I64, _I32, _I32, _P]
    L.or_conv_out_size.argtypes = [C.POINTER(ConvDesc)]
    for f in ("or_conv_fwd", "or_conv_dgrad", "or_conv_wgrad"):
        getattr(L, f).argtypes = [C.POINTER(ConvDesc), _P, _P, _P]
        getattr(L, f + "_at").argtypes = [C.POINTER(ConvDesc), _P, _P, _P, _I64, _P]
    L.or_weight_decay.argtypes = [_I64, _P, _P, _I32, _I32, _I32]
    L.or_weight_decay.restype = None
    L.or_sq_per_channel.argtypes = [_P, _I64, _I64, _I64, _D, _I32, _I32, _P, _P]
    L.or_sq_per_channel.restype = None
    L.or_sq_at.argtypes = [_P, _I64, _I64, _D, _I32, _I32, _P]
    L.or_sq_at.restype = _D
    L.or_rq_at.argtypes = [_P, _P, _I64, _I64, _D, _I32, _I32, _U64, _U64, _U64, _U64, _P]
    L.or_rq_at.restype = _D
    L.or_bn_fwd.argtypes = [_I64, _I32, _P, _D, _P, _P, C.POINTER(BnBits), _P, _P, _P, _P,
                            _P, _P, _P, _P, C.POINTER(BnOut)]
    L.or_bn_fwd.restype = _I32
    L.or_bn_bwd.argtypes = [_I64, _I32, _P, _D, _P, _P, _D, _P, _P, _I32, _I32, _I32, _I32,
                            _P, C.POINTER(C.c_double), _P, _P]
    L.or_bn_bwd.restype = _I32
    L.or_relu_bwd.argtypes = [_I64, _P, _P, _P]
    L.or_bn_apply_fixed.argtypes = [_I64, _I32, _P, _P, _P, _P, _P, _I32, _I32, _I32, _I32, _P,
                                    _P]
    L.or_update.argtypes = [_I64, _P, _P, _P, _D, _I32, _I32, _I32, _I32]
    L.or_quantize_image_u8.argtypes = [_P, _I64, _I32, _I32, _P]
    L.or_quantize_image_u8.restype = _D
    L.or_maxpool_fwd.argtypes = [_P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P,
                                 C.POINTER(C.c_int), C.POINTER(C.c_int)]
    L.or_maxpool_bwd.argtypes = [_P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _P]
    L.or_mse_grad.argtypes = [_P, _I64, _I32, _D, _P, _I32, _P]
    L.or_mse_grad.restype = _D
    L.or_u128_to_double.argtypes = [_U64, _U64]
    L.or_u128_to_double.restype = _D
    L.or_combine.argtypes = [C.POINTER(Term), _I32, _I32, _I64, _I64, _I32, _I32, _P]
    L.or_combine.restype = _D
    L.or_spatial_sum.argtypes = [_P, _I64, _I64, _I32, _I32, _I32, _D, _I32, _P]
    L.or_spatial_sum.restype = _D
    L.or_bilinear_up.argtypes = [_P, _I32, _I32, _I32, _I32, _I32, _D, _P, _P]
    L.or_bilinear_up.restype = _D
    L.or_bilinear_up_bwd.argtypes = [_P, _I32, _I32, _I32, _I32, _I32, _D, _P, _P]
    L.or_bilinear_up_bwd.restype = _D
    L.or_exp_f32_n.argtypes = [_P, _I64, _P]
    L.or_ce_grad.argtypes = [_P, _D, _P, _I64, _I32, _I32, _P, C.POINTER(C.c_int64)]
    L.or_ce_grad.restype = _D


def _ptr(a: np.ndarray):
    assert a.flags.c_contiguous
    return a.ctypes.data_as(C.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# ---------------------------------------------------------------- quantizers

def uq(x, k: int) -> np.ndarray:
    """Eq. (UQ): codes of UQ(x, k) for fp32 x (value = code * 2^(1-k))."""
    x = _c(x, np.float32)
    out = np.empty(x.shape, np.int32)
    lib().or_uq_f32(_ptr(x), x.size, k, _ptr(out))
    return out


def uq2(x, k: int) -> np.ndarray:
    """2*UQ(x/2, k) codes (value = code * 2^(2-k)), Sec. 3.1.1 / QBN block."""
    x = _c(x, np.float32)
    out = np.empty(x.shape, np.int32)
    lib().or_uq2_f32(_ptr(x), x.size, k, _ptr(out))
    return out


def sq_float(x, k: int):
    """Eq. (ScaleQ) on fp32 input: (codes, scale)."""
    x = _c(x, np.float32)
    out = np.empty(x.shape, np.int32)
    s = lib().or_sq_f32(_ptr(x), x.size, k, _ptr(out))
    return out, s


def sq_int(q, s: float, k: int, relu: bool = False):
    """Eq. (ScaleQ) on an integer-coded tensor (codes q, scale s): (codes, scale)."""
    q = _c(q, np.int64)
    out = np.empty(q.shape, np.int32)
    so = lib().or_sq_int64(_ptr(q), q.size, float(s), k, int(relu), _ptr(out))
    return out, so


def sq_per_channel(q, outer: int, C: int, inner: int, s: float, k: int, relu: bool = False):
    """Eq. (ScaleQ) with a per-channel Scale (Eq. (ScaleFactor) over each channel's elements)
    on an integer-coded tensor viewed as [outer][C][inner]: (codes, scales[C])."""
    q = _c(q, np.int64)
    assert q.size == outer * C * inner
    out = np.empty(q.shape, np.int32)
    sc = np.empty(C, np.float64)
    lib().or_sq_per_channel(_ptr(q), outer, C, inner, float(s), k, int(relu), _ptr(out), _ptr(sc))
    return out, sc


def sq_at(q, M: int, s: float, k: int, relu: bool = False):
    """Eq. (ScaleQ) codes of selected elements q of a tensor whose max |q| (after ReLU when
    relu) is M, and the output scale: the values sq_int gives at those elements."""
    q = _c(q, np.int64)
    out = np.empty(q.shape, np.int32)
    so = lib().or_sq_at(_ptr(q), q.size, int(M), float(s), k, int(relu), _ptr(out))
    return out, so


def rq_at(q, idx, M: int, s: float, k: int, gq_mode: int, seed: int, layer: int, step: int,
          tag: int = 0):
    """Eqs. (SQ),(SR),(GQ1)/(GQ2) codes of selected elements q (flat indices idx) of a tensor
    whose max |q| is M, and the output scale: the values rq_int gives at those elements."""
    q = _c(q, np.int64)
    idx = _c(idx, np.int64)
    assert q.shape == idx.shape
    out = np.empty(q.shape, np.int32)
    so = lib().or_rq_at(_ptr(q), _ptr(idx), q.size, int(M), float(s), k, gq_mode, seed, layer,
                        step, tag, _ptr(out))
    return out, so


def philox(ctr, key) -> np.ndarray:
    """Philox4x64-10 block for a 4-word counter and 2-word key."""
    c = _c(ctr, np.uint64)
    kk = _c(key, np.uint64)
    o = np.empty(4, np.uint64)
    lib().or_philox4x64_10(_ptr(c), _ptr(kk), _ptr(o))
    return o


def rq_uniform(seed, layer, step, tag, i) -> int:
    return int(lib().or_rq_uniform(seed, layer, step, tag, i))


def rq_int(q, s: float, k: int, gq_mode: int, seed: int, layer: int, step: int, tag: int = 0):
    """Eqs. (SQ),(SR) applied as Eq. (GQ1) (gq_mode=1) or Eq. (GQ2) (gq_mode=2)."""
    q = _c(q, np.int64)
    out = np.empty(q.shape, np.int32)
    so = lib().or_rq_int64(_ptr(q), q.size, float(s), k, gq_mode, seed, layer, step, tag,
                           _ptr(out))
    return out, so


def requant_master(m, k_u: int = 24, k_w: int = 8) -> np.ndarray:
    """Eq. (WQ1): W_q = UQ(W_m, k_W) from k_U-grid master codes."""
    m = _c(m, np.int32)
    out = np.empty(m.shape, np.int32)
    lib().or_requant_master(_ptr(m), m.size, k_u, k_w, _ptr(out))
    return out


def quantize_image_u8(img, c_out: int):
    """Network input: pixel/255 -> SQ8 codes, NHWC uint8 -> NHWC int8 with c_out channels."""
    img = _c(img, np.uint8)
    n, h, w, c = img.shape
    out = np.empty((n, h, w, c_out), np.int8)
    s = lib().or_quantize_image_u8(_ptr(img), n * h * w, c, c_out, _ptr(out))
    return out, s


def u128_to_double(v: int) -> float:
    return lib().or_u128_to_double((v >> 64) & (2**64 - 1), v & (2**64 - 1))


# ---------------------------------------------------------------- convolution

@dataclass
class Conv:
    n: int
    h: int
    w: int
    c: int
    k: int
    r: int
    s: int
    stride: int = 1
    pad: int = 0
    dil: int = 1
    groups: int = 1

    def desc(self) -> ConvDesc:
        d = ConvDesc(self.n, self.h, self.w, self.c, self.k, self.r, self.s, self.stride,
                     self.stride, self.pad, self.pad, self.dil, self.dil, self.groups, 0, 0)
        lib().or_conv_out_size(C.byref(d))
        return d

    @property
    def pq(self):
        d = self.desc()
        return d.p, d.q


def conv_fwd(cv: Conv, x, w) -> np.ndarray:
    """Direct 7-loop convolution: int8 NHWC x, int8 KRSC w -> int32 NPQK."""
    d = cv.desc()
    x = _c(x, np.int8)
    w = _c(w, np.int8)
    assert x.size == cv.n * cv.h * cv.w * cv.c
    assert w.size == cv.k * cv.r * cv.s * (cv.c // cv.groups)
    out = np.empty((cv.n, d.p, d.q, cv.k), np.int32)
    lib().or_conv_fwd(C.byref(d), _ptr(x), _ptr(w), _ptr(out))
    return out


def conv_dgrad(cv: Conv, e, w) -> np.ndarray:
    """Adjoint of conv_fwd in x: int8 e (NPQK), int8 w -> int64 NHWC (exact sums)."""
    d = cv.desc()
    e = _c(e, np.int8)
    w = _c(w, np.int8)
    assert e.size == cv.n * d.p * d.q * cv.k
    out = np.empty((cv.n, cv.h, cv.w, cv.c), np.int64)
    lib().or_conv_dgrad(C.byref(d), _ptr(e), _ptr(w), _ptr(out))
    return out


def conv_wgrad(cv: Conv, e, x) -> np.ndarray:
    """Adjoint of conv_fwd in w: int8 e (NPQK), int8 x (NHWC) -> int64 KRSC."""
    d = cv.desc()
    e = _c(e, np.int8)
    x = _c(x, np.int8)
    out = np.empty((cv.k, cv.r, cv.s, cv.c // cv.groups), np.int64)
    lib().or_conv_wgrad(C.byref(d), _ptr(e), _ptr(x), _ptr(out))
    return out


def _at(fname, cv: Conv, a, b, idx):
    d = cv.desc()
    a = _c(a, np.int8)
    b = _c(b, np.int8)
    idx = _c(idx, np.int64).ravel()
    out = np.empty(idx.shape, np.int64)
    getattr(lib(), fname)(C.byref(d), _ptr(a), _ptr(b), _ptr(idx), idx.size, _ptr(out))
    return out


def conv_fwd_at(cv: Conv, x, w, idx) -> np.ndarray:
    """conv_fwd at the flat NPQK output indices idx only (int64 sums), one by one."""
    return _at("or_conv_fwd_at", cv, x, w, idx)


def conv_dgrad_at(cv: Conv, e, w, idx) -> np.ndarray:
    """conv_dgrad at the flat NHWC input indices idx only."""
    return _at("or_conv_dgrad_at", cv, e, w, idx)


def conv_wgrad_at(cv: Conv, e, x, idx) -> np.ndarray:
    """conv_wgrad at the flat KRSC weight indices idx only."""
    return _at("or_conv_wgrad_at", cv, e, x, idx)


# ---------------------------------------------------------------- L1BN

@dataclass
class BnResult:
    X: np.ndarray
    A: np.ndarray
    c_mu: np.ndarray
    c_sigma: np.ndarray
    F: np.ndarray
    B: np.ndarray
    G: np.ndarray
    H: np.ndarray
    s_xhat: float
    s_a: float
    m_xhat: float
    m_y: float
    p_x: int
    p_a: int


def bn_fwd(acc, s_acc: float, gamma_codes, beta_codes, k_mu=16, k_sigma=16, k_xhat=16,
           k_gamma=8, k_beta=8, k_a=8) -> BnResult:
    """Quantized L1BN + ReLU + Q_A on conv accumulators acc[m, C] (Sec. 3.2.2-3.2.3)."""
    acc = _c(acc, np.int32)
    m, Cn = acc.reshape(-1, acc.shape[-1]).shape
    g = _c(gamma_codes, np.int32)
    b = _c(beta_codes, np.int32)
    X = np.empty(acc.shape, np.int16)
    A = np.empty(acc.shape, np.int8)
    cm = np.empty(Cn, np.int32)
    cs = np.empty(Cn, np.int32)
    F = np.empty(Cn, np.int64)
    B = np.empty(Cn, np.int64)
    G = np.empty(Cn, np.int64)
    H = np.empty(Cn, np.int64)
    bits = BnBits(k_mu, k_sigma, k_xhat, k_gamma, k_beta, k_a)
    o = BnOut()
    rc = lib().or_bn_fwd(m, Cn, _ptr(acc), float(s_acc), _ptr(g), _ptr(b), C.byref(bits),
                         _ptr(X), _ptr(A), _ptr(cm), _ptr(cs), _ptr(F), _ptr(B), _ptr(G),
                         _ptr(H), C.byref(o))
    if rc != 0:
        raise ValueError("or_bn_fwd: empty input")
    return BnResult(X, A, cm, cs, F, B, G, H, o.s_xhat, o.s_a, o.m_xhat, o.m_y, o.p_x, o.p_a)


def bn_apply_fixed(acc, F, B, G, H, p_x: int, p_a: int, k_xhat=16, k_a=8):
    """The L1BN element maps with constants fixed by an earlier call (frozen statistics):
    returns (X, A) for accumulators acc[m, C]."""
    acc = _c(acc, np.int32)
    C_ = acc.shape[-1]
    m = acc.size // C_
    F, B, G, H = (_c(v, np.int64) for v in (F, B, G, H))
    X = np.empty(acc.shape, np.int16)
    A = np.empty(acc.shape, np.int8)
    lib().or_bn_apply_fixed(m, C_, _ptr(acc), _ptr(F), _ptr(B), _ptr(G), _ptr(H), p_x, p_a,
                            k_xhat, k_a, _ptr(X), _ptr(A))
    return X, A


def bn_bwd(eA, s_e: float, A, X, s_x: float, gamma_codes, c_sigma, k_sigma=16, k_gamma=8,
           k_e2=16, k_e=8):
    """ReLU + quantized L1BN backward, then Q_E to the conv error (Sec. 3.3.1)."""
    eA = _c(eA, np.int8)
    A = _c(A, np.int8)
    X = _c(X, np.int16)
    Cn = eA.shape[-1]
    m = eA.size // Cn
    g = _c(gamma_codes, np.int32)
    cs = _c(c_sigma, np.int32)
    E = np.empty(eA.shape, np.int8)
    so = C.c_double(0)
    dg = np.empty(Cn, np.int64)
    db = np.empty(Cn, np.int64)
    rc = lib().or_bn_bwd(m, Cn, _ptr(eA), float(s_e), _ptr(A), _ptr(X), float(s_x), _ptr(g),
                         _ptr(cs), k_sigma, k_gamma, k_e2, k_e, _ptr(E), C.byref(so), _ptr(dg),
                         _ptr(db))
    if rc != 0:
        raise ValueError("or_bn_bwd: empty input")
    return E, so.value, dg, db


def relu_bwd(eA, A) -> np.ndarray:
    eA = _c(eA, np.int8)
    A = _c(A, np.int8)
    out = np.empty(eA.shape, np.int8)
    lib().or_relu_bwd(eA.size, _ptr(eA), _ptr(A), _ptr(out))
    return out


def update(master, gcodes, s_g: float, lr_log2: int, k_u=24, k_w=8, x2=False):
    """Eq. (UQ2) update of k_U-grid master codes; returns (new master, new W_q)."""
    m = np.array(master, dtype=np.int32, copy=True)
    g = _c(gcodes, np.int32)
    wq = np.empty(m.shape, np.int32)
    lib().or_update(m.size, _ptr(m), _ptr(wq), _ptr(g), float(s_g), lr_log2, k_u, k_w, int(x2))
    return m, wq


def weight_decay(master, shift: int, k_u=24, k_w=8):
    """Decoupled L2 weight decay of k_U-grid master codes (decay step 2^-shift); returns
    (new master, new W_q)."""
    m = np.array(master, dtype=np.int32, copy=True)
    wq = np.empty(m.shape, np.int32)
    lib().or_weight_decay(m.size, _ptr(m), _ptr(wq), shift, k_u, k_w)
    return m, wq


# ---------------------------------------------------------------- network glue

def maxpool_fwd(x, k: int, s: int, p: int = 0):
    """Max pooling of codes; returns (y, argmax tap index)."""
    x = _c(x, np.int8)
    n, h, w, c = x.shape
    P = (h + 2 * p - k) // s + 1
    Q = (w + 2 * p - k) // s + 1
    y = np.empty((n, P, Q, c), np.int8)
    a = np.empty((n, P, Q, c), np.uint8)
    ph, pw = C.c_int(), C.c_int()
    lib().or_maxpool_fwd(_ptr(x), n, h, w, c, k, s, p, _ptr(y), _ptr(a), C.byref(ph), C.byref(pw))
    return y, a


def maxpool_bwd(e, arg, in_shape, k: int, s: int, p: int = 0) -> np.ndarray:
    e = _c(e, np.int8)
    arg = _c(arg, np.uint8)
    n, h, w, c = in_shape
    ex = np.empty((n, h, w, c), np.int32)
    lib().or_maxpool_bwd(_ptr(e), _ptr(arg), n, h, w, c, k, s, p, _ptr(ex))
    return ex


def mse_grad(z, s_z: float, labels, k: int = 8):
    """Q_E of the MSE-loss gradient z s_z - onehot(label) on quantized logits."""
    z = _c(z, np.int8)
    lab = _c(labels, np.uint8)
    c = z.shape[-1]
    E = np.empty(z.shape, np.int8)
    s = lib().or_mse_grad(_ptr(z), z.size // c, c, float(s_z), _ptr(lab), k, _ptr(E))
    return E, s


# ---------------------------------------------------------------- DeepLab glue

@dataclass
class CombineTerm:
    """One operand of combine(): integer codes (int8 or int16) with real value
    a_c v + b_c, a_c = scale (or gamma_q,c scale for a BN affine term), b_c = 0 (or beta_q,c).
    codes are [n, hw, c] (or [n, c] with bcast: one value per image, broadcast over hw)."""
    codes: np.ndarray
    scale: float
    c_offset: int = 0
    bcast: bool = False
    gamma: np.ndarray = None
    beta: np.ndarray = None
    k_gamma: int = 8
    k_beta: int = 8


def combine(terms, n: int, hw: int, c_out: int, concat: bool = False, relu: bool = False):
    """Sum (or channel concatenation) of quantized tensors in real units, then SQ8
    (Eqs. (AQ1)/(EQ) applied to a residual add, a sum of errors, the ASPP concat)."""
    keep, arr = [], (Term * len(terms))()
    for t, T in zip(terms, arr):
        codes = np.ascontiguousarray(t.codes)
        assert codes.dtype in (np.int8, np.int16)
        keep.append(codes)
        T.codes = codes.ctypes.data
        T.is16 = int(codes.dtype == np.int16)
        T.c = codes.shape[-1]
        T.c_offset = t.c_offset
        T.bcast = int(t.bcast)
        T.scale = float(t.scale)
        if t.gamma is not None:
            g = _c(t.gamma, np.int32); b = _c(t.beta, np.int32)
            keep += [g, b]
            T.gamma, T.beta = g.ctypes.data, b.ctypes.data
        else:
            T.gamma = T.beta = None
        T.k_gamma, T.k_beta = t.k_gamma, t.k_beta
    out = np.empty((n * hw * c_out,), np.int8)
    s = lib().or_combine(arr, len(terms), int(concat), n, hw, c_out, int(relu), _ptr(out))
    return out, s


def spatial_sum(x, s: float, mean: bool, c_offset: int = 0, c: int = None):
    """Per image sum (mean) over the pixels of channels [c_offset, c_offset + c) of
    x [n, h, w, c_total], then SQ8; returns ([n, c] codes, scale)."""
    x = _c(x, np.int8)
    n, c_total = x.shape[0], x.shape[-1]
    hw = x.size // (n * c_total)
    c = c_total - c_offset if c is None else c
    out = np.empty((n, c), np.int8)
    so = lib().or_spatial_sum(_ptr(x), n, hw, c_total, c_offset, c, float(s), int(mean), _ptr(out))
    return out, so


def bilinear_up(x, s: float, f: int):
    """x8-style bilinear upsampling with aligned corners (exact integer numerators, then
    SQ8); returns (codes [n, (h-1)f+1, (w-1)f+1, c], scale, numerators int32)."""
    x = _c(x, np.int8)
    n, h, w, c = x.shape
    H, W = (h - 1) * f + 1, (w - 1) * f + 1
    acc = np.empty((n, H, W, c), np.int32)
    out = np.empty((n, H, W, c), np.int8)
    so = lib().or_bilinear_up(_ptr(x), n, h, w, c, f, float(s), _ptr(acc), _ptr(out))
    return out, so, acc


def bilinear_up_bwd(e, s: float, f: int, in_shape):
    e = _c(e, np.int8)
    n, h, w, c = in_shape
    assert e.shape == (n, (h - 1) * f + 1, (w - 1) * f + 1, c)
    out = np.empty((n, h, w, c), np.int8)
    acc = np.empty((n, h, w, c), np.int64)
    so = lib().or_bilinear_up_bwd(_ptr(e), n, h, w, c, f, float(s), _ptr(acc), _ptr(out))
    return out, so, acc


def exp_f32(t) -> np.ndarray:
    """The fp32 exponential of the softmax head (Cody-Waite reduction + degree-7 Taylor)."""
    t = _c(t, np.float32)
    out = np.empty(t.shape, np.float32)
    lib().or_exp_f32_n(_ptr(t), t.size, _ptr(out))
    return out


def ce_grad(z, s_z: float, labels, ignore: int = 255):
    """Softmax cross-entropy gradient on quantized logits, SQ8; returns (E, scale, n_valid)."""
    z = _c(z, np.int8)
    lab = _c(labels, np.uint8)
    c = z.shape[-1]
    E = np.empty(z.shape, np.int8)
    nv = C.c_int64()
    s = lib().or_ce_grad(_ptr(z), float(s_z), _ptr(lab), z.size // c, c, ignore, _ptr(E),
                         C.byref(nv))
    return E, s, nv.value
