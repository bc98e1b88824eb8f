"""Thin Python binding of the iq C ABI (``include/iq.h``).

Argument marshalling only: every step of the computation runs in the CUDA
kernels of ``libiq.so``.  Tensors are torch CUDA tensors used as plain device
memory; the stream defaults to torch's current stream.  There is no fallback:
if the library cannot be loaded the import-time ``load()`` raises.
"""
from __future__ import annotations

import ctypes as C
import os

import torch

from . import build as _build

IQ_OK, IQ_ERR_INVALID_ARG, IQ_ERR_UNSUPPORTED, IQ_ERR_WORKSPACE = 0, 1, 2, 3
IQ_ERR_OVERFLOW_RISK, IQ_ERR_TIMEOUT, IQ_ERR_CUDA = 4, 5, 6
IQ_I8, IQ_I16, IQ_I32, IQ_I64, IQ_F32, IQ_U8 = 1, 2, 3, 4, 5, 6
IQ_MODE_UQ, IQ_MODE_UQ2, IQ_MODE_SQ, IQ_MODE_SQ_RELU, IQ_MODE_RQ_GQ1, IQ_MODE_RQ_GQ2 = range(6)
IQ_BN_S_XHAT, IQ_BN_M_XHAT, IQ_BN_M_Y, IQ_BN_S_ACC, IQ_BN_S_A, IQ_BN_SCALES = 0, 1, 2, 3, 4, 8

EXPORTS = [
    "iq_status_str", "iq_version", "iq_launch_count", "iq_conv_out_size", "iq_quantize_workspace_size",
    "iq_conv_fwd_workspace_size", "iq_conv_dgrad_workspace_size", "iq_conv_wgrad_workspace_size",
    "iq_bn_int_workspace_size", "iq_quantize", "iq_quantize_image_u8", "iq_requantize",
    "iq_requantize_per_channel_workspace_size", "iq_requantize_per_channel",
    "iq_gemm_s8_nibble_workspace_size", "iq_gemm_s8_nibble", "iq_weight_decay",
    "iq_weight_requant", "iq_conv_fwd", "iq_conv_dgrad", "iq_conv_wgrad", "iq_bn_int_fwd",
    "iq_bn_int_bwd", "iq_relu_bwd", "iq_update", "iq_maxpool_fwd", "iq_maxpool_bwd",
    "iq_upsample_workspace_size", "iq_upsample_fwd", "iq_upsample_bwd", "iq_upsample_wgrad",
    "iq_mse_grad", "iq_bn_int_fwd_noalloc", "iq_combine_workspace_size", "iq_combine",
    "iq_spatial_sum_workspace_size", "iq_spatial_sum", "iq_avgpool_bwd", "iq_channel_slice",
    "iq_bilinear_workspace_size", "iq_bilinear_up_fwd", "iq_bilinear_up_bwd", "iq_ce_grad",
    "iq_bn_update", "iq_device_status", "iq_rq_epoch_advance", "iq_rq_epoch_set",
    "iq_kernel_timing_begin", "iq_kernel_timing_end", "iq_wait_selftest", "iq_conv_fwd_frozen",
]
IQ_KERNEL_CONV_PIXEL_MAJOR, IQ_KERNEL_CONV_CHANNEL_MAJOR, IQ_KERNEL_CONV_WGRAD = 1, 2, 3
IQ_KERNEL_CONV_CPASYNC, IQ_KERNEL_CONV_GATHER, IQ_KERNEL_CONV_SIMT = 4, 5, 6
(IQ_KERNEL_BN_DEV, IQ_KERNEL_BN_REQUANT, IQ_KERNEL_BNB_PASS1, IQ_KERNEL_BNB_PASS2,
 IQ_KERNEL_BNB_PASS3, IQ_KERNEL_COMBINE_MAX, IQ_KERNEL_COMBINE_CODES, IQ_KERNEL_SQ_CODES,
 IQ_KERNEL_CODES_TO_F16, IQ_KERNEL_ABSMAX, IQ_KERNEL_RQ_CODES) = range(10, 21)
KERNEL_NAMES = {1: "k_conv_tct (forward / data gradient)", 2: "k_conv_tcc (channel-major)",
                3: "k_conv_tct (weight gradient)", 4: "k_conv_tcq", 5: "k_conv_tcp",
                6: "k_conv_simt", 10: "k_bn_dev", 11: "k_bn_requant", 12: "k_bnb_pass1",
                13: "k_bnb_pass2", 14: "k_bnb_pass3", 15: "iq_combine max pass",
                16: "iq_combine codes pass", 17: "SQ codes (k_sq_i32_i8x4 / k_sq_int)",
                18: "k_codes_to_f16", 19: "k_absmax_int", 20: "k_rq_int"}
CONV_KERNELS = (1, 2, 3, 4, 5, 6)


class IqError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn}: {status_str(code)} ({code})")
        self.code = code


class ConvDesc(C.Structure):
    _fields_ = [(n, C.c_int32) for n in
                ("n", "h", "w", "c", "k", "r", "s", "stride_h", "stride_w", "pad_h", "pad_w",
                 "dil_h", "dil_w", "groups", "layout", "k_w", "k_a", "flags")]


IQ_LAYOUT_NHWC, IQ_LAYOUT_NCHW = 0, 1
IQ_CONV_X_F16_READY, IQ_CONV_E_F16_READY = 1, 2


class BnBits(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("k_mu", "k_sigma", "k_xhat", "k_gamma", "k_beta", "k_a")]


class Term(C.Structure):
    """iq_term: one operand of iq_combine (device pointers inside)."""
    _fields_ = [("codes", C.c_void_p), ("dtype", C.c_int32), ("c", C.c_int32),
                ("c_offset", C.c_int32), ("bcast", C.c_int32), ("scale", C.c_void_p),
                ("gamma", C.c_void_p), ("beta", C.c_void_p), ("k_gamma", C.c_int32),
                ("k_beta", C.c_int32)]


class KernelTime(C.Structure):
    """iq_kernel_time: summed event time and MACs of one (kernel, operation) pair."""
    _fields_ = [("kernel", C.c_int32), ("op", C.c_int32), ("launches", C.c_int32),
                ("pad", C.c_int32), ("ms", C.c_double), ("macs", C.c_double),
                ("dense_macs", C.c_double), ("bytes", C.c_double)]


IQ_MAX_TERMS = 8


_P = C.c_void_p
_I = C.c_int
_I32 = C.c_int32
_I64 = C.c_int64
_U64 = C.c_uint64
_SZ = C.c_size_t
_L = None


def load(path: str | None = None):
    """Load libiq.so (building it in-tree if needed).  Raises if unavailable."""
    global _L
    if _L is not None:
        return _L
    if path is None:
        path = _build.LIB if os.path.exists(_build.LIB) else _build.build()
    L = C.CDLL(path)
    L.iq_status_str.restype = C.c_char_p
    L.iq_status_str.argtypes = [_I]
    L.iq_version.restype = _I
    L.iq_launch_count.restype = C.c_ulonglong
    L.iq_launch_count.argtypes = []
    L.iq_conv_out_size.argtypes = [C.POINTER(ConvDesc), C.POINTER(_I32), C.POINTER(_I32)]
    L.iq_quantize_workspace_size.argtypes = [_I64, C.POINTER(_SZ)]
    L.iq_conv_fwd_workspace_size.argtypes = [C.POINTER(ConvDesc), _I, C.POINTER(_SZ)]
    L.iq_conv_dgrad_workspace_size.argtypes = [C.POINTER(ConvDesc), C.POINTER(_SZ)]
    L.iq_conv_wgrad_workspace_size.argtypes = [C.POINTER(ConvDesc), C.POINTER(_SZ)]
    L.iq_bn_int_workspace_size.argtypes = [_I64, _I32, C.POINTER(_SZ)]
    L.iq_quantize.argtypes = [_P, _I64, _I, _I, _I, _P, _P, _P, _SZ, _P]
    L.iq_quantize_image_u8.argtypes = [_P, _I32, _I32, _I32, _I32, _I, _I32, _P, _P, _P, _SZ, _P]
    L.iq_weight_decay.argtypes = [_P, _P, _I64, _I, _I, _I, _P]
    L.iq_gemm_s8_nibble_workspace_size.argtypes = [_I32, _I32, _I32, C.POINTER(_SZ)]
    L.iq_gemm_s8_nibble.argtypes = [_P, _P, _P, _I32, _I32, _I32, _P, _SZ, _P]
    L.iq_requantize_per_channel_workspace_size.argtypes = [_I32, C.POINTER(_SZ)]
    L.iq_requantize_per_channel.argtypes = [_P, _I, _I64, _I32, _I64, _P, _I, _I, _P, _I, _P, _P,
                                            _SZ, _P]
    L.iq_requantize.argtypes = [_P, _I, _I64, _P, _I, _I, _U64, _U64, _U64, _U64, _P, _I, _P, _P,
                                _SZ, _P]
    L.iq_weight_requant.argtypes = [_P, _P, _I64, _I, _I, _P]
    L.iq_conv_fwd.argtypes = [C.POINTER(ConvDesc), _P, _P, _P, _P, _P, C.POINTER(BnBits), _I, _I,
                              _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P]
    L.iq_conv_fwd_frozen.argtypes = [C.POINTER(ConvDesc), _P, _P, _P, C.POINTER(BnBits), _I, _I,
                                     _P, _P, _P, _P, _SZ, _P]
    L.iq_conv_dgrad.argtypes = [C.POINTER(ConvDesc), _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ,
                                _P]
    L.iq_conv_wgrad.argtypes = [C.POINTER(ConvDesc), _P, _P, _P, _P, _I, _U64, _U64, _U64, _P, _P,
                                _P, _P, _P, _P, _SZ, _P]
    L.iq_bn_int_fwd.argtypes = [_P, _I64, _I32, _P, _P, _P, C.POINTER(BnBits), _P, _P, _P, _P, _P,
                                _P, _P, _SZ, _P]
    L.iq_bn_int_bwd.argtypes = [_P, _P, _P, _P, _I64, _I32, _P, _P, _P, C.POINTER(BnBits), _I, _P,
                                _P, _P, _P, _P, _P, _SZ, _P]
    L.iq_relu_bwd.argtypes = [_P, _P, _I64, _P, _P, _P]
    L.iq_update.argtypes = [_P, _P, _P, _P, _I64, _I, _I, _I, _I, _P]
    L.iq_maxpool_fwd.argtypes = [_P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P, _P]
    L.iq_maxpool_bwd.argtypes = [_P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P,
                                 _SZ, _P]
    L.iq_upsample_workspace_size.argtypes = [_I32, _I32, _I32, _I32, _I32, C.POINTER(_SZ)]
    L.iq_upsample_fwd.argtypes = [_P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P,
                                  _P, _SZ, _P]
    L.iq_upsample_bwd.argtypes = [_P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P,
                                  _P, _SZ, _P]
    L.iq_upsample_wgrad.argtypes = [_P, _P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _I32, _I,
                                    _U64, _U64, _U64, _P, _P, _P, _P, _SZ, _P]
    L.iq_mse_grad.argtypes = [_P, _P, _P, _I64, _I32, _P, _P, _P, _SZ, _P]
    L.iq_bn_int_fwd_noalloc.argtypes = [_P, _I64, _I32, _P, _P, _P, C.POINTER(BnBits), _P, _P,
                                        _P, _P, _P, _P, _P]
    L.iq_combine_workspace_size.argtypes = [C.POINTER(Term), _I32, C.POINTER(_SZ)]
    L.iq_combine.argtypes = [C.POINTER(Term), _I32, _I32, _I64, _I64, _I32, _I32, _P, _P, _P, _P,
                             _SZ, _P]
    L.iq_spatial_sum_workspace_size.argtypes = [_I64, _I32, C.POINTER(_SZ)]
    L.iq_spatial_sum.argtypes = [_P, _P, _I64, _I64, _I32, _I32, _I32, _I32, _P, _P, _P, _SZ, _P]
    L.iq_avgpool_bwd.argtypes = [_P, _P, _I64, _I64, _I32, _P, _P, _P]
    L.iq_channel_slice.argtypes = [_P, _I64, _I32, _I32, _I32, _P, _P]
    L.iq_bilinear_workspace_size.argtypes = [_I32, _I32, _I32, _I32, C.POINTER(_SZ)]
    L.iq_bilinear_up_fwd.argtypes = [_P, _P, _I32, _I32, _I32, _I32, _I32, _P, _P, _P, _SZ, _P]
    L.iq_bilinear_up_bwd.argtypes = [_P, _P, _I32, _I32, _I32, _I32, _I32, _P, _P, _P, _SZ, _P]
    L.iq_ce_grad.argtypes = [_P, _P, _P, _I64, _I32, _I32, _P, _P, _P, _P, _SZ, _P]
    L.iq_bn_update.argtypes = [_P, _P, _P, _P, _P, _P, _P, _P, _I32, C.POINTER(BnBits), _I, _I,
                               _U64, _U64, _U64, _P, _SZ, _P]
    L.iq_device_status.argtypes = [C.POINTER(_I32), _P]
    L.iq_kernel_timing_begin.argtypes = []
    L.iq_kernel_timing_end.argtypes = [C.POINTER(KernelTime), _I32, C.POINTER(_I32)]
    L.iq_rq_epoch_advance.argtypes = [_P]
    L.iq_rq_epoch_set.argtypes = [_U64, _P]
    L.iq_wait_selftest.argtypes = [C.c_longlong, _P]
    for f in EXPORTS:
        if f not in ("iq_status_str", "iq_version", "iq_launch_count"):
            getattr(L, f).restype = _I
    _L = L
    return L


def launch_count() -> int:
    return int(load().iq_launch_count())


def iq_kernel_timing_begin():
    """Start bracketing every tensor-core conv kernel launch with CUDA events (eager calls)."""
    _check("iq_kernel_timing_begin", load().iq_kernel_timing_begin())


def iq_kernel_timing_end(capacity=64):
    """Stop, wait for the events and return [{kernel, op, launches, ms, macs, dense_macs,
    bytes}] per (kernel, op)."""
    out = (KernelTime * capacity)()
    n = _I32(0)
    _check("iq_kernel_timing_end", load().iq_kernel_timing_end(out, capacity, C.byref(n)))
    return [{"kernel": out[i].kernel, "op": out[i].op, "launches": out[i].launches,
             "ms": out[i].ms, "macs": out[i].macs, "dense_macs": out[i].dense_macs,
             "bytes": out[i].bytes} for i in range(n.value)]


def iq_device_status(stream=None) -> int:
    """Synchronize the stream, return and clear the sticky device status of the tensor-core
    kernels (0: every bounded wait completed).  Raises IqError(IQ_ERR_TIMEOUT) when a wait
    gave up, since the outputs since the last check are then not valid."""
    code = _I32(0)
    _check("iq_device_status", load().iq_device_status(C.byref(code), _stream(stream)))
    return code.value


def iq_wait_selftest(limit_cycles=1 << 20, stream=None):
    """Enqueue the bounded-wait self-test kernel (its wait must give up: status code 5)."""
    _check("iq_wait_selftest", load().iq_wait_selftest(C.c_longlong(limit_cycles),
                                                       _stream(stream)))


def iq_rq_epoch_advance(stream=None):
    """Add 1 to the stochastic-rounding epoch (the fourth Philox counter word) on the stream."""
    _check("iq_rq_epoch_advance", load().iq_rq_epoch_advance(_stream(stream)))


def iq_rq_epoch_set(value: int, stream=None):
    _check("iq_rq_epoch_set", load().iq_rq_epoch_set(value, _stream(stream)))


def status_str(code: int) -> str:
    return load().iq_status_str(code).decode()


def _p(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn: str, rc: int):
    if rc != IQ_OK:
        raise IqError(fn, rc)


def _ws(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


def conv_desc(n, h, w, c, k, r, s, stride=1, pad=0, dil=1, groups=1, layout=IQ_LAYOUT_NHWC,
              k_w=0, k_a=0, flags=0) -> ConvDesc:
    """iq_conv_desc; layout IQ_LAYOUT_NCHW takes NCHW activations / errors and KCRS filters,
    k_w / k_a the weight and activation code widths (0: 8 bits); flags
    IQ_CONV_X_F16_READY: the x_f16 buffer of the forward already holds the input's fp16 copy."""
    return ConvDesc(n, h, w, c, k, r, s, stride, stride, pad, pad, dil, dil, groups, layout, k_w,
                    k_a, flags)


def bn_bits(k_mu=16, k_sigma=16, k_xhat=16, k_gamma=8, k_beta=8, k_a=8) -> BnBits:
    return BnBits(k_mu, k_sigma, k_xhat, k_gamma, k_beta, k_a)


# ---------------------------------------------------------------- queries

def iq_conv_out_size(d: ConvDesc):
    p, q = _I32(), _I32()
    _check("iq_conv_out_size", load().iq_conv_out_size(C.byref(d), C.byref(p), C.byref(q)))
    return p.value, q.value


def _size(fn, *args) -> int:
    b = _SZ()
    _check(fn, getattr(load(), fn)(*args, C.byref(b)))
    return b.value


def iq_quantize_workspace_size(n: int) -> int:
    return _size("iq_quantize_workspace_size", n)


def iq_conv_fwd_workspace_size(d: ConvDesc, with_bn: bool = False) -> int:
    return _size("iq_conv_fwd_workspace_size", C.byref(d), int(with_bn))


def iq_conv_dgrad_workspace_size(d: ConvDesc) -> int:
    return _size("iq_conv_dgrad_workspace_size", C.byref(d))


def iq_conv_wgrad_workspace_size(d: ConvDesc) -> int:
    return _size("iq_conv_wgrad_workspace_size", C.byref(d))


def iq_bn_int_workspace_size(m: int, c: int) -> int:
    return _size("iq_bn_int_workspace_size", m, c)


# ---------------------------------------------------------------- operations

def iq_quantize(x, k, mode, codes, scale, ws=None, stream=None):
    out_dtype = {torch.int8: IQ_I8, torch.int16: IQ_I16, torch.int32: IQ_I32}[codes.dtype]
    if ws is None:
        ws = _ws(iq_quantize_workspace_size(x.numel()), x.device)
    _check("iq_quantize", load().iq_quantize(_p(x), x.numel(), k, mode, out_dtype, _p(codes),
                                             _p(scale), _p(ws), ws.numel(), _stream(stream)))


def iq_quantize_image_u8(img, nchw, c_out, codes, scale, ws=None, stream=None):
    if nchw:
        n, c, h, w = img.shape
    else:
        n, h, w, c = img.shape
    if ws is None:
        ws = _ws(iq_quantize_workspace_size(img.numel()), img.device)
    _check("iq_quantize_image_u8",
           load().iq_quantize_image_u8(_p(img), n, h, w, c, int(nchw), c_out, _p(codes),
                                       _p(scale), _p(ws), ws.numel(), _stream(stream)))


def iq_requantize(q, s_in, k, mode, codes, s_out, seed=0, layer=0, step=0, tag=0, ws=None,
                  stream=None):
    in_dtype = {torch.int32: IQ_I32, torch.int64: IQ_I64}[q.dtype]
    out_dtype = {torch.int8: IQ_I8, torch.int16: IQ_I16, torch.int32: IQ_I32}[codes.dtype]
    if ws is None:
        ws = _ws(iq_quantize_workspace_size(q.numel()), q.device)
    _check("iq_requantize",
           load().iq_requantize(_p(q), in_dtype, q.numel(), _p(s_in), k, mode, seed, layer, step,
                                tag, _p(codes), out_dtype, _p(s_out), _p(ws), ws.numel(),
                                _stream(stream)))


def iq_requantize_per_channel_workspace_size(c: int) -> int:
    n = _SZ(0)
    _check("iq_requantize_per_channel_workspace_size",
           load().iq_requantize_per_channel_workspace_size(c, C.byref(n)))
    return n.value


def iq_requantize_per_channel(q, outer, c, inner, s_in, k, codes, s_out, relu=False, ws=None,
                              stream=None):
    """Eq. (ScaleQ) with a per-channel Scale on q viewed as [outer][c][inner]; s_out[c]."""
    in_dtype = {torch.int32: IQ_I32, torch.int64: IQ_I64}[q.dtype]
    out_dtype = {torch.int8: IQ_I8, torch.int16: IQ_I16, torch.int32: IQ_I32}[codes.dtype]
    if ws is None:
        ws = _ws(iq_requantize_per_channel_workspace_size(c), q.device)
    _check("iq_requantize_per_channel",
           load().iq_requantize_per_channel(_p(q), in_dtype, outer, c, inner, _p(s_in), k,
                                            int(relu), _p(codes), out_dtype, _p(s_out), _p(ws),
                                            ws.numel(), _stream(stream)))


def iq_weight_decay(master, wq, shift, k_u=24, k_w=8, stream=None):
    """Decoupled L2 decay of the k_u-grid masters (decay step 2^-shift), W_q regenerated."""
    _check("iq_weight_decay", load().iq_weight_decay(_p(master), _p(wq), master.numel(), shift,
                                                     k_u, k_w, _stream(stream)))


def iq_gemm_s8_nibble(a, b, c, ws=None, stream=None):
    """c[m][n] = a[m][k] b[n][k]^T (int8 -> int32, exact) on the fp8 nibble-split route."""
    m, k = a.shape
    n = b.shape[0]
    if ws is None:
        nb = _SZ(0)
        _check("iq_gemm_s8_nibble_workspace_size",
               load().iq_gemm_s8_nibble_workspace_size(m, n, k, C.byref(nb)))
        ws = _ws(nb.value, a.device)
    _check("iq_gemm_s8_nibble",
           load().iq_gemm_s8_nibble(_p(a), _p(b), _p(c), m, n, k, _p(ws), ws.numel(),
                                    _stream(stream)))


def iq_weight_requant(master, wq, k_u=24, k_w=8, stream=None):
    _check("iq_weight_requant", load().iq_weight_requant(_p(master), _p(wq), master.numel(), k_u,
                                                         k_w, _stream(stream)))


def iq_conv_fwd(d: ConvDesc, x, s_x, w, a, s_a, gamma=None, beta=None, bits=None, use_bn=False,
                relu=True, xhat=None, bn_codes=None, bn_scales=None, frozen_out=None, acc_out=None,
                x_f16=None, a_f16=None, ws=None, stream=None):
    if ws is None:
        ws = _ws(iq_conv_fwd_workspace_size(d, use_bn), x.device)
    _check("iq_conv_fwd",
           load().iq_conv_fwd(C.byref(d), _p(x), _p(s_x), _p(w), _p(gamma), _p(beta),
                              C.byref(bits) if bits is not None else None, int(use_bn),
                              int(relu), _p(a), _p(s_a), _p(xhat), _p(bn_codes), _p(bn_scales),
                              _p(frozen_out), _p(acc_out), _p(x_f16), _p(a_f16), _p(ws),
                              ws.numel(), _stream(stream)))


def iq_conv_fwd_frozen(d: ConvDesc, x, w, frozen, a, use_bn=False, relu=True, bits=None,
                       xhat=None, x_f16=None, ws=None, stream=None):
    if ws is None:
        ws = _ws(iq_conv_fwd_workspace_size(d, use_bn), x.device)
    _check("iq_conv_fwd_frozen",
           load().iq_conv_fwd_frozen(C.byref(d), _p(x), _p(w), _p(frozen),
                                     C.byref(bits) if bits is not None else None, int(use_bn),
                                     int(relu), _p(a), _p(xhat), _p(x_f16), _p(ws), ws.numel(),
                                     _stream(stream)))


def iq_conv_dgrad(d: ConvDesc, e, s_e, w, dx, s_dx, acc_out=None, e_f16=None, dx_mask=None,
                  dx_f16=None, ws=None, stream=None):
    if ws is None:
        ws = _ws(iq_conv_dgrad_workspace_size(d), e.device)
    _check("iq_conv_dgrad",
           load().iq_conv_dgrad(C.byref(d), _p(e), _p(s_e), _p(w), _p(dx), _p(s_dx), _p(acc_out),
                                _p(e_f16), _p(dx_mask), _p(dx_f16), _p(ws), ws.numel(),
                                _stream(stream)))


def iq_conv_wgrad(d: ConvDesc, e, s_e, x, s_x, g, s_g, gq_mode=1, seed=0, layer=0, step=0,
                  g_acc_out=None, e_f16=None, x_f16=None, ws=None, stream=None):
    if ws is None:
        ws = _ws(iq_conv_wgrad_workspace_size(d), e.device)
    _check("iq_conv_wgrad",
           load().iq_conv_wgrad(C.byref(d), _p(e), _p(s_e), _p(x), _p(s_x), gq_mode, seed, layer,
                                step, _p(g), _p(s_g), _p(g_acc_out), _p(e_f16), _p(x_f16),
                                _p(ws), ws.numel(), _stream(stream)))


def iq_bn_int_fwd(acc, s_acc, gamma, beta, a, s_a, xhat=None, bn_codes=None, bn_scales=None,
                  bn_fixed=None, bits=None, ws=None, stream=None):
    c = acc.shape[-1]
    m = acc.numel() // c
    if ws is None:
        ws = _ws(iq_bn_int_workspace_size(m, c), acc.device)
    _check("iq_bn_int_fwd",
           load().iq_bn_int_fwd(_p(acc), m, c, _p(s_acc), _p(gamma), _p(beta),
                                C.byref(bits) if bits is not None else None, _p(xhat), _p(a),
                                _p(s_a), _p(bn_codes), _p(bn_scales), _p(bn_fixed), _p(ws),
                                ws.numel(), _stream(stream)))


def iq_bn_int_bwd(e_a, s_e, a, xhat, gamma, bn_codes, bn_scales, e, s_e_out, dgamma=None,
                  dbeta=None, k_e2=16, bits=None, e_f16=None, ws=None, stream=None):
    c = e_a.shape[-1]
    m = e_a.numel() // c
    if ws is None:
        ws = _ws(iq_bn_int_workspace_size(m, c), e_a.device)
    _check("iq_bn_int_bwd",
           load().iq_bn_int_bwd(_p(e_a), _p(s_e), _p(a), _p(xhat), m, c, _p(gamma), _p(bn_codes),
                                _p(bn_scales), C.byref(bits) if bits is not None else None, k_e2,
                                _p(e), _p(s_e_out), _p(dgamma), _p(dbeta), _p(e_f16), _p(ws),
                                ws.numel(), _stream(stream)))


def iq_relu_bwd(e_a, a, e, e_f16=None, stream=None):
    _check("iq_relu_bwd", load().iq_relu_bwd(_p(e_a), _p(a), e_a.numel(), _p(e), _p(e_f16),
                                             _stream(stream)))


def iq_update(master, wq, g, s_g, lr_log2, k_u=24, k_w=8, x2=False, stream=None):
    _check("iq_update", load().iq_update(_p(master), _p(wq), _p(g), _p(s_g), master.numel(),
                                         lr_log2, k_u, k_w, int(x2), _stream(stream)))


# ---------------------------------------------------------------- network glue

def iq_maxpool_fwd(x, k, s, p, y, arg, y_f16=None, stream=None):
    n, h, w, c = x.shape
    _check("iq_maxpool_fwd", load().iq_maxpool_fwd(_p(x), n, h, w, c, k, s, p, _p(y), _p(arg),
                                                   _p(y_f16), _stream(stream)))


def iq_maxpool_bwd(e, s_e, arg, in_shape, k, s, p, ex, s_ex, ws=None, stream=None):
    n, h, w, c = in_shape
    if ws is None:
        ws = _ws(n * h * w * c * 4 + 4096, e.device)
    _check("iq_maxpool_bwd", load().iq_maxpool_bwd(_p(e), _p(s_e), _p(arg), n, h, w, c, k, s, p,
                                                   _p(ex), _p(s_ex), _p(ws), ws.numel(),
                                                   _stream(stream)))


def iq_upsample_workspace_size(n, h, w, c, R) -> int:
    return _size("iq_upsample_workspace_size", n, h, w, c, R)


def iq_upsample_fwd(x, s_x, w, R, stride, pad, out, s_out, acc_out=None, ws=None, stream=None):
    n, h, wd, c = x.shape
    if ws is None:
        ws = _ws(iq_upsample_workspace_size(n, h, wd, c, R), x.device)
    _check("iq_upsample_fwd", load().iq_upsample_fwd(_p(x), _p(s_x), _p(w), n, h, wd, c, R, stride,
                                                     pad, _p(out), _p(s_out), _p(acc_out), _p(ws),
                                                     ws.numel(), _stream(stream)))


def iq_upsample_bwd(E, s_e, w, x_shape, R, stride, pad, ex, s_ex, acc_out=None, ws=None,
                    stream=None):
    n, h, wd, c = x_shape
    if ws is None:
        ws = _ws(iq_upsample_workspace_size(n, h, wd, c, R), E.device)
    _check("iq_upsample_bwd", load().iq_upsample_bwd(_p(E), _p(s_e), _p(w), n, h, wd, c, R, stride,
                                                     pad, _p(ex), _p(s_ex), _p(acc_out), _p(ws),
                                                     ws.numel(), _stream(stream)))


def iq_upsample_wgrad(x, s_x, E, s_e, R, stride, pad, g, s_g, gq_mode=2, seed=0, layer=0, step=0,
                      g_acc_out=None, ws=None, stream=None):
    n, h, wd, c = x.shape
    if ws is None:
        ws = _ws(iq_upsample_workspace_size(n, h, wd, c, R), x.device)
    _check("iq_upsample_wgrad",
           load().iq_upsample_wgrad(_p(x), _p(s_x), _p(E), _p(s_e), n, h, wd, c, R, stride, pad,
                                    gq_mode, seed, layer, step, _p(g), _p(s_g), _p(g_acc_out),
                                    _p(ws), ws.numel(), _stream(stream)))


def iq_mse_grad(z, s_z, labels, E, s_e, ws=None, stream=None):
    c = z.shape[-1]
    if ws is None:
        ws = _ws(4096, z.device)
    _check("iq_mse_grad", load().iq_mse_grad(_p(z), _p(s_z), _p(labels), z.numel() // c, c, _p(E),
                                             _p(s_e), _p(ws), ws.numel(), _stream(stream)))


def iq_bn_int_fwd_noalloc(acc, s_acc, gamma, beta, a, s_a, xhat=None, bn_codes=None,
                          bn_scales=None, bn_fixed=None, bits=None, stream=None):
    """iq_bn_int_fwd for callers that cannot allocate: no workspace argument."""
    c = acc.shape[-1]
    m = acc.numel() // c
    _check("iq_bn_int_fwd_noalloc",
           load().iq_bn_int_fwd_noalloc(_p(acc), m, c, _p(s_acc), _p(gamma), _p(beta),
                                        C.byref(bits) if bits is not None else None, _p(xhat),
                                        _p(a), _p(s_a), _p(bn_codes), _p(bn_scales),
                                        _p(bn_fixed), _stream(stream)))


# ---------------------------------------------------------------- DeepLab glue

def term(codes, scale, c_offset=0, bcast=False, gamma=None, beta=None, k_gamma=8, k_beta=8):
    """An iq_term over device tensors: codes int8/int16 [..., c], scale a device double
    (tensor, or an int device address such as bn_scales' IQ_BN_S_XHAT element)."""
    dt = {torch.int8: IQ_I8, torch.int16: IQ_I16}[codes.dtype]
    return Term(codes.data_ptr(), dt, codes.shape[-1], c_offset, int(bcast), _p(scale),
                _p(gamma), _p(beta), k_gamma, k_beta)


def iq_combine_workspace_size(terms) -> int:
    arr = (Term * len(terms))(*terms)
    b = _SZ()
    _check("iq_combine_workspace_size", load().iq_combine_workspace_size(arr, len(terms), C.byref(b)))
    return b.value


def iq_combine(terms, n, hw, c_out, out, s_out, concat=False, relu=False, out_f16=None, ws=None,
               stream=None):
    arr = (Term * len(terms))(*terms)
    if ws is None:
        ws = _ws(iq_combine_workspace_size(terms), out.device)
    _check("iq_combine", load().iq_combine(arr, len(terms), int(concat), n, hw, c_out, int(relu),
                                           _p(out), _p(s_out), _p(out_f16), _p(ws), ws.numel(),
                                           _stream(stream)))


def iq_spatial_sum_workspace_size(n, c) -> int:
    return _size("iq_spatial_sum_workspace_size", n, c)


def iq_spatial_sum(x, s_x, out, s_out, mean=True, c_off=0, c=None, ws=None, stream=None):
    n, c_total = x.shape[0], x.shape[-1]
    hw = x.numel() // (n * c_total)
    c = c_total - c_off if c is None else c
    if ws is None:
        ws = _ws(iq_spatial_sum_workspace_size(n, c), x.device)
    _check("iq_spatial_sum", load().iq_spatial_sum(_p(x), _p(s_x), n, hw, c_total, c_off, c,
                                                   int(mean), _p(out), _p(s_out), _p(ws),
                                                   ws.numel(), _stream(stream)))


def iq_avgpool_bwd(e, s_e, hw, s_ex, ex=None, stream=None):
    n, c = e.shape[0], e.shape[-1]
    _check("iq_avgpool_bwd", load().iq_avgpool_bwd(_p(e), _p(s_e), n, hw, c, _p(ex), _p(s_ex),
                                                   _stream(stream)))


def iq_channel_slice(x, c_off, c, out, stream=None):
    c_total = x.shape[-1]
    _check("iq_channel_slice", load().iq_channel_slice(_p(x), x.numel() // c_total, c_total, c_off,
                                                       c, _p(out), _stream(stream)))


def iq_bilinear_workspace_size(n, h, w, c) -> int:
    return _size("iq_bilinear_workspace_size", n, h, w, c)


def iq_bilinear_up_fwd(x, s_x, f, out, s_out, ws=None, stream=None):
    n, h, w, c = x.shape
    if ws is None:
        ws = _ws(iq_bilinear_workspace_size(n, h, w, c), x.device)
    _check("iq_bilinear_up_fwd", load().iq_bilinear_up_fwd(_p(x), _p(s_x), n, h, w, c, f, _p(out),
                                                           _p(s_out), _p(ws), ws.numel(),
                                                           _stream(stream)))


def iq_bilinear_up_bwd(e, s_e, f, in_shape, ex, s_ex, ws=None, stream=None):
    n, h, w, c = in_shape
    if ws is None:
        ws = _ws(iq_bilinear_workspace_size(n, h, w, c), e.device)
    _check("iq_bilinear_up_bwd", load().iq_bilinear_up_bwd(_p(e), _p(s_e), n, h, w, c, f, _p(ex),
                                                           _p(s_ex), _p(ws), ws.numel(),
                                                           _stream(stream)))


def iq_ce_grad(z, s_z, labels, E, s_e, n_valid=None, ignore=255, ws=None, stream=None):
    c = z.shape[-1]
    if ws is None:
        ws = _ws(4096, z.device)
    _check("iq_ce_grad", load().iq_ce_grad(_p(z), _p(s_z), _p(labels), z.numel() // c, c, ignore,
                                           _p(E), _p(s_e), _p(n_valid), _p(ws), ws.numel(),
                                           _stream(stream)))


def iq_bn_update(gamma_master, beta_master, gamma, beta, dgamma, dbeta, s_e, bn_scales, lr_log2,
                 seed, layer, step, k_u=24, bits=None, ws=None, stream=None):
    """ws is accepted for compatibility and ignored: the update needs no scratch."""
    c = gamma.numel()
    _check("iq_bn_update", load().iq_bn_update(_p(gamma_master), _p(beta_master), _p(gamma),
                                               _p(beta), _p(dgamma), _p(dbeta), _p(s_e),
                                               _p(bn_scales), c,
                                               C.byref(bits) if bits is not None else None,
                                               lr_log2, k_u, seed, layer, step, None, 0,
                                               _stream(stream)))
