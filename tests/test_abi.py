"""CPU-side checks of the C ABI: the library builds and loads, exports every entry point
that include/iq.h declares, and rejects bad arguments before launching anything."""
import ctypes as C
import os
import re
import subprocess

import pytest

from paper_2011_14504_gb300 import build as B
from paper_2011_14504_gb300 import iq

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_entry_points():
    src = open(os.path.join(ROOT, "include", "iq.h")).read()
    return sorted(set(re.findall(r"^\s*(?:iq_status|const char\*|int|unsigned long long)\s+(iq_\w+)\s*\(", src,
                                 re.M)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return iq.load()


def test_every_declared_symbol_is_exported(lib):
    decl = declared_entry_points()
    assert len(decl) >= 19
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (iq_\w+)", out))
    missing = [d for d in decl if d not in exported]
    assert not missing, missing
    assert sorted(decl) == sorted(iq.EXPORTS)


def test_status_strings_and_version(lib):
    assert iq.status_str(0) == "ok"
    assert "workspace" in iq.status_str(3)
    assert lib.iq_version() >= 1


def test_conv_out_size_and_workspace_queries(lib):
    d = iq.conv_desc(1, 32, 32, 64, 64, 3, 3, 1, 1)
    assert iq.iq_conv_out_size(d) == (32, 32)
    d2 = iq.conv_desc(2, 65, 65, 256, 256, 3, 3, 1, 24, 24)    # ASPP rate 24 on 65x65
    assert iq.iq_conv_out_size(d2) == (65, 65)
    d3 = iq.conv_desc(16, 513, 513, 4, 64, 7, 7, 2, 3)          # stem
    assert iq.iq_conv_out_size(d3) == (257, 257)
    assert iq.iq_conv_fwd_workspace_size(d) >= 32 * 32 * 64 * 4
    assert iq.iq_conv_dgrad_workspace_size(d) >= 32 * 32 * 64 * 4
    assert iq.iq_conv_wgrad_workspace_size(d) >= 64 * 9 * 64 * 8
    assert iq.iq_bn_int_workspace_size(1024, 64) > 0
    # NCHW calls stage their transposes in front of the NHWC workspace
    dn = iq.conv_desc(1, 32, 32, 64, 64, 3, 3, 1, 1, layout=iq.IQ_LAYOUT_NCHW)
    for f in (iq.iq_conv_fwd_workspace_size, iq.iq_conv_dgrad_workspace_size,
              iq.iq_conv_wgrad_workspace_size):
        assert f(dn) >= f(d) + 2 * 32 * 32 * 64


def test_conv_desc_layout_and_widths_validated(lib):
    """The descriptor's layout and code widths: NHWC / NCHW, k_w and k_a in 2..8 (0: 8 bits),
    flags from IQ_CONV_X_F16_READY | IQ_CONV_E_F16_READY; anything else is rejected by the
    host-side checks."""
    ok = [dict(), dict(layout=iq.IQ_LAYOUT_NCHW), dict(k_w=4, k_a=4), dict(k_w=2, k_a=8),
          dict(flags=iq.IQ_CONV_X_F16_READY), dict(flags=iq.IQ_CONV_E_F16_READY),
          dict(flags=iq.IQ_CONV_X_F16_READY | iq.IQ_CONV_E_F16_READY)]
    bad = [dict(layout=2), dict(layout=-1), dict(k_w=1), dict(k_w=9), dict(k_a=1), dict(k_a=16),
           dict(flags=4), dict(flags=-1)]
    for kw in ok:
        assert iq.iq_conv_out_size(iq.conv_desc(1, 8, 8, 8, 8, 3, 3, 1, 1, **kw)) == (8, 8)
    for kw in bad:
        with pytest.raises(iq.IqError) as e:
            iq.iq_conv_out_size(iq.conv_desc(1, 8, 8, 8, 8, 3, 3, 1, 1, **kw))
        assert e.value.code == iq.IQ_ERR_INVALID_ARG


def test_kernel_timing_host_side(lib):
    # with nothing launched between begin and end: no rows, no device work; null outputs
    # are rejected
    iq.iq_kernel_timing_begin()
    assert iq.iq_kernel_timing_end() == []
    n = C.c_int32(0)
    assert lib.iq_kernel_timing_end(None, 4, C.byref(n)) == iq.IQ_ERR_INVALID_ARG
    out = (iq.KernelTime * 2)()
    assert lib.iq_kernel_timing_end(out, 2, None) == iq.IQ_ERR_INVALID_ARG
    # the struct layout the header declares: 4 int32 then 4 doubles
    assert C.sizeof(iq.KernelTime) == 48


def test_invalid_arguments_rejected_before_launch(lib):
    bad = iq.conv_desc(1, 8, 8, 6, 4, 3, 3, 1, 1, 1, 4)        # C not divisible by groups
    with pytest.raises(iq.IqError) as e:
        iq.iq_conv_out_size(bad)
    assert e.value.code == iq.IQ_ERR_INVALID_ARG
    d = iq.conv_desc(1, 8, 8, 8, 8, 3, 3, 1, 1)
    rc = lib.iq_conv_fwd(C.byref(d), None, None, None, None, None, None, 0, 1, None, None, None,
                         None, None, None, None, None, None, None, 0, None)
    assert rc == iq.IQ_ERR_INVALID_ARG
    # a shape beyond the int32 accumulation bound: 1024*12*12*127^2 >= 2^31
    big = iq.conv_desc(1, 12, 12, 1024, 8, 12, 12)
    rc = lib.iq_conv_fwd(C.byref(big), 1, 1, 1, None, None, None, 0, 1, 1, 1, None, None, None,
                         None, None, None, None, None, 0, None)
    assert rc == iq.IQ_ERR_OVERFLOW_RISK
    # workspace too small
    rc = lib.iq_conv_fwd(C.byref(d), 1, 1, 1, None, None, None, 0, 1, 1, 1, None, None, None,
                         None, None, None, None, None, 16, None)
    assert rc == iq.IQ_ERR_WORKSPACE
    # an fp16 carrier that is not 16-byte aligned
    rc = lib.iq_conv_fwd(C.byref(d), 16, 1, 1, None, None, None, 0, 1, 1, 1, None, None, None,
                         None, None, 24, None, None, 1 << 30, None)
    assert rc == iq.IQ_ERR_INVALID_ARG
    # an fp16 output copy that is not 16-byte aligned
    rc = lib.iq_conv_fwd(C.byref(d), 16, 1, 16, None, None, None, 0, 1, 16, 1, None, None, None,
                         None, None, None, 24, None, 1 << 30, None)
    assert rc == iq.IQ_ERR_INVALID_ARG
    # the same for the other producers of fp16 copies, rejected before any launch
    assert lib.iq_relu_bwd(16, 16, 32, 16, 24, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_relu_bwd(16, 16, 40, 16, 32, None) == iq.IQ_ERR_INVALID_ARG   # n % 16
    assert lib.iq_maxpool_fwd(16, 1, 8, 8, 16, 2, 2, 0, 16, 16, 24, None) == iq.IQ_ERR_INVALID_ARG
    # the data gradient's ReLU mask and fp16 copy: NHWC only, the copy 16-byte aligned
    dn = iq.conv_desc(1, 8, 8, 16, 16, 3, 3, 1, 1, layout=iq.IQ_LAYOUT_NCHW)
    assert lib.iq_conv_dgrad(C.byref(dn), 16, 16, 16, 16, 16, None, None, 16, None, 16, 1 << 20,
                             None) == iq.IQ_ERR_UNSUPPORTED
    assert lib.iq_conv_dgrad(C.byref(d), 16, 16, 16, 16, 16, None, None, 16, 24, 16, 1 << 30,
                             None) == iq.IQ_ERR_INVALID_ARG
    # bad bit width / dtype combination
    rc = lib.iq_quantize(1, 10, 16, iq.IQ_MODE_UQ, iq.IQ_I8, 1, 1, 1, 4096, None)
    assert rc == iq.IQ_ERR_INVALID_ARG
    rc = lib.iq_requantize(1, iq.IQ_I32, 10, 1, 8, 99, 0, 0, 0, 0, 1, iq.IQ_I8, 1, 1, 4096, None)
    assert rc == iq.IQ_ERR_INVALID_ARG
    # BN needs C % 4 == 0
    rc = lib.iq_bn_int_fwd(16, 10, 6, 1, 1, 1, None, None, 16, 1, None, None, None, 16, 1 << 20,
                           None)
    assert rc == iq.IQ_ERR_UNSUPPORTED
    rc = lib.iq_update(1, 1, 1, 1, 10, -1, 24, 8, 0, None)
    assert rc == iq.IQ_ERR_INVALID_ARG


def test_glue_arguments_rejected_before_launch(lib):
    T = iq.Term
    ok = T(16, iq.IQ_I8, 8, 0, 0, 16, None, None, 8, 8)
    arr = (T * 9)(*([ok] * 9))
    assert lib.iq_combine(arr, 0, 0, 1, 4, 8, 0, 16, 16, None, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_combine(arr, 9, 0, 1, 4, 8, 0, 16, 16, None, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    # a sum whose operand does not cover every output channel
    assert lib.iq_combine(arr, 2, 0, 1, 4, 16, 0, 16, 16, None, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    # a concatenation operand past the last channel
    off = (T * 1)(T(16, iq.IQ_I8, 8, 4, 0, 16, None, None, 8, 8))
    assert lib.iq_combine(off, 1, 1, 1, 4, 8, 0, 16, 16, None, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    # gamma without beta, bad dtype
    half = (T * 1)(T(16, iq.IQ_I8, 8, 0, 0, 16, 16, None, 8, 8))
    assert lib.iq_combine(half, 1, 0, 1, 4, 8, 0, 16, 16, None, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    wide = (T * 1)(T(16, iq.IQ_I32, 8, 0, 0, 16, None, None, 8, 8))
    assert lib.iq_combine(wide, 1, 0, 1, 4, 8, 0, 16, 16, None, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    need = C.c_size_t()
    assert lib.iq_combine_workspace_size(arr, 2, C.byref(need)) == 0 and need.value >= 256 + 2 * 128
    assert lib.iq_combine(arr, 2, 0, 1, 4, 8, 0, 16, 16, None, 16, 64, None) == iq.IQ_ERR_WORKSPACE
    # an fp16 output copy off a 16-byte boundary
    assert lib.iq_combine(arr, 2, 0, 1, 4, 8, 0, 16, 16, 24, 16, 1 << 20, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_spatial_sum(16, 16, 2, 9, 8, 4, 8, 1, 16, 16, 16, 4096, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_spatial_sum(16, 16, 2, 9, 8, 0, 8, 1, 16, 16, 16, 8, None) == iq.IQ_ERR_WORKSPACE
    assert lib.iq_avgpool_bwd(None, 16, 2, 9, 8, None, 16, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_channel_slice(16, 10, 8, 6, 4, 16, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_bilinear_up_fwd(16, 16, 1, 4, 4, 3, 0, 16, 16, 16, 4096, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_bilinear_up_bwd(16, 16, 1, 4, 4, 3, 8, 16, 16, 16, 64, None) == iq.IQ_ERR_WORKSPACE
    assert lib.iq_ce_grad(16, 16, 16, 10, 2000, 255, 16, 16, None, 16, 4096, None) == iq.IQ_ERR_INVALID_ARG
    assert lib.iq_ce_grad(16, 16, 16, 10, 21, 255, 16, 16, None, 16, 8, None) == iq.IQ_ERR_WORKSPACE
    assert lib.iq_bn_update(16, 16, 16, 16, 16, None, 16, 16, 8, None, 10, 24, 0, 0, 0, 16, 1 << 16,
                            None) == iq.IQ_ERR_INVALID_ARG
    # more channels than the one-launch update takes (its workspace is reserved: NULL is fine)
    assert lib.iq_bn_update(16, 16, 16, 16, 16, 16, 16, 16, 4097, None, 10, 24, 0, 0, 0, None, 0,
                            None) == iq.IQ_ERR_UNSUPPORTED
