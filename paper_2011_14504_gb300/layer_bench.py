"""Time one integer 3x3 convolution layer (stride 1, padding 1), or one integer L1BN,
through the C ABI; or run one step of a network once (a profiling target).

    python -m paper_2011_14504_gb300.layer_bench [N,H,C,K] [time|once]
    python -m paper_2011_14504_gb300.layer_bench bn M,C [time|once]
    python -m paper_2011_14504_gb300.layer_bench step deeplab|fcn BATCH [train|infer]
    python -m paper_2011_14504_gb300.layer_bench gemm M,N,K [time|once]
    python -m paper_2011_14504_gb300.layer_bench join C16,C8 [time|once]

Runs iq_conv_fwd (with ReLU and the SQ8 requantisation of the output), iq_conv_dgrad and
iq_conv_wgrad (GQ8 gradient) of an N x H x H x C -> K layer on random 8-bit codes.  "time"
(the default) prints each call's CUDA-event duration over 10 calls after 3 warm-up calls and
the int8 multiply-accumulate rate it implies (2 ops per MAC); "once" makes one call of each,
which is the form used under a profiler.  The bn form runs iq_bn_int_fwd on M x C random
int32 accumulators (L1BN, ReLU, Q_A) and iq_bn_int_bwd on random 8-bit errors, and prints
each call's duration and its DRAM bytes per element over that time.  The join form times
iq_combine on a residual join of two int16 operands and a sum of two int8 errors.
"""
import sys

import torch

from . import iq


def _time(f, mode):
    if mode != "time":
        f()
        return None
    for _ in range(3):
        f()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(10):
        f()
    t1.record()
    torch.cuda.synchronize()
    return t0.elapsed_time(t1) / 10


def bn_main(argv):
    m, c = [int(v) for v in (argv[0] if argv else "67600,1024").split(",")]
    mode = argv[1] if len(argv) > 1 else "time"
    dev = "cuda"
    g = torch.Generator(device=dev)
    g.manual_seed(1)
    acc = (torch.randn((m, c), generator=g, device=dev) * 4000).to(torch.int32)
    gam = torch.randint(-127, 128, (c,), generator=g, device=dev, dtype=torch.int32)
    bet = torch.randint(-127, 128, (c,), generator=g, device=dev, dtype=torch.int32)
    ea = torch.randint(-127, 128, (m, c), generator=g, device=dev, dtype=torch.int8)
    s_acc = torch.tensor([2.0 ** -14], dtype=torch.float64, device=dev)
    s_e = torch.tensor([2.0 ** -21], dtype=torch.float64, device=dev)
    a = torch.empty((m, c), dtype=torch.int8, device=dev)
    x = torch.empty((m, c), dtype=torch.int16, device=dev)
    e = torch.empty((m, c), dtype=torch.int8, device=dev)
    codes = torch.empty(2 * c, dtype=torch.int32, device=dev)
    scal = torch.empty(iq.IQ_BN_SCALES, dtype=torch.float64, device=dev)
    s_a, s_out = torch.empty_like(s_acc), torch.empty_like(s_acc)
    ws = torch.empty(iq.iq_bn_int_workspace_size(m, c), dtype=torch.uint8, device=dev)
    fwd = lambda: iq.iq_bn_int_fwd(acc, s_acc, gam, bet, a, s_a, xhat=x, bn_codes=codes,
                                   bn_scales=scal, ws=ws)
    bwd = lambda: iq.iq_bn_int_bwd(ea, s_e, a, x, gam, codes, scal, e, s_out, ws=ws)
    # bytes per element: fwd reads the int32 sums three times (sums, deviation,
    # requantisation) and
    # writes X (int16) and A (int8); bwd reads e_a, A, X three times and writes E (int8)
    for name, f, nb in (("bn_fwd", fwd, 15), ("bn_bwd", bwd, 13)):
        ms = _time(f, mode)
        if ms is not None:
            print(f"{name}: {ms:.3f} ms  {nb * m * c / ms / 1e6:.0f} GB/s at {nb} B/element")
    torch.cuda.synchronize()
    print("ok")


def join_main(argv):
    """One residual join of two int16 X-code operands with the BN affine and ReLU (the
    downsampling blocks' form) and one sum of two int8 errors, both 65 x 65 x C at batch 16
    (the stage-3 and stage-4 shapes of the DeepLab step), through iq_combine with the fp16
    output copy."""
    c16, c8 = [int(v) for v in (argv[0] if argv else "1024,2048").split(",")]
    mode = argv[1] if len(argv) > 1 else "time"
    dev = "cuda"
    g = torch.Generator(device=dev)
    g.manual_seed(3)
    n, hw = 16, 65 * 65

    def sc(v):
        return torch.tensor([v], dtype=torch.float64, device=dev)

    keep = []
    cases = []
    X = [torch.randint(-32767, 32768, (n, hw, c16), generator=g, device=dev, dtype=torch.int16)
         for _ in range(2)]
    gb = [torch.randint(-127, 128, (c16,), generator=g, device=dev, dtype=torch.int32)
          for _ in range(4)]
    s16 = [sc(2.5e-5), sc(3.1e-5)]
    keep += X + gb + s16
    cases.append(("residual join, int16 + int16", c16, True, 9,
                  [iq.term(X[0], s16[0], gamma=gb[0], beta=gb[1]),
                   iq.term(X[1], s16[1], gamma=gb[2], beta=gb[3])]))
    E = [torch.randint(-127, 128, (n, hw, c8), generator=g, device=dev, dtype=torch.int8)
         for _ in range(2)]
    s8 = [sc(1.1e-6), sc(0.9e-6)]
    keep += E + s8
    cases.append(("error sum, int8 + int8", c8, False, 5, [iq.term(E[0], s8[0]),
                                                           iq.term(E[1], s8[1])]))
    for name, c, relu, nb, terms in cases:
        out = torch.empty((n, hw, c), dtype=torch.int8, device=dev)
        out16 = torch.empty(out.numel(), dtype=torch.float16, device=dev)
        so = sc(0.0)
        ws = torch.empty(iq.iq_combine_workspace_size(terms), dtype=torch.uint8, device=dev)
        f = lambda: iq.iq_combine(terms, n, hw, c, out, so, relu=relu, out_f16=out16, ws=ws)
        ms = _time(f, mode)
        if ms is not None:
            # both passes read the operands, the codes pass writes the codes and their copy
            print(f"{name} (c = {c}): {ms:.3f} ms  {(nb + 2) * n * hw * c / ms / 1e6:.0f} GB/s "
                  f"at {nb + 2} B/element")
    torch.cuda.synchronize()
    assert iq.iq_device_status() == 0
    print("ok")


def step_main(argv):
    """Exactly one training step (or inference pass) of the full-width network on synthetic
    inputs (batch BATCH, 513 x 513 or 512 x 512), no warm-up: under a profiler every launch
    of the run belongs to that one step."""
    import numpy as np
    from . import synthetic as S
    net_name, batch = argv[0], int(argv[1])
    train = (argv[2] if len(argv) > 2 else "train") == "train"
    g = S.rng(7)
    if net_name == "deeplab":
        from .deeplab import DeepLabV3R50
        net = DeepLabV3R50(batch, 513, 513, classes=21, train=train)
        img = torch.from_numpy(S.images_u8(g, batch, 513, 513)).cuda()
        lab = torch.from_numpy(S.labels_uniform_ignore(g, batch, 513, 513, 21)).cuda()
    else:
        from .fcn import FcnVgg16
        net = FcnVgg16(batch, 512, 512, classes=150, train=train)
        img = torch.from_numpy(S.images_u8(g, batch, 512, 512)).cuda()
        lab = torch.from_numpy(S.labels_voronoi(g, batch, 512, 512, 150)).cuda()
    torch.cuda.synchronize()
    l0 = iq.launch_count()
    if train:
        net.train_step(img, lab)
    else:
        net.forward(img)
    torch.cuda.synchronize()
    assert iq.iq_device_status() == 0
    print(f"{net_name} batch {batch} {'train step' if train else 'inference'}: "
          f"{iq.launch_count() - l0} library launches")
    print("ok")


def gemm_main(argv):
    """The exact int8 GEMM C = A B^T two ways: the fp8 nibble-split route (iq_gemm_s8_nibble,
    four kind::f8f6f4 MMAs per k-step) and the fp16-carrier route of a 1x1 iq_conv_fwd."""
    m, n, k = [int(v) for v in (argv[0] if argv else "8192,8192,4096").split(",")]
    mode = argv[1] if len(argv) > 1 else "time"
    dev = "cuda"
    g = torch.Generator(device=dev)
    g.manual_seed(3)
    a = torch.randint(-128, 128, (m, k), generator=g, device=dev, dtype=torch.int8)
    b = torch.randint(-128, 128, (n, k), generator=g, device=dev, dtype=torch.int8)
    c = torch.empty((m, n), dtype=torch.int32, device=dev)
    d = iq.conv_desc(1, 1, m, k, n, 1, 1)
    acc = torch.empty((1, 1, m, n), dtype=torch.int32, device=dev)
    codes = torch.empty((1, 1, m, n), dtype=torch.int8, device=dev)
    one = torch.ones(1, dtype=torch.float64, device=dev)
    s_out = torch.empty(1, dtype=torch.float64, device=dev)
    ws = torch.empty(iq.iq_conv_fwd_workspace_size(d, False), dtype=torch.uint8, device=dev)
    routes = [("fp8 nibble split (kind::f8f6f4)", lambda: iq.iq_gemm_s8_nibble(a, b, c)),
              ("fp16 carriers (kind::f16, 1x1 conv)",
               lambda: iq.iq_conv_fwd(d, a, one, b, codes, s_out, relu=False, acc_out=acc, ws=ws))]
    for name, f in routes:
        ms = _time(f, mode)
        if ms is not None:
            print(f"{name}: {ms:.3f} ms  {2.0 * m * n * k / ms / 1e9:.0f} TOPS (whole call)")
    if mode == "time":
        iq.iq_kernel_timing_begin()
        for _, f in routes:
            f()
        for r in iq.iq_kernel_timing_end():
            if r["op"] in (1, 4):
                print(f"kernel {r['kernel']}: {r['ms']:.3f} ms  "
                      f"{2.0 * r['macs'] / r['ms'] / 1e9:.0f} TOPS")
    torch.cuda.synchronize()
    print("ok")


def main(argv=None):
    argv = sys.argv[1:] if argv is None else argv
    if argv and argv[0] == "bn":
        return bn_main(argv[1:])
    if argv and argv[0] == "step":
        return step_main(argv[1:])
    if argv and argv[0] == "gemm":
        return gemm_main(argv[1:])
    if argv and argv[0] == "join":
        return join_main(argv[1:])
    n, h, c, k = [int(v) for v in (argv[0] if argv else "8,128,256,256").split(",")]
    mode = argv[1] if len(argv) > 1 else "time"
    dev = "cuda"
    d = iq.conv_desc(n, h, h, c, k, 3, 3, 1, 1)
    x = torch.randint(-127, 128, (n, h, h, c), dtype=torch.int8, device=dev)
    wq = torch.randint(-127, 128, (k, 3, 3, c), dtype=torch.int8, device=dev)
    e = torch.randint(-127, 128, (n, h, h, k), dtype=torch.int8, device=dev)
    a = torch.empty((n, h, h, k), dtype=torch.int8, device=dev)
    dx = torch.empty((n, h, h, c), dtype=torch.int8, device=dev)
    g = torch.empty((k, 3, 3, c), dtype=torch.int8, device=dev)
    sx = torch.tensor([0.01], dtype=torch.float64, device=dev)
    sa, sdx, sg = torch.empty_like(sx), torch.empty_like(sx), torch.empty_like(sx)
    wsz = max(iq.iq_conv_fwd_workspace_size(d), iq.iq_conv_dgrad_workspace_size(d),
              iq.iq_conv_wgrad_workspace_size(d))
    ws = torch.empty(wsz, dtype=torch.uint8, device=dev)
    macs = n * h * h * k * 9 * c
    ops = {"fwd": lambda: iq.iq_conv_fwd(d, x, sx, wq, a, sa, relu=True, ws=ws),
           "dgrad": lambda: iq.iq_conv_dgrad(d, e, sx, wq, dx, sdx, ws=ws),
           "wgrad": lambda: iq.iq_conv_wgrad(d, e, sx, x, sx, g, sg, gq_mode=2, ws=ws)}
    for name, f in ops.items():
        if mode == "time":
            for _ in range(3):
                f()
            torch.cuda.synchronize()
            t0 = torch.cuda.Event(enable_timing=True)
            t1 = torch.cuda.Event(enable_timing=True)
            t0.record()
            for _ in range(10):
                f()
            t1.record()
            torch.cuda.synchronize()
            ms = t0.elapsed_time(t1) / 10
            print(f"{name}: {ms:.3f} ms  {2 * macs / ms / 1e9:.1f} TOPS")
        else:
            f()
    torch.cuda.synchronize()
    print("ok")


if __name__ == "__main__":
    main()
