"""Time one integer 3x3 convolution layer (stride 1, padding 1) through the C ABI.

    python -m paper_2011_14504_gb300.layer_bench [N,H,C,K] [time|once]

Runs iq_conv_fwd (with ReLU and the SQ8 requantisation of the output), iq_conv_dgrad and
iq_conv_wgrad (GQ8 gradient) of an N x H x H x C -> K layer on random 8-bit codes.  "time"
(the default) prints each call's CUDA-event duration over 10 calls after 3 warm-up calls and
the int8 multiply-accumulate rate it implies (2 ops per MAC); "once" makes one call of each,
which is the form used under a profiler.
"""
import sys

import torch

from . import iq


def main(argv=None):
    argv = sys.argv[1:] if argv is None else argv
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
