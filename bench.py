"""Benchmark: the FCN-VGG16 quantized training step (int8 conv fwd + dgrad + wgrad, the
paper's Sec. 3 dataflow) on synthetic 512x512 segmentation batches.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line.  `value` is the int8 convolution throughput of the whole step in
TOPS (2 x MACs of every forward, data-gradient and weight-gradient convolution, the
decoder included, divided by the device time of the step), summed over all ranks.
Inputs are resident in HBM during the timed region; the working set of a step (several
GB) is far larger than the 129 MB L2, so no flush is needed between steps.  With
--gpus N > 1 (torchrun) every rank trains its own replica on its own batch (weak
scaling, no data-path collective).  --impl reference times the CPU oracle on a bounded
sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

BATCH, IMG, CLASSES, SITES = 16, 512, 150, 64
WORKLOAD = "fcn_vgg16_train_step"


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, \
            "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx = max(mx, float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(n_gpus: int):
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if os.environ.get("IQ_BENCH_GLOO") is None else "gloo")
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(v: float, world: int, device) -> float:
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ oracle (CPU) leg

def oracle_sample_step():
    """One FCN-VGG16 training step of the CPU oracle on a bounded sample of the workload:
    one image at 128x128 (the full-width network), about 10-30 s of CPU work."""
    import numpy as np
    from oracle.fcn import OracleFcn
    from paper_2011_14504_gb300 import synthetic as S
    n, h = 1, 128
    chans = S.fcn_vgg16_channels(CLASSES, 1.0)
    wts, up = S.fcn_vgg16_weights(0, CLASSES, 1.0)
    ora = OracleFcn(chans, wts, up, CLASSES, seed=0)
    g = S.rng(1)
    img = S.images_u8(g, n, h, h)
    lab = S.labels_voronoi(g, n, h, h, CLASSES, sites=SITES)
    macs = fcn_step_macs(n, h, h, CLASSES)

    def run():
        tr = ora.forward(img)
        ora.backward_update(tr, lab)
    return run, macs, f"FCN-VGG16 train step, N={n}, {h}x{h}, full width, {CLASSES} classes"


def fcn_step_macs(n, h, w, classes, width=1.0):
    from paper_2011_14504_gb300 import synthetic as S
    hh, ww = h, w
    f = dg = 0
    for name, cin, cout, r, pad, relu in S.fcn_vgg16_channels(classes, width):
        if name == "pool":
            hh, ww = hh // 2, ww // 2
            continue
        m = n * hh * ww * cout * r * r * (3 if cin == 4 else cin)
        f += m
        if cin != 4:
            dg += m
    up = n * h * w * classes * 4
    return f + dg + f + 3 * up


def cpu_threads():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def run_reference(args, rank, world):
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    run, macs, sample = oracle_sample_step()
    for _ in range(min(args.warmup, 1)):
        run()
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        run()
        times.append(time.perf_counter() - t0)
    t = sum(times) / len(times)
    v = 2 * macs / t / 1e12
    line = {"impl": "reference", "metric": "int8 conv TOPS (fwd+bwd)", "value": v, "unit": "TOPS",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": t * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int8", "data": "synthetic",
            "config": {"workload": WORKLOAD, "global_batch": BATCH * args.gpus,
                       "image": f"3x{IMG}x{IMG}", "classes": CLASSES},
            "cpu_baseline": {"value": v, "unit": "TOPS", "cores": cpu_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------------ GPU leg

def run_ours(args, rank, world, local):
    import numpy as np
    import torch

    from paper_2011_14504_gb300 import iq
    from paper_2011_14504_gb300 import synthetic as S
    from paper_2011_14504_gb300.fcn import FcnVgg16

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    iq.load()
    net = FcnVgg16(BATCH, IMG, IMG, classes=CLASSES, seed=rank, lr_log2=10, device=str(dev))
    g = S.rng(1000 + rank)
    img_np = S.images_u8(g, BATCH, IMG, IMG)
    lab_np = S.labels_voronoi(g, BATCH, IMG, IMG, CLASSES, sites=SITES)
    img = torch.from_numpy(img_np).to(dev)
    lab = torch.from_numpy(lab_np).to(dev)
    stream = torch.cuda.current_stream(dev)

    # per-operation attribution with events on the launching stream
    op_events = {}

    def timed(kind, fn):
        def wrap(*a, **k):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn(*a, **k)
            e1.record(stream)
            op_events.setdefault(kind, []).append((e0, e1, a[0]))
        return wrap

    for _ in range(args.warmup):
        net.train_step(img, lab)
    torch.cuda.synchronize(dev)

    orig = {k: getattr(iq, k) for k in ("iq_conv_fwd", "iq_conv_dgrad", "iq_conv_wgrad")}
    import paper_2011_14504_gb300.fcn as fcn_mod
    for k, f in orig.items():
        setattr(fcn_mod.iq, k, timed(k, f))
    launches0 = iq.launch_count()
    barrier(world)
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for _ in range(args.steps):
            net.train_step(img, lab)
        t_end.record(stream)
        torch.cuda.synchronize(dev)
    barrier(world)
    launches = iq.launch_count() - launches0
    for k, f in orig.items():
        setattr(fcn_mod.iq, k, f)
    ms_total = t_start.elapsed_time(t_end)
    ms_total = max_over_ranks(ms_total, world, dev)
    ms_step = ms_total / args.steps
    macs = net.macs_step
    tops = 2 * macs * world / (ms_step * 1e-3) / 1e12

    # roofline of the dominant conv operation (per-call event durations)
    per = {}
    for kind, evs in op_events.items():
        per[kind] = sum(e0.elapsed_time(e1) for e0, e1, _ in evs)
    dom = max(per, key=per.get)
    conv_macs = {"iq_conv_fwd": sum(L.macs for L in net.convs),
                 "iq_conv_dgrad": sum(L.macs for L in net.convs if L.layer_id > 0),
                 "iq_conv_wgrad": sum(L.macs for L in net.convs)}
    n_calls = len(op_events[dom]) // args.steps
    ms_call = per[dom] / len(op_events[dom])
    flops_call = 2 * conv_macs[dom] / n_calls
    pk, pk_kind = peaks()
    peak_tf = pk.get("bf16_tflops_sustained", pk.get("bf16_tflops"))
    achieved = flops_call / (ms_call * 1e-3) / 1e12
    roofline = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peak_tf,
                "unit": "TFLOP/s", "frac": achieved / peak_tf, "traffic": None,
                "peak_source": f"{pk_kind} fp16/bf16 dense sustained (MEASURED_PEAKS.json)",
                "share_of_step": per[dom] / ms_total,
                "op_ms_per_step": {k: v / args.steps for k, v in per.items()}}

    # end to end: host (pinned) inputs copied in, a result scalar read back, every step
    img_h = torch.from_numpy(img_np).pin_memory()
    lab_h = torch.from_numpy(lab_np).pin_memory()
    res_h = torch.empty(1, dtype=torch.float64).pin_memory()
    img_d = torch.empty_like(img)
    lab_d = torch.empty_like(lab)
    e2e_steps = max(1, min(args.steps, 3))
    barrier(world)
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        img_d.copy_(img_h, non_blocking=True)
        lab_d.copy_(lab_h, non_blocking=True)
        net.train_step(img_d, lab_d)
        res_h.copy_(net.s_Ez, non_blocking=True)     # max |z s_z - onehot| / 127
    e1.record(stream)
    torch.cuda.synchronize(dev)
    ms_e2e = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)
    tops_e2e = 2 * macs * world / (ms_e2e * 1e-3) / 1e12

    if rank == 0:
        cpu = None
        try:
            import oracle
            oracle.build()
            run, omacs, sample = oracle_sample_step()
            t0 = time.perf_counter()
            run()
            t = time.perf_counter() - t0
            cpu = {"value": 2 * omacs / t / 1e12, "unit": "TOPS", "cores": cpu_threads(),
                   "kind": "oracle", "sample": sample, "seconds": t}
        except Exception as ex:   # the GPU number stands on its own
            cpu = {"value": None, "unit": "TOPS", "cores": cpu_threads(), "kind": "oracle",
                   "sample": f"failed: {ex}"}
        line = {"metric": "int8 conv TOPS (fwd+bwd)", "value": tops, "unit": "TOPS",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "int8", "data": "synthetic",
                "images_per_s": BATCH * world / (ms_step * 1e-3),
                "config": {"workload": WORKLOAD, "global_batch": BATCH * world,
                           "image": f"3x{IMG}x{IMG}", "classes": CLASSES,
                           "labels": f"voronoi {SITES} sites", "macs_per_image_step":
                               macs // BATCH, "parallelism": f"replicas x{world}",
                           "l2": "working set >> 129 MB L2, no flush"},
                "e2e": {"value": tops_e2e, "unit": "TOPS",
                        "h2d_bytes_per_step": img_h.numel() + lab_h.numel(),
                        "d2h_bytes_per_step": 8, "images_per_s": BATCH * world /
                        (ms_e2e * 1e-3)},
                "gpu_launches": launches,
                "roofline": roofline,
                "clocks": clk.summary(),
                "cpu_baseline": cpu}
        print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    args = ap.parse_args()
    rank, world, local = dist_setup(args.gpus)
    if args.impl == "reference":
        rc = run_reference(args, rank, world)
    else:
        rc = run_ours(args, rank, world, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return rc


if __name__ == "__main__":
    sys.exit(main())
