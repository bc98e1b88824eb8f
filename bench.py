"""Benchmark: the FCN-VGG16 quantized training step (int8 conv fwd + dgrad + wgrad, the
paper's Sec. 3 dataflow) on synthetic 512x512 segmentation batches.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload fcn_vgg16_train|deeplabv3_r50_train|fcn_vgg16_infer|
                              deeplabv3_r50_infer]

The default workload is the FCN-VGG16 training step (batch 16, 512x512, 150 classes);
the others are the DeepLabv3-ResNet50 training step (batch 16, 513x513, 21 classes, 5%
ignored labels) and the two inference passes (batch 8).

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

SITES = 64


class Workload:
    """One benchmarked configuration: the network, its inputs and what a step counts."""

    def __init__(self, name: str):
        self.name = name
        self.fcn = name.startswith("fcn")
        self.train = name.endswith("train")
        self.batch = 16 if self.train else 8
        self.img = 512 if self.fcn else 513
        self.classes = 150 if self.fcn else 21
        self.labels = f"voronoi {SITES} sites" if self.fcn else "uniform, 5% ignore (255)"

    def config(self, world: int) -> dict:
        return {"workload": self.name + "_step" if self.train else self.name,
                "global_batch": self.batch * world, "image": f"3x{self.img}x{self.img}",
                "classes": self.classes, "labels": self.labels if self.train else None}

    def inputs(self, g, n, h):
        from paper_2011_14504_gb300 import synthetic as S
        img = S.images_u8(g, n, h, h)
        if not self.train:
            return img, None
        if self.fcn:
            return img, S.labels_voronoi(g, n, h, h, self.classes, sites=SITES)
        return img, S.labels_uniform_ignore(g, n, h, h, self.classes)

    def build(self, dev, seed):
        if self.fcn:
            from paper_2011_14504_gb300.fcn import FcnVgg16
            return FcnVgg16(self.batch, self.img, self.img, classes=self.classes, seed=seed,
                            lr_log2=10, device=str(dev), train=self.train)
        from paper_2011_14504_gb300.deeplab import DeepLabV3R50
        return DeepLabV3R50(self.batch, self.img, self.img, classes=self.classes, seed=seed,
                            lr_log2=10, device=str(dev), train=self.train)

    def step(self, net, img, lab):
        if self.train:
            net.train_step(img, lab)
        else:
            net.forward(img)

    def result(self, net):
        """The scalar read back every end-to-end step: the loss-gradient scale (training)
        or the logits scale (inference)."""
        if self.train:
            return net.s_Ez if self.fcn else net.s_E
        return net.s_z

    def macs(self, net) -> int:
        return net.macs_step if self.train else net.macs_forward

    def conv_macs(self, net) -> dict:
        """MACs per step of each convolution entry point (the decoder of FCN excluded)."""
        if self.fcn:
            layers = [(L.macs, L.layer_id == 0) for L in net.convs]
        else:
            layers = [(L.macs, L is net.stem) for L in net.layers.values()]
        f = sum(m for m, _ in layers)
        return {"iq_conv_fwd": f, "iq_conv_dgrad": sum(m for m, first in layers if not first),
                "iq_conv_wgrad": f}


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, \
            "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 50 ms while running."""

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
                 "--format=csv,noheader,nounits", "-lms", "50"],
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

def oracle_sample_step(wl: Workload):
    """One step of the CPU oracle on a bounded sample of the workload (the full-width
    network, one image at 128x128 (FCN) or 129x129 (DeepLab), about 10-30 s of CPU work)."""
    from paper_2011_14504_gb300 import synthetic as S
    g = S.rng(1)
    if wl.fcn:
        from oracle.fcn import OracleFcn
        n, h = 1, 128
        chans = S.fcn_vgg16_channels(wl.classes, 1.0)
        wts, up = S.fcn_vgg16_weights(0, wl.classes, 1.0)
        ora = OracleFcn(chans, wts, up, wl.classes, seed=0)
        macs = fcn_step_macs(n, h, h, wl.classes)
        if not wl.train:
            macs = fcn_forward_macs(n, h, h, wl.classes)
        name = "FCN-VGG16"
    else:
        from oracle.deeplab import OracleDeepLab
        n, h = 1, 129
        sp = S.deeplabv3_r50_spec(wl.classes, 1.0)
        w, gm, bm = S.deeplabv3_r50_init(0, sp)
        ora = OracleDeepLab(sp, w, gm, bm, seed=0)
        macs = deeplab_macs(sp, n, h, wl.train)
        name = "DeepLabv3-ResNet50"
    img, lab = wl.inputs(g, n, h)

    def run():
        tr = ora.forward(img)
        if wl.train:
            ora.backward_update(tr, lab)
    kind = "train step" if wl.train else "inference"
    return run, macs, f"{name} {kind}, N={n}, {h}x{h}, full width, {wl.classes} classes"


def deeplab_macs(sp, n, h, train):
    """Forward (+ data and weight gradient) MACs of the DeepLab convolutions for n images of
    h x h, from the conv geometry alone."""
    def out(sz, cv):
        return (sz + 2 * cv.pad - cv.dil * (cv.r - 1) - 1) // cv.stride + 1
    per = []
    sz = out(h, sp.stem)
    per.append((n * sz * sz * sp.stem.cout * 49 * 3, True))
    sz = (sz + 2 - 3) // 2 + 1
    for b in sp.blocks:
        s1 = sz
        for cv in (b.conv1, b.conv2, b.conv3):
            o = out(s1, cv)
            per.append((n * o * o * cv.cout * cv.r * cv.r * cv.cin, False))
            s1 = o
        if b.down:
            per.append((n * s1 * s1 * b.down.cout * b.down.cin, False))
        sz = s1
    for cv in list(sp.aspp) + [sp.project, sp.head, sp.cls]:
        per.append((n * sz * sz * cv.cout * cv.r * cv.r * cv.cin, False))
    per.append((n * sp.pool_conv.cout * sp.pool_conv.cin, False))
    f = sum(m for m, _ in per)
    if not train:
        return f
    return f + sum(m for m, first in per if not first) + f


def fcn_forward_macs(n, h, w, classes, width=1.0):
    from paper_2011_14504_gb300 import synthetic as S
    hh, ww, f = h, w, 0
    for name, cin, cout, r, pad, relu in S.fcn_vgg16_channels(classes, width):
        if name == "pool":
            hh, ww = hh // 2, ww // 2
            continue
        f += n * hh * ww * cout * r * r * (3 if cin == 4 else cin)
    return f + n * h * w * classes * 4


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
    wl = Workload(args.workload)
    run, macs, sample = oracle_sample_step(wl)
    for _ in range(min(args.warmup, 1)):
        run()
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        run()
        times.append(time.perf_counter() - t0)
    t = sum(times) / len(times)
    v = 2 * macs / t / 1e12
    line = {"impl": "reference", "metric": metric_name(wl), "value": v, "unit": "TOPS",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": t * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int8", "data": "synthetic",
            "config": wl.config(args.gpus),
            "cpu_baseline": {"value": v, "unit": "TOPS", "cores": cpu_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def metric_name(wl: Workload) -> str:
    return "int8 conv TOPS (fwd+bwd)" if wl.train else "int8 conv TOPS (fwd)"


# ------------------------------------------------------------------ GPU leg

def run_ours(args, rank, world, local):
    import numpy as np
    import torch

    from paper_2011_14504_gb300 import iq
    from paper_2011_14504_gb300 import synthetic as S

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    iq.load()
    wl = Workload(args.workload)
    net = wl.build(dev, rank)
    g = S.rng(1000 + rank)
    img_np, lab_np = wl.inputs(g, wl.batch, wl.img)
    img = torch.from_numpy(img_np).to(dev)
    lab = torch.from_numpy(lab_np).to(dev) if lab_np is not None else None
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
        wl.step(net, img, lab)
    torch.cuda.synchronize(dev)

    # The step as a CUDA graph (one captured step, replayed): every kernel of the step is
    # still launched and run, without the per-launch host work.  The stochastic-rounding epoch
    # advances at the end of each replay, so every step draws new random numbers.  A step that
    # cannot be captured runs eagerly.
    graph, graph_launches = None, 0
    try:
        side = torch.cuda.Stream(dev)
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            wl.step(net, img, lab)
        stream.wait_stream(side)
        torch.cuda.synchronize(dev)
        graph = torch.cuda.CUDAGraph()
        l0 = iq.launch_count()
        with torch.cuda.graph(graph):
            wl.step(net, img, lab)
            iq.iq_rq_epoch_advance()
        graph_launches = iq.launch_count() - l0
        graph.replay()
        torch.cuda.synchronize(dev)
        iq.iq_device_status(stream)
    except Exception as ex:     # not capturable here: time the eager step instead
        graph = None
        print(f"# CUDA graph capture unavailable ({type(ex).__name__}: {ex}); eager steps",
              file=sys.stderr)
        torch.cuda.synchronize(dev)

    def run_step():
        if graph is not None:
            graph.replay()
        else:
            wl.step(net, img, lab)

    launches0 = iq.launch_count()
    barrier(world)
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for _ in range(args.steps):
            run_step()
        t_end.record(stream)
        torch.cuda.synchronize(dev)
    barrier(world)
    launches = (graph_launches * args.steps if graph is not None
                else iq.launch_count() - launches0)
    iq.iq_device_status(stream)     # raises if a bounded device wait gave up

    # per-operation attribution (eager steps, CUDA events around each conv call on the stream)
    # and, inside those calls, events around every launch of the tensor-core conv kernels
    orig = {k: getattr(iq, k) for k in ("iq_conv_fwd", "iq_conv_dgrad", "iq_conv_wgrad")}
    for k, f in orig.items():
        setattr(iq, k, timed(k, f))
    iq.iq_kernel_timing_begin()
    for _ in range(args.steps):
        wl.step(net, img, lab)
    torch.cuda.synchronize(dev)
    ktimes = iq.iq_kernel_timing_end()
    for k, f in orig.items():
        setattr(iq, k, f)
    ms_total = t_start.elapsed_time(t_end)
    ms_total = max_over_ranks(ms_total, world, dev)
    ms_step = ms_total / args.steps
    macs = wl.macs(net)
    tops = 2 * macs * world / (ms_step * 1e-3) / 1e12

    # roofline of the dominant kernel: the tensor-core conv kernel with the largest summed
    # event time over the attribution steps; achieved = its algorithmic flops (2 x the MACs
    # of the calls that launched it) / its summed launch time
    per = {}
    for kind, evs in op_events.items():
        per[kind] = sum(e0.elapsed_time(e1) for e0, e1, _ in evs)
    byk = {}
    for r in ktimes:
        t = byk.setdefault(r["kernel"], {"ms": 0.0, "macs": 0.0, "launches": 0})
        t["ms"] += r["ms"]
        t["macs"] += r["macs"]
        t["launches"] += r["launches"]
    pk, pk_kind = peaks()
    peak_tf = pk.get("bf16_tflops_sustained", pk.get("bf16_tflops"))
    dk = max(byk, key=lambda k: byk[k]["ms"])
    kt = byk[dk]
    achieved = 2 * kt["macs"] / (kt["ms"] * 1e-3) / 1e12
    roofline = {"bound": "tensor", "kernel": iq.KERNEL_NAMES.get(dk, str(dk)),
                "achieved": achieved, "peak": peak_tf, "unit": "TFLOP/s",
                "frac": achieved / peak_tf, "traffic": None,
                "peak_source": f"{pk_kind} fp16/bf16 dense sustained (MEASURED_PEAKS.json)",
                "launches_per_step": kt["launches"] / args.steps,
                "kernel_ms_per_step": kt["ms"] / args.steps,
                "share_of_step": kt["ms"] / args.steps / (ms_total / args.steps),
                "kernels_ms_per_step": {iq.KERNEL_NAMES.get(k, str(k)): v["ms"] / args.steps
                                        for k, v in byk.items()},
                "op_ms_per_step": {k: v / args.steps for k, v in per.items()}}

    # end to end: host (pinned) inputs copied in, a result scalar read back, every step
    img_h = torch.from_numpy(img_np).pin_memory()
    lab_h = torch.from_numpy(lab_np).pin_memory() if lab is not None else None
    res_h = torch.empty(1, dtype=torch.float64).pin_memory()
    img_d = torch.empty_like(img)
    lab_d = torch.empty_like(lab) if lab is not None else None
    e2e_steps = max(1, min(args.steps, 3))
    barrier(world)
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        if graph is not None:
            # the captured step reads the static input buffers
            img.copy_(img_h, non_blocking=True)
            if lab is not None:
                lab.copy_(lab_h, non_blocking=True)
            graph.replay()
        else:
            img_d.copy_(img_h, non_blocking=True)
            if lab_d is not None:
                lab_d.copy_(lab_h, non_blocking=True)
            wl.step(net, img_d, lab_d)
        res_h.copy_(wl.result(net), non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    iq.iq_device_status(stream)
    ms_e2e = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)
    tops_e2e = 2 * macs * world / (ms_e2e * 1e-3) / 1e12

    if rank == 0:
        cpu = None
        try:
            import oracle
            oracle.build()
            run, omacs, sample = oracle_sample_step(wl)
            t0 = time.perf_counter()
            run()
            t = time.perf_counter() - t0
            cpu = {"value": 2 * omacs / t / 1e12, "unit": "TOPS", "cores": cpu_threads(),
                   "kind": "oracle", "sample": sample, "seconds": t}
        except Exception as ex:   # the GPU number stands on its own
            cpu = {"value": None, "unit": "TOPS", "cores": cpu_threads(), "kind": "oracle",
                   "sample": f"failed: {ex}"}
        cfg = wl.config(world)
        cfg.update({"macs_per_image_step": macs // wl.batch, "parallelism": f"replicas x{world}",
                    "l2": "working set >> 129 MB L2, no flush",
                    "launch": "cuda graph of one step, replayed" if graph is not None
                    else "eager"})
        line = {"metric": metric_name(wl), "value": tops, "unit": "TOPS",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "int8", "data": "synthetic",
                "images_per_s": wl.batch * world / (ms_step * 1e-3),
                "config": cfg,
                "e2e": {"value": tops_e2e, "unit": "TOPS",
                        "h2d_bytes_per_step": img_h.numel() + (lab_h.numel() if lab_h is not None
                                                               else 0),
                        "d2h_bytes_per_step": 8, "images_per_s": wl.batch * world /
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
    ap.add_argument("--workload", default="fcn_vgg16_train",
                    choices=["fcn_vgg16_train", "deeplabv3_r50_train", "fcn_vgg16_infer",
                             "deeplabv3_r50_infer"])
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
