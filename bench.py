"""Benchmark of the TBN hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Workload (default): the VGG-small TBN conv stack at batch 128 on CIFAR-sized
input (3x32x32 bf16 ~ N(0,1), six 3x3/p1 layers 128-128-256-256-512-512,
ReLU, 2x2 max pool after every second layer, He-normal weights), seed 1.
One step = one pass of the whole hot path over the batch: re-quantize every
layer's real-valued weights (Eq. 3 + Eq. 5 + packing, one grouped launch),
NCHW -> NHWC, six two-bit convolutions (Eq. 1) with fused ReLU, three max
pools.  The metric is TBN-conv TFLOP/s: the algorithmic 2*N*K*P*Q*C*R*S
flops of the six convolutions per step over the step's device time (every
launch of the step included); images/s is reported beside it.

Timing: the step is captured once in a CUDA graph; W warm-up replays, then
K timed replays, each timed with CUDA events recorded inside the graph
(start/end of the step and around every tensor-core convolution), a 512 MiB
L2 flush between replays (outside the timed events).  nvidia-smi samples the
SM clock from the last second of warm-up to the end of the timed region.

The e2e figure replays a second graph that adds, each step, the copy of the
input batch from pinned host memory and the copy of the output feature map
back to pinned host memory.

Under torchrun (N > 1) every rank runs its own batch on its own GPU (data
parallel replicas, no collective on the data path): value = the images of all
ranks over the slowest rank's time.

--impl reference times the CPU oracle (plain C, fp64) on the same workload:
a bounded sample of images through re-quantization + the six convolutions +
glue, reported in the same unit.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

WORKLOAD = "vgg_small_b128_cifar"
METRIC = "TBN conv TFLOP/s (VGG-small b128 forward incl. per-step re-quantization)"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = os.path.join(ROOT, "_build", "clocks.%d.csv" % os.getpid())

    def start(self):
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self, t0: float, t1: float):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 10:
                    continue
                try:
                    ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                    rows.append((ts, float(parts[2]), float(parts[3]), parts[6:10]))
                except Exception:
                    continue
        os.remove(self.path)
        sel = [r for r in rows if t0 - 1.5 <= r[0] <= t1 + 1.0] or rows
        if not sel:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in sel for i, v in enumerate(r[3]) if v == "Active"})
        return {"sm_mhz": float(np.median([r[1] for r in sel])),
                "sm_max_mhz": float(max(r[2] for r in sel)), "reasons": reasons,
                "samples": len(sel)}


# ------------------------------------------------------------------ our arm
def run_ours(args, rank, world, local_rank):
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import nets

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    net = nets.vgg_small(device=dev)
    N = net.N
    flops = net.flops
    tc_layers = [i for i, l in enumerate(net.layers)
                 if tbn.tbn_conv2d_select_algo(torch.bfloat16, tbn.TBN_NHWC, N, l.spec.C,
                                               l.in_hw[0], l.in_hw[1], l.spec.K, l.spec.R,
                                               l.spec.S, (l.spec.stride,) * 2,
                                               (l.spec.pad,) * 2) == tbn.TBN_CONV_IMPLICIT_GEMM]
    tc_flops = N * sum(net.layers[i].flops_per_image for i in tc_layers)

    stream = torch.cuda.Stream(device=dev)
    # eager warm-up outside capture: resolves per-device state and kernel attributes
    with torch.cuda.stream(stream):
        net.forward(requantize=True)
    torch.cuda.synchronize(dev)
    if tbn.tbn_device_error() != 0:
        raise RuntimeError("device error word set after warm-up")

    ev_step = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
    ev_conv = {i: [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
               for i in tc_layers}

    def hook(i, layer, when):
        if i in ev_conv:
            ev_conv[i][0 if when == "before" else 1].record()

    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            ev_step[0].record()
            net.forward(requantize=True, conv_hook=hook)
            ev_step[1].record()
    torch.cuda.synchronize(dev)

    flush = torch.empty(512 * 1024 * 1024, dtype=torch.uint8, device=dev)
    sampler = ClockSampler(local_rank)
    sampler.start()
    # warm-up: W replays, and at least --min-warmup-s of replays so clocks settle
    t_w = time.time()
    w = 0
    while w < args.warmup or time.time() - t_w < args.min_warmup_s:
        with torch.cuda.stream(stream):
            flush.zero_()
            graph.replay()
        w += 1
        if w % 50 == 0:
            torch.cuda.synchronize(dev)
    torch.cuda.synchronize(dev)

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    t0 = time.time()
    step_ms, conv_ms = [], []
    for _ in range(args.steps):
        with torch.cuda.stream(stream):
            flush.zero_()
            graph.replay()
        stream.synchronize()
        step_ms.append(ev_step[0].elapsed_time(ev_step[1]))
        conv_ms.append(sum(ev_conv[i][0].elapsed_time(ev_conv[i][1]) for i in tc_layers))
    torch.cuda.synchronize(dev)
    t1 = time.time()
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop(t0, t1)

    total_ms = float(np.sum(step_ms))
    if world > 1:
        t = torch.tensor([total_ms], dtype=torch.float64, device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_per_step = total_ms / args.steps
    value = world * flops * args.steps / (total_ms * 1e-3) / 1e12
    images_per_s = world * N * args.steps / (total_ms * 1e-3)

    # e2e: pinned host input -> device, step, output -> pinned host
    x_host = net.x_in.cpu().pin_memory()
    out_host = torch.empty(net.out.shape, dtype=net.out.dtype).pin_memory()
    g2 = torch.cuda.CUDAGraph()
    ev_e = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
    with torch.cuda.stream(stream):
        with torch.cuda.graph(g2, stream=stream):
            ev_e[0].record()
            net.x_in.copy_(x_host, non_blocking=True)
            net.forward(requantize=True)
            out_host.copy_(net.out, non_blocking=True)
            ev_e[1].record()
    for _ in range(3):
        with torch.cuda.stream(stream):
            g2.replay()
    torch.cuda.synchronize(dev)
    e2e_ms = []
    for _ in range(args.steps):
        with torch.cuda.stream(stream):
            flush.zero_()
            g2.replay()
        stream.synchronize()
        e2e_ms.append(ev_e[0].elapsed_time(ev_e[1]))
    e2e_total = float(np.sum(e2e_ms))
    if world > 1:
        t = torch.tensor([e2e_total], dtype=torch.float64, device=dev)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        e2e_total = float(t.item())
    e2e_value = world * flops * args.steps / (e2e_total * 1e-3) / 1e12

    err = tbn.tbn_device_error()
    peaks, peak_kind = load_peaks()
    tc_ms = float(np.mean(conv_ms)) / max(1, len(tc_layers))  # mean per launch
    achieved = (tc_flops / max(1, len(tc_layers))) / (tc_ms * 1e-3) / 1e12
    peak = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    roofline = {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak,
                "unit": "TFLOP/s", "frac": round(achieved / peak, 4), "traffic": None,
                "kernel": "conv_igemm_kernel (tcgen05 implicit GEMM), layers %s" %
                          ",".join("c%d" % (i + 1) for i in tc_layers),
                "peak_kind": "%s bf16 dense, sustained" % peak_kind}

    result = {
        "metric": METRIC, "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) input, He-normal weights)",
        "config": {"workload": WORKLOAD, "global_batch": N * world, "image": [3, 32, 32],
                   "layers": "3x3/p1 128-128-256-256-512-512, 2x2 pool every 2nd",
                   "requantize_per_step": True, "parallelism": "replicas x%d" % world,
                   "l2": "512 MiB flush between timed steps"},
        "images_per_s": round(images_per_s, 1),
        "tbn_conv_gflop_per_step": round(flops * world / 1e9, 3),
        "e2e": {"value": round(e2e_value, 3), "unit": "TFLOP/s",
                "h2d_bytes_per_step": int(x_host.numel() * x_host.element_size()),
                "d2h_bytes_per_step": int(out_host.numel() * out_host.element_size()),
                "ms_per_step": round(e2e_total / args.steps, 5)},
        "gpu_launches": net.launches_per_forward(True) * args.steps,
        "roofline": roofline,
        "clocks": clocks,
        "device_error_word": err,
    }
    return result


# ------------------------------------------------------------------ CPU oracle
def oracle_forward_one_image(orc, x_img_nchw_f32, Ws, specs):
    """Re-quantize every layer and run one image through the stack on the CPU
    oracle (Eq. 3, Eq. 5, Eq. 1 + ReLU + max pool)."""
    h = x_img_nchw_f32[None]
    flops = 0
    for W, s in zip(Ws, specs):
        K = W.shape[0]
        wt, al = orc.quantize(W.reshape(K, -1))
        y, _ = orc.conv2d_nchw(h, wt.reshape(W.shape), al, (s.stride, s.stride),
                               (s.pad, s.pad))
        flops += 2 * K * y.shape[2] * y.shape[3] * s.C * s.R * s.S
        y = orc.epilogue(y, None, relu=s.relu)
        if s.pool is not None:
            y = orc.maxpool2d_nchw(y, (s.pool[0],) * 2, (s.pool[1],) * 2)
        h = y.astype(np.float32)
    return flops


def run_cpu_oracle(target_s: float = 10.0, max_s: float = 30.0, max_images: int | None = None):
    import oracle
    from paper_1701_00485_gb300 import inputs
    orc = oracle.default()
    x, Ws = inputs.vgg_small_inputs(1)
    specs = inputs.VGG_SMALL["convs"]
    xf = x.float().numpy()
    Wn = [W.numpy() for W in Ws]
    t0 = time.time()
    flops = 0
    images = 0
    while True:
        flops += oracle_forward_one_image(orc, xf[images % x.shape[0]], Wn, specs)
        images += 1
        el = time.time() - t0
        if el >= target_s or el >= max_s or (max_images and images >= max_images):
            break
    el = time.time() - t0
    return {"value": flops / el / 1e12, "unit": "TFLOP/s", "cores": orc.num_threads(),
            "kind": "oracle", "images": images, "seconds": round(el, 3),
            "images_per_s": images / el,
            "sample": "%d image(s) of the VGG-small b128 batch, each through re-quantization "
                      "of all six layers + six convolutions + ReLU/pool glue (fp64 C oracle)"
                      % images}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--min-warmup-s", type=float, default=1.0,
                    help="keep replaying warm-up steps for at least this long (clock settling)")
    args = ap.parse_args()

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        # the reference arm is the CPU oracle; rank 0 alone runs it
        if rank != 0:
            return 0
        per_step = []
        cb = None
        for _ in range(max(1, args.warmup)):
            run_cpu_oracle(target_s=0.0, max_images=1)
        for _ in range(args.steps):
            cb = run_cpu_oracle(target_s=0.0, max_images=1)
            per_step.append(cb["seconds"])
        total = float(np.sum(per_step))
        img_flops = cb["value"] * 1e12 * cb["seconds"]
        value = img_flops * args.steps / total / 1e12
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": total / args.steps * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic (seeded N(0,1) input, He-normal weights)",
                "config": {"workload": WORKLOAD, "global_batch": 128, "image": [3, 32, 32],
                           "step_sample": "1 image of the 128-image batch per step"},
                "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cb["cores"],
                                 "kind": "oracle",
                                 "sample": "1 image per step through re-quantization + six "
                                           "convolutions + glue"},
                "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0

    if world > 1:
        torch.distributed.init_process_group("nccl")
    # the CPU baseline forks no workers after CUDA init: run it first
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = run_cpu_oracle()
    res = run_ours(args, rank, world, local_rank)
    if rank == 0:
        if cpu is not None:
            res["cpu_baseline"] = {k: cpu[k] for k in ("value", "unit", "cores", "kind", "sample")}
            res["cpu_baseline"]["images_per_s"] = round(cpu["images_per_s"], 4)
        print(json.dumps(res))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
