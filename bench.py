"""Benchmark of the TBN hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload vgg_small|gemv|quantize]

Default workload: the VGG-small TBN conv stack at batch 128 on CIFAR-sized
input (3x32x32 bf16 ~ N(0,1), six 3x3/p1 layers 128-128-256-256-512-512,
ReLU, 2x2 max pool after every second layer, He-normal weights), seed 1.
One step = one pass of the whole hot path over the batch: re-quantize every
layer's real-valued weights (Eq. 3 + Eq. 5 + packing, one grouped launch),
NCHW -> NHWC, six two-bit convolutions (Eq. 1) with fused ReLU and, after
every second layer, the fused 2x2 max pool.  The metric is TBN-conv TFLOP/s:
the algorithmic 2*N*K*P*Q*C*R*S flops of the six convolutions per step over
the step's device time (every launch of the step included); images/s is
reported beside it.

Timing: the step is captured in a CUDA graph; W warm-up replays (and at
least --min-warmup-s seconds of them, so the clocks settle), then K timed
replays, each bracketed by CUDA events recorded inside the graph, with a
512 MiB write between replays that flushes L2 (outside the timed events).
nvidia-smi samples the SM clock through the timed regions.  A second timed
region replays an instrumented copy of the graph with events around every
tensor-core convolution: the roofline entry (the tcgen05 conv kernel) is
its flops over those durations.  The e2e figure replays a third graph that
adds, each step, the copy of the input batch from pinned host memory and the
copy of the output feature map back to pinned host memory.

Under torchrun (N > 1) every rank runs its own batch on its own GPU (data
parallel replicas, no collective on the data path): value = the work of all
ranks over the slowest rank's time.

--workload gemv       batch-1/8 fully-connected layers, K_out = K_in in
                      {4096, 8192, 16384}: HBM GB/s on the 2-bit stream
--workload quantize   tbn_quantize_pack on 8192^2 and 16384^2 fp32 matrices:
                      HBM GB/s at 4.25 bytes per weight
--workload backward   Algorithm 1's TwoBitBackward through the six VGG-small
                      convolutions at batch 128: the filter gradients of all
                      six layers and the input gradients of c2..c6 (the
                      image itself needs none), 309.2 GFLOP per step
--impl reference      the CPU oracle (plain C, fp64) on the VGG-small
                      workload: one image of the batch per step through
                      re-quantization + the six convolutions + glue.
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
FLUSH_BYTES = 512 * 1024 * 1024

# DRAM bytes (read + write) per convolution launch, mean over the five
# implicit-GEMM launches of one step (c2..c6), from the ncu capture summarised in profiles/vgg_small_b128_launches.md.
# Valid only for the kernel sources it was measured on (hash below); otherwise the
# roofline entry reports null.
CONV_TRAFFIC = {"sources": ["paper_1701_00485_gb300/csrc/tbn_conv_igemm.cu",
                            "paper_1701_00485_gb300/csrc/tbn_device.cuh"],
                "sha256_16": "07de82155ed5eaf3", "bytes_per_launch": 14.54e6}


def measured_traffic(rec):
    import hashlib
    h = hashlib.sha256()
    for f in rec["sources"]:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return rec["bytes_per_launch"] if h.hexdigest()[:16] == rec["sha256_16"] else None


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


class L2Flush:
    """Evicts the step's data from L2 between timed replays: writes a 512 MiB
    buffer (larger than the 129 MB L2) and, in "write+read" mode, then reads
    another 512 MiB buffer, so the write's dirty lines are written back
    before the timed region instead of during it (L2 ends up holding clean,
    unrelated lines)."""

    def __init__(self, dev, mode):
        self.mode = mode
        self.w = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
        self.r = torch.ones(FLUSH_BYTES // 4, dtype=torch.int32, device=dev) if mode == "write+read" else None
        self.acc = torch.empty((), dtype=torch.int32, device=dev)

    def zero_(self):
        self.w.zero_()
        if self.r is not None:
            torch.sum(self.r, dim=0, dtype=torch.int32, out=self.acc)


def timed_replays(graph, stream, flush, ev, steps, dev):
    """Replay `graph` `steps` times, flushing L2 before each replay; returns
    the per-replay device times (ms) between the graph's own events ev."""
    out = []
    for _ in range(steps):
        with torch.cuda.stream(stream):
            flush.zero_()
            graph.replay()
        stream.synchronize()
        out.append(ev[0].elapsed_time(ev[1]))
    return out


def warm(graph, stream, flush, steps, min_s, dev):
    t = time.time()
    w = 0
    while w < steps or time.time() - t < min_s:
        with torch.cuda.stream(stream):
            flush.zero_()
            graph.replay()
        w += 1
        if w % 50 == 0:
            torch.cuda.synchronize(dev)
    torch.cuda.synchronize(dev)


def max_over_ranks(x: float, world: int, dev) -> float:
    if world == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        torch.distributed.barrier()


# ------------------------------------------------------------------ VGG-small
def run_vgg(args, rank, world, local_rank):
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

    def capture(body):
        ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            with torch.cuda.graph(g, stream=stream):
                ev[0].record()
                body()
                ev[1].record()
        torch.cuda.synchronize(dev)
        return g, ev

    # plain step: the timed graph
    graph, ev_step = capture(lambda: net.forward(requantize=True))
    # instrumented step: events around every tensor-core convolution
    ev_conv = {i: [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
               for i in range(len(net.layers))}

    ev_quant = torch.cuda.Event(enable_timing=True, external=True)

    def hook(i, layer, when):
        if i < 0:
            ev_quant.record()
        elif i in ev_conv:
            ev_conv[i][0 if when == "before" else 1].record()

    graph_i, ev_i = capture(lambda: net.forward(requantize=True, conv_hook=hook))

    # roofline graph: the tensor-core convolutions alone, back to back as in
    # the step (each layer reads the previous layer's output), bracketed by
    # one pair of events so the launches overlap as they do in the step
    def tc_chain():
        for i in tc_layers:
            l = net.layers[i]
            s = l.spec
            h = net.layers[i - 1].pooled if net.layers[i - 1].pooled is not None else \
                net.layers[i - 1].y
            tbn.tbn_conv2d_fwd(h, l.codes, l.alpha, s.K, s.R, s.S, (s.stride, s.stride),
                               (s.pad, s.pad), layout=tbn.TBN_NHWC, relu=s.relu, out=l.y,
                               pool=2 if s.pool == (2, 2) else 0)

    assert tc_layers and tc_layers[0] > 0 and \
        tc_layers == list(range(tc_layers[0], tc_layers[-1] + 1)) and \
        all(net.layers[i].pooled is None for i in tc_layers), "chain of fused layers"
    graph_c, ev_c = capture(tc_chain)
    # e2e step: host input in, output feature map out
    x_host = net.x_in.cpu().pin_memory()
    out_host = torch.empty(net.out.shape, dtype=net.out.dtype).pin_memory()

    def e2e_body():
        net.x_in.copy_(x_host, non_blocking=True)
        net.forward(requantize=True)
        out_host.copy_(net.out, non_blocking=True)

    graph_e, ev_e = capture(e2e_body)

    flush = L2Flush(dev, args.l2_flush)
    sampler = ClockSampler(local_rank)
    sampler.start()
    warm(graph, stream, flush, args.warmup, args.min_warmup_s, dev)

    barrier(world)
    torch.cuda.synchronize(dev)
    t0 = time.time()
    step_ms = timed_replays(graph, stream, flush, ev_step, args.steps, dev)
    torch.cuda.synchronize(dev)
    barrier(world)
    # roofline region: the tensor-core chain alone, then the instrumented
    # graph (per-layer breakdown; its events between layers stop the overlap)
    chain_ms = timed_replays(graph_c, stream, flush, ev_c, args.steps, dev)
    conv_ms = []
    layer_ms = np.zeros(len(net.layers))
    quant_ms = 0.0
    prefix_ms = 0.0
    for _ in range(args.steps):
        with torch.cuda.stream(stream):
            flush.zero_()
            graph_i.replay()
        stream.synchronize()
        conv_ms.append(sum(ev_conv[i][0].elapsed_time(ev_conv[i][1]) for i in tc_layers))
        layer_ms += [ev_conv[i][0].elapsed_time(ev_conv[i][1]) for i in range(len(net.layers))]
        quant_ms += ev_i[0].elapsed_time(ev_quant)
        prefix_ms += ev_quant.elapsed_time(ev_conv[0][0])
    t1 = time.time()
    clocks = sampler.stop(t0, t1)

    total_ms = max_over_ranks(float(np.sum(step_ms)), world, dev)
    ms_per_step = total_ms / args.steps
    value = world * flops * args.steps / (total_ms * 1e-3) / 1e12
    images_per_s = world * N * args.steps / (total_ms * 1e-3)

    warm(graph_e, stream, flush, 3, 0.0, dev)
    e2e_ms = timed_replays(graph_e, stream, flush, ev_e, args.steps, dev)
    e2e_total = max_over_ranks(float(np.sum(e2e_ms)), world, dev)
    e2e_value = world * flops * args.steps / (e2e_total * 1e-3) / 1e12

    err = tbn.tbn_device_error()
    peaks, peak_kind = load_peaks()
    tc_launch_ms = float(np.mean(chain_ms)) / len(tc_layers)   # mean per launch in the chain
    achieved = (tc_flops / len(tc_layers)) / (tc_launch_ms * 1e-3) / 1e12
    achieved_isolated = tc_flops / (float(np.mean(conv_ms)) * 1e-3) / 1e12
    peak = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    burst = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    roofline = {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak,
                "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
                # the step runs at full SM clock (see "clocks"), so the burst
                # peak is the stricter denominator: reported beside it
                "peak_burst": burst, "frac_burst": round(achieved / burst, 4),
                "timing": "the %d launches back to back in one graph, L2 flushed before each "
                          "replay, %.2f us per launch; with events between the layers (no launch "
                          "overlap) %.1f TFLOP/s" % (len(tc_layers), 1e3 * tc_launch_ms,
                                                    achieved_isolated),
                "traffic": measured_traffic(CONV_TRAFFIC),
                "kernel": "conv_igemm_kernel (tcgen05 implicit GEMM), %d launches per step "
                          "(layers %s)" % (len(tc_layers),
                                           ",".join("c%d" % (i + 1) for i in tc_layers)),
                "peak_kind": "%s bf16 dense, sustained" % peak_kind}
    return {
        "metric": METRIC, "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) input, He-normal weights)",
        "config": {"workload": WORKLOAD, "global_batch": N * world, "image": [3, 32, 32],
                   "layers": "3x3/p1 128-128-256-256-512-512, 2x2 pool every 2nd",
                   "requantize_per_step": True, "parallelism": "replicas x%d" % world,
                   "l2": "512 MiB %s between timed steps" % args.l2_flush},
        "images_per_s": round(images_per_s, 1),
        "breakdown_note": "per layer from events between the layers, which stop the launch "
                          "overlap of the plain step: the parts sum to more than ms_per_step",
        "breakdown_us": dict([("quantize", round(1e3 * quant_ms / args.steps, 2)),
                              ("nchw_to_nhwc", round(1e3 * prefix_ms / args.steps, 2))] +
                             [("c%d" % (i + 1), round(1e3 * layer_ms[i] / args.steps, 2))
                              for i in range(len(net.layers))]),
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


# ------------------------------------------------------------------ HBM-bound paths
def _rotating_graph(fn_list, stream, dev):
    """One graph that calls each fn once (launches rotate over buffers that
    together exceed L2), bracketed by events."""
    ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(g, stream=stream):
            ev[0].record()
            for fn in fn_list:
                fn()
            ev[1].record()
    torch.cuda.synchronize(dev)
    return g, ev


def run_gemv(args, rank, world, local_rank):
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    stream = torch.cuda.Stream(device=dev)
    sweep = []
    sampler = ClockSampler(local_rank)
    sampler.start()
    t0 = time.time()
    for K in args.gemv_sizes:
        W, _ = inputs.gemv_inputs(K, 1)
        codes, alpha = tbn.tbn_quantize_pack(W.to(dev))
        del W
        code_bytes = codes.numel() * 4
        copies = max(2, int(np.ceil(3 * l2 / code_bytes)))
        bufs = [codes] + [codes.clone() for _ in range(copies - 1)]
        for B in args.gemv_batches:
            gx = torch.Generator(device=dev)
            gx.manual_seed(1000 * K + B)
            x = torch.randn((B, K), generator=gx, device=dev).to(torch.bfloat16)
            y = torch.empty((B, K), dtype=torch.bfloat16, device=dev)
            ws_bytes = tbn.tbn_linear_workspace_bytes(B, K, K, torch.float32)
            ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=dev)
            x32 = x.float()
            reps = max(copies, 64)
            # "mma": tbn_linear_fwd with bf16 activations (tensor-core GEMV);
            # "table-f32": tbn_linear_fwd_ws with fp32 activations (the
            # batch-1 table-lookup GEMV, the path for fp32 inputs);
            # "conv-f32": tbn_linear_fwd with fp32 activations and no scratch
            # (the 1x1-convolution path those inputs take otherwise)
            paths = ["mma", "table-f32", "conv-f32"] if ws_bytes > 0 else ["mma"]
            for path in paths:
                if path == "table-f32":
                    fns = [(lambda c=bufs[r % copies]:
                            tbn.tbn_linear_fwd_ws(x32, c, alpha, K, ws, out=y))
                           for r in range(reps)]
                elif path == "conv-f32":
                    fns = [(lambda c=bufs[r % copies]: tbn.tbn_linear_fwd(x32, c, alpha, K, out=y))
                           for r in range(reps)]
                else:
                    fns = [(lambda c=bufs[r % copies]: tbn.tbn_linear_fwd(x, c, alpha, K, out=y))
                           for r in range(reps)]
                with torch.cuda.stream(stream):
                    fns[0]()
                torch.cuda.synchronize(dev)
                g, ev = _rotating_graph(fns, stream, dev)
                for _ in range(max(3, args.warmup)):
                    g.replay()
                torch.cuda.synchronize(dev)
                ms = []
                for _ in range(max(3, args.steps // 20)):
                    with torch.cuda.stream(stream):
                        g.replay()
                    stream.synchronize()
                    ms.append(ev[0].elapsed_time(ev[1]) / reps)
                t = float(np.median(ms)) * 1e-3
                byts = code_bytes + 4 * K + (4 if path.endswith("f32") else 2) * B * K + 2 * B * K
                sweep.append({"K": K, "B": B, "path": path, "us_per_call": round(t * 1e6, 3),
                              "gbs": round(byts / t / 1e9, 1),
                              "frac_hbm": round(byts / t / 1e9 / hbm, 4),
                              "tflops": round(2 * B * K * K / t / 1e12, 3)})
                del g
        del bufs
        torch.cuda.empty_cache()
    clocks = sampler.stop(t0, time.time())
    head = ([s for s in sweep if s["K"] == 16384 and s["B"] == 1 and s["path"] == "mma"] or
            sweep)[0]
    head_kernel = "gemv_tma_kernel (mma.sync)"
    return {"metric": "TBN GEMV HBM GB/s (B=1, K_out=K_in=16384, 2-bit weight stream)",
            "value": head["gbs"], "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (He-normal weights, N(0,1) activations)",
            "config": {"workload": "gemv_sweep", "l2": "rotating weight copies > 3x L2"},
            "roofline": {"bound": "hbm", "achieved": head["gbs"], "peak": hbm, "unit": "GB/s",
                         "frac": round(head["gbs"] / hbm, 4), "traffic": None,
                         "kernel": head_kernel, "peak_kind": peak_kind},
            "sweep": sweep, "clocks": clocks}


def run_quantize(args, rank, world, local_rank):
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    stream = torch.cuda.Stream(device=dev)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    sweep = []
    sampler = ClockSampler(local_rank)
    sampler.start()
    t0 = time.time()
    for K in args.quant_sizes:
        W, _ = inputs.gemv_inputs(K, 1)
        W = W.to(dev)
        codes = torch.empty((K, K // 16), dtype=torch.int32, device=dev)
        alpha = torch.empty((K,), dtype=torch.float32, device=dev)
        g, ev = _rotating_graph([lambda: tbn.tbn_quantize_pack(W, codes, alpha)], stream, dev)
        for _ in range(max(3, args.warmup)):
            g.replay()
        torch.cuda.synchronize(dev)
        ms = timed_replays(g, stream, flush, ev, max(5, args.steps // 10), dev)
        t = float(np.median(ms)) * 1e-3
        byts = K * K * 4.25 + 4 * K
        sweep.append({"K": K, "n": K, "us": round(t * 1e6, 2), "gbs": round(byts / t / 1e9, 1),
                      "frac_hbm": round(byts / t / 1e9 / hbm, 4)})
        del W, codes, alpha
        torch.cuda.empty_cache()
    clocks = sampler.stop(t0, time.time())
    head = sweep[-1]
    return {"metric": "TBN quantize+pack HBM GB/s (16384 x 16384 fp32, 4.25 B/weight)",
            "value": head["gbs"], "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (He-normal weights)",
            "config": {"workload": "quantize_16384", "l2": "512 MiB flush between timed steps"},
            "roofline": {"bound": "hbm", "achieved": head["gbs"], "peak": hbm, "unit": "GB/s",
                         "frac": head["frac_hbm"], "traffic": None,
                         "kernel": "quantize_pack_kernel", "peak_kind": peak_kind},
            "sweep": sweep, "clocks": clocks}


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


def run_backward(args, rank, world, local_rank):
    """TwoBitBackward for every VGG-small layer: dx (tensor-core forward
    kernels on the transposed filters) and dW^ (CUDA-core fp32 kernel)."""
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    stream = torch.cuda.Stream(device=dev)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    N = 128
    layers = []
    hw = 32
    for i, s in enumerate(inputs.VGG_SMALL["convs"]):
        st, pd = (s.stride, s.stride), (s.pad, s.pad)
        P, Q = tbn.conv_out_hw(hw, hw, s.R, s.S, st, pd)
        x = torch.randn((N, hw, hw, s.C), generator=g, device=dev).to(torch.bfloat16)
        dy = torch.randn((N, P, Q, s.K), generator=g, device=dev).to(torch.bfloat16)
        W = inputs.he_normal(s.K, s.C, s.R, s.S, inputs.generator(100 + i))
        codes, alpha = tbn.tbn_quantize_pack(
            W.permute(0, 2, 3, 1).reshape(s.K, -1).contiguous().to(dev))
        shape = (N, s.C, hw, hw, s.K, s.R, s.S, st[0], st[1], pd[0], pd[1])
        wsd = torch.empty(max(256, tbn.lib().tbn_conv2d_bwd_data_workspace_bytes(*shape)),
                          dtype=torch.uint8, device=dev)
        wsf = torch.empty(max(256, tbn.lib().tbn_conv2d_bwd_filter_workspace_bytes(*shape)),
                          dtype=torch.uint8, device=dev)
        flops = 2 * N * s.K * P * Q * s.C * s.R * s.S
        layers.append(dict(s=s, hw=hw, st=st, pd=pd, x=x, dy=dy, codes=codes, alpha=alpha,
                           wsd=wsd, wsf=wsf, flops=flops))
        if s.pool is not None:
            hw = (P - s.pool[0]) // s.pool[1] + 1
        else:
            hw = P

    def data_fn(L):
        s = L["s"]
        return lambda: tbn.tbn_conv2d_bwd_data(L["dy"], L["codes"], L["alpha"], s.C,
                                               (L["hw"], L["hw"]), s.R, s.S, L["st"], L["pd"],
                                               workspace=L["wsd"])

    def filt_fn(L):
        s = L["s"]
        return lambda: tbn.tbn_conv2d_bwd_filter(L["x"], L["dy"], s.R, s.S, L["st"], L["pd"],
                                                 workspace=L["wsf"])

    def time_graph(fns, reps):
        with torch.cuda.stream(stream):
            for f in fns:
                f()
        torch.cuda.synchronize(dev)
        gr, ev = _rotating_graph(fns, stream, dev)
        for _ in range(max(3, args.warmup)):
            gr.replay()
        ms = []
        for _ in range(reps):
            with torch.cuda.stream(stream):
                flush.fill_(1)
                gr.replay()
            stream.synchronize()
            ms.append(ev[0].elapsed_time(ev[1]))
        return float(np.median(ms))

    sampler = ClockSampler(local_rank)
    sampler.start()
    t0 = time.time()
    reps = max(5, args.steps // 10)
    # the first layer's input gradient (w.r.t. the image) is not part of the pass
    step_fns = [filt_fn(layers[0])] + [f(L) for L in layers[1:] for f in (data_fn, filt_fn)]
    ms_all = time_graph(step_fns, reps)
    ms_data = time_graph([data_fn(L) for L in layers[1:]], reps)
    ms_filt = time_graph([filt_fn(L) for L in layers], reps)
    per_layer = []
    for i, L in enumerate(layers):
        per_layer.append({"layer": "c%d" % (i + 1),
                          "data_us": round(1e3 * time_graph([data_fn(L)], reps), 2),
                          "filter_us": round(1e3 * time_graph([filt_fn(L)], reps), 2)})
    clocks = sampler.stop(t0, time.time())
    gflop = sum(L["flops"] for L in layers) / 1e9              # one gradient of every layer
    gflop_data = sum(L["flops"] for L in layers[1:]) / 1e9
    value = (gflop + gflop_data) / ms_all
    bf16_peak = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops"]))
    filt_tf = gflop / ms_filt
    return {"metric": "TBN TwoBitBackward TFLOP/s (VGG-small b128, input + filter gradients)",
            "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": 1, "steps": reps,
            "warmup": args.warmup, "ms_per_step": round(ms_all, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (N(0,1) activations and output gradients, He-normal weights)",
            "config": {"workload": "vgg_small_b128_backward", "global_batch": N,
                       "l2": "512 MiB write between timed steps"},
            "gflop_per_step": round(gflop + gflop_data, 3),
            "input_grad_tflops": round(gflop_data / ms_data, 3),
            "filter_grad_tflops": round(filt_tf, 3),
            "per_layer_us": per_layer,
            "roofline": {"bound": "tensor", "achieved": round(filt_tf, 3), "peak": bf16_peak,
                         "unit": "TFLOP/s", "frac": round(filt_tf / bf16_peak, 4), "traffic": None,
                         "kernel": "bwd_filter_tc_kernel (tcgen05 M128 N128 bf16, accumulator "
                                   "in tensor memory, cp.async ring; c1: bwd_filter_kernel on "
                                   "mma.sync), 6 launches + slice reductions",
                         "peak_kind": "%s bf16 dense, sustained" % peak_kind,
                         "input_grad_vs_bf16_peak": round(gflop_data / ms_data / bf16_peak, 4)},
            "clocks": clocks}


def run_cpu_oracle_backward(target_s: float = 10.0, max_s: float = 30.0):
    """The oracle's TwoBitBackward (both gradients) through the six VGG-small
    layers, one image of the batch at a time."""
    import oracle
    from paper_1701_00485_gb300 import inputs
    orc = oracle.default()
    rng = np.random.default_rng(5)
    specs = inputs.VGG_SMALL["convs"]
    shapes, hw = [], 32
    for i, s in enumerate(specs):
        P, Q = oracle.out_hw(hw, hw, s.R, s.S, (s.stride,) * 2, (s.pad,) * 2)
        wt = rng.choice(np.array([-2, -1, 1, 2], dtype=np.int8), size=(s.K, s.C, s.R, s.S))
        shapes.append((s, hw, P, Q, wt, rng.random(s.K) + 0.5))
        hw = (P - s.pool[0]) // s.pool[1] + 1 if s.pool is not None else P
    t0 = time.time()
    flops, images = 0, 0
    while True:
        for s, h, P, Q, wt, al in shapes:
            x = rng.standard_normal((1, s.C, h, h)).astype(np.float32)
            dy = rng.standard_normal((1, s.K, P, Q)).astype(np.float32)
            orc.conv2d_bwd_data(dy, wt, al, (h, h), (s.stride,) * 2, (s.pad,) * 2)
            orc.conv2d_bwd_filter(x, dy, (s.R, s.S), (s.stride,) * 2, (s.pad,) * 2)
            flops += 2 * 2 * s.K * P * Q * s.C * s.R * s.S
        images += 1
        el = time.time() - t0
        if el >= target_s or el >= max_s:
            break
    return {"value": flops / el / 1e12, "unit": "TFLOP/s", "cores": orc.num_threads(),
            "kind": "oracle",
            "sample": "%d image(s): input and filter gradients of the six VGG-small layers "
                      "(fp64 C oracle)" % images}


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
    ap.add_argument("--workload", choices=["vgg_small", "gemv", "quantize", "backward"],
                    default="vgg_small")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--gemv-sizes", type=int, nargs="+", default=[4096, 8192, 16384],
                    help="K_out = K_in of the GEMV workload")
    ap.add_argument("--gemv-batches", type=int, nargs="+", default=[1, 8])
    ap.add_argument("--quant-sizes", type=int, nargs="+", default=[8192, 16384],
                    help="square fp32 matrices of the quantize workload")
    ap.add_argument("--l2-flush", choices=["write", "write+read"], default="write",
                    help="L2 eviction between timed steps (write+read also drains the dirty lines)")
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
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload == "vgg_small":
        cpu = run_cpu_oracle()
    elif rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload == "backward":
        cpu = run_cpu_oracle_backward()
    runner = {"vgg_small": run_vgg, "gemv": run_gemv, "quantize": run_quantize,
              "backward": run_backward}[args.workload]
    res = runner(args, rank, world, local_rank)
    if rank == 0:
        if cpu is not None:
            res["cpu_baseline"] = {k: cpu[k] for k in ("value", "unit", "cores", "kind", "sample")}
            if "images_per_s" in cpu:
                res["cpu_baseline"]["images_per_s"] = round(cpu["images_per_s"], 4)
        print(json.dumps(res))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
