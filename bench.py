"""Benchmark of the TBN hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload alexnet|vgg_small|resnet18|lenet|gemv|quantize|backward]
                    [--no-extras] [--no-cpu-baseline] [--eager-steps K]

Default workload: the AlexNet-shaped TBN network at batch 256 (3x227x227
bf16 ~ N(0,1); conv 96x11x11/4, 256x5x5/p2, 384x3x3/p1, 384x3x3/p1,
256x3x3/p1 with 3x3/2 max pools; FC 9216-4096-4096-1000; He-normal weights,
two-bit with per-output-neuron alpha), seed 2.  One step is one pass of the
whole hot path over the batch: re-quantization of every layer's real-valued
weights (Eq. 3 + Eq. 5 + packing, one grouped launch; Algorithm 1 runs the
quantization loop before each forward), the input's NCHW -> NHWC change, the
five two-bit convolutions (Eq. 1) with fused ReLU, the three max pools and
the three fully-connected layers (Section 3).  The metric is TBN TFLOP/s:
the algorithmic 2*N*K*P*Q*C*R*S flops of the convolutions plus 2*B*K_in*K_out
of the FC layers (581.25 GFLOP per step) over the step's device time, every
launch of the step included; images/s is reported beside it, and the
inference form (codes quantized once, no re-quantization) as an extra key.

Timing: the step is captured in a CUDA graph; W warm-up replays (and at
least --min-warmup-s seconds of them, so the clocks settle), then K timed
replays, each bracketed by CUDA events recorded inside the graph, with a
512 MiB write and a 256 MiB read between replays that flush L2 (outside the
timed events).
nvidia-smi samples the SM clock through the timed regions.  The roofline
entry is the tcgen05 implicit-GEMM kernel: its launches of one step (the
five convolutions and the three FC layers) replayed back to back in a graph
of their own after an L2 flush, algorithmic flops over that time.  The e2e
figure replays a graph that adds, each step, the copy of a whole input
batch from pinned host memory and of the logits back to pinned host memory;
the copy of the next batch runs on a second stream once the step's layout
change has consumed the current one, so it overlaps the convolutions.

Extra keys of the default run (each its own small timed region): VGG-small
b128 and ResNet-18 b128 forward TFLOP/s and images/s, the LeNet-like layer's
quantize + conv latency, the quantizer's and the GEMV's HBM GB/s, and the
fused quantize-and-convolve launch against the two-launch path.

Under torchrun (N > 1) every rank runs its own batch on its own GPU (data
parallel replicas, no collective on the data path): value = the work of all
ranks over the slowest rank's time.

--workload vgg_small  VGG-small b128 (re-quantized per forward) as the line
--workload resnet18   ResNet-18 b128 as the line
--workload gemv       batch-1/8 fully-connected layers, K_out = K_in in
                      {4096, 8192, 16384}: HBM GB/s on the 2-bit stream
--workload quantize   tbn_quantize_pack on 8192^2 and 16384^2 fp32 matrices:
                      HBM GB/s at 4.25 bytes per weight
--workload backward   Algorithm 1's TwoBitBackward through the six VGG-small
                      convolutions at batch 128
--impl reference      the CPU oracle (plain C, fp64) on the AlexNet
                      workload: one image of the batch per step through
                      re-quantization + the five convolutions + pools + FC.
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

# used only when MEASURED_PEAKS.json is absent (one earlier GB300 measurement)
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}
FLUSH_BYTES = 512 * 1024 * 1024

WORKLOADS = {
    "alexnet": ("alexnet_b256", "TBN TFLOP/s (AlexNet b256 forward incl. per-step re-quantization)"),
    "vgg_small": ("vgg_small_b128_cifar",
                  "TBN conv TFLOP/s (VGG-small b128 forward incl. per-step re-quantization)"),
    "resnet18": ("resnet18_b128", "TBN conv TFLOP/s (ResNet-18 b128, two-bit convolutions)"),
}

# DRAM bytes (read + write) per implicit-GEMM launch of the AlexNet b256 step,
# mean over its eight launches, from the full-size ncu capture summarised in
# profiles/alexnet_b256_launches.md.  Valid only for the kernel sources it was
# measured on (hash below); otherwise the roofline entry reports null.
CONV_TRAFFIC = {"sources": ["paper_1701_00485_gb300/csrc/tbn_conv_igemm.cuh",
                            "paper_1701_00485_gb300/csrc/tbn_conv_igemm.cu",
                            "paper_1701_00485_gb300/csrc/tbn_device.cuh"],
                "sha256_16": "2edd57ba5c2ffeed", "bytes_per_launch": 48.08e6}


def measured_traffic(rec):
    import hashlib
    if rec["sha256_16"] is None:
        return None
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


L2_NOTE = "512 MiB write + 256 MiB read between timed steps (L2 flushed, no dirty lines left)"


class L2Flush:
    """Evicts the step's data from L2 between timed replays by writing a
    512 MiB buffer (larger than the 129 MB L2), then reading a 256 MiB one:
    the read replaces the written (dirty) lines with clean ones, so their
    write-back to HBM happens here and not inside the next timed step."""

    def __init__(self, dev):
        self.w = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
        self.r = torch.zeros(FLUSH_BYTES // 8, dtype=torch.int32, device=dev)

    def zero_(self):
        self.w.zero_()
        self.r.sum()


def capture(body, stream, dev):
    """A CUDA graph of body() bracketed by two timing events recorded inside it."""
    ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(g, stream=stream):
            ev[0].record()
            body()
            ev[1].record()
    torch.cuda.synchronize(dev)
    return g, ev


def timed_replays(graph, stream, flush, ev, steps):
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


def pick_peak(peaks, clocks):
    """Burst peak when the timed region ran at the maximum SM clock with no
    power cap (a kernel timed that way is not power-limited), else the
    sustained one; returns (peak, kind, other)."""
    burst = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    sust = peaks.get("bf16_tflops_sustained")
    at_max = (clocks.get("sm_mhz") is not None and clocks.get("sm_max_mhz") is not None and
              clocks["sm_mhz"] >= 0.97 * clocks["sm_max_mhz"] and
              "sw_power_cap" not in clocks.get("reasons", []))
    if at_max or sust is None:
        return burst, "burst", (float(sust) if sust is not None else None)
    return float(sust), "sustained", burst


# ------------------------------------------------------------------ networks
def net_spec(name, dev, batch=None):
    """The network of a workload and the closures the benchmark times: the
    whole step, the inference form, the implicit-GEMM launches of one step
    (for the roofline) and every launch of the step on its own."""
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import nets

    def conv_call(h, l, s, pool=0):
        return lambda: tbn.tbn_conv2d_fwd(h, l.codes, l.alpha, s.K, s.R, s.S, (s.stride,) * 2,
                                          (s.pad,) * 2, layout=tbn.TBN_NHWC, relu=s.relu,
                                          out=l.y, pool=pool)

    def is_igemm(N, C, hw, s):
        return tbn.tbn_conv2d_select_algo(torch.bfloat16, tbn.TBN_NHWC, N, C, hw[0], hw[1], s.K,
                                          s.R, s.S, (s.stride,) * 2, (s.pad,) * 2) == \
            tbn.TBN_CONV_IMPLICIT_GEMM

    chain, chain_flops, layers = [], 0, []
    if name in ("alexnet", "vgg_small"):
        net = nets.alexnet(batch, device=dev) if name == "alexnet" else nets.vgg_small(batch, device=dev)
        F = net.features if name == "alexnet" else net
        N = F.N
        if F.s2d:
            s0 = F.layers[0].spec
            layers.append(("space_to_depth", lambda: tbn.tbn_space_to_depth(
                F.x_in, s0.R, s0.S, (s0.stride,) * 2, (s0.pad,) * 2, layout=tbn.TBN_NCHW,
                out=F.x_s2d)))
            h = F.x_s2d
        else:
            layers.append(("nchw_to_nhwc", lambda: tbn.tbn_nchw_to_nhwc(F.x_in, out=F.x_nhwc)))
            h = F.x_nhwc
        for i, l in enumerate(F.layers):
            s = l.spec
            if i == 0 and F.s2d:
                fn = (lambda h=h, l=l, s=s: tbn.tbn_conv2d_fwd(
                    h, l.codes, l.alpha, s.K, s.R, s.S, (s.stride,) * 2, (s.pad,) * 2,
                    layout=tbn.TBN_S2D_NHWC, in_chw=F.in_chw, relu=s.relu, out=l.y))
            else:
                fn = conv_call(h, l, s, 2 if s.pool == (2, 2) else 0)
            layers.append(("conv%d" % (i + 1), fn))
            if (i == 0 and F.s2d) or is_igemm(N, s.C, l.in_hw, s):
                chain.append(fn)
                chain_flops += N * l.flops_per_image
            h = l.y
            if l.pooled is not None:
                k, st = s.pool
                layers.append(("pool%d" % (i + 1),
                               (lambda hh=h, ll=l, k=k, st=st:
                                tbn.tbn_maxpool2d_nhwc(hh, (k, k), (st, st), out=ll.pooled))))
                h = l.pooled
        if name == "alexnet":
            hh = h.reshape(N, -1)
            for j, (W, codes, alpha, relu, y) in enumerate(net.classifier.layers):
                fn = (lambda hh=hh, c=codes, a=alpha, r=relu, y=y:
                      tbn.tbn_linear_fwd_ws(hh, c, a, c.shape[0], net.classifier.workspace,
                                            relu=r, out=y))
                layers.append(("fc%d" % (j + 6), fn))
                chain.append(fn)
                chain_flops += 2 * N * W.shape[0] * W.shape[1]
                hh = y
            flops = net.flops
            cfg = {"workload": "alexnet_b256", "global_batch": N, "image": [3, 227, 227],
                   "layers": "conv 96x11x11/4, 256x5x5/p2, 384x3x3/p1, 384x3x3/p1, "
                             "256x3x3/p1, 3x3/2 max pools; FC 9216-4096-4096-1000",
                   "requantize_per_step": True}
            kernel_desc = "conv_igemm_kernel (tcgen05 implicit GEMM): conv1 (space-to-depth " \
                          "input, filter resident in tensor memory), " \
                          "conv2 (32-channel TMA), conv3-5, fc6-8 (1x1, split K; their " \
                          "ordered split sums included in the chain time)"
        else:
            flops = net.flops
            cfg = {"workload": "vgg_small_b128_cifar", "global_batch": N, "image": [3, 32, 32],
                   "layers": "3x3/p1 128-128-256-256-512-512, 2x2 pool every 2nd",
                   "requantize_per_step": True}
            kernel_desc = "conv_igemm_kernel (tcgen05 implicit GEMM), layers c2-c6"
        step = lambda: net.forward(requantize=True)
        infer = lambda: net.forward(requantize=False)
        quant = net.quantize
        tbn_flops = flops
    elif name == "resnet18":
        net = nets.resnet18(batch, device=dev)
        N = net.N
        layers.append(("stem", net.stem))
        h = net.pool_y
        for a, b, d in net.blocks:
            for c, x_in, res, relu in ((a, h, None, None), (d, h, None, None),
                                       (b, a.y, (d.y if d is not None else h), True)):
                if c is None:
                    continue
                fn = (lambda c=c, x_in=x_in, res=res, relu=relu: c.run(x_in, residual=res, relu=relu))
                layers.append((c.name, fn))
                chain.append(fn)
                chain_flops += N * c.flops_per_image
            h = b.y
        layers.append(("head", lambda hh=h: net.head(hh)))
        step = lambda: net.forward(requantize=True)
        infer = lambda: net.forward(requantize=False)
        quant = net.quantize
        tbn_flops = net.tbn_flops
        flops = tbn_flops
        cfg = {"workload": "resnet18_b128", "global_batch": N, "image": [3, 224, 224],
               "layers": "fp32 7x7/2 stem + 3x3/2 max pool, 8 basic blocks of two-bit 3x3 "
                         "convs (1x1/2 two-bit projections), global average pool, fp32 FC "
                         "512-1000", "requantize_per_step": True}
        kernel_desc = "conv_igemm_kernel (tcgen05 implicit GEMM), all 19 two-bit convolutions"
    else:
        raise ValueError(name)
    return dict(net=net, N=N, step=step, infer=infer, quant=quant, flops=flops,
                tbn_flops=tbn_flops, chain=chain, chain_flops=chain_flops, layers=layers,
                cfg=cfg, kernel_desc=kernel_desc,
                launches=net.launches_per_forward(True))


def run_network(args, rank, world, local_rank, name, full=True, steps=None, warmup=None):
    import paper_1701_00485_gb300 as tbn
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    steps = args.steps if steps is None else steps
    warmup = args.warmup if warmup is None else warmup
    sp = net_spec(name, dev)
    net, N = sp["net"], sp["N"]
    stream = torch.cuda.Stream(device=dev)
    # eager warm-up outside capture: resolves per-device state and kernel attributes
    with torch.cuda.stream(stream):
        sp["step"]()
    torch.cuda.synchronize(dev)
    if tbn.tbn_device_error() != 0:
        raise RuntimeError("device error word set after warm-up")

    def chain_body():
        for fn in sp["chain"]:
            fn()

    graph, ev_step = capture(sp["step"], stream, dev)
    graph_inf, ev_inf = capture(sp["infer"], stream, dev)
    graph_q, ev_q = capture(sp["quant"], stream, dev)
    graph_c, ev_c = capture(chain_body, stream, dev)
    flush = L2Flush(dev)
    sampler = ClockSampler(local_rank)
    sampler.start()
    warm(graph, stream, flush, warmup, args.min_warmup_s if full else 0.2, dev)

    barrier(world)
    torch.cuda.synchronize(dev)
    t0 = time.time()
    step_ms = timed_replays(graph, stream, flush, ev_step, steps)
    torch.cuda.synchronize(dev)
    barrier(world)
    inf_ms = timed_replays(graph_inf, stream, flush, ev_inf, steps)
    chain_ms = timed_replays(graph_c, stream, flush, ev_c, steps)
    quant_ms = timed_replays(graph_q, stream, flush, ev_q, max(3, steps // 2))
    breakdown = {}
    if full:
        reps = max(3, min(steps, 10))
        for label, fn in sp["layers"]:
            g, ev = capture(fn, stream, dev)
            breakdown[label] = round(1e3 * float(np.median(timed_replays(g, stream, flush, ev, reps))), 2)
            del g
    t1 = time.time()
    clocks = sampler.stop(t0, t1)

    total_ms = max_over_ranks(float(np.sum(step_ms)), world, dev)
    ms_per_step = total_ms / steps
    value = world * sp["flops"] * steps / (total_ms * 1e-3) / 1e12
    images_per_s = world * N * steps / (total_ms * 1e-3)
    inf_step = float(np.mean(inf_ms))
    chain_step = float(np.mean(chain_ms))
    peaks, peak_kind = load_peaks()
    peak, which, other = pick_peak(peaks, clocks)
    achieved = sp["chain_flops"] / (chain_step * 1e-3) / 1e12
    roofline = {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak,
                "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
                "peak_kind": "%s bf16 dense, %s" % (peak_kind, which),
                "timing": "the %d implicit-GEMM launches of one step back to back in one graph, "
                          "L2 flushed before each replay: %.2f us per step (%.1f GFLOP)"
                          % (len(sp["chain"]), 1e3 * chain_step, sp["chain_flops"] / 1e9),
                "traffic": measured_traffic(CONV_TRAFFIC) if name == "alexnet" else None,
                "kernel": sp["kernel_desc"]}
    if other is not None:
        roofline["frac_" + ("sustained" if which == "burst" else "burst")] = round(achieved / other, 4)
    res = {
        "metric": WORKLOADS[name][1], "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": world,
        "steps": steps, "warmup": warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) input, He-normal weights)",
        "config": dict(sp["cfg"], global_batch=N * world, parallelism="replicas x%d" % world,
                       l2=L2_NOTE),
        "images_per_s": round(images_per_s, 1),
        "tbn_gflop_per_step": round(sp["tbn_flops"] * world / 1e9, 3),
        "inference_form": {"note": "codes and alpha quantized once (no re-quantization in the step)",
                           "ms_per_step": round(inf_step, 5),
                           "tflops": round(sp["flops"] / (inf_step * 1e-3) / 1e12, 3),
                           "images_per_s": round(N / (inf_step * 1e-3), 1)},
        "requantize_us": round(1e3 * float(np.median(quant_ms)), 2),
        "roofline": roofline,
        "gpu_launches": sp["launches"] * steps,
        "clocks": clocks,
    }
    if name == "resnet18":
        res["tbn_conv_tflops_chain"] = round(achieved, 3)
        res["dense_gflop_per_step"] = round(net.dense_flops / 1e9, 3)
    if full:
        res["breakdown_us"] = breakdown
        res["breakdown_note"] = "each launch alone in its own graph after an L2 flush (no " \
                                "overlap with its neighbours): the parts sum to more than the step"
        # e2e: host input in, logits out, every step.  Each step copies a
        # whole input batch from pinned host memory and reads its logits
        # back.  The next step's batch is copied on a second stream as soon
        # as this step's layout change (the only kernel that reads the input
        # buffer) has been issued, so the copy overlaps the convolutions;
        # both streams are joined before the step ends.
        net_e = sp["net"]
        x_host = net_e.x_in.cpu().pin_memory()
        out = net_e.out
        out_host = torch.empty(out.shape, dtype=out.dtype).pin_memory()
        copy_stream = torch.cuda.Stream(device=dev)

        def e2e_body():
            cur = torch.cuda.current_stream(dev)

            def prefetch(i, layer, when):
                if i == 0 and when == "before":   # the input has been consumed
                    copy_stream.wait_stream(cur)
                    with torch.cuda.stream(copy_stream):
                        net_e.x_in.copy_(x_host, non_blocking=True)

            net_e.forward(requantize=True, conv_hook=prefetch)
            cur.wait_stream(copy_stream)
            out_host.copy_(out, non_blocking=True)

        graph_e, ev_e = capture(e2e_body, stream, dev)
        warm(graph_e, stream, flush, 3, 0.0, dev)
        e2e_ms = timed_replays(graph_e, stream, flush, ev_e, steps)
        e2e_total = max_over_ranks(float(np.sum(e2e_ms)), world, dev)
        res["e2e"] = {"value": round(world * sp["flops"] * steps / (e2e_total * 1e-3) / 1e12, 3),
                      "unit": "TFLOP/s",
                      "h2d_bytes_per_step": int(x_host.numel() * x_host.element_size()),
                      "d2h_bytes_per_step": int(out_host.numel() * out_host.element_size()),
                      "ms_per_step": round(e2e_total / steps, 5),
                      "pipeline": "each step: its logits read back, and the next batch copied "
                                  "from pinned host memory on a second stream once the layout "
                                  "change has consumed the current one (overlapping the "
                                  "convolutions)"}
    res["device_error_word"] = tbn.tbn_device_error()
    del graph, graph_inf, graph_q, graph_c
    return res


# ------------------------------------------------------------------ single layers
def run_lenet(args, local_rank, reps=50):
    """The LeNet-like layer (config 1): quantize + pack [20, 25] fp32 weights,
    then the fp32 direct convolution of 16 x 1 x 28 x 28 fp32 inputs;
    latency per pass (launch-bound: 9.2 MFLOP)."""
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    dev = torch.device("cuda", local_rank)
    x, W = inputs.lenet_inputs(0)
    x, W = x.to(dev), W.reshape(20, -1).contiguous().to(dev)
    codes = torch.empty((20, tbn.packed_words(25)), dtype=torch.int32, device=dev)
    alpha = torch.empty((20,), dtype=torch.float32, device=dev)
    y = torch.empty((16, 20, 24, 24), dtype=torch.float32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def body():
        tbn.tbn_quantize_pack(W, codes, alpha)
        tbn.tbn_conv2d_fwd(x, codes, alpha, 20, 5, 5, layout=tbn.TBN_NCHW, out=y)

    with torch.cuda.stream(stream):
        body()
    torch.cuda.synchronize(dev)
    g, ev = capture(body, stream, dev)
    flush = L2Flush(dev)
    warm(g, stream, flush, 5, 0.0, dev)
    ms = timed_replays(g, stream, flush, ev, reps)
    t = float(np.median(ms))
    return {"workload": "lenet_like_conv_b16", "us_per_pass": round(1e3 * t, 2),
            "tflops": round(2 * 16 * 20 * 24 * 24 * 25 / (t * 1e-3) / 1e12, 4),
            "note": "quantize + pack, then the fp32 direct convolution; two launches, "
                    "launch-latency bound"}


def _rotating_graph(fn_list, stream, dev):
    """One graph that calls each fn once (launches rotate over buffers that
    together exceed L2), bracketed by events."""
    def body():
        for fn in fn_list:
            fn()
    return capture(body, stream, dev)


def run_gemv(args, rank, world, local_rank, sizes=None, batches=None, reps=None):
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    stream = torch.cuda.Stream(device=dev)
    sizes = args.gemv_sizes if sizes is None else sizes
    batches = args.gemv_batches if batches is None else batches
    reps_t = max(3, args.steps // 20) if reps is None else reps
    sweep = []
    sampler = ClockSampler(local_rank)
    sampler.start()
    t0 = time.time()
    for K in sizes:
        W, _ = inputs.gemv_inputs(K, 1)
        codes, alpha = tbn.tbn_quantize_pack(W.to(dev))
        del W
        code_bytes = codes.numel() * 4
        copies = max(2, int(np.ceil(3 * l2 / code_bytes)))
        bufs = [codes] + [codes.clone() for _ in range(copies - 1)]
        # the fp8 tensor-core path reads its own prepared copy of the codes
        f8 = tbn.tbn_linear_f8_prepared_words(K, K) > 0
        pbufs = [tbn.tbn_linear_prepare_f8(c, K) for c in bufs] if f8 else []
        for B in batches:
            gx = torch.Generator(device=dev)
            gx.manual_seed(1000 * K + B)
            x = torch.randn((B, K), generator=gx, device=dev).to(torch.bfloat16)
            y = torch.empty((B, K), dtype=torch.bfloat16, device=dev)
            ws_bytes = tbn.tbn_linear_workspace_bytes(B, K, K, torch.float32)
            ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=dev)
            x32 = x.float()
            reps = max(copies, 64)
            # "mma": bf16 activations (tensor-core GEMV); "table-f32": fp32
            # activations on the batch-1 table-lookup GEMV (tbn_linear_fwd_ws);
            # "tcgen05-f8": batch 1 on the fp8 tensor-core path
            paths = ["mma", "table-f32"] if ws_bytes > 0 else ["mma"]
            f8_ws = tbn.tbn_linear_f8_workspace_bytes(B, K, K) if f8 else 0
            if f8_ws > 0:
                paths.append("tcgen05-f8")
                wsf = torch.empty(f8_ws, dtype=torch.uint8, device=dev)
            for path in paths:
                if path == "tcgen05-f8":
                    fns = [(lambda c=pbufs[r % copies]:
                            tbn.tbn_linear_fwd_f8(x, c, alpha, K, wsf, out=y))
                           for r in range(reps)]
                elif path == "table-f32":
                    fns = [(lambda c=bufs[r % copies]:
                            tbn.tbn_linear_fwd_ws(x32, c, alpha, K, ws, out=y))
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
                for _ in range(reps_t):
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
        del bufs, pbufs
        torch.cuda.empty_cache()
    clocks = sampler.stop(t0, time.time())
    head = ([s for s in sweep if s["K"] == 16384 and s["B"] == 1 and s["path"] == "mma"] or
            sweep)[0]
    return {"metric": "TBN GEMV HBM GB/s (B=1, K_out=K_in=16384, 2-bit weight stream)",
            "value": head["gbs"], "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (He-normal weights, N(0,1) activations)",
            "config": {"workload": "gemv_sweep", "l2": "rotating weight copies > 3x L2"},
            "roofline": {"bound": "hbm", "achieved": head["gbs"], "peak": hbm, "unit": "GB/s",
                         "frac": round(head["gbs"] / hbm, 4), "traffic": None,
                         "kernel": "gemv_tma_kernel (mma.sync)", "peak_kind": peak_kind},
            "sweep": sweep, "clocks": clocks}


def run_quantize(args, rank, world, local_rank, sizes=None, reps=None):
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    stream = torch.cuda.Stream(device=dev)
    flush = L2Flush(dev)
    sizes = args.quant_sizes if sizes is None else sizes
    reps = max(5, args.steps // 10) if reps is None else reps
    sweep = []
    sampler = ClockSampler(local_rank)
    sampler.start()
    t0 = time.time()
    for K in sizes:
        W, _ = inputs.gemv_inputs(K, 1)
        W = W.to(dev)
        codes = torch.empty((K, K // 16), dtype=torch.int32, device=dev)
        alpha = torch.empty((K,), dtype=torch.float32, device=dev)
        g, ev = capture(lambda: tbn.tbn_quantize_pack(W, codes, alpha), stream, dev)
        for _ in range(max(3, args.warmup)):
            g.replay()
        torch.cuda.synchronize(dev)
        ms = timed_replays(g, stream, flush, ev, reps)
        t = float(np.median(ms)) * 1e-3
        byts = K * K * 4.25 + 4 * K
        sweep.append({"K": K, "n": K, "us": round(t * 1e6, 2), "gbs": round(byts / t / 1e9, 1),
                      "frac_hbm": round(byts / t / 1e9 / hbm, 4)})
        del W, codes, alpha, g
        torch.cuda.empty_cache()
    clocks = sampler.stop(t0, time.time())
    head = sweep[-1]
    return {"metric": "TBN quantize+pack HBM GB/s (16384 x 16384 fp32, 4.25 B/weight)",
            "value": head["gbs"], "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (He-normal weights)",
            "config": {"workload": "quantize_16384", "l2": L2_NOTE},
            "roofline": {"bound": "hbm", "achieved": head["gbs"], "peak": hbm, "unit": "GB/s",
                         "frac": head["frac_hbm"], "traffic": None,
                         "kernel": "quantize_pack_kernel", "peak_kind": peak_kind},
            "sweep": sweep, "clocks": clocks}


# ------------------------------------------------- fused quantize + convolve
FUSED_LAYERS = (
    # name, N, C, K, R, pad, H (stride 1, square maps, NHWC bf16)
    ("alexnet_conv3_b256", 256, 256, 384, 3, 1, 13),
    ("vgg_c4_b128", 128, 256, 256, 3, 1, 16),
    ("vgg_c6_b8", 8, 512, 512, 3, 1, 8),
)


def run_fused_quant_conv(args, local_rank, reps=5):
    """Per layer: the fp32 filters quantized and the convolution run (a) as
    two launches (tbn_quantize_pack, tbn_conv2d_fwd) and (b) as the one fused
    launch (tbn_conv2d_fwd_quant), each replayed from a graph after an L2
    flush; both give bitwise the same codes, alpha and output."""
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.Stream(device=dev)
    flush = L2Flush(dev)
    out = []
    for name, N, C, K, R, pad, H in FUSED_LAYERS:
        g = inputs.generator(5)
        x = torch.randn(N, H, H, C, generator=g).to(torch.bfloat16).to(dev)
        W = inputs.normal((K, R * R * C), (2.0 / (C * R * R)) ** 0.5, g).to(dev)
        codes = torch.empty((K, tbn.packed_words(R * R * C)), dtype=torch.int32, device=dev)
        alpha = torch.empty((K,), dtype=torch.float32, device=dev)
        ws = torch.empty(64, dtype=torch.uint8, device=dev)
        y = torch.empty((N, H, H, K), dtype=torch.bfloat16, device=dev)

        def separate():
            tbn.tbn_quantize_pack(W, codes, alpha)
            tbn.tbn_conv2d_fwd(x, codes, alpha, K, R, R, (1, 1), (pad, pad), relu=True,
                               algo=tbn.TBN_CONV_IMPLICIT_GEMM, out=y)

        def fused():
            tbn.tbn_conv2d_fwd_quant(x, W, K, R, R, (1, 1), (pad, pad), relu=True, codes=codes,
                                     alpha=alpha, workspace=ws, out=y)
        row = {"layer": name}
        for key, fn in (("separate_us", separate), ("fused_us", fused)):
            with torch.cuda.stream(stream):
                fn()   # once outside the capture: the library's one-time kernel set-up
            torch.cuda.synchronize(dev)
            gr, ev = capture(fn, stream, dev)
            for _ in range(max(3, args.warmup)):
                gr.replay()
            torch.cuda.synchronize(dev)
            row[key] = round(float(np.median(timed_replays(gr, stream, flush, ev, reps))) * 1e3, 2)
            del gr
        out.append(row)
        del x, W, codes, alpha, ws, y
        torch.cuda.empty_cache()
    return {"layers": out, "note": "graph replay after an L2 flush; separate = quantize "
            "launch + convolution launch, fused = one cooperative launch with a grid barrier"}


# ------------------------------------------------------------------ backward
def run_backward(args, rank, world, local_rank):
    """TwoBitBackward for every VGG-small layer: dx (tensor-core forward
    kernels on the transposed filters) and dW^ (CUDA-core fp32 kernel)."""
    import paper_1701_00485_gb300 as tbn
    from paper_1701_00485_gb300 import inputs
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    stream = torch.cuda.Stream(device=dev)
    flush = L2Flush(dev)
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
                flush.zero_()
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
    bf16_peak, which, _ = pick_peak(peaks, clocks)
    filt_tf = gflop / ms_filt
    return {"metric": "TBN TwoBitBackward TFLOP/s (VGG-small b128, input + filter gradients)",
            "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": 1, "steps": reps,
            "warmup": args.warmup, "ms_per_step": round(ms_all, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (N(0,1) activations and output gradients, He-normal weights)",
            "config": {"workload": "vgg_small_b128_backward", "global_batch": N,
                       "l2": L2_NOTE},
            "gflop_per_step": round(gflop + gflop_data, 3),
            "input_grad_tflops": round(gflop_data / ms_data, 3),
            "filter_grad_tflops": round(filt_tf, 3),
            "per_layer_us": per_layer,
            "roofline": {"bound": "tensor", "achieved": round(filt_tf, 3), "peak": bf16_peak,
                         "unit": "TFLOP/s", "frac": round(filt_tf / bf16_peak, 4), "traffic": None,
                         "kernel": "bwd_filter_tc_kernel (tcgen05 M128 N128 bf16, accumulator "
                                   "in tensor memory, cp.async ring; c1: bwd_filter_kernel on "
                                   "mma.sync), 6 launches + slice reductions",
                         "peak_kind": "%s bf16 dense, %s" % (peak_kind, which),
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




# ------------------------------------------------------------------ CPU oracle
def oracle_alexnet_one_image(orc, x_img_nchw_f32, Ws, Wfc, specs, fcs):
    """Re-quantize every layer and run one image through the AlexNet-shaped
    network on the CPU oracle (Eq. 3, Eq. 5, Eq. 1 + ReLU + max pool, the FC
    layers of Section 3 on the NHWC flattening); returns its TBN flops."""
    h = x_img_nchw_f32[None]
    flops = 0
    for W, s in zip(Ws, specs):
        K = W.shape[0]
        wt, al = orc.quantize(W.reshape(K, -1))
        y, _ = orc.conv2d_nchw(h, wt.reshape(W.shape), al, (s.stride,) * 2, (s.pad,) * 2)
        flops += 2 * K * y.shape[2] * y.shape[3] * s.C * s.R * s.S
        y = orc.epilogue(y, None, relu=s.relu)
        if s.pool is not None:
            y = orc.maxpool2d_nchw(y, (s.pool[0],) * 2, (s.pool[1],) * 2)
        h = y.astype(np.float32)
    v = np.ascontiguousarray(h.transpose(0, 2, 3, 1).reshape(1, -1))
    for W, (kin, kout, relu) in zip(Wfc, fcs):
        wt, al = orc.quantize(W)
        y, _ = orc.linear(v, wt, al)
        flops += 2 * kin * kout
        v = orc.epilogue(y, None, relu=relu).astype(np.float32)
    return flops


def run_cpu_oracle(target_s: float = 10.0, max_images: int | None = None, threads=None):
    """The oracle as it stands on the host cores: whole images of the AlexNet
    b256 batch, each through re-quantization of all eight layers + the
    network; returns TFLOP/s over the sample."""
    import oracle
    from paper_1701_00485_gb300 import inputs
    orc = oracle.default()
    cores = orc.num_threads() if threads is None else threads
    if threads is not None:
        orc.set_num_threads(threads)
    x, Ws, Wfc = inputs.alexnet_inputs(2, batch=8)
    specs, fcs = inputs.ALEXNET["convs"], inputs.ALEXNET["fcs"]
    xf = x.float().numpy()
    Wn = [W.numpy() for W in Ws]
    Wfn = [W.numpy() for W in Wfc]
    t0 = time.time()
    flops, images = 0, 0
    try:
        while True:
            flops += oracle_alexnet_one_image(orc, xf[images % xf.shape[0]], Wn, Wfn, specs, fcs)
            images += 1
            el = time.time() - t0
            if el >= target_s or (max_images and images >= max_images):
                break
    finally:
        if threads is not None:
            orc.set_num_threads(os.cpu_count() or 1)
    el = time.time() - t0
    return {"value": flops / el / 1e12, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
            "images": images, "seconds": round(el, 3), "images_per_s": images / el,
            "sample": "%d image(s) of the AlexNet b256 batch, each through re-quantization of "
                      "all eight layers + five convolutions + ReLU/pool glue + three FC layers "
                      "(fp64 C oracle, %d thread(s))" % (images, cores)}


def cpu_baseline_line():
    """All-core sample (about 10 s) and a single-thread image."""
    allc = run_cpu_oracle(target_s=10.0)
    one = run_cpu_oracle(target_s=0.0, max_images=1, threads=1)
    line = {k: allc[k] for k in ("value", "unit", "cores", "kind", "sample")}
    line["images_per_s"] = round(allc["images_per_s"], 4)
    line["single_thread"] = {"value": one["value"], "unit": "TFLOP/s", "cores": 1,
                             "seconds_per_image": one["seconds"]}
    return line


def reference_arm(args, rank):
    """The reference arm: the CPU oracle on the AlexNet workload, one image of
    the batch per step (plus its re-quantization), on the host cores."""
    if rank != 0:
        return 0
    per_step, cb = [], None
    for _ in range(max(1, args.warmup)):
        run_cpu_oracle(target_s=0.0, max_images=1)
    for _ in range(args.steps):
        cb = run_cpu_oracle(target_s=0.0, max_images=1)
        per_step.append(cb["seconds"])
    total = float(np.sum(per_step))
    img_flops = cb["value"] * 1e12 * cb["seconds"]
    value = img_flops * args.steps / total / 1e12
    line = {"impl": "reference", "metric": WORKLOADS["alexnet"][1], "value": value,
            "unit": "TFLOP/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": total / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded N(0,1) input, He-normal weights)",
            "config": {"workload": "alexnet_b256", "global_batch": 256, "image": [3, 227, 227],
                       "step_sample": "1 image of the 256-image batch per step"},
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cb["cores"],
                             "kind": "oracle",
                             "sample": "1 image per step through re-quantization + five "
                                       "convolutions + glue + three FC layers"},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["alexnet", "vgg_small", "resnet18", "lenet", "gemv",
                                           "quantize", "backward"], default="alexnet")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="only the headline workload (no VGG/ResNet/LeNet/GEMV/quantizer keys)")
    ap.add_argument("--gemv-sizes", type=int, nargs="+", default=[4096, 8192, 16384],
                    help="K_out = K_in of the GEMV workload")
    ap.add_argument("--gemv-batches", type=int, nargs="+", default=[1, 8])
    ap.add_argument("--quant-sizes", type=int, nargs="+", default=[8192, 16384],
                    help="square fp32 matrices of the quantize workload")
    ap.add_argument("--min-warmup-s", type=float, default=1.0,
                    help="keep replaying warm-up steps for at least this long (clock settling)")
    ap.add_argument("--eager-steps", type=int, default=0,
                    help="for profilers: run the network workload's step eagerly this many "
                         "times (no graphs, no timing, no JSON line) and exit")
    args = ap.parse_args()

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        return reference_arm(args, rank)
    if args.eager_steps > 0:
        import paper_1701_00485_gb300 as tbn
        torch.cuda.set_device(local_rank)
        sp = net_spec(args.workload, torch.device("cuda", local_rank))
        for _ in range(args.eager_steps):
            sp["step"]()
        torch.cuda.synchronize()
        print("eager steps %d, device error word %d" % (args.eager_steps, tbn.tbn_device_error()))
        return 0

    if world > 1:
        torch.distributed.init_process_group("nccl")
    # the CPU baseline forks no workers after CUDA init: run it first
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload == "alexnet":
        cpu = cpu_baseline_line()
    elif rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload == "backward":
        cpu = run_cpu_oracle_backward()
    if args.workload in WORKLOADS:
        res = run_network(args, rank, world, local_rank, args.workload)
        if args.workload == "alexnet" and not args.no_extras and world == 1:
            k = min(args.steps, 20)
            extras = {}
            for name in ("vgg_small", "resnet18"):
                r = run_network(args, rank, world, local_rank, name, full=False, steps=k,
                                warmup=min(args.warmup, 5))
                extras[name] = {kk: r[kk] for kk in ("value", "unit", "ms_per_step",
                                                     "images_per_s", "inference_form",
                                                     "requantize_us", "roofline", "clocks")}
                if name == "resnet18":
                    extras[name]["note"] = "value: 434.06 GFLOP of two-bit convolutions over " \
                                           "the whole step (fp32 stem and FC included in the " \
                                           "time); roofline: the 19 two-bit convolutions alone"
                torch.cuda.empty_cache()
            extras["lenet"] = run_lenet(args, local_rank)
            q = run_quantize(args, rank, world, local_rank, reps=5)
            extras["quantize"] = {"sweep": q["sweep"], "clocks": q["clocks"]}
            gm = run_gemv(args, rank, world, local_rank, reps=3)
            extras["gemv"] = {"sweep": gm["sweep"], "clocks": gm["clocks"]}
            extras["fused_quant_conv"] = run_fused_quant_conv(args, local_rank)
            res["extras"] = extras
    else:
        runner = {"lenet": None, "gemv": run_gemv, "quantize": run_quantize,
                  "backward": run_backward}[args.workload]
        if runner is None:
            res = dict(run_lenet(args, local_rank), n_gpus=1)
        else:
            res = runner(args, rank, world, local_rank)
    if rank == 0:
        if cpu is not None:
            res["cpu_baseline"] = cpu
        print(json.dumps(res))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
