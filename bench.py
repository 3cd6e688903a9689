#!/usr/bin/env python
"""Benchmark: ResNet-50 v1.5 pure-FP16 training step, batch 256 per GPU, on GB300.

One step = forward, backward and the FP16 SGD update of the whole network on
one synthetic ImageNet-shaped batch (224x224x3 images ~ N(0,1) per channel,
labels uniform over 1000 classes), all of it in libpf16's kernels, replayed
from one CUDA graph.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl pf16|reference]

`--impl reference` times the CPU oracle (the plain binary64 reference
implementation) on the host cores on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "ResNet-50 pure-FP16 train images/s at batch 256 on 1 GB300; conv TFLOP/s vs FP16 peak"
UNIT = "images/s"
BATCH = 256
WORKLOAD = "ResNet-50 v1.5 pure-FP16 training step (fwd + bwd + FP16 SGD momentum), batch 256, 224x224x3"


def peaks():
    p = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "src": "fallback"}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            m = json.load(f)
        p.update({k: float(m[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained") if k in m})
        p["src"] = "measured"
    except (OSError, ValueError, KeyError):
        pass
    return p


def preload(stream, ms):
    """Keep `stream` busy for about `ms` milliseconds (a one-thread spin
    kernel), so that the host enqueues the calls timed after it before the GPU
    reaches their first event: the events then bracket device time only, not
    the host's argument marshalling and tensor-map encoding of an idle stream."""
    import torch

    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(ms * 2.2e6))  # SM clock cycles (at most ~2.1 GHz)


class ClockSampler:
    """nvidia-smi clock / throttle samples every 200 ms while running."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            try:
                pw.append(float(f[3]))
            except ValueError:
                pass
            for nm, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)), "reasons": sorted(reasons),
                "samples": len(sm), **({"power_w": float(np.median(pw)), "power_w_max": float(max(pw))} if pw else {})}


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def max_over_ranks(v, dist, device):
    """The largest of every rank's v: a replica job ends with its slowest rank
    (dist None: one process)."""
    if dist is None:
        return float(v)
    import torch

    t = torch.tensor([float(v)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world, per_rank_batch, steps, ms):
    """Images per second of the whole job: every rank's images over the slowest
    rank's time (weak scaling: each rank trains its own batch)."""
    return world * per_rank_batch * steps / (ms / 1e3)


# --------------------------------------------------------------------------- CPU oracle
def oracle_step_time(batch=1, image=224, reps=1):
    """Time the oracle's ResNet-50 training step (binary64 C loops, OpenMP) on
    `batch` images; returns (seconds per step, threads)."""
    import oracle
    from oracle import resnet50 as oresnet
    from paper_1911_07384_gb300 import synthetic as syn

    oracle.build()
    net = oresnet.OracleResNet50(batch, image, 1000, seed_cfg=4)
    imgs = syn.images_f16(syn.seed_for(4, "x"), batch, image, image, 3)
    labs = syn.labels(syn.seed_for(4, "labels"), batch)
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        net.step(imgs, labs)
        times.append(time.perf_counter() - t0)
    return float(np.median(times)), oracle.num_threads()


def run_reference(args, rank, world):
    if rank != 0:
        return 0
    sample_batch = 1
    # warm-up: one step on a small image (builds the library, pages code in)
    oracle_step_time(1, 64, 1)
    t_all = []
    for _ in range(args.steps):
        t, cores = oracle_step_time(sample_batch, 224, 1)
        t_all.append(t)
    total = float(np.sum(t_all))
    value = args.steps * sample_batch / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "global_batch": BATCH * args.gpus, "sample_per_step": sample_batch},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{sample_batch} image(s) of 224x224 per step: full fwd+bwd+SGD of "
                                   "ResNet-50 in binary64 over binary16 tensors"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------- GPU
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="pf16", choices=["pf16", "reference"])
    ap.add_argument("--batch", type=int, default=BATCH)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--conv", default=None,
                    help="time one conv pass instead of the step: N,H,W,C,K,R,S,stride,pad")
    ap.add_argument("--pass", dest="conv_pass", default="fwd", choices=["fwd", "dgrad", "wgrad"])
    ap.add_argument("--stats", action="store_true",
                    help="with --conv --pass fwd: the forward that also reduces the BatchNorm statistics of its "
                         "output (pf16_conv_fwd_bnstats, as the training step calls it)")
    ap.add_argument("--bn", default=None,
                    help="time one BatchNorm pass instead of the step: N,H,W,C (ReLU + residual, s=0.25)")
    ap.add_argument("--bn-pass", default="fwd", choices=["fwd", "bwd"])
    ap.add_argument("--nvtx", action="store_true",
                    help="name every library call of the step with an NVTX range (pf16:<kind>:<shape>) for "
                         "profilers; host-side only, the replayed step graph is unchanged")
    ap.add_argument("--bn-in-operand", action="store_true",
                    help="apply each block's second BatchNorm in its last conv's operand path (off by default)")
    ap.add_argument("--bn-swap", action="store_true",
                    help="the BN-swap variant (Sec. 4.1) in every block's last BatchNorm (off in the headline run)")
    ap.add_argument("--layers", action="store_true",
                    help="per-layer CUDA-event times of one eager step (median of 3), one JSON line each")
    ap.add_argument("--ingest-traffic", default=None, metavar="CSV",
                    help="store k_gemm DRAM bytes per launch from an ncu CSV of one step, then exit")
    ap.add_argument("--sweep", default=None, choices=["cfg2", "cfg3"],
                    help="per-layer conv lines: cfg2 = every distinct ResNet-50 conv at N=64, "
                         "cfg3 = the N=256 pure-GEMM 1x1 layers")
    ap.add_argument("--tc-rate", action="store_true",
                    help="the library's MMA-only probe: kind::f16 tcgen05 TFLOP/s for N = 64..256, f16 and f32 "
                         "accumulators, one or two accumulator chains; one JSON line each")
    args = ap.parse_args()
    rank, world, local = dist_env()
    if args.ingest_traffic:
        return ingest_traffic(args.ingest_traffic)
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.conv:
        print(json.dumps(time_conv(tuple(int(v) for v in args.conv.split(",")), args.conv_pass, stats=args.stats,
                                   steps=args.steps, warmup=args.warmup)), flush=True)
        return 0
    if args.sweep:
        return run_sweep(args)
    if args.layers:
        return run_layers(args)
    if args.tc_rate:
        return run_tc_rate()
    if args.bn:
        print(json.dumps(time_bn(tuple(int(v) for v in args.bn.split(",")), args.bn_pass, args.steps,
                                 args.warmup)), flush=True)
        return 0
    if args.warmup < 3:
        args.warmup = 3

    import torch

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if dist is not None:
            dist.barrier()

    from paper_1911_07384_gb300 import pf16
    from paper_1911_07384_gb300 import synthetic as syn
    from paper_1911_07384_gb300.resnet50 import ResNet50

    N = args.batch
    net = ResNet50(batch=N, seed_cfg=4, bn_swap=args.bn_swap, wgrad_branch=True, bn_in_operand=args.bn_in_operand)
    if args.nvtx:
        from paper_1911_07384_gb300.resnet50 import nvtx_hook

        net.hook = nvtx_hook
    imgs = syn.images_f16(syn.seed_for(4, "x", rank), N)
    labs = syn.labels(syn.seed_for(4, "labels", rank), N)
    net.set_batch(imgs, labs)

    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        net.step()  # eager warm-up: first-call setup happens outside the capture
    torch.cuda.synchronize()
    rc = pf16.sync_status(stream)
    if rc != 0:
        raise RuntimeError(f"device status {rc} after warm-up step")
    graph = torch.cuda.CUDAGraph()
    n0 = pf16.kernel_launches()
    with torch.cuda.graph(graph, stream=stream):
        net.step()
    launches = pf16.kernel_launches() - n0  # libpf16 kernels recorded into the step graph
    if launches != count_launches(net):
        raise RuntimeError(f"step graph holds {launches} libpf16 kernels, the call plan "
                           f"predicts {count_launches(net)}")

    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()

    # ---------------- device-timed region: K graph replays, inputs resident in HBM
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            ev0.record(stream)
            for _ in range(args.steps):
                graph.replay()
            ev1.record(stream)
        torch.cuda.synchronize()
        barrier()
    ms = ev0.elapsed_time(ev1)
    rc = pf16.sync_status(stream)
    if rc != 0:
        raise RuntimeError(f"device status {rc} after timed steps")
    ms_max = max_over_ranks(ms, dist, "cuda")
    loss = float(np.uint16(net.loss.cpu().numpy().view(np.uint16)[0]).view(np.float16))
    value = job_throughput(world, N, args.steps, ms_max)

    # ---------------- end to end through host buffers (pinned), copies in the timed region.
    # Two input buffers, as a prefetching loader keeps them: step i reads buffer i % 2,
    # whose host-to-device copy ran on a copy stream while step i - 1 computed; a copy
    # into a buffer waits for the step that last read it.  Every step's copies and its
    # loss read-back lie between the two events.
    x_bufs, l_bufs = [net.x, torch.empty_like(net.x)], [net.labels, torch.empty_like(net.labels)]
    net.x, net.labels = x_bufs[1], l_bufs[1]
    graph_b = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph_b, stream=stream):
        net.step()
    net.x, net.labels = x_bufs[0], l_bufs[0]
    graphs = [graph, graph_b]
    h_img = torch.from_numpy(imgs.reshape(-1).view(np.int16)).pin_memory()
    h_lab = torch.from_numpy(labs.astype(np.int32)).pin_memory()
    h_loss = torch.empty(1, dtype=torch.int16).pin_memory()
    copy_stream = torch.cuda.Stream()
    done = [torch.cuda.Event(), torch.cuda.Event()]
    ready = [torch.cuda.Event(), torch.cuda.Event()]

    def load(b, after=None):
        with torch.cuda.stream(copy_stream):
            if after is not None:
                copy_stream.wait_event(after)
            x_bufs[b].copy_(h_img, non_blocking=True)
            l_bufs[b].copy_(h_lab, non_blocking=True)
            ready[b].record(copy_stream)

    for b in (0, 1):  # warm both graphs on their own buffers
        load(b)
        stream.wait_event(ready[b])
        graphs[b].replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        load(0, after=e0)
        for i in range(args.steps):
            b = i % 2
            if i + 1 < args.steps:
                load(1 - b, after=done[1 - b] if i >= 1 else e0)
            stream.wait_event(ready[b])
            graphs[b].replay()
            done[b].record(stream)
            h_loss.copy_(net.loss, non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dist, "cuda")
    e2e = {"value": job_throughput(world, N, args.steps, e2e_ms), "unit": UNIT,
           "h2d_bytes_per_step": int(h_img.numel() * 2 + h_lab.numel() * 4), "d2h_bytes_per_step": 2}

    # ---------------- dominant kernel (the tcgen05 conv GEMM): per-call CUDA events
    conv = conv_roofline(net, stream, reps=3)
    pk = peaks()
    peak = pk["bf16_tflops_sustained"]  # FP16 and BF16 share the dense tensor rate
    kr = kernel_roofline(pk)
    mma = pf16.tc_rate(256, reps=20000)  # the FP16 kind::f16 MMA rate of this GPU (the library's probe)
    # the aggregate over every conv call of the step; its per-launch DRAM traffic
    # is not measured (a whole-step capture is not made); the single dominant
    # launch class with its captured traffic is roofline_kernel
    roof = {"bound": "tensor", "achieved": conv["tflops"], "peak": peak, "unit": "TFLOP/s",
            "frac": conv["tflops"] / peak, "traffic": None,
            "algorithmic_bytes_per_launch": conv["bytes_per_launch"],
            "peak_f16_mma_probe": mma, "frac_of_f16_mma_probe": conv["tflops"] / mma,
            "kernel": "k_gemm (all conv passes of the step, split-K reduce included)",
            "peak_src": f"{pk['src']} bf16 dense sustained; f16 MMA probe measured in this run"}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": WORKLOAD, "global_batch": N * world, "per_gpu_batch": N,
                   "image": "224x224x3 NHWC", "parallelism": f"replicas{world}" if world > 1 else "single",
                   "l2": "working set (~25 GB of activations per step) far larger than L2; no flush needed",
                   **({"bn_swap": True} if args.bn_swap else {}),
                   **({"bn_in_operand": True} if args.bn_in_operand else {})},
        "loss": loss,
        "clocks": clocks.summary(),
        "e2e": e2e,
        "gpu_launches": launches * args.steps,
        "roofline": roof,
        "roofline_kernel": kr,
        "conv": {"tflops": conv["tflops"], "ms_per_step": conv["ms"], "gflop_per_step": conv["gflop"],
                 "frac_of_dense_peak": conv["tflops"] / pk["bf16_tflops"], "by_pass": conv["by_pass"]},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t, cores = oracle_step_time(1, 224, 1)
        line["cpu_baseline"] = {"value": 1.0 / t, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": "1 image of 224x224: full fwd+bwd+SGD of ResNet-50 in binary64 "
                                          "over binary16 tensors (batch statistics over that image)"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def run_tc_rate():
    """pf16_tc_rate over tile widths, accumulator types and chain counts, against
    the measured bf16 cuBLAS peaks the rooflines use."""
    import torch

    from paper_1911_07384_gb300 import pf16

    torch.cuda.init()
    pk = peaks()
    for n in (64, 128, 192, 256):
        for f32 in (False, True):
            for chains in (1, 2):
                tf = pf16.tc_rate(n, f32_accum=f32, chains=chains, reps=20000)
                print(json.dumps({"probe": "tcgen05.mma kind::f16 M=128", "n": n, "accumulator": "f32" if f32 else "f16",
                                  "chains": chains, "tflops": tf,
                                  "of_bf16_burst": tf / pk["bf16_tflops"], "peak_src": pk["src"]}),
                      flush=True)
    if pf16.sync_status() != 0:
        raise RuntimeError("device status after the rate probe")
    return 0


def run_layers(args):
    """Every library call of one training step timed with CUDA events on the
    launching stream (eager, median of 3 steps; the stream is pre-loaded so that
    each pair of events brackets device time only), aggregated per (call, shape).
    Convs report TFLOP/s; BatchNorm reports GB/s of its minimum bytes (forward
    x, y, residual, ReLU mask; backward x, dy, dx, residual gradient, mask)."""
    import collections

    import torch

    from paper_1911_07384_gb300 import pf16
    from paper_1911_07384_gb300 import synthetic as syn
    from paper_1911_07384_gb300.resnet50 import ResNet50

    net = ResNet50(batch=args.batch, seed_cfg=4, bn_in_operand=args.bn_in_operand)
    net.set_batch(syn.images_f16(syn.seed_for(4, "x", 0), args.batch),
                  syn.labels(syn.seed_for(4, "labels", 0), args.batch))
    stream = torch.cuda.Stream()
    recs = []

    def hook(kind, layer, fn, *a, **kw):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn(*a, **kw)
        e1.record(stream)
        recs.append((kind, layer, e0, e1))

    with torch.cuda.stream(stream):
        net.step()
    torch.cuda.synchronize()
    runs = []
    for _ in range(3):
        recs.clear()
        net.hook = hook
        preload(stream, 300)
        h0 = time.perf_counter()
        with torch.cuda.stream(stream):
            net.step()
        host_ms = 1e3 * (time.perf_counter() - h0)
        net.hook = None
        torch.cuda.synchronize()
        if host_ms > 250:
            raise RuntimeError(f"the step's host enqueue ({host_ms:.0f} ms) outlasted the stream pre-load")
        runs.append([(k, l, e0.elapsed_time(e1)) for k, l, e0, e1 in recs])
    if pf16.sync_status(stream) != 0:
        raise RuntimeError("device status error")
    agg = collections.OrderedDict()
    for i, (kind, layer, _) in enumerate(runs[0]):
        t = float(np.median([r[i][2] for r in runs]))
        if kind.startswith("conv"):
            d = layer.desc
            key = (kind, (d.n, d.h, d.w, d.c, d.k, d.r, d.s, d.stride, d.pad))
            work, unit = layer.flops / 1e12, "TFLOP/s"
        elif kind.startswith("bn"):
            d = layer.desc
            key = (kind, (d.n, d.h, d.w, d.c, int(d.flags)))
            relu, res = d.flags & pf16.PF16_BN_RELU, d.flags & pf16.PF16_BN_RESIDUAL
            e = layer.elems
            if kind == "bn_pool_fwd":  # x read; pooled output, positions (a byte each) and ReLU bits written
                work = (2.0 * e + 0.5 * e + 0.25 * e + e / 8) / 1e9
            else:
                units = (2 + (1 if res else 0)) if kind == "bn_fwd" else (3 + (1 if res else 0))
                work = (2.0 * layer.elems * units + (layer.elems / 8 if relu else 0)) / 1e9
            unit = "GB/s"
        else:
            key, work, unit = (kind, ()), 0.0, ""
        a = agg.setdefault(key, [0, 0.0, 0.0, unit])
        a[0] += 1
        a[1] += t
        a[2] += work
    total = sum(a[1] for a in agg.values())
    for (kind, shape), (n, t, work, unit) in sorted(agg.items(), key=lambda kv: -kv[1][1]):
        line = {"call": kind, "shape": list(shape), "n": n, "ms": t, "share": t / total}
        if unit:
            line["rate"] = work / (t / 1e3)
            line["unit"] = unit
        print(json.dumps(line), flush=True)
    print(json.dumps({"total_ms": total, "note": "sum of per-call event times of an eager step"}))
    return 0


CFG3 = [(256, 56, 56, 256, 64, 1, 1, 1, 0), (256, 28, 28, 512, 128, 1, 1, 1, 0),
        (256, 14, 14, 1024, 256, 1, 1, 1, 0), (256, 7, 7, 512, 2048, 1, 1, 1, 0)]


_POOLS = {}


def pooled_f16(tensor, shape, std=1.0):
    """Seeded N(0, std^2) binary16 timing inputs of `shape`: the prefix of one
    pool per tensor kind, drawn once (and again only when a larger shape asks),
    so that a sweep over many layers does not redraw every tensor."""
    from paper_1911_07384_gb300 import synthetic as syn

    n = int(np.prod(shape))
    p = _POOLS.get((tensor, std))
    if p is None or p.size < n:
        p = syn.normal_f16(syn.seed_for(2, tensor), (n,), std)
        _POOLS[(tensor, std)] = p
    return p[:n].reshape(shape)


def run_sweep(args):
    from paper_1911_07384_gb300.resnet50 import conv_shapes

    if args.sweep == "cfg3":
        shapes = [(f"cfg3_{i}", s) for i, s in enumerate(CFG3)]
    else:
        seen, shapes = set(), []
        for name, s in conv_shapes(64):
            if s not in seen:
                seen.add(s)
                shapes.append((name, s))
    big = max(s[0] * s[1] * s[2] * max(s[3], s[4]) for _, s in shapes)
    pooled_f16("x", (big,))
    pooled_f16("dy", (big,), 0.01)
    for name, s in shapes:
        for ps in ("fwd", "dgrad", "wgrad"):
            if ps == "dgrad" and s[3] == 3:
                continue
            r = time_conv(s, ps, args.steps, args.warmup)
            r["layer"] = name
            print(json.dumps(r), flush=True)
    return 0


def time_conv(shape, conv_pass, steps, warmup, stats=False):
    """One convolution pass on synthetic N(0,1) inputs, He weights, dy ~ N(0, 0.01^2):
    `steps` launches timed with CUDA events on the launching stream; when the
    operands fit in L2 a 256 MiB buffer is rewritten between launches.  stats:
    the forward also reduces the BatchNorm statistics of its output, as the
    training step's forwards do."""
    import torch

    from paper_1911_07384_gb300 import pf16
    from paper_1911_07384_gb300 import synthetic as syn

    N, H, W, C, K, R, S, st, pd = shape
    d = pf16.conv_desc(*shape)
    P, Q = d.out_hw()
    dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).cuda()
    x = dev(pooled_f16("x", (N, H, W, C)))
    w = dev(syn.he_normal_f16(syn.seed_for(2, "w"), K, R, S, C))
    dy = dev(pooled_f16("dy", (N, P, Q, K), 0.01))
    y = torch.empty(N * P * Q * K, dtype=torch.int16, device="cuda")
    dx = torch.empty(N * H * W * C, dtype=torch.int16, device="cuda")
    dw = torch.empty(K * R * S * C, dtype=torch.int16, device="cuda")
    p = {"fwd": pf16.PF16_PASS_FWD, "dgrad": pf16.PF16_PASS_DGRAD, "wgrad": pf16.PF16_PASS_WGRAD}[conv_pass]
    wsb = pf16.conv_workspace_size(d, p)
    ws = torch.empty(max(wsb, 1), dtype=torch.uint8, device="cuda")
    flush = None
    io_bytes = 2 * (x.numel() + w.numel() + (y.numel() if conv_pass != "dgrad" else dy.numel()))
    if io_bytes < 2 * 135 * 2 ** 20:
        flush = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")
    st = torch.empty(pf16.conv_bnstats_size(d), dtype=torch.uint8, device="cuda") if stats else None
    fn = {"fwd": (lambda: pf16.conv_fwd_bnstats(d, x, w, y, st, ws)) if stats else (lambda: pf16.conv_fwd(d, x, w, y, ws)),
          "dgrad": lambda: pf16.conv_dgrad(d, dy, w, dx),
          "wgrad": lambda: pf16.conv_wgrad(d, x, dy, dw, ws)}[conv_pass]
    for _ in range(max(warmup, 3)):
        fn()
    torch.cuda.synchronize()
    times = []
    s = torch.cuda.current_stream()
    for _ in range(steps):
        if flush is not None:
            flush.fill_(1)
        preload(s, 2)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(s)
        fn()
        e1.record(s)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    assert pf16.sync_status() == 0
    ms = float(np.median(times))
    flops = 2.0 * N * P * Q * K * C * R * S
    byts = 2.0 * {"fwd": N * H * W * C + K * R * S * C + N * P * Q * K,
                  "dgrad": N * P * Q * K + K * R * S * C + N * H * W * C,
                  "wgrad": N * H * W * C + N * P * Q * K + K * R * S * C}[conv_pass]
    pk = peaks()
    tf = flops / ms / 1e9
    gbs = byts / ms / 1e6
    attainable = min(pk["bf16_tflops"], byts and flops / byts * pk["hbm_gbs"] / 1e3)
    del x, w, dy, y, dx, dw, ws, flush
    return {"metric": "conv pass TFLOP/s", "conv": list(shape), "pass": conv_pass, "bn_stats": bool(stats), "ms": ms,
            "ms_best": float(np.min(times)), "tflops": tf, "gbs": gbs,
            "frac_of_dense_peak": tf / pk["bf16_tflops"],
            "frac_of_attainable": tf / attainable, "arith_intensity": flops / byts,
            "workspace_bytes": wsb, "l2_flush": io_bytes < 2 * 135 * 2 ** 20}


def time_bn(shape, bn_pass, steps, warmup):
    """One BatchNorm pass (x0.25, residual, ReLU) timed with CUDA events.  Bytes
    are the algorithmic minimum of the pass: forward reads x and the residual
    and writes y and the ReLU bit mask; backward reads x, dy and the mask and
    writes dx and the residual gradient."""
    import torch

    from paper_1911_07384_gb300 import pf16
    from paper_1911_07384_gb300 import synthetic as syn

    N, H, W, C = shape
    R = N * H * W
    dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).cuda()
    e = lambda n: torch.empty(n, dtype=torch.int16, device="cuda")
    x, res, dy = dev(syn.normal_f16(11, (R * C,))), dev(syn.normal_f16(12, (R * C,))), dev(
        syn.normal_f16(13, (R * C,), 0.01))
    one = np.float16(1.0).view(np.uint16)
    g, b = dev(np.full(C, one, np.uint16)), dev(np.zeros(C, np.uint16))
    y, mean, inv, dx, dg, db, dr = e(R * C), e(C), e(C), e(R * C), e(C), e(C), e(R * C)
    mask = torch.empty(R * C // 8, dtype=torch.uint8, device="cuda")
    d = pf16.bn_desc(N, H, W, C, 0x00A8, 0x3400, pf16.PF16_BN_RELU | pf16.PF16_BN_RESIDUAL)
    ws = torch.empty(pf16.bn_workspace_size(d), dtype=torch.uint8, device="cuda")
    fwd = lambda: pf16.bn_fwd_bwd(d, 0, ws, x=x, gamma=g, beta=b, residual=res, y=y, mean=mean, invstd=inv,
                                  relu_mask=mask)
    bwd = lambda: pf16.bn_fwd_bwd(d, 1, ws, x=x, gamma=g, mean=mean, invstd=inv, dy=dy, relu_mask=mask,
                                  dx=dx, dgamma=dg, dbeta=db, dresidual=dr)
    fwd()
    fn = fwd if bn_pass == "fwd" else bwd
    for _ in range(max(warmup, 3)):
        fn()
    torch.cuda.synchronize()
    times = []
    s = torch.cuda.current_stream()
    for _ in range(steps):
        preload(s, 2)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(s)
        fn()
        e1.record(s)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    assert pf16.sync_status() == 0
    ms = float(np.median(times))
    byts = 2.0 * R * C * (3 if bn_pass == "fwd" else 4) + R * C / 8  # + the ReLU bit mask
    pk = peaks()
    return {"metric": "BatchNorm pass GB/s", "bn": list(shape), "pass": bn_pass, "ms": ms,
            "ms_best": float(np.min(times)), "gbs": byts / ms / 1e6,
            "frac_of_hbm": byts / ms / 1e6 / pk["hbm_gbs"], "algorithmic_bytes": byts}


# The dominant launch class of the step, k_gemm<256> (BN = 256, plain epilogue;
# a quarter of the step's kernel time in the ncu launch list), on its largest
# call: the 56x56, 64 -> 256 1x1 forward with the fused BatchNorm statistics
# (four calls per step, 26.3 GFLOP and 514 MB of |x|+|w|+|y| per launch; AI 51
# flop/B, so HBM-bound).  Its DRAM traffic comes from one ncu capture of that
# single launch (bench.py --conv ... --stats under ncu -c 1).
KERNEL_LAYER = (256, 56, 56, 64, 256, 1, 1, 1, 0)
KERNEL_NAME = "k_gemm<256> (plain epilogue, forward statistics), 56x56 64->256 1x1 forward, batch 256"
TRAFFIC_JSON = os.path.join(ROOT, "profiles", "k_gemm_256_conv_56x56_64to256_fwd_stats_b256_traffic.json")
GEMM_SOURCES = ["pf16_gemm.cu", "pf16_epi.cuh", "pf16_api.cu", "pf16_internal.h", "pf16_ptx.cuh"]


def wgrad_is_gemm(h, w, c, k, r, s, st, pad):
    """Whether a layer's weight gradient runs as k_gemm launches: not the stem's
    (k_stem_wgrad) nor the 3x3 64-channel layers' on padded rows of 64
    (k_wgrad3x3_halo)."""
    if c == 3:
        return False
    return not (r == 3 and s == 3 and st == 1 and pad == 1 and c == 64 and k == 64 and w + 2 <= 64)


def gemm_source_digest():
    """sha256 over the conv GEMM kernel and the code that plans its launches."""
    import hashlib

    h = hashlib.sha256()
    for nm in GEMM_SOURCES:
        with open(os.path.join(ROOT, "paper_1911_07384_gb300", "csrc", nm), "rb") as f:
            h.update(nm.encode() + b"\0" + f.read())
    return h.hexdigest()


def ingest_traffic(csv_path):
    """DRAM traffic of the one k_gemm launch in an ncu CSV (metrics
    gpu__time_duration.sum, dram__bytes_read.sum, dram__bytes_write.sum) of
    `bench.py --conv <KERNEL_LAYER> --pass fwd --stats`, stored with the digest
    of the sources it was measured on."""
    import csv as _csv

    with open(csv_path) as f:
        rows = [r for r in _csv.reader(f)]
    hi = next(i for i, r in enumerate(rows) if "Kernel Name" in r)
    h = rows[hi]
    ki, mi, ui, vi, ii = (h.index("Kernel Name"), h.index("Metric Name"), h.index("Metric Unit"),
                          h.index("Metric Value"), h.index("ID"))
    scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "ns": 1, "nsecond": 1,
             "usecond": 1e3, "msecond": 1e6}
    per = {}
    for r in rows[hi + 1:]:
        if len(r) <= vi or "k_gemm" not in r[ki]:
            continue
        per.setdefault(r[ii], {})[r[mi]] = float(r[vi].replace(",", "")) * scale[r[ui]]
    if len(per) != 1:
        raise SystemExit(f"{csv_path}: {len(per)} k_gemm launches, expected the one captured launch")
    v = next(iter(per.values()))
    rd, wr = v["dram__bytes_read.sum"], v["dram__bytes_write.sum"]
    N, H, W, C, K, R, S, st, pd = KERNEL_LAYER
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    out = {"kernel": KERNEL_NAME, "layer": list(KERNEL_LAYER), "dram_read_bytes": rd, "dram_write_bytes": wr,
           "traffic_per_launch": rd + wr, "ncu_time_ns": v.get("gpu__time_duration.sum"),
           "algorithmic_bytes": 2 * (N * H * W * C + K * R * S * C + N * P * Q * K),
           "source_sha256": gemm_source_digest()}
    with open(TRAFFIC_JSON, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    print(json.dumps(out))
    return 0


def gemm_traffic():
    """Stored DRAM bytes of the one-launch capture, or None once the sources changed."""
    try:
        with open(TRAFFIC_JSON) as f:
            t = json.load(f)
    except (OSError, ValueError):
        return None
    return t["traffic_per_launch"] if t.get("source_sha256") == gemm_source_digest() else None


def kernel_roofline(pk, reps=10):
    """The dominant launch class on its largest call of the step, timed alone
    with CUDA events on a pre-loaded stream (its operands are larger than L2):
    algorithmic bytes |x|+|w|+|y| per launch over the launch time, against the
    measured copy bandwidth (the layer is HBM-bound); the tensor rate beside
    it for context."""
    r = time_conv(KERNEL_LAYER, "fwd", reps, 3, stats=True)
    byts = r["gbs"] * r["ms"] * 1e6
    return {"bound": "hbm", "kernel": KERNEL_NAME, "achieved": r["gbs"], "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": r["gbs"] / pk["hbm_gbs"], "traffic": gemm_traffic(), "algorithmic_bytes": byts,
            "ms_per_launch": r["ms"], "tflops": r["tflops"], "gflop_per_launch": r["tflops"] * r["ms"],
            "peak_src": f"{pk['src']} HBM copy"}


def one_phase_launch(d):
    """Whether the library runs a stride-2 data gradient's four stride phases
    as one launch: every phase has taps, and all share the output grid and
    the first dy row / column they read (as the library's planner decides)."""
    if d.stride != 2 or d.r == 1:
        return False

    def axis(n, k, ph):
        offs = [(ph + d.pad - r) // 2 for r in range(k) if (ph + d.pad - r) % 2 == 0]
        return (-(-(n - ph) // 2), min(offs)) if offs else None

    phases = [(axis(d.h, d.r, ph), axis(d.w, d.s, pw)) for ph in (0, 1) for pw in (0, 1)]
    return all(a is not None and b is not None for a, b in phases) and len(set(phases)) == 1


def count_launches(net):
    """Kernels of one step, counted by replaying the call sequence with a hook."""
    from paper_1911_07384_gb300 import pf16

    per = {"conv_fwd": 0, "conv_dgrad": 0, "conv_wgrad": 0, "bn_fwd": 2, "bn_bwd": 3, "maxpool_fwd": 1,
           "maxpool_bwd": 1, "avgpool_fwd": 1, "avgpool_bwd": 1, "softmax_xent": 2, "sgd": 1}
    total = 0
    for c in net.convs:
        d = c.desc
        stem = d.c == 3
        total += 1 + (1 if stem else 0)                      # fwd (+ the stem's space-to-depth)
        if not stem:
            phases = d.stride * d.stride if d.r > 1 and not one_phase_launch(d) else 1
            total += phases  # dgrad (a strided 1x1 also zero-fills dx, by a memset node)
        ws = pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD)
        total += 1 + (1 if ws else 0) + (2 if stem else 0)  # wgrad (+ split-K reduce, + the stem's s2d, scatter)
    # forward statistics come from the conv; backward ones from the data gradient where fused
    # (the swap variant's backward takes a second statistics pass)
    # (a BatchNorm applied in the next conv's operand path launches no apply pass)
    total += sum(per["bn_fwd"] + per["bn_bwd"] - (1 if getattr(b, "fused_bwd", False) else 0)
                 - (1 if getattr(b, "fused_apply", False) else 0)
                 + (1 if b.desc.flags & pf16.PF16_BN_SWAP else 0) for b in net.bns)
    # (the stem's fused BatchNorm + pooling forward: the BatchNorm's statistics final and the
    # fused pass -- the BatchNorm's count above, with no pooling launch)
    total += (0 if getattr(net, "stem_fused", False) else per["maxpool_fwd"]) + per["maxpool_bwd"]
    total += per["avgpool_fwd"] + per["avgpool_bwd"]
    total += per["softmax_xent"] + 2 * per["sgd"]
    return total


def conv_roofline(net, stream, reps=3):
    """Eager steps with CUDA events around every conv call on the launching
    stream (the stream pre-loaded, so that the events time the device only):
    algorithmic conv FLOPs / summed conv-call time."""
    import torch

    recs = []

    def hook(kind, layer, fn, *a, **kw):
        if kind.startswith("conv_"):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn(*a, **kw)
            e1.record(stream)
            recs.append((kind, layer, e0, e1))
            return None
        return fn(*a, **kw)

    totals = []
    by_pass = {"conv_fwd": [0.0, 0.0], "conv_dgrad": [0.0, 0.0], "conv_wgrad": [0.0, 0.0]}
    side, net.side = net.side, None  # per-call events need every call on `stream`, in program order
    for _ in range(reps):
        recs.clear()
        net.hook = hook
        preload(stream, 300)
        h0 = time.perf_counter()
        with torch.cuda.stream(stream):
            net.step()
        host_ms = 1e3 * (time.perf_counter() - h0)
        net.hook = None
        torch.cuda.synchronize()
        if host_ms > 250:
            raise RuntimeError(f"the step's host enqueue ({host_ms:.0f} ms) outlasted the stream pre-load")
        ms = 0.0
        for kind, layer, e0, e1 in recs:
            t = e0.elapsed_time(e1)
            ms += t
            by_pass[kind][0] += t
            by_pass[kind][1] += layer.flops
        totals.append(ms)
    net.side = side
    ms = float(np.median(totals))
    gflop = net.conv_flops() / 1e9
    # algorithmic bytes of a pass: |x| + |w| + |y| in FP16, each touched once
    byts, gemms = 0, 0
    for c in net.convs:
        d = c.desc
        P = (d.h + 2 * d.pad - d.r) // d.stride + 1
        Q = (d.w + 2 * d.pad - d.s) // d.stride + 1
        one = 2 * (d.n * d.h * d.w * d.c + d.k * d.r * d.s * d.c + d.n * P * Q * d.k)
        stem = d.c == 3
        # the k_gemm launches the stored traffic covers: every pass but the weight
        # gradients of other kernels (k_stem_wgrad, k_wgrad3x3_halo)
        wg = wgrad_is_gemm(d.h, d.w, d.c, d.k, d.r, d.s, d.stride, d.pad)
        byts += one * ((1 if stem else 2) + (1 if wg else 0))
        dg = 1 if d.r == 1 or one_phase_launch(d) else d.stride * d.stride
        gemms += 1 + (0 if stem else dg) + (1 if wg else 0)
    out = {"ms": ms, "gflop": gflop, "tflops": gflop / ms, "by_pass": {}, "bytes_per_launch": byts / gemms}
    for k, (t, f) in by_pass.items():
        out["by_pass"][k] = {"ms": t / reps, "tflops": (f / reps) / 1e9 / (t / reps) if t else None}
    return out


if __name__ == "__main__":
    sys.exit(main())
