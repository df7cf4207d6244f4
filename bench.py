#!/usr/bin/env python
"""Benchmark of the bit-precise convolution hot path on GB300.

Headline (one JSON line on rank 0): effective int MAC/s of the 3x3
convolution N8 C64 -> 64 on 56x56 (pad 1) over the bit-width sweep -- lane
widths b = 1..8 for activations and weights, all four signed/unsigned
combinations, int32 accumulation requantized to a packed b-bit output. One
step runs the 32 layers (one CUDA graph of 32 kernel launches). Weights are
prepared once, as an inference deployment does at load time.

Also reported: the packed elementwise ops (add, sub, mul, ReLU, requantize)
plus pack/unpack and max-pool in GB/s on 2^28-lane arrays at every width;
the conv kernel's roofline fraction; the same metric end to end through the
C ABI from pinned host buffers; the CPU oracle timed on the host cores.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl samd|reference]
                  [--workload sweep|vgg16|resnet50|conv1x]
"""
from __future__ import annotations

import argparse
import glob
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

L2_FLUSH_BYTES = 512 << 20  # > 129 MB L2
L2_BYTES = 129 * 10**6
METRIC = "effective int MAC/s for b-bit conv2d vs bit width (fraction of int8 TC peak); packed-op GB/s"


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="samd", choices=["samd", "reference"])
    ap.add_argument("--workload", default="sweep", choices=["sweep", "vgg16", "resnet50", "conv1x"])
    ap.add_argument("--no-packed-ops", action="store_true")
    ap.add_argument("--profile-fused-pool", action="store_true",
                    help="VGG-16 conv7 (N16 C256->256 56x56, u4 x s4 -> u4) with the 2x2 max-pool fused into its "
                         "epilogue, one untimed call and one more, and exit: the command ncu captures for the fused "
                         "pool")
    ap.add_argument("--profile-ops", action="store_true",
                    help="launch each packed op once at 2^28 lanes (b = 1, 4, 8; pack, unpack, the five elementwise "
                         "ops) and the VGG-16 block-1 max-pool, after one untimed warm-up launch of each, and exit: "
                         "the command ncu captures for the packed ops' DRAM counters")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--layers", type=str, default="", help="comma-separated layer indices (profiling aid)")
    ap.add_argument("--tiles-per-cta", type=int, default=0,
                    help="samd_conv2d_set_min_tiles_per_cta for the step (0: 8 for the sweep's 32 concurrent "
                         "small layers, else the library default)")
    ap.add_argument("--l2", default="rotate", choices=["rotate", "flush"],
                    help="keep a step's data out of L2 by cycling through sets of inputs larger than L2 in "
                         "total (rotate), or by flushing L2 before every step (flush)")
    ap.add_argument("--streams", type=int, default=8,
                    help="independent layers of a step run on this many streams (graph branches)")
    ap.add_argument("--connections", type=int, default=0,
                    help="CUDA_DEVICE_MAX_CONNECTIONS for this process (hardware work queues the streams map "
                         "onto; 0: leave the environment as it is)")
    return ap.parse_args()


# ---- distributed plumbing ------------------------------------------------------------

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


class Dist:
    def __init__(self, backend):
        import torch.distributed as dist

        self.ws, self.rank, self.local = dist_env()
        self.dist = dist if self.ws > 1 else None
        if self.dist:
            dist.init_process_group(backend)

    def barrier(self):
        if self.dist:
            self.dist.barrier()

    def max(self, x: float) -> float:
        if not self.dist:
            return x
        import torch

        t = torch.tensor([x], dtype=torch.float64, device="cuda" if self.dist.get_backend() == "nccl" else "cpu")
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.dist:
            self.dist.destroy_process_group()


def whole_job_rate(d: Dist, units_per_step: float, steps: int, local_seconds: float):
    """Weak scaling over replicas: every rank runs `steps` steps of
    `units_per_step` units; the job took as long as its slowest rank. Returns
    (units per second over all ranks, ms per step of the slowest rank)."""
    slowest = d.max(local_seconds)
    return units_per_step * steps * d.ws / slowest, slowest / steps * 1e3


# ---- clocks ------------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax, "samples": len(sm),
                "reasons": sorted(reasons)}


# ---- CPU oracle baseline ---------------------------------------------------------------

def cpu_oracle_rate(layers, seconds: float, threads: int = 0):
    """The oracle's direct convolution on one image of each layer in turn, on
    `threads` host threads (0: all cores), until `seconds` have passed.
    Returns (MAC/s, threads, sample)."""
    import oracle
    from paper_1809_10572_gb300 import synth

    threads = threads or os.cpu_count() or 1
    done_macs, t0, k = 0, time.perf_counter(), 0
    names = []
    while time.perf_counter() - t0 < seconds or k == 0:
        layer = layers[k % len(layers)]
        s = layer.shape
        a = synth.lanes(synth.seed_for("cpu", k), (1, s.C, s.H, s.W), layer.ba, layer.sa)
        w = synth.lanes(synth.seed_for("cpuw", k), (s.K, s.C, s.R, s.S), layer.bw, layer.sw)
        oracle.conv2d(a, w, stride=s.stride, pad=s.pad, nthreads=threads)
        done_macs += s.macs // s.N
        names.append(layer.name)
        k += 1
    el = time.perf_counter() - t0
    sample = f"{k} single-image layer runs ({', '.join(sorted(set(names))[:4])}{'...' if len(set(names)) > 4 else ''}), " \
             f"{done_macs / 1e9:.2f} GMAC in {el:.1f} s"
    return done_macs / el, threads, sample


# ---- the reference arm: the CPU oracle ------------------------------------------------

def run_reference(args, layers):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    from paper_1809_10572_gb300 import synth

    threads = os.cpu_count() or 1
    # one step = one image of each layer of the workload (a bounded sample)
    inputs = []
    for i, layer in enumerate(layers):
        s = layer.shape
        inputs.append((synth.lanes(synth.seed_for("ref", i), (1, s.C, s.H, s.W), layer.ba, layer.sa),
                       synth.lanes(synth.seed_for("refw", i), (s.K, s.C, s.R, s.S), layer.bw, layer.sw), s))
    step_macs = sum(s.macs // s.N for _, _, s in inputs)

    def step():
        for a, w, s in inputs:
            oracle.conv2d(a, w, stride=s.stride, pad=s.pad, nthreads=threads)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    value = step_macs * args.steps / el
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "MAC/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": workload_config(args, layers),
        "cpu_baseline": {"value": value, "unit": "MAC/s", "cores": threads, "kind": "oracle",
                         "sample": f"one image of each of the {len(layers)} layers per step "
                                   f"({step_macs / 1e9:.2f} GMAC/step)"},
        "e2e": {"value": value, "unit": "MAC/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_config(args, layers):
    from paper_1809_10572_gb300 import workloads

    desc = {
        "sweep": "3x3 conv N8 C64->64 56x56 pad1 stride1; act=weight=out width b in 1..8, signs uu/us/su/ss "
                 "(32 layers), int32 acc requantized to packed b-bit; 32-bit words",
        "vgg16": "VGG-16 13 conv layers 224x224 batch16, u4 act x s4 wt -> u4, chained: each layer reads the "
                 "previous one's packed output, with the 4 2x2 max-pools between blocks in the timed step (fused "
                 "into the conv epilogue for conv4, conv7 and conv10; standalone after conv2)",
        "resnet50": "ResNet-50 v1.5 stage convs (52) batch64, u6 act x s2 wt -> u6",
        "conv1x": "3x3 conv N1 C16->16 32x32, u4 x s4, 64-bit words",
    }[args.workload]
    return {"workload": desc, "layers": len(layers), "macs_per_step": workloads.total_macs(layers),
            "l2": ("inputs larger than L2: independent sets of packed inputs, prepared weights and outputs, "
                   "together at least twice the L2, used in turn (one set per step), no flush; "
                   "value_l2_flushed: one set with L2 flushed (512 MiB write + 512 MiB read) before every step"
                   if args.l2 == "rotate" else
                   "flushed before every step (512 MiB write, then 512 MiB read); inputs resident in HBM"),
            "weights": "prepared once into the tensor-core operand layout (samd_conv2d_prepare), not in the step",
            "launch": f"one CUDA graph per step; independent layers fanned out over {args.streams} streams"
                      f"{f' ({args.connections} hardware work queues)' if args.connections else ''}; "
                      f"each CTA at least {args.tiles_per_cta or (8 if args.workload == 'sweep' else 4)} reference tiles "
                      f"of work (samd_conv2d_set_min_tiles_per_cta)",
            "parallelism": f"replicas x{args.gpus}"}


# ---- the samd arm ------------------------------------------------------------------------

def build_layers(layers, dev, chain=False):
    """Packed inputs, prepared weights and output buffers of every layer.
    With chain=True (VGG-16 as one network) only the first layer gets a
    synthetic input; every other layer reads the previous layer's packed
    output, or the 2x2 max-pool of it where the layer is marked pool_after
    (the pool's output buffer is the entry's "pooled")."""
    import torch

    from paper_1809_10572_gb300 import samd, synth, workloads

    built = []
    prev = None
    for i, layer in enumerate(layers):
        s = layer.shape
        fa = samd.fmt(layer.ba, layer.sa, 0, layer.word_bits)
        fw = samd.fmt(layer.bw, layer.sw, 0, layer.word_bits)
        fo = samd.fmt(layer.bo, layer.so, 0, layer.word_bits)
        if chain and prev is not None:
            a_w = prev
        else:
            a = synth.lanes_t(synth.seed_for("bench", i), (s.N * s.H * s.W, s.C), layer.ba, layer.sa, device=dev)
            a_w = samd.pack(synth.to_bytes_t(a), fa)
            del a
        w = synth.lanes_t(synth.seed_for("benchw", i), (s.K * s.R * s.S, s.C), layer.bw, layer.sw, device=dev)
        w_w = samd.pack(synth.to_bytes_t(w), fw)
        conv = samd.PreparedConv(w_w, s, fa, fw, fo)
        _, out = conv.outputs(want_acc=False)
        shift = workloads.harness_shift(layer.ba, layer.bw, layer.bo, s.C * s.R * s.S)
        opb = samd.samd_conv2d_operand_bits(s.desc(), fa, fw)  # 8: e4m3 operands, 16: fp16
        pooled, fused = None, False
        if chain and layer.pool_after:
            pooled = samd.empty_words(fo, s.N * (s.Ho // 2) * (s.Wo // 2), s.K, dev)
            # the pool fused into the convolution's epilogue where the kernel
            # supports it (samd_conv2d_prepared_pool2x2), else a second launch
            fused = conv.pool2x2_supported()
        built.append({"layer": layer, "conv": conv, "act": a_w, "out": out, "shift": shift, "operand_bits": opb,
                      "fo": fo, "pooled": pooled, "fused_pool": fused})
        prev = pooled if pooled is not None else out
    torch.cuda.synchronize()
    return built


def _graph_time(fn, stream, reps=7):
    """Median device time of fn's launches, captured once into a CUDA graph
    and replayed (no host launch cost in the measurement)."""
    import torch

    with torch.cuda.stream(stream):
        fn(stream)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn(torch.cuda.current_stream())
    cur = torch.cuda.current_stream()  # replay() launches the graph here
    ts = []
    for _ in range(reps):
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(cur)
        g.replay()
        s1.record(cur)
        s1.synchronize()
        ts.append(s0.elapsed_time(s1) * 1e-3)
    return statistics.median(ts)


def choose_pool_forms(built, stream):
    """For each layer whose 2x2 max-pool the kernel can fuse, time the fused
    call against the convolution followed by samd_maxpool2x2 (each alone, in
    a CUDA graph) and keep the faster; returns the measured times (the two
    forms give the same words, tests/test_gpu_pool.py)."""
    from paper_1809_10572_gb300 import samd

    forms = {}
    for b in built:
        if not b["fused_pool"]:
            continue
        s = b["layer"].shape

        def fused(st, b=b):
            b["conv"].pool2x2(b["act"], b["pooled"], b["shift"], stream=st)

        def two(st, b=b, s=s):
            b["conv"](b["act"], None, b["out"], b["shift"], stream=st)
            samd.samd_maxpool2x2(b["fo"], b["out"], b["pooled"], s.N, s.K, s.Ho, s.Wo, stream=st)

        tf, t2 = _graph_time(fused, stream), _graph_time(two, stream)
        b["fused_pool"] = tf < t2
        forms[b["layer"].name] = {"fused_us": tf * 1e6, "conv_then_pool_us": t2 * 1e6,
                                  "chosen": "fused" if tf < t2 else "conv then pool"}
    return forms


def unique_bytes(built):
    """Bytes of the distinct device tensors of a built workload."""
    seen, total = set(), 0
    for b in built:
        for t in (b["act"], b["out"], b["conv"].prepared, b.get("pooled")):
            if t is not None and t.data_ptr() not in seen:
                seen.add(t.data_ptr())
                total += t.numel() * t.element_size()
    return total


def launches_per_step(built):
    return sum(1 + (1 if b.get("pooled") is not None and not b.get("fused_pool") else 0) for b in built)


def run_chain(bs, stream):
    """The layers of a chained network in order on one stream: each
    convolution, then the 2x2 max-pool of its output where the network has
    one (fused into the convolution where the kernel supports it)."""
    from paper_1809_10572_gb300 import samd

    for b in bs:
        if b["fused_pool"]:
            b["conv"].pool2x2(b["act"], b["pooled"], b["shift"], stream=stream)
            continue
        b["conv"](b["act"], None, b["out"], b["shift"], stream=stream)
        if b["pooled"] is not None:
            s = b["layer"].shape
            samd.samd_maxpool2x2(b["fo"], b["out"], b["pooled"], s.N, s.K, s.Ho, s.Wo, stream=stream)


def time_packed_ops(dev, flush):
    """GB/s of pack/unpack, the five elementwise ops (spacer-free, and with one
    permanent spacer bit per lane) and max-pool at 2^28 lanes.

    Each figure times 8 launches back to back, rotating over independent sets
    of input and output buffers whose total is at least twice the L2: each
    launch finds its inputs in DRAM, and the write-back of one launch's output
    happens during the next one, inside the timed region (only the last
    launch's may escape it). L2 is flushed before the first launch."""
    import torch

    from paper_1809_10572_gb300 import samd, synth, workloads

    n = workloads.ELEMENTWISE_N
    res = {}
    reps = 8
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def n_sets(set_bytes):
        return max(2, -(-2 * L2_BYTES // set_bytes) + 1)

    def timed(fns, nbytes):
        ts = []
        for _ in range(3):
            flush()
            start.record()
            for i in range(reps):
                fns[i % len(fns)]()
            end.record()
            end.synchronize()
            ts.append(start.elapsed_time(end) * 1e-3)
        return reps * nbytes / statistics.median(ts) / 1e9

    for spacer in (0, 1):
        for signed in (False, True):
            tag = ("s" if signed else "u") + ("_spacer1" if spacer else "")
            for b in range(1, 9 - spacer):
                f = samd.fmt(b, signed, spacer)
                xb = synth.to_bytes_t(synth.lanes_t(synth.seed_for("ewx", b, signed), (n,), b, signed, device=dev))
                xw = samd.pack(xb, f)
                wbytes = xw.numel() * 4
                ns = n_sets(2 * wbytes + (n if spacer == 0 else 0))
                xws = [xw] + [xw.clone() for _ in range(ns - 1)]
                yws = [samd.pack(synth.to_bytes_t(synth.lanes_t(synth.seed_for("ewy", b, signed, k), (n,), b, signed,
                                                                device=dev)), f) for k in range(ns)]
                outs = [torch.empty_like(xw) for _ in range(ns)]
                if spacer == 0:
                    xbs = [xb] + [xb.clone() for _ in range(ns - 1)]
                    res.setdefault("pack", {}).setdefault(tag, []).append(timed(
                        [lambda k=k: samd.samd_pack(f, xbs[k], outs[k], 1, n) for k in range(ns)], n + wbytes))
                    res.setdefault("unpack", {}).setdefault(tag, []).append(timed(
                        [lambda k=k: samd.samd_unpack(f, xws[k], xbs[k], 1, n) for k in range(ns)], n + wbytes))
                    del xbs
                for op in workloads.ELEMENTWISE_OPS:
                    binary = op in ("add", "sub", "mul")
                    nb = (3 if binary else 2) * wbytes
                    res.setdefault(op, {}).setdefault(tag, []).append(timed(
                        [lambda k=k: samd.samd_elementwise(op, f, xws[k], yws[k] if binary else None, f, outs[k], n,
                                                           1 if op == "requant" else 0, 0) for k in range(ns)], nb))
                del xb, xw, xws, yws, outs
    # 2x2 max-pool on VGG-16 block-1 activations (224 x 224 x 64, u4): at
    # batch 128 (258 MB moved) and at the workload's batch 16 (32 MB)
    f = samd.fmt(4, False)
    C, H, W = 64, 224, 224
    for N, key in ((128, "maxpool2x2"), (16, "maxpool2x2_batch16")):
        xw = samd.pack(synth.to_bytes_t(synth.lanes_t(5, (N * H * W, C), 4, False, device=dev)), f)
        out = samd.empty_words(f, N * H * W // 4, C, dev)
        nb = (xw.numel() + out.numel()) * 4
        ns = n_sets(nb)
        xs = [xw] + [xw.clone() for _ in range(ns - 1)]
        outs = [out] + [torch.empty_like(out) for _ in range(ns - 1)]
        res[key] = {"u": [timed([lambda k=k: samd.samd_maxpool2x2(f, xs[k], outs[k], N, C, H, W) for k in range(ns)],
                                nb)]}
        del xw, out, xs, outs
    return res


def time_nchw_widemul(dev):
    """The paper's wide-multiply engine (NCHW packed along W, CUDA cores) on
    the sweep's 3x3 C64 -> 64 56x56 layer at batch 8, for the lane widths whose
    kernel row fits one 64-bit word: effective MAC/s, beside the tensor-core
    path's per-layer rates."""
    import torch

    from paper_1809_10572_gb300 import samd, synth

    shape = samd.ConvShape(8, 64, 56, 56, 64)
    out = {}
    for b, sa, sw in [(1, False, False), (1, True, True), (2, False, False), (2, True, True), (3, True, True),
                      (4, False, True), (4, True, True), (5, True, True)]:
        fa, fw = samd.fmt(b, sa), samd.fmt(b, sw)
        desc = shape.desc(samd.SAMD_NCHW)
        if samd.samd_conv2d_operand_bits(desc, fa, fw) == 0:
            continue
        a = samd.pack(synth.to_bytes_t(synth.lanes_t(1, (shape.N * shape.C * shape.H, shape.W), b, sa, device=dev)),
                      fa)
        w = samd.pack(synth.to_bytes_t(synth.lanes_t(2, (shape.K * shape.C * shape.R, shape.S), b, sw, device=dev)),
                      fw)
        ws = torch.empty(samd.samd_conv2d_workspace_size(desc, fa, fw), dtype=torch.uint8, device=dev)
        packed = samd.empty_words(fa, shape.N * shape.K * shape.Ho, shape.Wo, dev)
        run = lambda: samd.samd_conv2d(desc, fa, a, fw, w, None, fa, packed, b, ws)
        t = _best_time(run, reps=5)
        out[f"b{b}_{'s' if sa else 'u'}{'s' if sw else 'u'}"] = shape.macs / t
    return out


def profile_ops():
    """Each packed op once at 2^28 lanes for b = 1, 4, 8 (unsigned, 32-bit
    words), then the 2x2 max-pool of VGG-16 block 1 (N16 224x224 C64 u4). The
    first round of launches is a warm-up; the second is the one profiled
    (ncu -s <launches of one round>). Prints the order of the launches."""
    import torch

    from paper_1809_10572_gb300 import samd, synth, workloads

    dev = torch.device("cuda", 0)
    samd.load()
    n = workloads.ELEMENTWISE_N
    calls = []
    for b in (1, 4, 8):
        f = samd.fmt(b, False)
        xb = synth.to_bytes_t(synth.lanes_t(synth.seed_for("ewx", b, False), (n,), b, False, device=dev))
        xw = samd.pack(xb, f)
        yw = samd.pack(synth.to_bytes_t(synth.lanes_t(synth.seed_for("ewy", b, False, 0), (n,), b, False,
                                                      device=dev)), f)
        out = torch.empty_like(xw)
        ub = torch.empty_like(xb)
        calls.append((f"pack b{b}", lambda f=f, xb=xb, out=out: samd.samd_pack(f, xb, out, 1, n)))
        calls.append((f"unpack b{b}", lambda f=f, xw=xw, ub=ub: samd.samd_unpack(f, xw, ub, 1, n)))
        for op in workloads.ELEMENTWISE_OPS:
            binary = op in ("add", "sub", "mul")
            calls.append((f"{op} b{b}", lambda f=f, op=op, xw=xw, yw=yw, out=out, binary=binary: samd.samd_elementwise(
                op, f, xw, yw if binary else None, f, out, n, 1 if op == "requant" else 0, 0)))
    f4 = samd.fmt(4, False)
    N, C, H, W = 16, 64, 224, 224
    pin = samd.pack(synth.to_bytes_t(synth.lanes_t(5, (N * H * W, C), 4, False, device=dev)), f4)
    pout = samd.empty_words(f4, N * H * W // 4, C, dev)
    calls.append(("maxpool2x2 N16 C64 224x224 u4", lambda: samd.samd_maxpool2x2(f4, pin, pout, N, C, H, W)))
    for rnd in range(2):
        for name, fn in calls:
            fn()
        torch.cuda.synchronize()
    print(json.dumps({"profile_ops": [name for name, _ in calls], "launches_per_round": len(calls)}), flush=True)
    return 0


def profile_fused_pool():
    """VGG-16 conv7 with its pool fused (samd_conv2d_prepared_pool2x2): the
    first call is a warm-up, the second the one profiled (ncu -s 1 -c 1)."""
    import torch

    from paper_1809_10572_gb300 import samd, synth, workloads

    dev = torch.device("cuda", 0)
    samd.load()
    layer = next(l for l in workloads.vgg16() if l.name == "conv7")
    s = layer.shape
    fa, fw, fo = samd.fmt(layer.ba, layer.sa), samd.fmt(layer.bw, layer.sw), samd.fmt(layer.bo, layer.so)
    a_w = samd.pack(synth.to_bytes_t(synth.lanes_t(11, (s.N * s.H * s.W, s.C), layer.ba, layer.sa, device=dev)), fa)
    w_w = samd.pack(synth.to_bytes_t(synth.lanes_t(12, (s.K * s.R * s.S, s.C), layer.bw, layer.sw, device=dev)), fw)
    conv = samd.PreparedConv(w_w, s, fa, fw, fo)
    pooled = samd.empty_words(fo, s.N * (s.Ho // 2) * (s.Wo // 2), s.K, dev)
    shift = workloads.harness_shift(layer.ba, layer.bw, layer.bo, s.C * s.R * s.S)
    for _ in range(2):
        conv.pool2x2(a_w, pooled, shift)
    torch.cuda.synchronize()
    print(json.dumps({"profile_fused_pool": layer.name, "pooled_bytes": pooled.numel() * 4,
                      "input_bytes": a_w.numel() * 4}), flush=True)
    return 0


def csrc_digest():
    """sha256 over the kernel sources (file names and contents)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_1809_10572_gb300", "csrc")
    for f in sorted(glob.glob(os.path.join(csrc, "*.cu")) + glob.glob(os.path.join(csrc, "*.cuh"))):
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def measured_traffic(args):
    """DRAM bytes per conv launch of the sweep step from the committed ncu
    summary, if the kernel sources are still the ones it measured."""
    if args.workload != "sweep" or args.layers:
        return None, "measured for the full sweep step only"
    try:
        with open(os.path.join(ROOT, "profiles", "conv_kernel_sweep_traffic.json")) as fh:
            rec = json.load(fh)
    except (OSError, ValueError):
        return None, "no ncu traffic summary"
    if rec.get("csrc_sha256") != csrc_digest():
        return None, "kernel sources changed since the ncu traffic capture"
    return rec["dram_bytes_per_launch"], ("ncu dram__bytes_read.sum + dram__bytes_write.sum, mean over the step's "
                                          f"{rec['launches']} launches")


def run_samd(args, layers):
    import torch

    from paper_1809_10572_gb300 import samd, workloads

    ws, rank, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    d = Dist("nccl")
    samd.load()

    # the sweep's 32 small layers run concurrently: each keeps to a few SMs
    tpc = args.tiles_per_cta or (8 if args.workload == "sweep" else 4)
    samd.samd_conv2d_set_min_tiles_per_cta(tpc)
    chain = args.workload == "vgg16"  # one network: each layer reads the previous one's (pooled) output
    built = build_layers(layers, dev, chain)
    pool_forms = choose_pool_forms(built, torch.cuda.Stream(device=dev)) if chain else {}
    step_macs = workloads.total_macs(layers)
    # Between timed steps no step may find its data in L2. The step works on
    # one of R independent sets of inputs, prepared weights and outputs, the
    # next set each step, with R x (bytes of a set) at least twice the L2:
    # when a set comes round again, more than an L2's worth of other data has
    # passed through since. (--l2 flush keeps one set and flushes L2 instead;
    # the line reports that number too.)
    set_bytes = unique_bytes(built)
    n_sets = max(1, -(-2 * L2_BYTES // set_bytes)) if args.l2 == "rotate" else 1
    sets = [built] + [build_layers(layers, dev, chain) for _ in range(n_sets - 1)]
    for bs in sets[1:]:  # the same choice in every set
        for b, b0 in zip(bs, built):
            b["fused_pool"] = b0["fused_pool"]
    flush_w = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flush_r = torch.ones(L2_FLUSH_BYTES // 8, dtype=torch.int64, device=dev)

    def flush():
        # write a buffer larger than L2, then read another one: the timed
        # kernel starts with none of its data in L2 and no dirty lines left to
        # write back on its time
        flush_w.fill_(1)
        torch.sum(flush_r)

    stream = torch.cuda.Stream(device=dev)
    side = [torch.cuda.Stream(device=dev) for _ in range(max(1, args.streams))]

    def step_calls(main, bs):
        if chain:
            run_chain(bs, main)
            return
        # the layers of the workload are independent: fan them out over the
        # side streams and join them back into `main`
        for sd in side:
            sd.wait_stream(main)
        for i, b in enumerate(bs):
            b["conv"](b["act"], None, b["out"], b["shift"], stream=side[i % len(side)])
        for sd in side:
            main.wait_stream(sd)

    # first calls outside any capture (kernel attributes, tensor-map entry point)
    with torch.cuda.stream(stream):
        step_calls(stream, built)
    torch.cuda.synchronize()
    graphs = []
    for bs in sets:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step_calls(torch.cuda.current_stream(), bs)
        graphs.append(g)
    torch.cuda.synchronize()
    if samd.samd_device_status() != 0:
        raise RuntimeError("a kernel recorded a timeout")

    def timed_steps(use_flush, sample_clocks):
        """K steps after W warm-up steps; with use_flush one set and an L2
        flush before every step (outside the events), else the sets in turn."""
        gs = graphs[:1] if use_flush else graphs
        for w in range(args.warmup):
            if use_flush:
                flush()
            gs[w % len(gs)].replay()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        clocks = ClockSampler(local)
        if sample_clocks and rank == 0:
            clocks.start()
        d.barrier()
        torch.cuda.synchronize()
        t_wall = time.perf_counter()
        cur = torch.cuda.current_stream()
        for i in range(args.steps):
            if use_flush:
                flush()
            ev[i][0].record(cur)
            gs[(args.warmup + i) % len(gs)].replay()
            ev[i][1].record(cur)
        torch.cuda.synchronize()
        d.barrier()
        wall_s = time.perf_counter() - t_wall
        clk_s = clocks.stop() if sample_clocks and rank == 0 else None
        if samd.samd_device_status() != 0:
            raise RuntimeError("a kernel recorded a timeout")
        return [a.elapsed_time(b) * 1e-3 for a, b in ev], wall_s, clk_s

    # timed region
    step_s, wall, clk = timed_steps(args.l2 == "flush", True)
    value, ms_per_step = whole_job_rate(d, step_macs, args.steps, sum(step_s))
    if args.l2 == "rotate":  # the same step with one set and an L2 flush before every step
        flushed_s, _, _ = timed_steps(True, False)
        value_flushed, _ = whole_job_rate(d, step_macs, args.steps, sum(flushed_s))
    else:
        value_flushed = value
    l2_note = (f"inputs larger than L2: {n_sets} sets of packed inputs, prepared weights and outputs "
               f"({n_sets} x {set_bytes / 1e6:.1f} MB) used in turn, one set per step, no flush"
               if args.l2 == "rotate" else
               "flushed before every step (512 MiB write, then 512 MiB read); inputs resident in HBM")

    cur = torch.cuda.current_stream()
    # per-layer throughput (one graph per layer, replayed with events; each
    # layer alone, so with the library's default spread over the SMs)
    samd.samd_conv2d_set_min_tiles_per_cta(4)
    by_layer = {}
    for b in built:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            b["conv"](b["act"], None, b["out"], b["shift"], stream=torch.cuda.current_stream())
        ts = []
        for _ in range(5):
            flush()
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s0.record(cur)
            g.replay()
            s1.record(cur)
            s1.synchronize()
            ts.append(s0.elapsed_time(s1) * 1e-3)
        by_layer[b["layer"].name] = b["layer"].macs / statistics.median(ts)

    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        pass
    bf16_peak = peaks.get("bf16_tflops")
    peak_src = "measured" if bf16_peak else "fallback"
    bf16_peak = bf16_peak or 1900.0
    # The peak of each layer is that of its operand type: fp16 runs at the
    # bf16 rate (MEASURED_PEAKS.json, burst); e4m3 at the e4m3 rate measured
    # here (cuBLASLt through torch._scaled_mm), or at twice the bf16 rate (the
    # nominal 4.5 / 2.25 PFLOP/s dense ratio) if that cannot be measured. The
    # step's peak is the rate at which every layer would run at its own peak:
    # 2 x step MACs / sum of the layers' ideal times.
    e4m3 = measure_e4m3_peak(dev)
    e4m3_peak = e4m3["tflops"] or 2.0 * bf16_peak
    e4m3_src = "measured (torch._scaled_mm 8192^3)" if e4m3["tflops"] else f"2 x {peak_src} bf16"

    def layer_peak(b):
        return e4m3_peak if b["operand_bits"] == 8 else bf16_peak

    ideal_s = sum(2.0 * b["layer"].macs / (layer_peak(b) * 1e12) for b in built)
    step_peak = 2.0 * step_macs / ideal_s / 1e12
    n_e4m3 = sum(1 for b in built if b["operand_bits"] == 8)
    achieved_tflops = 2.0 * step_macs / (ms_per_step * 1e-3) / 1e12
    traffic, traffic_note = measured_traffic(args)
    roofline = {"kernel": "conv_kernel", "bound": "tensor", "achieved": achieved_tflops, "peak": step_peak,
                "unit": "TFLOP/s", "frac": achieved_tflops / step_peak, "traffic": traffic,
                "traffic_note": traffic_note,
                "peak_source": f"fp16 layers: {peak_src} bf16 burst {bf16_peak:.1f} TFLOP/s; e4m3 layers "
                               f"({n_e4m3} of {len(built)}): {e4m3_src} {e4m3_peak:.1f} TFLOP/s; MAC-weighted",
                "e4m3_peak": e4m3,
                "frac_vs_nominal_ratio": achieved_tflops / (2.0 * step_macs / sum(
                    2.0 * b["layer"].macs / ((2.0 if b["operand_bits"] == 8 else 1.0) * bf16_peak * 1e12)
                    for b in built) / 1e12),
                "note": ("achieved = 2 x direct-conv MACs of the step / step time (the step's "
                         f"{launches_per_step(built) - len(built)} standalone max-pool launches and "
                         f"{sum(1 for b in built if b.get('fused_pool'))} fused pool epilogues included, so "
                         "achieved is understated); " if chain else
                         "achieved = 2 x direct-conv MACs of the step / step time (all launches are the conv "
                         "kernel); ") + "frac_vs_nominal_ratio takes e4m3 at 2 x the bf16 peak instead"}

    line = {
        "metric": METRIC, "value": value, "unit": "MAC/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "e4m3 or f16 operands -> f32 tensor-core accumulation of exact integers (b-bit packed lanes)",
        "data": "synthetic",
        "config": workload_config(args, layers), "l2_sets": l2_note, "value_l2_flushed": value_flushed,
        "wall_s_timed_region": wall,
        "gpu_launches": args.steps * launches_per_step(built),
        "roofline": roofline,
    }
    if args.workload == "sweep":
        per_bits = {}
        for name, v in by_layer.items():
            per_bits.setdefault(name.split("_")[0], []).append(v)
        line["by_bits_mac_s"] = {k: statistics.mean(v) for k, v in per_bits.items()}
    line["by_layer_mac_s"] = by_layer
    if pool_forms:
        line["pool_forms"] = pool_forms

    # int8 tensor-core peak (for the metric's "fraction of int8 TC peak")
    if rank == 0:
        line["int8_tc_peak"] = measure_int8_peak(dev)
        if line["int8_tc_peak"].get("tops"):
            line["frac_of_int8_tc_peak"] = 2 * value / ws / (line["int8_tc_peak"]["tops"] * 1e12)

    # e2e: the same step through the C ABI from pinned host buffers
    if not args.no_e2e:
        line["e2e"] = measure_e2e(built, step_macs, args, dev, ws, d, chain)

    if rank == 0 and not args.no_packed_ops:
        ops = time_packed_ops(dev, flush)
        hbm = peaks.get("hbm_gbs") or 6800.0
        fr = [v / hbm for op, sg in ops.items() if op != "maxpool2x2_batch16" for vals in sg.values() for v in vals]
        line["packed_ops_gb_s"] = ops
        line["packed_ops_roofline"] = {"bound": "hbm", "peak": hbm, "unit": "GB/s",
                                       "peak_source": "measured" if peaks.get("hbm_gbs") else "fallback",
                                       "min_frac": min(fr), "median_frac": statistics.median(fr), "max_frac": max(fr),
                                       "n": 2 ** 28, "word_bits": 32,
                                       "bytes": "each input word read once + each output word written once",
                                       "timing": "8 launches back to back over rotating buffer sets of more than "
                                                 "twice the L2 (write-back of each output inside the timed region); "
                                                 "L2 flushed first"}
        line["nchw_widemul_mac_s"] = time_nchw_widemul(dev)
    line["clocks"] = clk
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, cores, sample = cpu_oracle_rate(layers, args.cpu_seconds)
        v1, _, sample1 = cpu_oracle_rate(layers, args.cpu_seconds / 3, threads=1)
        line["cpu_baseline"] = {"value": v, "unit": "MAC/s", "cores": cores, "kind": "oracle", "sample": sample,
                                "value_1thread": v1, "sample_1thread": sample1}
    if rank == 0:
        print(json.dumps(line), flush=True)
    d.close()
    return 0


def _best_time(fn, reps=5):
    import torch

    fn()
    torch.cuda.synchronize()
    best = None
    for _ in range(reps):
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record()
        fn()
        s1.record()
        s1.synchronize()
        t = s0.elapsed_time(s1) * 1e-3
        best = t if best is None else min(best, t)
    return best


def measure_int8_peak(dev):
    """Dense int8 tensor-core rate, the best of torch._int_mm (cuBLASLt) on
    8192^3 and the hand-written mma.sync m16n8k32 s8 loop (libsamd_peaks)."""
    import ctypes

    import torch

    from paper_1809_10572_gb300 import build as samd_build

    res = {}
    try:
        n = 8192
        a = torch.randint(-128, 127, (n, n), dtype=torch.int8, device=dev)
        b = torch.randint(-128, 127, (n, n), dtype=torch.int8, device=dev)
        res["int_mm_tops"] = 2 * n ** 3 / _best_time(lambda: torch._int_mm(a, b)) / 1e12
        del a, b
    except Exception as e:  # noqa: BLE001
        res["int_mm_tops"] = None
        res["int_mm_error"] = type(e).__name__
    try:
        lib = ctypes.CDLL(samd_build.build_peaks())
        lib.samd_peak_imma_s8.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                          ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_double)]
        lib.samd_peak_imma_s8.restype = ctypes.c_int
        scratch = torch.zeros(4, dtype=torch.int32, device=dev)
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        best = None
        for per_sm in (2, 4, 8):
            ms, macs = ctypes.c_float(0), ctypes.c_double(0)
            rc = lib.samd_peak_imma_s8(sms * per_sm, 4096, scratch.data_ptr(), ctypes.byref(ms), ctypes.byref(macs))
            if rc == 0 and ms.value > 0:
                tops = 2 * macs.value / (ms.value * 1e-3) / 1e12
                best = tops if best is None else max(best, tops)
        res["mma_sync_s8_tops"] = best
        # the binary MMA (m16n8k256 b1, AND + popcount): the bit-plane form of
        # a 1-2-bit convolution takes b^2 of its products per multiply-add
        lib.samd_peak_bmma_b1.argtypes = lib.samd_peak_imma_s8.argtypes
        lib.samd_peak_bmma_b1.restype = ctypes.c_int
        bbest = None
        for per_sm in (2, 4, 8):
            ms, ops = ctypes.c_float(0), ctypes.c_double(0)
            rc = lib.samd_peak_bmma_b1(sms * per_sm, 4096, scratch.data_ptr(), ctypes.byref(ms), ctypes.byref(ops))
            if rc == 0 and ms.value > 0:
                r = ops.value / (ms.value * 1e-3)
                bbest = r if bbest is None else max(bbest, r)
        res["mma_sync_b1_products_per_s"] = bbest
        if bbest:
            res["bitplane_mac_s"] = {"b1": bbest, "b2": bbest / 4}
    except Exception as e:  # noqa: BLE001
        res["mma_sync_s8_tops"] = None
        res["mma_sync_error"] = f"{type(e).__name__}: {e}"
    vals = [v for v in (res.get("int_mm_tops"), res.get("mma_sync_s8_tops")) if v]
    res["tops"] = max(vals) if vals else None
    res["how"] = ("best of torch._int_mm int8 8192^3 (best of 5) and a hand-written mma.sync m16n8k32 s8 loop on "
                  "register operands (2, 4, 8 blocks of 256 threads per SM, 4096 x 8 MMAs per warp); "
                  "mma_sync_b1_products_per_s: the same loop on mma.sync m16n8k256 b1 AND+popc; bitplane_mac_s: "
                  "the multiply-add rate of a bit-plane convolution built on it (b^2 binary products per b-bit MAC)")
    return res


def measure_e4m3_peak(dev):
    """Dense e4m3 tensor-core rate: torch._scaled_mm (cuBLASLt) on 8192^3 with
    unit scales and fp32... bf16 output, best of 5 -- the peak of the
    convolution's e4m3 layers."""
    import torch

    try:
        n = 8192
        a = torch.randn(n, n, device=dev).to(torch.float8_e4m3fn)
        b = torch.randn(n, n, device=dev).to(torch.float8_e4m3fn).t()
        one = torch.ones((), device=dev)
        t = _best_time(lambda: torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16))
        return {"tflops": 2 * n ** 3 / t / 1e12,
                "how": "torch._scaled_mm e4m3 x e4m3 -> bf16, 8192^3, unit scales, best of 5"}
    except Exception as e:  # noqa: BLE001
        return {"tflops": None, "how": f"torch._scaled_mm unavailable: {type(e).__name__}: {e}"}


def measure_e2e(built, step_macs, args, dev, ws, d, chain=False):
    import torch

    # a chained network copies in the first layer's input and copies out the
    # last layer's output; independent layers copy each layer's own
    ends = [built[0]] if chain else built
    host_in = [torch.empty(b["act"].shape, dtype=b["act"].dtype, pin_memory=True) for b in ends]
    last = built[-1]["pooled"] if (chain and built[-1]["pooled"] is not None) else built[-1]["out"]
    host_out = ([torch.empty(last.shape, dtype=last.dtype, pin_memory=True)] if chain else
                [torch.empty(b["out"].shape, dtype=b["out"].dtype, pin_memory=True) for b in built])
    for h, b in zip(host_in, ends):
        h.copy_(b["act"])
    dev_in = [b["act"] for b in ends] if chain else [torch.empty_like(b["act"]) for b in built]
    h2d = sum(t.numel() * t.element_size() for t in host_in)
    d2h = sum(t.numel() * t.element_size() for t in host_out)
    # each layer's copy in, convolution and copy out run in order on one of
    # the streams; the independent layers overlap across streams
    streams = [torch.cuda.Stream(device=dev) for _ in range(max(1, args.streams))]
    tpc = args.tiles_per_cta or (8 if args.workload == "sweep" else 4)

    from paper_1809_10572_gb300 import samd
    samd.samd_conv2d_set_min_tiles_per_cta(tpc)

    def calls(main):
        if chain:
            with torch.cuda.stream(main):
                dev_in[0].copy_(host_in[0], non_blocking=True)
                run_chain(built, main)
                host_out[0].copy_(last, non_blocking=True)
            return
        for st in streams:
            st.wait_stream(main)
        for i, (b, hi, di, ho) in enumerate(zip(built, host_in, dev_in, host_out)):
            st = streams[i % len(streams)]
            with torch.cuda.stream(st):
                di.copy_(hi, non_blocking=True)
                b["conv"](di, None, b["out"], b["shift"], stream=st)
                ho.copy_(b["out"], non_blocking=True)
        for st in streams:
            main.wait_stream(st)

    main_stream = torch.cuda.Stream(device=dev)

    def step_eager():
        with torch.cuda.stream(main_stream):
            calls(main_stream)
        main_stream.synchronize()

    # The same calls captured once into a CUDA graph (the copies from and to
    # pinned host memory are graph nodes and run on every replay): what a
    # serving loop does to keep the host's per-call cost off the step.
    step_eager()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=main_stream):
        calls(torch.cuda.current_stream())
    torch.cuda.synchronize()

    def step_graph():
        graph.replay()
        torch.cuda.current_stream().synchronize()

    def timed(step):
        for _ in range(max(1, args.warmup)):
            step()
        d.barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            step()
        return d.max(time.perf_counter() - t0)

    el = timed(step_graph)
    el_eager = timed(step_eager)
    if samd.samd_device_status() != 0:
        raise RuntimeError("a kernel recorded a timeout")
    how = ("one CUDA graph per step: pinned H2D of the network's packed input, the chained layers and pools, "
           "pinned D2H of the last packed output; host replays and waits each step" if chain else
           "one CUDA graph per step: per layer, on one of the step's streams, pinned H2D of its packed input, "
           "samd_conv2d_prepared, pinned D2H of its packed output; host replays and waits each step")
    return {"value": step_macs * args.steps * ws / el, "unit": "MAC/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "how": how,
            "eager_value": step_macs * args.steps * ws / el_eager,
            "eager_how": "the same calls issued from Python every step (no graph): host-bound"}


def main():
    args = parse_args()
    if args.connections:  # read by the CUDA runtime when it creates the context, so set before any CUDA call
        os.environ["CUDA_DEVICE_MAX_CONNECTIONS"] = str(args.connections)
    from paper_1809_10572_gb300 import workloads

    if args.profile_ops:
        return profile_ops()
    if args.profile_fused_pool:
        return profile_fused_pool()
    layers = workloads.WORKLOADS[args.workload]()
    if args.layers:
        idx = [int(t) for t in args.layers.split(",")]
        layers = [layers[i] for i in idx]
    if args.impl == "reference":
        return run_reference(args, layers)
    return run_samd(args, layers)


if __name__ == "__main__":
    sys.exit(main())
