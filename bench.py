#!/usr/bin/env python
"""Training-throughput benchmark of the parareal network on GB300.

Workload (default): parareal pre-activation ResNet-1001 torn into N=8 fine
subnetworks, batch 256, 3x64x64 synthetic N(0,1) images (stride-2 stem),
200 classes, bf16 -- the headline configuration.  A step is one whole
training iteration (Algorithm 1 forward, Algorithm 2 backward, SGD update).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config I]
                  [--paper-net resnet_nN|vgg16_4]

Prints one JSON line (rank 0).  For N > 1 (launched by torchrun) every rank
trains an independent replica on its own batch (the path is single-GPU by
design): value = images of all ranks / max over ranks of the timed region.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workloads as W  # noqa: E402

METRIC = "parareal-net training images/sec on 1 GB300; conv TFLOP/s as % of bf16 dense peak"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# CUDA-core fp32 peak: 152 SMs x 128 FP32 lanes x 2 FLOP (FMA) x 2.07 GHz max SM clock
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12
CONV_KINDS = ("conv_fwd", "conv_dgrad", "conv_wgrad", "conv_fwd_tc", "conv_dgrad_tc", "conv_wgrad_tc")


PAPER_NETS = {f"resnet_n{n}": (lambda n=n: W.paper_parareal_resnet(n)) for n in (1, 3, 6, 12, 18, 24)}
PAPER_NETS["vgg16_4"] = lambda: W.parareal_vgg16(coarse="paper")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-batch", type=int, default=1,
                    help="images per step of the reference arm (the CPU oracle)")
    ap.add_argument("--cpu-baseline-batch", type=int, default=12,
                    help="images of the cpu_baseline sample (about 15 s of oracle work on 16 cores)")
    ap.add_argument("--stream-fp32", type=int, default=None, choices=[0, 1],
                    help="keep the residual stream and correction tensors in fp32 (1) or bf16 (0); default: "
                         "the workload's (bf16 for the bf16 workloads)")
    ap.add_argument("--paper-net", default=None, choices=sorted(PAPER_NETS),
                    help="time one of the paper's own constructions instead of --config: Parareal "
                         "ResNet-N of Section 4.2 (batch 128, 3x32x32, 100 classes, the workload of "
                         "Table grad) or Parareal VGG-16-4 with the two-conv coarse blocks of Section 4.1")
    ap.add_argument("--tearing", default="none", choices=["none", "uniform", "flops", "bytes", "time"],
                    help="ResNet-1001 workloads: cut the body into subnetworks of equal RU count (uniform, "
                         "Section 4.2) or of equal cost (the remark after Table grad): algorithmic FLOPs, "
                         "HBM bytes, or the device time of each layer measured on the untorn network; "
                         "every choice but none also reports each subnetwork's measured time")
    ap.add_argument("--overlap", type=int, default=0,
                    help="run the last subnetwork's backward beside the coarse chain's (Algorithm 2 needs only "
                         "D_N for it), leaving this many SMs to the chain; 0 = phases in sequence")
    ap.add_argument("--inference", action="store_true",
                    help="time the eval-mode forward (pnn_infer) of the workload instead of training")
    ap.add_argument("--lr", type=float, default=None,
                    help="SGD learning rate (default: Section 4's 0.1; 0.01 for the VGG-16 workloads, whose "
                         "4096-wide FC head diverges within a few steps at 0.1 on a fixed synthetic batch; "
                         "the step's work does not depend on it)")
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's batch (profiling a small case of the same network)")
    ap.add_argument("--layer", default=None, choices=sorted(LAYERS),
                    help="time one grouped convolution launch of the ResNet-1001 N=8 workload (pnn_conv_run) "
                         "instead of the training step: a bottleneck conv (reduce = 1x1 out->mid, conv3x3 = "
                         "mid->mid, expand = 1x1 mid->out with the residual add) and a mode (fwd, dgrad, "
                         "wgrad), one instance per subnetwork at the stage its middle block sits in")
    ap.add_argument("--layer-impl", default="auto", choices=["auto", "tma", "gathered", "tma_tap"])
    return ap.parse_args()


# grouped-launch microbenchmark: the same layer of the 8 subnetworks of the
# 64x64 ResNet-1001 N=8 workload (batch 256; after the stride-2 stem the
# stages run at 32x32 / 16x16 / 8x8 with widths 64 / 128 / 256 and bottleneck
# widths 16 / 32 / 64); at the middle block of each subnetwork (uniform
# tearing [42 x 7, 39] of 333 bottlenecks, 111 per stage) the stages are
# [1, 1, 1, 2, 2, 3, 3, 3]
LAYER_STAGES = [1, 1, 1, 2, 2, 3, 3, 3]
STAGE_GEOM = {1: (32, 64, 16), 2: (16, 128, 32), 3: (8, 256, 64)}  # (hw, out, mid)
LAYERS = {f"{conv}_{mode}": (conv, mode) for conv in ("reduce", "conv3x3", "expand")
          for mode in ("fwd", "dgrad", "wgrad")}


def layer_instances(name, batch, stream_dt):
    """The instance list (host arrays and geometry) of a grouped layer launch."""
    conv, mode = LAYERS[name]
    rng = np.random.default_rng(7)
    out = []
    for st in LAYER_STAGES:
        hw, wide, mid = STAGE_GEOM[st]
        c, k, ks = {"reduce": (wide, mid, 1), "conv3x3": (mid, mid, 3), "expand": (mid, wide, 1)}[conv]
        out.append(dict(batch=batch, h=hw, w=hw, c=c, k=k, ksize=ks, stride=1, relu=1,
                        # the conv input: the stored BN input (the residual stream for reduce)
                        x_dt=stream_dt if conv == "reduce" else "bf16", mode=mode, conv=conv))
    return out


def layer_arm(args, rank):
    """Device time of one grouped conv launch of the training step, through
    pnn_conv_time (CUDA events around repeated launches of the kernel alone),
    with algorithmic bytes / FLOPs counted as the training step's profiler
    counts them (each operand read once, each result written once)."""
    import torch
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    if rank != 0:
        return
    torch.cuda.set_device(0)
    B = args.batch or 256
    sdt = "f32" if args.stream_fp32 == 1 else "bf16"
    insts = layer_instances(args.layer, B, sdt)
    conv, mode = LAYERS[args.layer]
    dev, flops, nbytes = [], 0.0, 0.0
    for g in insts:
        M = B * g["h"] * g["w"]
        xdt = torch.float32 if g["x_dt"] == "f32" else torch.bfloat16
        xb = 4 if g["x_dt"] == "f32" else 2
        d = {k: g[k] for k in ("batch", "h", "w", "c", "k", "ksize", "stride", "relu")}
        d["wt"] = (torch.randn(g["k"] * g["ksize"] ** 2 * g["c"], device="cuda") * 0.1).to(torch.bfloat16)
        d["x"] = torch.randn(M, g["c"], device="cuda").to(xdt)
        d["bn_scale"] = torch.rand(g["c"], device="cuda") + 0.5
        d["bn_shift"] = torch.randn(g["c"], device="cuda") * 0.1
        w_bytes = g["k"] * g["ksize"] ** 2 * g["c"] * 2
        macs = M * g["k"] * g["c"] * g["ksize"] ** 2
        flops += 2.0 * macs
        if mode == "fwd":
            ydt = torch.float32 if (conv == "expand" and sdt == "f32") else torch.bfloat16
            d["y"] = torch.empty(M, g["k"], device="cuda", dtype=ydt)
            d["y_mean"] = torch.empty(g["k"], device="cuda")
            d["y_rstd"] = torch.empty(g["k"], device="cuda")
            nbytes += M * g["c"] * xb + w_bytes + M * g["k"] * d["y"].element_size()
            if conv == "expand":
                d["res"] = torch.randn(M, g["k"], device="cuda").to(ydt)
                nbytes += M * g["k"] * d["res"].element_size()
        elif mode == "dgrad":
            d["dy"] = torch.randn(M, g["k"], device="cuda")
            d["dx"] = torch.empty(M, g["c"], device="cuda")
            nbytes += M * g["k"] * 4 + w_bytes + M * g["c"] * 4
            # every input here is a BN+ReLU value: its backward sums ride along
            d["bn_mean"] = torch.zeros(g["c"], device="cuda")
            d["bn_rstd"] = torch.ones(g["c"], device="cuda")
            d["dgamma"] = torch.empty(g["c"], device="cuda")
            d["dbeta"] = torch.empty(g["c"], device="cuda")
            nbytes += M * g["c"] * xb
        else:
            d["dy"] = torch.randn(M, g["k"], device="cuda")
            d["dw"] = torch.empty(g["k"] * g["ksize"] ** 2 * g["c"], device="cuda")
            nbytes += M * g["c"] * xb + M * g["k"] * 4 + g["k"] * g["ksize"] ** 2 * g["c"] * 4
        dev.append(d)
    pnn.conv_run({"fwd": "forward", "dgrad": "dgrad", "wgrad": "wgrad"}[mode], dev, impl=args.layer_impl)
    ms = pnn.conv_run({"fwd": "forward", "dgrad": "dgrad", "wgrad": "wgrad"}[mode], dev, impl=args.layer_impl,
                      repeat=max(1, args.steps))
    pk, src = peaks()
    gbs = nbytes / (ms / 1e3) / 1e9
    print(json.dumps({
        "metric": "grouped conv launch, algorithmic GB/s", "layer": args.layer, "impl": args.layer_impl,
        "value": gbs, "unit": "GB/s", "ms_per_launch": ms, "tflops": flops / (ms / 1e3) / 1e12,
        "frac_of_hbm": gbs / pk["hbm_gbs"], "frac_of_bf16_peak": flops / (ms / 1e3) / 1e12 / pk["bf16_tflops"],
        "peak_source": src, "instances": [(g["c"], g["k"], g["ksize"], g["h"]) for g in insts], "batch": B,
        "algorithmic_bytes": nbytes, "flops": flops, "residual_stream": sdt,
        "l2": "operands larger than L2" if nbytes > 129e6 else "operands within L2"}), flush=True)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return PEAKS_FALLBACK, "fallback"


# ---------------------------------------------------------------- clocks
class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.p = None

    def __enter__(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        return self

    def __exit__(self, *a):
        if self.p:
            self.p.terminate()
            self.p.wait(timeout=10)

    def summary(self):
        self.f.flush()
        rows = []
        with open(self.f.name) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.f.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------- distributed
def dist_setup(gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    return rank, local, world, dist


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(dist, v):
    if dist is None:
        return v
    import torch
    t = torch.tensor([v], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t[0])


# ---------------------------------------------------------------- CPU oracle
def oracle_sample(desc, batch):
    """One oracle training step on `batch` images of the same network."""
    from oracle import pnn_oracle as O
    d = W.with_batch(desc, batch)
    net = O.ParaNet(d)
    theta = W.init_params(net.spec, seed=0, bf16=d["precision"] == "bf16")
    x, labels = W.make_batch(d)
    prec = "bf16" if d["precision"] == "bf16" else "fp64"
    t0 = time.perf_counter()
    O.train_step(d, theta, x, labels, precision=prec)
    return time.perf_counter() - t0


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def config_of(args, desc, world=1, extra=None):
    """The `config` object of both arms' JSON lines."""
    B = desc["batch"]
    c = {"workload": desc["name"] + "_b%d_%dpx_c%d" % (B, desc["in_h"], desc["classes"]),
         "batch": B, "input": "3x%dx%d" % (desc["in_h"], desc["in_w"]), "classes": desc["classes"],
         "subnetworks": len(desc["segments"]), "correction": desc.get("correction", "residual"),
         "residual_stream": desc.get("residual_stream", "fp32"), "lr": args.lr,
         "tearing": "uniform" if args.tearing == "none" else args.tearing,
         "overlap_sms": args.overlap,
         "parallelism": "replicas" if world > 1 else "single-gpu"}
    c.update(extra or {})
    return c


def reference_arm(args, desc, rank):
    if rank != 0:
        return
    b = args.cpu_sample_batch
    for _ in range(args.warmup):
        oracle_sample(desc, b)
    ts = [oracle_sample(desc, b) for _ in range(args.steps)]
    total = sum(ts)
    value = b * args.steps / total
    sample = f"{b} image(s) of the same network per step (CPU fp64 oracle, one forward+backward+SGD)"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(args, desc, args.gpus),
        "cpu_baseline": {"value": value, "unit": "images/s", "cores": cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ---------------------------------------------------------------- our arm
def layer_times(desc, stream, steps=2):
    """Device ms of each body layer's forward and backward launches in the
    untorn network (the body as one segment), from an eager profiled step."""
    import copy
    import torch
    from paper_2103_08802_gb300 import pnn
    d1 = copy.deepcopy(desc)
    d1["segments"] = [len(desc["body"])]
    d1["coarse"] = []
    net = pnn.ParaNet(d1, seed=0, stream=stream)
    x, labels = W.make_batch(d1, seed=7)
    xd, ld = torch.from_numpy(x).cuda(), torch.from_numpy(labels).cuda()
    theta0 = net.get_params()
    for _ in range(2):
        net.train_step(xd, ld)
    t = [0.0] * len(desc["body"])
    for _ in range(steps):
        net.set_params(theta0)
        net.profile(True)
        net.forward(xd, ld)
        net.backward()
        for r in net.profile_trace():
            if r["phase"] in (1, 7) and r["block"] >= 0:
                t[r["block"]] += r["ms"] / steps
        net.profile(False)
    net.close()
    del net
    torch.cuda.empty_cache()
    return t


def retear(args, desc, stream):
    """The workload torn as --tearing asks, and a record of the cut: layers per
    segment, each segment's summed layer time measured on the untorn network,
    and the largest of them (the parallel phase's virtual wall-clock of
    Table grad if every subnetwork had a GPU of its own)."""
    from paper_2103_08802_gb300 import pnn
    t = layer_times(desc, stream)
    n = len(desc["segments"])
    if args.tearing == "uniform":
        seg = list(desc["segments"])
    else:
        cost = t if args.tearing == "time" else pnn.block_costs(desc, args.tearing)
        seg = pnn.partition(cost, n)
        desc = W.config(args.config, batch=args.batch, segments=seg)
    b = np.cumsum([0] + seg)
    seg_ms = [float(sum(t[b[j]:b[j + 1]])) for j in range(n)]
    rec = {"kind": args.tearing, "segments": seg, "segment_fine_ms": seg_ms,
           "virtual_fine_ms": max(seg_ms), "mean_segment_ms": float(np.mean(seg_ms)),
           "layer_ms_total": float(sum(t))}
    return desc, rec


KERNEL_SYMBOL = {("conv_fwd_tc", 0): "k_conv_fwd_tc", ("conv_fwd_tc", 1): "k_conv_fwd_tma",
                 ("conv_fwd_tc", 2): "k_conv_fwd_tma_w", ("conv_dgrad_tc", 0): "k_conv_dgrad_tc",
                 ("conv_dgrad_tc", 1): "k_conv_dgrad_tma", ("conv_dgrad_tc", 2): "k_conv_dgrad_tma_w",
                 ("conv_fwd_tc", 3): "k_conv_fwd_tma_h", ("conv_dgrad_tc", 3): "k_conv_dgrad_tma_h",
                 ("conv_wgrad_tc", 0): "k_conv_wgrad_tc", ("conv_wgrad_tc", 1): "k_conv_wgrad_tma",
                 ("bn_bwd_apply", 1): "k_bnb_apply8", ("bn_finalize", 0): "k_bn_fin"}


def dram_traffic(symbol):
    """The ncu record of `symbol` in profiles/dram_traffic.json, if it was taken
    on the kernel source as it stands (the file names the sha256 of the
    source file the kernel is built from); else None."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as f:
            rec = json.load(f).get(symbol)
    except (OSError, ValueError):
        return None
    if not rec:
        return None
    src = os.path.join(ROOT, "paper_2103_08802_gb300", "csrc", rec["source"])
    try:
        with open(src, "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != rec["source_sha256"]:
                return None
    except OSError:
        return None
    return rec


def launch_groups(trace, steps, n=14):
    """The n launch groups (kind, variant, first-instance shape, instances)
    with the most device time per step, with their algorithmic GB/s against
    the measured HBM peak."""
    pk, _ = peaks()
    groups = {}
    for r in trace or []:
        k = (r["kind"], r["variant"], r["shape"], r["instances"])
        g = groups.setdefault(k, [0.0, 0, 0.0])
        g[0] += r["ms"]; g[1] += 1; g[2] += r["bytes"]
    out = []
    for (kind, variant, shape, inst), (ms, cnt, by) in sorted(groups.items(), key=lambda kv: -kv[1][0])[:n]:
        gbs = by / (ms / 1e3) / 1e9 if ms else 0.0
        out.append({"kernel": KERNEL_SYMBOL.get((kind, variant), kind), "shape": list(shape), "instances": inst,
                    "launches_per_step": cnt / steps, "ms_per_step": ms / steps, "us_per_launch": 1e3 * ms / cnt,
                    "gbs": gbs, "frac_of_hbm": gbs / pk["hbm_gbs"]})
    return out


def roofline_of(prof, steps, trace=None):
    """Roofline record of the dominant kernel: the launch group (kind,
    variant, first-instance shape, instances) with the largest device time in
    a profiled window of `steps` steps, from the per-launch trace; without a
    trace, the dominant kind ({kind: (ms, launches, flops, bytes)})."""
    pk, src = peaks()
    if trace:
        groups = {}
        for r in trace:
            k = (r["kind"], r["variant"], r["shape"], r["instances"])
            g = groups.setdefault(k, [0.0, 0, 0.0, 0.0])
            g[0] += r["ms"]; g[1] += 1; g[2] += r["flops"]; g[3] += r["bytes"]
        # (a group with no algorithmic bytes or FLOPs -- the per-channel BN
        # finalisation, the head -- has no roof to be measured against)
        cand = {k: g for k, g in groups.items() if g[2] > 0 or g[3] > 0} or groups
        (kind, variant, shape, inst), (kms, kn, kfl, kby) = max(cand.items(), key=lambda kv: kv[1][0])
        name = KERNEL_SYMBOL.get((kind, variant), kind)
        what = {"kind": kind, "variant": variant, "first_instance_shape": list(shape), "instances": inst}
    else:
        cand = {k: v for k, v in prof.items() if v[2] > 0 or v[3] > 0} or prof
        name, (kms, kn, kfl, kby) = max(cand.items(), key=lambda kv: kv[1][0])
        kind, what = name, {"kind": name}
    per_launch_ms = kms / kn
    # the bound follows the kernel's algorithmic intensity: below the ridge point
    # (peak FLOP/s / peak B/s) the roof is HBM bandwidth
    ridge = pk["bf16_tflops_sustained"] * 1e12 / (pk["hbm_gbs"] * 1e9)
    intensity = kfl / kby if kby else float("inf")
    tflops = kfl / kn / (per_launch_ms / 1e3) / 1e12
    if kind.startswith("conv") and not kind.endswith("_tc") and intensity >= FP32_ALU_TFLOPS * 1e3 / pk["hbm_gbs"]:
        bound, peak, unit, achieved = "alu", FP32_ALU_TFLOPS, "TFLOP/s", tflops
    elif kind.endswith("_tc") and intensity >= ridge:
        bound, peak, unit, achieved = "tensor", pk["bf16_tflops_sustained"], "TFLOP/s", tflops
    else:
        bound, peak, unit = "hbm", pk["hbm_gbs"], "GB/s"
        achieved = kby / kn / (per_launch_ms / 1e3) / 1e9
    out = {"kernel": name, **what, "bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
           "frac": achieved / peak, "traffic": None, "intensity_flop_per_byte": intensity,
           "peak_source": (src + (" (hbm_gbs)" if bound == "hbm" else " (bf16_tflops_sustained)"))
           if bound != "alu" else "derived: 152 SM x 128 FP32 lanes x 2 x 2.07 GHz",
           "launches_per_step": kn / steps, "ms_per_launch": per_launch_ms,
           "algorithmic_bytes_per_launch": kby / kn, "flops_per_launch": kfl / kn}
    if kind.endswith("_tc"):
        # the contraction against the dense bf16 tensor peak as well
        out["tensor_tflops"] = tflops
        out["tensor_frac_of_bf16_sustained"] = tflops / pk["bf16_tflops_sustained"]
    rec = dram_traffic(name)
    if rec:
        # DRAM bytes / algorithmic bytes of the same grouped launch measured
        # alone (bench.py --layer), scaled to this group's algorithmic bytes
        ratio = rec["dram_bytes"] / rec["algorithmic_bytes"]
        out["traffic"] = ratio * kby / kn
        out["traffic_over_algorithmic"] = ratio
        out["traffic_source"] = rec["command"]
    return out


def infer_arm(args, desc, rank, local, world, dist):
    """Eval-mode forward throughput (pnn_infer, one CUDA graph per pass) of the
    same network: parameters and running statistics of a fresh net (the work
    does not depend on their values)."""
    import torch
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    torch.cuda.set_device(local)
    stream = torch.cuda.Stream()
    net = pnn.ParaNet(desc, seed=0, stream=stream, inference=True)
    B = desc["batch"]
    x, labels = W.make_batch(desc, seed=2000 + rank)
    xd = torch.from_numpy(x).cuda()
    logits = torch.empty(B * desc["classes"], dtype=torch.float32, device="cuda")
    for _ in range(max(3, args.warmup)):
        net.infer(xd, logits)
    net.sync()
    with Clocks(local) as clk:
        barrier(dist)
        torch.cuda.synchronize()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for _ in range(args.steps):
            net.infer(xd, logits)
        end.record(stream)
        torch.cuda.synchronize()
        ms = start.elapsed_time(end)
        barrier(dist)
    ms = max_over_ranks(dist, ms)
    clocks = clk.summary()
    net.sync()
    value = B * args.steps * world / (ms / 1e3)
    net.profile(True)
    for _ in range(args.steps):
        net.infer(xd, logits)
    prof = net.profile_read()
    net.profile(False)
    # end to end: pinned host images in, host logits out, every pass
    xh = torch.from_numpy(x).pin_memory()
    lh = torch.empty(B * desc["classes"], dtype=torch.float32).pin_memory()
    net.infer(xd, logits)
    net.sync()
    barrier(dist)
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            xd.copy_(xh, non_blocking=True)
            net.infer(xd, logits)
            lh.copy_(logits, non_blocking=True)
            stream.synchronize()
    e2e_s = max_over_ranks(dist, time.perf_counter() - t0)
    if rank != 0:
        return
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        from oracle import pnn_oracle as O
        d1 = W.with_batch(desc, args.cpu_baseline_batch)
        onet = O.ParaNet(d1, precision="bf16" if d1["precision"] == "bf16" else "fp64")
        theta = W.init_params(onet.spec, seed=0, bf16=d1["precision"] == "bf16")
        x1, _ = W.make_batch(d1)
        t = time.perf_counter()
        onet.infer(theta, x1, O.RunningStats(onet.spec))
        t = time.perf_counter() - t
        cpu = {"value": d1["batch"] / t, "unit": "images/s", "cores": cores(), "kind": "oracle",
               "sample": f"{d1['batch']} image(s) of the same network, one eval-mode forward of the CPU fp64 "
                         f"oracle ({t:.1f} s)"}
    out = {
        "metric": "parareal-net eval-mode forward images/sec on 1 GB300", "value": value, "unit": "images/s",
        "n_gpus": world, "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if desc["precision"] == "bf16" else "fp32", "data": "synthetic",
        "config": {"workload": desc["name"] + "_b%d_%dpx_c%d_inference" % (B, desc["in_h"], desc["classes"]),
                   "batch": B, "input": "3x%dx%d" % (desc["in_h"], desc["in_w"]), "classes": desc["classes"],
                   "subnetworks": len(desc["segments"]), "correction": desc.get("correction", "residual"),
                   "workspace_gb": net.workspace_bytes / 1e9,
                   "l2": "inputs larger than L2" if net.workspace_bytes > 129e6 else "workspace within L2",
                   "parallelism": "replicas" if world > 1 else "single-gpu"},
        "roofline": roofline_of(prof, args.steps),
        "kernels": {k: {"ms_per_step": v[0] / args.steps, "launches_per_step": v[1] / args.steps,
                        "gflop_per_step": v[2] / args.steps / 1e9, "gb_per_step": v[3] / args.steps / 1e9}
                    for k, v in sorted(prof.items(), key=lambda kv: -kv[1][0])},
        "cpu_baseline": cpu,
        "e2e": {"value": B * args.steps * world / e2e_s, "unit": "images/s",
                "h2d_bytes_per_step": int(x.nbytes), "d2h_bytes_per_step": int(B * desc["classes"] * 4)},
        "gpu_launches": sum(v[1] for v in prof.values()),
        "clocks": clocks,
    }
    print(json.dumps(out), flush=True)


def our_arm(args, desc, rank, local, world, dist):
    import torch
    from paper_2103_08802_gb300 import build, pnn

    build.build()
    torch.cuda.set_device(local)
    stream = torch.cuda.Stream()
    tearing = None
    if args.tearing != "none":
        if args.paper_net or args.config not in (2, 3, 4):
            raise SystemExit("--tearing applies to the ResNet-1001 configurations 2, 3 and 4")
        desc, tearing = retear(args, desc, stream)
    net = pnn.ParaNet(desc, seed=0, stream=stream, lr=args.lr,
                      overlap=args.overlap)
    B = desc["batch"]
    x, labels = W.make_batch(desc, seed=1000 + desc.get("config_index", 0) + rank)
    xd = torch.from_numpy(x).cuda()
    ld = torch.from_numpy(labels).cuda()
    loss = torch.zeros(1, device="cuda")
    # every measured section below starts again from the initial weights: a
    # fixed synthetic batch trained for dozens of steps at Section 4's lr can
    # diverge, and the step's work does not depend on the weights' values
    theta0 = net.get_params()
    torch.cuda.synchronize()

    for _ in range(max(3, args.warmup)):
        net.train_step(xd, ld, loss)
    net.sync()

    # ------------------------------------------------ timed region (device events)
    with Clocks(local) as clk:
        barrier(dist)
        torch.cuda.synchronize()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for _ in range(args.steps):
            net.train_step(xd, ld, loss)
        end.record(stream)
        torch.cuda.synchronize()
        ms = start.elapsed_time(end)
        barrier(dist)
    ms = max_over_ranks(dist, ms)
    clocks = clk.summary()
    net.sync()
    final_loss = float(loss.cpu())
    value = B * args.steps * world / (ms / 1e3)

    # ------------------------------------------------ per-kernel profile (eager steps)
    net.set_params(theta0)
    net.profile(True)
    for _ in range(args.steps):
        net.forward(xd, ld, loss)
        net.backward()
        net.sgd_step()
    prof = net.profile_read()
    trace = net.profile_trace()
    net.profile(False)
    fw, bw, up = net.launch_counts()
    launches_per_step = fw + bw + up
    phases_eager = net.timings()
    net.set_params(theta0)
    # the overlapped backward runs two phases at once: no per-phase split
    phases = net.time_phases(xd, ld, args.steps) if not args.overlap else None

    # ------------------------------------------------ end to end through the host API
    net.set_params(theta0)
    xh = torch.from_numpy(x).pin_memory()
    lh = torch.from_numpy(labels).pin_memory()
    net.train_step_host(xh, lh)  # captures the host-staged step graph
    barrier(dist)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        net.train_step_host(xh, lh)
    e2e_s = max_over_ranks(dist, time.perf_counter() - t0)
    e2e = {"value": B * args.steps * world / e2e_s, "unit": "images/s",
           "h2d_bytes_per_step": int(x.nbytes + labels.nbytes), "d2h_bytes_per_step": 4}

    if rank != 0:
        return
    pk, src = peaks()
    conv_ms = sum(prof[k][0] for k in CONV_KINDS if k in prof)
    conv_flops = sum(prof[k][2] for k in CONV_KINDS if k in prof)
    total_prof_ms = sum(v[0] for v in prof.values())
    roofline = roofline_of(prof, args.steps, trace)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        b = args.cpu_baseline_batch
        t = oracle_sample(desc, b)
        cpu = {"value": b / t, "unit": "images/s", "cores": cores(), "kind": "oracle",
               "sample": f"{b} image(s) of the same network, one forward+backward+SGD step of the CPU "
                         f"fp64 oracle ({t:.1f} s)"}
    out = {
        "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": world, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if desc["precision"] == "bf16" else "fp32",
        "data": "synthetic",
        "config": config_of(args, desc, world, {
            "l2": "inputs larger than L2 (%.1f GB workspace per step)" % (net.workspace_bytes / 1e9)}),
        "conv_tflops": conv_flops / (conv_ms / 1e3) / 1e12 if conv_ms else None,
        "conv_frac_of_bf16_peak": (conv_flops / (conv_ms / 1e3) / 1e12) / pk["bf16_tflops_sustained"] if conv_ms else None,
        "conv_share_of_device_time": conv_ms / total_prof_ms if total_prof_ms else None,
        "roofline": roofline,
        "launch_groups": launch_groups(trace, args.steps),
        "kernels": {k: {"ms_per_step": v[0] / args.steps, "launches_per_step": v[1] / args.steps,
                        "gflop_per_step": v[2] / args.steps / 1e9, "gb_per_step": v[3] / args.steps / 1e9}
                    for k, v in sorted(prof.items(), key=lambda kv: -kv[1][0])},
        "tearing": tearing,
        "phases_ms": phases,
        "phases_ms_eager": phases_eager,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
        "loss_after": final_loss,
    }
    print(json.dumps(out), flush=True)


def main():
    args = parse()
    rank, local, world, dist = dist_setup(args.gpus)
    if args.paper_net:
        desc = PAPER_NETS[args.paper_net]()
        if args.batch:
            desc["batch"] = args.batch
    else:
        desc = W.config(args.config, batch=args.batch)
    if args.lr is None:
        args.lr = 0.01 if desc["head"]["kind"] == "gap_mlp" else 0.1
    if args.stream_fp32 is not None and desc["precision"] == "bf16":
        desc["residual_stream"] = "fp32" if args.stream_fp32 else "bf16"
    if args.impl == "reference":
        reference_arm(args, desc, rank)
    elif args.layer:
        layer_arm(args, rank)
    elif args.inference:
        infer_arm(args, desc, rank, local, world, dist)
    else:
        our_arm(args, desc, rank, local, world, dist)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
