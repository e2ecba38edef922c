#!/usr/bin/env python3
"""Throughput of the multipoint-quantization hot path on GB300.

One step = every layer of the workload through the whole path: greedy points (mpq_quantize_layer),
output error (mpq_output_error), point allocation (mpq_allocate_points, budget mode) and
multipoint weights (mpq_reconstruct).  Metric: weight-elements x scale-candidates x points per
second, i.e. sum over layers of C*d*G*k_max per step / step time.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config c2] [--impl ours|reference]

Prints ONE JSON line on rank 0.  Multi-GPU (torchrun): every rank quantizes its own copy of the
workload (independent problems, no collective on the data path; weak scaling); value = units of
all ranks / max-over-ranks time.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "weight-elements x scale-candidates x points / s"
UNIT = "elem*cand*pt/s"
PROFILES = os.path.join(ROOT, "profiles")
KERNEL_SOURCES = {
    "output_error": ("paper_2002_09049_gb300/csrc/output_error.cu",
                     "paper_2002_09049_gb300/csrc/output_error_f16.cu",
                     "paper_2002_09049_gb300/csrc/output_error_pair.cu",
                     "paper_2002_09049_gb300/csrc/pair_common.cuh",
                     "paper_2002_09049_gb300/csrc/output_error_tc.cu",
                     "paper_2002_09049_gb300/csrc/sm100.cuh",
                     "paper_2002_09049_gb300/csrc/tf32_operands.cuh",
                     "paper_2002_09049_gb300/csrc/waits.cuh"),
    "quantize": ("paper_2002_09049_gb300/csrc/quantize.cu",
                 "paper_2002_09049_gb300/csrc/rounding.cuh",
                 "paper_2002_09049_gb300/csrc/sm100.cuh"),
    "allocate": "paper_2002_09049_gb300/csrc/allocate.cu",
    "reconstruct": "paper_2002_09049_gb300/csrc/reconstruct.cu",
    "center": "paper_2002_09049_gb300/csrc/center.cu",
}


CENTER_MODES = {"none": -1, "channel": 0, "layer": 1}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default="c5", choices=["c1", "c2", "c3", "c4", "c5"],
                    help="workload; c5 (the two large linear layers) is the largest")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--graph", type=int, default=1,
                    help="replay the multi-stream step as a captured CUDA graph (1) or launch it (0)")
    ap.add_argument("--streams", type=int, default=12,
                    help="CUDA streams the independent layers are spread over")
    ap.add_argument("--batch-alloc", type=int, default=1,
                    help="allocate every layer's points in one launch (1) or one launch per layer")
    ap.add_argument("--layers", default=None,
                    help="comma-separated layer indices to run (profiling a subset); default all")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--op", default="quantize", choices=["quantize", "clip", "infer", "adaptive"],
                    help="quantize: the multipoint path (Algorithm 1, Eq. 11, Algorithm 2, Eq. 4); "
                         "clip: the output-error-driven clipping factor search (Eq. 12); "
                         "infer: integer inference with the packed multipoint weights (Eq. 13)")
    ap.add_argument("--coef-bits", type=int, default=16, help="p of Eq. 13 for --op infer")
    ap.add_argument("--clip-candidates", type=int, default=20,
                    help="clipping factor candidates (c+1)/n x max|w| for --op clip")
    ap.add_argument("--center", default="none", choices=list(CENTER_MODES),
                    help="asymmetric sets (Eq. 1, B != 0) for --op quantize / infer: one centre per "
                         "channel or per layer, the points approximating the centred weights")
    return ap.parse_args()


# ------------------------------------------------------------------------------------------------
def dist_setup(args):
    from paper_2002_09049_gb300 import dist as dist_helpers
    return dist_helpers.world_from_env()


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def src_hash(rel):
    """First 16 hex digits of the sha256 of a source file (or of several, concatenated)."""
    h = hashlib.sha256()
    for r in ([rel] if isinstance(rel, str) else rel):
        with open(os.path.join(ROOT, r), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "sm_max_mhz": 2070.0}, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.15)
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------------------------
def layer_inputs(wl, li):
    from paper_2002_09049_gb300 import workloads as wlm
    return wlm.make_weights(wl, li), wlm.make_calibration(wl, li)


def kernel_units(wl, layer):
    return layer.C * layer.d * wl.G * wl.k_max


def quantize_bytes(wl, layer):
    """Algorithmic HBM bytes of one mpq_quantize_layer call: read W once, write k_max code planes,
    the scales and the residual norms."""
    return layer.C * (layer.d * (4 + wl.k_max) + 4 * wl.k_max + 4 * (wl.k_max + 1))


# Greedy search (lattice form), algorithmic lane operations.  Per element-step: |r|, u2 = 2a*G/smax
# (2), lattice-distance test (5), bucket index (3), 64-bit fixed point (6), three atomics (3) = 20;
# residual update and code emission: code (6), sign (1), fma (1), two stores (2), compensated square
# sum (4), max (1) = 15.  Per channel-step: clear, suffix scan and bucket reads of the
# 2*G*Qmax + 1 buckets (7 per bucket), fold (4 per (g, L)), fp32 screen and argmin (12 per g).
GREEDY_OPS_PER_ELEMENT_STEP = 35
ALU_LANES_PER_SM = 128   # fp32 / int32 lanes per SM (4 SMSPs x 32)


def quantize_ops(wl, layer, bits):
    qmax = (1 << (bits - 1)) - 1
    nb = 2 * wl.G * qmax + 1
    per_channel_step = 7 * nb + 4 * wl.G * qmax + 12 * wl.G
    return layer.C * wl.k_max * (GREEDY_OPS_PER_ELEMENT_STEP * layer.d + per_channel_step)


def reconstruct_bytes(wl, layer):
    """Algorithmic HBM bytes of one mpq_reconstruct call at the budget's average point count:
    n_avg code bytes + one fp32 write per weight (scales and counts are negligible)."""
    return layer.C * layer.d * (wl.beta + 4)


def contraction_flops(wl, layer):
    """Algorithmic flops of Eq. 11 for one layer: 2 * N * d * C * (k_max + 1)."""
    return 2 * wl.n_calib * layer.d * layer.C * (wl.k_max + 1)


def output_error_bytes(wl, layer):
    """Algorithmic HBM bytes of one mpq_output_error call: read X, W, the k_max code planes and the
    scales once, write the error table."""
    x = layer.C * wl.n_calib * layer.d if layer.groups > 1 else wl.n_calib * layer.d
    return 4 * x + layer.C * (layer.d * (4 + wl.k_max) + 4 * wl.k_max + 4 * (wl.k_max + 1))


def allocate_bytes(wl, layer):
    """Algorithmic HBM bytes of one mpq_allocate_points call: read the error table, write the
    point counts."""
    return 4 * layer.C * (wl.k_max + 1) + 4 * layer.C + 4


def run_ours(args, world, rank, local):
    import torch
    from paper_2002_09049_gb300 import _build, binding, pipeline, workloads as wlm
    from paper_2002_09049_gb300 import dist as dist_helpers

    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or world == 1:
        _build.build()
    if world > 1:
        torch.distributed.barrier()
    binding.load()

    wl = wlm.WORKLOADS[args.config]
    keep = None if args.layers is None else {int(x) for x in args.layers.split(",")}
    idx = [li for li in range(len(wl.layers)) if keep is None or li in keep]
    layers = [wl.layers[li] for li in idx]
    specs, Ws, Xs, Whs, Xhs = [], [], [], [], []
    for li, layer in zip(idx, layers):
        W, X = layer_inputs(wl, li)
        specs.append(pipeline.LayerSpec(C=layer.C, d=layer.d, N=wl.n_calib, groups=layer.groups,
                                        bits=wl.bits[0], G=wl.G, k_max=wl.k_max,
                                        budget_or_eps=wl.beta, center=CENTER_MODES[args.center]))
        Whs.append(torch.from_numpy(W).pin_memory())
        Xhs.append(torch.from_numpy(X).pin_memory())
        Ws.append(Whs[-1].to(dev))
        Xs.append(Xhs[-1].to(dev))
    net = pipeline.NetworkPlan(specs, dev, n_streams=args.streams,
                               batch_alloc=bool(args.batch_alloc))
    units_per_step = sum(kernel_units(wl, l) for l in layers) * len(wl.bits)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)  # 512 MB > L2
    stream = torch.cuda.current_stream()

    families = ["center", "quantize", "output_error", "allocate", "reconstruct"]

    graphs = []
    if args.graph:
        # one captured graph per bit width (the bit width is a launch argument); each bit width
        # has its own plan (output buffers), so the graphs replay concurrently on their own streams
        for n, b in enumerate(wl.bits):
            if n == 0:
                for sp in specs:
                    sp.bits = b
                plan_b = net
            else:
                plan_b = pipeline.NetworkPlan([dataclasses.replace(sp, bits=b) for sp in specs],
                                              dev, n_streams=args.streams,
                                              batch_alloc=bool(args.batch_alloc))
            graphs.append(pipeline.CapturedNetwork(plan_b, Ws, Xs))
    graph_streams = [torch.cuda.Stream(dev) for _ in graphs]

    def step():
        if len(graphs) == 1:
            graphs[0].replay()
            return
        if graphs:
            ev = torch.cuda.Event()
            ev.record(stream)
            for g, gs in zip(graphs, graph_streams):
                gs.wait_event(ev)
                with torch.cuda.stream(gs):
                    g.replay()
            for gs in graph_streams:
                e = torch.cuda.Event()
                e.record(gs)
                stream.wait_event(e)
            return
        for b in wl.bits:
            for sp in specs:
                sp.bits = b
            net.run_device(Ws, Xs, stream=stream)

    center_launches = {"none": 0, "channel": 1, "layer": 3}[args.center]
    # one kernel per call, plus the two pre-passes (ranges, X split) of every output error on the
    # CTA-pair kernel (shared calibration input, rows a multiple of 16 elements; torch buffers are
    # 16-byte aligned)
    range_launches = 2 * sum(1 for l in layers if l.groups == 1 and l.d % 16 == 0)
    alloc_launches = 1 if net.batch_alloc else len(layers)
    launches_per_step = ((3 + center_launches) * len(layers) + alloc_launches +
                         range_launches) * len(wl.bits)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    peaks, peak_src = measured_peaks()
    step_ms = []
    recs = []
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for _ in range(args.steps):
            flush.fill_(1.0)                    # evict L2 between steps (outside the timing)
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            step()
            z.record(stream)
            torch.cuda.synchronize()
            step_ms.append(a.elapsed_time(z))
    torch.cuda.synchronize()
    # Per-kernel durations for the roofline: the same steps once more with every layer on one
    # stream and CUDA events around each call, so no launch shares the GPU with another layer's.
    for _ in range(args.steps):
        flush.fill_(1.0)
        rec = []
        for b in wl.bits:
            for sp in specs:
                sp.bits = b
            evs = {}
            for i in net.order:
                evs[i] = [torch.cuda.Event(enable_timing=True) for _ in range(len(families) + 1)]
                net.plans[i].run_device(Ws[i], Xs[i], stream=stream,
                                        timing=lambda ph, e=evs[i]: e[ph].record(stream),
                                        finish=not net.batch_alloc)
            if net.batch_alloc:   # one allocation launch for every layer, then the reconstructions
                ab = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
                ab[0].record(stream)
                net.allocate_all(stream)
                ab[1].record(stream)
                for i in net.order:
                    evs[i][4].record(stream)
                    net.plans[i].run_reconstruct(stream)
                    evs[i][5].record(stream)
                evs["batch_alloc"] = ab
            rec.append(evs)
        torch.cuda.synchronize()
        recs.append(rec)
    if world > 1:
        torch.distributed.barrier()
    ms = dist_helpers.max_over_ranks(float(np.mean(step_ms)), device=dev)
    value = dist_helpers.aggregate_throughput(units_per_step, ms, world)

    # per-kernel-family device time from the events around every call (on its own stream)
    fam_ms = {f: 0.0 for f in families}
    fam_work = {f: 0.0 for f in families}     # flops (output error), lane-ops (quantize), bytes
    fam_bytes = {f: 0.0 for f in families}    # algorithmic HBM bytes of every family
    for rec in recs:
        for evs in rec:
            ab = evs.pop("batch_alloc", None)
            if ab is not None:
                fam_ms["allocate"] += ab[0].elapsed_time(ab[1])
            for i, e in evs.items():
                layer = layers[i]
                for k, f in enumerate(families):
                    if ab is not None and f == "allocate":
                        continue   # timed once for all layers above
                    fam_ms[f] += e[k].elapsed_time(e[k + 1])
                fam_work["output_error"] += contraction_flops(wl, layer)
                fam_work["quantize"] += quantize_ops(wl, layer, wl.bits[0])
                fam_work["reconstruct"] += reconstruct_bytes(wl, layer)
                fam_work["allocate"] += allocate_bytes(wl, layer)
                fam_work["center"] += 8 * layer.C * layer.d + 4 * layer.C
                fam_bytes["output_error"] += output_error_bytes(wl, layer)
                fam_bytes["quantize"] += quantize_bytes(wl, layer)
                fam_bytes["reconstruct"] += reconstruct_bytes(wl, layer)
                fam_bytes["allocate"] += allocate_bytes(wl, layer)
                fam_bytes["center"] += 8 * layer.C * layer.d + 4 * layer.C
    if args.center == "none":   # no centring call: its (empty) interval is not a kernel family
        families = [f for f in families if f != "center"]
        for t in (fam_ms, fam_work, fam_bytes):
            t.pop("center")
    total_fam = sum(fam_ms.values())
    dominant = max(fam_ms, key=fam_ms.get)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count

    roofline = dominant_roofline(dominant, fam_ms, fam_work, peaks, peak_src, wl, args,
                                 sm_count=sms)
    roofline["share"] = fam_ms[dominant] / total_fam if total_fam else None
    roofline["family_ms_per_step"] = {f: fam_ms[f] / args.steps for f in families}
    roofline["timing"] = ("CUDA events around every call in a single-stream pass of the same "
                          "steps inside bench.py (value itself is timed with layers on "
                          f"{args.streams} streams)")
    # every family against HBM (algorithmic bytes / its single-stream time), the greedy search
    # also against its ALU lane rate, the contraction against the tensor peak
    hbm = peaks["hbm_gbs"]
    fam_hbm = {}
    for f in families:
        t_s = fam_ms[f] / 1e3
        ach = fam_bytes[f] / t_s / 1e9 if t_s > 0 else None
        fam_hbm[f] = {"achieved": ach, "frac": ach / hbm if ach else None,
                      "bytes_per_step": fam_bytes[f] / args.steps,
                      "ms_per_step": fam_ms[f] / args.steps}
    roofline_greedy = greedy_roofline(fam_ms, fam_work, fam_bytes, peaks, peak_src, wl, args, sms)
    step_bytes = sum(fam_bytes.values()) / args.steps

    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": f"{args.config}: {wl.title}", "layers": len(layers),
                   "weights": sum(l.C * l.d for l in layers),
                   "channels": sum(l.C for l in layers), "bits": list(wl.bits),
                   "G": wl.G, "k_max": wl.k_max, "budget": wl.beta, "calib_rows": wl.n_calib,
                   "units_per_step": units_per_step, "l2": "flushed between steps (512 MB write)",
                   "streams": args.streams, "cuda_graph": bool(args.graph),
                   "batched_allocation": net.batch_alloc,
                   "center": args.center, "parallelism": f"replicas x{world}"},
        "roofline": roofline,
        "roofline_greedy": roofline_greedy,
        "hbm": {"achieved": step_bytes / (ms / 1e3) / 1e9, "peak": hbm, "unit": "GB/s",
                "frac": step_bytes / (ms / 1e3) / 1e9 / hbm, "bytes_per_step": step_bytes,
                "what": "algorithmic HBM bytes of the whole step (every call reads its inputs and "
                        "writes its outputs once) / ms_per_step",
                "families": fam_hbm},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk.summary(),
    }

    if not args.no_e2e:
        out["e2e"] = run_e2e(net, specs, Whs, Xhs, Ws, Xs, wl, args, stream, units_per_step)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        gpu_out = gpu_sample_outputs(net, specs, Ws, Xs, wl, stream, oracle_sample(
            wl, args.cpu_seconds))
        out["cpu_baseline"], orc_out = cpu_baseline(wl, args.cpu_seconds,
                                                    CENTER_MODES[args.center])
        out["parity"] = parity_report(wl, gpu_out, orc_out, CENTER_MODES[args.center])
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    return out if rank == 0 else None




def dominant_roofline(dominant, fam_ms, fam_work, peaks, peak_src, wl, args, sm_count=152):
    """Roofline entry of the kernel family with the largest measured time.

    output_error: tensor-pipe bound; achieved = algorithmic flops 2*N*d*C*(k_max+1) (the three
      fp16 split passes are not counted) / measured time; peak = measured bf16 dense burst peak
      (kind::f16 runs fp16 and bf16 operands at the same rate).
    quantize: ALU bound; achieved = algorithmic lane operations (quantize_ops) / time; peak = SMs x
      128 lanes x the maximum SM clock.
    reconstruct / allocate / center: HBM roofline; achieved = algorithmic bytes / time."""
    traffic = None
    tfile = os.path.join(PROFILES, "roofline_traffic.json")
    if os.path.exists(tfile):
        with open(tfile) as f:
            tr = json.load(f)
        ent = tr.get(args.config, {}).get(dominant)
        if ent and ent.get("source_sha") == src_hash(KERNEL_SOURCES[dominant]):
            traffic = ent.get("dram_bytes_per_launch")
    t_s = fam_ms[dominant] / 1e3
    if dominant == "output_error":
        peak = peaks["bf16_tflops"]
        ach = fam_work[dominant] / t_s / 1e12
        return {"kernel": "output_error_f16_kernel (Eq. 11, tcgen05 cta_group::2 kind::f16, "
                          "scaled fp16 hi/lo operands, 3 passes, X split ahead; after "
                          "pair_range_kernel and f16_split_kernel; output_error_tc_kernel for rows "
                          "not 16-byte multiples)",
                "bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                "frac": ach / peak, "traffic": traffic,
                "peak_source": f"{peak_src} bf16 dense burst (the fp16 rate of kind::f16)"}
    if dominant == "quantize":
        mhz = peaks.get("sm_max_mhz", 2070.0)
        peak = sm_count * ALU_LANES_PER_SM * mhz * 1e6 / 1e12
        ach = fam_work[dominant] / t_s / 1e12
        return {"kernel": "quantize_kernel (Eq. 7-9 lattice form, all k_max steps)", "bound": "alu",
                "achieved": ach, "peak": peak, "unit": "Tlane-op/s", "frac": ach / peak,
                "traffic": traffic,
                "peak_source": f"{sm_count} SMs x {ALU_LANES_PER_SM} lanes x {mhz:.0f} MHz "
                               f"(algorithmic ops: {GREEDY_OPS_PER_ELEMENT_STEP} per element-step "
                               "+ per channel-step scan, fold and screen)"}
    hbm = peaks["hbm_gbs"]
    ach = fam_work.get(dominant, 0.0) / t_s / 1e9
    names = {"reconstruct": "reconstruct_vec4_kernel (Eq. 4)",
             "allocate": "allocate_budget_kernel (Algorithm 2)",
             "center": "center_channel_kernel (Eq. 1 centre, centred weights)"}
    return {"kernel": names.get(dominant, dominant), "bound": "hbm", "achieved": ach, "peak": hbm,
            "unit": "GB/s", "frac": ach / hbm, "traffic": traffic,
            "peak_source": f"{peak_src} HBM copy"}


def greedy_roofline(fam_ms, fam_work, fam_bytes, peaks, peak_src, wl, args, sm_count):
    """The greedy search (mpq_quantize_layer) against HBM: algorithmic bytes (read W once, write
    the k_max code planes, the scales and the residual norms) / its single-stream time, with its
    lane-operation rate against the ALU peak beside it (the kernel is bound by instruction issue,
    not by HBM)."""
    hbm = peaks["hbm_gbs"]
    t_s = fam_ms["quantize"] / 1e3
    ach = fam_bytes["quantize"] / t_s / 1e9
    traffic = None
    tfile = os.path.join(PROFILES, "roofline_traffic.json")
    if os.path.exists(tfile):
        with open(tfile) as f:
            ent = json.load(f).get(args.config, {}).get("quantize")
        if ent and ent.get("source_sha") == src_hash(KERNEL_SOURCES["quantize"]):
            traffic = ent.get("dram_bytes_per_launch")
    mhz = peaks.get("sm_max_mhz", 2070.0)
    alu_peak = sm_count * ALU_LANES_PER_SM * mhz * 1e6 / 1e12
    alu = fam_work["quantize"] / t_s / 1e12
    n_launch = len(wl.layers) * len(wl.bits)
    return {"kernel": "quantize_kernel (Eq. 7-9, lattice form, all k_max steps in one launch)",
            "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
            "traffic": traffic, "peak_source": f"{peak_src} HBM copy",
            "bytes_per_launch": fam_bytes["quantize"] / args.steps / n_launch,
            "ms_per_step": fam_ms["quantize"] / args.steps,
            "alu": {"achieved": alu, "peak": alu_peak, "unit": "Tlane-op/s",
                    "frac": alu / alu_peak,
                    "peak_source": f"{sm_count} SMs x {ALU_LANES_PER_SM} lanes x {mhz:.0f} MHz; "
                                   f"{GREEDY_OPS_PER_ELEMENT_STEP} algorithmic lane operations "
                                   "per element-step + the per channel-step scan, fold and "
                                   "screen"}}


def run_e2e(net, specs, Whs, Xhs, Ws, Xs, wl, args, stream, units_per_step):
    """Same metric through the public network call with host buffers: per layer, H2D of W and X
    from pinned memory, the path, D2H of codes / scales / point counts -- all inside the timing.
    The step is NetworkPlan.run_host, captured into a CUDA graph like the device step (one graph
    per bit width; --graph 0 launches it call by call)."""
    import torch
    from paper_2002_09049_gb300 import pipeline
    # the inputs are copied in once per step; every bit width's outputs are copied out
    h2d = sum(w.numel() * 4 + x.numel() * 4 for w, x in zip(Whs, Xhs))
    d2h = sum(p.d2h_bytes() for p in net.plans) * len(wl.bits)
    graphs = []
    if args.graph:
        for n, b in enumerate(wl.bits):
            for sp in specs:
                sp.bits = b
            graphs.append(pipeline.CapturedNetwork(net, Ws, Xs, host=(Whs, Xhs),
                                                   copy_inputs=n == 0))

    def step():
        if graphs:
            for g in graphs:
                g.replay()
            return
        for n, b in enumerate(wl.bits):
            for sp in specs:
                sp.bits = b
            net.run_host(Whs, Xhs, Ws, Xs, stream=stream, copy_inputs=n == 0)

    for _ in range(max(1, args.warmup)):
        step()
    torch.cuda.synchronize()
    times = []
    for _ in range(args.steps):
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        z = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        step()
        z.record(stream)
        z.synchronize()
        times.append(a.elapsed_time(z))
    ms = float(np.mean(times))
    # the mean is the metric; the median is reported beside it because a host-side stall of
    # tens of ms now and then (seen in graph and call-by-call steps alike) lands in the mean
    return {"value": units_per_step / (ms / 1e3), "unit": UNIT, "ms_per_step": ms,
            "ms_per_step_median": float(np.median(times)),
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)}


# ------------------------------------------------------------------------------------------------
def oracle_sample(wl, target_s):
    """A bounded, proportional sample of the workload for the CPU oracle: every layer keeps the
    channels k = 0, stride, 2*stride, ...  Returns (sample list, stride)."""
    total_ch = wl.n_channels
    # rough oracle cost per channel (s, single core): quantize d*G*k_max*6ns + error d*N*(k+1)*1ns
    est = sum(l.C * (l.d * wl.G * wl.k_max * 6e-9 + l.d * wl.n_calib * (wl.k_max + 1) * 1.2e-9)
              for l in wl.layers) * len(wl.bits)
    cores = host_cores()
    stride = max(1, int(np.ceil(est / cores / target_s)))
    return stride


def run_oracle_step(wl, stride, threads, inputs, center=-1, collect=None):
    """The oracle over the sampled channels of every layer: centring (asymmetric sets), Algorithm
    1, Eq. 11, Algorithm 2 (budget, per layer, on the sample), Eq. 4.  Returns the metric units
    processed; with a dict ``collect``, also keeps each (bits, layer)'s codes, scales, error table
    and near-tie record there."""
    import oracle
    units = 0
    for b in wl.bits:
        for li, layer in enumerate(wl.layers):
            W, X = inputs[li]
            B = None
            if center >= 0:
                B, W = oracle.center(W, center)
            q = oracle.quantize_layer(W, b, wl.G, wl.k_max, want_residuals=False, threads=threads)
            groups = W.shape[0] if layer.groups > 1 else 1
            err = oracle.output_error(X, groups, W, q["codes"], q["scales"], wl.k_max,
                                      threads=threads)
            n, _ = oracle.allocate_budget(err.astype(np.float32), wl.k_max, wl.beta)
            oracle.reconstruct(q["codes"], q["scales"], n, center=B)
            units += W.shape[0] * layer.d * wl.G * wl.k_max
            if collect is not None:
                collect[(b, li)] = dict(W=W, codes=q["codes"], scales=q["scales"], err=err,
                                        best=q["best"], second=q["second"])
    return units


def sample_inputs(wl, stride):
    from paper_2002_09049_gb300 import workloads as wlm
    inputs = []
    for li, layer in enumerate(wl.layers):
        W, X = layer_inputs(wl, li)
        sel = np.arange(0, layer.C, stride)
        Ws = np.ascontiguousarray(W[sel])
        Xs = np.ascontiguousarray(X[sel]) if layer.groups > 1 else X
        inputs.append((Ws, Xs))
    return inputs


def cpu_baseline(wl, target_s, center=-1):
    """The oracle timed on the sampled channels; returns (cpu_baseline record, the oracle's
    outputs per (bits, layer) for the parity report)."""
    import oracle
    oracle.build()
    stride = oracle_sample(wl, target_s)
    threads = host_cores()
    inputs = sample_inputs(wl, stride)
    collect = {}
    t0 = time.perf_counter()
    units = run_oracle_step(wl, stride, threads, inputs, center, collect=collect)
    dt = time.perf_counter() - t0
    return ({"value": units / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
             "seconds": dt,
             "sample": f"every {stride}th channel of every layer of the same workload "
                       f"({units:.3e} units), oracle threads over channels"}, collect)


def gpu_sample_outputs(net, specs, Ws, Xs, wl, stream, stride):
    """Runs every bit width once more (one stream) and keeps the GPU's results for the parity
    report: codes, scales and reconstructions of the sampled channels (every stride-th), the whole
    error table and point counts of every layer (the allocation is checked on the full table)."""
    import torch
    out = {}
    for b in wl.bits:
        for sp in specs:
            sp.bits = b
        net.run_device(Ws, Xs, stream=stream)
        torch.cuda.synchronize()
        for li, p in enumerate(net.plans):
            sel = torch.arange(0, p.spec.C, stride, device=p.codes.device)
            out[(b, li)] = dict(codes=p.codes.index_select(1, sel).cpu().numpy(),
                                scales=p.scales.index_select(0, sel).cpu().numpy(),
                                err=p.err.cpu().numpy(), npoints=p.npoints.cpu().numpy(),
                                points_used=int(p.points_used.item()),
                                W_hat=p.W_hat.index_select(0, sel).cpu().numpy(),
                                center=None if p.center is None else
                                p.center.index_select(0, sel).cpu().numpy(), stride=stride)
    return out


NEAR_TIE_RTOL = 1e-6     # oracle top-two candidate errors this close (relative) are a near tie
VALUE_RTOL = 1e-5        # fp32 values (output errors) against the oracle's double results


def parity_report(wl, gpu, orc, center=-1):
    """GPU results against the oracle on the sampled channels, counted the way the parity bar
    states them: codes and scales bit-exact per greedy step except at a near tie (the oracle's
    error at the GPU's scale within 1e-6 relative of its best; the channel's later steps are then
    excluded), output errors within 1e-5 relative (channels that never diverged), point counts
    bit-exact against the oracle's allocation of the GPU's whole error table (Algorithm 2 as a
    sequential loop), reconstructions (Eq. 4) bit-exact."""
    import oracle
    rep = dict(channels=0, steps_compared=0, mismatch_steps=0, near_tie_mismatches=0,
               other_mismatches=0, diverged_steps_excluded=0, oracle_near_ties=0, err_values=0,
               err_max_rel=0.0, npoints_compared=0, npoints_mismatches=0,
               points_used_mismatches=0, reconstruct_mismatch_channels=0)
    K = wl.k_max
    for (b, li), o in orc.items():
        g = gpu[(b, li)]
        C_s = o["codes"].shape[1]
        rep["channels"] += C_s
        o_best, o_second = o["best"], o["second"]
        rep["oracle_near_ties"] += int(np.sum((o_second - o_best) <= NEAR_TIE_RTOL * o_second))
        for c in range(C_s):
            diverged = None
            for i in range(K):
                same = (g["scales"][c, i].tobytes() == o["scales"][c, i].tobytes() and
                        np.array_equal(g["codes"][i, c], o["codes"][i, c]))
                if same:
                    rep["steps_compared"] += 1
                    continue
                rep["mismatch_steps"] += 1
                if g["scales"][c, i].tobytes() == o["scales"][c, i].tobytes():
                    rep["other_mismatches"] += 1      # same scale, other codes: never a tie
                    rep["diverged_steps_excluded"] += K - 1 - i
                    diverged = i
                    break
                r = o["W"][c] if i == 0 else oracle.quantize_layer(
                    o["W"][c:c + 1], b, wl.G, i)["residuals"][i - 1, 0]
                E, s = oracle.candidate_errors(r, b, wl.G)
                hit = np.nonzero(s == g["scales"][c, i])[0]
                if hit.size and E[hit[0]] <= E.min() * (1 + NEAR_TIE_RTOL):
                    rep["near_tie_mismatches"] += 1
                else:
                    rep["other_mismatches"] += 1
                rep["diverged_steps_excluded"] += K - 1 - i
                diverged = i
                break
            if diverged is None:
                ge = g["err"][c * g["stride"]].astype(np.float64)
                oe = o["err"][c]
                f = np.isfinite(oe)
                if f.any():
                    rel = np.abs(ge[f] - oe[f]) / np.maximum(np.abs(oe[f]), 1e-300)
                    rep["err_max_rel"] = max(rep["err_max_rel"], float(rel.max()))
                    rep["err_values"] += int(f.sum())
        n_or, used_or = oracle.allocate_budget(g["err"], K, wl.beta)
        rep["npoints_compared"] += n_or.size
        rep["npoints_mismatches"] += int(np.sum(n_or != g["npoints"]))
        rep["points_used_mismatches"] += int(used_or != g["points_used"])
        sel_n = g["npoints"][::g["stride"]]
        W_or = oracle.reconstruct(g["codes"], g["scales"], sel_n, center=g["center"])
        rep["reconstruct_mismatch_channels"] += int(np.sum(
            np.any(W_or.view(np.uint32) != g["W_hat"].view(np.uint32), axis=1)))
    rep["err_rtol"] = VALUE_RTOL
    rep["near_tie_rtol"] = NEAR_TIE_RTOL
    rep["status"] = "pass" if (rep["other_mismatches"] == 0 and rep["npoints_mismatches"] == 0 and
                               rep["points_used_mismatches"] == 0 and
                               rep["reconstruct_mismatch_channels"] == 0 and
                               rep["err_max_rel"] <= VALUE_RTOL) else "fail"
    rep["sample"] = (f"every {next(iter(gpu.values()))['stride']}th channel of every layer "
                     "(the cpu_baseline sample); point counts on every channel")
    return rep


def run_reference(args, world, rank):
    """The oracle as the reference arm, on the host cores; rank 0 only."""
    if rank != 0:
        return None
    import oracle
    from paper_2002_09049_gb300 import workloads as wlm
    oracle.build()
    wl = wlm.WORKLOADS[args.config]
    per_step = max(2.0, 150.0 / max(1, args.steps + args.warmup))
    stride = oracle_sample(wl, per_step)
    threads = host_cores()
    inputs = sample_inputs(wl, stride)
    cen = CENTER_MODES[args.center]
    for _ in range(args.warmup):
        run_oracle_step(wl, stride, threads, inputs, cen)
    times, units = [], 0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        units = run_oracle_step(wl, stride, threads, inputs, cen)
        times.append(time.perf_counter() - t0)
    s = float(np.mean(times))
    value = units / s
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": f"{args.config}: {wl.title}", "bits": list(wl.bits), "G": wl.G,
                       "k_max": wl.k_max, "budget": wl.beta, "center": args.center},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"every {stride}th channel of every layer per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


CLIP_METRIC = "weight-elements x clip-candidates / s"
CLIP_UNIT = "elem*cand/s"


def clip_oracle_step(wl, stride, threads, inputs, n_cand):
    """The oracle's Eq. 12 search (per-channel candidates, errors, argmin) on the sampled channels."""
    import oracle
    units = 0
    for li, layer in enumerate(wl.layers):
        W, X = inputs[li]
        groups = W.shape[0] if layer.groups > 1 else 1
        clip = oracle.clip_candidates(W, n_cand, oracle.CLIP_PER_CHANNEL)
        err = oracle.clip_errors(X, groups, W, wl.bits[0], clip, threads=threads)
        oracle.clip_select(err.astype(np.float32), oracle.CLIP_PER_CHANNEL)
        units += W.shape[0] * W.shape[1] * n_cand
    return units


def clip_oracle_stride(wl, target_s, n_cand):
    est = sum(l.C * l.d * wl.n_calib * n_cand * 1.2e-9 for l in wl.layers)
    return max(1, int(np.ceil(est / host_cores() / target_s)))


def clip_launches(layer, n_cand):
    """Kernels one mpq_clip_search call launches: candidates and argmin, plus (tensor-core path) the
    X range and split and, per chunk of at most 4 GiB of residual planes, the planes and the
    contraction; else the shared-memory error kernel."""
    if layer.groups != 1 or layer.d % 16:
        return 3
    per_chunk = max(1, (1 << 32) // (4 * layer.d * n_cand))
    chunks = -(-layer.C // min(layer.C, per_chunk))
    return 4 + 2 * chunks


def run_clip(args, world, rank, local):
    """Eq. 12 over every layer of the workload: mpq_clip_search (per-channel candidates, output
    errors on the tensor cores, argmin) with layers on a pool of streams."""
    import torch
    from paper_2002_09049_gb300 import _build, binding
    from paper_2002_09049_gb300 import dist as dist_helpers
    from paper_2002_09049_gb300 import workloads as wlm

    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or world == 1:
        _build.build()
    if world > 1:
        torch.distributed.barrier()
    binding.load()
    wl = wlm.WORKLOADS[args.config]
    nc = args.clip_candidates
    bits = wl.bits[0]
    keep = None if args.layers is None else {int(x) for x in args.layers.split(",")}
    idx = [li for li in range(len(wl.layers)) if keep is None or li in keep]
    layers = [wl.layers[li] for li in idx]
    Ws, Xs, Whs, Xhs, outs = [], [], [], [], []
    for li, layer in zip(idx, layers):
        W, X = layer_inputs(wl, li)
        Whs.append(torch.from_numpy(W).pin_memory())
        Xhs.append(torch.from_numpy(X).pin_memory())
        Ws.append(Whs[-1].to(dev))
        Xs.append(Xhs[-1].to(dev))
        mk = lambda dt, shape: torch.empty(shape, dtype=dt, device=dev)
        outs.append((mk(torch.float32, (layer.C, nc)), mk(torch.float32, (layer.C, nc)),
                     mk(torch.int32, (layer.C,))))
    order = sorted(range(len(layers)), key=lambda i: -layers[i].C * layers[i].d)
    streams = [torch.cuda.Stream(dev) for _ in range(max(1, args.streams))]
    main = torch.cuda.current_stream()
    units_per_step = sum(l.C * l.d * nc for l in layers)
    flops_per_step = sum(2.0 * wl.n_calib * l.d * l.C * nc for l in layers)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    def call(i, st):
        c, e, b = outs[i]
        binding.mpq_clip_search(Xs[i], Ws[i], bits, nc, binding.MPQ_CLIP_PER_CHANNEL,
                                groups=layers[i].groups, clip=c, err=e, best=b, stream=st)

    def step():
        ev = torch.cuda.Event()
        ev.record(main)
        for st in streams:
            st.wait_event(ev)
        for n, i in enumerate(order):
            call(i, streams[n % len(streams)])
        for st in streams:
            e = torch.cuda.Event()
            e.record(st)
            main.wait_event(e)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    peaks, peak_src = measured_peaks()
    step_ms = []
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for _ in range(args.steps):
            flush.fill_(1.0)
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(main)
            step()
            z.record(main)
            torch.cuda.synchronize()
            step_ms.append(a.elapsed_time(z))
    # per-call durations on one stream for the roofline
    one_ms = []
    for _ in range(args.steps):
        flush.fill_(1.0)
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(order) + 1)]
        evs[0].record(main)
        for n, i in enumerate(order):
            call(i, main)
            evs[n + 1].record(main)
        torch.cuda.synchronize()
        one_ms.append(evs[0].elapsed_time(evs[-1]))
    if world > 1:
        torch.distributed.barrier()
    ms = dist_helpers.max_over_ranks(float(np.mean(step_ms)), device=dev)
    value = dist_helpers.aggregate_throughput(units_per_step, ms, world)
    t1 = float(np.mean(one_ms)) / 1e3
    peak = peaks["bf16_tflops"]
    ach = flops_per_step / t1 / 1e12
    roofline = {"kernel": "output_error_f16_kernel in clip mode (Eq. 12 residuals written once as "
                          "fp16 hi/lo planes by clip_planes_kernel and tile-copied into a tcgen05 "
                          "cta_group::2 kind::f16 3-pass contraction) + candidate, X range, X split "
                          "and argmin kernels",
                "bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                "frac": ach / peak, "traffic": None,
                "peak_source": f"{peak_src} bf16 dense burst (fp16 operands: the same rate)",
                "timing": "whole calls (candidates, errors, argmin) on one stream, CUDA events; "
                          "achieved = algorithmic flops 2*N*d*C*n_cand / that time",
                "single_stream_ms_per_step": t1 * 1e3}
    out = {"metric": CLIP_METRIC, "value": value, "unit": CLIP_UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
           "data": "synthetic",
           "config": {"workload": f"{args.config}: {wl.title}", "op": "clip (Eq. 12)",
                      "layers": len(layers), "clip_candidates": nc, "sets": "per channel",
                      "bits": bits, "calib_rows": wl.n_calib, "units_per_step": units_per_step,
                      "l2": "flushed between steps (512 MB write)", "streams": args.streams,
                      "parallelism": f"replicas x{world}"},
           "roofline": roofline,
           "gpu_launches": sum(clip_launches(l, nc) for l in layers) * args.steps,
           "clocks": clk.summary()}
    if not args.no_e2e:
        def e2e_step():
            ev = torch.cuda.Event()
            ev.record(main)
            for st in streams:
                st.wait_event(ev)
            host = []
            for n, i in enumerate(order):
                st = streams[n % len(streams)]
                with torch.cuda.stream(st):
                    Ws[i].copy_(Whs[i], non_blocking=True)
                    Xs[i].copy_(Xhs[i], non_blocking=True)
                    call(i, st)
                    c, e, b = outs[i]
                    host.append((c.to("cpu", non_blocking=True), e.to("cpu", non_blocking=True),
                                 b.to("cpu", non_blocking=True)))
            for st in streams:
                e = torch.cuda.Event()
                e.record(st)
                main.wait_event(e)
            return host
        for _ in range(max(1, args.warmup)):
            e2e_step()
        torch.cuda.synchronize()
        tms = []
        for _ in range(args.steps):
            flush.fill_(1.0)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            e2e_step()
            torch.cuda.synchronize()
            tms.append((time.perf_counter() - t0) * 1e3)
        e_ms = float(np.mean(tms))
        out["e2e"] = {"value": units_per_step / (e_ms / 1e3), "unit": CLIP_UNIT, "ms_per_step": e_ms,
                      "h2d_bytes_per_step": sum(w.numel() * 4 + x.numel() * 4
                                                for w, x in zip(Whs, Xhs)),
                      "d2h_bytes_per_step": sum(l.C * nc * 8 + l.C * 4 for l in layers)}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        stride = clip_oracle_stride(wl, args.cpu_seconds, nc)
        inputs = sample_inputs(wl, stride)
        t0 = time.perf_counter()
        units = clip_oracle_step(wl, stride, host_cores(), inputs, nc)
        dt = time.perf_counter() - t0
        out["cpu_baseline"] = {"value": units / dt, "unit": CLIP_UNIT, "cores": host_cores(),
                               "kind": "oracle", "seconds": dt,
                               "sample": f"every {stride}th channel of every layer ({units:.3e} "
                                         "units), oracle threads over channels"}
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    return out if rank == 0 else None


INFER_METRIC = "multipoint integer MACs / s"
INFER_UNIT = "MAC/s"


def infer_layers(args, wl, dev):
    """Per layer: quantize, output error and budget allocation on the device (not timed), the
    packed layer, and int8 inputs (T = the workload's calibration rows)."""
    import torch
    from paper_2002_09049_gb300 import binding
    keep = None if args.layers is None else {int(x) for x in args.layers.split(",")}
    out = []
    for li, layer in enumerate(wl.layers):
        if keep is not None and li not in keep:
            continue
        W, X = layer_inputs(wl, li)
        Wd, Xd = torch.from_numpy(W).to(dev), torch.from_numpy(X).to(dev)
        B = None
        if CENTER_MODES[args.center] >= 0:
            B, Wd = binding.mpq_center_weights(Wd, CENTER_MODES[args.center])
        codes, scales, _, _ = binding.mpq_quantize_layer(Wd, wl.bits[0], wl.G, wl.k_max)
        err = binding.mpq_output_error(Xd, Wd, codes, scales, wl.k_max,
                                       groups=layer.C if layer.groups > 1 else 1)
        npts, _ = binding.mpq_allocate_points(err, wl.k_max, binding.MPQ_ALLOC_BUDGET, wl.beta)
        n_host = npts.cpu().numpy()
        lay = binding.mpq_pack_layout(n_host, layer.d, wl.k_max, wl.bits[0], args.coef_bits,
                                      centered=B is not None)
        packed = binding.mpq_pack_points(codes, scales, n_host, lay, center=B)
        Xq = np.random.default_rng(900000 + li).integers(-128, 128, (wl.n_calib, layer.d))
        Xh = torch.from_numpy(Xq.astype(np.int8)).pin_memory()
        out.append(dict(layer=layer, lay=lay, packed=packed, Xh=Xh, X=Xh.to(dev),
                        Y=torch.empty((layer.C, wl.n_calib), dtype=torch.int32, device=dev),
                        macs=int(n_host.sum()) * layer.d * wl.n_calib,
                        codes=codes.cpu().numpy(), scales=scales.cpu().numpy(), n=n_host, Xq=Xq,
                        center=None if B is None else B.cpu().numpy()))
    return out


def run_infer(args, world, rank, local):
    """Eq. 13 over every layer: mpq_multipoint_linear on the packed layers, layers on streams."""
    import torch
    from paper_2002_09049_gb300 import _build, binding
    from paper_2002_09049_gb300 import dist as dist_helpers
    from paper_2002_09049_gb300 import workloads as wlm

    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or world == 1:
        _build.build()
    if world > 1:
        torch.distributed.barrier()
    binding.load()
    wl = wlm.WORKLOADS[args.config]
    L = infer_layers(args, wl, dev)
    order = sorted(range(len(L)), key=lambda i: -L[i]["macs"])
    streams = [torch.cuda.Stream(dev) for _ in range(max(1, args.streams))]
    main = torch.cuda.current_stream()
    macs = sum(x["macs"] for x in L)
    mma_macs = sum(x["lay"].rows * x["layer"].d * wl.n_calib for x in L)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    def call(i, st):
        x = L[i]
        binding.mpq_multipoint_linear(x["X"], x["lay"], x["packed"], Y=x["Y"], stream=st)

    def step():
        ev = torch.cuda.Event()
        ev.record(main)
        for st in streams:
            st.wait_event(ev)
        for n, i in enumerate(order):
            call(i, streams[n % len(streams)])
        for st in streams:
            e = torch.cuda.Event()
            e.record(st)
            main.wait_event(e)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    peaks, peak_src = measured_peaks()
    step_ms = []
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for _ in range(args.steps):
            flush.fill_(1.0)
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(main)
            step()
            z.record(main)
            torch.cuda.synchronize()
            step_ms.append(a.elapsed_time(z))
    one_ms = []
    for _ in range(args.steps):
        flush.fill_(1.0)
        a = torch.cuda.Event(enable_timing=True)
        z = torch.cuda.Event(enable_timing=True)
        a.record(main)
        for i in order:
            call(i, main)
        z.record(main)
        torch.cuda.synchronize()
        one_ms.append(a.elapsed_time(z))
    if world > 1:
        torch.distributed.barrier()
    ms = dist_helpers.max_over_ranks(float(np.mean(step_ms)), device=dev)
    value = dist_helpers.aggregate_throughput(macs, ms, world)
    t1 = float(np.mean(one_ms)) / 1e3
    peak = peaks["bf16_tflops"]
    ach = 2.0 * macs / t1 / 1e12
    roofline = {"kernel": "multipoint_linear_kernel (Eq. 13 step 1 on tcgen05 kind::f16 bf16, "
                          "steps 2-3 in the epilogue)",
                "bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                "frac": ach / peak, "traffic": None,
                "peak_source": f"{peak_src} bf16 dense burst",
                "timing": "all layers on one stream, CUDA events; achieved = 2 x the multipoint "
                          "MACs (used points only) / that time",
                "packed_row_macs_per_used_mac": mma_macs / macs,
                "single_stream_ms_per_step": t1 * 1e3}
    out = {"metric": INFER_METRIC, "value": value, "unit": INFER_UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int8 x int4",
           "data": "synthetic",
           "config": {"workload": f"{args.config}: {wl.title}", "op": "infer (Eq. 13)",
                      "layers": len(L), "inputs_per_layer": wl.n_calib, "p": args.coef_bits,
                      "points": f"budget {wl.beta} per channel (Algorithm 2)",
                      "center": args.center,
                      "macs_per_step": macs, "l2": "flushed between steps (512 MB write)",
                      "streams": args.streams, "parallelism": f"replicas x{world}"},
           "roofline": roofline, "gpu_launches": len(L) * args.steps, "clocks": clk.summary()}
    if not args.no_e2e:
        # inputs in on one copy stream (largest layer first), each layer's kernel as soon as its
        # inputs have landed, outputs out on a second copy stream into pinned buffers; captured
        # into a CUDA graph (one host call per step) unless --graph 0
        Yh = [torch.empty(x["Y"].shape, dtype=torch.int32).pin_memory() for x in L]
        copy_in, copy_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

        def e2e_launch(root):
            ev = torch.cuda.Event()
            ev.record(root)
            for st in streams + [copy_in, copy_out]:
                st.wait_event(ev)
            landed = {}
            for i in order:
                with torch.cuda.stream(copy_in):
                    L[i]["X"].copy_(L[i]["Xh"], non_blocking=True)
                landed[i] = torch.cuda.Event()
                landed[i].record(copy_in)
            for n, i in enumerate(order):
                st = streams[n % len(streams)]
                st.wait_event(landed[i])
                call(i, st)
                done = torch.cuda.Event()
                done.record(st)
                copy_out.wait_event(done)
                with torch.cuda.stream(copy_out):
                    Yh[i].copy_(L[i]["Y"], non_blocking=True)
            for st in streams + [copy_in, copy_out]:
                e = torch.cuda.Event()
                e.record(st)
                root.wait_event(e)

        side = torch.cuda.Stream(dev)
        side.wait_stream(main)
        with torch.cuda.stream(side):
            for _ in range(max(1, args.warmup)):
                e2e_launch(side)
        main.wait_stream(side)
        torch.cuda.synchronize()
        graph = None
        if args.graph:
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=side):
                e2e_launch(side)
            torch.cuda.synchronize()

        def e2e_step():
            if graph is not None:
                graph.replay()
            else:
                e2e_launch(main)
        e2e_step()
        torch.cuda.synchronize()
        tms = []
        for _ in range(args.steps):
            flush.fill_(1.0)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            e2e_step()
            torch.cuda.synchronize()
            tms.append((time.perf_counter() - t0) * 1e3)
        for x, y in zip(L, Yh):   # the host outputs are the device results
            if not torch.equal(y, x["Y"].cpu()):
                raise RuntimeError("end-to-end outputs differ from the device results")
        e_ms = float(np.mean(tms))
        out["e2e"] = {"value": macs / (e_ms / 1e3), "unit": INFER_UNIT, "ms_per_step": e_ms,
                      "h2d_bytes_per_step": sum(x["Xh"].numel() for x in L),
                      "d2h_bytes_per_step": sum(x["Y"].numel() * 4 for x in L)}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        t0 = time.perf_counter()
        units = 0
        for x in L:   # a channel sample of every layer, bounded to about --cpu-seconds
            C = x["layer"].C
            per_ch = x["macs"] / max(1, C) * 1.5e-9
            nc = max(1, min(C, int(args.cpu_seconds / len(L) / max(per_ch, 1e-12)) * host_cores()))
            oracle.multipoint_linear(x["Xq"].astype(np.int8), x["codes"], x["scales"], x["n"],
                                     args.coef_bits, channels=(0, nc), threads=host_cores(),
                                     center=x["center"])
            units += int(x["n"][:nc].sum()) * x["layer"].d * wl.n_calib
        dt = time.perf_counter() - t0
        out["cpu_baseline"] = {"value": units / dt, "unit": INFER_UNIT, "cores": host_cores(),
                               "kind": "oracle", "seconds": dt,
                               "sample": f"the first channels of every layer ({units:.3e} MACs), "
                                         "oracle threads over channels"}
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    return out if rank == 0 else None


ADAPTIVE_CAP = 10 ** 15      # no refusal: the search does not enumerate the grid
ADAPTIVE_METRIC = "weight-elements x points / s (adaptive grid of Eq. 10)"
ADAPTIVE_UNIT = "elem*pt/s"
ADAPTIVE_BUDGET_S = 20.0     # timed GPU work of one --op adaptive run, at most
# Algorithmic lane operations of the adaptive search, per code-level threshold (every element
# has Qmax of them a step): finding it (two correctly rounded divisions, rint, compare: 25),
# sorting it (4 radix passes of 2 loads, a match, a popc, a store: 48), its piece's running sums
# and fp32 lower bound (30); per element-step: the magnitude sort for Definition 1 (48), its gap
# (6), the update and code store (11).
ADAPTIVE_OPS_PER_THRESHOLD = 103
ADAPTIVE_OPS_PER_ELEMENT = 65


def adaptive_layers(wl):
    from paper_2002_09049_gb300 import binding
    qmax = (1 << (wl.bits[0] - 1)) - 1
    idx = [li for li, l in enumerate(wl.layers)
           if l.d * qmax <= binding.MPQ_ADAPTIVE_MAX_THRESHOLDS]
    if not idx:
        raise SystemExit("--op adaptive: no layer with d * Qmax <= MPQ_ADAPTIVE_MAX_THRESHOLDS")
    return idx


def adaptive_ops(wl, layer):
    qmax = (1 << (wl.bits[0] - 1)) - 1
    return layer.C * layer.d * wl.k_max * (ADAPTIVE_OPS_PER_THRESHOLD * qmax +
                                           ADAPTIVE_OPS_PER_ELEMENT)


def adaptive_oracle_step(wl, idx, per_layer, threads):
    """The oracle's adaptive grid (Eq. 10; its piecewise search, the definition's decisions
    without enumerating) on the first `per_layer` channels of every layer; returns the
    element-steps (C d k_max) it processed."""
    import oracle
    from concurrent.futures import ThreadPoolExecutor
    jobs = [(li, c) for li in idx for c in range(min(per_layer, wl.layers[li].C))]
    Ws = {li: layer_inputs(wl, li)[0] for li in idx}

    def one(job):
        li, c = job
        oracle.quantize_adaptive(Ws[li][c:c + 1], wl.bits[0], wl.k_max,
                                 max_candidates=ADAPTIVE_CAP, refuse="mark", piecewise=True)
        return wl.layers[li].d * wl.k_max

    with ThreadPoolExecutor(max_workers=threads) as ex:
        return sum(ex.map(one, jobs))


def run_adaptive(args, world, rank, local):
    """Algorithm 1 with the adaptive grid of Eq. 10 (Definition 1) on every layer of the workload:
    mpq_quantize_layer_adaptive per layer on a pool of streams; value = weight-element-steps
    (C d k_max summed over layers) per second.  One single-stream pass is timed first and the
    number of timed steps is cut to fit ADAPTIVE_BUDGET_S."""
    import torch
    from paper_2002_09049_gb300 import _build, binding
    from paper_2002_09049_gb300 import dist as dist_helpers
    from paper_2002_09049_gb300 import workloads as wlm

    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or world == 1:
        _build.build()
    if world > 1:
        torch.distributed.barrier()
    binding.load()
    wl = wlm.WORKLOADS[args.config]
    idx = adaptive_layers(wl)
    if args.layers is not None:
        keep = {int(x) for x in args.layers.split(",")}
        idx = [li for li in idx if li in keep]
    layers = [wl.layers[li] for li in idx]
    bits, k_max = wl.bits[0], wl.k_max
    Whs = [torch.from_numpy(layer_inputs(wl, li)[0]).pin_memory() for li in idx]
    Ws = [w.to(dev) for w in Whs]
    mk = lambda dt, shape: torch.empty(shape, dtype=dt, device=dev)
    outs = [(mk(torch.int8, (k_max, l.C, l.d)), mk(torch.float32, (l.C, k_max)),
             mk(torch.float32, (l.C, k_max + 1)), mk(torch.int64, (l.C, k_max))) for l in layers]
    hosts = [(torch.empty(o[0].shape, dtype=torch.int8, pin_memory=True),
              torch.empty(o[1].shape, dtype=torch.float32, pin_memory=True)) for o in outs]
    order = sorted(range(len(layers)), key=lambda i: -layers[i].C * layers[i].d)
    streams = [torch.cuda.Stream(dev) for _ in range(max(1, args.streams))]
    main = torch.cuda.current_stream()
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    def call(i, st):
        c, s_, r, n = outs[i]
        binding.mpq_quantize_layer_adaptive(Ws[i], bits, k_max, max_cand=ADAPTIVE_CAP, codes=c,
                                            scales=s_, resid_sq=r, ncand=n, stream=st)

    def step(host=False):
        ev = torch.cuda.Event()
        ev.record(main)
        for st in streams:
            st.wait_event(ev)
        for n, i in enumerate(order):
            st = streams[n % len(streams)]
            if host:
                with torch.cuda.stream(st):
                    Ws[i].copy_(Whs[i], non_blocking=True)
            call(i, st)
            if host:
                with torch.cuda.stream(st):
                    hosts[i][0].copy_(outs[i][0], non_blocking=True)
                    hosts[i][1].copy_(outs[i][1], non_blocking=True)
        for st in streams:
            e = torch.cuda.Event()
            e.record(st)
            main.wait_event(e)

    def one_stream():
        a = torch.cuda.Event(enable_timing=True)
        z = torch.cuda.Event(enable_timing=True)
        flush.fill_(1.0)
        a.record(main)
        for i in order:
            call(i, main)
        z.record(main)
        torch.cuda.synchronize()
        return a.elapsed_time(z)

    first_ms = one_stream()                     # also the first warm-up pass
    steps = max(1, min(args.steps, int(ADAPTIVE_BUDGET_S * 1e3 / max(first_ms, 1e-3) / 2)))
    warm = max(1, min(args.warmup, steps))
    for _ in range(warm):
        step()
    torch.cuda.synchronize()
    ncand = [o[3].cpu().numpy() for o in outs]
    grid_points = int(sum(np.maximum(n, 0).sum() for n in ncand))
    refused = int(sum((n < 0).sum() for n in ncand))
    units_per_step = sum(l.C * l.d * k_max for l in layers)
    step_ms = []
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for _ in range(steps):
            flush.fill_(1.0)
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(main)
            step()
            z.record(main)
            torch.cuda.synchronize()
            step_ms.append(a.elapsed_time(z))
    one_ms = [one_stream() for _ in range(steps)]
    if world > 1:
        torch.distributed.barrier()
    ms = dist_helpers.max_over_ranks(float(np.mean(step_ms)), device=dev)
    value = dist_helpers.aggregate_throughput(units_per_step, ms, world)
    t1 = float(np.mean(one_ms)) / 1e3
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    peaks, _ = measured_peaks()
    mhz = peaks.get("sm_max_mhz", 2070.0)
    alu_peak = sms * ALU_LANES_PER_SM * mhz * 1e6 / 1e12
    ach = sum(adaptive_ops(wl, l) for l in layers) / t1 / 1e12
    roofline = {"kernel": "adaptive_kernel (Algorithm 1 over the grid of Eq. 10: code-level "
                          "thresholds sorted, piecewise quadratic screened in fp32, settled in "
                          "double)", "bound": "alu", "achieved": ach, "peak": alu_peak,
                "unit": "Tlane-op/s", "frac": ach / alu_peak, "traffic": None,
                "peak_source": f"{sms} SMs x {ALU_LANES_PER_SM} lanes x {mhz:.0f} MHz; "
                               f"{ADAPTIVE_OPS_PER_THRESHOLD} lane operations per code-level "
                               f"threshold (Qmax per element-step) + {ADAPTIVE_OPS_PER_ELEMENT} "
                               "per element-step",
                "timing": "every layer on one stream, CUDA events",
                "single_stream_ms_per_step": t1 * 1e3}
    out = {"metric": ADAPTIVE_METRIC, "value": value, "unit": ADAPTIVE_UNIT, "n_gpus": world,
           "steps": steps, "warmup": warm, "ms_per_step": ms,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
           "data": "synthetic",
           "config": {"workload": f"{args.config}: {wl.title}",
                      "op": "adaptive grid (Def. 1 + Eq. 10)", "layers": len(layers),
                      "channels": sum(l.C for l in layers), "bits": bits, "k_max": k_max,
                      "eta": 2.0 ** -10, "grid_points_per_step": grid_points,
                      "refused_steps": refused, "units_per_step": units_per_step,
                      "first_pass_ms": first_ms,
                      "l2": "flushed between steps (512 MB write)", "streams": args.streams,
                      "parallelism": f"replicas x{world}"},
           "roofline": roofline, "gpu_launches": len(layers) * steps,
           "clocks": clk.summary()}
    if not args.no_e2e:
        step(host=True)
        torch.cuda.synchronize()
        times = []
        for _ in range(steps):
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(main)
            step(host=True)
            z.record(main)
            z.synchronize()
            times.append(a.elapsed_time(z))
        e_ms = float(np.mean(times))
        out["e2e"] = {"value": units_per_step / (e_ms / 1e3), "unit": ADAPTIVE_UNIT,
                      "ms_per_step": e_ms,
                      "h2d_bytes_per_step": int(sum(w.numel() * 4 for w in Whs)),
                      "d2h_bytes_per_step": int(sum(h[0].numel() + 4 * h[1].numel()
                                                    for h in hosts))}
    if not args.no_cpu_baseline and rank == 0:
        import oracle
        oracle.build()
        per_layer = 2
        t0 = time.perf_counter()
        units = adaptive_oracle_step(wl, idx, per_layer, host_cores())
        dt = time.perf_counter() - t0
        out["cpu_baseline"] = {"value": units / dt, "unit": ADAPTIVE_UNIT, "cores": host_cores(),
                               "kind": "oracle", "seconds": dt,
                               "sample": f"the first {per_layer} channels of every layer (the "
                                         "oracle's piecewise search), threads over channels"}
    return out


def run_adaptive_reference(args, world, rank):
    """The oracle's adaptive grid as the reference arm of --op adaptive, on the host cores."""
    if rank != 0:
        return None
    import oracle
    from paper_2002_09049_gb300 import workloads as wlm
    oracle.build()
    wl = wlm.WORKLOADS[args.config]
    idx = adaptive_layers(wl)
    per_layer = 2
    for _ in range(args.warmup):
        adaptive_oracle_step(wl, idx, 1, host_cores())
    times, units = [], 0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        units = adaptive_oracle_step(wl, idx, per_layer, host_cores())
        times.append(time.perf_counter() - t0)
    v = units / float(np.mean(times))
    return {"impl": "reference", "metric": ADAPTIVE_METRIC, "value": v, "unit": ADAPTIVE_UNIT,
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * float(np.mean(times)), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{args.config}: {wl.title}",
                       "op": "adaptive grid (Def. 1 + Eq. 10)", "bits": wl.bits[0],
                       "k_max": wl.k_max},
            "cpu_baseline": {"value": v, "unit": ADAPTIVE_UNIT, "cores": host_cores(),
                             "kind": "oracle",
                             "sample": f"the first {per_layer} channels of every layer per step "
                                       "(the oracle's piecewise search)"},
            "e2e": {"value": v, "unit": ADAPTIVE_UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def run_clip_reference(args, world, rank):
    """The oracle's Eq. 12 search as the reference arm of --op clip, on the host cores."""
    if rank != 0:
        return None
    import oracle
    from paper_2002_09049_gb300 import workloads as wlm
    oracle.build()
    wl = wlm.WORKLOADS[args.config]
    nc = args.clip_candidates
    per_step = max(2.0, 150.0 / max(1, args.steps + args.warmup))
    stride = clip_oracle_stride(wl, per_step, nc)
    inputs = sample_inputs(wl, stride)
    for _ in range(args.warmup):
        clip_oracle_step(wl, stride, host_cores(), inputs, nc)
    times, units = [], 0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        units = clip_oracle_step(wl, stride, host_cores(), inputs, nc)
        times.append(time.perf_counter() - t0)
    s = float(np.mean(times))
    value = units / s
    return {"impl": "reference", "metric": CLIP_METRIC, "value": value, "unit": CLIP_UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": f"{args.config}: {wl.title}", "op": "clip (Eq. 12)",
                       "clip_candidates": nc, "sets": "per channel"},
            "cpu_baseline": {"value": value, "unit": CLIP_UNIT, "cores": host_cores(),
                             "kind": "oracle",
                             "sample": f"every {stride}th channel of every layer per step"},
            "e2e": {"value": value, "unit": CLIP_UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    args = parse()
    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        if args.op == "infer":
            out = {"impl": "reference", "op": "infer",
                   "unavailable": "the integer inference path needs the device-quantized layers; "
                                  "its oracle is timed as cpu_baseline of --op infer"}
        else:
            out = {"clip": run_clip_reference,
                   "adaptive": run_adaptive_reference}.get(args.op, run_reference)(args, world, rank)
    elif args.op == "clip":
        out = run_clip(args, world, rank, local)
    elif args.op == "infer":
        out = run_infer(args, world, rank, local)
    elif args.op == "adaptive":
        out = run_adaptive(args, world, rank, local)
    else:
        out = run_ours(args, world, rank, local)
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
