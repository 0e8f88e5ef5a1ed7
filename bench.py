"""Benchmark: pattern- and connectivity-pruned 3x3 conv networks on one GB300.

Default workload: the VGG-16 conv trunk at 1x3x224x224 fp32 (13 pattern-pruned
convs, bias+ReLU, 4 fused 2x2 pools; conv1 keeps all kernels, the rest 30%).
A step is one frame through the whole trunk with ``pp_net_run`` (CUDA-graph
replay), inputs resident in HBM, L2 flushed between steps.

Printed JSON line (rank 0):
  value      surviving-weight GFLOP/s over all ranks (2 FLOP per kept MAC of the
             4 pattern taps; pruned kernels and taps never counted)
  ms_per_step  ms per frame
  e2e        the same metric through pp_net_run_host (pinned host buffers,
             H2D + run + D2H + sync every step)
  roofline   the dominant kernel of the pruned convs: its surviving-weight
             TFLOP/s over its launches timed inside the frame (op by op, events
             between the ops, L2 flushed once per frame) vs the FP32 FMA peak
             measured by pp_peak_probe in the same run (the method's roofline;
             the derived SMs x 128 lanes x 2 FLOP x max clock beside it);
             "tensor" adds the tensor-pipe view of the ops that run on the
             tensor cores (dense-tap FLOPs executed in their passes vs the
             tcgen05 MMA peak measured by the same probe)
  cpu_baseline the fp64 CPU oracle on this host's cores on a bounded sample
  configs    ms/frame, GFLOP/s, roofline fraction and tensor-pipe view of all
             five workloads

``--impl reference`` times the CPU oracle alone (the reference arm: the paper
ships no code) and prints the same metric.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

HBM_PEAK_GBS_FALLBACK = 6800.0
CONFIG_CPU_SECONDS = 4.0  # oracle sample per workload of the all-configs table
KERNEL_NAMES = {1: "ppconv_tm_kernel", 2: "ppconv_kernel", 3: "ppconv_tc_kernel", 4: "ppconv_tcf_kernel",
                5: "ppconv_direct_kernel"}
FP32_LANES_PER_SM = 128
SM_MAX_MHZ = 2070.0
L2_FLUSH_BYTES = 512 << 20
# Roofline denominators: FP32 FMA peak in TFLOP/s.  bench.py replaces it by the rate pp_peak_probe
# measures on the GPU it runs on (set_fp32_peak); the value below is the derived peak of a 152-SM
# GB300 at its maximum clock (152 x 128 lanes x 2 FLOP x 2.07 GHz), used before that and on the CPU.
FP32_PEAK_TFLOPS = 152 * FP32_LANES_PER_SM * 2 * SM_MAX_MHZ * 1e6 / 1e12  # 80.55


def set_fp32_peak(tflops: float):
    global FP32_PEAK_TFLOPS
    FP32_PEAK_TFLOPS = float(tflops)


def measure_peaks():
    """FP32 FMA and tcgen05 MMA (tf32, f16) peaks of this GPU by pp_peak_probe, each the best of 3
    launches of a few milliseconds, with the SM clock seen during the best one; plus the derived FP32
    peak (SMs x 128 lanes x 2 FLOP x maximum clock)."""
    import torch
    from paper_2004_11250_gb300 import ppconv as pp
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    out = {"sms": sms, "derived_fp32_tflops": round(sms * FP32_LANES_PER_SM * 2 * SM_MAX_MHZ * 1e6 / 1e12, 2),
           "derived_from": f"{sms} SMs x {FP32_LANES_PER_SM} FP32 lanes x 2 FLOP x {SM_MAX_MHZ:.0f} MHz"}
    for name, kind, iters in (("fp32_ffma", pp.PP_PROBE_FFMA, 1 << 16), ("tf32_mma", pp.PP_PROBE_MMA_TF32, 1 << 15),
                              ("f16_mma", pp.PP_PROBE_MMA_F16, 1 << 15)):
        pp.pp_peak_probe(kind, iters)  # warm-up (clocks ramp, code loads)
        best = max((pp.pp_peak_probe(kind, iters) for _ in range(3)), key=lambda r: r[0])
        out[name] = {"tflops": round(best[0], 2), "sm_mhz": round(best[1]), "ms": round(best[2], 3)}
    return out


def hbm_peak_gbs():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return HBM_PEAK_GBS_FALLBACK, "fallback"


# ----------------------------------------------------------------------------- workloads


def workload(name: str):
    from paper_2004_11250_gb300 import synth
    if name == "vgg16":
        return synth.cfg1_vgg16()
    if name == "single":
        return synth.cfg0_single()
    if name == "style":
        return synth.cfg2_style()
    if name == "vdsr":
        return synth.cfg3_vdsr()
    if name.startswith("sweep:"):  # sweep:C:P:keep, one point of the throughput sweep
        C, P, keep = name.split(":")[1:]
        return synth.cfg4_point(int(C), int(P), float(keep))
    if name.startswith("op:"):  # op:<workload>:<k>, op k of a network alone (for profiling one layer)
        base, k = name.split(":")[1:]
        return single_op(workload(base), int(k))
    raise ValueError(name)


def single_op(spec, k):
    """Op k of a network as a one-op network: same layer, flags and input shape; the input is seeded
    U(0, 1) (a ReLU network's activations are non-negative) and a skip, if any, is dropped."""
    from paper_2004_11250_gb300 import synth
    N, C, H, W = spec.x.shape
    for op in spec.ops[:k]:
        C = op.layer.Co
        if op.pool:
            H, W = H // 2, W // 2
    op = spec.ops[k]
    x = np.random.default_rng(k).uniform(0, 1, size=(N, C, H, W)).astype(np.float32)
    return synth.Net(f"{spec.name}_op{k}", x, [synth.Op(op.layer, relu=op.relu, pool=op.pool)])


def op_shapes(spec):
    """Per op: (N, Ci, Co, H, W, Ho, Wo, surviving FLOPs, compulsory bytes, pruned?)."""
    from paper_2004_11250_gb300 import synth
    N, C, H, W = spec.x.shape
    out = []
    for op in spec.ops:
        L = op.layer
        pruned = isinstance(L, synth.PrunedLayer)
        taps = 4 * L.nk if pruned else 9 * L.Co * L.Ci
        Ho, Wo = (H // 2, W // 2) if op.pool else (H, W)
        flops = 2 * N * H * W * taps
        nbytes = 4 * N * L.Ci * H * W + 4 * N * L.Co * Ho * Wo + 4 * L.Co
        nbytes += 21 * L.nk if pruned else 36 * L.Co * L.Ci
        if op.skip_from >= 0:
            nbytes += 4 * N * L.Co * H * W
        out.append(dict(N=N, Ci=L.Ci, Co=L.Co, H=H, W=W, Ho=Ho, Wo=Wo, flops=flops, bytes=nbytes, pruned=pruned))
        H, W = Ho, Wo
    return out


def roof_time_s(flops, nbytes, hbm):
    return max(flops / (FP32_PEAK_TFLOPS * 1e12), nbytes / (hbm * 1e9))


# ----------------------------------------------------------------------------- clocks


class ClockSampler:
    """nvidia-smi sampling (200 ms) during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": float(rows[0][2]) if rows[0][2].replace(".", "").isdigit() else None,
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------------------------- CPU oracle baseline


def cpu_oracle_sample(spec, target_s: float, seed: int = 0):
    """Time the fp64 oracle on a bounded sample of the workload: every op, restricted to its first
    ceil(f * Co) filters (at least one per oracle thread), on a seeded input of the op's input shape
    (one per distinct shape).  f is calibrated on the first
    pruned op so that the whole sample takes about target_s seconds.  Returns (GFLOP/s, f, seconds)."""
    from oracle import oracle as orc
    from paper_2004_11250_gb300 import synth
    rng = np.random.default_rng(seed)
    shapes = op_shapes(spec)
    total_flops = sum(s["flops"] for s in shapes)
    by_shape = {}  # one seeded input per distinct input shape (the timing does not depend on the values)
    inputs = []
    for s in shapes:
        key = (s["N"], s["Ci"], s["H"], s["W"])
        if key not in by_shape:
            by_shape[key] = rng.uniform(-1, 1, key).astype(np.float32)
        inputs.append(by_shape[key])
    pats = [orc.pattern_ids(op.layer.w, op.layer.mask, op.layer.taps) if isinstance(op.layer, synth.PrunedLayer)
            else None for op in spec.ops]

    nthr = max(1, orc.num_threads())

    def run(k, f):
        # at least one filter per oracle thread (it runs in parallel over images and filters)
        L = spec.ops[k].layer
        co = min(L.Co, max(nthr, int(math.ceil(f * L.Co))))
        t0 = time.perf_counter()
        if pats[k] is not None:
            orc.conv_pruned(inputs[k], L.w[:co], pats[k][:co], L.taps, None if L.bias is None else L.bias[:co])
        else:
            orc.conv_dense(inputs[k], L.w[:co], None if L.bias is None else L.bias[:co])
        dt = time.perf_counter() - t0
        s = shapes[k]
        return dt, s["flops"] * co / s["Co"]

    k0 = max(range(len(shapes)), key=lambda k: shapes[k]["flops"])
    f0 = min(1.0, nthr / max(1, shapes[k0]["Co"]))
    dt, fl = run(k0, f0)
    rate = fl / max(dt, 1e-9)
    f = min(1.0, target_s * rate / total_flops)
    t_all, fl_all, frames = 0.0, 0.0, 0
    while True:  # whole passes over the ops; repeat small workloads until about target_s of work
        for k in range(len(shapes)):
            dt, fl = run(k, f)
            t_all += dt
            fl_all += fl
        frames += 1
        if f < 1.0 or t_all >= 0.8 * target_s or frames >= 1000:
            break
    return fl_all / t_all / 1e9, f * frames, t_all


# ----------------------------------------------------------------------------- GPU timing


def time_net(dn, x, y, steps, warmup, flush, stream):
    import torch
    for _ in range(warmup):
        flush.zero_()
        dn.run(x, y, stream)
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for e0, e1 in evs:
        flush.zero_()
        e0.record(stream)
        dn.run(x, y, stream)
        e1.record(stream)
    torch.cuda.synchronize()
    return [e0.elapsed_time(e1) for e0, e1 in evs]


def time_ops(dn, acts, steps, flush, stream):
    """Average duration (ms) of every op's kernel launch alone, L2 flushed before each launch."""
    import torch
    from paper_2004_11250_gb300 import runner
    spec = dn.spec
    res = []
    for k, (op, L) in enumerate(zip(spec.ops, dn.layers)):
        xin, out = acts[k], acts[k + 1]
        skip = acts[op.skip_from] if op.skip_from >= 0 else None
        N, _, H, W = xin.shape
        flags = runner.op_flags(op)
        L.forward(xin, out, skip, N, H, W, flags, stream)
        ts = []
        for _ in range(steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            L.forward(xin, out, skip, N, H, W, flags, stream)
            e1.record(stream)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1))
        res.append(sum(ts) / len(ts))
    return res


def time_ops_in_frame(dn, acts, steps, flush, stream):
    """Median duration (ms) of every op inside a frame: the ops launched back to back in frame order on
    the stream with a CUDA event between consecutive ops, L2 flushed once before each frame (as in the
    timed frames).  The events break the overlap of one op's tail with the next op's start that the
    frame's graph gets from programmatic dependent launch, so the sum is a little above the frame time."""
    import torch
    from paper_2004_11250_gb300 import runner
    spec = dn.spec
    n = len(spec.ops)
    args = []
    for k, (op, L) in enumerate(zip(spec.ops, dn.layers)):
        xin = acts[k]
        N, _, H, W = xin.shape
        args.append((L, xin, acts[k + 1], acts[op.skip_from] if op.skip_from >= 0 else None, N, H, W,
                     runner.op_flags(op)))
    per = [[] for _ in range(n)]
    for rep in range(steps + 2):
        flush.zero_()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
        ev[0].record(stream)
        for k, (L, xin, out, skip, N, H, W, flags) in enumerate(args):
            L.forward(xin, out, skip, N, H, W, flags, stream)
            ev[k + 1].record(stream)
        ev[-1].synchronize()
        if rep >= 2:  # two warm frames first
            for k in range(n):
                per[k].append(ev[k].elapsed_time(ev[k + 1]))
    return [statistics.median(v) for v in per]


def time_graph_of_launches(dn, acts, reps, steps, stream):
    """Per-launch time (ms) of op 0 replayed back to back: one CUDA graph of `reps` launches of the op on the
    same buffers (no L2 flush between them: weights and input stay warm), replayed `steps` times.  With a
    launch far shorter than the launch latency this separates the kernel's own time from the latency of a
    lone launch."""
    import torch
    from paper_2004_11250_gb300 import runner
    op, L = dn.spec.ops[0], dn.layers[0]
    xin, out = acts[0], acts[1]
    N, _, H, W = xin.shape
    flags = runner.op_flags(op)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for _ in range(reps):
            L.forward(xin, out, None, N, H, W, flags, torch.cuda.current_stream())
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        g.replay()
    e1.record(stream)
    e1.synchronize()
    return e0.elapsed_time(e1) / (steps * reps)


def traffic_from_profile(kernel_hash: str, kernel: str = None, precision: str = "tf32x3"):
    """Per-launch DRAM bytes (read + write) from the committed ncu summary of the VGG-16 frame in this
    tensor-core arithmetic, of one kernel (average over its launches in the frame) or of all the frame's
    convs, if that summary was taken on the current kernel source."""
    name = "ppconv_vgg16_dram_traffic.txt" if precision == "tf32x3" else f"ppconv_vgg16_dram_traffic_{precision}.txt"
    path = os.path.join(ROOT, "profiles", name)
    try:
        kv = {}
        for line in open(path):
            if ":" in line:
                k, v = line.split(":", 1)
                kv[k.strip()] = v.strip()
        if kv.get("kernel_source_sha256") != kernel_hash:
            return None
        key = f"dram_bytes_per_launch_avg[{kernel}]" if kernel else "dram_bytes_per_launch_avg"
        return float(kv[key])
    except Exception:
        return None


def code_lines(text: str) -> str:
    """The source without its // comments and blank lines (the sources use no // inside strings)."""
    out = []
    for line in text.splitlines():
        k = line.find("//")
        line = (line if k < 0 else line[:k]).rstrip()
        if line:
            out.append(line)
    return "\n".join(out)


def kernel_source_hash():
    """sha256 over the conv kernel sources' code, comments left out (a profile taken on other code is
    stale; an edit of a comment does not change the kernels)."""
    import hashlib
    h = hashlib.sha256()
    for name in ("conv.cu", "conv_tm.cu", "conv_tc.cu", "conv_tcf.cu", "conv_direct.cu", "tc_ptx.cuh", "internal.h"):
        with open(os.path.join(ROOT, "paper_2004_11250_gb300", "csrc", name), encoding="utf-8") as f:
            h.update(code_lines(f.read()).encode())
    return h.hexdigest()


TENSOR_PEAKS = {}  # filled by main(): {"tf32": TFLOP/s, "f16": TFLOP/s} measured by pp_peak_probe


def tensor_view(shapes, kern, op_ms, pruned, f16=False):
    """Tensor-pipe view of the pruned ops that run on a tensor-core kernel: their dense 9-tap contraction
    in 3 passes (hi*hi, lo*hi, hi*lo) per second against the measured kind::tf32 (or kind::f16) MMA
    peak; None without such ops."""
    tc_ops = [k for k in pruned if kern[k] in ("ppconv_tc_kernel", "ppconv_tcf_kernel")]
    kind = "f16" if f16 else "tf32"
    if not tc_ops or kind not in TENSOR_PEAKS:
        return None
    tf = sum(3 * 2 * shapes[k]["N"] * shapes[k]["Ci"] * shapes[k]["Co"] * 9 * shapes[k]["H"] * shapes[k]["W"]
             for k in tc_ops)
    tt = sum(op_ms[k] for k in tc_ops) * 1e-3
    tpk = TENSOR_PEAKS[kind]
    return {"bound": "tensor", "ops": len(tc_ops), "achieved": round(tf / tt / 1e12, 2), "peak": round(tpk, 1),
            "unit": f"TFLOP/s ({kind}, dense 9-tap, 3 passes)", "frac": round(tf / tt / 1e12 / tpk, 4),
            "peak_source": f"measured: pp_peak_probe kind::{kind} MMA (M 128, N 256, K {16 if f16 else 8}), this run"}


def bench_config(name, steps, warmup, flush, stream, hbm, fold_too=False, precision=0):
    """ms/frame, GFLOP/s and per-op roofline fractions (op times taken inside the frame) of one workload,
    for the all-configs table; with fold_too also the frame time with the filter reorder folded into the
    next layer (Section 3 matrix reorder; activations between layers in reordered channel order)."""
    import torch
    from paper_2004_11250_gb300 import runner
    spec = workload(name)
    dn = runner.DeviceNet(spec, use_graph=True, precision=precision)
    try:
        x = torch.from_numpy(spec.x).cuda()
        y = torch.empty(dn.out_shape, device="cuda")
        ts = time_net(dn, x, y, steps, warmup, flush, stream)
        shapes = op_shapes(spec)
        acts = dn.run_layerwise(x)
        op_ms = time_ops_in_frame(dn, acts, max(3, steps // 2), flush, stream)
        flops = sum(s["flops"] for s in shapes)
        ms = statistics.median(ts)
        fr = [roof_time_s(s["flops"], s["bytes"], hbm) / (t * 1e-3) for s, t in zip(shapes, op_ms)]
        pr = [f for s, f in zip(shapes, fr) if s["pruned"]]
        del acts
        from paper_2004_11250_gb300 import ppconv as pp
        per_op = [KERNEL_NAMES.get(pp.pp_layer_kernel(L.handle), "?") if not L.dense else "dense" for L in dn.layers]
        kern = sorted(set(k for k in per_op if k != "dense"))
        tv = tensor_view(shapes, per_op, op_ms, [k for k, s in enumerate(shapes) if s["pruned"]], f16=precision == 1)
        graph_us = None
        if name == "single":
            graph_us = round(time_graph_of_launches(dn, dn.run_layerwise(x), 20, 10, stream) * 1e3, 3)
        res = {"ms_per_frame": round(ms, 4), "gflops": round(flops / (ms * 1e-3) / 1e9, 1), "kernels": kern,
               "op_us_in_frame": [round(t * 1e3, 2) for t in op_ms],
               "roofline_frac_min_pruned_op": round(min(pr), 3) if pr else None,
               "roofline_frac_median_pruned_op": round(statistics.median(pr), 3) if pr else None,
               "tensor_tflops": tv["achieved"] if tv else None, "tensor_frac": tv["frac"] if tv else None}
        if graph_us is not None:
            res["us_per_launch_graph_of_20"] = graph_us
            res["roofline_frac_graph_of_20"] = round(roof_time_s(shapes[0]["flops"], shapes[0]["bytes"], hbm)
                                                     / (graph_us * 1e-6), 4)
    finally:
        dn.close()
    if fold_too:
        dn = runner.DeviceNet(spec, use_graph=True, fold_perm=True)
        try:
            x = torch.from_numpy(spec.x).cuda()
            y = torch.empty(dn.out_shape, device="cuda")
            ts = time_net(dn, x, y, steps, warmup, flush, stream)
            res["ms_per_frame_perm_folded"] = round(statistics.median(ts), 4)
        finally:
            dn.close()
    return res


def bench_sweep(steps, flush, stream, hbm, precision=0):
    """Sweep workload: per point (C, P, keep) one layer at 8x56x56, its kernel autotuned at that shape;
    returns summary + per-point roofline fractions and the kernel used."""
    import torch
    from paper_2004_11250_gb300 import runner, synth
    fracs, total_ms = {}, 0.0
    for (C, P, keep) in synth.cfg4_points():
        spec = synth.cfg4_point(C, P, keep)
        L = runner.DeviceLayer(spec.ops[0].layer, precision=precision)
        try:
            from paper_2004_11250_gb300 import ppconv as pp
            pp.pp_layer_autotune(L.handle, 8, 56, 56, 0, stream)  # kernel choice at this shape, before timing
            x = torch.from_numpy(spec.x).cuda()
            y = torch.empty((8, C, 56, 56), device="cuda")
            L.forward(x, y, None, 8, 56, 56, 0, stream)
            ts = []
            for _ in range(steps):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                L.forward(x, y, None, 8, 56, 56, 0, stream)
                e1.record(stream)
                e1.synchronize()
                ts.append(e0.elapsed_time(e1))
            t = statistics.median(ts)
            s = op_shapes(spec)[0]
            fracs[f"C{C}_P{P}_k{keep}"] = round(roof_time_s(s["flops"], s["bytes"], hbm) / (t * 1e-3), 3)
            total_ms += t
        finally:
            L.close()
    v = list(fracs.values())
    return {"points": len(v), "ms_total": round(total_ms, 3), "roofline_frac_min": min(v),
            "roofline_frac_median": statistics.median(v), "per_point": fracs}


# ----------------------------------------------------------------------------- main


def dist_setup(args):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        backend = "nccl" if args.impl != "reference" else "gloo"
        dist.init_process_group(backend)
    return ws, rank, local


def max_over_ranks(t_ms, ws, device):
    """The slowest rank's time (every rank gets it); a collective only when ws > 1."""
    if ws == 1:
        return float(t_ms)
    import torch
    t = torch.tensor([float(t_ms)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_value(ws, flops_frame, steps, t_total_ms):
    """Whole-job throughput in GFLOP/s: every rank ran `steps` frames of `flops_frame` surviving FLOPs
    (replicas; weak scaling), timed by the slowest rank."""
    return ws * flops_frame * steps / (t_total_ms * 1e-3) / 1e9


def run_reference(args, ws, rank):
    if rank != 0:
        return
    from oracle import oracle as orc
    spec = workload(args.workload)
    per_step = max(1.0, min(8.0, 150.0 / max(1, args.steps + args.warmup)))
    for _ in range(args.warmup):
        cpu_oracle_sample(spec, per_step)
    vals, fs = [], []
    t0 = time.perf_counter()
    for _ in range(args.steps):
        v, f, _ = cpu_oracle_sample(spec, per_step)
        vals.append(v)
        fs.append(f)
    wall = time.perf_counter() - t0
    value = statistics.median(vals)
    flops = sum(s["flops"] for s in op_shapes(spec))
    line = {
        "impl": "reference", "metric": metric_name(args.workload), "value": round(value, 3), "unit": "GFLOP/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(flops / (value * 1e9) * 1e3, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_dict(args.workload),
        "cpu_baseline": {"value": round(value, 3), "unit": "GFLOP/s", "cores": orc.num_threads(), "kind": "oracle",
                         "sample": f"per step: every op of the workload on {statistics.median(fs):.4f} of its filters "
                                   f"(at least one per oracle thread; frames when >= 1), seeded inputs; "
                                   f"{wall:.1f} s for {args.steps} steps"},
        "e2e": {"value": round(value, 3), "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def metric_name(w):
    names = {"vgg16": "VGG-16 pattern-pruned conv trunk 1x3x224x224",
             "single": "single pattern-pruned layer 1x16x32x32",
             "style": "style-transfer residual trunk 1x128x128x128",
             "vdsr": "VDSR-shaped SR stack 1x1x720x1280"}
    if w.startswith("sweep:"):
        C, P, keep = w.split(":")[1:]
        name = f"sweep point 8x{C}x56x56, C_in = C_out = {C}, {P} patterns, keep {keep}"
    elif w.startswith("op:"):
        base, k = w.split(":")[1:]
        name = f"op {k} of the {names[base]} alone"
    else:
        name = names[w]
    return f"effective GFLOP/s (surviving MACs), {name}, fp32"


def config_dict(w):
    from paper_2004_11250_gb300 import synth
    spec = workload(w)
    return {"workload": metric_name(w).split(", ")[1], "batch": int(spec.x.shape[0]),
            "input": list(spec.x.shape), "convs": len(spec.ops),
            "surviving_gflop_per_frame": round(spec.surviving_flops() / 1e9, 4),
            "patterns": (f"{w.split(':')[2]} seed-chosen centre+3-neighbour patterns" if w.startswith("sweep:")
                         else "8 fixed centre+3-neighbour patterns"),
            "l2": "flushed between steps (512 MiB write)"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="vgg16",
                    help="vgg16 (default), single, style, vdsr, sweep:C:P:keep (one point of the sweep), or "
                         "op:<workload>:<k> (op k of a network alone, to profile one layer)")
    ap.add_argument("--precision", default="tf32x3", choices=["tf32x3", "f16x3"],
                    help="arithmetic of the tensor-core kernels for the timed frames (pp_layer_set_precision)")
    ap.add_argument("--fold-perm", action="store_true",
                    help="fold each layer's filter reorder into the next layer for the timed frames")
    ap.add_argument("--no-configs", action="store_true", help="skip the all-configs table")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--kernels", default="",
                    help="comma list, one per op (tm, reg, tc, flat, flat:R:S, direct, or auto to keep the autotuned "
                         "choice): pins each op's kernel (and for flat:R:S the flat kernel's rows per tile and "
                         "split) after pp_net_finalize, e.g. to profile the selection of an earlier run")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    ws, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return

    import torch
    torch.cuda.set_device(local)
    from paper_2004_11250_gb300 import build
    build.build()
    from paper_2004_11250_gb300 import runner
    hbm, hbm_src = hbm_peak_gbs()
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)  # flushes, copies and kernels all ordered on one stream
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    # measured peaks of this GPU (the roofline denominators), before anything is timed
    peaks = measure_peaks()
    set_fp32_peak(peaks["fp32_ffma"]["tflops"])
    TENSOR_PEAKS["tf32"] = peaks["tf32_mma"]["tflops"]
    TENSOR_PEAKS["f16"] = peaks["f16_mma"]["tflops"]
    spec = workload(args.workload)
    shapes = op_shapes(spec)
    flops_frame = sum(s["flops"] for s in shapes)
    precision = 1 if args.precision == "f16x3" else 0
    dn = runner.DeviceNet(spec, use_graph=True, fold_perm=args.fold_perm, precision=precision)
    if args.kernels:
        from paper_2004_11250_gb300 import ppconv as pp
        ids = {"tm": pp.PP_KERNEL_TMEM, "reg": pp.PP_KERNEL_REGISTER, "tc": pp.PP_KERNEL_TC,
               "flat": pp.PP_KERNEL_TC_FLAT, "direct": pp.PP_KERNEL_DIRECT}
        names = args.kernels.split(",")
        if len(names) != len(dn.layers):
            raise SystemExit(f"--kernels needs {len(dn.layers)} entries")
        for L, k, op, sh in zip(dn.layers, names, spec.ops, shapes):
            if k != "auto" and not L.dense:
                pp.pp_layer_set_kernel(L.handle, ids[k.split(":")[0]])
                if k.startswith("flat:"):
                    R, S = (int(v) for v in k.split(":")[1:])
                    pp.pp_layer_pin_flat_geometry(L.handle, sh["N"], sh["H"], sh["W"], runner.op_flags(op), R, S)
    x = torch.from_numpy(spec.x).cuda()
    y = torch.empty(dn.out_shape, device="cuda")
    torch.cuda.synchronize()

    clocks = ClockSampler(local)
    with torch.cuda.stream(stream):
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        clocks.start()
        ts = time_net(dn, x, y, args.steps, args.warmup, flush, stream)
        torch.cuda.synchronize()
        clk = clocks.stop()
    t_total_ms = max_over_ranks(sum(ts), ws, "cuda")
    if ws > 1:
        torch.distributed.barrier()
    ms_per_step = t_total_ms / args.steps
    value = job_value(ws, flops_frame, args.steps, t_total_ms)

    # per-op kernel durations inside the frame (op by op in frame order, events between the ops, L2 flushed
    # once per frame) -> roofline of the pruned convs; the same ops launched alone (L2 flushed before each
    # launch) are reported beside them
    acts = dn.run_layerwise(x, stream)
    torch.cuda.synchronize()
    op_ms = time_ops_in_frame(dn, acts, max(5, args.steps // 2), flush, stream)
    op_ms_alone = time_ops(dn, acts, max(5, args.steps // 2), flush, stream)
    del acts
    pruned = [k for k, s in enumerate(shapes) if s["pruned"]]
    kf = sum(shapes[k]["flops"] for k in pruned)
    kt = sum(op_ms[k] for k in pruned) * 1e-3
    achieved_all = kf / kt / 1e12
    # which kernel each op runs (autotuned by pp_net_finalize) and the tensor-pipe view
    from paper_2004_11250_gb300 import ppconv as pp
    kern = [KERNEL_NAMES.get(pp.pp_layer_kernel(L.handle), "?") if not L.dense else "ppconv_kernel (dense)"
            for L in dn.layers]
    # the flat kernel's tile geometry per op ("R:S", as --kernels flat:R:S takes it)
    geo = []
    for L, op, sh in zip(dn.layers, spec.ops, shapes):
        g = None
        if not L.dense and pp.pp_layer_kernel(L.handle) == pp.PP_KERNEL_TC_FLAT:
            R, S = pp.pp_layer_flat_geometry(L.handle, sh["N"], sh["H"], sh["W"], runner.op_flags(op))
            g = f"{R}:{S}" if R else "model"
        geo.append(g)
    tensor = tensor_view(shapes, kern, op_ms, pruned, f16=precision == 1)
    # the dominant kernel (most device time over the pruned ops): its surviving FLOPs per launch over
    # its mean launch duration, against the FP32 roofline of the method
    by_kern = {}
    for k in pruned:
        f, t = by_kern.get(kern[k], (0.0, 0.0))
        by_kern[kern[k]] = (f + shapes[k]["flops"], t + op_ms[k] * 1e-3)
    dom = max(by_kern, key=lambda n: by_kern[n][1])
    dom_ops = [k for k in pruned if kern[k] == dom]
    achieved = by_kern[dom][0] / by_kern[dom][1] / 1e12
    achieved_alone = sum(shapes[k]["flops"] for k in dom_ops) / (sum(op_ms_alone[k] for k in dom_ops) * 1e-3) / 1e12
    traffic = traffic_from_profile(kernel_source_hash(), dom, args.precision)
    # the dominant kernel's compulsory bytes per launch (its ops' inputs, outputs and compact weights)
    algo_bytes = sum(shapes[k]["bytes"] for k in dom_ops) / len(dom_ops)
    # the same op times scaled so that they add up to the graph frame (the events above break the overlap
    # of consecutive ops that programmatic dependent launch gives inside the graph): an apportioned view
    scale = ms_per_step / sum(op_ms)
    achieved_graph = achieved / scale
    layer_fracs = [round(roof_time_s(s["flops"], s["bytes"], hbm) / (t * 1e-3), 3) for s, t in zip(shapes, op_ms)]

    # end to end through the public API with host buffers
    xh = torch.from_numpy(spec.x).pin_memory()
    yh = torch.empty(dn.out_shape, dtype=torch.float32).pin_memory()
    for _ in range(args.warmup):
        dn.run_host(xh, yh, stream)
    e2e_t = []
    for _ in range(args.steps):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        dn.run_host(xh, yh, stream)
        e2e_t.append(time.perf_counter() - t0)
    e2e_value = ws * flops_frame / statistics.median(e2e_t) / 1e9

    configs = None
    if not args.no_configs and rank == 0:
        configs = {}
        for name in ("single", "vgg16", "style", "vdsr"):
            configs[name] = bench_config(name, 10, 3, flush, stream, hbm, fold_too=name in ("vgg16", "style"))
            if name != "single":  # the single 16-channel layer has no tensor-core layout
                configs[name]["f16x3"] = bench_config(name, 10, 3, flush, stream, hbm, precision=1)
        configs["sweep"] = bench_sweep(5, flush, stream, hbm)
        configs["sweep"]["f16x3"] = bench_sweep(5, flush, stream, hbm, precision=1)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu:
        from oracle import oracle as orc
        v, f, secs = cpu_oracle_sample(spec, args.cpu_seconds)
        cpu = {"value": round(v, 3), "unit": "GFLOP/s", "cores": orc.num_threads(), "kind": "oracle",
               "sample": (f"every op on its first {f:.4f} of filters, at least one per thread (seeded inputs), {secs:.1f} s" if f < 1 else
                          f"{f:.0f} whole frames of every op (seeded inputs), {secs:.1f} s")}
        if configs is not None:
            # the oracle beside every workload, same cores, a bounded sample each (the sweep: its middle point)
            from paper_2004_11250_gb300 import synth
            for name in configs:
                if name == args.workload:
                    cv, cf, cs = v, f, secs
                else:
                    cspec = synth.cfg4_point(256, 8, 0.35) if name == "sweep" else workload(name)
                    cv, cf, cs = cpu_oracle_sample(cspec, CONFIG_CPU_SECONDS)
                configs[name]["cpu_oracle"] = {
                    "gflops": round(cv, 3), "cores": orc.num_threads(),
                    "sample": ("sweep point C256 P8 keep 0.35: " if name == "sweep" else "")
                    + (f"every op on its first {cf:.4f} of filters (at least one per thread), {cs:.1f} s" if cf < 1 else
                       f"{cf:.0f} whole frames, {cs:.1f} s")}

    if rank == 0:
        line = {
            "metric": metric_name(args.workload), "value": round(value, 2), "unit": "GFLOP/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded; shapes and distributions of the workload, no dataset or trained weights)",
            "config": dict(config_dict(args.workload), perm_folded=bool(args.fold_perm),
                           tensor_core_precision=args.precision),
            "e2e": {"value": round(e2e_value, 2), "unit": "GFLOP/s", "h2d_bytes_per_step": int(xh.numel() * 4),
                    "d2h_bytes_per_step": int(yh.numel() * 4), "ms_per_step": round(statistics.median(e2e_t) * 1e3, 4)},
            "gpu_launches": len(spec.ops) * args.steps,
            "roofline": {"bound": "alu", "achieved": round(achieved, 3), "peak": round(FP32_PEAK_TFLOPS, 2),
                         "unit": "TFLOP/s", "frac": round(achieved / FP32_PEAK_TFLOPS, 4), "traffic": traffic,
                         "algorithmic_bytes": int(algo_bytes),
                         "frac_of_derived_peak": round(achieved / peaks["derived_fp32_tflops"], 4),
                         "kernel": f"{dom} ({len(dom_ops)} of the {len(pruned)} pruned convs, "
                                   f"{100 * by_kern[dom][1] / kt:.0f}% of their in-frame device time)",
                         "timing": "op by op in frame order, CUDA events between the ops on the launching "
                                   "stream, L2 flushed once per frame; median over frames",
                         "op_us_in_frame": [round(t * 1e3, 2) for t in op_ms],
                         "op_flops": [int(s["flops"]) for s in shapes],
                         "dominant_ops": dom_ops,
                         "frame_ms_op_by_op": round(sum(op_ms), 4),
                         "graph_apportioned": {"achieved": round(achieved_graph, 3),
                                               "frac": round(achieved_graph / FP32_PEAK_TFLOPS, 4),
                                               "scale": round(scale, 4),
                                               "timing": "op_us_in_frame x (ms_per_step / frame_ms_op_by_op): "
                                                         "the in-frame op times apportioned to the graph frame"},
                         "alone": {"achieved": round(achieved_alone, 3),
                                   "frac": round(achieved_alone / FP32_PEAK_TFLOPS, 4),
                                   "op_us": [round(t * 1e3, 2) for t in op_ms_alone],
                                   "timing": "each op launched alone, L2 flushed before every launch"},
                         "all_pruned_ops": {"achieved": round(achieved_all, 3),
                                            "frac": round(achieved_all / FP32_PEAK_TFLOPS, 4),
                                            "traffic": traffic_from_profile(kernel_source_hash(), None, args.precision),
                                            "kernels": sorted(by_kern)},
                         "tensor": tensor,
                         "peak_source": (f"measured: pp_peak_probe FFMA, {peaks['fp32_ffma']['tflops']} TFLOP/s at "
                                         f"{peaks['fp32_ffma']['sm_mhz']} MHz (this run)"),
                         "peaks": peaks,
                         "hbm_peak_gbs": hbm, "hbm_peak_source": hbm_src},
            "layer_roofline_frac": layer_fracs,
            "layer_kernels": kern,
            "layer_flat_geometry": geo,
            "clocks": clk,
            "cpu_baseline": cpu,
            "configs": configs,
        }
        print(json.dumps(line), flush=True)
    dn.close()
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
