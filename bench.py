#!/usr/bin/env python
"""Throughput of 8-bit quantized LSTM acoustic-model inference on GB300 (one JSON line on stdout).

A step is one qnn_lstm_forward over one batch of synthetic frames: per-frame activation
quantization, the integer products of every layer, recovery fused with the gates and the cell
update, the 8-bit output layer and its softmax. Default workload: the largest single-GPU one, a
projected LSTM (LSTMP) of 5 layers of 2048 cells with 512-unit projections, 80-dimensional input
frames, an 8192-class 8-bit softmax layer, batch 1024, T = 1000 frames. The same line also
carries the standalone quantized product at 16384 x 8192 x 8192 (`int8_gemm`) and the batch-1
5 x 500-cell workload (`batch1`).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl reference]

N > 1 runs under torchrun: every rank runs its own replica on its own batch (the sequences are
independent; there is no collective on the data path), and the value is the frames of all ranks
divided by the slowest rank's time. `--impl reference` times the CPU oracle instead, on a bounded
sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_1607_04683_gb300 import inputs  # noqa: E402

METRIC = "quantized LSTM frames/sec at batch B; int8 GEMM TOPS as % of GB300 int8 peak"
DEFAULT_WORKLOAD = inputs.LSTMP_5x2048P512_B1024.name
GEMM_SHAPE = inputs.QmatmulShape(16384, 8192, 8192)  # the largest product of the standalone sweep
L2_FLUSH_BYTES = 512 << 20  # > 129 MB L2


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(inputs.LSTM_WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true", help="skip the int8_gemm and batch1 keys")
    ap.add_argument("--sweep", action="store_true", help="standalone quantized matmul sweep instead")
    ap.add_argument("--shape", default="", help="with --sweep: one shape M,N,K only")
    ap.add_argument("--stream", action="store_true",
                    help="streaming server mode instead: per-frame latency and burst rate of a resident session")
    ap.add_argument("--frames", type=int, default=0,
                    help="profiling aid: run only the first N frames of the workload (same per-launch shapes)")
    ap.add_argument("--layers", type=int, default=0,
                    help="profiling aid: run only the first L layers of the workload (same per-launch shapes)")
    return ap.parse_args()


def max_over_ranks(ms: float, world: int, device=None) -> float:
    """The slowest rank's time: every rank contributes its own, all receive the maximum."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, max_ms: float, world: int) -> float:
    """Weak scaling: every rank runs its own copy of the workload (independent sequences; no data
    exchange), so the job processes world x units in the slowest rank's time."""
    return world * units_per_rank / (max_ms / 1e3)


def dist_info():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


# ---------------------------------------------------------------------------------------------
# algorithmic bytes of the dominant kernel (the persistent recurrent kernel), per launch
# ---------------------------------------------------------------------------------------------

def recurrent_bytes_per_launch(wl: inputs.LstmWorkload) -> int:
    """One launch runs the T recurrent steps of one layer over B sequences. Unique HBM bytes it
    must move: the layer's recurrent weight codes once (4H x R, plus P x H for a projection), and
    per frame of each sequence the recovered input product row (4H fp32) read, the previous
    output row (R fp32) read and the new output row (R fp32) written."""
    H, R, P = wl.hidden, wl.R, wl.proj
    weights = 4 * H * R + (P * H if P > 0 else 0)
    per_frame = 4 * H * 4 + 2 * R * 4
    return weights + wl.batch * wl.frames * per_frame


def small_ops_per_launch(wl: inputs.LstmWorkload) -> int:
    """Integer multiply-adds x 2 of one batch-of-few launch: every layer's input and recurrent
    products and the output layer's, for B T frames."""
    return ops_per_frame(wl) * wl.batch * wl.frames


def small_bytes_per_launch(wl: inputs.LstmWorkload) -> int:
    """Unique HBM bytes of one batch-of-few launch: every weight code once, the input frames,
    and the logits (or top-layer outputs) written."""
    H, R = wl.hidden, wl.R
    w = sum(4 * H * (wl.layer_in(l) + R) for l in range(wl.num_layers)) + wl.num_classes * R
    out = wl.num_classes if wl.num_classes > 0 else R
    return w + wl.batch * wl.frames * (wl.input_dim + out) * 4


def source_sha(sources) -> str:
    """Hash of the kernel's source files (the .cu and the headers its arithmetic comes from)."""
    h = hashlib.sha256()
    for name in sources:
        h.update(open(os.path.join(ROOT, "paper_1607_04683_gb300", "csrc", name), "rb").read())
    return h.hexdigest()[:16]


def gates_fused(wl) -> bool:
    """Whether the gate kernel computes the step's input product itself (the library's default for
    input widths up to 1024; QNN_TC_FUSE_X=0 turns it off)."""
    return os.environ.get("QNN_TC_FUSE_X") != "0" and max(wl.input_dim, wl.R) <= 1024


def gates_input_width(wl) -> float:
    """Input width of a layer, averaged over the layers (the first takes the frames, the rest R)."""
    return (wl.input_dim + (wl.num_layers - 1) * wl.R) / wl.num_layers


def gates_bytes_per_launch(wl) -> float:
    """Algorithmic DRAM bytes of one tensor-core recurrent step: the cell state read and written
    (B x H fp32 each way), the cell outputs written (B x H fp32), the recurrent input codes (B x R
    bytes) and the gate weight codes (4H x R bytes); plus, with the input product fused in, the
    step's input codes (B x I bytes) and the input weight codes (4H x I bytes), else the batched
    input products px (B x 4H fp32). I is averaged over the layers."""
    B, H, R = wl.batch, wl.hidden, wl.R
    common = 2 * B * H * 4 + B * H * 4 + B * R + 4 * H * R
    if gates_fused(wl):
        il = gates_input_width(wl)
        return float(common + B * il + 4 * H * il)
    return float(common + B * 4 * H * 4)


def traffic_record(kernel: str, workload: str, sources):
    """Per-launch DRAM bytes from the committed ncu summary, if taken on the current sources."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    try:
        sha = source_sha(sources)
        for line in open(path):
            f = line.split()
            if len(f) >= 4 and not line.startswith("#") and f[0] == kernel and f[1] == workload and f[3] == sha:
                return float(f[2])
    except OSError:
        pass
    return None


# ---------------------------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]
        return False

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
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------------------------
# CPU oracle timing (reference arm and cpu_baseline)
# ---------------------------------------------------------------------------------------------

def oracle_frames_per_s(wl, params, x, min_seconds=8.0, max_frames=None, reps_max=5):
    import oracle
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    xs = x[:1, : (max_frames or x.shape[1])]
    frames, t0 = 0, time.perf_counter()
    for _ in range(reps_max):
        oracle.lstm_forward(d, params, xs)
        frames += xs.shape[0] * xs.shape[1]
        if time.perf_counter() - t0 >= min_seconds:
            break
    dt = time.perf_counter() - t0
    return frames / dt, frames, dt


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def oracle_frames_per_s_threads(wl, params, x, frames, threads):
    """The oracle on `threads` sequences at once, one host thread each (its C calls release the
    interpreter lock, so they run in parallel; the oracle itself stays single-threaded per call)."""
    from concurrent.futures import ThreadPoolExecutor

    import oracle
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    seqs = [x[b % x.shape[0]: b % x.shape[0] + 1, :frames] for b in range(threads)]
    t0 = time.perf_counter()
    with ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(lambda xs: oracle.lstm_forward(d, params, xs), seqs))
    dt = time.perf_counter() - t0
    return threads * frames / dt, dt


def run_reference(args, wl, rank, world):
    """The CPU oracle as it stands, on the host's cores: each step runs the oracle on one sequence
    per core (one host thread each), every sequence cut to its first frames so that a step takes
    about a second or two."""
    if rank != 0:
        return 0
    cores = host_cores()
    params, x = wl.make(batch=min(wl.batch, cores))
    per_frame_ops = ops_per_frame(wl)
    sample_frames = max(1, min(wl.frames, int(2.0e9 / max(per_frame_ops, 1))))
    for _ in range(args.warmup):
        oracle_frames_per_s_threads(wl, params, x, sample_frames, cores)
    dt = 0.0
    for _ in range(args.steps):
        dt += oracle_frames_per_s_threads(wl, params, x, sample_frames, cores)[1]
    fps = args.steps * cores * sample_frames / dt
    sample = (f"per step: sequences 0..{cores - 1} (repeating past the batch), first {sample_frames} frames of "
              f"{wl.frames} each, one host thread per sequence")
    line = {
        "impl": "reference", "metric": METRIC, "value": fps, "unit": "frames/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u8", "data": "synthetic",
        "config": workload_config(wl),
        "cpu_baseline": {"value": fps, "unit": "frames/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": fps, "unit": "frames/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def ops_per_frame(wl) -> int:
    """Integer multiply-adds x 2 per frame: every layer's input and recurrent products, the
    projection, and the output layer."""
    H, R, P = wl.hidden, wl.R, wl.proj
    ops = 0
    for l in range(wl.num_layers):
        ops += 2 * 4 * H * (wl.layer_in(l) + R) + (2 * P * H if P > 0 else 0)
    if wl.num_classes > 0:
        ops += 2 * wl.num_classes * R
    return ops


def workload_config(wl):
    return {"workload": wl.name, "batch": wl.batch, "frames": wl.frames, "layers": wl.num_layers,
            "cells": wl.hidden, "proj": wl.proj, "input_dim": wl.input_dim, "classes": wl.num_classes,
            "output_layer": "8-bit" if wl.output_mode == 1 else ("float" if wl.output_mode == 2 else "none"),
            "activation_units": "per frame row", "weight_units": "per gate matrix",
            "l2": "flushed between timed steps (512 MiB write)"}


# ---------------------------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------------------------

def run_ours(args, wl, rank, world, local):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_1607_04683_gb300 import build as qbuild, qnn

    if not qbuild.up_to_date():
        if rank == 0:
            qbuild.build()
        if world > 1:
            dist.barrier()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    params, x = wl.make()
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, torch.from_numpy(params).to(dev))
    xd = torch.from_numpy(x).to(dev)
    ycols = wl.num_classes if wl.num_classes > 0 else wl.R
    yd = torch.empty((wl.batch, wl.frames, ycols), dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(args.warmup):
        model.forward(xd, y=yd)
    torch.cuda.synchronize()
    st = qnn.device_status()
    if st != qnn.QNN_OK:
        raise RuntimeError(f"device status after warm-up: {st}")

    # ---- timed region: device-resident inputs ----
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        barrier()
        torch.cuda.synchronize()
        for i in range(args.steps):
            flush.zero_()
            evs[i][0].record(stream)
            model.forward(xd, y=yd)
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        barrier()
    step_ms = [a.elapsed_time(b) for a, b in evs]
    # Per-kernel durations: the same K steps again with CUDA events around every launch (events
    # between back-to-back launches lengthen the step, so the step time above is taken without).
    # The layers of a multi-layer LSTMP run as a wavefront on one stream each, where a kernel's
    # events would also span other layers' kernels running beside it; the instrumented replay runs
    # the layers one after the other (QNN_TC_WAVE=0: the same kernels on the same data), so each
    # launch's events time that kernel alone.
    qnn.profile_read()
    qnn.profile_enable(True)
    wave_env = os.environ.get("QNN_TC_WAVE")
    os.environ["QNN_TC_WAVE"] = "0"
    prof_ms = 0.0  # the instrumented steps' own duration: a kernel's share of the step is taken from it
    for i in range(args.steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        model.forward(xd, y=yd)
        b.record(stream)
        b.synchronize()
        prof_ms += a.elapsed_time(b)
    torch.cuda.synchronize()
    qnn.profile_enable(False)
    if wave_env is None:
        del os.environ["QNN_TC_WAVE"]
    else:
        os.environ["QNN_TC_WAVE"] = wave_env
    prof = qnn.profile_read()
    total_ms = max_over_ranks(sum(step_ms), world, dev)
    frames_per_step = wl.batch * wl.frames
    value = whole_job_rate(frames_per_step * args.steps, total_ms, world)

    # ---- end to end: pinned host buffers through the C ABI, copies inside the timed region ----
    x_host = torch.from_numpy(x).pin_memory()
    y_host = torch.empty((wl.batch, wl.frames, ycols), dtype=torch.float32).pin_memory()
    for _ in range(2):
        model.forward(x_host, y=y_host)
    torch.cuda.synchronize()
    e2e_ms = 0.0
    barrier()
    for i in range(args.steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        model.forward(x_host, y=y_host)
        b.record(stream)
        b.synchronize()
        e2e_ms += a.elapsed_time(b)
    barrier()
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    e2e_value = whole_job_rate(frames_per_step * args.steps, e2e_ms, world)
    ok = qnn.device_status() == qnn.QNN_OK
    if not ok:
        raise RuntimeError("device status reported an error during the timed steps")

    if rank != 0:
        return 0

    peaks, peak_kind = measured_peaks()
    kname = max(prof, key=lambda k: prof[k][1])
    launches, kms = prof[kname]
    avg_s = kms / launches / 1e3
    roofline = None
    share = kms / prof_ms if world == 1 else None
    if kname == "lstm_recurrent":
        alg = recurrent_bytes_per_launch(wl)
        ach = alg / avg_s / 1e9
        roofline = {"bound": "hbm", "kernel": kname, "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                    "frac": ach / peaks["hbm_gbs"], "peak_kind": peak_kind,
                    "traffic": traffic_record(kname, wl.name, ["lstm.cu", "qnn_device.cuh"]), "alg_bytes_per_launch": alg,
                    "avg_launch_ms": avg_s * 1e3, "share_of_step": share}
    elif kname == "lstm_small":
        # the whole stack in one launch; its arithmetic is the integer products of every layer and
        # of the output layer, which run as dp4a (u8 x u8 -> s32): roofline = the measured dp4a rate
        ops = small_ops_per_launch(wl)
        ach = ops / avg_s / 1e12
        dp4a_peak = qnn.measure_peak(1)
        roofline = {"bound": "alu", "kernel": kname, "achieved": ach, "peak": dp4a_peak, "unit": "TOP/s",
                    "frac": ach / dp4a_peak, "peak_kind": "measured (qnn_measure_peak dp4a)",
                    "traffic": traffic_record(kname, wl.name, ["lstm_small.cu", "qnn_device.cuh"]), "alg_ops_per_launch": ops,
                    "alg_bytes_per_launch": small_bytes_per_launch(wl), "hbm_frac":
                        small_bytes_per_launch(wl) / avg_s / 1e9 / peaks["hbm_gbs"],
                    "avg_launch_ms": avg_s * 1e3, "share_of_step": share}
        # a frame of a layer is a chain of dependent steps: its time against the measured floor of
        # the kernel's per-frame synchronisation (cluster exchange + hand-over, no arithmetic)
        cs = (wl.hidden + 31) // 32
        floor_us = qnn.measure_exchange_floor(cs, 20000)
        us_frame = avg_s * 1e6 / wl.frames
        roofline["latency"] = {"us_per_frame": us_frame, "floor_us_per_frame": floor_us,
                               "frac": floor_us / us_frame, "cluster_blocks": cs,
                               "floor_kind": "measured (qnn_measure_exchange_floor)"}
    elif kname == "lstm_gates_tc":
        # one recurrent step of one layer: the tcgen05 gate product (with the input product fused
        # in, the library's default) and the LSTM cell in its epilogue. Fused, the step moves few
        # bytes (no px) and its work is the 2 B 4H (R + I) operations of the two products: reported
        # against the fp16 tensor peak, with its HBM rate beside; unfused against HBM.
        alg = gates_bytes_per_launch(wl)
        gbs = alg / avg_s / 1e9
        flops = 2.0 * wl.batch * 4 * wl.hidden * (wl.R + (gates_input_width(wl) if gates_fused(wl) else 0))
        tfs = flops / avg_s / 1e12
        traffic = traffic_record(kname, wl.name, ["qgemm_tc.cu", "qnn_device.cuh", "tc_ptx.cuh"])
        if gates_fused(wl):
            # the kernel runs inside a long step (thousands of launches per pass): the sustained peak
            tpk = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
            roofline = {"bound": "tensor", "kernel": kname, "achieved": tfs, "peak": tpk,
                        "unit": "TFLOP/s", "frac": tfs / tpk,
                        "peak_kind": f"{peak_kind} (fp16/bf16 dense, sustained)",
                        "traffic": traffic, "alg_flops_per_launch": flops, "alg_bytes_per_launch": alg,
                        "hbm_gbs": gbs, "hbm_frac": gbs / peaks["hbm_gbs"], "input_product": "fused",
                        "avg_launch_ms": avg_s * 1e3, "share_of_step": share}
        else:
            roofline = {"bound": "hbm", "kernel": kname, "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "frac": gbs / peaks["hbm_gbs"], "peak_kind": peak_kind, "traffic": traffic,
                        "alg_bytes_per_launch": alg, "tensor_tflops": tfs, "tensor_frac": tfs / peaks["bf16_tflops"],
                        "input_product": "batched", "avg_launch_ms": avg_s * 1e3, "share_of_step": share}
    line = {
        "metric": METRIC, "value": value, "unit": "frames/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u8", "data": "synthetic", "config": workload_config(wl),
        "gpu_launches": sum(v[0] for v in prof.values()),
        "kernels": {k: {"launches": v[0], "ms": v[1]} for k, v in sorted(prof.items(), key=lambda kv: -kv[1][1])},
        "int8_tops": ops_per_frame(wl) * frames_per_step * args.steps / (total_ms / 1e3) / 1e12,
        "roofline": roofline,
        "e2e": {"value": e2e_value, "unit": "frames/s", "h2d_bytes_per_step": int(x.nbytes),
                "d2h_bytes_per_step": int(wl.batch * wl.frames * ycols * 4)},
        "clocks": clk.summary(),
        # how the library ran the layers in the timed steps (the kernels' own durations above come
        # from a replay with the layers in sequence)
        "layer_schedule": ("wavefront: one stream per layer" if wl.num_layers >= 2 and wl.batch >= 64 and
                           os.environ.get("QNN_TC_WAVE") != "0" else "sequential"),
    }
    if world == 1 and not args.no_extras:
        line["int8_gemm"] = gemm_metric(qnn, torch, peaks, peak_kind, flush, max(5, args.steps))
        line["batch1"] = batch1_metric(qnn, torch, dev, flush, args.steps, args.warmup)
    if world == 1 and not args.no_cpu_baseline:
        sample_frames = min(wl.frames, max(1, int(3.0e9 / ops_per_frame(wl))))
        fps, frames, dt = oracle_frames_per_s(wl, params, x, min_seconds=8.0, max_frames=sample_frames)
        line["cpu_baseline"] = {"value": fps, "unit": "frames/s", "cores": 1, "kind": "oracle",
                                "sample": f"sequence 0 frames 0..{sample_frames}"
                                          f", repeated: {frames} frames in {dt:.1f} s, single thread"}
        cores = host_cores()
        fps_mt, dt_mt = oracle_frames_per_s_threads(wl, params, x, sample_frames, cores)
        line["cpu_baseline_mt"] = {"value": fps_mt, "unit": "frames/s", "cores": cores, "kind": "oracle",
                                   "sample": f"sequences 0..{cores - 1}, frames 0..{sample_frames} each, one host "
                                             f"thread per sequence on {cores} cores (os.sched_getaffinity): "
                                             f"{cores * sample_frames} frames in {dt_mt:.1f} s"}
    print(json.dumps(line), flush=True)
    return 0


def gemm_metric(qnn, torch, peaks, peak_kind, flush, reps):
    """The standalone quantized product at its largest sweep shape, 16384 x 8192 x 8192, codes in
    and fp32 out (eq. 1 offsets and eq. 3 recovery in the epilogue): tera-operations per second of
    the tensor-core product kernel alone and of the whole qnn_qmatmul call (which also converts both
    operands' codes to centered fp16 on every call), against the measured fp16 tensor peak (the
    datapath the exact product runs on) and the measured peak of the warp-level u8 integer MMA."""
    shape = GEMM_SHAPE
    W, A = inputs.make_qmatmul_operands(shape)
    Ag, Wg = torch.from_numpy(A).cuda(), torch.from_numpy(W).cuda()
    del W, A
    cw, pw, cs = qnn.qnn_quantize(Wg, qnn.PER_MATRIX)
    ca, pa, ra = qnn.qnn_quantize(Ag, qnn.PER_MATRIX)
    del Ag, Wg
    Y = torch.empty((shape.M, shape.N), dtype=torch.float32, device="cuda")
    for _ in range(2):
        qnn.qnn_qmatmul(ca, pa, 0, ra, cw, pw, cs, out=Y)
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        qnn.qnn_qmatmul(ca, pa, 0, ra, cw, pw, cs, out=Y)
        b.record()
        b.synchronize()
        ts.append(a.elapsed_time(b) / 1e3)
    qnn.profile_read()
    qnn.profile_enable(True)
    for _ in range(reps):
        flush.zero_()
        qnn.qnn_qmatmul(ca, pa, 0, ra, cw, pw, cs, out=Y)
    torch.cuda.synchronize()
    qnn.profile_enable(False)
    prof = qnn.profile_read()
    assert qnn.device_status() == qnn.QNN_OK
    n, kms = prof["qgemm_tc"]
    t_kernel = kms / n / 1e3
    t_call = statistics.median(ts)
    ops = 2.0 * shape.M * shape.N * shape.K
    imma = qnn.measure_peak(0)
    pk = peaks["bf16_tflops"]  # a kernel timed alone: the burst peak
    del ca, cw, Y
    torch.cuda.empty_cache()
    return {"M": shape.M, "N": shape.N, "K": shape.K, "unit": "TOP/s",
            "datapath": "tcgen05 kind::f16 on centered codes (exact integer sums; sm_103a has no kind::i8)",
            "kernel_tops": ops / t_kernel / 1e12, "kernel_ms": t_kernel * 1e3,
            "call_tops": ops / t_call / 1e12, "call_ms": t_call * 1e3,
            "centering_ms": (prof["center_fp16"][1] / prof["center_fp16"][0]) if "center_fp16" in prof else None,
            "peak": pk, "peak_kind": f"{peak_kind} (fp16/bf16 dense, burst)",
            "frac_kernel": ops / t_kernel / 1e12 / pk, "frac_call": ops / t_call / 1e12 / pk,
            "mma_u8_peak_tops": imma, "vs_mma_u8_peak_kernel": ops / t_kernel / 1e12 / imma,
            "l2": "flushed before every timed call"}


def batch1_metric(qnn, torch, dev, flush, steps, warmup):
    """The batch-1 workload (5 x 500 cells, 2000 classes, T = 300): frames per second of whole
    forward passes, and the per-frame time of the batch-of-few kernel against the measured floor of
    its per-frame synchronisation."""
    wl = inputs.LSTM_5x500_B1
    params, x = wl.make()
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, torch.from_numpy(params).to(dev))
    xd = torch.from_numpy(x).to(dev)
    yd = torch.empty((1, wl.frames, wl.num_classes), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(max(3, warmup)):
        model.forward(xd, y=yd)
    torch.cuda.synchronize()
    ms = []
    for _ in range(steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        model.forward(xd, y=yd)
        b.record(stream)
        b.synchronize()
        ms.append(a.elapsed_time(b))
    qnn.profile_read()
    qnn.profile_enable(True)
    for _ in range(steps):
        model.forward(xd, y=yd)
    torch.cuda.synchronize()
    qnn.profile_enable(False)
    prof = qnn.profile_read()
    assert qnn.device_status() == qnn.QNN_OK
    n, kms = prof["lstm_small"]
    us_frame = kms / n * 1e3 / wl.frames
    floor = qnn.measure_exchange_floor((wl.hidden + 31) // 32, 20000)
    model.close()
    return {"workload": wl.name, "value": wl.frames * steps / (sum(ms) / 1e3), "unit": "frames/s",
            "ms_per_step": sum(ms) / steps, "steps": steps, "kernel": "lstm_small",
            "us_per_frame": us_frame, "floor_us_per_frame": floor, "latency_frac": floor / us_frame}


def run_sweep(args):
    """Standalone quantized matmul sweep (K = N in {512, 2048, 8192}, M in {1, 16, 256, 4096,
    16384}, per-matrix units): one JSON line per shape with the product's TOPS (codes in, fp32
    out), the fp32-in rate including the activation quantizer, and the quantizer's GB/s. L2 is
    flushed before every timed repetition."""
    import torch

    from paper_1607_04683_gb300 import build as qbuild, qnn
    qbuild.build()
    torch.cuda.set_device(0)
    peaks, peak_kind = measured_peaks()
    imma = qnn.measure_peak(0)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    reps = max(3, args.steps)

    def timed(fn):
        ts = []
        for _ in range(reps + 1):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            ts.append(a.elapsed_time(b))
        return statistics.median(ts[1:]) / 1e3

    shapes = inputs.QMATMUL_SWEEP
    if args.shape:
        M, N, K = (int(v) for v in args.shape.split(","))
        shapes = [inputs.QmatmulShape(M, N, K)]
    for shape in shapes:
        W, A = inputs.make_qmatmul_operands(shape)
        Ag, Wg = torch.from_numpy(A).cuda(), torch.from_numpy(W).cuda()
        cw, pw, cs = qnn.qnn_quantize(Wg, qnn.PER_MATRIX)
        ca, pa, ra = qnn.qnn_quantize(Ag, qnn.PER_MATRIX)
        Y = torch.empty((shape.M, shape.N), dtype=torch.float32, device="cuda")
        t_mm = timed(lambda: qnn.qnn_qmatmul(ca, pa, 0, ra, cw, pw, cs, out=Y))
        t_q = timed(lambda: qnn.qnn_quantize(Ag, qnn.PER_MATRIX))
        t_qr = timed(lambda: qnn.qnn_quantize(Ag, qnn.PER_ROW))

        def both():
            c, p, r = qnn.qnn_quantize(Ag, qnn.PER_MATRIX)
            qnn.qnn_qmatmul(c, p, 0, r, cw, pw, cs, out=Y)
        t_all = timed(both)
        ops = 2.0 * shape.M * shape.N * shape.K
        mm_bytes = shape.M * shape.K + shape.N * shape.K + 4 * shape.M * shape.N
        print(json.dumps({
            "sweep": "qmatmul", "M": shape.M, "N": shape.N, "K": shape.K,
            "qmatmul_tops": ops / t_mm / 1e12, "qmatmul_ms": t_mm * 1e3,
            "datapath": "tcgen05 fp16 (exact centered codes)" if shape.M >= 128 else "mma.sync u8",
            "frac_of_datapath_peak": ops / t_mm / 1e12 / (peaks["bf16_tflops"] if shape.M >= 128 else imma),
            "frac_of_measured_mma_u8_peak": ops / t_mm / 1e12 / imma, "mma_u8_peak_tops": imma,
            "f16_tensor_peak_tflops": peaks["bf16_tflops"],
            "qmatmul_gbs": mm_bytes / t_mm / 1e9,
            "fp32_in_tops": ops / t_all / 1e12, "quantize_ms": t_q * 1e3,
            "quantize_gbs_alg": 5.0 * shape.M * shape.K / t_q / 1e9,
            "quantize_rows_gbs_alg": (5.0 * shape.M * shape.K + 20.0 * shape.M) / t_qr / 1e9,
            "hbm_peak_gbs": peaks["hbm_gbs"],
            "peak_kind": peak_kind, "l2": "flushed"}), flush=True)
        del Ag, Wg, cw, ca, Y
        torch.cuda.empty_cache()
    if args.shape:
        return 0
    # the on-the-fly quantizer alone, per-row units, on activation matrices shaped like the LSTM
    # layers' inputs (T*B frames x width; all larger than L2)
    gen = torch.Generator(device="cuda").manual_seed(7)
    for rows, cols, what in ((1024000, 512, "LSTMP 5x2048p512 layer input, T=1000 B=1024"),
                             (128000, 500, "LSTM 5x500 layer input, T=500 B=256"),
                             (131072, 2048, "rows of 2048 (two passes)")):
        X = torch.randn((rows, cols), device="cuda", generator=gen) * 1.7 + 0.3
        t_qr = timed(lambda: qnn.qnn_quantize(X, qnn.PER_ROW))
        alg = 5.0 * rows * cols + 20.0 * rows
        print(json.dumps({"sweep": "quantize", "rows": rows, "cols": cols, "granularity": "per row",
                          "what": what, "ms": t_qr * 1e3, "gbs_alg": alg / t_qr / 1e9,
                          "frac_of_hbm": alg / t_qr / 1e9 / peaks["hbm_gbs"], "hbm_peak_gbs": peaks["hbm_gbs"],
                          "peak_kind": peak_kind, "l2": "flushed"}), flush=True)
        del X
        torch.cuda.empty_cache()
    return 0


def run_stream(args):
    """Streaming server mode on the batch-1 workload's model (5 x 500 cells, 2000 classes): a
    session pushes one frame and pulls its posteriors before the next (round-trip latency seen by
    the host, wall clock), then pushes and pulls bursts of 64 frames (sustained rate). Inputs from
    host memory, outputs to host memory; one JSON line per measurement."""
    import numpy as np
    import torch

    from paper_1607_04683_gb300 import build as qbuild, qnn
    qbuild.build()
    torch.cuda.set_device(0)
    wl = inputs.LSTM_5x500_B1
    params, x = wl.make()
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, torch.from_numpy(params).cuda())
    T = x.shape[1]
    chunk = 1024
    # for comparison, the same frame-by-frame use through the batch call: one qnn_lstm_forward of
    # one frame per step, state carried on the device, input and output in pinned host memory
    # (measured before the session opens: its resident kernel holds the SMs this call needs)
    hs = torch.zeros((wl.num_layers, 1, wl.R), dtype=torch.float32, device="cuda")
    cs = torch.zeros((wl.num_layers, 1, wl.hidden), dtype=torch.float32, device="cuda")
    xh = torch.from_numpy(x).pin_memory()
    yh = torch.empty((1, 1, wl.num_classes), dtype=torch.float32).pin_memory()
    cur = torch.cuda.current_stream()
    lat_f = []
    for t in range(T):
        t0 = time.perf_counter()
        model.forward(xh[:, t:t + 1], y=yh, h_state=hs, c_state=cs)
        cur.synchronize()
        lat_f.append(time.perf_counter() - t0)
    lat_f = np.array(lat_f[20:]) * 1e6
    print(json.dumps({"bench": "stream", "mode": "frame by frame through qnn_lstm_forward (1 frame per call)",
                      "model": wl.name, "frames": int(lat_f.size), "latency_us_median": float(np.median(lat_f)),
                      "latency_us_p99": float(np.percentile(lat_f, 99))}), flush=True)
    s = qnn.LstmStream(model, 1, chunk=chunk, idle_seconds=10.0)
    lat = []
    for t in range(T):
        t0 = time.perf_counter()
        s.push(x[:, t:t + 1])
        s.pull(1)
        lat.append(time.perf_counter() - t0)
    lat = np.array(lat[20:]) * 1e6  # past the first launch's start
    print(json.dumps({"bench": "stream", "mode": "frame by frame (push 1, pull 1)", "model": wl.name,
                      "frames": int(lat.size), "latency_us_median": float(np.median(lat)),
                      "latency_us_p99": float(np.percentile(lat, 99)), "latency_us_min": float(lat.min()),
                      "chunk": chunk, "io": "host memory (host-mapped buffers)"}), flush=True)
    burst = 64
    reps = 40
    t0 = time.perf_counter()
    for i in range(reps):
        xs = x[:, (i * burst) % (T - burst):(i * burst) % (T - burst) + burst]
        s.push(xs)
        s.pull(burst)
    dt = time.perf_counter() - t0
    st = s.close()
    print(json.dumps({"bench": "stream", "mode": f"bursts of {burst} frames", "model": wl.name,
                      "frames": burst * reps, "frames_per_s": burst * reps / dt, "status": int(st),
                      "chunk": chunk}), flush=True)
    return 0 if st == qnn.QNN_OK else 1


def main():
    args = parse()
    if args.sweep:
        return run_sweep(args)
    if args.stream:
        return run_stream(args)
    rank, world, local = dist_info()
    wl = inputs.LSTM_WORKLOADS[args.workload]
    if args.frames or args.layers:  # a cut of the named workload (its name says so)
        import dataclasses
        cut = {}
        if args.frames:
            cut["frames"] = min(args.frames, wl.frames)
        if args.layers:
            cut["num_layers"] = min(args.layers, wl.num_layers)
        wl = dataclasses.replace(wl, name=f"{wl.name}_cut_L{cut.get('num_layers', wl.num_layers)}"
                                          f"_T{cut.get('frames', wl.frames)}", **cut)
    if world > 1 and args.impl == "ours":
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    try:
        if args.impl == "reference":
            return run_reference(args, wl, rank, world)
        return run_ours(args, wl, rank, world, local)
    finally:
        if world > 1 and args.impl == "ours":
            import torch.distributed as dist
            if dist.is_initialized():
                dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
