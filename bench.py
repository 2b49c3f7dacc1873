#!/usr/bin/env python
"""Throughput of the slice -> mix -> deslice coupling on GB300 (one JSON line).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload large_g_bf16|...] [--no-cpu-baseline]

A step is one pass of the whole forward hot path (fs_slice_fwd -> fs_mix ->
fs_deslice_fwd through the C ABI) over one batch of the named synthetic
workload, default N = 1,048,576 points, H = 8, d = 32, G = 1024, bf16
(inputs 512 MiB each, larger than the 129 MB L2, so no flush is needed between
steps).  Metric: Mpoints/s of the whole job (B*N points per step per rank).

--workload train_bf16 (B = 2, N = 524,288, G = 512, the workload with an upstream
gradient) times a training step instead: the forward and then fs_deslice_bwd ->
fs_mix_bwd -> fs_slice_bwd, every gradient of the coupling, and reports that
step's Mpoints/s on its own line (metric "train step ...").

Multi-GPU: the workload is replicated (each rank runs its own full copy; no
collective on the data path), so scaling is weak.  Launched with torchrun for
N > 1; rank 0 prints the line.  --shard instead splits one coupling's points
over the ranks, with NCCL all-reduces of the slice partials (and, with an
upstream gradient, of d_tokens_mixed and the parameter gradients): strong
scaling (App. G.4).

--impl reference times the fp64 CPU oracle (the only reference this method
has) on the host cores, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "slice+deslice Mpoints/s (N=1M, G=1024, bf16) and % of roofline"
UNIT = "Mpoints/s"
TRAIN_METRIC = "train step (slice+mix+deslice forward and backward) Mpoints/s"


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# DRAM traffic per C-ABI call at the full large_g_bf16 workload (N = 1,048,576).
# Source: ncu dram__bytes_read.sum + dram__bytes_write.sum of each call's kernels,
# captured at N = 262,144. The point-proportional kernels (stats, slice, px rows,
# deslice) are scaled x4; the W/Z' images and the split-partial reduction are not.
# Valid only for the kernel sources it was measured on, identified by the SHA-1 of
# _TRAFFIC_SOURCES.  When they change the figure is reported as null.
_TRAFFIC = {"sources_sha1": "7447527bf243e0c26dcdfcd4abea5c8647e400a3", "workload": "large_g_bf16", "N": 1048576,
            "fs_slice_fwd": 2.5530e9, "fs_deslice_fwd": 1.0684e9}


def _overrides(args):
    """Config entries that mark a run on a changed recipe."""
    o = {}
    if args.points:
        o["points_override"] = "N reduced for profiling; not the benchmark workload"
    if args.slots:
        o["slots_override"] = "G set to %d; not one of the named configurations" % args.slots
    if args.dtype:
        o["dtype_override"] = "inputs in %s; not the named configuration's dtype" % args.dtype
    return o


def _pipelined_e2e(K, stream, dev, ins, outs, compute):
    """K steps end to end, as a caller streaming batches through the C-ABI calls
    runs them: every step's inputs are copied in from pinned host memory and its
    outputs copied back.  Inputs and outputs are double-buffered, so step k + 1's
    inputs upload (one copy stream) and step k - 1's outputs download (another)
    while step k computes on `stream`.  The first upload and the last download
    are not hidden.  ins / outs: [(pinned host tensor, (device buffer 0, 1))];
    compute(j) enqueues one step on buffer set j.  Returns when all of it is
    enqueued on `stream` (the caller records its timing events around the call)."""
    import torch

    up_s, down_s = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    up_s.wait_stream(stream)  # nothing uploads before the caller's start event
    up, comp, down = ([torch.cuda.Event() for _ in range(K)] for _ in range(3))

    def upload(k):
        if k >= 2:
            up_s.wait_event(comp[k - 2])  # step k - 2 has finished reading these buffers
        with torch.cuda.stream(up_s):
            for h, d in ins:
                d[k % 2].copy_(h, non_blocking=True)
        up[k].record(up_s)

    upload(0)
    for k in range(K):
        if k + 1 < K:
            upload(k + 1)
        stream.wait_event(up[k])
        if k >= 2:
            stream.wait_event(down[k - 2])  # its output buffers have been copied out
        compute(k % 2)
        comp[k].record(stream)
        down_s.wait_event(comp[k])
        with torch.cuda.stream(down_s):
            for h, d in outs:
                h.copy_(d[k % 2], non_blocking=True)
        down[k].record(down_s)
    stream.wait_event(down[K - 1])


# The sources of the kernels whose DRAM traffic _TRAFFIC holds (the tensor-core
# forward: statistics, slice, deslice and their prep kernels).
_TRAFFIC_SOURCES = ("fs_tc.h", "fs_tc_common.cuh", "fs_tc_fwd.cu", "fs_tc_ptx.cuh")


def _sources_sha1():
    import hashlib

    h = hashlib.sha1()
    for f in _TRAFFIC_SOURCES:
        h.update(open(os.path.join(ROOT, "paper_2609_32525_gb300", "csrc", f), "rb").read())
    return h.hexdigest()


def _traffic(wl, call):
    if wl.name != _TRAFFIC["workload"] or wl.N != _TRAFFIC["N"] or _sources_sha1() != _TRAFFIC["sources_sha1"]:
        return None
    return _TRAFFIC[call]


def _algorithmic(wl):
    """Algorithmic work of one forward (per point, all heads; C = H*d):
    flops 8*C*G (logits twice, slice accumulate, deslice apply), bytes 4*C*e
    (slice reads x_mid and fx; deslice reads x_mid and writes out).  Each of the
    two streaming calls carries half of both."""
    C = wl.H * wl.d
    e = 2 if wl.dtype == "bf16" else 4
    P = wl.B * wl.N
    return {"flops": 8.0 * C * wl.G * P, "bytes": 4.0 * C * e * P,
            "flops_per_call": 4.0 * C * wl.G * P, "bytes_per_call": 2.0 * C * e * P}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms in the background."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id=None):
        self.path = tempfile.mktemp(prefix="fs_clocks_", suffix=".csv")
        cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits", "-lms", "200"]
        if gpu_id:
            cmd += ["-i", str(gpu_id)]
        try:
            self.f = open(self.path, "w")
            self.p = subprocess.Popen(cmd, stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def cpu_oracle_rate(wl, target_s=12.0, train=False):
    """The fp64 oracle as it stands, forward (slice over the sample, mix, deslice
    of the sample) on the first n points of the workload, all heads.  Returns
    (Mpoints/s, sample description, threads)."""
    from oracle import flashslice_oracle as orc

    def run(n):
        t0 = time.perf_counter()
        if train:
            orc.backward(wl.x_mid[:, :n], wl.fx[:, :n], wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout[:, :n], eps=wl.eps)
        else:
            orc.forward(wl.x_mid[:, :n], wl.fx[:, :n], wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
        return time.perf_counter() - t0

    n = min(wl.N, 4096)
    t = run(n)
    n2 = int(min(wl.N, max(n, n * target_s / max(t, 1e-3))))
    n2 = max(1024, (n2 // 1024) * 1024) if n2 >= 1024 else n2
    t2 = run(n2)
    threads = os.cpu_count()
    try:
        from threadpoolctl import threadpool_info

        threads = max([i.get("num_threads", 1) for i in threadpool_info()] + [1])
    except Exception:
        pass
    pts = wl.B * n2
    what = ("fp64 forward and backward (every gradient; the slice's sums over the sample)" if train else
            "fp64 forward (slice over the sample, mix, deslice of the sample)")
    desc = f"{wl.name}: first {n2} of {wl.N} points x B={wl.B}, all {wl.H} heads, {what}, {t2:.1f} s"
    return pts / t2 / 1e6, desc, threads


def run_reference(args):
    """--impl reference: the fp64 CPU oracle timed on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from oracle import flashslice_oracle as orc
    from paper_2609_32525_gb300.workloads import make_named

    wl = make_named(args.workload, n_override=args.points, g_override=args.slots, dtype_override=args.dtype)
    n = int(args.ref_points)
    train = wl.dout is not None  # the training workload: forward and backward, as its GPU line
    times = []
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        if train:
            orc.backward(wl.x_mid[:, :n], wl.fx[:, :n], wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout[:, :n], eps=wl.eps)
        else:
            orc.forward(wl.x_mid[:, :n], wl.fx[:, :n], wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    t = float(np.sum(times))
    value = wl.B * n * len(times) / t / 1e6
    what = "fp64 forward and backward" if train else "fp64 forward"
    line = {"impl": "reference", "metric": TRAIN_METRIC if train else METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl.name, "sample_points": n, "B": wl.B, "N": wl.N,
                                             "H": wl.H, "d": wl.d, "G": wl.G},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": f"first {n} points of {wl.name} per step, all heads, {what}"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)



def run_train(args, wl, dev, world, rank):
    """A training step of the coupling through the C ABI: the forward, then the
    backward of the deslice, the mix and the slice (every gradient)."""
    import torch
    import torch.distributed as dist

    from paper_2609_32525_gb300 import flashslice as fs
    from paper_2609_32525_gb300 import sharding

    def put(a, dt):
        return torch.from_numpy(a).to(device=dev, dtype=dt).contiguous()

    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    x, fx, dO = put(wl.x_mid, tdt), put(wl.fx, tdt), put(wl.dout, tdt)
    W, b, t, M = (put(getattr(wl, k), torch.float32) for k in ("W_slice", "bias", "tau", "M"))
    c = fs.Coupling(wl.B, wl.N, wl.H, wl.d, wl.G, tdt, wl.eps, device=dev, backward=True)
    s = c.shape
    stream = torch.cuda.current_stream()
    sep = args.separate_backward
    names = ("fs_slice_fwd", "fs_mix", "fs_deslice_fwd") + (
        ("fs_deslice_bwd", "fs_mix_bwd", "fs_slice_bwd") if sep else ("fs_coupling_bwd",))

    def step(ev=None, xs=x, fs_=fx, ds=dO, outs=None):
        out, dx, dfx = outs or (c.out, c.dx_mid, c.dfx)
        calls = (
            lambda: fs.fs_slice_fwd(s, xs, fs_, W, b, t, c.tokens, c.wsum, c.lse, True, c.ws_slice),
            lambda: fs.fs_mix(s, M, c.tokens, c.tokens_mixed),
            lambda: fs.fs_deslice_fwd(s, xs, W, b, t, c.tokens_mixed, c.lse, out, c.ws_deslice),
        )
        if sep:
            calls += (
                lambda: fs.fs_deslice_bwd(s, xs, W, b, t, c.tokens_mixed, c.lse, ds, c.d_tokens_mixed, dx, c.dW,
                                          c.dbias, c.dtau, False, c.ws_dbwd),
                lambda: fs.fs_mix_bwd(s, M, c.tokens, c.d_tokens_mixed, c.d_tokens, c.dM),
                lambda: fs.fs_slice_bwd(s, xs, fs_, W, b, t, c.tokens, c.wsum, c.lse, c.d_tokens, dx, dfx, c.dW,
                                        c.dbias, c.dtau, True, c.ws_sbwd),
            )
        else:
            calls += (
                lambda: fs.fs_coupling_bwd(s, xs, fs_, W, b, t, M, c.tokens, c.wsum, c.tokens_mixed, c.lse, ds,
                                           c.d_tokens_mixed, c.d_tokens, dx, dfx, c.dW, c.dbias, c.dtau, c.dM, False,
                                           c.ws_cbwd),
            )
        for i, call in enumerate(calls):
            if ev is not None:
                ev[i].record(stream)
            call()
        if ev is not None:
            ev[len(calls)].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if c.device_status() != fs.FS_OK:
        raise RuntimeError("device status after warm-up: " + fs.status_string(c.device_status()))
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        pass
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)] for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(uuid)
    time.sleep(0.3)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms_per_step = sharding.job_time_ms(t0.elapsed_time(t1), dev) / args.steps
    value = sharding.job_rate(wl.points, world, ms_per_step)
    call_ms = {n: float(np.mean([e[i].elapsed_time(e[i + 1]) for e in evs])) for i, n in enumerate(names)}
    assert c.device_status() == fs.FS_OK

    # End to end: pinned host x, fx, dO in; out, dx_mid and dfx back, every step,
    # pipelined as _pipelined_e2e describes.
    hx, hf, hd = (torch.from_numpy(a).to(tdt).pin_memory() for a in (wl.x_mid, wl.fx, wl.dout))
    hout = [torch.empty(c.out.shape, dtype=tdt).pin_memory() for _ in range(3)]
    ib = [[torch.empty_like(a) for _ in range(2)] for a in (x, fx, dO)]
    ob = [[torch.empty_like(a) for _ in range(2)] for a in (c.out, c.dx_mid, c.dfx)]
    ins, outs = list(zip((hx, hf, hd), ib)), list(zip(hout, ob))

    def e2e_compute(j):
        step(None, ib[0][j], ib[1][j], ib[2][j], (ob[0][j], ob[1][j], ob[2][j]))

    _pipelined_e2e(2, stream, dev, ins, outs, e2e_compute)
    torch.cuda.synchronize()
    assert c.device_status() == fs.FS_OK
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    _pipelined_e2e(args.e2e_steps, stream, dev, ins, outs, e2e_compute)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = sharding.job_time_ms(e0.elapsed_time(e1) / args.e2e_steps, dev)

    # Algorithmic work of a training step per point (C = H*d): forward 8*C*G flops,
    # each backward call 8*C*G (logits, dw and the two products of its pass), so
    # 24*C*G in all; bytes 11*C*e (forward 4, deslice backward 3, slice backward 4).
    C, e = wl.H * wl.d, (2 if wl.dtype == "bf16" else 4)
    P = wl.B * wl.N
    flops, bytes_ = 24.0 * C * wl.G * P, 11.0 * C * e * P
    per_call = {"fs_slice_fwd": 4.0 * C * wl.G * P, "fs_deslice_fwd": 4.0 * C * wl.G * P,
                "fs_deslice_bwd": 8.0 * C * wl.G * P, "fs_slice_bwd": 8.0 * C * wl.G * P,
                "fs_coupling_bwd": 16.0 * C * wl.G * P}
    per_call_bytes = {"fs_slice_fwd": 2.0 * C * e * P, "fs_deslice_fwd": 2.0 * C * e * P,
                      "fs_deslice_bwd": 3.0 * C * e * P, "fs_slice_bwd": 4.0 * C * e * P,
                      "fs_coupling_bwd": 7.0 * C * e * P}
    per_call = {k: v for k, v in per_call.items() if k in call_ms}
    per_call_bytes = {k: v for k, v in per_call_bytes.items() if k in call_ms}
    peaks = _peaks()
    dom = max(per_call, key=lambda k: call_ms[k])
    t_tensor, t_hbm = flops / (peaks["bf16_tflops"] * 1e12), bytes_ / (peaks["hbm_gbs"] * 1e9)
    roof_t = max(t_tensor, t_hbm)
    if t_tensor >= t_hbm:
        achieved = per_call[dom] / (call_ms[dom] * 1e-3) / 1e12
        bound = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                 "frac": achieved / peaks["bf16_tflops"], "peak_source": peaks["source"] + " bf16 burst"}
    else:
        achieved = per_call_bytes[dom] / (call_ms[dom] * 1e-3) / 1e9
        bound = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                 "frac": achieved / peaks["hbm_gbs"], "peak_source": peaks["source"] + " HBM copy"}
    roofline = {**bound, "traffic": None, "kernel": dom, "step_frac": roof_t / (ms_per_step * 1e-3),
                "call_ms": call_ms,
                "per_call_work": "forward calls 4*C*G flops and 2*C*e bytes per point each; the backward "
                                 "16*C*G flops and 7*C*e bytes (deslice backward 8*C*G and 3*C*e, slice "
                                 "backward 8*C*G and 4*C*e)"}
    line = {"metric": TRAIN_METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32",
            "data": "synthetic (seeded; " + wl.recipe + ")",
            "config": {"workload": wl.name, "B": wl.B, "N": wl.N, "H": wl.H, "d": wl.d, "G": wl.G,
                       "step": " + ".join(names), "parallelism": f"replicas x{world}",
                       "dot": ["bf16", "bf16x2"][s.dot],
                       "path": {"forward": ["simt", "tcgen05"][fs.path_for_shape(s)],
                                "backward": ["simt", "tcgen05"][fs.backward_path_for_shape(s)]},
                       **_overrides(args)},
            "clocks": clocks, "roofline": roofline,
            "gpu_launches": (fs.forward_launch_count(s) + (fs.backward_launch_count(s, True) if sep else
                                                           fs.coupling_bwd_launch_count(s, True))) * args.steps,
            "e2e": {"value": sharding.job_rate(wl.points, world, e2e_ms), "unit": UNIT,
                    "h2d_bytes_per_step": 3 * hx.numel() * hx.element_size(),
                    "d2h_bytes_per_step": sum(h_.numel() * h_.element_size() for h_ in hout), "ms_per_step": e2e_ms}}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, desc, threads = cpu_oracle_rate(wl, train=True)
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": desc}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


VARIANTS = ("tied", "untied", "frozen", "notokenattn")


def run_shard(args, wl, dev, world, rank):
    """--shard: one coupling point-sharded over the ranks (App. G.4).  Rank r holds
    points sharding.point_range(N, r, world) of every batch; a step is
    sharding.sharded_forward (the slice's unnormalised partials summed over ranks
    by NCCL, then finalize, mix, deslice of the local points) and, for a workload
    with an upstream gradient, sharding.sharded_backward (d_tokens_mixed summed,
    mix backward, slice backward, dW, dbias, dtau summed).  The total work is the
    workload's, whatever the number of ranks: scaling is strong."""
    import torch

    from paper_2609_32525_gb300 import flashslice as fs
    from paper_2609_32525_gb300 import sharding

    n0, n1 = sharding.point_range(wl.N, rank, world)
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32

    def put(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a)).to(device=dev, dtype=dt).contiguous()

    x, fx = put(wl.x_mid[:, n0:n1], tdt), put(wl.fx[:, n0:n1], tdt)
    dout = put(wl.dout[:, n0:n1], tdt) if wl.dout is not None else None
    W, b, t, M = (put(getattr(wl, k), torch.float32) for k in ("W_slice", "bias", "tau", "M"))
    ops = fs.ShardedCoupling(wl.B, n1 - n0, wl.H, wl.d, wl.G, x, fx, W, b, t, M, tdt, wl.eps, dout=dout, device=dev)
    train = dout is not None
    stream = torch.cuda.current_stream()

    def step():
        sharding.sharded_forward(ops)
        if train:
            sharding.sharded_backward(ops)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if ops.c.device_status() != fs.FS_OK:
        raise RuntimeError("device status after warm-up: " + fs.status_string(ops.c.device_status()))
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        pass
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(uuid)
    time.sleep(0.3)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms = sharding.job_time_ms(e0.elapsed_time(e1) / args.steps, dev)
    assert ops.c.device_status() == fs.FS_OK
    # the forward's kernels and the finalize of the summed partials; the backward's
    # calls all get the forward's lse
    per_step = fs.forward_launch_count(ops.c.shape) + 1 + (fs.backward_launch_count(ops.c.shape, True) if train else 0)
    line = {"metric": ("train step" if train else "coupling forward") + " Mpoints/s, point-sharded",
            "value": wl.points / (ms * 1e-3) / 1e6, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "strong",
            "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32",
            "data": "synthetic (seeded; " + wl.recipe + ")",
            "config": {"workload": wl.name, "B": wl.B, "N": wl.N, "H": wl.H, "d": wl.d, "G": wl.G,
                       "points_per_rank": n1 - n0, "parallelism": f"point-sharded x{world}",
                       "exchange": "NCCL all-reduce of (U, S)" + (", d_tokens_mixed, dW, dbias, dtau" if train else ""),
                       "path": ["simt", "tcgen05"][fs.path_for_shape(ops.c.shape)], **_overrides(args)},
            "clocks": clocks, "gpu_launches": per_step * args.steps}
    if rank == 0:
        print(json.dumps(line), flush=True)


def run_variant(args, wl, dev, world, rank):
    """One coupling forward of a variant of Sec. 3 (the variants table) on a forward
    workload, through the same C-ABI calls:
      untied      fs_slice_fwd, fs_mix, fs_deslice_fwd with its own (W', beta', tau')
                  and lse = NULL (the deslice computes its own statistics);
      frozen      a later layer slicing its own features fx2 with the layer-1 weights
                  and statistics: fs_slice_fwd_lse (no statistics pass), fs_mix,
                  fs_deslice_fwd with the layer-1 lse;
      notokenattn fs_slice_fwd, fs_mix_channels (a d x d map per head), fs_deslice_fwd.
    Timed like the default line (CUDA events on the launching stream, max over
    ranks); its work is the tied step's (8*C*G flops per point: the statistics a
    call recomputes are not algorithmic work)."""
    import torch

    from paper_2609_32525_gb300 import flashslice as fs
    from paper_2609_32525_gb300 import sharding

    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32

    def put(a, dt):
        return torch.from_numpy(a).to(device=dev, dtype=dt).contiguous()

    x, fx = put(wl.x_mid, tdt), put(wl.fx, tdt)
    W, b, t, M = (put(getattr(wl, k), torch.float32) for k in ("W_slice", "bias", "tau", "M"))
    c = fs.Coupling(wl.B, wl.N, wl.H, wl.d, wl.G, tdt, wl.eps, device=dev)
    s = c.shape
    stream = torch.cuda.current_stream()
    g = torch.Generator(device=dev)
    g.manual_seed(2609)
    f32 = dict(dtype=torch.float32, device=dev)
    # the second weight set, the later layer's features and the channel map, seeded:
    # W' ~ N(0, 1/d), beta' = 0, tau' = 0.7; fx2 ~ N(0, 1); Wc = I + N(0, 0.01)
    W2 = torch.randn(W.shape, generator=g, **f32) / wl.d ** 0.5
    b2, t2 = torch.zeros_like(b), torch.full_like(t, 0.7)
    fx2 = torch.randn(fx.shape, generator=g, **f32).to(tdt)
    Wc = torch.eye(wl.d, **f32).expand(wl.H, wl.d, wl.d) + 0.1 * torch.randn(wl.H, wl.d, wl.d, generator=g, **f32)
    Wc = Wc.contiguous()
    lse1 = torch.empty_like(c.lse)
    fs.fs_slice_fwd(s, x, fx, W, b, t, c.tokens, c.wsum, lse1, True, c.ws_slice)  # layer 1's statistics

    def step():
        if args.variant == "untied":
            fs.fs_slice_fwd(s, x, fx, W, b, t, c.tokens, c.wsum, c.lse, True, c.ws_slice)
            fs.fs_mix(s, M, c.tokens, c.tokens_mixed)
            fs.fs_deslice_fwd(s, x, W2, b2, t2, c.tokens_mixed, None, c.out, c.ws_deslice)
        elif args.variant == "frozen":
            fs.fs_slice_fwd_lse(s, x, fx2, W, b, t, lse1, c.tokens, c.wsum, True, c.ws_slice)
            fs.fs_mix(s, M, c.tokens, c.tokens_mixed)
            fs.fs_deslice_fwd(s, x, W, b, t, c.tokens_mixed, lse1, c.out, c.ws_deslice)
        elif args.variant == "notokenattn":
            fs.fs_slice_fwd(s, x, fx, W, b, t, c.tokens, c.wsum, c.lse, True, c.ws_slice)
            fs.fs_mix_channels(s, Wc, c.tokens, c.tokens_mixed)
            fs.fs_deslice_fwd(s, x, W, b, t, c.tokens_mixed, c.lse, c.out, c.ws_deslice)
        else:
            fs.fs_slice_fwd(s, x, fx, W, b, t, c.tokens, c.wsum, c.lse, True, c.ws_slice)
            fs.fs_mix(s, M, c.tokens, c.tokens_mixed)
            fs.fs_deslice_fwd(s, x, W, b, t, c.tokens_mixed, c.lse, c.out, c.ws_deslice)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if c.device_status() != fs.FS_OK:
        raise RuntimeError("device status after warm-up: " + fs.status_string(c.device_status()))
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(None)
    time.sleep(0.3)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step()
    t1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = sharding.job_time_ms(t0.elapsed_time(t1), dev) / args.steps
    assert c.device_status() == fs.FS_OK
    alg, peaks = _algorithmic(wl), _peaks()
    roof_t = max(alg["flops"] / (peaks["bf16_tflops"] * 1e12), alg["bytes"] / (peaks["hbm_gbs"] * 1e9))
    line = {"metric": "coupling forward Mpoints/s, variant " + args.variant, "value": sharding.job_rate(wl.points, world, ms),
            "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
            "data": "synthetic (seeded; " + wl.recipe + ")",
            "config": {"workload": wl.name, "variant": args.variant, "B": wl.B, "N": wl.N, "H": wl.H, "d": wl.d,
                       "G": wl.G, "parallelism": f"replicas x{world}", **_overrides(args)},
            "clocks": clocks, "step_frac": roof_t / (ms * 1e-3)}
    if rank == 0:
        print(json.dumps(line), flush=True)


def build_parser() -> argparse.ArgumentParser:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="large_g_bf16")
    ap.add_argument("--variant", default=None, choices=VARIANTS,
                    help="time one coupling variant of the forward workload instead (Sec. 3 variants table)")
    ap.add_argument("--shard", action="store_true",
                    help="one coupling point-sharded over the ranks with NCCL all-reduces (App. G.4), "
                         "strong scaling, instead of one replica per rank")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--ref-points", type=int, default=16384)
    ap.add_argument("--points", type=int, default=None,
                    help="profiling runs only: the workload's recipe at a smaller N (the line says so)")
    ap.add_argument("--separate-backward", action="store_true",
                    help="training: the backward as fs_deslice_bwd, fs_mix_bwd, fs_slice_bwd instead of "
                         "fs_coupling_bwd")
    ap.add_argument("--slots", type=int, default=None,
                    help="the workload's recipe at another slot count G (the line says so)")
    ap.add_argument("--dtype", default=None, choices=["bf16", "f32"],
                    help="the workload's recipe with inputs of this dtype (the line says so)")
    return ap


def main():
    args = build_parser().parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    from paper_2609_32525_gb300 import build as _build

    if not os.path.exists(_build.LIB):
        _build.build()
    from paper_2609_32525_gb300 import flashslice as fs
    from paper_2609_32525_gb300 import sharding
    from paper_2609_32525_gb300.workloads import make_named

    wl = make_named(args.workload, n_override=args.points, g_override=args.slots, dtype_override=args.dtype)
    if args.shard:
        run_shard(args, wl, dev, world, rank)
        if world > 1:
            dist.destroy_process_group()
        return
    if wl.dout is not None:
        return run_train(args, wl, dev, world, rank)
    if args.variant is not None:
        return run_variant(args, wl, dev, world, rank)
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32

    def put(a, dt):
        return torch.from_numpy(a).to(device=dev, dtype=dt).contiguous()

    x, fx = put(wl.x_mid, tdt), put(wl.fx, tdt)
    W, b, t, M = (put(getattr(wl, k), torch.float32) for k in ("W_slice", "bias", "tau", "M"))
    c = fs.Coupling(wl.B, wl.N, wl.H, wl.d, wl.G, tdt, wl.eps, device=dev)
    s = c.shape
    stream = torch.cuda.current_stream()

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        fs.fs_slice_fwd(s, x, fx, W, b, t, c.tokens, c.wsum, c.lse, True, c.ws_slice)
        if ev is not None:
            ev[1].record(stream)
        fs.fs_mix(s, M, c.tokens, c.tokens_mixed)
        if ev is not None:
            ev[2].record(stream)
        fs.fs_deslice_fwd(s, x, W, b, t, c.tokens_mixed, c.lse, c.out, c.ws_deslice)
        if ev is not None:
            ev[3].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if c.device_status() != fs.FS_OK:
        raise RuntimeError("device status after warm-up: " + fs.status_string(c.device_status()))

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        pass
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(uuid)
    time.sleep(0.3)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = t_start.elapsed_time(t_end)
    slice_ms = float(np.mean([e[0].elapsed_time(e[1]) for e in evs]))
    mix_ms = float(np.mean([e[1].elapsed_time(e[2]) for e in evs]))
    desl_ms = float(np.mean([e[2].elapsed_time(e[3]) for e in evs]))
    total_ms = sharding.job_time_ms(total_ms, dev)
    ms_per_step = total_ms / args.steps
    value = sharding.job_rate(wl.points, world, ms_per_step)
    assert c.device_status() == fs.FS_OK

    # End to end through the C-ABI calls with host buffers (pinned x, fx in; out back
    # every step), pipelined as _pipelined_e2e describes.
    hx = torch.from_numpy(wl.x_mid).to(tdt).pin_memory()
    hf = torch.from_numpy(wl.fx).to(tdt).pin_memory()
    hout = torch.empty(c.out.shape, dtype=tdt).pin_memory()
    xb, fb, ob = ([torch.empty_like(a) for _ in range(2)] for a in (x, fx, c.out))

    def e2e_compute(j):
        fs.fs_slice_fwd(s, xb[j], fb[j], W, b, t, c.tokens, c.wsum, c.lse, True, c.ws_slice)
        fs.fs_mix(s, M, c.tokens, c.tokens_mixed)
        fs.fs_deslice_fwd(s, xb[j], W, b, t, c.tokens_mixed, c.lse, ob[j], c.ws_deslice)

    ins, outs = [(hx, xb), (hf, fb)], [(hout, ob)]
    _pipelined_e2e(2, stream, dev, ins, outs, e2e_compute)
    torch.cuda.synchronize()
    assert c.device_status() == fs.FS_OK
    if world > 1:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    _pipelined_e2e(args.e2e_steps, stream, dev, ins, outs, e2e_compute)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / args.e2e_steps
    e2e_ms = sharding.job_time_ms(e2e_ms, dev)
    e2e_val = sharding.job_rate(wl.points, world, e2e_ms)
    h2d = 2 * hx.numel() * hx.element_size()
    d2h = hout.numel() * hout.element_size()

    peaks = _peaks()
    alg = _algorithmic(wl)
    dom_name, dom_ms = ("fs_slice_fwd", slice_ms) if slice_ms >= desl_ms else ("fs_deslice_fwd", desl_ms)
    t_tensor = alg["flops"] / (peaks["bf16_tflops"] * 1e12)
    t_hbm = alg["bytes"] / (peaks["hbm_gbs"] * 1e9)
    roof_t = max(t_tensor, t_hbm)
    if t_tensor >= t_hbm:
        achieved = alg["flops_per_call"] / (dom_ms * 1e-3) / 1e12
        bound = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                 "frac": achieved / peaks["bf16_tflops"], "peak_source": peaks["source"] + " bf16 burst",
                 "frac_sustained": achieved / peaks["bf16_tflops_sustained"]}
    else:
        achieved = alg["bytes_per_call"] / (dom_ms * 1e-3) / 1e9
        bound = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                 "frac": achieved / peaks["hbm_gbs"], "peak_source": peaks["source"] + " HBM copy"}
    roofline = {**bound, "traffic": _traffic(wl, dom_name), "kernel": dom_name,
                "traffic_unit": "bytes per call (ncu DRAM read + write)",
                "step_frac": roof_t / (ms_per_step * 1e-3),
                "call_ms": {"fs_slice_fwd": slice_ms, "fs_mix": mix_ms, "fs_deslice_fwd": desl_ms},
                "per_call_work": "4*C*G flops and 2*C*e bytes per point for each of slice and deslice"}

    # Each of the three sweeps (statistics, slice, deslice) makes one exponential per
    # point, head and slot; at 32 ex2 per clock per SM (measured on GB300) that floor
    # lies above the tensor roofline, so the MUFU rate is reported beside it.
    n_exp = float(wl.B * wl.N * wl.H * wl.G)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    mufu_peak = 32.0 * sms * float(clocks.get("sm_mhz") or 2070.0) * 1e6 / 1e9
    exps = {"fs_slice_fwd": 2 * n_exp, "fs_deslice_fwd": n_exp}
    call_ms = {"fs_slice_fwd": slice_ms, "fs_deslice_fwd": desl_ms}
    roofline["mufu"] = {"unit": "Gexp/s", "peak": mufu_peak, "exps_per_call": exps,
                        "achieved": {k: exps[k] / (call_ms[k] * 1e-3) / 1e9 for k in exps},
                        "frac": {k: exps[k] / (call_ms[k] * 1e-3) / 1e9 / mufu_peak for k in exps},
                        "step_frac": 3 * n_exp / (ms_per_step * 1e-3) / 1e9 / mufu_peak}

    launches = fs.forward_launch_count(s) * args.steps
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32",
            "data": "synthetic (seeded; " + wl.recipe + ")",
            "config": {"workload": wl.name, "B": wl.B, "N": wl.N, "H": wl.H, "d": wl.d, "G": wl.G,
                       "step": "fs_slice_fwd + fs_mix + fs_deslice_fwd", "parallelism": f"replicas x{world}",
                       "l2": "inputs 2 x %d MiB > 129 MB L2, no flush" % (hx.numel() * hx.element_size() >> 20),
                       "path": ["simt", "tcgen05"][fs.path_for_shape(s)],
                       **_overrides(args)},
            "clocks": clocks, "gpu_launches": launches, "roofline": roofline,
            "e2e": {"value": e2e_val, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_ms}}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, desc, threads = cpu_oracle_rate(wl)
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": desc}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
