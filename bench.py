#!/usr/bin/env python3
"""Throughput of the GB300 DLA forward path (one JSON line on stdout).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dla|reference]

Headline: prefill tokens/s of the regime-shift workload (B=2, H=16, T=16384,
d=128, C=32, bf16 inputs, fp32 states) -- one step is one dla_forward call
over the whole batch (scan, snapshots, read-out), inputs resident in HBM.
The same line carries the decode workload (256 sequences x 32 heads, d=128,
C=64, fp32 cache pre-filled by an 8K-token prefill; one step is one
dla_decode_step for every stream), the roofline of the dominant kernel of
each (CUDA events on the library's stream), the end-to-end figure through the
public API with host buffers, and the fp64 oracle timed on the host cores
(cpu_baseline).  The path shards by independent (batch, head) streams, so
N > 1 runs N independent replicas (weak scaling, no collective on the data
path).  ``--impl reference`` times the oracle instead (the reference arm).
"""
from __future__ import annotations

import argparse
import datetime
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

PREFILL_METRIC = "DLA tokens/sec (prefill, T=16K, C=32)"
DECODE_METRIC = "DLA decode tokens/sec"
FP32_LANES_PER_SM = 128  # FFMA lanes per SM (Blackwell)


# ---------------------------------------------------------------- helpers

def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), bf16=float(p["bf16_tflops"]),
                    bf16_sustained=float(p["bf16_tflops_sustained"]), sm_max_mhz=float(p.get("sm_max_mhz", 2070.0)),
                    source="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, sm_max_mhz=2070.0, source="fallback")


class Dist:
    def __init__(self):
        self.rank = int(os.environ.get("RANK", "0"))
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch
            import torch.distributed as dist
            backend = "nccl" if torch.cuda.is_available() else "gloo"
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def reduce(self, x, op):
        if not self.pg:
            return x
        import torch
        dev = torch.device("cuda", self.local) if torch.cuda.is_available() else torch.device("cpu")
        t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX if op == "max" else self.pg.ReduceOp.SUM)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


class Clocks:
    """nvidia-smi sampling (every 50 ms) around a timed region and the untimed
    steps of the same work run just before it (a timed region of a few tens of
    ms holds one sample at most); samples whose timestamp falls inside the
    timed region are also counted apart."""

    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None
        self.region = None  # wall-clock (start, end) of the timed region

    def mark(self, t0, t1):
        self.region = (t0, t1)

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="dla_clocks_", suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return self.summarize(lines, self.region)

    @staticmethod
    def summarize(lines, region=None):
        """The clock record of nvidia-smi CSV lines (the fields of Q)."""
        rows = []
        for line in lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 11:
                rows.append(parts)
        if not rows:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return float("nan")

        def stamp(x):  # nvidia-smi's local time, e.g. 2026/12/02 15:01:16.123
            try:
                return datetime.datetime.strptime(x, "%Y/%m/%d %H:%M:%S.%f").timestamp()
            except ValueError:
                return None

        loaded = [r for r in rows if num(r[5]) > 0] or rows
        sm = [num(r[2]) for r in loaded]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in loaded for i in range(4) if r[7 + i].lower().startswith("active")})
        rec = {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(num(r[3]) for r in rows),
               "power_w_max": max(num(r[4]) for r in rows), "samples": len(rows), "samples_under_load": len(loaded),
               "reasons": reasons, "interval_ms": 50}
        if region is not None:
            inside = [r for r in rows if (stamp(r[0]) or -1.0) >= region[0] - 0.05 and (stamp(r[0]) or -1.0) <= region[1] + 0.05]
            rec["samples_in_timed_region"] = len(inside)
            if inside:
                rec["sm_mhz_in_timed_region"] = statistics.median(num(r[2]) for r in inside)
        return rec


def kernel_table(timing, steps):
    total = sum(ms for _, ms in timing.values()) or 1.0
    return {k: {"launches": n, "ms_total": round(ms, 4), "ms_per_launch": round(ms / n, 5) if n else None,
                "share": round(ms / total, 4)} for k, (n, ms) in timing.items() if n}


# ---------------------------------------------------------------- prefill

_INPUTS = {}  # device inputs of the headline workload: (workload, q, k, v, lambda)


def bench_backward(args, dist, pk, steps=3, warmup=2):
    """dla_backward on the headline workload's inputs and decisions: dQ, dK, dV
    and dlambda of the read-out for a seeded upstream gradient, timed with CUDA
    events; the device status is checked."""
    import torch

    from paper_2606_10650_gb300 import dla

    w, qt, kt, vt, lt = _INPUTS[args.workload]
    B, T, H, d = kt.shape
    fwd = dla.forward(qt, kt, vt, lt, tau=w.tau, capacity=w.C, eps=w.eps, rms_eps=w.rms_eps)
    g = torch.randn((B, T, H, d), dtype=torch.float32, device=kt.device,
                    generator=torch.Generator(device=kt.device).manual_seed(11))
    del fwd["o"]

    def step():
        return dla.backward(qt, kt, vt, lt, fwd["boundary"], fwd["merge_log"], g, capacity=w.C)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    if dla.dla_sync_status() != 0:
        raise RuntimeError("backward: device status reports a failure")
    dla.dla_timing_read(reset=True)
    dla.dla_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        out = step()
    e1.record()
    torch.cuda.synchronize()
    dla.dla_timing_enable(False)
    if dla.dla_sync_status() != 0:
        raise RuntimeError("backward: device status reports a failure in the timed steps")
    launches = sum(v_[0] for v_ in dla.dla_timing_read(reset=True).values())
    ms = e0.elapsed_time(e1) / steps
    del out
    # five d-long contractions per token pair s <= t: q_t.k_s, g_t.v_s and the
    # three weighted gradient products (dq, dk, dv)
    algorithmic = 10.0 * d * (T * (T + 1) / 2) * B * H
    return {"workload": f"{w.name}: B={B} H={H} T={T} d={d} C={w.C}, decisions of a forward call, "
                        "upstream gradient N(0, 1)",
            "value": round(B * T / ms * 1e3, 1), "unit": "tokens/s", "ms_per_step": round(ms, 3), "steps": steps,
            "outputs": "dQ, dK, dV [B, T, H, d] and dlambda [B, T, H, C], fp32",
            "algorithmic_tflops": round(algorithmic / (ms * 1e-3) / 1e12, 2),
            "algorithmic_flops": "10*d*T(T+1)/2*B*H (five d-long contractions per token pair s <= t)",
            "note": "quadratic in T per stream (every token pair s <= t, 64 x 64 tiles on mma.sync)",
            "gpu_launches": launches}


def bench_dla_i(args, dist, pk, capacity=128, steps=5, warmup=3):
    """DLA(I) (dynamic merging without the capacity bound) on the headline
    workload's inputs: capacity 128 lies above every stream's segment count, so
    no capacity merge occurs; the device status and the absence of merges are
    checked."""
    import torch

    from paper_2606_10650_gb300 import dla

    w, qt, kt, vt, lt0 = _INPUTS[args.workload]
    B, T, H, d = kt.shape
    lt = torch.ones((B, T, H, capacity), dtype=torch.float32, device=kt.device)
    lt[..., : w.C] = lt0

    def step():
        return dla.forward(qt, kt, vt, lt, tau=w.tau, capacity=capacity, eps=w.eps, rms_eps=w.rms_eps)

    for _ in range(warmup):
        r = step()
    torch.cuda.synchronize()
    if dla.dla_sync_status() != 0 or int((r["merge_log"] >= 0).sum().item()) != 0:
        raise RuntimeError("DLA(I): a device failure or a capacity merge")
    dla.dla_timing_read(reset=True)
    dla.dla_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        r = step()
    e1.record()
    torch.cuda.synchronize()
    dla.dla_timing_enable(False)
    if dla.dla_sync_status() != 0:
        raise RuntimeError("DLA(I): device status reports a failure in the timed steps")
    launches = sum(v_[0] for v_ in dla.dla_timing_read(reset=True).values())
    ms = e0.elapsed_time(e1) / steps
    seg = r["boundary"].sum(dim=2)
    return {"workload": f"{w.name}: B={B} H={H} T={T} d={d}, capacity {capacity} (DLA(I): no capacity merge)",
            "value": round(B * T / ms * 1e3, 1), "unit": "tokens/s", "ms_per_step": round(ms, 4), "steps": steps,
            "segments_per_stream": {"min": int(seg.min()), "max": int(seg.max()), "mean": round(float(seg.float().mean()), 1)},
            "merges": 0, "gpu_launches": launches}


def _time_steps(step, steps, warmup, before=None):
    """Mean CUDA-event time (ms) of `step` over `steps` calls after `warmup`
    untimed ones; `before` (untimed) runs ahead of every call; the library's
    launches inside the timed calls are counted."""
    import torch

    from paper_2606_10650_gb300 import dla

    for _ in range(warmup):
        if before:
            before()
        step()
    torch.cuda.synchronize()
    if dla.dla_sync_status() != 0:
        raise RuntimeError("device status reports a failure in the warm-up calls")
    dla.dla_timing_read(reset=True)
    total = 0.0
    for _ in range(steps):
        if before:
            before()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        dla.dla_timing_enable(True)
        e0.record()
        step()
        e1.record()
        torch.cuda.synchronize()
        dla.dla_timing_enable(False)
        total += e0.elapsed_time(e1)
    if dla.dla_sync_status() != 0:
        raise RuntimeError("device status reports a failure in the timed calls")
    launches = sum(v_[0] for v_ in dla.dla_timing_read(reset=True).values())
    return total / steps, launches


def bench_packed(args, dist, pk, steps=10, warmup=3):
    """dla_forward_varlen on the headline workload's tokens regrouped as a
    packed batch of four rows of different lengths (the serving layout,
    cu_seqlens offsets), each row from an empty cache."""
    import torch

    from paper_2606_10650_gb300 import dla

    w, qt, kt, vt, lt = _INPUTS[args.workload]
    B, T, H, d = kt.shape
    if B != 2 or T % 4:
        return None
    cuts = [(0, 0, 3 * T // 4), (0, 3 * T // 4, T), (1, 0, T // 2), (1, T // 2, T)]  # (batch row, t0, t1)
    lens = [t1 - t0 for _, t0, t1 in cuts]
    pq, pk_, pv, pl = (torch.cat([x[b, t0:t1] for b, t0, t1 in cuts]).contiguous() for x in (qt, kt, vt, lt))
    cu = torch.tensor([0] + list(__import__("itertools").accumulate(lens)), dtype=torch.int32, device=kt.device)
    mx = max(lens)
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    o = torch.empty_like(pq, dtype=torch.float32)
    bnd = torch.empty((len(lens), H, mx), dtype=torch.uint8, device=kt.device)
    ml = torch.empty((len(lens), H, mx), dtype=torch.int32, device=kt.device)
    cache = dla.Cache(len(lens), H, w.C, d, device=kt.device)
    ws = dla.dla_forward_varlen(p, cu, mx, pq, pk_, pv, pl, o, cache, bnd, ml)  # sizes the workspace once

    def step():
        dla.dla_forward_varlen(p, cu, mx, pq, pk_, pv, pl, o, cache, bnd, ml, workspace=ws)

    ms, launches = _time_steps(step, steps, warmup)
    tokens = sum(lens)
    return {"workload": f"{w.name} tokens regrouped: {len(lens)} packed rows of {lens} tokens, H={H} d={d} C={w.C}, "
                        "each row from an empty cache (dla_forward_varlen, cu_seqlens)",
            "value": round(tokens / ms * 1e3, 1), "unit": "tokens/s", "ms_per_step": round(ms, 4), "steps": steps,
            "gpu_launches": launches}


def bench_continuation(args, dist, pk, steps=10, warmup=3):
    """Prefill continuation: dla_forward with from_cache = 1 over the second
    half of the headline workload's rows, on top of the cache the first half
    left; the cache is restored (untimed) before every call."""
    import torch

    from paper_2606_10650_gb300 import dla

    w, qt, kt, vt, lt = _INPUTS[args.workload]
    B, T, H, d = kt.shape
    half = T // 2
    q2, k2, v2, l2 = (x[:, half:].contiguous() for x in (qt, kt, vt, lt))
    cache = dla.Cache(B, H, w.C, d, device=kt.device)
    dla.forward(qt[:, :half].contiguous(), kt[:, :half].contiguous(), vt[:, :half].contiguous(),
                lt[:, :half].contiguous(), tau=w.tau, capacity=w.C, eps=w.eps, rms_eps=w.rms_eps, want_o=False,
                cache=cache)
    saved = cache.buf.clone()
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps, from_cache=1)
    o = torch.empty((B, T - half, H, d), dtype=torch.float32, device=kt.device)
    bnd = torch.empty((B, H, T - half), dtype=torch.uint8, device=kt.device)
    ml = torch.empty((B, H, T - half), dtype=torch.int32, device=kt.device)
    nb = dla.dla_forward_workspace(p, B, T - half, H, d, d, dla.DLA_BF16, True)
    buf = torch.empty(nb + 256, dtype=torch.uint8, device=kt.device)
    ws = (buf, (buf.data_ptr() + 255) // 256 * 256, nb)

    def restore():
        cache.buf.copy_(saved)

    def step():
        dla.dla_forward(p, q2, k2, v2, l2, o, cache, bnd, ml, workspace=ws)

    ms, launches = _time_steps(step, steps, warmup, before=restore)
    return {"workload": f"{w.name}: B={B} H={H} d={d} C={w.C}, tokens {half}..{T - 1} of every row on top of the "
                        f"cache of tokens 0..{half - 1} (from_cache = 1; the cache restored, untimed, before each call)",
            "value": round(B * (T - half) / ms * 1e3, 1), "unit": "tokens/s", "ms_per_step": round(ms, 4),
            "steps": steps, "gpu_launches": launches}


def bench_prefill(args, dist, pk, workload=None, steps=None, warmup=None, headline=True):
    """One workload's prefill: warm-up, `steps` timed dla_forward calls (the
    default concurrent schedule), the call's device status checked, the kernels
    timed alone (serial schedule) and the timed run's decision trace checked
    against the serial run's.  With `headline`, also the end-to-end figure
    through dla_forward_host."""
    import numpy as np
    import torch

    from paper_2606_10650_gb300 import dla
    from paper_2606_10650_gb300 import workloads as W

    workload = workload or args.workload
    steps = args.steps if steps is None else steps
    warmup = args.warmup if warmup is None else warmup
    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    w = W.get(workload, **({"T": args.T} if (args.T and headline) else {}))
    q, k, v, lam = W.host_batch_parallel(w, T=w.T)
    qt, kt, vt = (W.to_device(x, w.dtype, dev) for x in (q, k, v))
    lt = torch.from_numpy(lam).to(dev)
    del q, k, v, lam
    if headline:
        _INPUTS[workload] = (w, qt, kt, vt, lt)  # reused by the backward and DLA(I) lines
    B, T, H, d = kt.shape
    p = dla.make_params(w.tau, w.C, w.eps, w.rms_eps)
    in_code = dla.DLA_BF16 if w.dtype == "bf16" else dla.DLA_F32
    cache = dla.Cache(B, H, w.C, d, device=dev)
    o = torch.empty((B, T, H, d), dtype=torch.float32, device=dev)
    bnd = torch.empty((B, H, T), dtype=torch.uint8, device=dev)
    ml = torch.empty((B, H, T), dtype=torch.int32, device=dev)
    nb = dla.dla_forward_workspace(p, B, T, H, d, d, in_code, True)
    if args.ws_gb:
        nb = max(min(nb, int(args.ws_gb * (1 << 30))), dla.dla_forward_min_workspace(p, B, T, H, d, d, in_code, True))
    buf = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    ws = (buf, (buf.data_ptr() + 255) // 256 * 256, nb)
    stream = torch.cuda.current_stream()

    def step():
        dla.dla_forward(p, qt, kt, vt, lt, o, cache, bnd, ml, workspace=ws, stream=stream)

    def check_status(what):
        st = dla.dla_sync_status(stream)
        if st != 0 or dla.workspace_status(ws) != 0:
            raise RuntimeError(f"{workload}: device status {st} after {what} (a bounded wait gave up or a "
                               "device check failed): the timing would not be valid")

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    check_status("the warm-up steps")
    dla.dla_timing_read(reset=True)
    clocks = Clocks(dist.local) if headline else None
    if clocks:
        # the clock record: sampled through 0.5 s of the same steps, untimed,
        # right before the timed region, and through the timed region itself
        clocks.start()
        t_soak = time.time() + 0.5
        n_soak = 0
        while time.time() < t_soak:
            step()
            n_soak += 1
            if n_soak % 16 == 0:
                torch.cuda.synchronize()
    dist.barrier()
    torch.cuda.synchronize()
    dla.dla_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0 = time.time()
    e0.record(stream)
    for _ in range(steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    w1 = time.time()
    dla.dla_timing_enable(False)
    dist.barrier()
    if clocks:
        clocks.mark(w0, w1)
    clk = clocks.stop() if clocks else None
    if clk is not None:
        clk["untimed_steps_before"] = n_soak
    ms = e0.elapsed_time(e1) / steps
    timing = dla.dla_timing_read(reset=True)
    check_status("the timed steps")
    ms_max = dist.reduce(ms, "max")
    tokens = B * T
    # the timed run's decisions, checked below against a serial-schedule run
    timed_trace = (bnd.clone(), ml.clone(), cache.view("m").clone(), cache.view("n").clone())
    # algorithmic work from the decision trace: m_t = live states after token t
    m_t = torch.cumsum(bnd.to(torch.int64), 2) - torch.cumsum((ml >= 0).to(torch.int64), 2)
    sum_m = int(m_t.sum().item())
    del m_t
    BH = B * H
    flops_total = 2.0 * d * d * (sum_m + 2 * T * BH)
    kt_tab = kernel_table(timing, steps)
    tc_path = (w.dtype == "bf16" and d == 128)
    # Each kernel alone on the device: the same forward pass under the serial
    # schedule (pre-pass, scan, read-out one after another), timed after the
    # step.  Inside the step the kernels overlap and the read-out is paced by
    # the scan, so their in-step durations are not their speeds.
    solo, solo_steps, validated = {}, min(steps, 5), None
    if tc_path:
        os.environ["DLA_SCHEDULE"] = "serial"
        try:
            step()
            torch.cuda.synchronize()
            dla.dla_timing_read(reset=True)
            dla.dla_timing_enable(True)
            for _ in range(solo_steps):
                step()
            torch.cuda.synchronize()
            dla.dla_timing_enable(False)
            solo = dla.dla_timing_read(reset=True)
            check_status("the serial-schedule steps")
        finally:
            os.environ.pop("DLA_SCHEDULE", None)
        same = [torch.equal(a_, b_) for a_, b_ in zip(timed_trace, (bnd, ml, cache.view("m"), cache.view("n")))]
        if not all(same):
            raise RuntimeError(f"{workload}: the timed run's decisions differ from the serial schedule's "
                               f"(boundary, merge_log, m, n equal: {same})")
        validated = ("device status 0 after the warm-up, timed and serial steps; the timed run's boundary flags, "
                     "merge indices and final live / token counts equal a serial-schedule run on the same inputs")
    del timed_trace
    t_in = {k_: (n_, ms_) for k_, (n_, ms_) in timing.items()}
    fp32_peak = pk_fp32(pk)
    rooflines, sm_ms = {}, {}
    n_sms = 152
    scan_sms = 2 * BH if 2 * BH <= n_sms else min(BH, n_sms)

    def per_launch(table, name):
        n_, ms_ = table.get(name, (0, 0.0))
        return (ms_ / n_) if n_ else None

    for name in ("readout", "scan", "gram"):
        t_solo = per_launch(solo, name) if solo else None
        t_step = per_launch(t_in, name)
        t = t_solo if t_solo is not None else t_step
        if t is None:
            continue
        n_launch = t_in.get(name, (0, 0.0))[0] / steps  # launches per step inside the timed region
        timing_note = (f"CUDA events around each launch of the kernel alone on the device (serial schedule, "
                       f"{solo_steps} forward passes after the timed steps); inside the timed step it lasts "
                       f"{t_step:.4f} ms per launch, overlapped" if t_solo is not None else
                       "CUDA events around each launch inside the timed steps")
        if name == "readout":
            work = 2.0 * d * d * sum_m / max(n_launch, 1)
            peak = pk["bf16"] if tc_path else fp32_peak
            ach = work / (t * 1e-3) / 1e12
            rooflines[name] = {
                "kernel": "readout (snapshot and intra-interval parts, K2)", "bound": "tensor" if tc_path else "alu",
                "achieved": round(ach, 3), "peak": round(peak, 2), "unit": "TFLOP/s", "frac": round(ach / peak, 4),
                "traffic": None, "ms_per_launch": round(t, 5),
                "peak_note": ("measured bf16 dense GEMM (burst) of MEASURED_PEAKS.json" if tc_path else
                              "fp32 FFMA: 152 SMs x 128 lanes x 2 flop x sm_max_mhz"),
                "work_per_launch": f"2*d^2*sum_t m_t / launches = {work:.4g} flop", "timing": timing_note,
                "executed_note": ("each snapshot-state product runs as one fp16 MMA per interval (fp16 pool "
                                  "entries, Q converted to fp16; fp16 runs at the bf16 dense rate), so the executed "
                                  "snapshot flops equal the algorithmic count; the intra-interval products (Q K^T, "
                                  "Pt V) come on top" if tc_path else "")}
            sm_ms[name] = t * n_launch * n_sms
        elif name == "scan":
            work = 4.0 * d * d * T * BH / max(n_launch, 1)  # x_t = v^T S k and the state build, 2 d^2 each per token
            peak = pk["bf16"] if tc_path else fp32_peak
            ach = work / (t * 1e-3) / 1e12
            rooflines[name] = {
                "kernel": "scan (K1)", "bound": "tensor" if tc_path else "alu", "achieved": round(ach, 3),
                "peak": round(peak, 2), "unit": "TFLOP/s", "frac": round(ach / peak, 4), "traffic": None,
                "ms_per_launch": round(t, 5),
                "peak_note": ("measured bf16 dense GEMM (burst) of MEASURED_PEAKS.json" if tc_path else
                              "fp32 FFMA: 152 SMs x 128 lanes x 2 flop x sm_max_mhz"),
                "work_per_launch": f"4*d^2*T*B*H / launches = {work:.4g} flop", "timing": timing_note,
                "note": (f"latency-bound: each (batch, head) stream is sequential; {scan_sms} CTAs "
                         f"({'pairs' if scan_sms == 2 * BH else 'one per stream'})")}
            sm_ms[name] = t * n_launch * scan_sms
        elif name == "gram":
            nch = (T + 63) // 64
            work = (2.0 * B * T * H * d * 2 + BH * nch * (2 * 64 * 64 + 64) * 4) / max(n_launch, 1)
            ach = work / (t * 1e-3) / 1e9
            rooflines[name] = {
                "kernel": "Gram pre-pass (K0)", "bound": "hbm", "achieved": round(ach, 1), "peak": pk["hbm"],
                "unit": "GB/s", "frac": round(ach / pk["hbm"], 4), "traffic": None, "ms_per_launch": round(t, 5),
                "work_per_launch": f"k, v read (bf16) + Gram tables written (fp32) = {work:.4g} bytes",
                "timing": timing_note}
            sm_ms[name] = t * n_launch * n_sms
    # DRAM traffic per launch from profiles/traffic.json, while the kernel's source is the one
    # captured and the workload is the one captured (else null)
    tr = captured_traffic("readout_tc_kernel", f"{workload} B{B} H{H} T{T} d{d}")
    if tr and "readout" in rooflines and tc_path:
        rooflines["readout"]["traffic"] = tr["bytes_per_launch"]
        rooflines["readout"]["traffic_note"] = ("dram__bytes_read.sum + dram__bytes_write.sum of one full-size "
                                                f"launch (ncu, {tr['summary']})")
    # dominant kernel: the one carrying the largest share of the step's algorithmic work,
    # the read-out (2 d^2 sum_t m_t of the prefill's 2 d^2 (sum_t m_t + 2T) flops); the
    # latency-bound scan sets the step's critical path (see rooflines.scan and the SM-time
    # shares in the note)
    dominant = "readout" if "readout" in rooflines else (max(sm_ms, key=lambda k_: sm_ms[k_]) if sm_ms else None)
    roof = dict(rooflines[dominant]) if dominant else None
    if roof is not None:
        share = sum_m / (sum_m + 2.0 * T * BH) if dominant == "readout" else None
        roof["dominance"] = ((f"largest share of the algorithmic work ({share:.3f} of 2 d^2 (sum_t m_t + 2T)); "
                              if share is not None else "") +
                             "SM-time per step (ms alone x SMs occupied): " +
                             ", ".join(f"{k_} {v_:.1f} SM-ms" for k_, v_ in sm_ms.items()))
    # end to end through the C ABI with host buffers: every step, dla_forward_host
    # copies q, k, v, lambda in from page-locked host memory (piece by piece beside
    # the scan on the concurrent schedule), runs the forward pass and copies o back
    e2e = None
    if headline and not args.no_e2e:
        qh, kh, vh = (x.cpu().pin_memory() for x in (qt, kt, vt))
        lh = lt.cpu().pin_memory()
        oh = torch.empty(o.shape, dtype=o.dtype).pin_memory()
        n_e2e = max(2, min(steps, 10))
        hnb = dla.dla_forward_host_workspace(p, B, T, H, d, d, in_code, True)
        hbuf = torch.empty(hnb + 256, dtype=torch.uint8, device=dev)
        hws = (hbuf, (hbuf.data_ptr() + 255) // 256 * 256, hnb)

        def e2e_step():
            dla.dla_forward_host(p, qh, kh, vh, lh, oh, cache, bnd, ml, workspace=hws, stream=stream)

        e2e_step()
        torch.cuda.synchronize()
        if dla.dla_sync_status(stream) != 0 or dla.workspace_status(hws) != 0:
            raise RuntimeError("dla_forward_host: device status reports a failure")
        dist.barrier()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(n_e2e):
            e2e_step()
        a1.record(stream)
        torch.cuda.synchronize()
        if dla.dla_sync_status(stream) != 0:
            raise RuntimeError("dla_forward_host: device status reports a failure in the timed steps")
        e_ms = dist.reduce(a0.elapsed_time(a1) / n_e2e, "max")
        hb = sum(x.numel() * x.element_size() for x in (qh, kh, vh, lh))
        e2e = {"value": round(dist.world * tokens / (e_ms * 1e-3), 1), "unit": "tokens/s", "ms_per_step": round(e_ms, 4),
               "h2d_bytes_per_step": hb, "d2h_bytes_per_step": oh.numel() * oh.element_size(), "steps": n_e2e,
               "call": "dla_forward_host (C ABI, page-locked host buffers in and out)"}
        del hbuf, hws
    res = {"value": dist.world * tokens / (ms_max * 1e-3), "ms_per_step": ms_max, "tokens_per_step": tokens,
           "roofline": roof, "rooflines": rooflines, "kernels": kt_tab,
           "kernels_alone": kernel_table(solo, solo_steps) if solo else None, "tc_path": tc_path, "clocks": clk,
           "e2e": e2e, "validated": validated, "steps": steps,
           "gpu_launches": sum(n_ for n_, _ in timing.values()),
           "algorithmic_tflops": flops_total / (ms_max * 1e-3) / 1e12, "sum_m": sum_m,
           "boundaries": int(bnd.sum().item()), "merges": int((ml >= 0).sum().item()),
           "workload": f"{w.name}: B={w.B} H={w.H} T={w.T} d={w.d} C={w.C} {w.dtype} inputs, fp32 states"}
    del qt, kt, vt, lt, o, buf, cache
    torch.cuda.empty_cache()
    return res


def captured_traffic(kernel, workload, table=None):
    """The DRAM traffic record of `kernel` in `table` (default
    profiles/traffic.json: bytes per launch from one ncu capture), if it was
    taken on `workload` and the kernel's source file (relative to the
    repository root) still has the recorded hash; else None."""
    import hashlib
    root = os.path.dirname(os.path.abspath(__file__))
    try:
        with open(table or os.path.join(root, "profiles", "traffic.json")) as f:
            rec = json.load(f).get(kernel)
        if not rec or rec.get("workload") != workload:
            return None
        with open(os.path.join(root, rec["source"]), "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()
        return rec if sha.startswith(rec["sha256_prefix"]) else None
    except (OSError, ValueError, KeyError):
        return None


def pk_fp32(pk):
    return 152 * FP32_LANES_PER_SM * 2 * pk["sm_max_mhz"] * 1e6 / 1e12


# ---------------------------------------------------------------- decode

def bench_decode(args, dist, pk):
    import torch

    from paper_2606_10650_gb300 import dla
    from paper_2606_10650_gb300 import workloads as W

    dev = torch.device("cuda", dist.local)
    w = W.get("decode")
    B, H, d, C, Tp = w.B, w.H, w.d, w.C, w.T
    if args.decode_batch:
        B = args.decode_batch
    p = dla.make_params(w.tau, C, w.eps, w.rms_eps)
    cache = dla.Cache(B, H, C, d, device=dev)
    gb = 32 if B % 32 == 0 else B
    nb = dla.dla_forward_workspace(p, gb, Tp, H, d, d, dla.DLA_BF16, False)
    buf = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    ws = (buf, (buf.data_ptr() + 255) // 256 * 256, nb)
    t0 = time.time()
    for g in range(B // gb):  # seeded 8K-token prefill, 32 sequences at a time, scan only (o = NULL)
        _, kk, vv, _ = W.device_iid_batch(w, gb, Tp, seed=w.seed * 1000 + g, device=dev, with_lam=False)
        dla.dla_forward(p, None, kk, vv, None, None, cache.sub(g * gb, gb), None, None, workspace=ws)
        del kk, vv
    torch.cuda.synchronize()
    prefill_s = time.time() - t0
    del buf
    nsteps = args.warmup + args.steps
    wd = W.get("decode", B=B)
    qs, ks, vs, ls = W.device_decode_steps(wd, nsteps, seed=w.seed * 1000 + 999, device=dev)
    o = torch.empty((B, H, d), dtype=torch.float32, device=dev)
    bflag = torch.empty((B, H), dtype=torch.uint8, device=dev)
    midx = torch.empty((B, H), dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    def step(i):
        dla.dla_decode_step(p, cache, qs[i], ks[i], vs[i], ls[i], o, bflag, midx, stream=stream)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    m_before = cache.view("m").to(torch.int64)
    bytes_per_step = float(((m_before + 1) * d * d * 4).sum().item())
    dla.dla_timing_read(reset=True)
    dist.barrier()
    torch.cuda.synchronize()
    dla.dla_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    nb_fire = 0
    for i in range(args.warmup, nsteps):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    dla.dla_timing_enable(False)
    dist.barrier()
    ms = dist.reduce(e0.elapsed_time(e1) / args.steps, "max")
    timing = dla.dla_timing_read(reset=True)
    if dla.dla_sync_status(stream) != 0:
        raise RuntimeError("decode: device status reports a failure in the timed steps")
    dn, dms = timing["decode"]
    achieved = bytes_per_step / (dms / dn * 1e-3) / 1e9
    roof = {"kernel": "decode", "bound": "hbm", "achieved": round(achieved, 1), "peak": pk["hbm"], "unit": "GB/s",
            "frac": round(achieved / pk["hbm"], 4), "traffic": None,
            "work_per_launch": f"sum over streams (m+1)*d^2*4 = {bytes_per_step:.4g} bytes"}
    nb_fire = int(bflag.sum().item())
    # end to end: host q, k, v, lambda in, o out
    e2e = None
    if not args.no_e2e:
        qh, kh, vh, lh = (x[:4].cpu().pin_memory() for x in (qs, ks, vs, ls))
        oh = torch.empty(o.shape, dtype=o.dtype).pin_memory()
        qd, kd, vd, ld = (torch.empty_like(x[0]) for x in (qs, ks, vs, ls))
        n_e2e = max(2, min(args.steps, 8))
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for i in range(n_e2e):
            j = i % 4
            qd.copy_(qh[j], non_blocking=True)
            kd.copy_(kh[j], non_blocking=True)
            vd.copy_(vh[j], non_blocking=True)
            ld.copy_(lh[j], non_blocking=True)
            dla.dla_decode_step(p, cache, qd, kd, vd, ld, o, bflag, midx, stream=stream)
            oh.copy_(o, non_blocking=True)
        a1.record(stream)
        torch.cuda.synchronize()
        e_ms = dist.reduce(a0.elapsed_time(a1) / n_e2e, "max")
        e2e = {"value": round(dist.world * B / (e_ms * 1e-3), 1), "unit": "tokens/s", "ms_per_step": round(e_ms, 4),
               "h2d_bytes_per_step": sum(x[0].numel() * x.element_size() for x in (qh, kh, vh, lh)),
               "d2h_bytes_per_step": oh.numel() * oh.element_size(), "steps": n_e2e}
    res = {"metric": DECODE_METRIC, "value": round(dist.world * B / (ms * 1e-3), 1), "unit": "tokens/s",
           "ms_per_step": round(ms, 4), "steps": args.steps, "higher_is_better": True,
           "config": {"workload": f"decode: {B} sequences x H={H}, d={d}, C={C}, fp32 cache after a seeded "
                                  f"{Tp}-token i.i.d. prefill; bf16 q/k/v N(0,1/128) per step",
                      "l2": f"cache {cache.buf.numel() / 1e9:.1f} GB >> L2"},
           "roofline": roof, "kernels": kernel_table(timing, args.steps), "e2e": e2e,
           "gpu_launches": sum(n for n, _ in timing.values()), "prefill_setup_s": round(prefill_s, 2),
           "boundaries_last_step": nb_fire}
    del cache, qs, ks, vs, ls
    torch.cuda.empty_cache()
    return res


# ---------------------------------------------------------------- oracle timings

def oracle_sample(workload, tokens, heads=None, threads=None):
    """The fp64 oracle over the first `tokens` tokens of every head of batch
    row 0 (read-out at every token).  Returns (seconds, threads, token-heads)."""
    import numpy as np
    from concurrent.futures import ThreadPoolExecutor

    import oracle
    from paper_2606_10650_gb300 import workloads as W

    w = W.get(workload)
    H = w.H if heads is None else heads
    streams = []
    for h in range(H):
        g = W.StreamGen(w, 0, h)
        q, kk, vv = g.tokens()
        streams.append((q[:tokens], kk[:tokens], vv[:tokens], g.lam()[:tokens]))
    n = threads or min(len(streams), os.cpu_count() or 1)

    def one(s):
        st = oracle.Stream(w.C, w.d, w.d, w.tau, w.eps, w.rms_eps)
        st.run(*s)

    oracle.lib()
    t0 = time.time()
    with ThreadPoolExecutor(n) as ex:
        list(ex.map(one, streams))
    return time.time() - t0, n, H * tokens


def cpu_baseline(args):
    secs, n, th = oracle_sample(args.workload, args.cpu_tokens)
    return {"value": round(args.cpu_tokens / secs, 2), "unit": "tokens/s", "cores": n, "kind": "oracle",
            "seconds": round(secs, 2),
            "sample": f"{args.workload} workload, batch row 0, all {th // args.cpu_tokens} heads, first "
                      f"{args.cpu_tokens} tokens, read-out at every token (a token = all heads of one position)"}


def run_reference(args, dist):
    cfg = config_of(args)
    if dist.rank != 0:
        return
    tok = args.ref_tokens
    for _ in range(args.warmup):
        oracle_sample(args.workload, tok)
    times = []
    cores = 1
    for _ in range(args.steps):
        s, cores, _ = oracle_sample(args.workload, tok)
        times.append(s)
    ms = 1e3 * sum(times) / len(times)
    val = tok / (ms * 1e-3)
    line = {"impl": "reference", "metric": PREFILL_METRIC, "value": round(val, 2), "unit": "tokens/s", "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": cfg,
            "cpu_baseline": {"value": round(val, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"each step: batch row 0, all heads, first {tok} tokens of the {args.workload} "
                                       "workload, read-out at every token"},
            "e2e": {"value": round(val, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def config_of(args):
    from paper_2606_10650_gb300 import workloads as W
    w = W.get(args.workload, **({"T": args.T} if args.T else {}))
    return {"workload": f"{w.name}: B={w.B} H={w.H} T={w.T} d={w.d} C={w.C} {w.dtype} inputs, fp32 states, "
                        f"tau={w.tau}, lambda U({w.lam_lo},{w.lam_hi})",
            "global_batch": w.B, "seq_len": w.T, "parallelism": "replicas",
            "l2": "inputs (q,k,v,lambda: %.0f MB) larger than L2" % (
                (3 * w.B * w.T * w.H * w.d * (2 if w.dtype == 'bf16' else 4) + 4 * w.B * w.T * w.H * w.C) / 1e6)}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="dla", choices=["dla", "reference"])
    ap.add_argument("--workload", default="regime")
    ap.add_argument("--T", type=int, default=0)
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the standard and long prefill lines")
    ap.add_argument("--decode-batch", type=int, default=0)
    ap.add_argument("--ws-gb", type=float, default=0.0, help="cap the prefill workspace (GiB)")
    ap.add_argument("--cpu-tokens", type=int, default=8192)
    # the reference arm's sample per step: the same as cpu_baseline's (first 8192
    # tokens of batch row 0, all heads, about 2 s on 16 host cores), so that the
    # two oracle rates describe one sample
    ap.add_argument("--ref-tokens", type=int, default=8192)
    args = ap.parse_args()
    args.warmup = max(args.warmup, 0)
    dist = Dist()
    if args.impl == "reference":
        run_reference(args, dist)
        dist.close()
        return
    import __graft_entry__
    __graft_entry__.build()
    pk = peaks()
    pre = None if args.no_prefill else bench_prefill(args, dist, pk)
    others = {}
    if not (args.no_prefill or args.no_configs):
        for name in ("standard", "long"):  # the other prefill workloads, fewer steps
            r = bench_prefill(args, dist, pk, workload=name, steps=min(args.steps, 10), warmup=max(args.warmup, 3),
                              headline=False)
            others[name] = {k_: r[k_] for k_ in ("workload", "value", "ms_per_step", "steps", "roofline",
                                                 "kernels_alone", "validated", "gpu_launches", "algorithmic_tflops",
                                                 "boundaries", "merges", "sum_m")}
            others[name]["value"] = round(others[name]["value"], 1)
            others[name]["unit"] = "tokens/s"
            others[name]["algorithmic_frac_of_peak"] = round(r["algorithmic_tflops"] / pk["bf16"], 4)
    extra = {}
    if pre and pre["tc_path"] and not args.no_configs and args.workload in _INPUTS:
        for key, fn in (("backward", bench_backward), ("dla_i", bench_dla_i), ("packed", bench_packed),
                        ("continuation", bench_continuation)):
            try:
                extra[key] = fn(args, dist, pk)
            except (RuntimeError, MemoryError) as exc:  # reported in the line; the headline stands
                extra[key] = {"error": str(exc)}
                import torch

                from paper_2606_10650_gb300 import dla
                torch.cuda.synchronize()
                dla.dla_sync_status()
    _INPUTS.clear()
    dec = None if args.no_decode else bench_decode(args, dist, pk)
    cpu = cpu_baseline(args) if (dist.rank == 0 and dist.world == 1 and not args.no_cpu) else None
    if dist.rank == 0:
        line = {"metric": PREFILL_METRIC, "unit": "tokens/s", "n_gpus": dist.world, "steps": args.steps,
                "warmup": args.warmup, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16" if (pre and pre["tc_path"]) else "f32", "data": "synthetic (seeded regime-shift streams; no dataset)",
                "config": config_of(args), "peaks_source": pk["source"]}
        if pre:
            line.update(value=round(pre["value"], 1), ms_per_step=round(pre["ms_per_step"], 4),
                        roofline=pre["roofline"], rooflines=pre["rooflines"], kernels=pre["kernels"],
                        kernels_alone=pre["kernels_alone"], clocks=pre["clocks"], e2e=pre["e2e"],
                        gpu_launches=pre["gpu_launches"],
                        algorithmic_tflops=round(pre["algorithmic_tflops"], 3),
                        algorithmic_frac_of_peak=round(pre["algorithmic_tflops"] / pk["bf16"], 4),
                        validated=pre["validated"],
                        trace={"sum_m": pre["sum_m"], "boundaries": pre["boundaries"], "merges": pre["merges"]})
        if others:
            line["other_prefill_workloads"] = others
        if extra:
            line.update(extra)
        if dec:
            line["decode"] = dec
        line["cpu_baseline"] = cpu
        print(json.dumps(line))
    dist.close()


if __name__ == "__main__":
    main()
