#!/usr/bin/env python3
"""Benchmark of SONIQ's inference hot path on GB300.

Default workload: the ResNet-18-shaped 3x3 convolution (batch 64, 14x14x256 ->
256, 70% of input channels at 4 bits and 30% at 8 bits) run as implicit GEMM.
One step = one pass of the per-inference path over the batch:
    soniq_quantize_act (max-abs scale + quantize + pack the NHWC input)
    soniq_mp_conv2d    (tcgen05 implicit GEMM + fused scale epilogue)
Weights are packed once before timing (offline, Sec. 3: the layout is fixed
after training).  The metric is effective TOPS = 2 * M * N * K / step time
with the logical (unpadded) K = 9 * 256.

--suite adds the other workload families (linear, MLP up-projection, decode
GEMV, precision sweep) as a per-kernel table under "suite".
--impl reference times the CPU oracle on bounded samples of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "mixed-precision GEMM effective TOPS (and GEMV GB/s) and % of roofline on 1 GB300"
L2_FLUSH_BYTES = 256 << 20       # > 129 MB L2
# dram__bytes_read.sum + dram__bytes_write.sum of one mp_mma_kernel launch on the
# default conv workload, from an ncu capture of `python bench.py --case conv_4b8b`
# (to be reset to None whenever the kernel changes after that capture)
CONV_TRAFFIC_BYTES = 2994176.0


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return dict(hbm=float(d["hbm_gbs"]), bf16=float(d["bf16_tflops"]),
                    bf16_sus=float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


# --------------------------------------------------------------------------
# clocks sampled during the timed region
# --------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"soniq_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
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
        self.fh.close()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax = float(parts[2])
                except ValueError:
                    continue
                for name, flag in zip(names, parts[5:9]):
                    if flag.lower() == "active":
                        reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------

def conv_ops(spec, count):
    """Logical integer ops per group: 2 * M * C_out * (R*S*count_g)."""
    return [2 * spec.M * spec.C_out * spec.R * spec.S * c for c in count]


def mixed_peak(ops, kinds, pk):
    """Tensor peak for a step that runs ops[g] on the pipe of kinds[g]
    (0: E4M3 at 2x the bf16 rate, 1: fp16 at the bf16 rate)."""
    t = sum(o / (pk["bf16"] * (2.0 if k == 0 else 1.0)) for o, k in zip(ops, kinds))
    return sum(ops) / t if t > 0 else pk["bf16"]


def run_gpu(args):
    import torch
    import torch.distributed as dist

    from paper_2311_14114_gb300 import soniq as sq
    from paper_2311_14114_gb300 import workloads as wl

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    pk = peaks()

    spec = wl.CONV_RESNET
    d = wl.make_conv(spec)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    stream = torch.cuda.current_stream()
    X = torch.from_numpy(d["X"]).cuda().reshape(-1, spec.C)
    Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
    cd = sq.conv_desc(spec.batch, spec.H, spec.W, spec.C_out, spec.R, spec.S, spec.stride, spec.pad)
    P, Q = sq.conv_out_hw(cd)
    Xp = torch.empty((spec.batch * spec.H * spec.W, lay.row_bytes()), dtype=torch.uint8, device="cuda")
    s_a = torch.empty(2, dtype=torch.float32, device="cuda")
    Y = torch.empty((spec.batch, P, Q, spec.C_out), dtype=torch.float16, device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")

    def step():
        sq.quantize_act(lay, X, "tensor", s_a=s_a, Ap=Xp)
        sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, Y=Y)

    for _ in range(max(args.warmup, 3)):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    if sq.sync_status() != 0:
        raise RuntimeError("device error during warm-up")

    # The device-timed steps replay CUDA graphs of the two library calls (as a
    # serving loop would), so host-side call overhead does not sit between the
    # events; the end-to-end number below goes through the plain API calls.
    side = torch.cuda.Stream()
    side.wait_stream(stream)
    n0 = sq.launch_count()
    g_step, g_quant, g_conv = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_step, stream=side):
        step()
    launches_per_step = sq.launch_count() - n0
    with torch.cuda.graph(g_quant, stream=side):
        sq.quantize_act(lay, X, "tensor", s_a=s_a, Ap=Xp)
    with torch.cuda.graph(g_conv, stream=side):
        sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, Y=Y)
    for _ in range(max(args.warmup, 3)):
        flush.zero_()
        g_step.replay()
    torch.cuda.synchronize()

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    for i in range(args.steps):
        flush.zero_()                       # L2 flushed between timed steps (outside the events)
        a, _, c = ev[i]
        a.record(stream)
        g_step.replay()
        c.record(stream)
    torch.cuda.synchronize()
    launches = launches_per_step * args.steps
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    if sq.sync_status() != 0:
        raise RuntimeError("device error during the timed steps")
    step_ms = [a.elapsed_time(c) for a, b, c in ev]
    total_ms = sum(step_ms)
    # the two kernels alone, same flush and replay discipline (roofline of the conv)
    conv_ms, quant_ms = [], []
    for g, out in ((g_conv, conv_ms), (g_quant, quant_ms)):
        for i in range(args.steps):
            flush.zero_()
            a, _, c = ev[i]
            a.record(stream)
            g.replay()
            c.record(stream)
        torch.cuda.synchronize()
        out.extend(a.elapsed_time(c) for a, _, c in ev)
    if world > 1:
        t = torch.tensor([total_ms, sum(conv_ms)], dtype=torch.float64, device="cuda")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms, conv_total = float(t[0]), float(t[1])
    else:
        conv_total = sum(conv_ms)
    ms_per_step = total_ms / args.steps
    ops = spec.ops
    value = world * ops / (ms_per_step * 1e-3) / 1e12

    # ---- end to end through host buffers ----
    # Every step uploads its own input from pinned host memory, runs the two
    # API calls and reads its output back.  As in a serving loop, the copies of
    # neighbouring steps overlap this step's kernels: uploads, kernels and
    # downloads run on three streams with two sets of buffers.
    NB = 2
    Xh = [torch.from_numpy(d["X"]).reshape(-1, spec.C).pin_memory() for _ in range(NB)]
    Yh = [torch.empty((spec.batch, P, Q, spec.C_out), dtype=torch.float16).pin_memory() for _ in range(NB)]
    Xd = [torch.empty_like(X) for _ in range(NB)]
    Xpd = [torch.empty_like(Xp) for _ in range(NB)]
    sad = [torch.empty_like(s_a) for _ in range(NB)]
    Yd = [torch.empty_like(Y) for _ in range(NB)]
    s_up, s_cmp, s_down = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    for st_ in (s_up, s_cmp, s_down):
        st_.wait_stream(stream)
    up_done = [torch.cuda.Event() for _ in range(NB)]
    cmp_done = [torch.cuda.Event() for _ in range(NB)]
    down_done = [torch.cuda.Event() for _ in range(NB)]
    used = [False] * NB

    def e2e_step(i):
        k = i % NB
        with torch.cuda.stream(s_up):
            if used[k]:
                s_up.wait_event(cmp_done[k])          # the kernels of step i - NB have read Xd[k]
            Xd[k].copy_(Xh[k], non_blocking=True)
            up_done[k].record(s_up)
        with torch.cuda.stream(s_cmp):
            s_cmp.wait_event(up_done[k])
            if used[k]:
                s_cmp.wait_event(down_done[k])        # Yd[k] of step i - NB has been read back
            sq.quantize_act(lay, Xd[k], "tensor", s_a=sad[k], Ap=Xpd[k], stream=s_cmp)
            sq.mp_conv2d(lay, cd, Xpd[k], sad[k], Wp, s_w, Y=Yd[k], stream=s_cmp)
            cmp_done[k].record(s_cmp)
        with torch.cuda.stream(s_down):
            s_down.wait_event(cmp_done[k])
            Yh[k].copy_(Yd[k], non_blocking=True)
            down_done[k].record(s_down)
        used[k] = True

    for i in range(3):
        e2e_step(i)
    torch.cuda.synchronize()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e_start.record(s_up)
    for i in range(args.steps):
        e2e_step(i)
    e_end.record(s_down)
    torch.cuda.synchronize()
    if sq.sync_status() != 0:
        raise RuntimeError("device error during the end-to-end steps")
    e2e_ms = e_start.elapsed_time(e_end) / args.steps
    if world > 1:
        t = torch.tensor([e2e_ms], dtype=torch.float64, device="cuda")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_ms = float(t[0])
    e2e_value = world * ops / (e2e_ms * 1e-3) / 1e12

    # ---- roofline of the dominant kernel (the implicit-GEMM conv) ----
    conv_avg_ms = conv_total / args.steps
    achieved = ops / (conv_avg_ms * 1e-3) / 1e12
    kinds = [0 if b <= 4 else 1 for b in d["bits"]]
    peak = mixed_peak(conv_ops(spec, d["count"]), kinds, pk)
    roofline = {"kernel": "mp_mma_kernel (implicit-GEMM conv)", "bound": "tensor",
                "achieved": round(achieved, 2), "peak": round(peak, 1), "unit": "TFLOP/s",
                "frac": round(achieved / peak, 4), "traffic": args.traffic,
                "peak_source": f"{pk['src']}: bf16 {pk['bf16']} TFLOP/s burst; E4M3 = 2x bf16 "
                               f"(nominal ratio), fp16 = bf16 rate; time-weighted over the groups",
                "quantize_us": round(statistics.mean(quant_ms) * 1e3, 2),
                "conv_us": round(conv_avg_ms * 1e3, 2)}

    out = {"metric": METRIC, "value": round(value, 3), "unit": "TOPS", "n_gpus": world,
           "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": round(ms_per_step, 5),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "u8xs8->i32 (E4M3/fp16 tensor pipes, exact)", "data": "synthetic",
           "config": {"workload": spec.name, "M": spec.M, "N": spec.C_out, "K": spec.K,
                      "bits": d["bits"], "count": d["count"], "parallelism": f"replicas{world}",
                      "l2": "flushed between timed steps (256 MB write)",
                      "launch": "the step (both library calls) replayed as one CUDA graph; e2e: plain API calls"},
           "e2e": {"value": round(e2e_value, 3), "unit": "TOPS",
                   "h2d_bytes_per_step": int(Xh[0].numel() * 2), "d2h_bytes_per_step": int(Yh[0].numel() * 2),
                   "ms_per_step": round(e2e_ms, 5),
                   "pipelining": "upload, kernels and download of neighbouring steps overlap (3 streams, 2 buffer sets)"},
           "gpu_launches": int(launches),
           "roofline": roofline,
           "clocks": clk}
    if args.suite:
        out["suite"] = run_suite(args, sq, wl, pk, flush)
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(spec, d, budget_s=args.cpu_seconds)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


def _time_events(fn, steps, flush, stream):
    """Median device time of fn (a library call), replayed as a CUDA graph so
    that host call overhead is not timed; L2 flushed before every replay."""
    import torch
    for _ in range(2):
        fn()
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(stream)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        fn()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for _ in range(3):
        flush.zero_()
        g.replay()
    for i in range(steps):
        flush.zero_()
        ev[i][0].record(stream)
        g.replay()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    return statistics.median(a.elapsed_time(b) for a, b in ev)


def run_suite(args, sq, wl, pk, flush):
    """Per-kernel measurements for the other workload families."""
    import torch
    stream = torch.cuda.current_stream()
    rows = []

    def linear_case(spec, kind):
        d = wl.make_linear(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        A = torch.from_numpy(d["A"]).cuda()
        W = torch.from_numpy(d["W"]).cuda()
        Wp, s_w = sq.pack_weights(lay, W)
        Ap, s_a = sq.quantize_act(lay, A)
        Y = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
        gemm_ms = _time_events(lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y), args.steps, flush, stream)
        quant_ms = _time_events(lambda: sq.quantize_act(lay, A, "tensor", s_a=s_a, Ap=Ap), args.steps, flush, stream)
        pack_ms = _time_events(lambda: sq.pack_weights(lay, W, Wp=Wp, s_w=s_w), max(3, args.steps // 4), flush, stream)
        ops = spec.ops
        kinds = [0 if b <= 4 else 1 for b in d["bits"]]
        peak = mixed_peak([2 * spec.M * spec.N * c for c in d["count"]], kinds, pk)
        wbytes = sum(c * b for c, b in zip(d["count"], d["bits"])) / 8 * spec.N
        abytes = spec.M * spec.K * 2 + spec.M * sum(c * b for c, b in zip(d["count"], d["bits"])) / 8
        r = {"workload": spec.name, "M": spec.M, "N": spec.N, "K": spec.K, "bits": d["bits"],
             "gemm_us": round(gemm_ms * 1e3, 2), "TOPS": round(ops / (gemm_ms * 1e-3) / 1e12, 2),
             "quantize_us": round(quant_ms * 1e3, 2),
             "quantize_GBps": round(abytes / (quant_ms * 1e-3) / 1e9, 1),
             "pack_weights_us": round(pack_ms * 1e3, 2)}
        if kind == "gemv":
            moved = Wp.numel() + s_w.numel() * 4
            r["path"] = "CUDA-core GEMV" if spec.M <= 12 else "tensor-core kernel"
            r["gemv_GBps_algorithmic"] = round(wbytes / (gemm_ms * 1e-3) / 1e9, 1)
            r["frac_hbm"] = round(wbytes / (gemm_ms * 1e-3) / 1e9 / pk["hbm"], 4)
            r["weight_bytes_moved"] = int(moved)
        else:
            r["frac_tensor_peak"] = round(ops / (gemm_ms * 1e-3) / 1e12 / peak, 4)
            r["peak_TFLOPs"] = round(peak, 1)
        rows.append(r)

    linear_case(wl.LINEAR_SMALL, "gemm")
    linear_case(wl.MLP_UP, "gemm")
    for m in (1, 4, 16):
        linear_case(wl.DECODE[m], "gemv")
    pts = wl.sweep_specs() if args.full_sweep else [
        s for s in wl.sweep_specs() if (s.bits_lo, s.bits_hi) in ((2, 8), (4, 8), (1, 4), (3, 6))]
    for s in pts:
        try:
            linear_case(s, "gemm")
        except Exception as e:  # report, do not hide
            rows.append({"workload": s.name, "error": str(e)})
    conv_b = wl.CONV_RESNET_1B4B
    d = wl.make_conv(conv_b)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    X = torch.from_numpy(d["X"]).cuda().reshape(-1, conv_b.C)
    Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
    Xp, s_a = sq.quantize_act(lay, X)
    cd = sq.conv_desc(conv_b.batch, conv_b.H, conv_b.W, conv_b.C_out)
    Y = torch.empty((conv_b.batch, 14, 14, conv_b.C_out), dtype=torch.float16, device="cuda")
    ms = _time_events(lambda: sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, Y=Y), args.steps, flush, stream)
    kinds = [0 if b <= 4 else 1 for b in d["bits"]]
    peak = mixed_peak(conv_ops(conv_b, d["count"]), kinds, pk)
    rows.append({"workload": conv_b.name, "conv_us": round(ms * 1e3, 2),
                 "TOPS": round(conv_b.ops / (ms * 1e-3) / 1e12, 2),
                 "frac_tensor_peak": round(conv_b.ops / (ms * 1e-3) / 1e12 / peak, 4)})
    return rows


# --------------------------------------------------------------------------
# CPU oracle (baseline leg and the reference arm)
# --------------------------------------------------------------------------

def _threads():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_conv_sample(spec, d, n_pix):
    """The oracle pipeline for the conv step on n_pix output pixels: scales,
    codes and packing of the whole input, weights once, accumulators and
    epilogue for the sampled pixels."""
    import oracle
    rng = np.random.default_rng(0)
    pix = np.sort(rng.choice(spec.M, size=min(n_pix, spec.M), replace=False))
    return oracle.conv2d(d["X"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], spec.R, spec.S,
                         stride=spec.stride, pad=spec.pad, pix=pix), len(pix)


def cpu_baseline(spec, d, budget_s=12.0):
    import oracle
    oracle.build()
    t0 = time.perf_counter()
    oracle_conv_sample(spec, d, 256)
    t1 = time.perf_counter() - t0
    n_pix = int(min(spec.M, max(256, 256 * budget_s / max(t1, 1e-3))))
    t0 = time.perf_counter()
    _, n = oracle_conv_sample(spec, d, n_pix)
    dt = time.perf_counter() - t0
    ops = 2 * n * spec.C_out * spec.K
    return {"value": round(ops / dt / 1e12, 6), "unit": "TOPS", "cores": _threads(), "kind": "oracle",
            "sample": f"{n} of {spec.M} output pixels (full-input scales/codes/packing, sampled "
                      f"accumulators + epilogue), {dt:.1f} s",
            "seconds": round(dt, 2)}


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2311_14114_gb300 import workloads as wl
    import oracle
    oracle.build()
    spec = wl.CONV_RESNET
    d = wl.make_conv(spec)
    per_step_pix = 192
    for _ in range(args.warmup):
        oracle_conv_sample(spec, d, 32)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        _, n = oracle_conv_sample(spec, d, per_step_pix)
        times.append(time.perf_counter() - t0)
    dt = sum(times)
    ops = 2 * per_step_pix * spec.C_out * spec.K * args.steps
    value = ops / dt / 1e12
    sample = (f"each step: {per_step_pix} of {spec.M} output pixels (full-input scales/codes/"
              f"packing, sampled accumulators + epilogue)")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64 (CPU oracle)",
        "data": "synthetic",
        "config": {"workload": spec.name, "M": spec.M, "N": spec.C_out, "K": spec.K, "bits": d["bits"]},
        "cpu_baseline": {"value": round(value, 6), "unit": "TOPS", "cores": _threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def run_case(args):
    """One kernel family on one workload, for profiling (ncu) and tuning:
    conv_4b8b | conv_1b4b | quant_conv | gemm:MxNxK:lo:hi:frac | gemv:M."""
    import torch
    from paper_2311_14114_gb300 import soniq as sq
    from paper_2311_14114_gb300 import workloads as wl
    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    stream = torch.cuda.current_stream()
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    name = args.case
    if name.startswith("conv") or name == "quant_conv":
        spec = wl.CONV_RESNET_1B4B if name == "conv_1b4b" else wl.CONV_RESNET
        d = wl.make_conv(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
        X = torch.from_numpy(d["X"]).cuda().reshape(-1, spec.C)
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
        Xp, s_a = sq.quantize_act(lay, X)
        cd = sq.conv_desc(spec.batch, spec.H, spec.W, spec.C_out, spec.R, spec.S, spec.stride, spec.pad)
        Y = torch.empty((spec.batch, 14, 14, spec.C_out), dtype=torch.float16, device="cuda")
        if name == "quant_conv":
            fn, ops = (lambda: sq.quantize_act(lay, X, "tensor", s_a=s_a, Ap=Xp)), 0
        else:
            fn, ops = (lambda: sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, Y=Y)), spec.ops
    elif name.startswith("gemm:"):
        _, shape, lo, hi, frac = name.split(":")
        M, N, K = (int(x) for x in shape.split("x"))
        spec = wl.LinearSpec(name, M=M, K=K, N=N, bits_lo=int(lo), bits_hi=int(hi), frac_hi=float(frac))
        d = wl.make_linear(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
        Ap, s_a = sq.quantize_act(lay, torch.from_numpy(d["A"]).cuda())
        Y = torch.empty((M, N), dtype=torch.float16, device="cuda")
        fn, ops = (lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y, flags=sq.FLAG_FORCE_MMA)), spec.ops
    elif name.startswith("gemv:"):
        spec = wl.DECODE[int(name.split(":")[1])]
        d = wl.make_linear(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
        Ap, s_a = sq.quantize_act(lay, torch.from_numpy(d["A"]).cuda())
        Y = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
        fn, ops = (lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y)), spec.ops
    else:
        raise SystemExit(f"unknown case {name}")
    ms = _time_events(fn, args.steps, flush, stream)
    if sq.sync_status() != 0:
        raise RuntimeError("device error")
    print(json.dumps({"case": name, "us": round(ms * 1e3, 2),
                      "TOPS": round(ops / (ms * 1e-3) / 1e12, 2) if ops else None}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="soniq", choices=["soniq", "reference"])
    ap.add_argument("--suite", action="store_true")
    ap.add_argument("--full-sweep", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--case", default=None, help="profile one kernel family on one workload")
    ap.add_argument("--traffic", type=float, default=CONV_TRAFFIC_BYTES,
                    help="DRAM bytes per conv launch from an ncu capture of the current kernel")
    args = ap.parse_args()
    if args.case:
        run_case(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
