#!/usr/bin/env python3
"""Benchmark of SONIQ's inference hot path on GB300.

Headline workload: the precision-sweep GEMM M=8192, K=N=4096 at the point
4-bit low / 8-bit high / 25 % high channels (1024 of 4096 channels at 8 bits),
activations fp16 ~N(0,1), weights ~N(0, 0.02).  One step = one pass of the
per-inference path over the batch:
    soniq_quantize_act (per-tensor max-abs scale + quantize + pack, Sec. 3 steps 1-2)
    soniq_mp_gemm      (exact integer products per precision group + scale epilogue)
Weights are packed once before timing (offline: the layout is fixed after
training).  The metric is effective TOPS = 2 * M * N * K / step time with the
logical (unpadded) K.

The default run also prints a "suite" with every other workload family: the
small linear layer, the ResNet-18 conv (4/8 and 1/4 bits), the MLP
up-projection, the decode GEMV (M = 1, 4, 16; GB/s of packed weights), the
per-tensor quantize (GB/s) and all 60 points of the precision sweep, each as
TOPS or GB/s and as a fraction of its roofline.

--impl reference times the CPU oracle on the same workload (bounded samples,
extrapolated to a full step as stated in its line).
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "mixed-precision GEMM effective TOPS (and GEMV GB/s) and % of roofline on 1 GB300"
L2_FLUSH_BYTES = 256 << 20       # > 129 MB L2
KERNEL_SOURCES = ("paper_2311_14114_gb300/csrc/staged_gemm.cu", "paper_2311_14114_gb300/csrc/tc_ptx.cuh")
# dram__bytes_read.sum + dram__bytes_write.sum of one soniq_mp_gemm call on the
# headline workload (its three kernels: activation expand, weight expand,
# staged tcgen05 GEMM), from one ncu capture, keyed by the sha256 of the
# kernel sources it was captured with: a different source reports null.
TRAFFIC = {"sha256": "2060e0fb153469afb64f575cabc46f15742c583ec4c60635a20cdff1b7dac587",
           "bytes": 157481984,
           "capture": "ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum: expansion (activations and weights, one launch) 31.58 MB read + 2.55 MB written, staged 2-SM GEMM 82.04 MB read + 41.32 MB written (one call)"}


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return dict(hbm=float(d["hbm_gbs"]), bf16=float(d["bf16_tflops"]),
                    bf16_sus=float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


def kernel_sha():
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def headline_spec():
    from paper_2311_14114_gb300 import workloads as wl
    return wl.SWEEP_HEADLINE


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
# rooflines
# --------------------------------------------------------------------------

def group_kinds(bits_a, bits_w, codes=None, N=None):
    """Tensor pipe of each group on the staged path: 0 = E4M3 (codes <= 4 bits
    on both sides), 1 = fp16, 2 = E2M1 (codes <= 2 bits on both sides, when such
    groups hold at least 60 % of the padded weight codes `codes`, the row holds
    at least 2048 of them, and 240-column tiles pad N by at most 7 %: the rule
    the library applies)."""
    kinds = [0 if (a <= 4 and w <= 4) else 1 for a, w in zip(bits_a, bits_w)]
    if codes is not None and N is not None and sum(codes) >= 2048 and -(-N // 240) * 240 * 100 <= N * 107:
        elig = [a <= 2 and w <= 2 and c > 0 for a, w, c in zip(bits_a, bits_w, codes)]
        if 5 * sum(c for c, e in zip(codes, elig) if e) >= 3 * sum(codes):
            kinds = [2 if e else k for k, e in zip(kinds, elig)]
    return kinds


def padded_codes(count, pad_unit=128, taps=1):
    """Padded weight codes per group (the staged path's K per group)."""
    ru = lambda x, u: (x + u - 1) // u * u
    return [ru(taps * ru(c, pad_unit), 128) if c > 0 else 0 for c in count]


def mixed_peak(ops, kinds, pk):
    """Tensor peak for work that runs ops[g] on the pipe of kinds[g] (E4M3 at
    2x the measured bf16 rate and E2M1 at 6x, the nominal fp8:bf16 and
    fp4:bf16 dense ratios; fp16 at the bf16 rate), time-weighted over the groups."""
    ratio = {0: 2.0, 1: 1.0, 2: 6.0}
    t = sum(o / (pk["bf16"] * ratio[k]) for o, k in zip(ops, kinds) if o > 0)
    return sum(ops) / t if t > 0 else pk["bf16"]


def linear_ops(M, N, count):
    return [2 * M * N * c for c in count]


def quant_bytes(M, K, count, bits):
    """Algorithmic bytes of an activation quantize: fp16 read + packed codes written."""
    return M * K * 2 + M * sum(c * b for c, b in zip(count, bits)) / 8


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------

def _graph(fn, stream):
    import torch
    side = torch.cuda.Stream()
    side.wait_stream(stream)
    with torch.cuda.stream(side):
        fn()                                # scratch buffers of this stream exist before capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        fn()
    return g


def _time_graph(g, steps, flush, stream, warm=3):
    """Per-replay device times (ms) of a captured graph; L2 flushed before each
    replay, outside the events."""
    import torch
    for _ in range(warm):
        flush.zero_()
        g.replay()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for i in range(steps):
        flush.zero_()
        ev[i][0].record(stream)
        g.replay()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in ev]


def max_over_ranks(x, world, device):
    """The largest x over the ranks of the process group (x itself for one
    rank): the job's time is its slowest replica's."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t[0])


def job_tops(ops_per_rank, ms_per_step, world):
    """Whole-job throughput: the operations of every replica over the slowest
    replica's time per step."""
    return world * ops_per_rank / (ms_per_step * 1e-3) / 1e12


def _time_fn(fn, steps, flush, stream):
    """Mean device time (ms) of a library call replayed as a CUDA graph (the
    mean, not the median: event timestamps here tick in steps of about 2 us,
    which a median of short calls would keep)."""
    return statistics.mean(_time_graph(_graph(fn, stream), steps, flush, stream))


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

    spec = headline_spec()
    d = wl.make_linear(spec)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    stream = torch.cuda.current_stream()
    A = torch.from_numpy(d["A"]).cuda()
    Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
    Ap = torch.empty((spec.M, lay.row_bytes()), dtype=torch.uint8, device="cuda")
    s_a = torch.empty(2, dtype=torch.float32, device="cuda")
    Y = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")

    def quant():
        sq.quantize_act(lay, A, "tensor", s_a=s_a, Ap=Ap)

    def gemm():
        sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y)

    def step():
        quant()
        gemm()

    for _ in range(max(args.warmup, 3)):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    if sq.sync_status() != 0:
        raise RuntimeError("device error during warm-up")

    # The device-timed steps replay a CUDA graph of the two library calls (as a
    # serving loop would), so host call overhead does not sit between the
    # events; the end-to-end number below goes through the plain API calls.
    n0 = sq.launch_count()
    g_step = _graph(step, stream)
    launches_per_step = (sq.launch_count() - n0) // 2     # the call before capture and the captured one
    g_quant, g_gemm = _graph(quant, stream), _graph(gemm, stream)

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    step_ms = _time_graph(g_step, args.steps, flush, stream, warm=max(args.warmup, 3))
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    if sq.sync_status() != 0:
        raise RuntimeError("device error during the timed steps")
    launches = launches_per_step * args.steps
    # the two kernels alone, same flush and replay discipline
    gemm_ms = _time_graph(g_gemm, args.steps, flush, stream)
    quant_ms = _time_graph(g_quant, args.steps, flush, stream)
    total_ms = max_over_ranks(sum(step_ms), world, "cuda")
    ms_per_step = total_ms / args.steps
    ops = spec.ops
    value = job_tops(ops, ms_per_step, world)

    # ---- end to end through host buffers ----
    # Every step uploads its own input from pinned host memory, runs the two
    # API calls and reads its output back.  As in a serving loop, the copies of
    # neighbouring steps overlap this step's kernels: uploads, kernels and
    # downloads run on three streams with two sets of buffers.
    NB = 2
    Ah = [torch.from_numpy(d["A"]).pin_memory() for _ in range(NB)]
    Yh = [torch.empty((spec.M, spec.N), dtype=torch.float16).pin_memory() for _ in range(NB)]
    Ad = [torch.empty_like(A) for _ in range(NB)]
    Apd = [torch.empty_like(Ap) for _ in range(NB)]
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
                s_up.wait_event(cmp_done[k])          # the kernels of step i - NB have read Ad[k]
            Ad[k].copy_(Ah[k], non_blocking=True)
            up_done[k].record(s_up)
        with torch.cuda.stream(s_cmp):
            s_cmp.wait_event(up_done[k])
            if used[k]:
                s_cmp.wait_event(down_done[k])        # Yd[k] of step i - NB has been read back
            sq.quantize_act(lay, Ad[k], "tensor", s_a=sad[k], Ap=Apd[k], stream=s_cmp)
            sq.mp_gemm(lay, Apd[k], sad[k], Wp, s_w, Y=Yd[k], stream=s_cmp)
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
    e2e_ms = max_over_ranks(e_start.elapsed_time(e_end) / args.steps, world, "cuda")
    e2e_value = job_tops(ops, e2e_ms, world)

    # ---- roofline of the dominant kernel (the tensor-core GEMM) ----
    gemm_avg = statistics.mean(gemm_ms)
    achieved = ops / (gemm_avg * 1e-3) / 1e12
    kinds = group_kinds(d["bits"], d["bits"], padded_codes(d["count"]), spec.N)
    peak = mixed_peak(linear_ops(spec.M, spec.N, d["count"]), kinds, pk)
    sha = kernel_sha()
    traffic = TRAFFIC["bytes"] if TRAFFIC["sha256"] == sha else None
    roofline = {"kernel": "soniq_mp_gemm call (operand expand + staged tcgen05 GEMM)", "bound": "tensor",
                "achieved": round(achieved, 2), "peak": round(peak, 1), "unit": "TFLOP/s",
                "frac": round(achieved / peak, 4), "traffic": traffic,
                "peak_source": f"{pk['src']}: bf16 {pk['bf16']} TFLOP/s burst; E4M3 = 2x bf16 "
                               f"(nominal ratio), fp16 = bf16 rate; time-weighted over the groups",
                "gemm_us": round(gemm_avg * 1e3, 2),
                "quantize_us": round(statistics.mean(quant_ms) * 1e3, 2),
                "quantize_GBps": round(quant_bytes(spec.M, spec.K, d["count"], d["bits"])
                                       / (statistics.mean(quant_ms) * 1e-3) / 1e9, 1)}

    out = {"metric": METRIC, "value": round(value, 3), "unit": "TOPS", "n_gpus": world,
           "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": round(ms_per_step, 5),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "u8xs8->i32 (E4M3/fp16 tensor pipes, exact)", "data": "synthetic",
           "config": headline_config(spec, d, world),
           "e2e": {"value": round(e2e_value, 3), "unit": "TOPS",
                   "h2d_bytes_per_step": int(Ah[0].numel() * 2), "d2h_bytes_per_step": int(Yh[0].numel() * 2),
                   "ms_per_step": round(e2e_ms, 5),
                   "pipelining": "upload, kernels and download of neighbouring steps overlap (3 streams, 2 buffer sets)"},
           "gpu_launches": int(launches),
           "roofline": roofline,
           "clocks": clk}
    if not args.no_suite:
        out["suite"] = run_suite(args, sq, wl, pk, flush, d)
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(args.cpu_seconds)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


def headline_config(spec, d, world):
    """The `config` of both arms' lines (identical)."""
    return {"workload": spec.name, "M": spec.M, "N": spec.N, "K": spec.K, "bits": d["bits"],
            "count": d["count"], "parallelism": f"replicas{world}",
            "l2": "flushed between timed steps (256 MB write)",
            "launch": "the step (both library calls) replayed as one CUDA graph; e2e: plain API calls"}


def run_suite(args, sq, wl, pk, flush, head):
    """Every workload family, each library call replayed as a CUDA graph after
    an L2 flush (mean of the replays)."""
    import torch
    stream = torch.cuda.current_stream()
    steps = max(5, args.suite_steps)
    rows = []

    def linear_case(spec, d=None, gemv=False):
        d = wl.make_linear(spec) if d is None else d
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        A = torch.from_numpy(d["A"]).cuda()
        W = torch.from_numpy(d["W"]).cuda()
        Wp, s_w = sq.pack_weights(lay, W)
        Ap, s_a = sq.quantize_act(lay, A)
        Y = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
        gemm_ms = _time_fn(lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y), steps, flush, stream)
        quant_ms = _time_fn(lambda: sq.quantize_act(lay, A, "tensor", s_a=s_a, Ap=Ap), steps, flush, stream)
        ops = spec.ops
        r = {"workload": spec.name, "M": spec.M, "N": spec.N, "K": spec.K, "bits": d["bits"],
             "count": d["count"], "gemm_us": round(gemm_ms * 1e3, 2),
             "TOPS": round(ops / (gemm_ms * 1e-3) / 1e12, 2), "quantize_us": round(quant_ms * 1e3, 2),
             "quantize_GBps": round(quant_bytes(spec.M, spec.K, d["count"], d["bits"]) / (quant_ms * 1e-3) / 1e9, 1)}
        if gemv:
            wbytes = sum(c * b for c, b in zip(d["count"], d["bits"])) / 8 * spec.N
            gbs = wbytes / (gemm_ms * 1e-3) / 1e9
            r["path"] = sq.gemm_path(lay, spec.M, spec.N)
            r["GBps_packed_weights"] = round(gbs, 1)
            r["frac_hbm_measured"] = round(gbs / pk["hbm"], 4)
            r["frac_hbm_8TBps"] = round(gbs / 8000.0, 4)
            r["weight_bytes_algorithmic"] = int(wbytes)
            r["weight_bytes_moved"] = int(Wp.numel() + s_w.numel() * 4)
        else:
            staged = sq.gemm_path(lay, spec.M, spec.N).startswith("tensor-core staged")
            kinds = group_kinds(d["bits"], d["bits"], padded_codes(d["count"]) if staged else None, spec.N)
            peak = mixed_peak(linear_ops(spec.M, spec.N, d["count"]), kinds, pk)
            r["frac_tensor_peak"] = round(ops / (gemm_ms * 1e-3) / 1e12 / peak, 4)
            r["peak_TFLOPs"] = round(peak, 1)
        rows.append(r)
        del A, W, Wp, Ap, Y

    def conv_case(spec):
        d = wl.make_conv(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
        X = torch.from_numpy(d["X"]).cuda().reshape(-1, spec.C)
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
        Xp, s_a = sq.quantize_act(lay, X)
        cd = sq.conv_desc(spec.batch, spec.H, spec.W, spec.C_out, spec.R, spec.S, spec.stride, spec.pad)
        P, Q = sq.conv_out_hw(cd)
        Y = torch.empty((spec.batch, P, Q, spec.C_out), dtype=torch.float16, device="cuda")
        ms = _time_fn(lambda: sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, Y=Y), steps, flush, stream)
        qms = _time_fn(lambda: sq.quantize_act(lay, X, "tensor", s_a=s_a, Ap=Xp), steps, flush, stream)
        ops = [2 * spec.M * spec.C_out * spec.R * spec.S * c for c in d["count"]]
        # the bench's convolutions take the staged path (E2M1 where the plan uses it)
        peak = mixed_peak(ops, group_kinds(d["bits"], d["bits"], padded_codes(d["count"], 32, spec.R * spec.S),
                                           spec.C_out), pk)
        qb = quant_bytes(spec.batch * spec.H * spec.W, spec.C, d["count"], d["bits"])
        rows.append({"workload": spec.name, "M": spec.M, "N": spec.C_out, "K": spec.K, "bits": d["bits"],
                     "count": d["count"], "conv_us": round(ms * 1e3, 2),
                     "TOPS": round(spec.ops / (ms * 1e-3) / 1e12, 2),
                     "frac_tensor_peak": round(spec.ops / (ms * 1e-3) / 1e12 / peak, 4),
                     "peak_TFLOPs": round(peak, 1), "quantize_us": round(qms * 1e3, 2),
                     "quantize_GBps": round(qb / (qms * 1e-3) / 1e9, 1),
                     "quantize_frac_hbm": round(qb / (qms * 1e-3) / 1e9 / pk["hbm"], 4)})

    def fused_quant_case(spec, bits2, frac2):
        """The layer's epilogue writing the next layer's packed codes (quantize-in-
        epilogue) against the unfused pair: fp16 outputs, then soniq_quantize_act
        with the next layer's calibrated scales."""
        d = wl.make_linear(spec)
        perm2, count2, _ = wl.assignment(np.random.default_rng(spec.seed + 1), spec.N, frac2, 0)
        lay2 = sq.Layout(perm2, count2, bits2)
        order = sq.next_layer_row_order(lay2)
        Wa = np.zeros((len(order), spec.K), np.float32)
        Wa[order >= 0] = d["W"][order[order >= 0]]
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(Wa).cuda())
        A = torch.from_numpy(d["A"]).cuda()
        Ap, s_a = sq.quantize_act(lay, A)
        s2 = torch.tensor([0.6, 1.8], dtype=torch.float32, device="cuda")
        nxt = sq.NextLayer(lay2, s2, M=spec.M)
        Y = torch.empty((spec.M, len(order)), dtype=torch.float16, device="cuda")
        X2 = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
        Ap2 = torch.empty_like(nxt.Ap)
        cols = torch.from_numpy(np.flatnonzero(order >= 0)).cuda()
        chans = torch.from_numpy(order[order >= 0]).cuda()

        def unfused():
            sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y)
            X2[:, chans] = Y[:, cols]          # the next layer's input in channel order (not timed below)
            sq.quantize_act(lay2, X2, "calibrated", s_a=s2, Ap=Ap2)

        gemm_ms = _time_fn(lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y), steps, flush, stream)
        unfused()
        q_ms = _time_fn(lambda: sq.quantize_act(lay2, X2, "calibrated", s_a=s2, Ap=Ap2), steps, flush, stream)
        fused_ms = _time_fn(lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y, next=nxt), steps, flush, stream)
        codes_ms = _time_fn(lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, next=nxt, write_y=False), steps, flush,
                            stream)
        same = bool(torch.equal(nxt.Ap, Ap2))
        rows.append({"workload": spec.name + "_then_next_layer_quantize", "M": spec.M, "N": len(order),
                     "K": spec.K, "bits": d["bits"], "next_bits": bits2, "next_count": count2,
                     "gemm_us": round(gemm_ms * 1e3, 2), "separate_quantize_us": round(q_ms * 1e3, 2),
                     "unfused_us": round((gemm_ms + q_ms) * 1e3, 2), "fused_us": round(fused_ms * 1e3, 2),
                     "fused_codes_only_us": round(codes_ms * 1e3, 2), "codes_identical": same})

    linear_case(wl.LINEAR_SMALL)
    def phase2_case(spec):
        """Algorithm 1 Phase II forward: every step quantizes both fp32 master
        weight matrices and the activations on the fly, then runs the GEMMs."""
        from paper_2311_14114_gb300.phase2 import FakeQuantMLP
        d = wl.make_phase2(spec)
        net = FakeQuantMLP(d["layers"], M=spec.M, sub_k=spec.sub_k)
        X = torch.from_numpy(d["X"]).cuda()
        step_ms = _time_fn(lambda: net.forward(X), steps, flush, stream)
        macs = sum(K * N for K, N in zip(spec.widths[:-1], spec.widths[1:])) * spec.M
        pack_ms = sum(_time_fn(lambda i=i: sq.pack_weights(net.layouts[i], net.W[i], Wp=net.Wp[i], s_w=net.s_w[i]),
                               steps, flush, stream) for i in range(len(net.layouts)))
        rows.append({"workload": spec.name, "M": spec.M, "widths": list(spec.widths), "bits": list(spec.bits),
                     "step_us": round(step_ms * 1e3, 2), "TOPS": round(2 * macs / (step_ms * 1e-3) / 1e12, 2),
                     "weight_quantize_us": round(pack_ms * 1e3, 2),
                     "step": "pack both fp32 weight matrices, quantize the activations, GEMM, per layer"})

    fused_quant_case(wl.MLP_UP, [2, 8], 0.2)
    phase2_case(wl.PHASE2_MLP)
    conv_case(wl.CONV_RESNET)
    conv_case(wl.CONV_RESNET_1B4B)
    linear_case(wl.MLP_UP)
    for m in (1, 4, 16):
        linear_case(wl.DECODE[m], gemv=True)
    # the 60 sweep points share the headline point's seeded A and W draws; each
    # point has its own seeded precision assignment (same as its own workload's)
    for s in wl.sweep_specs():
        perm, count, _ = wl.assignment(np.random.default_rng(s.seed), s.K, s.frac_hi, s.n_outliers)
        d = dict(A=head["A"], W=head["W"], perm=perm, count=count, bits=[s.bits_lo, s.bits_hi])
        try:
            linear_case(s, d)
        except Exception as e:  # report, do not hide
            rows.append({"workload": s.name, "error": str(e)})
    return rows


# --------------------------------------------------------------------------
# CPU oracle (baseline leg and the reference arm)
# --------------------------------------------------------------------------

def _threads():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_step_parts(d, rows, s_w=None, J=None):
    """The oracle's pipeline for one headline step, in two timed parts:
    per-tensor scales, codes and packing of the whole input (t_q), and exact
    accumulators plus the fp64 epilogue for the output rows `rows` (t_acc).
    Weight codes are made once, outside the timing (offline in both arms)."""
    import oracle
    if J is None:
        s_w = oracle.weight_scales(d["W"], d["perm"], d["count"])
        J = oracle.weight_codes(d["W"], d["perm"], d["count"], d["bits"], s_w)
    t0 = time.perf_counter()
    A32 = d["A"].astype(np.float32)
    s_a = oracle.act_scales(A32, d["perm"], d["count"])
    U = oracle.act_codes(A32, d["perm"], d["count"], d["bits"], s_a)
    oracle.pack_act_rows(U, d["count"], d["bits"], 128)
    t1 = time.perf_counter()
    acc = oracle.gemm_acc(U, J, d["count"], rows=rows)
    oracle.epilogue(acc, s_a, s_w, d["bits"], d["bits"], rows=rows)
    t2 = time.perf_counter()
    return t1 - t0, t2 - t1, s_w, J


def oracle_worker(args):
    """Runs in a child process (OMP_NUM_THREADS set by the parent): times the
    oracle on the headline workload and prints one JSON line."""
    from paper_2311_14114_gb300 import workloads as wl
    import oracle
    oracle.build()
    spec = headline_spec()
    d = wl.make_linear(spec)
    rng = np.random.default_rng(0)
    probe = np.sort(rng.choice(spec.M, size=8, replace=False))
    tq, ta, s_w, J = oracle_step_parts(d, probe)
    per_row = ta / len(probe)
    n = int(min(spec.M, max(8, (args.cpu_seconds - tq) / max(per_row, 1e-6))))
    rows = np.sort(rng.choice(spec.M, size=n, replace=False))
    tq, ta, _, _ = oracle_step_parts(d, rows, s_w, J)
    print(json.dumps({"t_q": tq, "t_acc": ta, "rows": n, "M": spec.M}), flush=True)


def _oracle_child(threads, seconds):
    env = dict(os.environ, OMP_NUM_THREADS=str(threads))
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-worker",
                        "--cpu-seconds", str(seconds)], capture_output=True, text=True, env=env, timeout=900)
    if r.returncode != 0:
        raise RuntimeError(f"oracle worker failed: {r.stderr[-2000:]}")
    return json.loads(r.stdout.strip().splitlines()[-1])


def _extrapolated(res, ops_full):
    """Full-step oracle time: the whole-input quantize plus the sampled
    accumulator time scaled to all M rows; returns (TOPS, step seconds)."""
    t_step = res["t_q"] + res["t_acc"] * res["M"] / res["rows"]
    return ops_full / t_step / 1e12, t_step


def cpu_baseline(budget_s=12.0):
    spec = headline_spec()
    cores = _threads()
    one = _oracle_child(1, budget_s)
    allc = _oracle_child(cores, budget_s)
    v1, t1 = _extrapolated(one, spec.ops)
    va, ta = _extrapolated(allc, spec.ops)
    return {"value": round(va, 6), "unit": "TOPS", "cores": cores, "kind": "oracle",
            "sample": (f"headline workload; per-tensor scales, codes and packing of all {spec.M} rows "
                       f"({allc['t_q']:.2f} s), exact accumulators + fp64 epilogue for {allc['rows']} sampled "
                       f"output rows ({allc['t_acc']:.2f} s), scaled to a full step of {ta:.1f} s"),
            "single_thread": {"value": round(v1, 6), "unit": "TOPS", "cores": 1,
                              "sample": f"{one['rows']} sampled rows, full step {t1:.1f} s"}}


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2311_14114_gb300 import workloads as wl
    import oracle
    oracle.build()
    spec = headline_spec()
    d = wl.make_linear(spec)
    rng = np.random.default_rng(1)
    rows_per_step = 16
    s_w = J = None
    for _ in range(args.warmup):
        _, _, s_w, J = oracle_step_parts(d, np.arange(2), s_w, J)
    t_steps = []
    for _ in range(args.steps):
        rows = np.sort(rng.choice(spec.M, size=rows_per_step, replace=False))
        tq, ta, s_w, J = oracle_step_parts(d, rows, s_w, J)
        t_steps.append(tq + ta * spec.M / rows_per_step)
    t_step = sum(t_steps) / len(t_steps)
    value = spec.ops / t_step / 1e12
    sample = (f"each step: per-tensor scales, codes and packing of all {spec.M} rows, exact accumulators + "
              f"fp64 epilogue for {rows_per_step} sampled output rows, scaled to all rows")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(t_step * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64 (CPU oracle)",
        "data": "synthetic",
        "config": headline_config(spec, d, world),
        "cpu_baseline": {"value": round(value, 6), "unit": "TOPS", "cores": _threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def run_case(args):
    """One kernel family on one workload, for profiling (ncu) and tuning:
    headline | quant_headline | conv_4b8b | conv_1b4b | quant_conv | mlp_next | mlp_next_codes |
    gemm:MxNxK:lo:hi:frac | quant:MxNxK:lo:hi:frac | gemv:M."""
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
    elif name.startswith(("gemm:", "quant:")) or name in ("headline", "quant_headline"):
        if name.startswith(("gemm:", "quant:")):
            _, shape, lo, hi, frac = name.split(":")
            M, N, K = (int(x) for x in shape.split("x"))
            spec = wl.LinearSpec(name, M=M, K=K, N=N, bits_lo=int(lo), bits_hi=int(hi), frac_hi=float(frac))
        else:
            spec = headline_spec()
        d = wl.make_linear(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
        A = torch.from_numpy(d["A"]).cuda()
        Ap, s_a = sq.quantize_act(lay, A)
        Y = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
        if name == "quant_headline" or name.startswith("quant:"):
            fn, ops = (lambda: sq.quantize_act(lay, A, "tensor", s_a=s_a, Ap=Ap)), 0
        else:
            fn, ops = (lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y, flags=args.flags)), spec.ops
    elif name in ("mlp_next", "mlp_next_codes"):
        # the MLP up-projection whose epilogue writes the next layer's codes
        spec = wl.MLP_UP
        d = wl.make_linear(spec)
        perm2, count2, _ = wl.assignment(np.random.default_rng(spec.seed + 1), spec.N, 0.2, 0)
        lay2 = sq.Layout(perm2, count2, [2, 8])
        order = sq.next_layer_row_order(lay2)
        Wa = np.zeros((len(order), spec.K), np.float32)
        Wa[order >= 0] = d["W"][order[order >= 0]]
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(Wa).cuda())
        Ap, s_a = sq.quantize_act(lay, torch.from_numpy(d["A"]).cuda())
        nxt = sq.NextLayer(lay2, torch.tensor([0.6, 1.8], dtype=torch.float32, device="cuda"), M=spec.M)
        Y = torch.empty((spec.M, len(order)), dtype=torch.float16, device="cuda")
        wy = name == "mlp_next"
        fn, ops = (lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y if wy else None, next=nxt, write_y=wy)), spec.ops
    elif name.startswith("gemv:"):
        spec = wl.DECODE[int(name.split(":")[1])]
        d = wl.make_linear(spec)
        lay = sq.Layout(d["perm"], d["count"], d["bits"])
        Wp, s_w = sq.pack_weights(lay, torch.from_numpy(d["W"]).cuda())
        Ap, s_a = sq.quantize_act(lay, torch.from_numpy(d["A"]).cuda())
        Y = torch.empty((spec.M, spec.N), dtype=torch.float16, device="cuda")
        fn, ops = (lambda: sq.mp_gemm(lay, Ap, s_a, Wp, s_w, Y=Y, flags=args.flags)), spec.ops
    else:
        raise SystemExit(f"unknown case {name}")
    ms = _time_fn(fn, args.steps, flush, stream)
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
    ap.add_argument("--no-suite", action="store_true", help="skip the per-workload suite")
    ap.add_argument("--suite-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--case", default=None, help="time one kernel family on one workload")
    ap.add_argument("--flags", type=int, default=0, help="soniq_mp_gemm flags for --case")
    ap.add_argument("--oracle-worker", action="store_true", help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.oracle_worker:
        oracle_worker(args)
    elif args.case:
        run_case(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
