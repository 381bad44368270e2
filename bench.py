#!/usr/bin/env python
"""Benchmark of the FP8 / NVFP4 quantized linear layer on GB300.

A step is one pass of the NVFP4 linear of the denoiser's MLP up-projection
(x [4608, 3072] bf16, W [12288, 3072]): dynamic NVFP4 activation quantization
(amax + quantize), then the block-scaled tensor-core GEMM whose epilogue writes
the bf16 output [4608, 12288] and re-quantizes it to NVFP4 for the next layer
with a calibrated static scale.  The weight is quantized offline (once).
Metric: TFLOP/s of the step (2*M*N*K per step), higher is better.

The JSON line also carries measurements of the other hot-path rows (quantizer
GB/s, FP8 GEMM, small-M translator linears, the 8-block linear stack) under
"rows", the roofline of the dominant kernel, an end-to-end number through the
public API with host buffers, and the CPU oracle timed on the host cores.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

M, K, N = 4608, 3072, 12288
STEP_FLOPS = 2 * M * N * K
EV_EVERY = 8                     # timing events bracket one GEMM in this many steps
WORKLOAD = "nvfp4_mlp_up_4608x12288x3072_fused"
L2_BYTES = 129 * 2 ** 20
FP4_PER_BF16 = 13.5 / 2.25       # nominal dense FP4 : BF16 tensor rate
FP8_PER_BF16 = 4.5 / 2.25


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=16384)
    ap.add_argument("--warmup", type=int, default=32)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-rows", action="store_true", help="skip the secondary row measurements")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return {"hbm_gbs": p["hbm_gbs"], "bf16": p["bf16_tflops"],
                "bf16_sustained": p.get("bf16_tflops_sustained", p["bf16_tflops"]),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


# ------------------------------------------------------------ distributed --

class Dist:
    """One process per GPU (torchrun env).  Ranks run independent replicas of
    the workload (weak scaling); the only collectives are a barrier and a max
    over ranks of the timed duration."""

    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local_rank = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch
            import torch.distributed as dist
            backend = "nccl" if torch.cuda.is_available() else "gloo"
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self):
        if self.pg is not None:
            self.pg.barrier()

    def max(self, v: float) -> float:
        if self.pg is None:
            return v
        import torch
        dev = "cuda" if torch.cuda.is_available() and self.pg.get_backend() == "nccl" else "cpu"
        t = torch.tensor([float(v)], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg is not None:
            self.pg.destroy_process_group()


# ----------------------------------------------------------------- clocks --

class Clocks:
    """nvidia-smi samples (every 200 ms) taken while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(index), f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.count(",") >= 8]
        os.unlink(self.f.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": float(rows[0][2]),
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max(float(r[3]) for r in rows)}


# ------------------------------------------------------------- our arm ---

def to_dev(bits, torch):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def graph_of(fn, torch, stream):
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    return g


def timed(fn, reps: int, torch, stream):
    """Device time per call of fn (a graph replay or a launch sequence), with
    events on the launching stream, synchronised on both sides."""
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        fn()
    b.record(stream)
    b.synchronize()
    return a.elapsed_time(b) / 1e3 / reps


def run_ours(args, dist: Dist):
    import torch

    from paper_2609_21849_gb300 import build, qlin, synthetic
    build.build()
    qlin.load_library()
    torch.cuda.set_device(dist.local_rank)
    pk = peaks()
    fp4_peak = pk["bf16"] * FP4_PER_BF16
    fp8_peak = pk["bf16"] * FP8_PER_BF16
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)

    # ---- workload: R rotating input/output sets, together larger than L2
    x_bits, w_bits = synthetic.nvfp4_mlp_up()
    R = 4
    xs = [to_dev(x_bits, torch) for _ in range(R)]
    w_dev = to_dev(w_bits, torch)
    ws = qlin.alloc_workspace()
    Wq = [qlin.qlin_quantize_weight(w_dev, qlin.QLIN_FMT_NVFP4, workspace=ws) for _ in range(R)]
    del w_dev
    As = [qlin.alloc_nvfp4(M, K) for _ in range(R)]
    wss = [qlin.alloc_workspace() for _ in range(R)]
    ys = [torch.empty((M, N), dtype=torch.bfloat16, device="cuda") for _ in range(R)]
    yqs = [qlin.alloc_nvfp4(M, N) for _ in range(R)]
    # calibration (post-training): dynamic scale of a first run's output
    qlin.qlin_quantize_act_nvfp4(xs[0], None, As[0], wss[0])
    qlin.qlin_gemm_nvfp4(As[0], Wq[0], ys[0])
    cal = qlin.qlin_quantize_act_nvfp4(ys[0])
    next_scale = cal.tensor_scale.clone()
    del cal
    torch.cuda.synchronize()
    set_bytes = (M * K * 2 + M * K // 2 + Wq[0].codes.numel() + Wq[0].scales.numel()
                 + M * N * 2 + M * N // 2 + yqs[0].scales.numel())

    def step(r):
        qlin.qlin_quantize_act_nvfp4(xs[r], None, As[r], wss[r])
        qlin.qlin_linear_fused(As[r], Wq[r], ys[r], next_scale, yqs[r])

    # one graph holds S steps, replayed back to back for the timed region.
    # Timing events (external event nodes) bracket one GEMM in EV_EVERY: an
    # event node between two kernels breaks their programmatic launch overlap
    # (measured: events around every GEMM stretched the step from 87 to
    # 100 us), so the GEMM's duration is sampled rather than bracketed
    # everywhere.
    S = 4 * R
    try:
        evs = [(torch.cuda.Event(enable_timing=True, external=True),
                torch.cuda.Event(enable_timing=True, external=True))
               for _ in range(S // EV_EVERY)]
    except TypeError:
        evs = None

    def s_steps():
        for i in range(S):
            r = i % R
            timed_gemm = evs is not None and i % EV_EVERY == 0
            qlin.qlin_quantize_act_nvfp4(xs[r], None, As[r], wss[r])
            if timed_gemm:
                evs[i // EV_EVERY][0].record(stream)
            qlin.qlin_linear_fused(As[r], Wq[r], ys[r], next_scale, yqs[r])
            if timed_gemm:
                evs[i // EV_EVERY][1].record(stream)

    for r in range(R):          # first launches outside capture (attributes)
        step(r)
    torch.cuda.synchronize()
    g = graph_of(s_steps, torch, stream)
    replays = max(1, args.steps // S)
    steps = replays * S
    warm = max(1, -(-args.warmup // S))
    for _ in range(warm):
        g.replay()
    torch.cuda.synchronize()

    dist.barrier()
    torch.cuda.synchronize()
    clocks = Clocks(dist.local_rank)
    time.sleep(0.25)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(replays):
        g.replay()
    t1.record(stream)
    t1.synchronize()
    clk = clocks.stop()
    torch.cuda.synchronize()
    dist.barrier()
    sec = dist.max(t0.elapsed_time(t1) / 1e3)
    per_step = sec / steps
    value = STEP_FLOPS * steps * dist.world / sec / 1e12

    if evs:
        gemm_s = statistics.mean(a.elapsed_time(b) for a, b in evs) / 1e3
    else:
        gemm_s = timed(lambda: qlin.qlin_linear_fused(As[0], Wq[0], ys[0], next_scale, yqs[0]),
                       200, torch, stream)
    gemm_tflops = STEP_FLOPS / gemm_s / 1e12

    # ---- end to end through the public API with host buffers: every step
    # copies its x in from pinned host memory and its y out to pinned host
    # memory inside the timed region.  The copies run on streams of their own,
    # so one step's compute overlaps the next step's input copy and the
    # previous step's output copy, as a serving loop does; events keep each
    # step's copy-in -> compute -> copy-out order and each set's reuse order.
    x_host = torch.from_numpy(x_bits.view(np.int16)).pin_memory()
    y_hosts = [torch.empty((M, N), dtype=torch.int16).pin_memory() for _ in range(R)]
    # (the output copy, 113 MB, runs at ~190 GB/s device -> host; splitting it
    # over several streams measured no faster)
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(R)]
    ev_comp = [torch.cuda.Event() for _ in range(R)]
    ev_out = [torch.cuda.Event() for _ in range(R)]

    def e2e_step(i):
        r = i % R
        s_in.wait_event(ev_comp[r])             # the set's last compute has read xs[r]
        with torch.cuda.stream(s_in):
            xs[r].view(torch.int16).copy_(x_host, non_blocking=True)
        ev_in[r].record(s_in)
        stream.wait_event(ev_in[r])
        stream.wait_event(ev_out[r])            # the set's last output has been read
        with torch.cuda.stream(stream):
            step(r)
        ev_comp[r].record(stream)
        s_out.wait_event(ev_comp[r])
        with torch.cuda.stream(s_out):
            y_hosts[r].copy_(ys[r].view(torch.int16), non_blocking=True)
        ev_out[r].record(s_out)

    def e2e_run(n):
        torch.cuda.synchronize()
        for r in range(R):
            ev_comp[r].record(stream)
            ev_out[r].record(stream)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        s_in.wait_event(a)
        s_out.wait_event(a)
        for i in range(n):
            e2e_step(i)
        for r in range(R):
            stream.wait_event(ev_out[r])
        b.record(stream)
        b.synchronize()
        return a.elapsed_time(b) / 1e3 / n

    e2e_run(2 * R)                              # warm-up
    n_e2e = max(4 * R, min(200, steps // 10))
    e2e_sec = dist.max(e2e_run(n_e2e))
    e2e = {"value": round(STEP_FLOPS * dist.world / e2e_sec / 1e12, 2), "unit": "TFLOP/s",
           "h2d_bytes_per_step": M * K * 2, "d2h_bytes_per_step": M * N * 2,
           "ms_per_step": round(e2e_sec * 1e3, 4),
           "copies": "pinned host buffers; input copy, compute and output copy on three "
                     "streams, consecutive steps overlapped"}

    traffic = committed_traffic()
    out = {
        "metric": "NVFP4 quantized-linear throughput (TFLOP/s, 2*M*N*K per step)",
        "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": dist.world, "steps": steps,
        "warmup": warm * S, "ms_per_step": round(per_step * 1e3, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "nvfp4 (e2m1 x e4m3 block scales), fp32 accumulate, bf16 out",
        "data": "synthetic (seeded; shapes of FLUX.2-klein at 1024^2, random weights)",
        "config": {"workload": WORKLOAD, "M": M, "N": N, "K": K,
                   "step": "dynamic NVFP4 act quant (one read of x: grid-wide amax + quant) + NVFP4 GEMM + bf16 out + fused NVFP4 requant",
                   "l2": f"{R} rotating input/output sets of {set_bytes / 2**20:.0f} MiB each (> 129 MiB L2)",
                   "graph": f"CUDA graph of {S} steps replayed {replays}x",
                   "gemm_timing": f"CUDA events around 1 GEMM in {EV_EVERY} inside the timed graph",
                   "parallelism": f"replicas x{dist.world}"},
        "gpu_launches": 2 * steps,
        "clocks": clk,
        "e2e": e2e,
        "roofline": {"kernel": "gemm_kernel<nvfp4, BN=256, requant>", "bound": "tensor",
                     "achieved": round(gemm_tflops, 1),
                     "peak": round(fp4_peak, 1), "unit": "TFLOP/s",
                     "peak_source": f"{pk['source']} bf16 burst {pk['bf16']} TFLOP/s x nominal FP4:BF16 {FP4_PER_BF16:g}",
                     "frac": round(gemm_tflops / fp4_peak, 4),
                     "traffic": traffic,
                     "algorithmic": f"{STEP_FLOPS / 1e9:.2f} GFLOP per launch; {gemm_s * 1e6:.2f} us avg launch"},
    }
    if not args.no_rows:
        out["rows"] = measure_rows(torch, qlin, synthetic, stream, pk, fp4_peak, fp8_peak)
    del xs, As, ys, yqs, Wq
    torch.cuda.empty_cache()
    if dist.rank == 0 and not args.no_cpu:
        out["cpu_baseline"] = cpu_baseline(budget_s=15.0)
    return out


def committed_traffic():
    """Per-launch DRAM bytes of the GEMM from the committed ncu summary, if it
    was taken on the current kernel source; else None."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    rec = json.load(open(path))
    h = hashlib.sha256()
    for f in rec.get("sources", []):
        h.update(open(os.path.join(ROOT, f), "rb").read())
    if h.hexdigest() != rec.get("sha256"):
        return None
    return rec.get("dram_bytes_per_launch")


def measure_rows(torch, qlin, synthetic, stream, pk, fp4_peak, fp8_peak):
    """Secondary rows, each in a CUDA graph, cold L2 by rotating buffers."""
    hbm = pk["hbm_gbs"]
    rows = {}

    def g_time(fn, reps_in_graph, replays=20):
        fn()
        torch.cuda.synchronize()
        g = graph_of(lambda: [fn() for _ in range(reps_in_graph)], torch, stream)
        g.replay()
        return timed(g.replay, replays, torch, stream) / reps_in_graph

    # quantizers on the 4608 x 3072 activations: 8 rotating inputs (226 MB)
    x_bits = synthetic.act_entry_outliers(2, M, K)
    R = 8
    xs = [to_dev(x_bits, torch) for _ in range(R)]
    qs = [qlin.alloc_nvfp4(M, K) for _ in range(R)]
    f8 = [qlin.alloc_fp8(M, K, False) for _ in range(R)]
    wsp = [qlin.alloc_workspace() for _ in range(R)]
    sc = torch.tensor([np.float32(0.01)], device="cuda")
    c = [0]

    def nxt():
        c[0] = (c[0] + 1) % R
        return c[0]
    elems = M * K
    t = g_time(lambda: (lambda r: qlin.qlin_quantize_act_nvfp4(xs[r], sc, qs[r]))(nxt()), R)
    rows["a2_quant_nvfp4_static"] = {"us": round(t * 1e6, 2), "GB/s": round(2.5625 * elems / t / 1e9, 1),
                                     "frac_hbm": round(2.5625 * elems / t / 1e9 / hbm, 3),
                                     "bytes_per_elem": 2.5625}
    t = g_time(lambda: (lambda r: qlin.qlin_quantize_act_nvfp4(xs[r], None, qs[r], wsp[r]))(nxt()), R)
    rows["a1a2_quant_nvfp4_dynamic"] = {"us": round(t * 1e6, 2), "GB/s": round(4.5625 * elems / t / 1e9, 1),
                                        "frac_hbm": round(4.5625 * elems / t / 1e9 / hbm, 3),
                                        "bytes_per_elem": 4.5625}
    t = g_time(lambda: (lambda r: qlin.qlin_quantize_act_fp8(xs[r], sc, f8[r]))(nxt()), R)
    rows["a3_quant_fp8_static"] = {"us": round(t * 1e6, 2), "GB/s": round(3 * elems / t / 1e9, 1),
                                   "frac_hbm": round(3 * elems / t / 1e9 / hbm, 3), "bytes_per_elem": 3}
    t = g_time(lambda: (lambda r: qlin.qlin_quantize_act_fp8(xs[r], None, f8[r], wsp[r]))(nxt()), R)
    rows["a3_quant_fp8_dynamic"] = {"us": round(t * 1e6, 2), "GB/s": round(5 * elems / t / 1e9, 1),
                                    "bytes_per_elem": 5}
    del xs, qs, f8

    # weight quantization (offline): NVFP4 [12288, 3072], FP8 per channel [3072, 3072]
    (wb,) = synthetic.weights(2, [(N, K)], 0.02)
    wd = [to_dev(wb, torch) for _ in range(2)]
    wq = [qlin.alloc_nvfp4(N, K) for _ in range(2)]
    t = g_time(lambda: (lambda r: qlin.qlin_quantize_weight(wd[r % 2], qlin.QLIN_FMT_NVFP4, wq[r % 2], wsp[r]))(nxt()), 2)
    rows["a4_weight_quant_nvfp4"] = {"us": round(t * 1e6, 2), "GB/s": round(4.5625 * N * K / t / 1e9, 1)}
    del wd, wq

    # FP8 linear 4608 x 3072 x 3072 (per-tensor act scale, per-channel W scale)
    x8, w8 = synthetic.fp8_linear()
    Rg = 4
    A8 = [qlin.qlin_quantize_act_fp8(to_dev(x8, torch)) for _ in range(Rg)]
    W8 = [qlin.qlin_quantize_weight(to_dev(w8, torch), qlin.QLIN_FMT_FP8) for _ in range(Rg)]
    y8 = [torch.empty((M, K), dtype=torch.bfloat16, device="cuda") for _ in range(Rg)]
    t = g_time(lambda: (lambda r: qlin.qlin_gemm_fp8(A8[r % Rg], W8[r % Rg], y8[r % Rg]))(nxt()), Rg * 2)
    fl = 2 * M * K * K
    rows["a6_gemm_fp8"] = {"us": round(t * 1e6, 2), "TFLOP/s": round(fl / t / 1e12, 1),
                           "frac_fp8_peak": round(fl / t / 1e12 / fp8_peak, 3),
                           "peak": round(fp8_peak, 1)}
    del A8, W8, y8

    # NVFP4 GEMM alone (no requant) on the MLP up-projection
    xb, wb2 = synthetic.nvfp4_mlp_up()
    A4 = [qlin.qlin_quantize_act_nvfp4(to_dev(xb, torch)) for _ in range(2)]
    W4 = [qlin.qlin_quantize_weight(to_dev(wb2, torch), qlin.QLIN_FMT_NVFP4) for _ in range(2)]
    y4 = [torch.empty((M, N), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    t = g_time(lambda: (lambda r: qlin.qlin_gemm_nvfp4(A4[r % 2], W4[r % 2], y4[r % 2]))(nxt()), 4)
    rows["a5_gemm_nvfp4"] = {"us": round(t * 1e6, 2), "TFLOP/s": round(STEP_FLOPS / t / 1e12, 1),
                             "frac_fp4_peak": round(STEP_FLOPS / t / 1e12 / fp4_peak, 3)}
    # the same linear with the next layer's input quantized at y's own dynamic
    # scale (epilogue amax + a quantizer pass over y: 113 MB read, 35 MB written)
    yq4 = [qlin.alloc_nvfp4(M, N) for _ in range(2)]
    wsd = [qlin.alloc_workspace() for _ in range(2)]
    t = g_time(lambda: (lambda r: qlin.qlin_linear_dynamic(A4[r % 2], W4[r % 2], y4[r % 2], yq4[r % 2],
                                                           wsd[r % 2]))(nxt()), 4)
    rows["f1_linear_dynamic_nvfp4"] = {"us": round(t * 1e6, 2), "TFLOP/s": round(STEP_FLOPS / t / 1e12, 1),
                                       "note": "GEMM with output-amax epilogue + NVFP4 quantizer over y"}
    del A4, W4, y4, yq4

    # small-M translator linears (batch 1, 512 tokens), both formats, latency
    x1, x2, w1, w2 = synthetic.translator()
    res = {}
    for fmt in ("nvfp4", "fp8"):
        for (xb_, wb_, tag) in ((x1, w1, "512x2560x1024"), (x2, w2, "512x1024x2560")):
            if fmt == "nvfp4":
                A = qlin.qlin_quantize_act_nvfp4(to_dev(xb_, torch))
                W = qlin.qlin_quantize_weight(to_dev(wb_, torch), qlin.QLIN_FMT_NVFP4)
                fn = lambda A=A, W=W: qlin.qlin_gemm_nvfp4(A, W, yy)
            else:
                A = qlin.qlin_quantize_act_fp8(to_dev(xb_, torch))
                W = qlin.qlin_quantize_weight(to_dev(wb_, torch), qlin.QLIN_FMT_FP8)
                fn = lambda A=A, W=W: qlin.qlin_gemm_fp8(A, W, yy)
            yy = torch.empty((A.rows, W.rows), dtype=torch.bfloat16, device="cuda")
            t = g_time(fn, 20)
            fl = 2 * A.rows * W.rows * A.K
            res[f"{fmt}_{tag}"] = {"us": round(t * 1e6, 2), "TFLOP/s": round(fl / t / 1e12, 1)}
    rows["a8_small_m"] = res

    # the 8-block linear stack, B = 1, 2, 4 (one forward = one graph)
    from paper_2609_21849_gb300 import stack
    res = {}
    wlist = list(synthetic.stack_weights(8, 4))
    for B in (1, 2, 4):
        st = stack.build_stack(B, weights=wlist)
        x = to_dev(synthetic.stack_input(B), torch)
        st.calibrate(x)
        st.forward(x)
        torch.cuda.synchronize()
        g = graph_of(lambda: st.forward(x), torch, stream)
        g.replay()
        t = timed(g.replay, 5, torch, stream)
        res[f"B{B}"] = {"M": st.M, "ms": round(t * 1e3, 3), "TFLOP/s": round(st.flops / t / 1e12, 1),
                        "frac_fp4_peak": round(st.flops / t / 1e12 / fp4_peak, 3),
                        "gemm_launches": len(st.layers)}
        del st, x, g
        torch.cuda.empty_cache()
    rows["a9_stack"] = res

    # precision ladder (Table 2's BF16 / FP16 / FP8 / NVFP4 axis) on the same
    # 8-block stack at B = 1, every linear chained from the stack input:
    #  bf16:  unquantized linears (QKV's value columns feed the out-projection
    #         as a strided view);
    #  fp16:  the same with fp16 operands;
    #  fp8:   W8A8, per-channel weight scales, static calibrated activation
    #         scales, each epilogue writing the next layer's FP8 input;
    #  nvfp4: the fused NVFP4 chain (the a9 B = 1 forward).
    x = to_dev(synthetic.stack_input(1), torch)
    M1 = x.shape[0]
    V0 = 2 * synthetic.HIDDEN
    wbf = [(name, to_dev(wb_, torch)) for (_, name, wb_) in wlist]
    ybf = [torch.empty((M1, w.shape[0]), dtype=torch.bfloat16, device="cuda") for _, w in wbf]

    def fwd_bf16():
        a = x
        for (name, w), y in zip(wbf, ybf):
            qlin.qlin_gemm_bf16(a, w, y)
            a = y[:, V0:] if name == "qkv" else y
    # fp16: the same chain with fp16 operands (converted once, outside the
    # timed region).  Without the blocks' norms the activations grow about
    # 3x per block, so the fp16 chain starts from x * 2^-6 (an exact
    # rescale; its last output would otherwise overflow fp16).
    x16 = (x.float() * 2.0 ** -6).half()   # exact rescale: keeps the chain inside fp16's range
    w16 = [(name, w.half()) for name, w in wbf]
    y16 = [torch.empty_like(y, dtype=torch.float16) for y in ybf]

    def fwd_fp16():
        a = x16
        for (name, w), y in zip(w16, y16):
            qlin.qlin_gemm_fp16(a, w, y)
            a = y[:, V0:] if name == "qkv" else y
    w8 = [(name, qlin.qlin_quantize_weight(w, qlin.QLIN_FMT_FP8)) for name, w in wbf]
    win = [(V0, w.shape[0] - V0) if name == "qkv" else (0, w.shape[0]) for name, w in wbf]
    a8 = [qlin.qlin_quantize_act_fp8(x)] + [qlin.alloc_fp8(M1, n, False) for (_, n) in win]
    nxt8 = [torch.ones(1, dtype=torch.float32, device="cuda") for _ in w8]
    for i, ((name, W), (c0, n)) in enumerate(zip(w8, win)):   # calibration
        qlin.qlin_gemm_fp8(a8[i], W, ybf[i])
        qlin.qlin_quantize_act_fp8(ybf[i][:, c0:c0 + n].contiguous(), None, a8[i + 1])
        nxt8[i].copy_(a8[i + 1].scale)

    def fwd_fp8():
        qlin.qlin_quantize_act_fp8(x, None, a8[0], wsp[0])
        for i, ((name, W), (c0, n)) in enumerate(zip(w8, win)):
            qlin.qlin_linear_fused_fp8(a8[i], W, ybf[i], nxt8[i], a8[i + 1], c0)
    st = stack.build_stack(1, weights=wlist)
    st.calibrate(x)

    def fwd_nvfp4():
        st.forward(x)
    # The 16-bit chains run at the power cap (the SM clock drops under
    # sustained load), so the precisions are timed in interleaved rounds of
    # about 0.6 s each, with the SM clock sampled during each; "ms_x_ghz"
    # (time x median clock) compares them per clock cycle.
    ladder, graphs = {}, {}
    for tag, fn in (("bf16", fwd_bf16), ("fp16", fwd_fp16), ("fp8", fwd_fp8), ("nvfp4", fwd_nvfp4)):
        fn()
        torch.cuda.synchronize()
        graphs[tag] = graph_of(fn, torch, stream)
        graphs[tag].replay()
    runs = {tag: [] for tag in graphs}
    for _ in range(3):
        for tag, g in graphs.items():
            reps = max(3, int(0.6 / max(timed(g.replay, 1, torch, stream), 1e-4)))
            clk = Clocks(int(os.environ.get("LOCAL_RANK", 0)))
            t = timed(g.replay, reps, torch, stream)
            runs[tag].append((t, clk.stop()))
    for tag, rs in runs.items():
        t = statistics.median(r[0] for r in rs)
        mhz = [r[1]["sm_mhz"] for r in rs if r[1].get("sm_mhz")]
        reasons = sorted({x for r in rs for x in r[1].get("reasons", [])})
        ladder[tag] = {"ms": round(t * 1e3, 3), "TFLOP/s": round(st.flops / t / 1e12, 1),
                       "sm_mhz": statistics.median(mhz) if mhz else None, "reasons": reasons}
        if mhz:
            ladder[tag]["ms_x_ghz"] = round(t * 1e3 * statistics.median(mhz) / 1e3, 3)
    del graphs
    for tag in ("fp16", "fp8", "nvfp4"):
        ladder[tag]["speedup_vs_bf16"] = round(ladder["bf16"]["ms"] / ladder[tag]["ms"], 2)
    rows["f2_precision_ladder_stack_B1"] = ladder
    del wbf, ybf, w8, a8, st, x16, w16, y16
    torch.cuda.empty_cache()

    # weight streaming (Sec. 4, "Weight streaming") on the NVFP4 stack: a
    # resident fraction of the layers, the rest copied from pinned host memory
    # through two device slots.  M is the measured pinned host -> device rate;
    # L the resident forward's time per linear; W a streamed layer's bytes.
    # Two device slots (the paper's floor) unless "_slotsN" says otherwise.
    # "model_ms" is the event-level timing of the slot schedule with
    # per-layer L split by FLOPs; "delta_ms" the paper's (N - K) * W / M with
    # N - K the layers that model finds waiting on their copy.
    from paper_2609_21849_gb300 import streaming
    big = max(wlist, key=lambda t: t[2].size)[2].shape
    hb = torch.empty(big[0] * big[1] // 2 + qlin.qlin_nvfp4_scale_bytes(*big), dtype=torch.uint8).pin_memory()
    db = torch.empty_like(hb, device="cuda")
    db.copy_(hb, non_blocking=True)
    t_cp = timed(lambda: db.copy_(hb, non_blocking=True), 20, torch, torch.cuda.current_stream())
    M_rate = hb.numel() / t_cp
    del hb, db
    stream_rows = {"M_GB/s": round(M_rate / 1e9, 1)}
    for B in (1, 4):
        st = stack.build_stack(B, weights=wlist)
        x = to_dev(synthetic.stack_input(B), torch)
        st.calibrate(x)
        st.forward(x)
        torch.cuda.synchronize()
        g = graph_of(lambda: st.forward(x), torch, stream)
        g.replay()
        t_res = statistics.median(timed(g.replay, 3, torch, stream) for _ in range(3))
        del g
        n = len(st.layers)
        wbytes = [l.W.codes.numel() + l.W.scales.numel() for l in st.layers]
        fl = [2 * st.M * l.N * l.K for l in st.layers]
        L_i = [t_res * f / st.flops for f in fl]
        C_i = [w / M_rate for w in wbytes]
        W_mean = sum(wbytes) / n
        res = {"resident_ms": round(t_res * 1e3, 3),
               "lambda": round(streaming.reservoir_lambda(t_res / n, M_rate, W_mean), 3)}
        for frac, slots in ((0.75, 2), (0.5, 2), (0.25, 2), (0.0, 2), (0.25, 3), (0.0, 3)):
            ss = streaming.StreamedStack(st, frac, release=False, n_slots=slots)
            ss.forward(x, stream)
            torch.cuda.synchronize()
            g = graph_of(lambda: ss.forward(x, stream), torch, stream)
            g.replay()
            t = statistics.median(timed(g.replay, 3, torch, stream) for _ in range(3))
            model_t, awaited = streaming.simulate(ss.resident, L_i, C_i, slots)
            dev_w = sum(w for w, r in zip(wbytes, ss.resident) if r) + ss.slot_bytes
            res[f"ws{int(frac * 100)}" + ("" if slots == 2 else f"_slots{slots}")] = {
                "ms": round(t * 1e3, 3), "overhead_pct": round((t / t_res - 1) * 100, 1),
                "model_ms": round(model_t * 1e3, 3), "awaited_layers": awaited,
                "delta_ms": round(streaming.predicted_overhead(n, n - awaited, W_mean, M_rate) * 1e3, 3),
                "device_weight_MB": round(dev_w / 1e6, 1)}
            del g, ss
        res["all_resident_weight_MB"] = round(sum(wbytes) / 1e6, 1)
        assert qlin.qlin_sync_status() == 0
        stream_rows[f"B{B}"] = res
        del st, x
        torch.cuda.empty_cache()
    rows["f3_weight_streaming_stack"] = stream_rows
    return rows


# ------------------------------------------------------------ CPU oracle ---

def cpu_sample_step(aq_full_scale, x_bits, wq, rows, s_next, cols=None):
    """The oracle's restatement of one step on a sample: quantize the sampled
    activation rows (with the full tensor's dynamic scale), exact fp64 GEMM
    against the weight rows of the output columns `cols` (a slice; all by
    default), bf16 rounding, re-quantization."""
    import oracle
    a = oracle.quant_nvfp4(np.ascontiguousarray(x_bits[rows]), aq_full_scale)
    if cols is not None:
        wq = (np.ascontiguousarray(wq[0][cols]), np.ascontiguousarray(wq[1][cols]), wq[2])
    y, _, _ = oracle.gemm_nvfp4(a, wq)
    y16 = oracle.round_bf16_array(y)
    oracle.quant_nvfp4(y16, s_next)


def cpu_setup():
    import oracle
    from paper_2609_21849_gb300 import synthetic
    oracle.build()
    x_bits, w_bits = synthetic.nvfp4_mlp_up()
    wq = oracle.quant_nvfp4(w_bits)                      # offline, not timed
    s_dec = oracle.nvfp4_tensor_scale(oracle.amax_bf16(x_bits))
    return oracle, x_bits, wq, s_dec


def cpu_baseline(budget_s: float = 15.0):
    """The oracle timed on the host cores on a row sample of the step, sized to
    roughly budget_s seconds (the full 4608-row step when that fits)."""
    oracle, x_bits, wq, s_dec = cpu_setup()
    rng = np.random.default_rng(0)
    probe = 64
    t0 = time.perf_counter()
    cpu_sample_step(s_dec, x_bits, wq, np.sort(rng.choice(M, probe, replace=False)), 0.01)
    per_row = (time.perf_counter() - t0) / probe
    n = int(max(probe, min(M, budget_s / max(per_row, 1e-6))))
    rows = np.sort(rng.choice(M, n, replace=False))
    t0 = time.perf_counter()
    cpu_sample_step(s_dec, x_bits, wq, rows, 0.01)
    dt = time.perf_counter() - t0
    return {"value": round(2 * n * N * K / dt / 1e12, 6), "unit": "TFLOP/s",
            "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{n} of {M} token rows of the step (quantize rows, fp64 GEMM vs all 12288 "
                      f"weight rows, bf16 round, re-quantize); {dt:.1f} s"}


def run_reference(args, dist: Dist, budget_s: float = 60.0):
    """The reference arm: the CPU oracle as it stands, on this host's cores
    (rank 0 only), each step a bounded sample of the same workload sized so
    that warm-up and steps together take about budget_s: up to 16 token rows
    against all output columns, or one row against a window of columns when
    the step count leaves less than a row per step."""
    if dist.rank != 0:
        return None
    oracle, x_bits, wq, s_dec = cpu_setup()
    rng = np.random.default_rng(1)
    # step cost = fixed + per_out * outputs, from two probes (the step's
    # whole pipeline: quantize, GEMM, bf16, re-quantize)
    def probe(n_rows, n_cols):
        t = time.perf_counter()
        cpu_sample_step(s_dec, x_bits, wq, np.arange(n_rows), 0.01, slice(0, n_cols))
        return time.perf_counter() - t
    probe(1, 64)
    small, large = probe(1, 64), probe(2, 2048)
    per_out = max((large - small) / (2 * 2048 - 64), 1e-9)
    fixed = max(small - 64 * per_out, 0.0)
    per_step = budget_s / max(args.steps + args.warmup, 1)
    outs = max(per_step - fixed, 0.0) / per_out
    rows_per_step = int(min(16, max(1, outs // N)))
    cols = int(min(N, max(64, outs // rows_per_step // 64 * 64)))

    def sample():
        r = np.sort(rng.choice(M, rows_per_step, replace=False))
        c0 = int(rng.integers(0, (N - cols) // 64 + 1)) * 64
        return r, slice(c0, c0 + cols)

    for _ in range(args.warmup):
        r, c = sample()
        cpu_sample_step(s_dec, x_bits, wq, r, 0.01, c)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        r, c = sample()
        cpu_sample_step(s_dec, x_bits, wq, r, 0.01, c)
    dt = time.perf_counter() - t0
    v = 2 * rows_per_step * cols * K * args.steps / dt / 1e12
    return {"impl": "reference", "metric": "NVFP4 quantized-linear throughput (TFLOP/s, 2*M*N*K per step)",
            "value": round(v, 6), "unit": "TFLOP/s", "n_gpus": 0, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(dt / args.steps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64 (oracle)",
            "data": "synthetic (seeded)", "config": {"workload": WORKLOAD, "M": M, "N": N, "K": K,
                                                     "sample_rows_per_step": rows_per_step,
                                                     "sample_cols_per_step": cols},
            "cpu_baseline": {"value": round(v, 6), "unit": "TFLOP/s", "cores": oracle.num_threads(),
                             "kind": "oracle",
                             "sample": f"{rows_per_step} of {M} token rows x {cols} of {N} output "
                                       f"columns per step"},
            "e2e": {"value": round(v, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    args = parse()
    if args.impl == "reference":
        # CPU only: no process group needed; non-zero ranks exit without work
        rank = int(os.environ.get("RANK", "0"))
        if rank != 0:
            return 0
        out = run_reference(args, _Rank0())
        print(json.dumps(out))
        return 0
    dist = Dist()
    try:
        out = run_ours(args, dist)
        if dist.rank == 0:
            print(json.dumps(out))
    finally:
        dist.close()
    return 0


class _Rank0:
    rank = 0
    world = 1


if __name__ == "__main__":
    sys.exit(main())
