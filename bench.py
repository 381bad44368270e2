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
    ap.add_argument("--no-rows", action="store_true",
                    help="time the step only: skip the quantizer, GEMM, translator and secondary rows")
    ap.add_argument("--sustained-s", type=float, default=1.0,
                    help="seconds of step replay after the timed region for the clock samples (0: none)")
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

    # Steps run as CUDA graphs: a graph of S steps replayed back to back, and
    # a graph of the remaining n % S steps, so that exactly --warmup and
    # --steps steps run.  Timing events (external event nodes) bracket one
    # GEMM in EV_EVERY: an event node between two kernels breaks their
    # programmatic launch overlap (measured: events around every GEMM
    # stretched the step from 87 to 100 us), so the GEMM's duration is
    # sampled rather than bracketed everywhere.
    S = 4 * R
    graphs = {}

    def graph_for(n):
        if n not in graphs:
            try:
                evs = [(torch.cuda.Event(enable_timing=True, external=True),
                        torch.cuda.Event(enable_timing=True, external=True))
                       for _ in range((n + EV_EVERY - 1) // EV_EVERY)]
            except TypeError:
                evs = []

            def steps_n():
                for i in range(n):
                    r = i % R
                    timed_gemm = bool(evs) and i % EV_EVERY == 0
                    qlin.qlin_quantize_act_nvfp4(xs[r], None, As[r], wss[r])
                    if timed_gemm:
                        evs[i // EV_EVERY][0].record(stream)
                    qlin.qlin_linear_fused(As[r], Wq[r], ys[r], next_scale, yqs[r])
                    if timed_gemm:
                        evs[i // EV_EVERY][1].record(stream)
            graphs[n] = (graph_of(steps_n, torch, stream), evs)
        return graphs[n]

    def run_steps(n):
        """Replay exactly n steps; returns the graphs whose events were recorded."""
        used = []
        if n >= S:
            g, evs = graph_for(S)
            for _ in range(n // S):
                g.replay()
            used.append(evs)
        if n % S:
            g, evs = graph_for(n % S)
            g.replay()
            used.append(evs)
        return used

    for r in range(R):          # first launches outside capture (attributes)
        step(r)
    torch.cuda.synchronize()
    graph_for(S)
    if args.steps % S:
        graph_for(args.steps % S)
    if args.warmup % S:
        graph_for(args.warmup % S)
    steps, warm = args.steps, args.warmup
    run_steps(warm)
    torch.cuda.synchronize()

    # Clock samples: nvidia-smi polls every 200 ms, from just before the timed
    # region through a sustained window of the same graph replayed for about
    # a second right after it (a timed region of a few steps is shorter than
    # the sampling period).
    dist.barrier()
    torch.cuda.synchronize()
    clocks = Clocks(dist.local_rank)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    used = run_steps(steps)
    t1.record(stream)
    t1.synchronize()
    torch.cuda.synchronize()
    dist.barrier()
    sec = dist.max(t0.elapsed_time(t1) / 1e3)
    per_step = sec / steps
    value = STEP_FLOPS * steps * dist.world / sec / 1e12
    gemm_samples = [a.elapsed_time(b) / 1e3 for evs in used for a, b in evs]
    if gemm_samples:
        gemm_s = statistics.mean(gemm_samples)
    else:
        gemm_s = timed(lambda: qlin.qlin_linear_fused(As[0], Wq[0], ys[0], next_scale, yqs[0]),
                       200, torch, stream)
    gemm_tflops = STEP_FLOPS / gemm_s / 1e12
    sus_steps = (S * max(1, int(args.sustained_s / max(per_step, 1e-6)) // S)
                 if args.sustained_s > 0 else 0)
    s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0.record(stream)
    sus_used = run_steps(sus_steps)
    s1.record(stream)
    s1.synchronize()
    clk = clocks.stop()
    clk["window"] = (f"timed region ({sec * 1e3:.2f} ms) plus a sustained replay of the same "
                     f"step graph right after it ({sus_steps} steps)")
    sus_sec = s0.elapsed_time(s1) / 1e3
    sus_gemm = [a.elapsed_time(b) / 1e3 for evs in sus_used for a, b in evs]
    sustained = {"steps": sus_steps,
                 "ms_per_step": round(sus_sec / sus_steps * 1e3, 5) if sus_steps else None,
                 "value": round(STEP_FLOPS * sus_steps / sus_sec / 1e12, 2) if sus_steps else None,
                 "gemm_us": round(statistics.mean(sus_gemm) * 1e6, 2) if sus_gemm else None}

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
                     "streams, consecutive steps overlapped; y (bf16) is read back every step, "
                     "the re-quantized y_q stays on the device as the next layer's input"}

    # ---- measured tensor-core ceilings (MMA-only probe, every SM at once)
    from paper_2609_21849_gb300 import probe
    ceil = probe.ceilings(sm_max_mhz=float(clk.get("sm_max_mhz") or 2070.0))
    sms = ceil["nvfp4_pair_256x256x64"]["sms"]
    mhz = float(clk.get("sm_mhz") or clk.get("sm_max_mhz") or 2070.0)
    fp4_ceil = ceil["nvfp4_pair_256x256x64"]["flop_per_cycle_per_sm"] * sms * mhz * 1e6 / 1e12
    fp8_ceil = ceil["fp8_pair_256x256x32"]["flop_per_cycle_per_sm"] * sms * mhz * 1e6 / 1e12

    traffic = committed_traffic()
    out = {
        "metric": "NVFP4 quantized-linear throughput (TFLOP/s, 2*M*N*K per step)",
        "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": dist.world, "steps": steps,
        "warmup": warm, "ms_per_step": round(per_step * 1e3, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "nvfp4 (e2m1 x e4m3 block scales), fp32 accumulate, bf16 out",
        "data": "synthetic (seeded; shapes of FLUX.2-klein at 1024^2, random weights)",
        "config": {"workload": WORKLOAD, "M": M, "N": N, "K": K,
                   "step": "dynamic NVFP4 act quant (one read of x: grid-wide amax + quant) + NVFP4 GEMM + bf16 out + fused NVFP4 requant",
                   "l2": f"{R} rotating input/output sets of {set_bytes / 2**20:.0f} MiB each (> 129 MiB L2)",
                   "graph": f"CUDA graphs of {S} steps (replayed {steps // S}x) and of the "
                            f"remaining {steps % S} steps",
                   "gemm_timing": f"CUDA events around 1 GEMM in {EV_EVERY} inside the timed graphs "
                                  f"({len(gemm_samples)} samples)",
                   "parallelism": f"replicas x{dist.world}"},
        "gpu_launches": 2 * steps,
        "clocks": clk,
        "sustained": sustained,
        "e2e": e2e,
        "roofline": {"kernel": "gemm_kernel<nvfp4, BN=256, requant>", "bound": "tensor",
                     "achieved": round(gemm_tflops, 1),
                     "peak": round(fp4_peak, 1), "unit": "TFLOP/s",
                     "peak_source": f"{pk['source']} bf16 burst {pk['bf16']} TFLOP/s x nominal FP4:BF16 {FP4_PER_BF16:g}",
                     "frac": round(gemm_tflops / fp4_peak, 4),
                     "mma_ceiling": round(fp4_ceil, 1),
                     "frac_of_mma_ceiling": round(gemm_tflops / fp4_ceil, 4),
                     "mma_ceiling_source": f"measured kind::mxf4nvf4 CTA-pair MMA rate "
                                           f"({ceil['nvfp4_pair_256x256x64']['flop_per_cycle_per_sm']:.0f} "
                                           f"FLOP/cycle/SM) x {sms} SMs x {mhz:.0f} MHz (median sampled SM clock)",
                     "traffic": traffic,
                     "algorithmic": f"{STEP_FLOPS / 1e9:.2f} GFLOP per launch; {gemm_s * 1e6:.2f} us avg launch"},
        "mma_probe": ceil,
    }
    if not args.no_rows:
        out.update(measure_headline_rows(torch, qlin, synthetic, stream, pk, fp4_peak, fp8_peak,
                                         fp4_ceil, fp8_ceil))
        out["rows"] = measure_rows(torch, qlin, synthetic, stream, pk, fp4_peak, fp8_peak)
    del xs, As, ys, yqs, Wq
    torch.cuda.empty_cache()
    if dist.rank == 0 and not args.no_cpu:
        out["cpu_baseline"] = cpu_baseline(budget_s=15.0)
        out["cpu_baseline_configs"] = cpu_baseline_configs()
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


def g_time(torch, stream, fn, reps_in_graph, replays=20):
    """Device time per call of fn, captured reps_in_graph times in one CUDA
    graph and replayed (events on the launching stream)."""
    fn()
    torch.cuda.synchronize()
    g = graph_of(lambda: [fn() for _ in range(reps_in_graph)], torch, stream)
    g.replay()
    return timed(g.replay, replays, torch, stream) / reps_in_graph


def measure_headline_rows(torch, qlin, synthetic, stream, pk, fp4_peak, fp8_peak, fp4_ceil,
                          fp8_ceil):
    """The quantizer and GEMM rows the metric names (top-level keys of the
    line): each in a CUDA graph, cold L2 by rotating buffers larger than L2."""
    hbm = pk["hbm_gbs"]
    out = {}
    sc = torch.tensor([np.float32(0.01)], device="cuda")
    c = [0]

    def nxt(R):
        c[0] = (c[0] + 1) % R
        return c[0]

    # ---- NVFP4 / FP8 activation quantizers: x [4608, 3072] (config 3's
    # activations) and [18432, 3072] (the stack input at B = 4, 113 MB: the
    # steady-state bandwidth check)
    quant = {"kernel": "quant_nvfp4_kernel<static> (and onepass / two-pass dynamic routes)",
             "peak_GB/s": hbm, "peak_source": f"{pk['source']} HBM copy bandwidth"}
    for (Mq, tag) in ((M, "4608x3072"), (4 * M, "18432x3072")):
        x_bits = synthetic.act_entry_outliers(2, Mq, K)
        R = max(2, -(-2 * L2_BYTES // (Mq * K * 2)))        # rotation > 2x L2
        xs = [to_dev(x_bits, torch) for _ in range(R)]
        qs = [qlin.alloc_nvfp4(Mq, K) for _ in range(R)]
        f8 = [qlin.alloc_fp8(Mq, K, False) for _ in range(R)]
        wsp = [qlin.alloc_workspace() for _ in range(R)]
        elems = Mq * K
        row = {"rotating_inputs": R}
        t = g_time(torch, stream, lambda: (lambda r: qlin.qlin_quantize_act_nvfp4(xs[r], sc, qs[r]))(nxt(R)), R)
        row["nvfp4_static"] = {"us": round(t * 1e6, 2), "GB/s": round(2.5625 * elems / t / 1e9, 1),
                               "frac_hbm": round(2.5625 * elems / t / 1e9 / hbm, 3),
                               "bytes_per_elem": 2.5625}
        t = g_time(torch, stream, lambda: (lambda r: qlin.qlin_quantize_act_nvfp4(xs[r], None, qs[r], wsp[r]))(nxt(R)), R)
        row["nvfp4_dynamic"] = {
            "us": round(t * 1e6, 2),
            "route": "one read of x (x held on chip)" if Mq * K * 2 <= 152 * 224 * 1024 else "amax pass + quantizer",
            "GB/s_moved": round((2.5625 if Mq * K * 2 <= 152 * 224 * 1024 else 4.5625) * elems / t / 1e9, 1),
            "GB/s_at_4.5625": round(4.5625 * elems / t / 1e9, 1),
            "frac_hbm_moved": round((2.5625 if Mq * K * 2 <= 152 * 224 * 1024 else 4.5625) * elems / t / 1e9 / hbm, 3)}
        t = g_time(torch, stream, lambda: (lambda r: qlin.qlin_quantize_act_fp8(xs[r], sc, f8[r]))(nxt(R)), R)
        row["fp8_static"] = {"us": round(t * 1e6, 2), "GB/s": round(3 * elems / t / 1e9, 1),
                             "frac_hbm": round(3 * elems / t / 1e9 / hbm, 3), "bytes_per_elem": 3}
        quant[tag] = row
        del xs, qs, f8, wsp
        torch.cuda.empty_cache()
    out["quantizer"] = quant
    out["quant_nvfp4_static_GBps"] = quant["4608x3072"]["nvfp4_static"]["GB/s"]
    out["quant_nvfp4_static_frac_hbm"] = quant["4608x3072"]["nvfp4_static"]["frac_hbm"]
    out["quant_nvfp4_static_frac_hbm_18432x3072"] = quant["18432x3072"]["nvfp4_static"]["frac_hbm"]

    # ---- FP8 linear 4608 x 3072 x 3072 (per-tensor act scale, per-channel W scale)
    x8, w8 = synthetic.fp8_linear()
    Rg = 4
    A8 = [qlin.qlin_quantize_act_fp8(to_dev(x8, torch)) for _ in range(Rg)]
    W8 = [qlin.qlin_quantize_weight(to_dev(w8, torch), qlin.QLIN_FMT_FP8) for _ in range(Rg)]
    y8 = [torch.empty((M, K), dtype=torch.bfloat16, device="cuda") for _ in range(Rg)]
    t = g_time(torch, stream, lambda: (lambda r: qlin.qlin_gemm_fp8(A8[r % Rg], W8[r % Rg], y8[r % Rg]))(nxt(Rg)), Rg * 2)
    fl = 2 * M * K * K
    out["fp8_gemm"] = {"workload": "4608x3072x3072", "us": round(t * 1e6, 2),
                       "TFLOP/s": round(fl / t / 1e12, 1),
                       "frac": round(fl / t / 1e12 / fp8_peak, 3), "peak": round(fp8_peak, 1),
                       "peak_source": f"{pk['source']} bf16 burst x nominal FP8:BF16 {FP8_PER_BF16:g}",
                       "frac_of_mma_ceiling": round(fl / t / 1e12 / fp8_ceil, 3),
                       "mma_ceiling": round(fp8_ceil, 1)}
    del A8, W8, y8

    # ---- NVFP4 GEMM alone (no re-quantization) on the MLP up-projection
    xb, wb2 = synthetic.nvfp4_mlp_up()
    A4 = [qlin.qlin_quantize_act_nvfp4(to_dev(xb, torch)) for _ in range(2)]
    W4 = [qlin.qlin_quantize_weight(to_dev(wb2, torch), qlin.QLIN_FMT_NVFP4) for _ in range(2)]
    y4 = [torch.empty((M, N), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    t = g_time(torch, stream, lambda: (lambda r: qlin.qlin_gemm_nvfp4(A4[r % 2], W4[r % 2], y4[r % 2]))(nxt(2)), 4)
    out["nvfp4_gemm"] = {"workload": "4608x12288x3072, bf16 out, no re-quantization",
                         "us": round(t * 1e6, 2), "TFLOP/s": round(STEP_FLOPS / t / 1e12, 1),
                         "frac": round(STEP_FLOPS / t / 1e12 / fp4_peak, 3),
                         "frac_of_mma_ceiling": round(STEP_FLOPS / t / 1e12 / fp4_ceil, 3)}
    # the same linear with the next layer's input quantized at y's own dynamic
    # scale (epilogue amax + a quantizer pass over y: 113 MB read, 35 MB written)
    yq4 = [qlin.alloc_nvfp4(M, N) for _ in range(2)]
    wsd = [qlin.alloc_workspace() for _ in range(2)]
    t = g_time(torch, stream, lambda: (lambda r: qlin.qlin_linear_dynamic(A4[r % 2], W4[r % 2], y4[r % 2], yq4[r % 2],
                                                                          wsd[r % 2]))(nxt(2)), 4)
    out["f1_linear_dynamic_nvfp4"] = {"us": round(t * 1e6, 2), "TFLOP/s": round(STEP_FLOPS / t / 1e12, 1),
                                      "vs_plain_gemm": round(t * 1e6 / out["nvfp4_gemm"]["us"], 3),
                                      "note": "GEMM with output-amax epilogue + NVFP4 quantizer over y"}
    del A4, W4, y4, yq4

    # ---- small-M translator linears (batch 1, 512 tokens), both formats,
    # against max(compute bound, bytes bound)
    x1, x2, w1, w2 = synthetic.translator()
    res = {}
    for fmt in ("nvfp4", "fp8"):
        for (xb_, wb_, tag) in ((x1, w1, "512x2560x1024"), (x2, w2, "512x1024x2560")):
            if fmt == "nvfp4":
                A = qlin.qlin_quantize_act_nvfp4(to_dev(xb_, torch))
                W = qlin.qlin_quantize_weight(to_dev(wb_, torch), qlin.QLIN_FMT_NVFP4)
                fn = lambda A=A, W=W: qlin.qlin_gemm_nvfp4(A, W, yy)
                nbytes = (A.codes.numel() + A.scales.numel() + W.codes.numel() + W.scales.numel())
                peak = fp4_peak
            else:
                A = qlin.qlin_quantize_act_fp8(to_dev(xb_, torch))
                W = qlin.qlin_quantize_weight(to_dev(wb_, torch), qlin.QLIN_FMT_FP8)
                fn = lambda A=A, W=W: qlin.qlin_gemm_fp8(A, W, yy)
                nbytes = A.codes.numel() + W.codes.numel() + 4 * W.rows
                peak = fp8_peak
            yy = torch.empty((A.rows, W.rows), dtype=torch.bfloat16, device="cuda")
            nbytes += yy.numel() * 2
            t = g_time(torch, stream, fn, 20)
            fl = 2 * A.rows * W.rows * A.K
            bound = max(fl / (peak * 1e12), nbytes / (hbm * 1e9))
            res[f"{fmt}_{tag}"] = {"us": round(t * 1e6, 2), "TFLOP/s": round(fl / t / 1e12, 1),
                                   "bound_us": round(bound * 1e6, 3),
                                   "frac_of_bound": round(bound / t, 3),
                                   "bound": "bytes" if nbytes / (hbm * 1e9) > fl / (peak * 1e12) else "compute"}
    out["a8_small_m"] = res

    # ---- the translator MLP forward (Sec. 3's d3072 translator: 512 tokens,
    # 1024 -> 3072 -> 2560; dynamic input quantization, the first linear's
    # epilogue re-quantizing the hidden activations), one CUDA graph per
    # format, against the sum of its three kernels' max(compute, bytes) bounds
    from paper_2609_21849_gb300 import translator
    xt, w1t, w2t = synthetic.translator_mlp()
    xtd = to_dev(xt, torch)
    Mt, Kt = xt.shape
    Ht, Ot = w1t.shape[0], w2t.shape[0]
    tr = {}
    for fmt in ("nvfp4", "fp8"):
        t = translator.build_translator(fmt, w1t, w2t, Mt)
        t.calibrate(xtd)
        tm = g_time(torch, stream, lambda t=t: t.forward(xtd, stream), 20)
        qb = 0.5625 if fmt == "nvfp4" else 1.0          # bytes per quantized element
        peak = fp4_peak if fmt == "nvfp4" else fp8_peak
        f1, f2 = 2 * Mt * Ht * Kt, 2 * Mt * Ot * Ht
        b0 = Mt * Kt * (2 + qb)                          # quantizer: read x, write x_q
        b1 = (Mt * Kt + Ht * Kt + Mt * Ht) * qb          # x_q, W1 in; h_q out
        b2 = (Mt * Ht + Ot * Ht) * qb + Mt * Ot * 2      # h_q, W2 in; bf16 y out
        bound = (b0 / (hbm * 1e9) + max(f1 / (peak * 1e12), b1 / (hbm * 1e9))
                 + max(f2 / (peak * 1e12), b2 / (hbm * 1e9)))
        tr[fmt] = {"us": round(tm * 1e6, 2), "TFLOP/s": round(t.flops / tm / 1e12, 1),
                   "bound_us": round(bound * 1e6, 3), "frac_of_bound": round(bound / tm, 3),
                   "launches": 3, "note": "one forward per graph node group, weights L2-warm"}
        del t
    out["f4_translator_mlp"] = tr
    return out


def measure_rows(torch, qlin, synthetic, stream, pk, fp4_peak, fp8_peak):
    """Secondary rows (stack, precision ladder, weight streaming), each in a
    CUDA graph."""
    rows = {}
    wsp = [qlin.alloc_workspace()]

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


def _time_rows(step, total_rows, flops_per_row, budget_s, probe_rows):
    """Time the oracle's step on a row sample of about budget_s (all rows
    when that fits): the sample grows 2x to 4x per probe until one takes
    half the budget (at least two probes).  A step costs a fixed part (decoding the weights) plus
    a part per row; the last two probes give both, and so the full-size time
    when the sample is not all rows."""
    def run(n):
        t0 = time.perf_counter()
        step(n)
        return time.perf_counter() - t0
    pts = []
    n = min(probe_rows, total_rows)
    while True:
        pts.append((n, run(n)))
        t = pts[-1][1]
        if n >= total_rows or (t >= budget_s / 2 and len(pts) > 1):
            break
        n = min(total_rows, max(2 * n, min(4 * n, int(n * budget_s / max(t, 1e-6)))))
    n, dt = pts[-1]
    if len(pts) > 1 and n > pts[-2][0]:
        per_row = max((dt - pts[-2][1]) / (n - pts[-2][0]), 1e-12)
        fixed = max(dt - n * per_row, 0.0)
    else:
        per_row, fixed = dt / n, 0.0
    full = dt if n >= total_rows else fixed + per_row * total_rows
    return {"value": round(flops_per_row * n / dt / 1e12, 6), "unit": "TFLOP/s",
            "rows": n, "of_rows": total_rows, "seconds": round(dt, 2),
            "fixed_seconds": round(fixed, 3), "full_size_seconds": round(full, 2),
            "extrapolated": n < total_rows}


def cpu_baseline_configs(budget_s: float = 2.0):
    """The oracle as it stands, timed on the host cores, single-threaded and
    on every core, for each workload: the tiny NVFP4 linear, the FP8 linear
    and the translator linears in full where the budget allows, the MLP
    up-projection, and the 8-block stack per layer on sampled token rows
    (extrapolated to all rows, and labelled so).  A step is what the GPU path
    does: activation quantization with the full tensor's scale, the exact
    fp64 GEMM, bf16 rounding (and, where the workload has it, the
    re-quantization of the output); weight quantization is offline."""
    import oracle
    from paper_2609_21849_gb300 import synthetic
    oracle.build()
    rng = np.random.default_rng(7)
    cases = {}

    def nvfp4_linear(x, wq, s_next=None):
        s = oracle.nvfp4_tensor_scale(oracle.amax_bf16(x))

        def step(n):
            rows = np.sort(rng.choice(x.shape[0], n, replace=False))
            a = oracle.quant_nvfp4(np.ascontiguousarray(x[rows]), s)
            y, _, _ = oracle.gemm_nvfp4(a, wq)
            y16 = oracle.round_bf16_array(y)
            if s_next is not None:
                oracle.quant_nvfp4(y16, s_next)
        return step

    x, w = synthetic.tiny_nvfp4()
    cases["tiny_nvfp4_128x256x256"] = (nvfp4_linear(x, oracle.quant_nvfp4(w)), 128, 2 * 256 * 256, 16)
    x8, w8 = synthetic.fp8_linear()
    wq8 = oracle.quant_fp8_rows(w8)
    s8 = oracle.fp8_tensor_scale(oracle.amax_bf16(x8))

    def fp8_step(n):
        rows = np.sort(rng.choice(M, n, replace=False))
        a = oracle.quant_fp8(np.ascontiguousarray(x8[rows]), s8)
        y, _, _ = oracle.gemm_fp8(a, wq8)
        oracle.round_bf16_array(y)
    cases["fp8_linear_4608x3072x3072"] = (fp8_step, M, 2 * K * K, 4)
    xu, wu = synthetic.nvfp4_mlp_up()
    cases["nvfp4_mlp_up_4608x12288x3072_fused"] = (nvfp4_linear(xu, oracle.quant_nvfp4(wu), 0.01),
                                                   M, 2 * N * K, 4)
    x1, x2, w1, w2 = synthetic.translator()
    tq = [(x1, oracle.quant_nvfp4(w1), oracle.quant_fp8_rows(w1)),
          (x2, oracle.quant_nvfp4(w2), oracle.quant_fp8_rows(w2))]

    def translator_step(n):
        for xt, wq4, wqf in tq:
            nvfp4_linear(xt, wq4)(n)
            sf = oracle.fp8_tensor_scale(oracle.amax_bf16(xt))
            rows = np.sort(rng.choice(xt.shape[0], n, replace=False))
            y, _, _ = oracle.gemm_fp8(oracle.quant_fp8(np.ascontiguousarray(xt[rows]), sf), wqf)
            oracle.round_bf16_array(y)
    cases["translator_512x2560x1024_512x1024x2560_nvfp4_fp8"] = (
        translator_step, 512, 2 * 2 * (2560 * 1024 + 1024 * 2560), 4)

    # the stack: one block's 4 layers chained on the sampled rows (layers are
    # row-local once their static scales are fixed; the 8 blocks have the
    # same shapes, so the stack takes 8x a block)
    wl = list(synthetic.stack_weights(1, 4))
    wsq = [(name, oracle.quant_nvfp4(wb)) for (_, name, wb) in wl]
    del wl
    xs5 = synthetic.stack_input(1)
    s5 = oracle.nvfp4_tensor_scale(oracle.amax_bf16(xs5))

    def stack_step(n):
        rows = np.sort(rng.choice(xs5.shape[0], n, replace=False))
        a = oracle.quant_nvfp4(np.ascontiguousarray(xs5[rows]), s5)
        for name, wq in wsq:
            y, _, _ = oracle.gemm_nvfp4(a, wq)
            y16 = oracle.round_bf16_array(y)
            win = np.ascontiguousarray(y16[:, 2 * K:] if name == "qkv" else y16)
            a = oracle.quant_nvfp4(win, oracle.nvfp4_tensor_scale(oracle.amax_bf16(win)))
    per_row5 = 2 * (3 * K * K + K * K + 2 * N * K)

    res = {}
    all_threads = oracle.num_threads()
    for threads in (1, all_threads):
        oracle.set_num_threads(threads)
        tag = "1_thread" if threads == 1 else f"{threads}_threads"
        for name, (fn, total, fpr, probe_n) in cases.items():
            res.setdefault(name, {})[tag] = _time_rows(fn, total, fpr, budget_s, probe_n)
        r5 = _time_rows(stack_step, M, per_row5, budget_s, 1)
        r5["stack_full_size_seconds"] = {f"B{b}": round(8 * b * r5["full_size_seconds"], 1)
                                         for b in (1, 2, 4)}
        r5["note"] = ("one block's 4 layers chained on sampled token rows; the 8-block stack "
                      "at 4608*B rows extrapolated as 8 blocks x B x (fixed + per-row cost)")
        res.setdefault("stack_block", {})[tag] = r5
    oracle.set_num_threads(all_threads)
    return {"kind": "oracle", "cores": all_threads, "configs": res}


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
