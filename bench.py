"""Benchmark of the NVFP4 W4A4KV4 hot path on GB300.

One step = one pass of the path over one batch of synthetic inputs of the
Qwen-32B-shaped prefill layer (M = 8192 tokens, the largest single-GPU
workload): for each linear (qkv, o, gate_up, down) the FP32 tensor scale of
its bf16 activation and NVFP4 quantization of the activation (one launch),
then the block-scaled FP4 GEMM to bf16.  Weights are quantized once, before
timing.  The headline value is the GEMM FLOPs of the step divided by its
device time (TFLOP/s); the roofline entry is the step's dominant kernel, the
gate_up GEMM (8192 x 55296 x 5120), against the dense FP4 tensor peak.

The decode-attention half of the metric is measured in the same run on the
Qwen-14B-shaped decode workload (batch 64, 40/8 heads, 16384-token NVFP4
cache): per step, quantize-and-append one new K/V token per sequence and run
decode attention over the cache; reported as algorithmic HBM GB/s under
"decode_attention".

Timing: CUDA events on the launching stream around each step, L2 flushed
(256 MiB write) between steps, steps replayed from a CUDA graph.  Clocks are
sampled with nvidia-smi while the timed loops run.  `--impl reference` times
the CPU oracle instead, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

GEMM_WL = "qwen32b_prefill_linears_m8192"
ATTN_WL = "qwen14b_decode_attention_b64_t16384"
# Reported beside the headline (same step form, graph-replayed, L2 flushed): the single linear, the
# 1.5B prefill linears, and the decode-batch linears with their K/V append.
OTHER_LINEAR_WLS = ("w4a4_linear_m16_k1536_n1536", "qwen1.5b_prefill_linears_m2048", "qwen14b_decode_linears_m256")
METRIC = "NVFP4 GEMM TFLOP/s & FP4-KV decode-attn HBM GB/s vs GB300 roofline"
FP4_OVER_BF16 = 13.5 / 2.25  # nominal dense FP4 / BF16 tensor ratio of GB300
CSRC = os.path.join(ROOT, "paper_2606_15682_gb300", "csrc")
# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one ncu capture of the
# same kernel and shape (commands in profiles/).  Each entry holds only while the kernel sources
# hash to the value they had at capture time; otherwise the line reports traffic = null.
NCU_TRAFFIC = {
    "gemm": {"bytes": 205745920 + 861377536, "sources": ("gemm.cu", "common.cuh"), "sha": "1dc61211627969f1",
             "shape": (8192, 55296, 5120),
             "profile": "profiles/gemm_qwen32b_prefill_gate_up_m8192_n55296_k5120.md"},
    "attention": {"bytes": 1208722432 + 22210816, "sources": ("attention.cu", "common.cuh"),
                  "sha": "2e035c943bb67759", "shape": (64, 16384),
                  "profile": "profiles/attention_qwen14b_decode_b64_t16384.md (attn_partial_kernel)"},
}


def ncu_traffic(kind, shape):
    e = NCU_TRAFFIC[kind]
    h = hashlib.sha256()
    for f in e["sources"]:
        with open(os.path.join(CSRC, f), "rb") as fh:
            h.update(fh.read())
    if e["bytes"] is None:
        return None
    return e["bytes"] if h.hexdigest()[:16] == e["sha"] and tuple(shape) == e["shape"] else None


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "src": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "src": "fallback"}


# ------------------------------------------------------- replica reduction ---
# N > 1 runs N independent replicas (the path has no exchange step): every rank
# times the same work on its own GPU; the job's time is the slowest rank's and
# its work is the sum over ranks.

def reduce_max_over_ranks(values, world):
    """Element-wise maximum of `values` over the ranks (gloo all_reduce)."""
    import torch
    vals = torch.tensor(values, dtype=torch.float64)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(vals, op=dist.ReduceOp.MAX)
    return vals.tolist()


def whole_job_rate(work_per_rank, world, ms_max):
    """Units per second for the whole job: all ranks' work over the slowest rank's time."""
    return world * work_per_rank / (ms_max * 1e-3)


# ------------------------------------------------------------ clocks ---

class ClockSampler:
    """nvidia-smi clock/throttle sampling in a background process."""

    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.rows = []
        self.proc = None
        self.windows = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-i", str(self.dev), "-lms", "50"], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        def reader():
            for line in self.proc.stdout:
                self.rows.append((time.time(), line.strip()))
        self.t = threading.Thread(target=reader, daemon=True)
        self.t.start()

    def mark(self, t0, t1):
        self.windows.append((t0, t1))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.t.join(timeout=2)

    def summary(self):
        parsed = []
        for ts, line in self.rows:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                parsed.append((ts, float(f[2]), float(f[3]), f[5:9]))
            except ValueError:
                continue
        if not parsed:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        inside = [p for p in parsed if any(a - 0.06 <= p[0] <= b + 0.06 for a, b in self.windows)]
        use = inside or parsed
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for p in use for i, v in enumerate(p[3]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(p[1] for p in use), "sm_max_mhz": max(p[2] for p in use),
                "reasons": reasons, "samples": len(use), "in_timed_region": bool(inside)}


# ---------------------------------------------------------- our arm ---

def run_ours(args, rank, world):
    import numpy as np
    import torch

    from paper_2606_15682_gb300 import build as B
    B.build()
    from paper_2606_15682_gb300 import nvfp4 as N
    from paper_2606_15682_gb300 import synth

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(device=dev)
    peaks = load_peaks()
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    sampler = ClockSampler(dev.index)
    sampler.start()

    # ---------------- GEMM step: prefill linears with on-the-fly activation quantization
    def build_layers(wl):
        """The workload's linears: bf16 activations, weights quantized once (MMA scales)."""
        Mw = synth.WORKLOADS[wl]["M"]
        out_layers, out_flops = [], 0
        for name, (Nn, K) in synth.WORKLOADS[wl]["linears"].items():
            a, W = synth.linear_inputs(wl, name, device=dev)
            gw = torch.empty(1, dtype=torch.float32, device=dev)
            wc = torch.empty(Nn, K // 2, dtype=torch.uint8, device=dev)
            ws = torch.empty(N.nvfp4_scales_bytes(Nn, K, N.SCALES_MMA), dtype=torch.uint8, device=dev)
            N.nvfp4_tensor_scale(W, gw)
            N.nvfp4_quantize(W, gw, wc, ws, N.SCALES_MMA)
            del W
            out_layers.append(dict(name=name, N=Nn, K=K, a=a, wc=wc, ws=ws, gw=gw,
                                   ga=torch.empty(1, dtype=torch.float32, device=dev),
                                   qstate=torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device=dev),
                                   ac=torch.empty(Mw, K // 2, dtype=torch.uint8, device=dev),
                                   asf=torch.empty(N.nvfp4_scales_bytes(Mw, K, N.SCALES_MMA), dtype=torch.uint8,
                                                   device=dev),
                                   out=torch.empty(Mw, Nn, dtype=torch.bfloat16, device=dev),
                                   ev=[torch.cuda.Event(enable_timing=True) for _ in range(2)]))
            out_flops += 2 * Mw * Nn * K
        torch.cuda.synchronize()
        return Mw, out_layers, out_flops

    M, layers, flops = build_layers(GEMM_WL)

    def gemm_step(record_gemm_events, layer_list=None, Mw=None):
        for L in (layers if layer_list is None else layer_list):
            N.nvfp4_quantize_dynamic(L["a"], L["qstate"], L["ga"], L["ac"], L["asf"], N.SCALES_MMA)
            if record_gemm_events:
                L["ev"][0].record()
            N.nvfp4_linear(L["ac"], L["asf"], L["ga"], L["wc"], L["ws"], L["gw"], L["out"], M if Mw is None else Mw,
                           L["N"], L["K"])
            if record_gemm_events:
                L["ev"][1].record()

    with torch.cuda.stream(stream):
        gemm_step(False)
        stream.synchronize()
        graph = torch.cuda.CUDAGraph()
        n0 = N.nvfp4_launch_count()
        with torch.cuda.graph(graph, stream=stream):
            gemm_step(False)
        launches_per_step = N.nvfp4_launch_count() - n0
    torch.cuda.synchronize()

    def timed_loop(replay, steps, warmup, per_step_extra=None):
        with torch.cuda.stream(stream):
            for _ in range(warmup):
                replay()
                flush_buf.zero_()
            stream.synchronize()
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
            barrier()
            t0 = time.time()
            for i in range(steps):
                evs[i][0].record(stream)
                replay()
                evs[i][1].record(stream)
                if per_step_extra:
                    per_step_extra(i)
                flush_buf.zero_()
            stream.synchronize()
            t1 = time.time()
            barrier()
        sampler.mark(t0, t1)
        return [a.elapsed_time(b) for a, b in evs]

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    step_ms = timed_loop(graph.replay, args.steps, args.warmup)
    # GEMM-only kernel durations (same work, eager launches with events between kernels).
    gemm_ms = {L["name"]: [] for L in layers}
    with torch.cuda.stream(stream):
        for _ in range(max(3, min(args.steps, 20))):
            torch.cuda._sleep(2_000_000)  # ~1 ms of device time: the host enqueues the whole step meanwhile
            gemm_step(True)
            stream.synchronize()
            for L in layers:
                gemm_ms[L["name"]].append(L["ev"][0].elapsed_time(L["ev"][1]))
            flush_buf.zero_()
    gemm_mean = {k: statistics.mean(v) for k, v in gemm_ms.items()}

    # e2e: host activations (pinned) -> device, full path, outputs -> pinned host, every step.
    host_a = [L["a"].cpu().pin_memory() for L in layers]
    host_o = [torch.empty(L["out"].shape, dtype=torch.bfloat16).pin_memory() for L in layers]
    h2d = sum(t.numel() * t.element_size() for t in host_a)
    d2h = sum(t.numel() * t.element_size() for t in host_o)

    # Copies run on their own streams so each layer's H2D, compute and D2H
    # overlap the others' (the two copy directions also run concurrently).
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev_fork = torch.cuda.Event()
    ev_in = [torch.cuda.Event() for _ in layers]
    ev_c = [torch.cuda.Event() for _ in layers]
    ev_join = torch.cuda.Event()

    def e2e_step():
        ev_fork.record(stream)
        s_in.wait_event(ev_fork)
        s_out.wait_event(ev_fork)
        with torch.cuda.stream(s_in):
            for L, ha, e in zip(layers, host_a, ev_in):
                L["a"].copy_(ha, non_blocking=True)
                e.record(s_in)
        for L, ho, ei, ec in zip(layers, host_o, ev_in, ev_c):
            stream.wait_event(ei)
            N.nvfp4_quantize_dynamic(L["a"], L["qstate"], L["ga"], L["ac"], L["asf"], N.SCALES_MMA)
            N.nvfp4_linear(L["ac"], L["asf"], L["ga"], L["wc"], L["ws"], L["gw"], L["out"], M, L["N"], L["K"])
            ec.record(stream)
            s_out.wait_event(ec)
            with torch.cuda.stream(s_out):
                ho.copy_(L["out"], non_blocking=True)
        ev_join.record(s_out)
        stream.wait_event(ev_join)

    e2e_ms = timed_loop(e2e_step, max(3, min(args.steps, 50)), args.warmup)

    # ---------------- the other linear workloads (reported beside the headline, not in it)
    def gemm_bytes(Mm, Nn, K):
        # Algorithmic bytes: codes 0.5 B/elem, scales 1/16 B/elem, bf16 output 2 B/elem, each operand once.
        return Mm * K * (0.5 + 1 / 16) + Nn * K * (0.5 + 1 / 16) + Mm * Nn * 2

    fp4_peak = peaks["bf16_tflops"] * FP4_OVER_BF16

    def graph_of(fn):
        with torch.cuda.stream(stream):
            fn()
            stream.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                fn()
        torch.cuda.synchronize()
        return g

    def roofline_of(flop, byt, ms):
        s_ = ms * 1e-3
        t_mem, t_cmp = byt / (peaks["hbm_gbs"] * 1e9), flop / (fp4_peak * 1e12)
        if t_cmp >= t_mem:
            return {"bound": "tensor", "achieved": flop / s_ / 1e12, "peak": fp4_peak, "unit": "TFLOP/s",
                    "frac": flop / s_ / 1e12 / fp4_peak}
        return {"bound": "hbm", "achieved": byt / s_ / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": byt / s_ / 1e9 / peaks["hbm_gbs"]}

    other_steps = min(args.steps, 10)
    other = {}
    for wl in OTHER_LINEAR_WLS:
        Mw, lw, fw = build_layers(wl)
        g = graph_of(lambda lw=lw, Mw=Mw: gemm_step(False, lw, Mw))
        ms_w = statistics.mean(timed_loop(g.replay, other_steps, args.warmup))
        per = {}
        with torch.cuda.stream(stream):
            for _ in range(3):
                flush_buf.zero_()
                torch.cuda._sleep(2_000_000)
                gemm_step(True, lw, Mw)
                stream.synchronize()
                for L in lw:
                    per.setdefault(L["name"], []).append(L["ev"][0].elapsed_time(L["ev"][1]))
        byt = sum(gemm_bytes(Mw, L["N"], L["K"]) for L in lw)
        # Each GEMM also back to back, as a graph-replayed serving loop runs it: a CUDA
        # graph of launches that rotate over enough copies of W (codes and scales,
        # > 256 MiB in all) that every launch streams W from DRAM; per-launch time =
        # graph time / launches.  The single-launch times above include the launch
        # latency that such a loop hides.
        b2b = {}
        for L in lw:
            wbytes = L["wc"].numel() + L["ws"].numel()
            copies = min(256, max(2, -(-(256 << 20) // wbytes)))
            wcs = [(L["wc"], L["ws"])] + [(L["wc"].clone(), L["ws"].clone()) for _ in range(copies - 1)]
            launches = 2 * copies

            def rep(L=L, wcs=wcs, n=launches, Mw=Mw):
                for i in range(n):
                    wc_i, ws_i = wcs[i % len(wcs)]
                    N.nvfp4_linear(L["ac"], L["asf"], L["ga"], wc_i, ws_i, L["gw"], L["out"], Mw, L["N"], L["K"])

            gb = graph_of(rep)
            b2b[L["name"]] = statistics.mean(timed_loop(gb.replay, 3, 1)) / launches
            del gb, wcs
            torch.cuda.empty_cache()
        entry = {"step": "per linear: tensor scale + quantize activation (one launch) + NVFP4 GEMM",
                 "ms_per_step": ms_w, "tflops": fw / (ms_w * 1e-3) / 1e12,
                 "gemm_us": {k: 1e3 * statistics.median(v) for k, v in per.items()},
                 "gemm_roofline": {k: roofline_of(2 * Mw * L["N"] * L["K"], gemm_bytes(Mw, L["N"], L["K"]),
                                                  statistics.median(per[L["name"]])) for k, L in
                                   ((L["name"], L) for L in lw)},
                 "gemm_us_back_to_back": {k: 1e3 * v for k, v in b2b.items()},
                 "gemm_roofline_back_to_back": {L["name"]: roofline_of(2 * Mw * L["N"] * L["K"],
                                                                       gemm_bytes(Mw, L["N"], L["K"]),
                                                                       b2b[L["name"]]) for L in lw},
                 "algorithmic_gemm_bytes": byt}
        if Mw <= 32 and all(L["K"] <= 1536 for L in lw):
            # The same step through nvfp4_linear_dynamic: tensor scale,
            # quantization and GEMM of each linear in one launch (bit-identical
            # outputs, checked in the GPU tests).
            def one_launch_step(lw=lw):
                for L in lw:
                    N.nvfp4_linear_dynamic(L["a"], L["wc"], L["ws"], L["gw"], L["out"], L["N"], g_a=L["ga"])

            gf = graph_of(one_launch_step)
            ms_f = statistics.mean(timed_loop(gf.replay, other_steps, args.warmup))
            entry["one_launch"] = {"step": "per linear: nvfp4_linear_dynamic (tensor scale, quantization and "
                                           "GEMM in one launch)",
                                   "ms_per_step": ms_f, "tflops": fw / (ms_f * 1e-3) / 1e12}
            del gf
        kva = synth.WORKLOADS[wl].get("kv_append")
        if kva:
            # One new token for each of n_new sequences, K and V quantized and appended.
            n_new, hk = kva["n_new"], kva["num_kv_heads"]
            gen = torch.Generator(device=dev)
            gen.manual_seed(synth.seed_for(wl, "kv_append") % (1 << 62))
            kn = torch.randn(n_new, hk, 128, generator=gen, device=dev).to(torch.bfloat16)
            vn = torch.randn(n_new, hk, 128, generator=gen, device=dev).to(torch.bfloat16)
            c3_cache = N.KVCache(n_new, hk, 16, float(kn.float().abs().max()) / 2688,
                                 float(vn.float().abs().max()) / 2688, device=dev)
            seq_a = torch.arange(n_new, dtype=torch.int32, device=dev)
            pos_a = torch.full((n_new,), 7, dtype=torch.int32, device=dev)
            ga_ = graph_of(lambda: N.kv_append_nvfp4(c3_cache, kn, vn, seq_a, pos_a))
            ms_a = statistics.mean(timed_loop(ga_.replay, other_steps, args.warmup))
            a_bytes = n_new * hk * 2 * (256 + 72)
            entry["kv_append"] = {"rows": n_new * hk, "us": 1e3 * ms_a, "algorithmic_bytes": a_bytes,
                                  "gbs": a_bytes / (ms_a * 1e-3) / 1e9}
            del c3_cache, kn, vn
        other[wl] = entry
        del lw, g
        torch.cuda.empty_cache()

    # ---------------- MXFP4 W4A4 (the format variant): per linear, the activation
    # rotated by H_32/sqrt(32) per 32-element block and MXFP4-quantized in one
    # launch (no tensor-wide scale, so no amax pass), then the MXFP4 GEMM
    # against W rotated and quantized once.
    def build_mx_layers(wl):
        Mw = synth.WORKLOADS[wl]["M"]
        out_layers, out_flops = [], 0
        for name, (Nn, K) in synth.WORKLOADS[wl]["linears"].items():
            a, W = synth.linear_inputs(wl, name, device=dev)
            wc = torch.empty(Nn, K // 2, dtype=torch.uint8, device=dev)
            ws = torch.empty(N.mxfp4_scales_bytes(Nn, K, N.SCALES_MMA), dtype=torch.uint8, device=dev)
            N.mxfp4_quantize(W, wc, ws, N.SCALES_MMA, rotate=True)
            del W
            out_layers.append(dict(name=name, N=Nn, K=K, a=a, wc=wc, ws=ws,
                                   ac=torch.empty(Mw, K // 2, dtype=torch.uint8, device=dev),
                                   asf=torch.empty(N.mxfp4_scales_bytes(Mw, K, N.SCALES_MMA), dtype=torch.uint8,
                                                   device=dev),
                                   out=torch.empty(Mw, Nn, dtype=torch.bfloat16, device=dev),
                                   ev=[torch.cuda.Event(enable_timing=True) for _ in range(3)]))
            out_flops += 2 * Mw * Nn * K
        torch.cuda.synchronize()
        return Mw, out_layers, out_flops

    def mx_step(lw, Mw, record=False):
        for L in lw:
            if record:
                L["ev"][0].record()
            N.mxfp4_quantize(L["a"], L["ac"], L["asf"], N.SCALES_MMA, rotate=True)
            if record:
                L["ev"][1].record()
            N.mxfp4_linear(L["ac"], L["asf"], L["wc"], L["ws"], L["out"], Mw, L["N"], L["K"])
            if record:
                L["ev"][2].record()

    mx = {}
    for wl in ("qwen1.5b_prefill_linears_m2048", GEMM_WL):
        Mw, lw, fw = build_mx_layers(wl)
        g = graph_of(lambda lw=lw, Mw=Mw: mx_step(lw, Mw))
        ms_w = statistics.mean(timed_loop(g.replay, other_steps, args.warmup))
        q_ms, g_ms = {}, {}
        with torch.cuda.stream(stream):
            for _ in range(3):
                flush_buf.zero_()
                torch.cuda._sleep(2_000_000)
                mx_step(lw, Mw, record=True)
                stream.synchronize()
                for L in lw:
                    q_ms.setdefault(L["name"], []).append(L["ev"][0].elapsed_time(L["ev"][1]))
                    g_ms.setdefault(L["name"], []).append(L["ev"][1].elapsed_time(L["ev"][2]))
        q_bytes = {L["name"]: Mw * L["K"] * (2 + 0.5 + 1 / 16) for L in lw}
        mx[wl] = {"step": "per linear: rotate (H_32 blocks) + MXFP4 quantize activation (one launch) + MXFP4 GEMM",
                  "ms_per_step": ms_w, "tflops": fw / (ms_w * 1e-3) / 1e12,
                  "gemm_us": {k: 1e3 * statistics.median(v) for k, v in g_ms.items()},
                  "gemm_roofline": {L["name"]: roofline_of(2 * Mw * L["N"] * L["K"], gemm_bytes(Mw, L["N"], L["K"]),
                                                           statistics.median(g_ms[L["name"]])) for L in lw},
                  "quantize_us": {k: 1e3 * statistics.median(v) for k, v in q_ms.items()},
                  "quantize_gbs": {k: q_bytes[k] / (statistics.median(v) * 1e-3) / 1e9 for k, v in q_ms.items()},
                  "quantize_roofline": {k: {"bound": "hbm", "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                            "frac": q_bytes[k] / (statistics.median(v) * 1e-3) / 1e9 / peaks["hbm_gbs"]}
                                        for k, v in q_ms.items()}}
        del lw, g
        torch.cuda.empty_cache()

    # ---------------- decode attention over the NVFP4 cache
    aw = synth.WORKLOADS[ATTN_WL]
    Bq, hq, hkv, T = aw["batch"], aw["num_q_heads"], aw["num_kv_heads"], aw["context"]
    rec = synth.kv_recipe(ATTN_WL, device=dev)
    gk = torch.zeros(1, dtype=torch.float32, device=dev)
    gv = torch.zeros(1, dtype=torch.float32, device=dev)
    kv_chunks = []
    for b in range(Bq):
        k, v = rec.kv(T, seed=synth.seed_for(ATTN_WL, f"kv:{b}") % (1 << 62))
        kv_chunks.append((k, v))
    K_all = torch.stack([c[0] for c in kv_chunks]).view(-1, 128)
    V_all = torch.stack([c[1] for c in kv_chunks]).view(-1, 128)
    del kv_chunks
    N.nvfp4_tensor_scale(K_all, gk)
    N.nvfp4_tensor_scale(V_all, gv)
    cache = N.KVCache(Bq, hkv, T, gk.item(), gv.item(), device=dev)
    seq = torch.arange(Bq, dtype=torch.int32, device=dev).repeat_interleave(T)
    pos = torch.arange(T, dtype=torch.int32, device=dev).repeat(Bq)
    N.kv_append_nvfp4(cache, K_all.view(-1, hkv, 128), V_all.view(-1, hkv, 128), seq, pos)
    # The cache fill itself (a4 at prefill size: every token of every sequence,
    # K and V quantized and written), timed as a single launch after an L2 flush.
    fill_ms = []
    with torch.cuda.stream(stream):
        for _ in range(3):
            flush_buf.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            N.kv_append_nvfp4(cache, K_all.view(-1, hkv, 128), V_all.view(-1, hkv, 128), seq, pos)
            e1.record()
            stream.synchronize()
            fill_ms.append(e0.elapsed_time(e1))
    fill_bytes = Bq * T * hkv * 2 * (256 + 72)  # bf16 K and V rows in; codes and scales out
    fill_gbs = fill_bytes / (statistics.median(fill_ms) * 1e-3) / 1e9
    del K_all, V_all, seq, pos
    cache.seq_lens.fill_(T)
    q = rec.queries(Bq, hq, seed=synth.seed_for(ATTN_WL, "q") % (1 << 62))
    k_new, v_new = rec.kv(Bq, seed=synth.seed_for(ATTN_WL, "new") % (1 << 62))
    seq_new = torch.arange(Bq, dtype=torch.int32, device=dev)
    pos_new = torch.full((Bq,), T - 1, dtype=torch.int32, device=dev)
    attn_ws = torch.empty(N.decode_attention_nvfp4_workspace_size(Bq, hq, T) // 4, dtype=torch.float32, device=dev)
    attn_out = torch.empty(Bq, hq, 128, dtype=torch.bfloat16, device=dev)
    scale = 1.0 / math.sqrt(128)
    ev_a = [torch.cuda.Event(enable_timing=True) for _ in range(2)]

    def attn_step(record=False):
        N.kv_append_nvfp4(cache, k_new, v_new, seq_new, pos_new)
        if record:
            ev_a[0].record()
        N.decode_attention_nvfp4(cache, q, scale, attn_out, attn_ws)
        if record:
            ev_a[1].record()

    with torch.cuda.stream(stream):
        attn_step()
        stream.synchronize()
        agraph = torch.cuda.CUDAGraph()
        n0 = N.nvfp4_launch_count()
        with torch.cuda.graph(agraph, stream=stream):
            attn_step()
        attn_launches = N.nvfp4_launch_count() - n0
    attn_step_ms = timed_loop(agraph.replay, args.steps, args.warmup)
    attn_kernel_ms = []
    with torch.cuda.stream(stream):
        for _ in range(max(3, min(args.steps, 20))):
            torch.cuda._sleep(2_000_000)
            attn_step(True)
            stream.synchronize()
            attn_kernel_ms.append(ev_a[0].elapsed_time(ev_a[1]))
    sampler.stop()
    status = N.nvfp4_get_device_status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the bench")

    # ---------------- reduce over ranks (max time, summed work)
    ms_step = statistics.mean(step_ms)
    ms_e2e = statistics.mean(e2e_ms)
    ms_attn_step = statistics.mean(attn_step_ms)
    ms_attn_kernel = statistics.mean(attn_kernel_ms)
    ms_step, ms_e2e, ms_attn_step, ms_attn_kernel = reduce_max_over_ranks(
        [ms_step, ms_e2e, ms_attn_step, ms_attn_kernel], world)

    dom = max(layers, key=lambda L: gemm_mean[L["name"]])
    d_flops = 2 * M * dom["N"] * dom["K"]
    d_bytes = gemm_bytes(M, dom["N"], dom["K"])
    d_s = gemm_mean[dom["name"]] * 1e-3
    t_mem, t_cmp = d_bytes / (peaks["hbm_gbs"] * 1e9), d_flops / (fp4_peak * 1e12)
    if t_cmp >= t_mem:
        roof = {"bound": "tensor", "achieved": d_flops / d_s / 1e12, "peak": fp4_peak, "unit": "TFLOP/s"}
    else:
        roof = {"bound": "hbm", "achieved": d_bytes / d_s / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = ncu_traffic("gemm", (M, dom["N"], dom["K"]))
    roof["kernel"] = f"nvfp4_gemm_pair_kernel ({dom['name']}: {M}x{dom['N']}x{dom['K']})"
    roof["peak_src"] = (f"{peaks['src']}: bf16 {peaks['bf16_tflops']} TFLOP/s x {FP4_OVER_BF16:g} nominal FP4/BF16"
                        if roof["bound"] == "tensor" else f"{peaks['src']} HBM copy")
    roof["also"] = {"tflops": d_flops / d_s / 1e12, "tflops_frac_of_fp4_peak": d_flops / d_s / 1e12 / fp4_peak,
                    "gbs": d_bytes / d_s / 1e9, "gbs_frac": d_bytes / d_s / 1e9 / peaks["hbm_gbs"]}

    kv_tokens = Bq * hkv * T
    attn_bytes = kv_tokens * 2 * (64 + 8) + q.numel() * 2 + attn_out.numel() * 2
    attn_gbs = attn_bytes / (ms_attn_kernel * 1e-3) / 1e9

    result = {
        "metric": METRIC,
        "value": whole_job_rate(flops, world, ms_step) / 1e12,
        "unit": "TFLOP/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "e2m1 x e2m1 -> f32 accumulate -> bf16 (e4m3 block scales)",
        "data": "synthetic (seeded; Qwen-shaped activations with outlier channels, N(0,0.02) weights)",
        "config": {"workload": GEMM_WL, "M": M,
                   "linears": {L["name"]: [L["N"], L["K"]] for L in layers},
                   "step": "per linear: tensor scale + quantize activation (one launch) + NVFP4 GEMM (weights pre-quantized)",
                   "l2": "flushed between steps (256 MiB write)", "graph": "CUDA graph replay",
                   "parallelism": f"replicas x{world}"},
        "gemm_ms": gemm_mean,
        "roofline": roof,
        "e2e": {"value": whole_job_rate(flops, world, ms_e2e) / 1e12, "unit": "TFLOP/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e},
        "gpu_launches": launches_per_step * args.steps,
        "decode_attention": {
            "workload": ATTN_WL, "value": world * attn_gbs, "unit": "GB/s",
            "ms_attention": ms_attn_kernel, "ms_per_step": ms_attn_step,
            "step": "append 1 token/sequence (kv_append_nvfp4) + decode_attention_nvfp4",
            "algorithmic_bytes": attn_bytes,
            "roofline": {"bound": "hbm", "achieved": attn_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": attn_gbs / peaks["hbm_gbs"], "traffic": ncu_traffic("attention", (Bq, T)),
                         "kernel": "attn_partial_kernel + attn_combine_kernel (one decode_attention_nvfp4 call)"},
            "gpu_launches": attn_launches * args.steps,
            "kv_fill": {"step": "kv_append_nvfp4 of the whole cache (B x T tokens, H_kv heads, K and V)",
                        "tokens": Bq * T, "us": 1e3 * statistics.median(fill_ms), "algorithmic_bytes": fill_bytes,
                        "gbs": fill_gbs, "frac": fill_gbs / peaks["hbm_gbs"]},
        },
        "attention_gbs": world * attn_gbs,
        "attention_frac": attn_gbs / peaks["hbm_gbs"],
        "other_workloads": other,
        "mxfp4_w4a4": mx,
        "clocks": sampler.summary(),
    }
    if rank == 0 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(args.cpu_seconds)
    return result


# ------------------------------------------------------- oracle arm ---

class OracleSample:
    """Bounded oracle steps on the bench workload.

    One step: for each of the workload's 4 linears, the tensor scale of the
    whole activation, quantization of its first `rows` rows, and the fp64
    dequantized GEMM against the first `cols` output columns of the weight
    (all when fewer).  The weights' first `cols_max` rows are quantized once,
    with their whole-tensor scales, when the sample is built."""

    def __init__(self, cols_max):
        from oracle import nvfp4_oracle as O
        from paper_2606_15682_gb300 import synth
        self.O = O
        self.prep = []
        for name, (Nn, K) in synth.WORKLOADS[GEMM_WL]["linears"].items():
            a, W = synth.linear_inputs(GEMM_WL, name)
            Wf = W.float().numpy()
            del W
            gw = O.tensor_scale(Wf)
            n = min(cols_max, Nn)
            wc, ws = O.quantize(Wf[:n], gw)
            del Wf
            self.prep.append((a.float().numpy(), wc, ws, gw, n, K))

    def step(self, rows=64, cols=None):
        O = self.O
        fl = 0
        for a, wc, ws, gw, n, K in self.prep:
            n = n if cols is None else min(cols, n)
            ga = O.tensor_scale(a)
            ac, as_ = O.quantize(a[:rows], ga)
            O.linear(ac, as_, ga, wc[:n], ws[:n], gw)
            fl += 2 * rows * n * K
        return fl

    def sample_text(self, rows, cols):
        return (f"{rows} activation rows x the first {cols} output columns (all when fewer) of each of the 4 "
                f"linears of {GEMM_WL} per step (tensor scale of the whole activation + quantize the rows + "
                f"fp64 dequantized GEMM)")


def calibrated_cols(sample, budget_s, cols_max):
    """Output columns per linear that make one 64-row step take about budget_s."""
    t0 = time.perf_counter()
    sample.step(rows=64, cols=64)
    t = time.perf_counter() - t0
    return int(max(16, min(cols_max, 64 * budget_s / max(t, 1e-6))))


CPU_COLS_MAX = 2048


def cpu_baseline(seconds=15.0):
    """The oracle timed on the host cores for about `seconds` (rank 0, N = 1)."""
    sample = OracleSample(CPU_COLS_MAX)
    cols = calibrated_cols(sample, 2.0, CPU_COLS_MAX)
    t0 = time.perf_counter()
    fl = 0
    n = 0
    while True:
        fl += sample.step(rows=64, cols=cols)
        n += 1
        if time.perf_counter() - t0 > seconds:
            break
    dt = time.perf_counter() - t0
    return {"value": fl / dt / 1e12, "unit": "TFLOP/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{n} steps of {sample.sample_text(64, cols)}, {dt:.1f} s"}


def run_reference(args):
    """The oracle as it stands, on the host cores.  Each step is a bounded
    sample of the workload: 64 activation rows against the first `cols`
    output columns of each of the 4 linears.  `cols` is chosen from one
    calibration step so that warm-up and timed steps together take about
    90 s of host time, whatever --steps and --warmup ask for."""
    n_steps = args.steps + max(args.warmup, 1)
    sample = OracleSample(CPU_COLS_MAX)
    cols = calibrated_cols(sample, 90.0 / n_steps, CPU_COLS_MAX)
    for _ in range(max(args.warmup, 1)):
        sample.step(rows=64, cols=cols)
    times = []
    fl = 0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        fl = sample.step(rows=64, cols=cols)
        times.append(time.perf_counter() - t0)
    ms = statistics.mean(times) * 1e3
    value = fl / (ms * 1e-3) / 1e12
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64 (dequantized)", "data": "synthetic",
            "config": {"workload": GEMM_WL, "sample_rows": 64, "sample_cols": cols},
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": os.cpu_count(), "kind": "oracle",
                             "sample": sample.sample_text(64, cols)},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    if args.gpus != world:
        # N GPUs means N ranks, one per GPU, started by torch.distributed.run.
        sys.exit(f"bench.py: --gpus {args.gpus} but WORLD_SIZE={world}; launch N > 1 with "
                 f"python -m torch.distributed.run --nproc-per-node {args.gpus} bench.py --gpus {args.gpus}")
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)))
        return
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    res = run_ours(args, rank, world)
    if rank == 0:
        print(json.dumps(res))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
