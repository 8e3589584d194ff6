"""Run one kernel of the hot path on one workload a few times (for profilers).

    python -m paper_2606_15682_gb300.cases gemm --workload qwen1.5b_prefill_linears_m2048 --linear gate_up
    python -m paper_2606_15682_gb300.cases quantize --workload qwen1.5b_prefill_linears_m2048 --linear down
    python -m paper_2606_15682_gb300.cases quantize_dynamic --workload qwen32b_prefill_linears_m8192 --linear down
    python -m paper_2606_15682_gb300.cases attention --batch 64 --context 16384
    python -m paper_2606_15682_gb300.cases gemm_swiglu --workload qwen32b_prefill_linears_m8192
    python -m paper_2606_15682_gb300.cases mx_gemm --workload qwen32b_prefill_linears_m8192 --linear down
    python -m paper_2606_15682_gb300.cases mx_quantize --workload qwen32b_prefill_linears_m8192 --linear down --rotate
    python -m paper_2606_15682_gb300.cases mx_gemm_swiglu --workload qwen32b_prefill_linears_m8192 --rotate
    NVFP4_TIMELINE=1 python -m paper_2606_15682_gb300.cases quantize_timeline --workload qwen1.5b_prefill_linears_m2048 --linear qkv
    NVFP4_TIMELINE=1 python -m paper_2606_15682_gb300.cases gemm_timeline --workload w4a4_linear_m16_k1536_n1536 --linear linear
    python -m paper_2606_15682_gb300.cases linear_dynamic --workload w4a4_linear_m16_k1536_n1536 --linear linear

Inputs are seeded synthetic tensors (paper_2606_15682_gb300.synth); for the
attention case the cache is filled with seeded random codes and scales
directly, which is enough to time the kernel.  Prints the mean CUDA-event time
of the measured call.  quantize_timeline (timeline build, NVFP4_TIMELINE=1)
prints, for one launch of the one-launch dynamic quantizer after an L2 flush,
when its blocks started, finished their loads, arrived at the grid barrier,
were released and issued their stores; gemm_timeline the same for one
single-CTA or split-K GEMM launch (set-up, first stage issued and landed, last
MMA issued, last accumulator seen by the epilogue or, split-K, the partial
drained into shared memory, stores complete, exit).
"""
from __future__ import annotations

import argparse
import math

import torch

from . import build as _build

_build.build()
from . import nvfp4 as N  # noqa: E402
from . import synth  # noqa: E402


def _quantized(x):
    g = torch.empty(1, dtype=torch.float32, device=x.device)
    N.nvfp4_tensor_scale(x, g)
    c = torch.empty(x.shape[0], x.shape[1] // 2, dtype=torch.uint8, device=x.device)
    s = torch.empty(N.nvfp4_scales_bytes(x.shape[0], x.shape[1], N.SCALES_MMA), dtype=torch.uint8, device=x.device)
    N.nvfp4_quantize(x, g, c, s, N.SCALES_MMA)
    return c, s, g


def _time(fn, iters):
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    fn()
    torch.cuda.synchronize()
    ev[0].record()
    for _ in range(iters):
        fn()
    ev[1].record()
    torch.cuda.synchronize()
    return ev[0].elapsed_time(ev[1]) / iters


def _quantize_timeline(a, dev):
    import ctypes
    if not hasattr(N._lib, "nvfp4_timeline_quantize_dynamic"):
        raise SystemExit("quantize_timeline needs the timeline build: run with NVFP4_TIMELINE=1")
    read = N._lib.nvfp4_timeline_quantize_dynamic
    read.argtypes = [ctypes.c_void_p]
    read.restype = ctypes.c_int
    x, _ = synth.linear_inputs(a.workload, a.linear, device=dev)
    M, K = x.shape
    state = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device=dev)
    g = torch.empty(1, dtype=torch.float32, device=dev)
    c = torch.empty(M, K // 2, dtype=torch.uint8, device=dev)
    s = torch.empty(N.nvfp4_scales_bytes(M, K, N.SCALES_MMA), dtype=torch.uint8, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()  # the zeroed barrier state is ordered before the first call
    for _ in range(3):
        N.nvfp4_quantize_dynamic(x, state, g, c, s, N.SCALES_MMA)
    host = (ctypes.c_ulonglong * (2048 * 5))()
    read(host)  # clears the stamps of the warm-up calls
    flush.zero_()
    torch.cuda._sleep(1_000_000)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record()
    N.nvfp4_quantize_dynamic(x, state, g, c, s, N.SCALES_MMA)
    ev[1].record()
    if read(host) != 0:
        raise SystemExit("reading the timeline failed")
    assert N.nvfp4_get_device_status() == 0
    rows = [host[5 * b:5 * b + 5] for b in range(2048) if host[5 * b] != 0]
    t0 = min(r[0] for r in rows)
    print(f"{a.workload}/{a.linear}: x {M}x{K} bf16 ({M * K * 2 / 1e6:.1f} MB), {len(rows)} blocks, "
          f"event {ev[0].elapsed_time(ev[1]) * 1e3:.2f} us, in-kernel span "
          f"{(max(r[4] for r in rows) - t0) / 1e3:.2f} us")
    for e, name in enumerate(["entry", "loads done", "arrived", "released", "stores issued"]):
        v = sorted(r[e] - t0 for r in rows)
        print(f"  {name:13s} min {v[0] / 1e3:6.2f}  median {v[len(v) // 2] / 1e3:6.2f}  max {v[-1] / 1e3:6.2f} us")


def _gemm_timeline(a, dev):
    import ctypes
    if not hasattr(N._lib, "nvfp4_timeline_gemm"):
        raise SystemExit("gemm_timeline needs the timeline build: run with NVFP4_TIMELINE=1")
    read = N._lib.nvfp4_timeline_gemm
    read.argtypes = [ctypes.c_void_p]
    read.restype = ctypes.c_int
    x, W = synth.linear_inputs(a.workload, a.linear, device=dev)
    M, K = x.shape
    Nn = W.shape[0]
    ac, asf, ga = _quantized(x)
    wc, wsf, gw = _quantized(W)
    out = torch.empty(M, Nn, dtype=torch.bfloat16, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(3):
        N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K)
    host = (ctypes.c_ulonglong * (1024 * 8))()
    read(host)  # clears the warm-up launches' stamps
    flush.zero_()
    torch.cuda._sleep(1_000_000)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record()
    N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K)
    ev[1].record()
    if read(host) != 0:
        raise SystemExit("reading the timeline failed")
    assert N.nvfp4_get_device_status() == 0
    rows = [host[8 * c:8 * c + 8] for c in range(1024) if host[8 * c] != 0]
    if not rows:
        raise SystemExit("no stamps: this shape runs neither the single-CTA nor the split-K GEMM kernel")
    t0 = min(r[0] for r in rows)
    print(f"{a.workload}/{a.linear}: {M}x{Nn}x{K}, {len(rows)} CTAs, event {ev[0].elapsed_time(ev[1]) * 1e3:.2f} us, "
          f"in-kernel span {(max(r[7] for r in rows) - t0) / 1e3:.2f} us")
    names = ["entry", "set-up done", "1st stage issued", "1st stage landed", "last MMA issued",
             "acc. seen/drained", "stores done", "exit"]
    for e, name in enumerate(names):
        v = sorted(r[e] - t0 for r in rows if r[e] != 0)
        if v:
            print(f"  {name:16s} min {v[0] / 1e3:6.2f}  median {v[len(v) // 2] / 1e3:6.2f}  max {v[-1] / 1e3:6.2f} us")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("kernel", choices=["gemm", "gemm_swiglu", "quantize", "quantize_dynamic", "tensor_scale",
                                       "attention", "mx_gemm", "mx_quantize", "mx_gemm_swiglu", "quantize_timeline",
                                       "gemm_timeline", "linear_dynamic"])
    ap.add_argument("--rotate", action="store_true", help="MXFP4: 32-element block rotation before quantizing")
    ap.add_argument("--workload", default="qwen1.5b_prefill_linears_m2048")
    ap.add_argument("--linear", default="gate_up")
    ap.add_argument("--batch", type=int, default=64)
    ap.add_argument("--context", type=int, default=16384)
    ap.add_argument("--iters", type=int, default=3)
    ap.add_argument("--rows", type=int, default=None,
                    help="gemm/quantize: activation rows instead of the workload's M (smaller profiler cases)")
    ap.add_argument("--kv-format", choices=["e2m1", "e1m2"], default="e2m1")
    a = ap.parse_args()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    if a.kernel == "quantize_timeline":
        _quantize_timeline(a, dev)
        return
    if a.kernel == "gemm_timeline":
        _gemm_timeline(a, dev)
        return
    if a.kernel == "gemm_swiglu":
        # gate_up of the workload with SwiGLU + NVFP4 quantization of the down
        # projection's input in the epilogue, against the same GEMM with bf16
        # output followed by the one-launch quantizer on an [M, I] tensor.
        x, W = synth.linear_inputs(a.workload, "gate_up", device=dev)
        M, K = x.shape
        I = W.shape[0] // 2
        Wi = torch.empty_like(W)
        N.nvfp4_interleave_gate_up(W[:I].contiguous(), W[I:].contiguous(), Wi)
        del W
        ac, asf, ga = _quantized(x)
        wc, wsf, gw = _quantized(Wi)
        del Wi
        g_out = torch.tensor([0.05], dtype=torch.float32, device=dev)
        qc = torch.empty(M, I // 2, dtype=torch.uint8, device=dev)
        qs = torch.empty(N.nvfp4_scales_bytes(M, I, N.SCALES_MMA), dtype=torch.uint8, device=dev)
        ms_f = _time(lambda: N.nvfp4_linear_swiglu_quantize(ac, asf, ga, wc, wsf, gw, M, I, K, g_out, qc, qs), a.iters)
        out = torch.empty(M, 2 * I, dtype=torch.bfloat16, device=dev)
        h = out[:, :I].contiguous()
        st = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device=dev)
        g_h = torch.empty(1, dtype=torch.float32, device=dev)

        def unfused():
            N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, 2 * I, K)
            N.nvfp4_quantize_dynamic(h, st, g_h, qc, qs, N.SCALES_MMA)
        ms_u = _time(unfused, a.iters)
        print(f"gemm_swiglu {a.workload} {M}x{2 * I}x{K}: fused {ms_f * 1e3:.1f} us "
              f"({2 * M * 2 * I * K / ms_f / 1e9:.1f} TFLOP/s); bf16 GEMM + quantize of h {ms_u * 1e3:.1f} us "
              f"(SwiGLU itself not included)")
    elif a.kernel == "mx_gemm_swiglu":
        # MXFP4 gate_up with SwiGLU + MXFP4 quantization of h in the epilogue,
        # against the MXFP4 GEMM with bf16 output followed by mxfp4_quantize of h.
        x, W = synth.linear_inputs(a.workload, "gate_up", device=dev)
        M, K = x.shape
        I = W.shape[0] // 2
        Wi = torch.empty_like(W)
        N.nvfp4_interleave_gate_up(W[:I].contiguous(), W[I:].contiguous(), Wi)
        del W

        def mxq(t):
            c = torch.empty(t.shape[0], t.shape[1] // 2, dtype=torch.uint8, device=dev)
            sc = torch.empty(N.mxfp4_scales_bytes(t.shape[0], t.shape[1], N.SCALES_MMA), dtype=torch.uint8, device=dev)
            N.mxfp4_quantize(t, c, sc, N.SCALES_MMA, rotate=a.rotate)
            return c, sc
        ac, asf = mxq(x)
        wc, wsf = mxq(Wi)
        del Wi
        qc = torch.empty(M, I // 2, dtype=torch.uint8, device=dev)
        qs = torch.empty(N.mxfp4_scales_bytes(M, I, N.SCALES_MMA), dtype=torch.uint8, device=dev)
        ms_f = _time(lambda: N.mxfp4_linear_swiglu_quantize(ac, asf, wc, wsf, M, I, K, qc, qs, rotate=a.rotate),
                     a.iters)
        out = torch.empty(M, 2 * I, dtype=torch.bfloat16, device=dev)
        h = out[:, :I].contiguous()

        def unfused():
            N.mxfp4_linear(ac, asf, wc, wsf, out, M, 2 * I, K)
            N.mxfp4_quantize(h, qc, qs, N.SCALES_MMA, rotate=a.rotate)
        ms_u = _time(unfused, a.iters)
        print(f"mx_gemm_swiglu{' (rotated)' if a.rotate else ''} {a.workload} {M}x{2 * I}x{K}: fused {ms_f * 1e3:.1f} us "
              f"({2 * M * 2 * I * K / ms_f / 1e9:.1f} TFLOP/s); bf16 GEMM + MXFP4 quantize of h {ms_u * 1e3:.1f} us "
              f"(SwiGLU itself not included)")
    elif a.kernel in ("mx_gemm", "mx_quantize"):
        x, W = synth.linear_inputs(a.workload, a.linear, device=dev)
        M, K = x.shape
        Nn = W.shape[0]

        def mx(t):
            c = torch.empty(t.shape[0], t.shape[1] // 2, dtype=torch.uint8, device=dev)
            sc = torch.empty(N.mxfp4_scales_bytes(t.shape[0], t.shape[1], N.SCALES_MMA), dtype=torch.uint8, device=dev)
            return c, sc
        ac, asf = mx(x)
        if a.kernel == "mx_quantize":
            ms = _time(lambda: N.mxfp4_quantize(x, ac, asf, N.SCALES_MMA, rotate=a.rotate), a.iters)
            byt = M * K * (2 + 0.5 + 1 / 16)
            print(f"mx_quantize{' (rotated)' if a.rotate else ''} {a.workload}/{a.linear} {M}x{K}: "
                  f"{ms * 1e3:.1f} us, {byt / ms / 1e6:.0f} GB/s")
        else:
            wc, wsf = mx(W)
            N.mxfp4_quantize(x, ac, asf, N.SCALES_MMA, rotate=a.rotate)
            N.mxfp4_quantize(W, wc, wsf, N.SCALES_MMA, rotate=a.rotate)
            del W
            out = torch.empty(M, Nn, dtype=torch.bfloat16, device=dev)
            ms = _time(lambda: N.mxfp4_linear(ac, asf, wc, wsf, out, M, Nn, K), a.iters)
            print(f"mx_gemm {a.workload}/{a.linear} {M}x{Nn}x{K}: {ms * 1e3:.1f} us, "
                  f"{2 * M * Nn * K / ms / 1e9:.1f} TFLOP/s")
    elif a.kernel == "linear_dynamic":
        # Tensor scale, quantization and GEMM in one launch (M <= 32), against
        # the one-launch quantizer followed by the GEMM.
        x, W = synth.linear_inputs(a.workload, a.linear, device=dev)
        M, K = x.shape
        Nn = W.shape[0]
        wc, wsf, gw = _quantized(W)
        del W
        out = torch.empty(M, Nn, dtype=torch.bfloat16, device=dev)
        ga = torch.empty(1, dtype=torch.float32, device=dev)
        ms_f = _time(lambda: N.nvfp4_linear_dynamic(x, wc, wsf, gw, out, Nn, g_a=ga), a.iters)
        st = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device=dev)
        ac = torch.empty(M, K // 2, dtype=torch.uint8, device=dev)
        asf = torch.empty(N.nvfp4_scales_bytes(M, K, N.SCALES_MMA), dtype=torch.uint8, device=dev)

        def two_calls():
            N.nvfp4_quantize_dynamic(x, st, ga, ac, asf, N.SCALES_MMA)
            N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K)
        ms_u = _time(two_calls, a.iters)
        print(f"linear_dynamic {a.workload}/{a.linear} {M}x{Nn}x{K}: one launch {ms_f * 1e3:.1f} us, "
              f"quantize_dynamic + linear {ms_u * 1e3:.1f} us")
    elif a.kernel in ("gemm", "quantize", "quantize_dynamic", "tensor_scale"):
        x, W = synth.linear_inputs(a.workload, a.linear, M=a.rows, device=dev)
        M, K = x.shape
        Nn = W.shape[0]
        if a.kernel == "gemm":
            ac, asf, ga = _quantized(x)
            wc, wsf, gw = _quantized(W)
            del W
            out = torch.empty(M, Nn, dtype=torch.bfloat16, device=dev)
            ms = _time(lambda: N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K), a.iters)
            print(f"gemm {a.workload}/{a.linear} {M}x{Nn}x{K}: {ms * 1e3:.1f} us, "
                  f"{2 * M * Nn * K / ms / 1e9:.1f} TFLOP/s")
        else:
            g = torch.empty(1, dtype=torch.float32, device=dev)
            N.nvfp4_tensor_scale(x, g)
            c = torch.empty(M, K // 2, dtype=torch.uint8, device=dev)
            s = torch.empty(N.nvfp4_scales_bytes(M, K, N.SCALES_MMA), dtype=torch.uint8, device=dev)
            if a.kernel == "quantize":
                ms = _time(lambda: N.nvfp4_quantize(x, g, c, s, N.SCALES_MMA), a.iters)
                byt = M * K * (2 + 0.5 + 1 / 16)
            elif a.kernel == "quantize_dynamic":
                st = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device=dev)
                ms = _time(lambda: N.nvfp4_quantize_dynamic(x, st, g, c, s, N.SCALES_MMA), a.iters)
                byt = M * K * (2 + 2 + 0.5 + 1 / 16)  # x read twice (amax pass, quantize pass)
            else:
                ms = _time(lambda: N.nvfp4_tensor_scale(x, g), a.iters)
                byt = M * K * 2
            print(f"{a.kernel} {a.workload}/{a.linear} {M}x{K}: {ms * 1e3:.1f} us, {byt / ms / 1e6:.0f} GB/s")
    else:
        B, hq, hkv, T = a.batch, 40, 8, a.context
        gen = torch.Generator(device=dev)
        gen.manual_seed(5)
        cache = N.KVCache(B, hkv, T, 0.01, 0.01, device=dev,
                          kv_format=N.KV_E1M2 if a.kv_format == "e1m2" else N.KV_E2M1)
        for t in (cache.k_codes, cache.v_codes):
            t.copy_(torch.randint(0, 256, t.shape, generator=gen, device=dev, dtype=torch.int32).to(torch.uint8))
        for t in (cache.k_scales, cache.v_scales):
            t.copy_(torch.randint(0x20, 0x58, t.shape, generator=gen, device=dev, dtype=torch.int32).to(torch.uint8))
        cache.seq_lens.fill_(T)
        q = torch.randn(B, hq, 128, generator=gen, device=dev).to(torch.bfloat16)
        ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, T) // 4, dtype=torch.float32, device=dev)
        out = torch.empty(B, hq, 128, dtype=torch.bfloat16, device=dev)
        ms = _time(lambda: N.decode_attention_nvfp4(cache, q, 1 / math.sqrt(128), out, ws), a.iters)
        byt = B * hkv * T * 144
        print(f"attention {a.kv_format} B={B} T={T}: {ms * 1e3:.1f} us, {byt / ms / 1e6:.0f} GB/s (K/V codes+scales)")
    assert N.nvfp4_get_device_status() == 0


if __name__ == "__main__":
    main()
