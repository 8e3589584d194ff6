"""Host-only checks of the C ABI: the library builds, loads, exports every
function include/nvfp4.h declares, and rejects bad arguments before any
launch.  No call here reaches a GPU."""
import ctypes

import pytest

from _util import header_functions, lib


def test_header_declares_the_hot_path_calls():
    names = header_functions()
    for n in ["nvfp4_tensor_scale", "nvfp4_quantize", "nvfp4_linear", "kv_append_nvfp4",
              "decode_attention_nvfp4", "decode_attention_nvfp4_workspace_size", "nvfp4_get_device_status"]:
        assert n in names


def test_library_exports_every_declared_symbol():
    N = lib()
    so = ctypes.CDLL(N.LIB_PATH)
    for name in header_functions():
        assert hasattr(so, name), name
    assert sorted(N.EXPORTED) == header_functions()


def test_bounds_checked_build_compiles_and_exports_every_call():
    """The NVFP4_DEBUG variant (store indices checked, NVFP4_ERR_BOUNDS instead
    of a write) builds and exports the same C ABI."""
    import os
    from paper_2606_15682_gb300 import build as B
    path = B.build(debug=True)
    assert os.path.basename(os.path.dirname(path)) == "_build_debug"
    so = ctypes.CDLL(path)
    for name in header_functions():
        assert hasattr(so, name), name
    so.nvfp4_status_string.restype = ctypes.c_char_p
    assert b"bounds" in so.nvfp4_status_string(8)


def test_timeline_build_compiles_and_exports_every_call():
    """The NVFP4_TIMELINE variant (per-block stamps in the one-launch
    quantizer) builds, exports the same C ABI plus its stamp reader, and the
    release build does not export the reader."""
    import os
    import pytest
    from paper_2606_15682_gb300 import build as B
    path = B.build(timeline=True)
    assert os.path.basename(os.path.dirname(path)) == "_build_timeline"
    so = ctypes.CDLL(path)
    for name in header_functions():
        assert hasattr(so, name), name
    assert hasattr(so, "nvfp4_timeline_quantize_dynamic") and hasattr(so, "nvfp4_timeline_gemm")
    assert not hasattr(ctypes.CDLL(B.build(timeline=False, debug=False)), "nvfp4_timeline_quantize_dynamic")
    with pytest.raises(ValueError):
        B.build(debug=True, timeline=True)


def test_status_strings_and_sizes():
    N = lib()
    assert N.nvfp4_status_string(0) == "ok"
    assert "capacity" in N.nvfp4_status_string(7)
    assert "bounds" in N.nvfp4_status_string(8)
    assert N.nvfp4_scales_bytes(130, 256, N.SCALES_ROWMAJOR) == 130 * 16
    assert N.nvfp4_scales_bytes(130, 256, N.SCALES_MMA) == 256 * 16
    assert N.decode_attention_nvfp4_workspace_size(64, 40, 16384) > 0
    assert N.decode_attention_nvfp4_workspace_size(0, 40, 16384) == 0


def test_argument_validation_before_launch():
    N = lib()
    L = N._lib
    p = ctypes.c_void_p(0x10000)      # aligned, never dereferenced: validation fails first
    odd = ctypes.c_void_p(0x10001)
    s = ctypes.c_void_p(0)
    # null pointers
    assert L.nvfp4_linear(None, p, p, p, p, p, 128, 128, 256, p, 128, s) == 1
    assert L.nvfp4_tensor_scale(p, 4, 16, 16, None, s) == 1
    # shapes: K not a multiple of 256, N not a multiple of 16, ldo < N
    assert L.nvfp4_linear(p, p, p, p, p, p, 128, 128, 192, p, 128, s) == 2
    assert L.nvfp4_linear(p, p, p, p, p, p, 128, 120, 256, p, 128, s) == 2
    assert L.nvfp4_linear(p, p, p, p, p, p, 128, 128, 256, p, 64, s) == 2
    assert L.nvfp4_quantize(p, 4, 40, 40, p, p, p, 0, s) == 2            # cols % 16
    assert L.nvfp4_quantize(p, 4, 32, 32, p, p, p, 1, s) == 2            # MMA layout needs cols % 64
    assert L.nvfp4_quantize(p, 4, 64, 64, p, p, p, 7, s) == 1            # bad layout enum
    # alignment
    assert L.nvfp4_linear(odd, p, p, p, p, p, 128, 128, 256, p, 128, s) == 3
    assert L.nvfp4_quantize(odd, 4, 64, 64, p, p, p, 1, s) == 3
    assert L.nvfp4_quantize(p, 4, 64, 68, p, p, p, 1, s) == 3            # ld % 8
    # fused gate_up + SwiGLU + quantize: I % 128, K % 256, null g_out
    assert L.nvfp4_linear_swiglu_quantize(p, p, p, p, p, p, 256, 192, 512, p, p, p, s) == 2
    assert L.nvfp4_linear_swiglu_quantize(p, p, p, p, p, p, 256, 256, 384, p, p, p, s) == 2
    assert L.nvfp4_linear_swiglu_quantize(p, p, p, p, p, p, 256, 256, 512, None, p, p, s) == 1
    assert L.nvfp4_linear_swiglu_quantize(p, p, p, p, p, p, 256, 256, 512, p, odd, p, s) == 3
    assert L.nvfp4_interleave_gate_up(p, p, 24, 64, p, s) == 2                # I % 16
    assert L.nvfp4_interleave_gate_up(p, p, 32, 40, p, s) == 2                # row bytes % 16
    st = ctypes.c_void_p(0x20000)
    assert L.nvfp4_quantize_dynamic(p, 4, 64, 64, None, p, p, p, 1, s) == 1   # no state
    assert L.nvfp4_quantize_dynamic(p, 4, 64, 64, st, None, p, p, 1, s) == 1  # no g
    assert L.nvfp4_quantize_dynamic(p, 4, 64, 64, odd, p, p, p, 1, s) == 3    # state not 16-B aligned
    assert L.nvfp4_quantize_dynamic(p, 4, 32, 32, st, p, p, p, 1, s) == 2     # MMA layout needs cols % 64
    assert L.nvfp4_quantize_dynamic(p, 4, 64, 64, st, p, p, p, 9, s) == 1     # bad layout enum
    assert L.nvfp4_quantize_dynamic(p, 4, 64, 64, st, p, None, p, 1, s) == 1  # no codes
    # one-launch quantize + linear: M <= 32 and K <= 1536, else UNSUPPORTED
    ld = L.nvfp4_linear_dynamic
    assert ld(None, 16, 1536, 1536, p, p, p, 1536, p, 1536, None, s) == 1
    assert ld(p, 16, 1536, 1536, p, p, None, 1536, p, 1536, None, s) == 1
    assert ld(p, 33, 1536, 1536, p, p, p, 1536, p, 1536, None, s) == 4
    assert ld(p, 16, 1792, 1792, p, p, p, 1536, p, 1536, None, s) == 4
    assert ld(p, 0, 1536, 1536, p, p, p, 1536, p, 1536, None, s) == 2
    assert ld(p, 16, 1280 + 64, 1344, p, p, p, 1536, p, 1536, None, s) == 2   # K % 256
    assert ld(p, 16, 1536, 1528, p, p, p, 1536, p, 1536, None, s) == 2        # ld_x < K
    assert ld(p, 16, 1536, 1536, p, p, p, 1544, p, 1536, None, s) == 2        # ldo < N
    assert ld(p, 16, 1536, 1536, p, p, p, 120 + 4, p, 128, None, s) == 2      # N % 16
    assert ld(odd, 16, 1536, 1536, p, p, p, 1536, p, 1536, None, s) == 3
    assert ld(p, 16, 1536, 1540, p, p, p, 1536, p, 1536, None, s) == 3        # ld_x % 8
    assert ld(p, 16, 1536, 1536, p, p, p, 1536, p, 1536, odd, s) == 3         # g_a_out 4-B aligned


def test_mxfp4_validation_before_launch():
    N = lib()
    L = N._lib
    p = ctypes.c_void_p(0x10000)
    odd = ctypes.c_void_p(0x10008)       # 8-B but not 16-B aligned
    s = ctypes.c_void_p(0)
    assert N.mxfp4_scales_bytes(130, 256, N.SCALES_ROWMAJOR) == 130 * 8
    assert N.mxfp4_scales_bytes(130, 256, N.SCALES_MMA) == N.nvfp4_scales_bytes(130, 256, N.SCALES_MMA)
    assert L.mxfp4_quantize(p, 4, 48, 48, 0, p, p, 0, s) == 2         # cols % 32
    assert L.mxfp4_quantize(p, 4, 96, 96, 0, p, p, 1, s) == 2         # MMA layout needs cols % 64
    assert L.mxfp4_quantize(p, 4, 64, 64, 2, p, p, 1, s) == 1         # rotate must be 0 or 1
    assert L.mxfp4_quantize(p, 4, 64, 64, 0, p, p, 5, s) == 1         # bad layout enum
    assert L.mxfp4_quantize(odd, 4, 64, 64, 0, p, p, 1, s) == 3       # x alignment
    assert L.mxfp4_quantize(p, 4, 64, 64, 0, odd, p, 1, s) == 3       # codes 16-B aligned
    assert L.mxfp4_quantize(p, 4, 64, 64, 0, None, p, 1, s) == 1      # no codes
    assert L.mxfp4_quantize(None, 0, 64, 64, 0, None, None, 1, s) == 0   # empty: nothing to do
    assert L.mxfp4_linear(None, p, p, p, 128, 128, 256, p, 128, s) == 1
    assert L.mxfp4_linear(p, p, p, p, 128, 128, 192, p, 128, s) == 2  # K % 256
    assert L.mxfp4_linear(p, p, p, p, 128, 120, 256, p, 128, s) == 2  # N % 16
    assert L.mxfp4_linear(p, odd, p, p, 128, 128, 256, p, 128, s) == 3
    assert L.mxfp4_linear_swiglu_quantize(p, p, p, p, 256, 192, 512, 0, p, p, s) == 2    # I % 128
    assert L.mxfp4_linear_swiglu_quantize(p, p, p, p, 256, 256, 384, 0, p, p, s) == 2    # K % 256
    assert L.mxfp4_linear_swiglu_quantize(p, p, p, p, 256, 256, 512, 3, p, p, s) == 1    # rotate 0/1
    assert L.mxfp4_linear_swiglu_quantize(p, p, p, p, 256, 256, 512, 0, None, p, s) == 1
    assert L.mxfp4_linear_swiglu_quantize(p, p, p, p, 256, 256, 512, 0, odd, p, s) == 3


def test_fault_injection_knob_validation():
    N = lib()
    assert N._lib.nvfp4_debug_inject_fault(5) == 1
    assert N._lib.nvfp4_debug_inject_fault(N.FAULT_GEMM_SKIP_STAGE) == 0
    assert N._lib.nvfp4_debug_inject_fault(N.FAULT_ATTN_SKIP_STAGE) == 0
    assert N._lib.nvfp4_debug_inject_fault(N.FAULT_NONE) == 0


def test_kv_and_attention_validation():
    N = lib()
    import torch  # noqa: F401  (struct only; no device memory)

    def cache(**kw):
        c = N.KVCacheStruct(0x10000, 0x10000, 0x10000, 0x10000, 0x10000, 2, 2, 128, 64, 1.0, 1.0)
        for k, v in kw.items():
            setattr(c, k, v)
        return c
    L = N._lib
    p = ctypes.c_void_p(0x10000)
    s = ctypes.c_void_p(0)
    assert L.kv_append_nvfp4(ctypes.byref(cache(head_dim=64)), p, p, p, p, 1, None, s) == 2
    assert L.kv_append_nvfp4(ctypes.byref(cache(k_gscale=0.0)), p, p, p, p, 1, None, s) == 1
    assert L.kv_append_nvfp4(ctypes.byref(cache()), None, p, p, p, 1, None, s) == 1
    # KV element format must be one of the enum's values
    assert L.kv_append_nvfp4(ctypes.byref(cache(kv_format=2)), p, p, p, p, 1, None, s) == 1
    assert L.decode_attention_nvfp4(ctypes.byref(cache(kv_format=-1)), p, 4, ctypes.c_float(0.1), p, p, 1 << 30, s) == 1
    # fused RoPE append: table required, and it must cover every cache position
    odd = ctypes.c_void_p(0x10004)
    assert L.kv_append_rope_nvfp4(ctypes.byref(cache()), p, p, p, p, 1, None, 64, None, s) == 1
    assert L.kv_append_rope_nvfp4(ctypes.byref(cache()), p, p, p, p, 1, p, 63, None, s) == 2
    assert L.kv_append_rope_nvfp4(ctypes.byref(cache()), p, p, p, p, 1, odd, 64, None, s) == 3
    assert L.nvfp4_rope_table(p, 16, 127, ctypes.c_float(1e6), s) == 2          # odd head_dim
    assert L.nvfp4_rope_table(p, 16, 128, ctypes.c_float(0.5), s) == 1          # theta <= 1
    assert L.nvfp4_rope_table(None, 16, 128, ctypes.c_float(1e6), s) == 1
    assert L.nvfp4_rope_table(None, 0, 128, ctypes.c_float(1e6), s) == 0        # empty: nothing to do
    ws = N.decode_attention_nvfp4_workspace_size(2, 4, 64)
    assert L.decode_attention_nvfp4(ctypes.byref(cache()), p, 3, ctypes.c_float(0.1), p, p, ws, s) == 2   # 3 % 2
    assert L.decode_attention_nvfp4(ctypes.byref(cache()), p, 18, ctypes.c_float(0.1), p, p, 1 << 30, s) == 2  # group 9
    assert L.decode_attention_nvfp4(ctypes.byref(cache()), p, 4, ctypes.c_float(0.1), p, p, ws - 16, s) == 2
    assert L.decode_attention_nvfp4(ctypes.byref(cache()), p, 4, ctypes.c_float(-1.0), p, p, ws, s) == 1
    ws_odd = N.decode_attention_nvfp4_workspace_size(2, 4, 63)
    assert L.decode_attention_nvfp4(ctypes.byref(cache(capacity=63)), p, 4, ctypes.c_float(0.1), p, p, ws_odd, s) == 2
    # attention with the output quantized for the o projection
    f = ctypes.c_float(0.1)
    assert L.decode_attention_nvfp4_quantize(ctypes.byref(cache()), p, 4, f, None, p, p, p, ws, s) == 1     # no g_out
    assert L.decode_attention_nvfp4_quantize(ctypes.byref(cache()), p, 4, f, p, None, p, p, ws, s) == 1     # no codes
    assert L.decode_attention_nvfp4_quantize(ctypes.byref(cache()), p, 3, f, p, p, p, p, ws, s) == 2        # 3 % 2
    assert L.decode_attention_nvfp4_quantize(ctypes.byref(cache()), p, 4, f, p, p, p, p, ws - 16, s) == 2   # workspace
    assert L.decode_attention_nvfp4_quantize(ctypes.byref(cache()), p, 4, f, p, odd, p, p, ws, s) == 3      # codes align
    assert L.decode_attention_nvfp4_quantize(ctypes.byref(cache(kv_format=5)), p, 4, f, p, p, p, p, ws, s) == 1
    # Q-FIT calibration: arguments checked before any CUDA call
    qws = N.nvfp4_qfit_workspace_size(2, 64, 4, 2, 3, 3)
    assert qws > 0 and N.nvfp4_qfit_workspace_size(2, 64, 4, 3, 3, 3) == 0          # 4 % 3
    assert N.nvfp4_qfit_workspace_size(2, 8193, 4, 2, 3, 3) == 0                        # > 8192 tokens
    assert N.nvfp4_qfit_workspace_size(2, 64, 4, 2, 0, 3) == 0                          # empty grid
    Q = L.nvfp4_qfit_calibrate
    ok = (p, p, p, 2, 64, 4, 2, 128, p, 64, 3, 3, ctypes.c_double(1e-6), 0, p, p, p, None, p, qws, s)
    def qcall(**kw):
        a = list(ok)
        for i, val in kw.items():
            a[int(i[1:])] = val
        return Q(*a)
    assert qcall(a0=None) == 1                                   # no queries
    assert qcall(a13=2) == 1                                     # kv format
    assert qcall(a12=ctypes.c_double(0.0)) == 1                  # eps
    assert qcall(a7=64) == 2                                     # head_dim
    assert qcall(a9=63) == 2                                     # table shorter than the cache
    assert qcall(a19=qws - 1) == 2                               # workspace
    assert qcall(a18=ctypes.c_void_p(0x10010)) == 3              # workspace alignment
    # static-scratch attention: a problem whose partials exceed the fixed
    # scratch is refused on the host, before any CUDA call
    big = cache(batch=64, num_kv_heads=1, capacity=131072)
    assert N.decode_attention_nvfp4_workspace_size(64, 8, 131072) > N.ATTN_STATIC_SCRATCH_BYTES
    assert L.decode_attention_nvfp4_static_scratch(ctypes.byref(big), p, 8, f, p, s) == 2
    assert L.decode_attention_nvfp4_static_scratch(ctypes.byref(cache()), p, 4, f, None, s) == 1
