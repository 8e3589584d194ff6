"""Thin ctypes binding of libnvfp4.so (include/nvfp4.h).

Argument marshalling only: every function takes torch CUDA tensors (or plain
integers for scalars), passes their device pointers and the current CUDA
stream to the C entry point of the same name, and raises ``NVFP4Error`` on a
non-OK status.  No computation happens here, and there is no CPU fallback:
if the library is missing, importing this module fails.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
# NVFP4_DEBUG=1 selects the bounds-checked build, NVFP4_TIMELINE=1 the
# timeline build (paper_2606_15682_gb300.build).
LIB_PATH = os.path.join(_PKG, "_build_debug" if os.environ.get("NVFP4_DEBUG") == "1" else
                        ("_build_timeline" if os.environ.get("NVFP4_TIMELINE") == "1" else "_build"), "libnvfp4.so")

SCALES_ROWMAJOR = 0
SCALES_MMA = 1

STATUS = {0: "ok", 1: "invalid argument", 2: "shape", 3: "alignment", 4: "unsupported", 5: "cuda",
          6: "timeout", 7: "capacity"}


class NVFP4Error(RuntimeError):
    def __init__(self, fn, code):
        self.code = code
        super().__init__(f"{fn} failed: {STATUS.get(code, code)} ({code})")


if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: run paper_2606_15682_gb300.build.build() first")
_lib = ctypes.CDLL(LIB_PATH)

_p, _i64, _i32, _f32, _sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float, ctypes.c_size_t


class KVCacheStruct(ctypes.Structure):
    _fields_ = [("k_codes", _p), ("k_scales", _p), ("v_codes", _p), ("v_scales", _p), ("seq_lens", _p),
                ("batch", _i32), ("num_kv_heads", _i32), ("head_dim", _i32), ("capacity", _i32),
                ("k_gscale", _f32), ("v_gscale", _f32), ("kv_format", _i32)]


def _sig(name, args, res=ctypes.c_int):
    f = getattr(_lib, name)
    f.argtypes = args
    f.restype = res
    return f


_tensor_scale = _sig("nvfp4_tensor_scale", [_p, _i64, _i64, _i64, _p, _p])
_quantize = _sig("nvfp4_quantize", [_p, _i64, _i64, _i64, _p, _p, _p, ctypes.c_int, _p])
_quantize_dynamic = _sig("nvfp4_quantize_dynamic", [_p, _i64, _i64, _i64, _p, _p, _p, _p, ctypes.c_int, _p])
_relayout = _sig("nvfp4_scales_relayout", [_p, _p, _i64, _i64, ctypes.c_int, ctypes.c_int, _p])
_linear = _sig("nvfp4_linear", [_p, _p, _p, _p, _p, _p, _i64, _i64, _i64, _p, _i64, _p])
_linear_dynamic = _sig("nvfp4_linear_dynamic", [_p, _i64, _i64, _i64, _p, _p, _p, _i64, _p, _i64, _p, _p])
_linear_swiglu = _sig("nvfp4_linear_swiglu_quantize", [_p, _p, _p, _p, _p, _p, _i64, _i64, _i64, _p, _p, _p, _p])
_interleave = _sig("nvfp4_interleave_gate_up", [_p, _p, _i64, _i64, _p, _p])
_kv_append = _sig("kv_append_nvfp4", [ctypes.POINTER(KVCacheStruct), _p, _p, _p, _p, _i64, _p, _p])
_kv_append_rope = _sig("kv_append_rope_nvfp4",
                       [ctypes.POINTER(KVCacheStruct), _p, _p, _p, _p, _i64, _p, _i64, _p, _p])
_rope_table = _sig("nvfp4_rope_table", [_p, _i64, _i32, _f32, _p])
_attn_ws = _sig("decode_attention_nvfp4_workspace_size", [_i32, _i32, _i32], _sz)
_attn = _sig("decode_attention_nvfp4", [ctypes.POINTER(KVCacheStruct), _p, _i32, _f32, _p, _p, _sz, _p])
_attn_quant = _sig("decode_attention_nvfp4_quantize",
                   [ctypes.POINTER(KVCacheStruct), _p, _i32, _f32, _p, _p, _p, _p, _sz, _p])
_attn_static = _sig("decode_attention_nvfp4_static_scratch", [ctypes.POINTER(KVCacheStruct), _p, _i32, _f32, _p, _p])
_qfit_ws = _sig("nvfp4_qfit_workspace_size", [_i32, _i32, _i32, _i32, _i32, _i32], _sz)
_qfit = _sig("nvfp4_qfit_calibrate", [_p, _p, _p, _i32, _i32, _i32, _i32, _i32, _p, _i64, _i32, _i32,
                                      ctypes.c_double, _i32, _p, _p, _p, _p, _p, _sz, _p])
_get_status = _sig("nvfp4_get_device_status", [ctypes.POINTER(_i32), _p])
_status_string = _sig("nvfp4_status_string", [ctypes.c_int], ctypes.c_char_p)
_launch_count = _sig("nvfp4_launch_count", [], ctypes.c_uint64)
_scales_bytes = _sig("nvfp4_scales_bytes", [_i64, _i64, ctypes.c_int], _sz)
_mx_scales_bytes = _sig("mxfp4_scales_bytes", [_i64, _i64, ctypes.c_int], _sz)
_inject_fault = _sig("nvfp4_debug_inject_fault", [ctypes.c_int])
FAULT_NONE, FAULT_ATTN_SKIP_STAGE, FAULT_GEMM_SKIP_STAGE = 0, 1, 2


def nvfp4_debug_inject_fault(what):
    """Test-only: arm one injected fault for the next call of its kind (see include/nvfp4.h)."""
    _check("nvfp4_debug_inject_fault", _inject_fault(what))
_mx_quantize = _sig("mxfp4_quantize", [_p, _i64, _i64, _i64, ctypes.c_int, _p, _p, ctypes.c_int, _p])
_mx_linear = _sig("mxfp4_linear", [_p, _p, _p, _p, _i64, _i64, _i64, _p, _i64, _p])
_mx_linear_swiglu = _sig("mxfp4_linear_swiglu_quantize", [_p, _p, _p, _p, _i64, _i64, _i64, ctypes.c_int, _p, _p, _p])


# The current stream's raw handle without building a torch.cuda.Stream object
# (0.1 us instead of ~3 us per call); the public call where it is absent.
_raw_current_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(stream):
    if stream is None:
        if _raw_current_stream is not None:
            return ctypes.c_void_p(_raw_current_stream(torch.cuda.current_device()))
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _ptr(t):
    """Device pointer of a dense tensor (None -> NULL)."""
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensor arguments must be contiguous (row-padded 2-D inputs go through the ld argument)")
    return ctypes.c_void_p(t.data_ptr())


def _mat(x):
    """(pointer, rows, cols, ld) of a 2-D row-major tensor whose rows may be padded."""
    if x.dim() != 2 or (x.shape[1] > 1 and x.stride(1) != 1):
        raise ValueError("expected a 2-D row-major tensor")
    rows, cols = x.shape
    ld = x.stride(0) if rows > 1 else cols
    if rows > 1 and ld < cols:
        raise ValueError("rows overlap")
    return ctypes.c_void_p(x.data_ptr()), rows, cols, ld


def _check(fn, code):
    if code != 0:
        raise NVFP4Error(fn, code)


# ----------------------------------------------------------------- calls ---

def nvfp4_scales_bytes(rows, cols, layout):
    return int(_scales_bytes(rows, cols, layout))


def nvfp4_tensor_scale(x, g, stream=None):
    """g[0] <- amax(|x|) / (6*448) (device)."""
    _check("nvfp4_tensor_scale", _tensor_scale(*_mat(x), _ptr(g), _stream(stream)))


def nvfp4_quantize(x, g, codes, scales, layout=SCALES_MMA, stream=None):
    _check("nvfp4_quantize", _quantize(*_mat(x), _ptr(g), _ptr(codes), _ptr(scales), layout, _stream(stream)))


DYNAMIC_STATE_BYTES = 16
KV_E2M1, KV_E1M2 = 0, 1


def nvfp4_quantize_dynamic(x, state, g, codes, scales, layout=SCALES_MMA, stream=None):
    """Tensor scale + quantization in one launch; `state` is a zero-filled
    device buffer of DYNAMIC_STATE_BYTES bytes owned by the caller."""
    _check("nvfp4_quantize_dynamic",
           _quantize_dynamic(*_mat(x), _ptr(state), _ptr(g), _ptr(codes), _ptr(scales), layout, _stream(stream)))


def nvfp4_scales_relayout(src, dst, rows, cols, from_layout, to_layout, stream=None):
    _check("nvfp4_scales_relayout", _relayout(_ptr(src), _ptr(dst), rows, cols, from_layout, to_layout,
                                              _stream(stream)))


def nvfp4_linear(a_codes, a_scales, g_a, w_codes, w_scales, g_w, out, M, N, K, ldo=None, stream=None):
    _check("nvfp4_linear", _linear(_ptr(a_codes), _ptr(a_scales), _ptr(g_a), _ptr(w_codes), _ptr(w_scales),
                                   _ptr(g_w), M, N, K, _ptr(out), N if ldo is None else ldo, _stream(stream)))


def nvfp4_linear_dynamic(x, w_codes, w_scales, g_w, out, N, ldo=None, g_a=None, stream=None):
    """Tensor scale, quantization of the bf16 activation x [M, K] (M <= 32,
    K <= 1536) and the linear layer with W in one launch; g_a (optional
    device float) receives the tensor scale."""
    ptr, M, K, ld = _mat(x)
    _check("nvfp4_linear_dynamic", _linear_dynamic(ptr, M, K, ld, _ptr(w_codes), _ptr(w_scales), _ptr(g_w), N,
                                                   _ptr(out), N if ldo is None else ldo, _ptr(g_a),
                                                   _stream(stream)))


def mxfp4_scales_bytes(rows, cols, layout):
    return int(_mx_scales_bytes(rows, cols, layout))


def mxfp4_quantize(x, codes, scales, layout=SCALES_MMA, rotate=False, stream=None):
    """MXFP4 codes and E8M0 block scales of a bf16 [rows, cols] tensor
    (optionally after the 32-element block rotation)."""
    _check("mxfp4_quantize", _mx_quantize(*_mat(x), int(bool(rotate)), _ptr(codes), _ptr(scales), layout,
                                          _stream(stream)))


def mxfp4_linear(a_codes, a_scales, w_codes, w_scales, out, M, N, K, ldo=None, stream=None):
    _check("mxfp4_linear", _mx_linear(_ptr(a_codes), _ptr(a_scales), _ptr(w_codes), _ptr(w_scales), M, N, K,
                                      _ptr(out), N if ldo is None else ldo, _stream(stream)))


def mxfp4_linear_swiglu_quantize(a_codes, a_scales, w_codes, w_scales, M, I, K, out_codes, out_scales,
                                  rotate=False, stream=None):
    _check("mxfp4_linear_swiglu_quantize",
           _mx_linear_swiglu(_ptr(a_codes), _ptr(a_scales), _ptr(w_codes), _ptr(w_scales), M, I, K,
                             int(bool(rotate)), _ptr(out_codes), _ptr(out_scales), _stream(stream)))


def nvfp4_linear_swiglu_quantize(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, I, K, g_out,
                                 out_codes, out_scales, stream=None):
    _check("nvfp4_linear_swiglu_quantize",
           _linear_swiglu(_ptr(a_codes), _ptr(a_scales), _ptr(g_a), _ptr(w_codes), _ptr(w_scales), _ptr(g_w),
                          M, I, K, _ptr(g_out), _ptr(out_codes), _ptr(out_scales), _stream(stream)))


def nvfp4_interleave_gate_up(w_gate, w_up, w_out, stream=None):
    _check("nvfp4_interleave_gate_up",
           _interleave(_ptr(w_gate), _ptr(w_up), w_gate.shape[0], w_gate.shape[1] * w_gate.element_size(),
                       _ptr(w_out), _stream(stream)))


def kv_append_nvfp4(cache, k, v, seq_idx, pos, k_shift=None, stream=None):
    s = cache.struct()
    _check("kv_append_nvfp4", _kv_append(ctypes.byref(s), _ptr(k), _ptr(v), _ptr(seq_idx), _ptr(pos), k.shape[0],
                                         _ptr(k_shift), _stream(stream)))


def kv_append_rope_nvfp4(cache, k_pre, v, seq_idx, pos, rope_table, k_shift=None, stream=None):
    """rope_table: float32 [n_pos, 64, 2] (see nvfp4_rope_table), n_pos >= cache.capacity."""
    s = cache.struct()
    _check("kv_append_rope_nvfp4",
           _kv_append_rope(ctypes.byref(s), _ptr(k_pre), _ptr(v), _ptr(seq_idx), _ptr(pos), k_pre.shape[0],
                           _ptr(rope_table), rope_table.shape[0], _ptr(k_shift), _stream(stream)))


def nvfp4_rope_table(table, theta=1.0e6, stream=None):
    """Fill table (float32 [n_pos, head_dim/2, 2]) with (cos, sin) of p * theta^(-2i/head_dim)."""
    _check("nvfp4_rope_table", _rope_table(_ptr(table), table.shape[0], 2 * table.shape[1], theta, _stream(stream)))


def decode_attention_nvfp4_workspace_size(batch, num_q_heads, capacity):
    return int(_attn_ws(batch, num_q_heads, capacity))


def decode_attention_nvfp4(cache, q, softmax_scale, out, workspace, stream=None):
    s = cache.struct()
    _check("decode_attention_nvfp4", _attn(ctypes.byref(s), _ptr(q), q.shape[1], softmax_scale, _ptr(out),
                                           _ptr(workspace), workspace.numel() * workspace.element_size(),
                                           _stream(stream)))


ATTN_STATIC_SCRATCH_BYTES = 24 << 20


def decode_attention_nvfp4_quantize(cache, q, softmax_scale, g_out, out_codes, out_scales, workspace, stream=None):
    """out_codes [batch, H_q*64] uint8, out_scales MMA layout for [batch, H_q*128]."""
    s = cache.struct()
    _check("decode_attention_nvfp4_quantize",
           _attn_quant(ctypes.byref(s), _ptr(q), q.shape[1], softmax_scale, _ptr(g_out), _ptr(out_codes),
                       _ptr(out_scales), _ptr(workspace), workspace.numel() * workspace.element_size(),
                       _stream(stream)))


def decode_attention_nvfp4_static_scratch(cache, q, softmax_scale, out, stream=None):
    """Decode attention whose partials live in the library's own device scratch (no workspace)."""
    s = cache.struct()
    _check("decode_attention_nvfp4_static_scratch", _attn_static(ctypes.byref(s), _ptr(q), q.shape[1], softmax_scale,
                                                                 _ptr(out), _stream(stream)))


def nvfp4_qfit_workspace_size(batch, tokens, num_q_heads, num_kv_heads, grid_s, grid_m):
    return int(_qfit_ws(batch, tokens, num_q_heads, num_kv_heads, grid_s, grid_m))


def nvfp4_qfit_calibrate(q_pre, k_pre, v, rope_table, grid_s, grid_m, eps, kv_format, s_q, s_k, m, errors,
                         workspace, stream=None):
    """q_pre [B, T, H_q, 128], k_pre and v [B, T, H_kv, 128] bf16; rope_table fp32 [n, 64, 2];
    s_q, s_k, m fp32 device outputs; errors: a host (CPU) float64 tensor of grid_s * grid_m, or None."""
    B, T, hq, d = q_pre.shape
    hkv = k_pre.shape[2]
    if errors is not None and (errors.device.type != "cpu" or errors.dtype != torch.float64 or
                               not errors.is_contiguous() or errors.numel() != grid_s * grid_m):
        raise ValueError("errors must be a contiguous CPU float64 tensor of grid_s * grid_m")
    _check("nvfp4_qfit_calibrate",
           _qfit(_ptr(q_pre), _ptr(k_pre), _ptr(v), B, T, hq, hkv, d, _ptr(rope_table), rope_table.shape[0], grid_s,
                 grid_m, float(eps), kv_format, _ptr(s_q), _ptr(s_k), _ptr(m),
                 None if errors is None else ctypes.c_void_p(errors.data_ptr()), _ptr(workspace),
                 workspace.numel() * workspace.element_size(), _stream(stream)))


def nvfp4_get_device_status(stream=None):
    v = _i32(0)
    _check("nvfp4_get_device_status", _get_status(ctypes.byref(v), _stream(stream)))
    return int(v.value)


def nvfp4_status_string(code):
    return _status_string(code).decode()


def nvfp4_launch_count():
    return int(_launch_count())


# ------------------------------------------------------------- KV cache ---

class KVCache:
    """Caller-owned NVFP4 KV cache buffers (layout of include/nvfp4.h)."""

    def __init__(self, batch, num_kv_heads, capacity, k_gscale, v_gscale, head_dim=128, device="cuda", kv_format=0):
        self.batch, self.num_kv_heads, self.capacity, self.head_dim = batch, num_kv_heads, capacity, head_dim
        self.kv_format = kv_format  # KV_E2M1 or KV_E1M2
        self.k_gscale, self.v_gscale = float(k_gscale), float(v_gscale)
        shape = (batch, num_kv_heads, capacity)
        self.k_codes = torch.zeros(shape + (head_dim // 2,), dtype=torch.uint8, device=device)
        self.v_codes = torch.zeros_like(self.k_codes)
        self.k_scales = torch.zeros(shape + (head_dim // 16,), dtype=torch.uint8, device=device)
        self.v_scales = torch.zeros_like(self.k_scales)
        self.seq_lens = torch.zeros(batch, dtype=torch.int32, device=device)

    def struct(self):
        return KVCacheStruct(self.k_codes.data_ptr(), self.k_scales.data_ptr(), self.v_codes.data_ptr(),
                             self.v_scales.data_ptr(), self.seq_lens.data_ptr(), self.batch, self.num_kv_heads,
                             self.head_dim, self.capacity, self.k_gscale, self.v_gscale, self.kv_format)


EXPORTED = ["nvfp4_scales_bytes", "nvfp4_tensor_scale", "nvfp4_quantize", "nvfp4_quantize_dynamic", "nvfp4_scales_relayout", "nvfp4_linear",
            "nvfp4_linear_dynamic",
            "nvfp4_linear_swiglu_quantize", "nvfp4_interleave_gate_up",
            "mxfp4_scales_bytes", "mxfp4_quantize", "mxfp4_linear", "mxfp4_linear_swiglu_quantize",
            "kv_append_nvfp4", "kv_append_rope_nvfp4", "nvfp4_rope_table", "decode_attention_nvfp4_workspace_size", "decode_attention_nvfp4",
            "decode_attention_nvfp4_quantize",
            "decode_attention_nvfp4_static_scratch", "nvfp4_qfit_workspace_size", "nvfp4_qfit_calibrate",
            "nvfp4_get_device_status", "nvfp4_status_string", "nvfp4_launch_count", "nvfp4_debug_inject_fault"]
