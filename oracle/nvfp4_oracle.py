"""CPU oracle for the NVFP4 W4A4KV4 hot path -- TEST INFRASTRUCTURE ONLY.

Only the test suite, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this module.  The product
path (the CUDA library and its Python binding) never calls it, and this module
imports nothing from the product package: the two share no code.

Everything here is the plain definition of what the path computes, written for
readability, not speed:

* the NVFP4 format (Appendix A, table "Quantization configurations of MXFP4 and
  NVFP4"): E2M1 elements, one FP8-E4M3 scale per block of 16 elements, one FP32
  per-tensor scale;
* the quantizer that maps a bf16 tensor onto that format (the paper fixes the
  format but not the recipe; the reading used is spelled out in ``quantize``);
* the linear layer on dequantized operands in fp64 (every linear of the decoder
  is quantized, Appendix D.1);
* decode attention over a quantized KV cache, ``z = softmax(Q K^T / sqrt(d)) V``
  with quantized K and V (Sec. 2.1), in fp64;
* the inference-time Q-FIT key shift ``K~ = R(K_pre / s) - m`` applied before
  the KV cache is quantized (Eq. 2, Appendix D.3), and the RoPE / paired scaling
  pieces needed to state its invariances (Sec. 2.1, Eq. 2);
* the fused step RoPE -> shift -> quantize -> append, with RoPE in fp32 from a
  (cos, sin) table in a fixed order of operations (``rope_f32``);
* the gate_up projection with the SwiGLU product and the NVFP4 quantization of
  the down projection's input fused behind it (``linear_swiglu_quantize``);
* the E1M2 element grid for the KV cache (``e1m2_*``, ``element="e1m2"``);
* the Q-FIT calibration (Algorithm 1): the paired pre-RoPE scale and the
  post-RoPE shift chosen by a grid search on the KV4 attention error
  (``qfit_calibrate``).

Floating-point conventions: the quantizer's arithmetic is IEEE fp32 with
round-to-nearest-even (numpy float32 scalars/arrays, no fused multiply-add);
everything downstream of dequantization is fp64.

Parity status: every function here is pinned by ``tests/test_oracle_pins.py``
(format tables, hand-worked ties in ``tests/golden/``, closed forms, library
routines and brute force on tiny inputs); none is "parity unpinned".
"""
from __future__ import annotations

import numpy as np

# ---------------------------------------------------------------------------
# E2M1 elements (Appendix A: FP4 with 2 exponent bits and 1 mantissa bit).
# A 4-bit code is  s e1 e0 m : sign, exponent (bias 1), mantissa.
#   e == 0 : subnormal, value = m * 0.5
#   e >= 1 : value = 2**(e-1) * (1 + m/2)
# The eight magnitudes are therefore 0, 0.5, 1, 1.5, 2, 3, 4, 6.
# ---------------------------------------------------------------------------


def e2m1_decode(code):
    """Value of 4-bit E2M1 codes (array of ints 0..15) as float64."""
    code = np.asarray(code, dtype=np.int64)
    sign = np.where(code & 0x8, -1.0, 1.0)
    e = (code >> 1) & 0x3
    m = code & 0x1
    mag = np.where(e == 0, m * 0.5, np.ldexp(1.0 + m / 2.0, e - 1))
    return sign * mag


E2M1_GRID = e2m1_decode(np.arange(8))  # non-negative magnitudes, index == code


def e2m1_encode(v):
    """Round float values onto E2M1, round-to-nearest-even, saturating at 6.

    The nearest grid point is chosen by brute force over the eight magnitudes;
    on an exact tie the code with an even index (even mantissa bit) wins.
    Values beyond 6 saturate to 6 ("satfinite").  The sign bit is kept, also
    when the magnitude rounds to zero (``-0.1 -> 0x8``).
    Inputs must be finite.
    """
    v = np.asarray(v, dtype=np.float64)
    flat = v.reshape(-1)
    out = np.empty(flat.shape, dtype=np.uint8)
    step = 1 << 20
    for lo in range(0, flat.size, step):
        x = flat[lo:lo + step]
        mag = np.abs(x)
        dist = np.abs(mag[:, None] - E2M1_GRID[None, :])          # (n, 8)
        best = dist.min(axis=1, keepdims=True)
        cand = dist == best                                          # ties: <= 2 adjacent
        even = cand & ((np.arange(8) % 2) == 0)[None, :]
        idx = np.where(even.any(axis=1), even.argmax(axis=1), cand.argmax(axis=1))
        idx = np.where(mag >= 6.0, 7, idx)
        out[lo:lo + step] = (idx | (np.signbit(x).astype(np.int64) << 3)).astype(np.uint8)
    return out.reshape(v.shape)


# ---------------------------------------------------------------------------
# FP8 E4M3 block scales (Appendix A).  OCP E4M3 "FN": 1 sign, 4 exponent bits
# (bias 7), 3 mantissa bits, no infinities, S.1111.111 is NaN, max 448.
# NVFP4 block scales are non-negative, i.e. the unsigned view the tensor core
# consumes; the encoder never produces the sign bit nor 0x7F.
# ---------------------------------------------------------------------------

E4M3_MAX = 448.0


def e4m3_decode(code):
    """Value of 8-bit E4M3 codes (array of ints 0..255) as float64 (NaN for 0x7F/0xFF)."""
    code = np.asarray(code, dtype=np.int64)
    sign = np.where(code & 0x80, -1.0, 1.0)
    e = (code >> 3) & 0xF
    m = code & 0x7
    mag = np.where(e == 0, np.ldexp(m / 8.0, -6), np.ldexp(1.0 + m / 8.0, e - 7))
    mag = np.where((e == 15) & (m == 7), np.nan, mag)
    return sign * mag


def e4m3_encode_nonneg(s):
    """Round non-negative values onto E4M3 (RNE), saturating to 448 ("satfinite").

    For s in binade [2**E, 2**(E+1)) with E >= -6 the representable values are
    multiples of 2**(E-3); below 2**-6 (subnormals) they are multiples of 2**-9.
    The value is rounded to the nearest multiple with ties to even (an even
    multiple is an even mantissa), then clamped to 448.  +inf saturates too.
    """
    s = np.asarray(s, dtype=np.float64)
    if np.any(np.isnan(s)) or np.any(s < 0):
        raise ValueError("e4m3_encode_nonneg: inputs must be non-negative and not NaN")
    finite = np.isfinite(s)
    sf = np.where(finite, s, 0.0)
    _, ex = np.frexp(sf)                    # sf = f * 2**ex, f in [0.5, 1)
    binade = np.maximum(ex - 1, -6)         # floor(log2(sf)), clamped to the subnormal range
    quantum = np.ldexp(1.0, binade - 3)
    val = np.rint(sf / quantum) * quantum   # np.rint: round half to even; the division is exact
    val = np.where(finite, np.minimum(val, E4M3_MAX), E4M3_MAX)
    return _e4m3_code_of_value(val)


def _e4m3_code_of_value(val):
    """Code of exactly representable non-negative E4M3 values."""
    val = np.asarray(val, dtype=np.float64)
    code = np.zeros(val.shape, dtype=np.int64)
    sub = (val > 0) & (val < 2.0 ** -6)
    code = np.where(sub, np.rint(val / 2.0 ** -9).astype(np.int64), code)
    nrm = val >= 2.0 ** -6
    _, ex = np.frexp(np.where(nrm, val, 1.0))
    E = ex - 1
    mant = np.rint((np.ldexp(np.where(nrm, val, 1.0), -E) - 1.0) * 8).astype(np.int64)
    code = np.where(nrm, ((E + 7) << 3) | mant, code)
    return code.astype(np.uint8)


# ---------------------------------------------------------------------------
# NVFP4 tensor quantization.
# ---------------------------------------------------------------------------

# ---------------------------------------------------------------------------
# E1M2 elements: the 4-bit KV-cache element of the paper's QAT runs (the
# Q-FIT section uses E1M2 for the KV cache; the paper names the format but not
# its bias).  Reading: 1 sign bit, 1 exponent bit with bias 0, 2 mantissa
# bits, so  e == 0: m/2 (subnormal), e == 1: 2 + m/2  -- the uniform grid
# 0, 0.5, ..., 3.5.  A magnitude is then k/2 with k = 0..7.
# Storage in this library's KV cache: the two's-complement nibble of
# n = sign * k (n in -7..7; the pattern of -8 is never written).
# ---------------------------------------------------------------------------

E1M2_MAX = 3.5


def e1m2_decode(nib):
    """Value of stored E1M2 nibbles (array of ints 0..15): n/2, n = nib as a
    4-bit two's-complement integer."""
    nib = np.asarray(nib, dtype=np.int64)
    n = np.where(nib >= 8, nib - 16, nib)
    return n.astype(np.float64) / 2.0


def e1m2_encode(v):
    """Round values onto E1M2: k = RNE(2|v|) (ties to even k, i.e. to an even
    mantissa), saturated at 7 (3.5); stored as the nibble of sign * k.  A
    negative value that rounds to zero is stored as 0 (one zero in two's
    complement)."""
    v = np.asarray(v, dtype=np.float64)
    k = np.minimum(np.rint(np.abs(v) * 2.0), 7).astype(np.int64)
    n = np.where(np.signbit(v), -k, k)
    return (n & 0xF).astype(np.uint8)


BLOCK = 16                    # elements per E4M3 block scale (Appendix A)
TENSOR_SCALE_DIV = np.float32(6.0 * 448.0)   # largest E2M1 magnitude x largest E4M3 scale


def bf16_bits_to_f32(bits):
    """bf16 bit patterns (uint16) -> exactly equal float32 values."""
    bits = np.asarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32)


def tensor_scale(x_f32):
    """FP32 per-tensor scale g = amax(|x|) / (6 * 448), fp32 division.

    With this g the largest element of the tensor maps onto the largest
    representable NVFP4 value (E2M1 6 times E4M3 448).  An all-zero tensor gets
    g = 1 (any positive g quantizes it to zero codes and zero scales).
    """
    amax = np.float32(np.max(np.abs(np.asarray(x_f32, dtype=np.float32)))) if np.size(x_f32) else np.float32(0)
    if amax == 0:
        return np.float32(1.0)
    return np.float32(amax / TENSOR_SCALE_DIV)


def quantize(x_f32, g, element="e2m1"):
    """NVFP4-quantize a [rows, cols] tensor along its rows (cols % 16 == 0).
    element="e1m2" swaps the element grid for the E1M2 KV variant (step 2
    then divides by 3.5 g instead of 6 g and step 4 rounds onto E1M2).

    Reading of the format (the paper gives the format, not the recipe), per
    block b of 16 consecutive elements of a row, all fp32 RNE:
      1. amax_b = max |x_i|
      2. s_f = amax_b / (6 * g)                       (product, then quotient)
      3. S = E4M3_RNE_satfinite(s_f)                  (block scale code)
      4. if S == 0: codes are the signs only (signed zeros)
         else:      v_i = x_i * (1 / (S * g))          (product, reciprocal, product)
                    code_i = E2M1_RNE_satfinite(v_i)  (sign kept)
    Returns (codes uint8 [rows, cols/2] with element 2j in the low nibble of
    byte j and element 2j+1 in the high nibble, scales uint8 [rows, cols/16]).
    """
    x = np.asarray(x_f32, dtype=np.float32)
    rows, cols = x.shape
    if cols % BLOCK:
        raise ValueError("cols must be a multiple of 16")
    g = np.float32(g)
    if not (np.isfinite(g) and g > 0):
        raise ValueError("tensor scale must be positive and finite")
    xb = x.reshape(rows, cols // BLOCK, BLOCK)
    amax = np.max(np.abs(xb), axis=2)                               # exact
    qmax = np.float32(6.0) if element == "e2m1" else np.float32(E1M2_MAX)
    six_g = np.float32(qmax * g)
    with np.errstate(over="ignore", divide="ignore"):
        s_f = (amax / six_g).astype(np.float32)
    S = e4m3_encode_nonneg(s_f)                                      # uint8 [rows, cols/16]
    S_val = e4m3_decode(S).astype(np.float32)                        # exact
    d = (S_val * g).astype(np.float32)
    zero_scale = S == 0
    with np.errstate(divide="ignore", over="ignore"):
        r = np.where(zero_scale, np.float32(0.0), np.float32(1.0) / np.where(zero_scale, np.float32(1.0), d))
    r = r.astype(np.float32)
    v = (xb * r[:, :, None]).astype(np.float32)                     # zero scale -> signed zeros
    codes = (e2m1_encode(v) if element == "e2m1" else e1m2_encode(v)).reshape(rows, cols)
    packed = (codes[:, 0::2] | (codes[:, 1::2] << 4)).astype(np.uint8)
    return packed, S


def unpack_codes(packed):
    """uint8 [rows, cols/2] -> 4-bit codes [rows, cols] (low nibble first)."""
    packed = np.asarray(packed, dtype=np.uint8)
    out = np.empty(packed.shape[:-1] + (packed.shape[-1] * 2,), dtype=np.uint8)
    out[..., 0::2] = packed & 0xF
    out[..., 1::2] = packed >> 4
    return out


def dequantize(packed, scales, g, element="e2m1"):
    """x_hat = e2m1(code) * e4m3(S) * g (or e1m2(code) ...), evaluated in fp64 (exact)."""
    codes = unpack_codes(packed)
    vals = e2m1_decode(codes) if element == "e2m1" else e1m2_decode(codes)
    rows, cols = codes.shape[-2], codes.shape[-1]
    s = e4m3_decode(scales).astype(np.float64)
    s = np.repeat(s, BLOCK, axis=-1)
    return vals * s * np.float64(np.float32(g))


# ---------------------------------------------------------------------------
# Block-scale storage order consumed by the tensor core ("MMA layout").
# Rows are grouped in tiles of 128, K-blocks in groups of 4 (64 elements).
# Each (row-tile, k-group) pair owns 512 contiguous bytes; pairs are stored
# k-group-fastest.  Inside a 512-byte atom, row r and k-block kb sit at byte
#     (r % 32) * 16 + ((r % 128) // 32) * 4 + (kb % 4).
# Rows beyond the tensor (padding up to a multiple of 128) hold zero.
# ---------------------------------------------------------------------------


def mma_scale_bytes(rows, cols):
    return ((rows + 127) // 128) * 128 * (cols // BLOCK)


def _mma_offsets(rows, kblocks):
    """Byte offset of every (row, k-block) scale in the MMA layout, [rows, kblocks]."""
    kgroups = kblocks // 4
    r = np.arange(rows, dtype=np.int64)[:, None]
    kb = np.arange(kblocks, dtype=np.int64)[None, :]
    return ((r // 128) * kgroups + kb // 4) * 512 + (r % 32) * 16 + ((r % 128) // 32) * 4 + kb % 4


def scales_to_mma(scales):
    """Row-major [rows, cols/16] scales -> flat MMA-layout byte array (padding rows zero)."""
    scales = np.asarray(scales, dtype=np.uint8)
    rows, kblocks = scales.shape
    if kblocks % 4:
        raise ValueError("cols must be a multiple of 64 for the MMA layout")
    out = np.zeros(mma_scale_bytes(rows, kblocks * BLOCK), dtype=np.uint8)
    out[_mma_offsets(rows, kblocks)] = scales
    return out


def scales_from_mma(flat, rows, cols):
    """Inverse of ``scales_to_mma`` (drops padding rows)."""
    flat = np.asarray(flat, dtype=np.uint8).reshape(-1)
    return flat[_mma_offsets(rows, cols // BLOCK)]


# ---------------------------------------------------------------------------
# Linear layer on NVFP4 operands (every linear of the decoder, Appendix D.1).
# D[m, n] = sum_k A_hat[m, k] * W_hat[n, k]  in fp64 on the dequantized inputs.
# ---------------------------------------------------------------------------


def linear(a_codes, a_scales, g_a, w_codes, w_scales, g_w):
    """fp64 reference of the NVFP4 linear: dequantize both operands, multiply."""
    a = dequantize(a_codes, a_scales, g_a)
    w = dequantize(w_codes, w_scales, g_w)
    return a @ w.T


def silu(x):
    """SiLU(x) = x * sigmoid(x) = x / (1 + e^-x), fp64 (the SwiGLU gate of the
    evaluated models' MLP, whose output feeds the quantized down projection)."""
    x = np.asarray(x, dtype=np.float64)
    return x / (1.0 + np.exp(-x))


def interleave_gate_up(w_gate, w_up):
    """Row order of the gate/up weight for the fused SwiGLU epilogue: blocks of
    16 gate rows alternate with the matching 16 up rows,
        out[32 j + t] = gate[16 j + t],  out[32 j + 16 + t] = up[16 j + t],  t < 16."""
    g = np.asarray(w_gate); u = np.asarray(w_up)
    I = g.shape[0]
    out = np.empty((2 * I,) + g.shape[1:], dtype=g.dtype)
    for j in range(I // 16):
        out[32 * j:32 * j + 16] = g[16 * j:16 * j + 16]
        out[32 * j + 16:32 * j + 32] = u[16 * j:16 * j + 16]
    return out


def linear_swiglu_quantize(a_codes, a_scales, g_a, wg_codes, wg_scales, wu_codes, wu_scales, g_w, g_out):
    """The down projection's input, h = SiLU(A W_gate^T) * (A W_up^T), from the
    NVFP4 operands in fp64, then NVFP4-quantized with the static scale g_out
    (same recipe as ``quantize``, applied to h rounded to fp32).  Returns
    (h fp64, codes, scales)."""
    G = linear(a_codes, a_scales, g_a, wg_codes, wg_scales, g_w)
    U = linear(a_codes, a_scales, g_a, wu_codes, wu_scales, g_w)
    h = silu(G) * U
    codes, scales = quantize(h.astype(np.float32), np.float32(g_out))
    return h, codes, scales


def linear_rows(a_codes, a_scales, g_a, w_codes, w_scales, g_w, rows):
    """Same as ``linear`` for a subset of output rows (large shapes)."""
    rows = np.asarray(rows)
    a = dequantize(a_codes[rows], a_scales[rows], g_a)
    w = dequantize(w_codes, w_scales, g_w)
    return a @ w.T


# ---------------------------------------------------------------------------
# KV cache: per-token NVFP4 rows with a static per-layer tensor scale.
# Cache arrays (one set for K, one for V):
#     codes  uint8 [batch, kv_heads, capacity, head_dim/2]
#     scales uint8 [batch, kv_heads, capacity, head_dim/16]
# Blocks of 16 run along head_dim, so every appended token is self-contained.
# ---------------------------------------------------------------------------


def kv_append(k_codes, k_scales, v_codes, v_scales, k_new, v_new, seq_idx, pos, g_k, g_v, k_shift=None,
              element="e2m1"):
    """Quantize and store new K/V rows in place.

    k_new, v_new: float32 [n_new, kv_heads, head_dim] (bf16 values, post-RoPE K).
    k_shift: optional float32 [kv_heads, head_dim]: the Q-FIT post-RoPE shift m,
    subtracted in fp32 before quantization, K~ = R(K) - m (Eq. 2).
    """
    k = np.asarray(k_new, dtype=np.float32)
    v = np.asarray(v_new, dtype=np.float32)
    n_new, hkv, d = k.shape
    if k_shift is not None:
        k = (k - np.asarray(k_shift, dtype=np.float32)[None, :, :]).astype(np.float32)
    kc, ks = quantize(k.reshape(n_new * hkv, d), g_k, element)
    vc, vs = quantize(v.reshape(n_new * hkv, d), g_v, element)
    kc = kc.reshape(n_new, hkv, d // 2); ks = ks.reshape(n_new, hkv, d // BLOCK)
    vc = vc.reshape(n_new, hkv, d // 2); vs = vs.reshape(n_new, hkv, d // BLOCK)
    for i in range(n_new):
        b, p = int(seq_idx[i]), int(pos[i])
        k_codes[b, :, p] = kc[i]; k_scales[b, :, p] = ks[i]
        v_codes[b, :, p] = vc[i]; v_scales[b, :, p] = vs[i]


def decode_attention(q_f32, k_codes, k_scales, v_codes, v_scales, seq_lens, g_k, g_v, softmax_scale,
                     batches=None, heads=None, element="e2m1"):
    """fp64 decode attention over the NVFP4 cache (Sec. 2.1).

    For query head h of sequence b, with KV head kv = h // (H_q / H_kv)
    (contiguous grouped-query replication):
        s_t = softmax_scale * (q . K_hat_t),  t < seq_lens[b]
        o   = sum_t softmax(s)_t * V_hat_t
    q_f32: [batch, H_q, d].  Returns fp64 [len(batches), len(heads), d].
    A sequence with no cached token has no softmax; its output is defined as
    zeros (the library's reading; the paper does not consider that case).
    """
    q = np.asarray(q_f32, dtype=np.float64)
    B, Hq, d = q.shape
    Hkv = k_codes.shape[1]
    if Hq % Hkv:
        raise ValueError("H_q must be a multiple of H_kv")
    group = Hq // Hkv
    batches = range(B) if batches is None else batches
    heads = range(Hq) if heads is None else heads
    scale = np.float64(np.float32(softmax_scale))
    out = np.zeros((len(batches), len(heads), d))
    for i, b in enumerate(batches):
        T = int(seq_lens[b])
        if T == 0:
            continue
        cache = {}
        for j, h in enumerate(heads):
            kv = h // group
            if kv not in cache:
                cache[kv] = (dequantize(k_codes[b, kv, :T], k_scales[b, kv, :T], g_k, element),
                             dequantize(v_codes[b, kv, :T], v_scales[b, kv, :T], g_v, element))
            K, V = cache[kv]
            out[i, j] = attention_fp64(q[b, h], K, V, scale)
    return out


def attention_fp64(q, K, V, scale):
    """softmax(scale * K q) V for one query vector, numerically stable, fp64."""
    s = (K @ q) * scale
    s = s - s.max()
    p = np.exp(s)
    p /= p.sum()
    return p @ V


# ---------------------------------------------------------------------------
# RoPE and the Q-FIT transforms (Sec. 2.1, Eq. 2).  Used to state invariances.
# RoPE rotates channel pairs (r, r + d/2) by angle pos * theta**(-2r/d).
# ---------------------------------------------------------------------------


def rope(x, positions, theta=1.0e6):
    """Apply RoPE to x [..., T, d] at integer positions [T] (fp64)."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-np.arange(half) * 2.0 / d)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def rope_table(n_pos, head_dim=128, theta=1.0e6):
    """RoPE (cos, sin) table, float32 [n_pos, head_dim/2, 2]: the fp64 values of
    cos/sin(pos * theta^(-2i/d)), i < d/2, rounded once to fp32 (Sec. 2.1; the
    rotate-half pairing of ``rope``)."""
    half = head_dim // 2
    inv = theta ** (-np.arange(half) * 2.0 / head_dim)
    ang = np.arange(n_pos, dtype=np.float64)[:, None] * inv[None, :]
    return np.stack([np.cos(ang), np.sin(ang)], axis=-1).astype(np.float32)


def rope_f32(x_f32, positions, table):
    """RoPE in fp32 from a (cos, sin) table, the order of operations fixed so a
    kernel can reproduce it exactly (round-to-nearest-even, no fused multiply-add):
        y[i]       = fl(fl(x[i] * c_i) - fl(x[i + d/2] * s_i))
        y[i + d/2] = fl(fl(x[i] * s_i) + fl(x[i + d/2] * c_i)),   i < d/2.
    x_f32 [n, ..., d] (one row per position), positions [n]."""
    x = np.asarray(x_f32, dtype=np.float32)
    half = x.shape[-1] // 2
    cs = np.asarray(table, dtype=np.float32)[np.asarray(positions)]      # [n, d/2, 2]
    shape = (x.shape[0],) + (1,) * (x.ndim - 2) + (half,)
    c = cs[..., 0].reshape(shape)
    sn = cs[..., 1].reshape(shape)
    x1, x2 = x[..., :half], x[..., half:]
    y1 = (x1 * c).astype(np.float32) - (x2 * sn).astype(np.float32)
    y2 = (x1 * sn).astype(np.float32) + (x2 * c).astype(np.float32)
    return np.concatenate([y1, y2], axis=-1).astype(np.float32)


def kv_append_rope(k_codes, k_scales, v_codes, v_scales, k_pre, v_new, seq_idx, pos, g_k, g_v, table,
                   k_shift=None, element="e2m1"):
    """The fused step before decode attention: K~ = RoPE(K_pre) - m (Eq. 2 with
    the pre-RoPE scaling s folded into the key projection), then quantize and
    store K~ and V as ``kv_append`` does.  k_pre: float32 [n_new, kv_heads, d]
    (bf16 values, before RoPE); RoPE and the shift in fp32 (``rope_f32``)."""
    k = rope_f32(k_pre, pos, table)
    kv_append(k_codes, k_scales, v_codes, v_scales, k, v_new, seq_idx, pos, g_k, g_v, k_shift, element)


def qfit_transform(q_pre, k_pre, s, m, positions, theta=1.0e6):
    """Q~ = R(Q_pre * s), K~ = R(K_pre / s) - m  (Eq. 2), fp64."""
    s = np.asarray(s, dtype=np.float64)
    return rope(q_pre * s, positions, theta), rope(k_pre / s, positions, theta) - np.asarray(m, np.float64)


# ---------------------------------------------------------------------------
# Q-FIT calibration (Algorithm 1, Sec. 4 / the Q-FIT appendix): choose the
# paired pre-RoPE scale S and the post-RoPE key shift m that minimize the MSE
# between a reference attention and the attention over the KV4 cache.
# Readings where the algorithm leaves a choice open:
#   * the calibration set is B sequences of T tokens at positions 0..T-1;
#     inputs are [B, T, heads, d];
#   * Attn is the causal attention of a decoder layer.  It is scored at the
#     last token of every sequence, which attends to all T tokens of its own
#     sequence: one decode step over the cached sequence.  (The paper averages
#     over every position of its calibration samples; the last-token subset
#     keeps the KV4 side a plain decode over one cache per grid point.)
#     Softmax scale 1/sqrt(d).
#   * RoPE is the fp32 table form ``rope_f32`` (tables from ``rope_table``);
#     the scaled keys K_pre / S_K are rounded to bf16 before RoPE, as a key
#     projection with S folded into its weights would produce them, and the
#     scaled, RoPE'd queries are rounded to bf16, the attention's input type.
#   * Q_KV4 uses a static tensor scale per grid point: g = amax / (qmax * 448)
#     of the tensor being cached (K~ - m over all sequences, or V).
#   * the shift template mu is the mean over all tokens of RoPE(K_pre), the
#     unscaled keys, as written; m(alpha_m) = alpha_m * mu at every alpha_s.
# ---------------------------------------------------------------------------


def _bf16_round(x):
    """Round fp32 values to bf16 (RNE) and back to fp32."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return (b << 16).astype(np.uint32).view(np.float32)


def _tokens(x):
    """[B, T, H, d] -> [B * T, H, d]."""
    x = np.asarray(x)
    return x.reshape((-1,) + x.shape[-2:])


def qfit_init_scale(k_pre, eps):
    """S_K^0[h, r] = max(max_t |K[t,h,r]|, max_t |K[t,h,r+d/2]|, eps) over every
    token of every sequence, shared by the pair (r, r + d/2) so the scaling
    commutes with RoPE.  k_pre [..., H_kv, d] -> [H_kv, d]."""
    k = np.abs(_tokens(k_pre).astype(np.float64))
    half = k.shape[-1] // 2
    m = np.maximum(k[..., :half].max(axis=0), k[..., half:].max(axis=0))
    s0 = np.maximum(m, eps)
    return np.concatenate([s0, s0], axis=-1)


def qfit_shift_template(k_pre, table):
    """mu = E_t[RoPE(K_pre)_t], the channel-wise mean of the post-RoPE keys over
    every token of every sequence (token t of a sequence at position t).
    k_pre [B, T, H_kv, d] -> fp64 [H_kv, d]."""
    k = np.asarray(k_pre, dtype=np.float32)
    B, T = k.shape[:2]
    pos = np.arange(T)
    rot = np.stack([rope_f32(k[b], pos, table) for b in range(B)])
    return rot.astype(np.float64).reshape((-1,) + k.shape[-2:]).mean(axis=0)


def qfit_reference(q_pre, k_pre, v, table):
    """Y_ref: the unquantized attention of the last token of each sequence,
    RoPE'd query against the RoPE'd keys and the values of all T tokens, fp64.
    Returns [B, H_q, d]."""
    q = np.asarray(q_pre, np.float32)
    k = np.asarray(k_pre, np.float32)
    vv = np.asarray(v, np.float64)
    B, T, hq, d = q.shape
    hkv = k.shape[2]
    group = hq // hkv
    pos = np.arange(T)
    scale = 1.0 / np.sqrt(d)
    out = np.zeros((B, hq, d))
    for b in range(B):
        k0 = rope_f32(k[b], pos, table).astype(np.float64)
        q0 = rope_f32(q[b, T - 1:T], np.array([T - 1]), table)[0].astype(np.float64)
        for h in range(hq):
            out[b, h] = attention_fp64(q0[h], k0[:, h // group], vv[b, :, h // group], scale)
    return out


def qfit_attention_error(q_pre, k_pre, v, table, s_k, s_q, m, element="e2m1", y_ref=None):
    """MSE between Y_ref and the attention of the last token of each sequence
    over the KV4 cache holding Q_KV4(RoPE(bf16(K_pre / s_k)) - m) and Q_KV4(V),
    with query bf16(RoPE(Q_pre * s_q)) (one grid point of Algorithm 1)."""
    q = np.asarray(q_pre, np.float32)
    k = np.asarray(k_pre, np.float32)
    vv = np.asarray(v, np.float32)
    B, T, hq, d = q.shape
    hkv = k.shape[2]
    group = hq // hkv
    qmax = 6.0 if element == "e2m1" else E1M2_MAX
    pos = np.arange(T)
    if y_ref is None:
        y_ref = qfit_reference(q_pre, k_pre, v, table)
    k_in = _bf16_round(k / np.asarray(s_k, np.float32)[None, None])
    kt = np.stack([rope_f32(k_in[b], pos, table) for b in range(B)])
    kt = (kt - np.asarray(m, np.float32)[None, None]).astype(np.float32)
    # static scales; an all-zero tensor gets scale 1 (the tensor-scale convention)
    a_k, a_v = np.abs(kt).max(), np.abs(vv).max()
    g_k = np.float32(a_k / np.float32(qmax * 448)) if a_k > 0 else np.float32(1.0)
    g_v = np.float32(a_v / np.float32(qmax * 448)) if a_v > 0 else np.float32(1.0)
    kc, ks = quantize(kt.reshape(-1, d), g_k, element)
    vc, vs = quantize(vv.reshape(-1, d), g_v, element)
    K = dequantize(kc, ks, g_k, element).reshape(B, T, hkv, d)
    V = dequantize(vc, vs, g_v, element).reshape(B, T, hkv, d)
    q_in = (q[:, T - 1] * np.asarray(s_q, np.float32)[None]).astype(np.float32)       # [B, H_q, d]
    qt = _bf16_round(rope_f32(q_in, np.full(B, T - 1), table)).astype(np.float64)
    scale = 1.0 / np.sqrt(d)
    y = np.stack([[attention_fp64(qt[b, h], K[b, :, h // group], V[b, :, h // group], scale) for h in range(hq)]
                  for b in range(B)])
    return float(np.mean((y - y_ref) ** 2))


def qfit_calibrate(q_pre, k_pre, v, table, grid_s, grid_m, eps=1e-6, element="e2m1"):
    """Algorithm 1 on B calibration sequences ([B, T, heads, d] inputs).
    Returns (s_q [H_q, d], s_k [H_kv, d], m [H_kv, d], errors[grid_s, grid_m]);
    the first grid point (in alpha_s-major order) with the least error wins."""
    hkv = np.asarray(k_pre).shape[2]
    hq = np.asarray(q_pre).shape[2]
    s0_k = qfit_init_scale(k_pre, eps)
    s0_q = np.repeat(s0_k, hq // hkv, axis=0)                      # Replicate to query heads
    mu = qfit_shift_template(k_pre, table)
    y_ref = qfit_reference(q_pre, k_pre, v, table)
    errors = np.full((grid_s, grid_m), np.inf)
    best = None
    for a in range(grid_s):
        alpha_s = a / grid_s
        s_k = (s0_k ** alpha_s).astype(np.float32)
        s_q = (s0_q ** alpha_s).astype(np.float32)
        for b in range(grid_m):
            alpha_m = b / grid_m
            m = (alpha_m * mu).astype(np.float32)
            e = qfit_attention_error(q_pre, k_pre, v, table, s_k, s_q, m, element, y_ref=y_ref)
            errors[a, b] = e
            if best is None or e < best[0]:
                best = (e, s_q, s_k, m)
    return best[1], best[2], best[3], errors
