"""CPU oracle for the MXFP4 format variant -- TEST INFRASTRUCTURE ONLY.

Only the test suite and ``bench.py``'s ``cpu_baseline`` / ``--impl reference``
legs may import this module; the product path never calls it and it imports
nothing from the product package.

MXFP4 (Appendix A, table "Quantization configurations of MXFP4 and NVFP4"):
E2M1 elements, one FP8-E8M0 (exponent-only) block scale per 32 elements and no
global scale.  Sec. 5 evaluates MXFP4 W4A4 deployments, and for MXFP4
configurations applies a block-wise rotation before quantization (Sec. 4,
"Additional implementation details").  The paper gives the format, not the
recipe; the readings used here are:

* shared exponent of a block (the OCP Microscaling rule the paper cites for
  the format): ``e = floor(log2(amax_b)) - 2`` (2 = exponent of E2M1's largest
  power of two, 4), clamped to E8M0's range [-127, 127]; an all-zero block
  takes e = -127.  The block scale is X = 2**e, stored as the E8M0 code e + 127.
* elements: ``code = E2M1_RNE_satfinite(x / X)`` with the sign kept (also for a
  value that rounds to zero), the same element encoder as NVFP4.  x / X is a
  division by a power of two; values in [6, 8) X saturate to 6 X.
* rotation (optional): each 32-element block of a row is multiplied by the
  normalized Sylvester-Hadamard matrix H_32 / sqrt(32) (orthogonal and
  symmetric, so rotating both operands of a linear along K preserves the
  product).  Because the rotated values decide the codes, the oracle computes
  them in the same fp32 arithmetic as the kernel: the fast Walsh-Hadamard
  butterflies (a + b, a - b) at strides 1, 2, 4, 8, 16, each result rounded to
  fp32, then one fp32 multiplication by fp32(1 / sqrt(32)).  ``rotate_blocks``
  is the fp64 definition (the matrix product) that pins it.
* linear: D = A_hat W_hat^T in fp64 on the dequantized operands, as for NVFP4;
  the fused gate_up form h = SiLU(G) * U (fp64), quantized from fp32 h.

Parity status: every function here is pinned by ``tests/test_oracle_pins_mx.py``
(the E8M0 table, closed forms of the shared exponent, exact round trips,
brute force over E2M1 grids, the Hadamard matrix's algebra); none is
"parity unpinned".
"""
from __future__ import annotations

import numpy as np

from oracle.nvfp4_oracle import e2m1_decode, e2m1_encode, scales_to_mma, scales_from_mma, silu, unpack_codes

MX_BLOCK = 32           # elements per E8M0 scale (Appendix A)
E2M1_EMAX = 2           # exponent of E2M1's largest power of two (4 = 2**2)
E8M0_BIAS = 127
E8M0_NAN = 0xFF


def e8m0_decode(code):
    """Value of E8M0 scale codes (exponent only, bias 127): 2**(code - 127), NaN for 0xFF."""
    code = np.asarray(code, dtype=np.int64)
    val = np.ldexp(1.0, code - E8M0_BIAS)
    return np.where(code == E8M0_NAN, np.nan, val)


def shared_exponent(amax):
    """e = floor(log2(amax)) - 2 clamped to [-127, 127]; -127 for amax == 0.

    amax is non-negative and finite; floor(log2) comes from the binary exponent
    (np.frexp is exact), so no logarithm is rounded."""
    amax = np.asarray(amax, dtype=np.float64)
    if np.any(amax < 0) or not np.all(np.isfinite(amax)):
        raise ValueError("amax must be finite and non-negative")
    _, ex = np.frexp(np.where(amax > 0, amax, 1.0))     # amax = f * 2**ex, f in [0.5, 1)
    e = (ex - 1) - E2M1_EMAX
    e = np.where(amax > 0, e, -E8M0_BIAS)
    return np.clip(e, -E8M0_BIAS, E8M0_BIAS).astype(np.int64)


def hadamard(n=MX_BLOCK):
    """Sylvester-Hadamard matrix H_n (entries +-1), n a power of two."""
    h = np.ones((1, 1))
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


def rotate_blocks(x, block=MX_BLOCK):
    """fp64 definition of the block rotation: every `block` consecutive
    elements of a row times H_block / sqrt(block)."""
    x = np.asarray(x, dtype=np.float64)
    rows, cols = x.shape
    if cols % block:
        raise ValueError("cols must be a multiple of the rotation block")
    h = hadamard(block) / np.sqrt(block)
    return (x.reshape(rows, cols // block, block) @ h).reshape(rows, cols)


def rotate_blocks_f32(x_f32):
    """The rotation as the quantizer computes it (fp32): butterflies at
    strides 1, 2, 4, 8, 16 over each 32-element block, every sum and
    difference rounded to fp32, then a multiplication by fp32(1/sqrt(32))."""
    x = np.asarray(x_f32, dtype=np.float32)
    rows, cols = x.shape
    if cols % MX_BLOCK:
        raise ValueError("cols must be a multiple of 32")
    v = x.reshape(rows, cols // MX_BLOCK, MX_BLOCK).copy()
    h = 1
    while h < MX_BLOCK:
        v = v.reshape(rows, cols // MX_BLOCK, MX_BLOCK // (2 * h), 2, h)
        a = v[:, :, :, 0, :].copy()
        b = v[:, :, :, 1, :].copy()
        v[:, :, :, 0, :] = (a + b).astype(np.float32)
        v[:, :, :, 1, :] = (a - b).astype(np.float32)
        v = v.reshape(rows, cols // MX_BLOCK, MX_BLOCK)
        h *= 2
    inv = np.float32(1.0 / np.sqrt(MX_BLOCK))
    return (v * inv).astype(np.float32).reshape(rows, cols)


def quantize_mx(x_f32, rotate=False):
    """MXFP4-quantize a [rows, cols] tensor along its rows (cols % 32 == 0).

    Per block of 32 consecutive elements (after the optional rotation):
      1. amax_b = max |x_i|                                   (exact)
      2. e = floor(log2(amax_b)) - 2, clamped to [-127, 127]  (-127 if amax_b == 0)
      3. code_i = E2M1_RNE_satfinite(x_i / 2**e)             (sign kept)
    Returns (codes uint8 [rows, cols/2], element 2j in the low nibble of byte
    j; scales uint8 [rows, cols/32] holding the E8M0 codes e + 127).
    """
    x = np.asarray(x_f32, dtype=np.float32)
    rows, cols = x.shape
    if cols % MX_BLOCK:
        raise ValueError("cols must be a multiple of 32")
    if rotate:
        x = rotate_blocks_f32(x)
    xb = x.reshape(rows, cols // MX_BLOCK, MX_BLOCK).astype(np.float64)
    amax = np.max(np.abs(xb), axis=2)
    e = shared_exponent(amax)
    v = np.ldexp(xb, -e[:, :, None])                 # exact: a power-of-two scaling in fp64
    codes = e2m1_encode(v).reshape(rows, cols)
    packed = (codes[:, 0::2] | (codes[:, 1::2] << 4)).astype(np.uint8)
    return packed, (e + E8M0_BIAS).astype(np.uint8)


def dequantize_mx(packed, scales):
    """x_hat = e2m1(code) * 2**(S - 127), in fp64 (exact)."""
    vals = e2m1_decode(unpack_codes(packed))
    s = np.repeat(e8m0_decode(scales), MX_BLOCK, axis=-1)
    return vals * s


def mx_scales_to_mma(scales):
    """Row-major [rows, cols/32] E8M0 scales -> the tensor-core byte order the
    library's GEMM reads: the 16-element-block MMA layout of the NVFP4 path,
    with each 32-element block's scale stored for both of its 16-element
    halves."""
    return scales_to_mma(np.repeat(np.asarray(scales, dtype=np.uint8), 2, axis=1))


def mx_scales_from_mma(flat, rows, cols):
    """Inverse of ``mx_scales_to_mma``; raises if the two halves of a block differ."""
    s16 = scales_from_mma(flat, rows, cols)
    if not np.array_equal(s16[:, 0::2], s16[:, 1::2]):
        raise ValueError("MMA-layout MX scales: the halves of a 32-element block differ")
    return s16[:, 0::2]


def linear_mx(a_codes, a_scales, w_codes, w_scales):
    """fp64 reference of the MXFP4 linear: dequantize both operands, multiply."""
    return dequantize_mx(a_codes, a_scales) @ dequantize_mx(w_codes, w_scales).T


def linear_mx_rows(a_codes, a_scales, w_codes, w_scales, rows):
    """The reference restricted to some output rows (full-size sampled checks)."""
    rows = np.asarray(rows)
    return dequantize_mx(a_codes[rows], a_scales[rows]) @ dequantize_mx(w_codes, w_scales).T


def linear_swiglu_quantize_mx(a_codes, a_scales, wg_codes, wg_scales, wu_codes, wu_scales, rotate=False, rows=None):
    """The down projection's input from MXFP4 operands: h = SiLU(A W_gate^T) *
    (A W_up^T) in fp64, then MXFP4-quantized (``quantize_mx``, optionally after
    the block rotation) from h rounded to fp32.  ``rows`` restricts to some
    rows of A.  Returns (h fp64, codes, scales)."""
    if rows is not None:
        a_codes, a_scales = a_codes[np.asarray(rows)], a_scales[np.asarray(rows)]
    G = linear_mx(a_codes, a_scales, wg_codes, wg_scales)
    U = linear_mx(a_codes, a_scales, wu_codes, wu_scales)
    h = silu(G) * U
    codes, scales = quantize_mx(h.astype(np.float32), rotate=rotate)
    return h, codes, scales
