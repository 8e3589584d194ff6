"""Helpers shared by the tests: library loading, tensor conversion, tolerances."""
import os
import re

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "nvfp4.h")

# Output tolerance of the GEMM and attention parity tests: the error of the
# bf16 output beyond its own final rounding (half a bf16 ulp of the output),
# normalised by the largest reference magnitude, must stay below 2e-3.
TOL = 2e-3


def lib():
    """Build (if needed) and import the ctypes binding."""
    from paper_2606_15682_gb300 import build as B
    B.build()
    from paper_2606_15682_gb300 import nvfp4 as N
    return N


def header_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*([a-z_0-9]+)\s*\(", text, flags=re.M)
    return sorted(set(n for n in names if n not in ("if", "while")))


def f32(t):
    """torch tensor (bf16 or other) -> numpy float32, exactly."""
    return t.detach().float().cpu().numpy()


def u8(t):
    return t.detach().cpu().numpy().astype(np.uint8)


def bf16_half_ulp(y):
    ay = np.abs(np.asarray(y, np.float64))
    e = np.floor(np.log2(np.maximum(ay, 2.0 ** -133)))
    return np.ldexp(1.0, (e - 8).astype(np.int64))


def errors(y_bf16, ref):
    """(beyond-rounding normwise error, plain normwise error, relative Frobenius error)."""
    y = np.asarray(y_bf16, np.float64)
    ref = np.asarray(ref, np.float64)
    scale = np.abs(ref).max()
    if scale == 0:
        return float(np.abs(y).max()), float(np.abs(y).max()), 0.0
    diff = np.abs(y - ref)
    beyond = np.maximum(diff - bf16_half_ulp(y), 0.0).max() / scale
    return float(beyond), float(diff.max() / scale), float(np.linalg.norm(y - ref) / np.linalg.norm(ref))


def assert_close(y_bf16, ref, tol=TOL, what=""):
    beyond, plain, fro = errors(y_bf16, ref)
    assert beyond <= tol, f"{what}: error beyond bf16 rounding {beyond:.3e} > {tol} (normwise {plain:.3e}, fro {fro:.3e})"
    return beyond, plain, fro


# ------------------------------------------------------------------------
# Bounded parity for the fused SwiGLU epilogues.  The kernels compute
# h = SiLU(G) U from fp32 accumulators as (G/2 + G/2 tanh(G/2)) U with the
# hardware tanh approximation, then quantize h.  Codes and scales cannot be
# required to equal the oracle's quantization of the exact h, but every one
# must be what the quantizer's recipe gives for some h' within the kernel's
# approximation error of the exact h; nothing else may differ.

# Bound on the error of tanh.approx.f32 relative to |tanh| (documented near
# 2^-11; a factor of two of margin).
TANH_APPROX_REL = 2.0 ** -10


def swiglu_tolerance(G, U, h):
    """Per-element bound on |h_kernel - h_exact|: the tanh approximation,
    |G/2| |dtanh| |U|, plus fp32 accumulation and rounding (2^-14 relative)."""
    G = np.abs(np.asarray(G, np.float64))
    U = np.abs(np.asarray(U, np.float64))
    return 0.5 * G * U * TANH_APPROX_REL + 2.0 ** -14 * (G * U + np.abs(np.asarray(h, np.float64))) + 1e-30


def _e2m1_value_range(v_lo, v_hi):
    from oracle import nvfp4_oracle as O
    return O.e2m1_decode(O.e2m1_encode(v_lo)), O.e2m1_decode(O.e2m1_encode(v_hi))


def assert_nvfp4_within(codes, scales_rm, h, tol, g, what=""):
    """codes uint8 [rows, cols/2], row-major E4M3 scales [rows, cols/16] from a
    kernel that quantized an approximation of h (fp64 [rows, cols]) with the
    static tensor scale g: every scale lies between the recipe's scales of the
    block's smallest and largest possible amax, every code between the codes
    of h -/+ tol under the kernel's own block scale."""
    from oracle import nvfp4_oracle as O
    h = np.asarray(h, np.float64)
    tol = np.asarray(tol, np.float64)
    rows, cols = h.shape
    nb = cols // 16
    g32 = np.float32(g)
    six_g = np.float32(6.0) * g32
    hb, tb = np.abs(h).reshape(rows, nb, 16), tol.reshape(rows, nb, 16)
    amax_lo = np.maximum(hb - tb, 0.0).max(axis=-1)
    amax_hi = (hb + tb).max(axis=-1)
    s_lo = np.nextafter((amax_lo / six_g).astype(np.float32), np.float32(0))
    s_hi = np.nextafter((amax_hi / six_g).astype(np.float32), np.float32(np.inf))
    S_lo = O.e4m3_encode_nonneg(np.maximum(s_lo, 0).astype(np.float64))
    S_hi = O.e4m3_encode_nonneg(s_hi.astype(np.float64))
    gs = np.asarray(scales_rm).astype(np.int64)
    bad = (gs < S_lo) | (gs > S_hi)
    assert not bad.any(), f"{what}: {bad.sum()} block scales outside the recipe's range, e.g. {np.argwhere(bad)[:3]}"
    d = (O.e4m3_decode(gs).astype(np.float32) * g32).astype(np.float32)
    r = np.where(d > 0, np.float32(1.0) / np.where(d > 0, d, 1), 0).astype(np.float64)
    r = np.repeat(r, 16, axis=1)
    lo, hi = _e2m1_value_range((h - tol) * r * (1 - 1e-6), (h + tol) * r * (1 + 1e-6))
    lo, hi = np.minimum(lo, hi), np.maximum(lo, hi)
    got = O.e2m1_decode(O.unpack_codes(codes))
    bad = (got < lo) | (got > hi)
    assert not bad.any(), f"{what}: {bad.sum()} codes outside the range of h -/+ tol, e.g. {np.argwhere(bad)[:3]}"


def assert_mxfp4_within(codes, scales_rm, t, tol_t, what=""):
    """MXFP4 form of assert_nvfp4_within: t (fp64 [rows, cols]) is the tensor
    the kernel approximated (rotated already when it rotates), tol_t its
    per-element bound; E8M0 scales per 32 elements, codes at the kernel's own
    scale 2^e."""
    from oracle import mxfp4_oracle as X
    from oracle import nvfp4_oracle as O
    t = np.asarray(t, np.float64)
    tol_t = np.asarray(tol_t, np.float64)
    rows, cols = t.shape
    nb = cols // 32
    tb, ub = np.abs(t).reshape(rows, nb, 32), tol_t.reshape(rows, nb, 32)
    e_lo = X.shared_exponent(np.maximum(tb - ub, 0.0).max(axis=-1))
    e_hi = X.shared_exponent((tb + ub).max(axis=-1))
    gs = np.asarray(scales_rm).astype(np.int64)
    e = gs - X.E8M0_BIAS
    bad = (e < e_lo) | (e > e_hi)
    assert not bad.any(), f"{what}: {bad.sum()} block scales outside the recipe's range, e.g. {np.argwhere(bad)[:3]}"
    inv = np.repeat(np.ldexp(1.0, -e), 32, axis=1)
    lo, hi = _e2m1_value_range((t - tol_t) * inv, (t + tol_t) * inv)
    lo, hi = np.minimum(lo, hi), np.maximum(lo, hi)
    got = O.e2m1_decode(O.unpack_codes(codes))
    bad = (got < lo) | (got > hi)
    assert not bad.any(), f"{what}: {bad.sum()} codes outside the range of t -/+ tol, e.g. {np.argwhere(bad)[:3]}"


def rotated_tolerance(h, tol):
    """Bound on the error of the fp32 32-point block rotation of an
    approximation of h: the exact rotation spreads each block's element
    bounds as sum(tol) / sqrt(32), and each of the butterflies' five rounded
    levels and the final product adds at most 2^-24 of the block's l1 norm."""
    h = np.abs(np.asarray(h, np.float64))
    rows, cols = h.shape
    tb = np.asarray(tol, np.float64).reshape(rows, cols // 32, 32).sum(axis=-1) / np.sqrt(32.0)
    hb = h.reshape(rows, cols // 32, 32).sum(axis=-1) * 8 * 2.0 ** -24
    return np.repeat(tb + hb, 32, axis=1)
