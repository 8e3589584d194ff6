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
