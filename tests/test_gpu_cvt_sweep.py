"""Hardware-conversion sweep: the quantizer's E4M3 and E2M1 encoders (the
device functions of csrc/nvfp4_quant.cuh, which wrap the hardware
cvt.rn.satfinite conversions) against the oracle's encoders over every
finite fp32 bit pattern.

Both encoders are monotone step functions of the magnitude, so they agree on
all 2^31 non-negative finite patterns exactly when they change code at the
same patterns, to the same codes.  A kernel walks every pattern and reports
each one whose code differs from its predecessor's; the oracle finds its own
change points by bisection over the patterns.  For E2M1 the kernel also
checks every negative finite pattern: its code must be the magnitude's code
with the sign bit (0x8) set, a negative value that rounds to zero included.
"""
import ctypes
import os
import shutil
import subprocess

import numpy as np
import pytest
import torch

from oracle import nvfp4_oracle as O

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2606_15682_gb300", "csrc")
LAST_FINITE = 0x7F7FFFFF
CAP = 1024

SWEEP_CU = r"""
#include <cstdint>
#include "nvfp4_quant.cuh"
using namespace nvfp4;

__device__ __forceinline__ uint32_t e2m1_code(float v) {
  float e[8] = {v, v, v, v, v, v, v, v};
  return e2m1x8(e) & 0xFu;
}
template <bool kE4M3>
__device__ __forceinline__ uint32_t code_of(uint32_t p) {
  const float v = __uint_as_float(p);
  return kE4M3 ? e4m3_rne_sat(v) : e2m1_code(v);
}
// Every p in (0, last] whose code differs from p - 1's: (p, code) pairs.
template <bool kE4M3>
__global__ void change_points(uint32_t last, uint32_t* out, uint32_t* n, uint32_t cap) {
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t q = 1 + blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; q <= last; q += stride) {
    const uint32_t p = static_cast<uint32_t>(q);
    const uint32_t c = code_of<kE4M3>(p);
    if (c != code_of<kE4M3>(p - 1)) {
      const uint32_t i = atomicAdd(n, 1u);
      if (i < cap) { out[2 * i] = p; out[2 * i + 1] = c; }
    }
  }
}
// Negative finite patterns whose E2M1 code is not the magnitude's code | 8.
__global__ void sign_mismatches(uint32_t last, unsigned long long* bad) {
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  unsigned long long local = 0;
  for (uint64_t q = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; q <= last; q += stride) {
    const uint32_t p = static_cast<uint32_t>(q);
    local += e2m1_code(__uint_as_float(p | 0x80000000u)) != (e2m1_code(__uint_as_float(p)) | 8u);
  }
  if (local) atomicAdd(bad, local);
}
extern "C" int sweep(int e4m3, uint32_t last, uint32_t* out_dev, uint32_t* n_dev, uint32_t cap) {
  if (e4m3) change_points<true><<<1216, 256>>>(last, out_dev, n_dev, cap);
  else change_points<false><<<1216, 256>>>(last, out_dev, n_dev, cap);
  return static_cast<int>(cudaDeviceSynchronize());
}
extern "C" int signs(uint32_t last, unsigned long long* bad_dev) {
  sign_mismatches<<<1216, 256>>>(last, bad_dev);
  return static_cast<int>(cudaDeviceSynchronize());
}
"""


@pytest.fixture(scope="module")
def sweep_lib(tmp_path_factory):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d = tmp_path_factory.mktemp("cvt_sweep")
    src = d / "sweep.cu"
    src.write_text(SWEEP_CU)
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    so = d / "libsweep.so"
    r = subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-I", CSRC,
                        "-Xcompiler", "-fPIC", "-shared", "-o", str(so), str(src)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    lib = ctypes.CDLL(str(so))
    lib.sweep.argtypes = [ctypes.c_int, ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint32]
    lib.signs.argtypes = [ctypes.c_uint32, ctypes.c_void_p]
    return lib


def gpu_change_points(lib, e4m3):
    out = torch.zeros(2 * CAP, dtype=torch.int64, device="cuda")  # viewed as uint32 pairs below
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert lib.sweep(int(e4m3), LAST_FINITE, out.data_ptr(), n.data_ptr(), CAP) == 0
    count = int(n.item())
    assert 0 < count <= CAP
    pairs = out.cpu().numpy().view(np.uint32)[: 2 * count].reshape(count, 2).astype(np.int64)
    return pairs[np.argsort(pairs[:, 0])]


def oracle_code(e4m3, p):
    v = np.array([p], dtype=np.uint32).view(np.float32)
    return int(O.e4m3_encode_nonneg(v)[0]) if e4m3 else int(O.e2m1_encode(v)[0])


def oracle_change_points(e4m3):
    """(p, code) where the oracle's code first reaches each larger value, by bisection."""
    top = oracle_code(e4m3, LAST_FINITE)
    points, c_prev = [], oracle_code(e4m3, 0)
    lo = 0
    while c_prev < top:
        hi = LAST_FINITE                                   # smallest p > lo with code(p) != c_prev
        a, b = lo, hi
        while b - a > 1:
            mid = (a + b) // 2
            if oracle_code(e4m3, mid) != c_prev:
                b = mid
            else:
                a = mid
        c = oracle_code(e4m3, b)
        assert c > c_prev, "the oracle encoder must be monotone"
        points.append((b, c))
        lo, c_prev = b, c
    return np.array(points, dtype=np.int64)


@pytest.mark.parametrize("e4m3", [True, False], ids=["e4m3", "e2m1"])
def test_encoder_change_points_match_oracle(sweep_lib, e4m3):
    assert oracle_code(e4m3, 0) == 0
    got = gpu_change_points(sweep_lib, e4m3)
    assert np.all(np.diff(got[:, 1]) > 0), "the device encoder must be monotone in the pattern"
    ref = oracle_change_points(e4m3)
    assert len(got) == len(ref) and np.array_equal(got, ref)
    # E4M3: every code 0x01..0x7E is reached (0x7E = 448 is the saturation value); E2M1: 1..7.
    assert list(got[:, 1]) == list(range(1, 0x7F if e4m3 else 8))


def test_e2m1_sign_of_every_negative_pattern(sweep_lib):
    bad = torch.zeros(1, dtype=torch.int64, device="cuda")
    assert sweep_lib.signs(LAST_FINITE, bad.data_ptr()) == 0
    assert int(bad.item()) == 0
