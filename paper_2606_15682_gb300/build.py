"""Build libnvfp4.so in-tree with nvcc for sm_103a (GB300).

Each CUDA translation unit is compiled in parallel, then linked into one
shared library under ``paper_2606_15682_gb300/_build``.  Re-running only
recompiles translation units whose sources or headers changed.

``build(debug=True)`` (or ``NVFP4_DEBUG=1`` in the environment) builds the
bounds-checked variant into ``_build_debug``: every computed store index of the
non-TMA kernels is checked against the extent the kernel derives from its
shape arguments, and a violation sets NVFP4_ERR_BOUNDS instead of writing.
The binding loads that variant when ``NVFP4_DEBUG=1``.

``build(timeline=True)`` (or ``NVFP4_TIMELINE=1``) builds a profiling variant
into ``_build_timeline``: the one-launch dynamic quantizer records per-block
globaltimer stamps (entry, loads done, barrier arrival, release, stores
issued), read back with ``nvfp4_timeline_quantize_dynamic`` (that build only).
The binding loads it when ``NVFP4_TIMELINE=1``.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "libnvfp4.so")
BUILD_DEBUG = os.path.join(PKG, "_build_debug")
BUILD_TIMELINE = os.path.join(PKG, "_build_timeline")
SOURCES = ["api.cu", "quantize.cu", "kv_append.cu", "attention.cu", "gemm.cu", "qfit.cu"]
HEADERS = ["common.cuh", "nvfp4_quant.cuh", os.path.join("..", "..", "include", "nvfp4.h")]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden", "-Xptxas", "-v"]


def _nvcc():
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found; the CUDA 13 toolkit is required to build libnvfp4.so")
    return cand


def _digest(src, flags):
    h = hashlib.sha256()
    for p in [src] + [os.path.join(CSRC, x) for x in HEADERS]:
        with open(p, "rb") as f:
            h.update(f.read())
    h.update(" ".join(ARCH + flags).encode())
    return h.hexdigest()[:16]


def _compile(nvcc, name, verbose, build_dir, flags):
    src = os.path.join(CSRC, name)
    obj = os.path.join(build_dir, name.replace(".cu", ".o"))
    stamp = obj + ".sha"
    dig = _digest(src, flags)
    if os.path.exists(obj) and os.path.exists(stamp) and open(stamp).read() == dig:
        return obj, ""
    cmd = [nvcc, *ARCH, *flags, "-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {name}:\n{r.stdout}\n{r.stderr}")
    with open(stamp, "w") as f:
        f.write(dig)
    return obj, (r.stderr if verbose else "")


def _variant(debug, timeline):
    if debug is None:
        debug = os.environ.get("NVFP4_DEBUG") == "1"
    if timeline is None:
        timeline = os.environ.get("NVFP4_TIMELINE") == "1"
    if debug and timeline:
        raise ValueError("the bounds-checked and the timeline builds are separate variants")
    return debug, timeline


def lib_path(debug: bool | None = None, timeline: bool | None = None) -> str:
    debug, timeline = _variant(debug, timeline)
    return os.path.join(BUILD_DEBUG if debug else (BUILD_TIMELINE if timeline else BUILD), "libnvfp4.so")


def build(verbose: bool = False, debug: bool | None = None, timeline: bool | None = None) -> str:
    debug, timeline = _variant(debug, timeline)
    build_dir = BUILD_DEBUG if debug else (BUILD_TIMELINE if timeline else BUILD)
    flags = FLAGS + (["-DNVFP4_DEBUG"] if debug else []) + (["-DNVFP4_TIMELINE"] if timeline else [])
    LIB = lib_path(debug, timeline)
    os.makedirs(build_dir, exist_ok=True)
    nvcc = _nvcc()
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(lambda s: _compile(nvcc, s, verbose, build_dir, flags), SOURCES))
    objs = [o for o, _ in results]
    for _, log in results:
        if log:
            sys.stderr.write(log)
    newest = max(os.path.getmtime(o) for o in objs)
    if not os.path.exists(LIB) or os.path.getmtime(LIB) < newest:
        tmp = LIB + ".tmp"
        # The driver's tensor-map encoder is fetched through the runtime's
        # entry-point query, so libcuda is not a link-time dependency.
        r = subprocess.run([nvcc, *ARCH, "-shared", "-o", tmp, *objs], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, debug=True if "--debug" in sys.argv else None))
