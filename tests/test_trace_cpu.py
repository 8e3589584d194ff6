"""Host-only check of the library's tracing: every C-ABI call opens an NVTX
range named after itself and closes it on return.  A tiny NVTX injection
library (the same mechanism a profiler uses to attach) records the pushes and
pops; the calls exercised here fail argument validation before any CUDA call,
so no GPU is needed."""
import os
import shutil
import subprocess
import sys
import textwrap

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

INJECTION_C = r"""
#include <stdio.h>
#include <stdlib.h>
#include <nvtx3/nvToolsExt.h>

static FILE* out;
static int on_push(const char* name) { fprintf(out, "push %s\n", name); fflush(out); return 0; }
static int on_pop(void) { fprintf(out, "pop\n"); fflush(out); return 0; }

int InitializeInjectionNvtx2(NvtxGetExportTableFunc_t get_table) {
  const NvtxExportTableCallbacks* cb = (const NvtxExportTableCallbacks*)get_table(NVTX_ETID_CALLBACKS);
  NvtxFunctionTable table = 0;
  unsigned int size = 0;
  if (!cb || !cb->GetModuleFunctionTable(NVTX_CB_MODULE_CORE, &table, &size)) return 0;
  if (size <= NVTX_CBID_CORE_RangePop) return 0;
  out = fopen(getenv("NVFP4_TRACE_LOG"), "w");
  if (!out) return 0;
  *table[NVTX_CBID_CORE_RangePushA] = (NvtxFunctionPointer)on_push;
  *table[NVTX_CBID_CORE_RangePop] = (NvtxFunctionPointer)on_pop;
  return 1;
}
"""

CALLS = textwrap.dedent("""
    import ctypes, sys
    sys.path.insert(0, {root!r})
    from paper_2606_15682_gb300 import nvfp4 as N
    L = N._lib
    p, s = ctypes.c_void_p(0x10000), ctypes.c_void_p(0)
    assert L.nvfp4_linear(None, p, p, p, p, p, 128, 128, 256, p, 128, s) == 1
    assert L.mxfp4_quantize(None, 0, 64, 64, 0, None, None, 1, s) == 0
    assert L.nvfp4_quantize(p, 4, 40, 40, p, p, p, 0, s) == 2
    assert L.mxfp4_linear_swiglu_quantize(p, p, p, p, 256, 192, 512, 0, p, p, s) == 2
""")


def _cuda_include():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(nvcc))), "include")
    return inc if os.path.isfile(os.path.join(inc, "nvtx3", "nvToolsExt.h")) else None


def test_each_abi_call_is_an_nvtx_range(tmp_path):
    from _util import lib
    lib()  # build the library in-tree if needed
    inc = _cuda_include()
    gcc = shutil.which("gcc")
    if inc is None or gcc is None:
        pytest.skip("needs gcc and the CUDA toolkit's NVTX headers")
    src = tmp_path / "inject.c"
    src.write_text(INJECTION_C)
    so = tmp_path / "libinject.so"
    r = subprocess.run([gcc, "-shared", "-fPIC", "-O1", "-I", inc, "-o", str(so), str(src)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    log = tmp_path / "trace.log"
    env = dict(os.environ, NVTX_INJECTION64_PATH=str(so), NVFP4_TRACE_LOG=str(log))
    r = subprocess.run([sys.executable, "-c", CALLS.format(root=ROOT)], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr
    events = log.read_text().split("\n")
    events = [e for e in events if e]
    assert events == ["push nvfp4_linear", "pop", "push mxfp4_quantize", "pop", "push nvfp4_quantize", "pop",
                      "push mxfp4_linear_swiglu_quantize", "pop"], events
