"""Decode attention without a caller workspace.

decode_attention_nvfp4_static_scratch is for callers that cannot allocate
device memory where they call attention (their runtime reserved all GPU memory
up front, or a host framework owns the allocator).  It keeps the split-KV
partials in a device array that the library holds itself.  This file checks,
through the C ABI, that two calls in a row give the same results as
decode_attention_nvfp4 with a caller workspace, and that problems too large
for the fixed scratch are refused before anything is launched.  Its name makes
pytest collect it last.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

from _util import assert_close, f32, lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return lib()


def _cache(N, B, hkv, T, seed):
    gen = torch.Generator(device="cuda")
    gen.manual_seed(seed)
    cache = N.KVCache(B, hkv, T, 0.013, 0.021)
    for t in (cache.k_codes, cache.v_codes):
        t.copy_(torch.randint(0, 256, t.shape, generator=gen, device="cuda", dtype=torch.int32).to(torch.uint8))
    for t in (cache.k_scales, cache.v_scales):
        t.copy_(torch.randint(0x28, 0x50, t.shape, generator=gen, device="cuda", dtype=torch.int32).to(torch.uint8))
    return cache, gen


def test_static_scratch_matches_workspace_version_twice(N):
    B, hq, hkv, T = 3, 10, 2, 2306
    cache, gen = _cache(N, B, hkv, T, seed=41)
    cache.seq_lens.copy_(torch.tensor([2306, 17, 1500], dtype=torch.int32))
    scale = 1.0 / math.sqrt(128)
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, T) // 4, dtype=torch.float32, device="cuda")
    for call in range(2):  # the scratch keeps the previous call's contents; results must not depend on them
        q = torch.randn(B, hq, 128, generator=gen, device="cuda").to(torch.bfloat16)
        ref = torch.empty(B, hq, 128, dtype=torch.bfloat16, device="cuda")
        got = torch.full((B, hq, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
        N.decode_attention_nvfp4(cache, q, scale, ref, ws)
        N.decode_attention_nvfp4_static_scratch(cache, q, scale, got)
        torch.cuda.synchronize()
        assert N.nvfp4_get_device_status() == 0
        r = f32(ref).astype(np.float64)
        assert np.isfinite(f32(got)).all()
        for b in range(B):
            assert_close(f32(got)[b], r[b], what=f"call {call} seq {b}")


def test_static_scratch_refuses_oversized_problems(N):
    # 64 sequences x 40 heads x 32 splits of 16384-token chunks need ~43 MB of partials > 24 MiB.
    need = N.decode_attention_nvfp4_workspace_size(64, 40, 32768)
    assert need > N.ATTN_STATIC_SCRATCH_BYTES
    s = N.KVCacheStruct(0x10000, 0x10000, 0x10000, 0x10000, 0x10000, 64, 8, 128, 32768, 1.0, 1.0)
    code = N._lib.decode_attention_nvfp4_static_scratch(ctypes.byref(s), ctypes.c_void_p(0x10000), 40,
                                                        ctypes.c_float(0.1), ctypes.c_void_p(0x10000), None)
    assert code == 2  # NVFP4_ERR_SHAPE, nothing launched
