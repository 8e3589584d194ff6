"""Decode attention without a caller workspace.

decode_attention_nvfp4_static_scratch is for callers that cannot allocate
device memory where they call attention (their runtime reserved all GPU memory
up front, or a host framework owns the allocator).  It keeps the split-KV
partials in a device array that the library holds itself.  This file checks,
through the C ABI, that two calls in a row give bit-identical results to
decode_attention_nvfp4 with a caller workspace (the two run the same
arithmetic), that those results match the oracle, and that problems too large
for the fixed scratch are refused before anything is launched.  Its name makes
pytest collect it last.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

from _util import assert_close, f32, lib, u8
from oracle import nvfp4_oracle as O

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
    lens = [2306, 17, 1500]
    cache.seq_lens.copy_(torch.tensor(lens, dtype=torch.int32))
    scale = 1.0 / math.sqrt(128)
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, T) // 4, dtype=torch.float32, device="cuda")
    for call in range(2):  # the scratch keeps the previous call's contents; results must not depend on them
        q = torch.randn(B, hq, 128, generator=gen, device="cuda").to(torch.bfloat16)
        ref = torch.full((B, hq, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
        got = torch.full((B, hq, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
        N.decode_attention_nvfp4(cache, q, scale, ref, ws)
        N.decode_attention_nvfp4_static_scratch(cache, q, scale, got)
        torch.cuda.synchronize()
        assert N.nvfp4_get_device_status() == 0
        assert torch.equal(got, ref), f"call {call}: static-scratch output differs from the workspace version"
        if call == 0:
            r = O.decode_attention(f32(q), u8(cache.k_codes), u8(cache.k_scales), u8(cache.v_codes),
                                   u8(cache.v_scales), lens, np.float32(0.013), np.float32(0.021), scale)
            for b in range(B):
                assert_close(f32(got)[b], r[b], what=f"seq {b} vs oracle")


def test_static_scratch_refuses_oversized_problems(N):
    # 64 sequences x 8 query heads over a 131072-token cache need 32.5 MiB of
    # partials, more than the 24 MiB scratch.  Every buffer is a real device
    # allocation of the declared shape (empty sequences), so the call would
    # stay inside them even if it launched; the refusal must come first.
    B, hkv, hq, T = 64, 1, 8, 131072
    need = N.decode_attention_nvfp4_workspace_size(B, hq, T)
    assert need > N.ATTN_STATIC_SCRATCH_BYTES
    cache = N.KVCache(B, hkv, T, 1.0, 1.0)
    q = torch.zeros(B, hq, 128, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(B, hq, 128, dtype=torch.bfloat16, device="cuda")
    before = N.nvfp4_launch_count()
    s = cache.struct()
    code = N._lib.decode_attention_nvfp4_static_scratch(ctypes.byref(s), ctypes.c_void_p(q.data_ptr()), hq,
                                                        ctypes.c_float(0.1), ctypes.c_void_p(out.data_ptr()), None)
    assert code == 2  # NVFP4_ERR_SHAPE
    assert N.nvfp4_launch_count() == before  # nothing launched
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
