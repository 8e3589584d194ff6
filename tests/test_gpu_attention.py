"""GPU parity of a4 (KV quantize + append, optional Q-FIT shift) and a5 (decode
attention over the NVFP4 cache) against the oracle."""
import math

import numpy as np
import pytest
import torch

from _util import assert_close, f32, lib, u8
from oracle import nvfp4_oracle as O
from paper_2606_15682_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return lib()


def oracle_cache(B, hkv, cap):
    kc = np.zeros((B, hkv, cap, 64), np.uint8); ks = np.zeros((B, hkv, cap, 8), np.uint8)
    return kc, ks, kc.copy(), ks.copy()


def gscale(N, x):
    g = torch.empty(1, dtype=torch.float32, device="cuda")
    N.nvfp4_tensor_scale(x.reshape(-1, x.shape[-1]), g)
    return g.item()


def fill(N, cache, k, v, seq, pos, shift=None):
    N.kv_append_nvfp4(cache, k.cuda(), v.cuda(), torch.as_tensor(seq, dtype=torch.int32, device="cuda"),
                      torch.as_tensor(pos, dtype=torch.int32, device="cuda"),
                      None if shift is None else shift.cuda())


@pytest.mark.parametrize("shifted", [False, True])
def test_kv_append_bit_exact(N, shifted):
    B, hkv, cap, n = 3, 2, 40, 50
    rec = synth.KVRecipe(hkv, seed=77)
    k, v = rec.kv(n, seed=5)
    shift = (f32(k).reshape(n, hkv, 128).mean(axis=0) * 0.7).astype(np.float32) if shifted else None
    kf = f32(k) - (shift if shifted else 0)
    gk, gv = O.tensor_scale(kf.astype(np.float32)), O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    rng = np.random.default_rng(3)
    seq = rng.integers(0, B, n); pos = rng.permutation(B * cap)[:n] % cap
    # unique (seq, pos) pairs so the write order does not matter
    pairs = {}
    for i in range(n):
        pairs[(seq[i], pos[i])] = i
    keep = np.array(sorted(pairs.values()))
    k, v, seq, pos = k[keep], v[keep], seq[keep], pos[keep]
    fill(N, cache, k, v, seq, pos, None if shift is None else torch.from_numpy(shift))
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv), k_shift=shift)
    assert np.array_equal(u8(cache.k_codes), rkc) and np.array_equal(u8(cache.k_scales), rks)
    assert np.array_equal(u8(cache.v_codes), rvc) and np.array_equal(u8(cache.v_scales), rvs)


@pytest.mark.parametrize("rope", [False, True])
@pytest.mark.parametrize("n", [1, 7, 33])
def test_kv_append_odd_row_counts_bit_exact(N, rope, n):
    """One KV head and an odd number of new tokens: the last warp of the
    append has idle lanes, which must neither read past the inputs nor write."""
    B, hkv, cap = 2, 1, 40
    rec = synth.KVRecipe(hkv, seed=13)
    k, v = rec.kv(n, seed=4)
    seq = np.arange(n) % B
    pos = (np.arange(n) // B) * 3 % cap
    table = O.rope_table(cap)
    kq = O.rope_f32(f32(k), pos, table) if rope else f32(k)
    shift = (kq.mean(axis=0) * 0.5).astype(np.float32)
    gk = O.tensor_scale((kq - shift).astype(np.float32))
    gv = O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    args = (k.cuda(), v.cuda(), torch.as_tensor(seq, dtype=torch.int32, device="cuda"),
            torch.as_tensor(pos, dtype=torch.int32, device="cuda"))
    if rope:
        N.kv_append_rope_nvfp4(cache, *args, torch.from_numpy(table).cuda(), torch.from_numpy(shift).cuda())
    else:
        N.kv_append_nvfp4(cache, *args, torch.from_numpy(shift).cuda())
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    if rope:
        O.kv_append_rope(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv), table,
                         k_shift=shift)
    else:
        O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv), k_shift=shift)
    assert np.array_equal(u8(cache.k_codes), rkc) and np.array_equal(u8(cache.k_scales), rks)
    assert np.array_equal(u8(cache.v_codes), rvc) and np.array_equal(u8(cache.v_scales), rvs)


def test_kv_append_out_of_range_sets_capacity_and_skips(N):
    B, hkv, cap = 2, 1, 8
    k = torch.randn(3, hkv, 128).to(torch.bfloat16)
    cache = N.KVCache(B, hkv, cap, 0.01, 0.01)
    N.nvfp4_get_device_status()
    fill(N, cache, k, k, [0, 1, 2], [8, 3, -1])
    assert N.nvfp4_get_device_status() == 7
    assert u8(cache.k_codes)[1, 0, 3].any()
    assert not u8(cache.k_codes)[0].any()


def run_attention(N, cache, q, scale):
    B, hq = q.shape[0], q.shape[1]
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, cache.capacity) // 4, dtype=torch.float32,
                     device="cuda")
    out = torch.full((B, hq, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    N.decode_attention_nvfp4(cache, q.cuda(), scale, out, ws)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("B,hq,hkv,lens", [
    (2, 10, 2, [1, 17]), (3, 40, 8, [1000, 15, 2049]), (1, 8, 8, [300]), (2, 8, 1, [4096, 1023]),
    (2, 6, 2, [0, 33])])
def test_decode_attention(N, B, hq, hkv, lens):
    cap = (max(max(lens), 1) + 6) & ~1  # decode attention needs an even capacity
    rec = synth.KVRecipe(hkv, seed=B * 100 + hq)
    T = sum(lens)
    k, v = rec.kv(max(T, 1), seed=11)
    seq = np.concatenate([np.full(l, b) for b, l in enumerate(lens)]).astype(np.int64)
    pos = np.concatenate([np.arange(l) for l in lens]).astype(np.int64)
    k, v = k[:T], v[:T]
    gk, gv = O.tensor_scale(f32(k)), O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    if T:
        fill(N, cache, k, v, seq, pos)
    cache.seq_lens.copy_(torch.tensor(lens, dtype=torch.int32))
    q = rec.queries(B, hq, seed=12)
    scale = 1.0 / math.sqrt(128)
    out = run_attention(N, cache, q, scale)
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    if T:
        O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv))
    assert np.array_equal(u8(cache.k_codes), rkc) and np.array_equal(u8(cache.v_scales), rvs)
    ref = O.decode_attention(f32(q), rkc, rks, rvc, rvs, lens, gk, gv, scale)
    got = f32(out)
    for b, l in enumerate(lens):
        if l == 0:
            assert not got[b].any(), "an empty sequence must give zeros"
        else:
            assert_close(got[b], ref[b], what=f"seq {b} len {l}")


def test_seq_len_beyond_capacity_is_clamped_and_reported(N):
    B, hq, hkv, cap = 1, 4, 1, 64
    rec = synth.KVRecipe(hkv, seed=3)
    k, v = rec.kv(cap, seed=1)
    gk, gv = O.tensor_scale(f32(k)), O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    fill(N, cache, k, v, np.zeros(cap, np.int64), np.arange(cap))
    cache.seq_lens.fill_(cap + 100)
    q = rec.queries(B, hq, seed=2)
    N.nvfp4_get_device_status()
    out = run_attention(N, cache, q, 0.088)
    assert N.nvfp4_get_device_status() == 7
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), np.zeros(cap, np.int64), np.arange(cap), np.float32(gk), np.float32(gv))
    ref = O.decode_attention(f32(q), rkc, rks, rvc, rvs, [cap], gk, gv, 0.088)
    assert_close(f32(out)[0], ref[0])


def test_decode_batch_kv_append_workload(N):
    """The decode-batch workload's K/V append: 256 new rows x 8 KV heads (one token per sequence)."""
    w = synth.WORKLOADS["qwen14b_decode_linears_m256"]["kv_append"]
    n, hkv = w["n_new"], w["num_kv_heads"]
    rec = synth.KVRecipe(hkv, seed=synth.seed_for("qwen14b_decode_linears_m256", "kv") % (1 << 31), device="cuda")
    k, v = rec.kv(n, seed=21)
    cap = 512
    pos = torch.randint(0, cap, (n,), generator=torch.Generator().manual_seed(2)).numpy()
    gk, gv = O.tensor_scale(f32(k)), O.tensor_scale(f32(v))
    cache = N.KVCache(n, hkv, cap, gk, gv)
    fill(N, cache, k, v, np.arange(n), pos)
    torch.cuda.synchronize()
    rkc, rks, rvc, rvs = oracle_cache(n, hkv, cap)
    O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), np.arange(n), pos, np.float32(gk), np.float32(gv))
    assert np.array_equal(u8(cache.k_codes), rkc) and np.array_equal(u8(cache.k_scales), rks)
    assert np.array_equal(u8(cache.v_codes), rvc) and np.array_equal(u8(cache.v_scales), rvs)


def test_full_size_decode_attention_workload(N):
    """B=64, 40/8 heads, 16384 tokens per sequence, in the bench's launch
    configuration; codes, scales and outputs checked on sampled sequences."""
    wl = "qwen14b_decode_attention_b64_t16384"
    w = synth.WORKLOADS[wl]
    B, hq, hkv, T = w["batch"], w["num_q_heads"], w["num_kv_heads"], w["context"]
    rec = synth.kv_recipe(wl, device="cuda")
    # Static per-layer scales from the amax of all generated K (resp. V).
    k_all = []
    v_all = []
    for b in range(B):
        k, v = rec.kv(T, seed=synth.seed_for(wl, f"kv:{b}") % (1 << 62))
        k_all.append(k); v_all.append(v)
    K = torch.stack(k_all); V = torch.stack(v_all)  # [B, T, hkv, 128]
    gk, gv = gscale(N, K.view(-1, 128)), gscale(N, V.view(-1, 128))
    # The oracle's scales: its own formula on the amax from a library reduction.
    gk_ref = O.tensor_scale(np.array([K.abs().max().float().item()], np.float32))
    gv_ref = O.tensor_scale(np.array([V.abs().max().float().item()], np.float32))
    assert np.float32(gk) == gk_ref and np.float32(gv) == gv_ref
    cache = N.KVCache(B, hkv, T, gk, gv)
    seq = torch.arange(B, dtype=torch.int32, device="cuda").repeat_interleave(T)
    pos = torch.arange(T, dtype=torch.int32, device="cuda").repeat(B)
    N.kv_append_nvfp4(cache, K.view(-1, hkv, 128), V.view(-1, hkv, 128), seq, pos)
    cache.seq_lens.fill_(T)
    q = rec.queries(B, hq, seed=synth.seed_for(wl, "q") % (1 << 62))
    out = run_attention(N, cache, q, 1.0 / math.sqrt(128))
    assert N.nvfp4_get_device_status() == 0
    for b in (0, 37, B - 1):
        kb, vb = f32(K[b]), f32(V[b])
        rkc, rks, rvc, rvs = oracle_cache(1, hkv, T)
        O.kv_append(rkc, rks, rvc, rvs, kb, vb, np.zeros(T, np.int64), np.arange(T), gk_ref, gv_ref)
        assert np.array_equal(u8(cache.k_codes[b:b + 1]), rkc) and np.array_equal(u8(cache.k_scales[b:b + 1]), rks)
        assert np.array_equal(u8(cache.v_codes[b:b + 1]), rvc) and np.array_equal(u8(cache.v_scales[b:b + 1]), rvs)
        ref = O.decode_attention(f32(q[b:b + 1]), rkc, rks, rvc, rvs, [T], gk_ref, gv_ref, 1.0 / math.sqrt(128))
        assert_close(f32(out[b]), ref[0], what=f"seq {b}")


# ------------------------- attention output quantized for the o projection ---

@pytest.mark.parametrize("B,hq,hkv,lens", [(3, 40, 8, [1000, 15, 2049]), (2, 8, 1, [0, 300]), (130, 8, 2, None)])
def test_decode_attention_quantize(N, B, hq, hkv, lens):
    """decode_attention_nvfp4_quantize: codes and scales bit-identical to the
    bf16 attention followed by nvfp4_quantize on the GPU, and to the oracle's
    quantizer applied to that bf16 attention output (the epilogue quantizes the
    attention's own bf16-rounded output); the attention output itself is within
    the attention's tolerance of the fp64 oracle, so the dequantized codes are
    within the quantization error bound plus that tolerance; padding scales
    zero."""
    if lens is None:
        lens = [int(x) for x in np.random.default_rng(B).integers(1, 65, B)]
    cap = (max(max(lens), 1) + 6) & ~1
    rec = synth.KVRecipe(hkv, seed=B * 7 + hq)
    T = sum(lens)
    k, v = rec.kv(max(T, 1), seed=13)
    seq = np.concatenate([np.full(l, b) for b, l in enumerate(lens)]).astype(np.int64)
    pos = np.concatenate([np.arange(l) for l in lens]).astype(np.int64)
    k, v = k[:T], v[:T]
    gk, gv = O.tensor_scale(f32(k)), O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    fill(N, cache, k, v, seq, pos)
    cache.seq_lens.copy_(torch.tensor(lens, dtype=torch.int32))
    q = rec.queries(B, hq, seed=14)
    scale = 1.0 / math.sqrt(128)
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv))
    ref = O.decode_attention(f32(q), rkc, rks, rvc, rvs, lens, gk, gv, scale).reshape(B, hq * 128)
    g_out = O.tensor_scale(ref.astype(np.float32))          # a calibrated static scale, from the oracle
    g_dev = torch.tensor([g_out], dtype=torch.float32, device="cuda")
    cols = hq * 128
    codes = torch.full((B, cols // 2), 0xEE, dtype=torch.uint8, device="cuda")
    scales = torch.full((N.nvfp4_scales_bytes(B, cols, 1),), 0xEE, dtype=torch.uint8, device="cuda")
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, cap) // 4, dtype=torch.float32, device="cuda")
    N.decode_attention_nvfp4_quantize(cache, q.cuda(), scale, g_dev, codes, scales, ws)
    out = run_attention(N, cache, q, scale)
    c2 = torch.empty_like(codes)
    s2 = torch.empty_like(scales)
    N.nvfp4_quantize(out.view(B, cols), g_dev, c2, s2, 1)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    assert torch.equal(codes, c2) and torch.equal(scales, s2), "differs from attention + nvfp4_quantize"
    oc, os_ = O.quantize(f32(out).reshape(B, cols), np.float32(g_out))
    gs = O.scales_from_mma(u8(scales), B, cols)
    assert np.array_equal(u8(codes), oc) and np.array_equal(gs, os_), "differs from the oracle's quantizer"
    for b in range(B):
        assert_close(f32(out).reshape(B, cols)[b], ref[b], what=f"attention output, seq {b}")
    deq = O.dequantize(u8(codes), gs, g_out)
    S = O.e4m3_decode(gs).repeat(16, axis=1)
    tol = 2e-3 * np.abs(ref).max(axis=1, keepdims=True)    # the attention's own tolerance, per sequence
    assert np.all(np.abs(deq - ref) <= 1.5 * S * np.float64(g_out) + tol)
    for b, l in enumerate(lens):
        if l == 0:
            assert not u8(codes)[b].any() and not gs[b].any(), "an empty sequence gives zero codes and scales"
    pad = np.setdiff1d(np.arange(O.mma_scale_bytes(B, cols)), O._mma_offsets(B, cols // 16).ravel())
    assert not u8(scales)[pad].any(), "padding rows of the output scales must be zero"


def test_decode_attention_quantize_invalid_g_out(N):
    B, hq, hkv, cap = 1, 8, 8, 64
    rec = synth.KVRecipe(hkv, seed=5)
    k, v = rec.kv(cap, seed=1)
    cache = N.KVCache(B, hkv, cap, O.tensor_scale(f32(k)), O.tensor_scale(f32(v)))
    fill(N, cache, k, v, np.zeros(cap, np.int64), np.arange(cap))
    cache.seq_lens.fill_(cap)
    q = rec.queries(B, hq, seed=2)
    codes = torch.full((B, hq * 64), 0xEE, dtype=torch.uint8, device="cuda")
    scales = torch.full((N.nvfp4_scales_bytes(B, hq * 128, 1),), 0xEE, dtype=torch.uint8, device="cuda")
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, cap) // 4, dtype=torch.float32, device="cuda")
    N.nvfp4_get_device_status()
    N.decode_attention_nvfp4_quantize(cache, q.cuda(), 0.088, torch.tensor([0.0], device="cuda"), codes, scales, ws)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 1
    assert not u8(codes).any() and not u8(scales).any()


# ----------------------------------- fused RoPE -> shift -> quantize -> append ---

def test_rope_table_matches_numpy(N):
    n_pos = 16384
    t = torch.empty(n_pos, 64, 2, dtype=torch.float32, device="cuda")
    N.nvfp4_rope_table(t, theta=1.0e6)
    torch.cuda.synchronize()
    ref = O.rope_table(n_pos)
    got = t.cpu().numpy()
    # both sides round an fp64 value once to fp32: equal except where the fp64
    # results straddle a rounding boundary (then one fp32 ulp apart)
    diff = np.abs(got.view(np.int32).astype(np.int64) - ref.view(np.int32).astype(np.int64))
    assert diff.max() <= 1 and (diff != 0).mean() < 1e-3, (diff.max(), (diff != 0).mean())


@pytest.mark.parametrize("shifted", [False, True])
def test_kv_append_rope_bit_exact(N, shifted):
    """Codes and scales equal the oracle's RoPE -> shift -> quantize on the same fp32 table."""
    B, hkv, cap, n = 3, 8, 64, 150
    rec = synth.KVRecipe(hkv, seed=91)
    k, v = rec.kv(n, seed=6)                     # bf16 [n, hkv, 128], used here as pre-RoPE keys
    rng = np.random.default_rng(11)
    seq = rng.integers(0, B, n); pos = rng.permutation(B * cap)[:n] % cap
    pairs = {}
    for i in range(n):
        pairs[(seq[i], pos[i])] = i
    keep = np.array(sorted(pairs.values()))
    k, v, seq, pos = k[keep], v[keep], seq[keep], pos[keep]
    table = O.rope_table(cap)
    krot = O.rope_f32(f32(k), pos, table)
    shift = (krot.mean(axis=0) * 0.5).astype(np.float32) if shifted else None
    gk = O.tensor_scale((krot - (shift if shifted else 0)).astype(np.float32))
    gv = O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    N.kv_append_rope_nvfp4(cache, k.cuda(), v.cuda(), torch.as_tensor(seq, dtype=torch.int32, device="cuda"),
                           torch.as_tensor(pos, dtype=torch.int32, device="cuda"), torch.from_numpy(table).cuda(),
                           None if shift is None else torch.from_numpy(shift).cuda())
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append_rope(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv), table,
                     k_shift=shift)
    assert np.array_equal(u8(cache.k_scales), rks) and np.array_equal(u8(cache.k_codes), rkc)
    assert np.array_equal(u8(cache.v_codes), rvc) and np.array_equal(u8(cache.v_scales), rvs)


def test_kv_append_rope_then_attention_matches_fp64(N):
    """End to end: pre-RoPE keys through the fused append, then decode attention,
    against fp64 attention on the oracle's dequantized cache."""
    B, hq, hkv, T = 2, 10, 2, 300
    cap = T + (T & 1)
    rec = synth.KVRecipe(hkv, seed=12)
    table = O.rope_table(cap)
    cache = N.KVCache(B, hkv, cap, 1.0, 1.0)
    ks, vs = [], []
    for b in range(B):
        k, v = rec.kv(T, seed=100 + b)
        ks.append(k); vs.append(v)
    kall = torch.cat(ks); vall = torch.cat(vs)
    seq = np.repeat(np.arange(B), T); pos = np.tile(np.arange(T), B)
    krot = O.rope_f32(f32(kall), pos, table)
    gk, gv = O.tensor_scale(krot), O.tensor_scale(f32(vall))
    cache.k_gscale, cache.v_gscale = float(gk), float(gv)
    N.kv_append_rope_nvfp4(cache, kall.cuda(), vall.cuda(), torch.as_tensor(seq, dtype=torch.int32, device="cuda"),
                           torch.as_tensor(pos, dtype=torch.int32, device="cuda"), torch.from_numpy(table).cuda())
    cache.seq_lens.fill_(T)
    q = rec.queries(B, hq, seed=7)
    out = torch.empty(B, hq, 128, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, cap) // 4, dtype=torch.float32, device="cuda")
    N.decode_attention_nvfp4(cache, q.cuda(), 1 / math.sqrt(128), out, ws)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append_rope(rkc, rks, rvc, rvs, f32(kall), f32(vall), seq, pos, np.float32(gk), np.float32(gv), table)
    ref = O.decode_attention(f32(q), rkc, rks, rvc, rvs, np.full(B, T), np.float32(gk), np.float32(gv),
                             1 / math.sqrt(128))
    for b in range(B):
        assert_close(f32(out)[b], ref[b], what=f"seq {b}")


# ------------------------------------------------------ E1M2 KV elements ---

@pytest.mark.parametrize("rope", [False, True])
def test_kv_append_e1m2_bit_exact(N, rope):
    B, hkv, cap, n = 3, 8, 64, 140
    rec = synth.KVRecipe(hkv, seed=33)
    k, v = rec.kv(n, seed=9)
    rng = np.random.default_rng(17)
    seq = rng.integers(0, B, n); pos = rng.permutation(B * cap)[:n] % cap
    pairs = {}
    for i in range(n):
        pairs[(seq[i], pos[i])] = i
    keep = np.array(sorted(pairs.values()))
    k, v, seq, pos = k[keep], v[keep], seq[keep], pos[keep]
    table = O.rope_table(cap)
    kq = O.rope_f32(f32(k), pos, table) if rope else f32(k)
    shift = (kq.mean(axis=0) * 0.5).astype(np.float32)
    gk = np.float32(np.abs(kq - shift).max() / (3.5 * 448))
    gv = np.float32(np.abs(f32(v)).max() / (3.5 * 448))
    cache = N.KVCache(B, hkv, cap, gk, gv, kv_format=N.KV_E1M2)
    args = (k.cuda(), v.cuda(), torch.as_tensor(seq, dtype=torch.int32, device="cuda"),
            torch.as_tensor(pos, dtype=torch.int32, device="cuda"))
    if rope:
        N.kv_append_rope_nvfp4(cache, *args, torch.from_numpy(table).cuda(), torch.from_numpy(shift).cuda())
    else:
        N.kv_append_nvfp4(cache, *args, torch.from_numpy(shift).cuda())
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    if rope:
        O.kv_append_rope(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, gk, gv, table, k_shift=shift, element="e1m2")
    else:
        O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, gk, gv, k_shift=shift, element="e1m2")
    assert np.array_equal(u8(cache.k_scales), rks) and np.array_equal(u8(cache.k_codes), rkc)
    assert np.array_equal(u8(cache.v_scales), rvs) and np.array_equal(u8(cache.v_codes), rvc)


@pytest.mark.parametrize("B,hq,hkv,lens", [(2, 10, 2, [300, 1030]), (3, 8, 8, [17, 2049, 1])])
def test_decode_attention_e1m2_matches_fp64(N, B, hq, hkv, lens):
    cap = (max(lens) + 6) & ~1
    rec = synth.KVRecipe(hkv, seed=58)
    cache = N.KVCache(B, hkv, cap, 1.0, 1.0, kv_format=N.KV_E1M2)
    ks, vs, seqs, poss = [], [], [], []
    for b, T in enumerate(lens):
        k, v = rec.kv(T, seed=300 + b)
        ks.append(k); vs.append(v); seqs.append(np.full(T, b)); poss.append(np.arange(T))
    kall, vall = torch.cat(ks), torch.cat(vs)
    seq, pos = np.concatenate(seqs), np.concatenate(poss)
    gk = np.float32(np.abs(f32(kall)).max() / (3.5 * 448)); gv = np.float32(np.abs(f32(vall)).max() / (3.5 * 448))
    cache.k_gscale, cache.v_gscale = float(gk), float(gv)
    N.kv_append_nvfp4(cache, kall.cuda(), vall.cuda(), torch.as_tensor(seq, dtype=torch.int32, device="cuda"),
                      torch.as_tensor(pos, dtype=torch.int32, device="cuda"))
    cache.seq_lens.copy_(torch.tensor(lens, dtype=torch.int32))
    q = rec.queries(B, hq, seed=5)
    out = torch.empty(B, hq, 128, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, hq, cap) // 4, dtype=torch.float32, device="cuda")
    N.decode_attention_nvfp4(cache, q.cuda(), 1 / math.sqrt(128), out, ws)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    # the oracle builds its own cache from the same inputs (the append is bit-exact, tested above)
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append(rkc, rks, rvc, rvs, f32(kall), f32(vall), seq, pos, gk, gv, element="e1m2")
    ref = O.decode_attention(f32(q), rkc, rks, rvc, rvs, np.array(lens), gk, gv, 1 / math.sqrt(128),
                             element="e1m2")
    for b in range(B):
        assert_close(f32(out)[b], ref[b], what=f"seq {b}")


# ------------------------------------------------ Q-FIT calibration (Alg. 1) ---

def _qfit_case(B, T, hq, hkv, seed, offset=6.0):
    rng = np.random.default_rng(seed)
    d = 128
    spread = np.exp(rng.standard_normal((hkv, d)))
    k = O._bf16_round((rng.standard_normal((B, T, hkv, d)) * spread + offset).astype(np.float32))
    q = O._bf16_round(rng.standard_normal((B, T, hq, d)).astype(np.float32))
    v = O._bf16_round(rng.standard_normal((B, T, hkv, d)).astype(np.float32))
    return q, k, v


@pytest.mark.parametrize("kv_format", ["e2m1", "e1m2"])
def test_qfit_calibration_matches_oracle_grid(N, kv_format):
    """nvfp4_qfit_calibrate (every step in the library's kernels) against the
    oracle's Algorithm 1: per-point errors close, the same best point, and the
    same transformation."""
    from paper_2606_15682_gb300 import qfit
    B, T, hq, hkv = 4, 255, 8, 2                          # odd T: the cache capacity rounds up
    q, k, v = _qfit_case(B, T, hq, hkv, seed=5)
    table = O.rope_table(T + 1)
    dev = "cuda"
    fmt = N.KV_E2M1 if kv_format == "e2m1" else N.KV_E1M2
    s_q, s_k, m, err = qfit.qfit_calibrate(torch.from_numpy(q).to(dev).to(torch.bfloat16),
                                           torch.from_numpy(k).to(dev).to(torch.bfloat16),
                                           torch.from_numpy(v).to(dev).to(torch.bfloat16),
                                           torch.from_numpy(table).to(dev), grid_s=3, grid_m=3, kv_format=fmt)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    r_sq, r_sk, r_m, r_err = O.qfit_calibrate(q, k, v, table, grid_s=3, grid_m=3, element=kv_format)
    err = err.numpy()
    # the GPU attention multiplies in f16 and rounds its output to bf16, its
    # reference is fp32: small relative differences in each point's error
    assert np.allclose(err, r_err, rtol=0.05, atol=1e-7), (err, r_err)
    assert np.unravel_index(err.argmin(), err.shape) == np.unravel_index(r_err.argmin(), r_err.shape)
    assert np.allclose(s_k.cpu().numpy(), r_sk, rtol=1e-6) and np.allclose(s_q.cpu().numpy(), r_sq, rtol=1e-6)
    assert np.allclose(m.cpu().numpy(), r_m, rtol=1e-5, atol=1e-6)
    assert r_err.min() < r_err[0, 0]            # the calibration improves on no transform


def test_injected_missing_stage_times_out_and_device_stays_usable(N):
    """Failure detection without a GPU fault: the test-only fault knob makes
    CTA 0's producer leave its first ring stage unissued (a barrier that
    nothing completes).  The consumers' bounded wait runs out after ~2 s, the
    call reports NVFP4_ERR_TIMEOUT, and the next call on the same cache is
    exact again."""
    import time
    B, hq, hkv, lens = 2, 10, 2, [300, 257]
    cap = 304
    rec = synth.KVRecipe(hkv, seed=41)
    T = sum(lens)
    k, v = rec.kv(T, seed=42)
    seq = np.concatenate([np.full(l, b) for b, l in enumerate(lens)]).astype(np.int64)
    pos = np.concatenate([np.arange(l) for l in lens]).astype(np.int64)
    gk, gv = O.tensor_scale(f32(k)), O.tensor_scale(f32(v))
    cache = N.KVCache(B, hkv, cap, gk, gv)
    fill(N, cache, k, v, seq, pos)
    cache.seq_lens.copy_(torch.tensor(lens, dtype=torch.int32))
    q = rec.queries(B, hq, seed=43)
    scale = 1.0 / math.sqrt(128)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    N.nvfp4_debug_inject_fault(N.FAULT_ATTN_SKIP_STAGE)
    try:
        t0 = time.time()
        run_attention(N, cache, q, scale)
        waited = time.time() - t0
    finally:
        N.nvfp4_debug_inject_fault(N.FAULT_NONE)
    assert N.nvfp4_get_device_status() == 6
    assert waited > 1.0, "the injected stage must be waited for (bounded) before the kernel gives up"
    out = run_attention(N, cache, q, scale)
    assert N.nvfp4_get_device_status() == 0
    rkc, rks, rvc, rvs = oracle_cache(B, hkv, cap)
    O.kv_append(rkc, rks, rvc, rvs, f32(k), f32(v), seq, pos, np.float32(gk), np.float32(gv))
    ref = O.decode_attention(f32(q), rkc, rks, rvc, rvs, lens, gk, gv, scale)
    for b in range(B):
        assert_close(f32(out)[b], ref[b], what=f"after the injected timeout, seq {b}")
