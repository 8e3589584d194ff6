"""One decode step of a fully quantized (W4A4KV4) transformer layer, chained
through the library's calls, against the same chain in the oracle.

GPU chain (every step a library kernel; RoPE of the queries and the residual
add are small torch glue):
  x -> nvfp4_quantize_dynamic -> nvfp4_linear (qkv)
    -> kv_append_rope_nvfp4 (RoPE on K, quantize, append K and V)
    -> decode_attention_nvfp4_quantize (attention, output as o's NVFP4 input)
    -> nvfp4_linear (o) -> + x -> nvfp4_quantize (static scale)
    -> nvfp4_linear_swiglu_quantize (gate_up, SwiGLU, down's NVFP4 input)
    -> nvfp4_linear (down)
The oracle runs the same steps on its own intermediate results (never the
GPU's).  The static scales of the attention output, of the residual sum and
of the SwiGLU output come from the oracle chain, as a calibration would.

Every single step is pinned bit-exactly or within 2e-3 by the other tests.
Through a chain, each re-quantization flips codes wherever the two chains'
bf16 intermediates straddle a rounding boundary, so the GPU and oracle layer
outputs drift apart by up to the FP4 quantization noise itself (a few per
cent here).  So the chain is judged against the exact layer: the same
computation in fp64 with no quantization at all.  The GPU's W4A4KV4 layer
must be as close to it as the oracle's W4A4KV4 layer is, and the two chains
must agree to well under the distance of unrelated outputs (a wrong layout,
transpose or scale position gives errors of order one)."""
import math

import numpy as np
import pytest
import torch

from _util import f32, lib, u8
from oracle import nvfp4_oracle as O

pytestmark = pytest.mark.gpu

B, H, HQ, HKV, D, I, CAP = 8, 512, 4, 2, 128, 256, 64


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return lib()


def bf16_np(x):
    """fp32 values of the bf16 rounding of x (the oracle's model of a bf16 output)."""
    return O._bf16_round(np.asarray(x, dtype=np.float32))


def quantized_weight(N, w_bf16):
    """Weight quantized once on the GPU (codes, MMA scales, g) and by the oracle."""
    dev = "cuda"
    g = torch.empty(1, dtype=torch.float32, device=dev)
    N.nvfp4_tensor_scale(w_bf16.to(dev), g)
    c = torch.empty(w_bf16.shape[0], w_bf16.shape[1] // 2, dtype=torch.uint8, device=dev)
    s = torch.empty(N.nvfp4_scales_bytes(w_bf16.shape[0], w_bf16.shape[1], 1), dtype=torch.uint8, device=dev)
    N.nvfp4_quantize(w_bf16.to(dev), g, c, s, 1)
    g_ref = O.tensor_scale(f32(w_bf16))
    rc, rs = O.quantize(f32(w_bf16), g_ref)
    return (c, s, g), (rc, rs, g_ref)


def gpu_dynamic(N, x):
    dev = "cuda"
    st = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device=dev)
    g = torch.empty(1, dtype=torch.float32, device=dev)
    c = torch.empty(x.shape[0], x.shape[1] // 2, dtype=torch.uint8, device=dev)
    s = torch.empty(N.nvfp4_scales_bytes(x.shape[0], x.shape[1], 1), dtype=torch.uint8, device=dev)
    N.nvfp4_quantize_dynamic(x, st, g, c, s, 1)
    return c, s, g


def gpu_linear(N, a, w, M, Nn, K):
    out = torch.empty(M, Nn, dtype=torch.bfloat16, device="cuda")
    N.nvfp4_linear(a[0], a[1], a[2], w[0], w[1], w[2], out, M, Nn, K)
    return out


def rope_torch(x, pos, table):
    """fp32 RoPE with the oracle's operation order (one rounding per product and sum)."""
    half = x.shape[-1] // 2
    cs = table[pos]                                   # [n, half, 2]
    c, s = cs[..., 0][:, None, :], cs[..., 1][:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x1 * s + x2 * c], dim=-1)


def test_fully_quantized_decode_layer_step(N):
    dev = "cuda"
    gen = torch.Generator().manual_seed(2606)
    x = torch.randn(B, H, generator=gen).to(torch.bfloat16)
    x[:, 7] *= 20.0                                   # an outlier channel
    w = lambda r, c: (torch.randn(r, c, generator=gen) * 0.04).to(torch.bfloat16)
    Wqkv, Wo, Wg, Wu, Wd = w((HQ + 2 * HKV) * D, H), w(H, HQ * D), w(I, H), w(I, H), w(H, I)
    Wgu = torch.from_numpy(O.interleave_gate_up(Wg.view(torch.int16).numpy(), Wu.view(torch.int16).numpy())).view(
        torch.bfloat16)
    qkv_w, qkv_w_ref = quantized_weight(N, Wqkv)
    o_w, o_w_ref = quantized_weight(N, Wo)
    gu_w, gu_w_ref = quantized_weight(N, Wgu)
    d_w, d_w_ref = quantized_weight(N, Wd)
    wg_ref = O.quantize(f32(Wg), gu_w_ref[2])
    wu_ref = O.quantize(f32(Wu), gu_w_ref[2])

    # Cache prefill: positions 0..len-1 of each sequence from seeded pre-RoPE K and V.
    rng = np.random.default_rng(7)
    lens = rng.integers(5, CAP - 4, B)
    n_pre = int(lens.sum())
    k_pre0 = (torch.randn(n_pre, HKV, D, generator=gen) * 2.0).to(torch.bfloat16)
    v0 = torch.randn(n_pre, HKV, D, generator=gen).to(torch.bfloat16)
    seq0 = np.concatenate([np.full(l, b) for b, l in enumerate(lens)]).astype(np.int64)
    pos0 = np.concatenate([np.arange(l) for l in lens]).astype(np.int64)
    table_ref = O.rope_table(CAP)
    kr = O.rope_f32(f32(k_pre0), pos0, table_ref)
    gk = O.tensor_scale(kr) * np.float32(2.0)         # static scales with headroom for the new tokens
    gv = O.tensor_scale(f32(v0)) * np.float32(2.0)
    cache = N.KVCache(B, HKV, CAP, float(gk), float(gv))
    table = torch.from_numpy(table_ref).to(dev)
    N.kv_append_rope_nvfp4(cache, k_pre0.to(dev), v0.to(dev), torch.as_tensor(seq0, dtype=torch.int32, device=dev),
                           torch.as_tensor(pos0, dtype=torch.int32, device=dev), table)
    rkc, rks, rvc, rvs = (np.zeros((B, HKV, CAP, 64), np.uint8), np.zeros((B, HKV, CAP, 8), np.uint8),
                          np.zeros((B, HKV, CAP, 64), np.uint8), np.zeros((B, HKV, CAP, 8), np.uint8))
    O.kv_append_rope(rkc, rks, rvc, rvs, f32(k_pre0), f32(v0), seq0, pos0, gk, gv, table_ref)
    torch.cuda.synchronize()
    assert np.array_equal(u8(cache.k_codes), rkc) and np.array_equal(u8(cache.v_codes), rvc)

    scale = 1.0 / math.sqrt(D)
    seq_new = np.arange(B)
    # ---------------- oracle chain
    gx = O.tensor_scale(f32(x))
    xc, xs = O.quantize(f32(x), gx)
    qkv_r = bf16_np(O.linear(xc, xs, gx, *qkv_w_ref))
    q_pre_r = qkv_r[:, :HQ * D].reshape(B, HQ, D)
    k_pre_r = qkv_r[:, HQ * D:(HQ + HKV) * D].reshape(B, HKV, D)
    v_r = qkv_r[:, (HQ + HKV) * D:].reshape(B, HKV, D)
    O.kv_append_rope(rkc, rks, rvc, rvs, k_pre_r, v_r, seq_new, lens, gk, gv, table_ref)
    q_r = bf16_np(O.rope_f32(q_pre_r, lens, table_ref))
    o_r = O.decode_attention(q_r, rkc, rks, rvc, rvs, lens + 1, gk, gv, scale).reshape(B, HQ * D)
    g_o = O.tensor_scale(bf16_np(o_r))
    oc_r, os_r = O.quantize(bf16_np(o_r), g_o)
    h_r = bf16_np(f32(x) + bf16_np(O.linear(oc_r, os_r, g_o, *o_w_ref)))
    gh = O.tensor_scale(h_r)
    hc_r, hs_r = O.quantize(h_r, gh)
    act_r, _, _ = O.linear_swiglu_quantize(hc_r, hs_r, gh, wg_ref[0], wg_ref[1], wu_ref[0], wu_ref[1], gu_w_ref[2],
                                           np.float32(1.0))
    g_m = O.tensor_scale(act_r.astype(np.float32))
    _, mc_r, ms_r = O.linear_swiglu_quantize(hc_r, hs_r, gh, wg_ref[0], wg_ref[1], wu_ref[0], wu_ref[1],
                                             gu_w_ref[2], g_m)
    y_r = O.linear(mc_r, ms_r, g_m, *d_w_ref)

    # ---------------- GPU chain
    xd = x.to(dev)
    xq = gpu_dynamic(N, xd)
    qkv = gpu_linear(N, xq, qkv_w, B, (HQ + 2 * HKV) * D, H)
    q_pre = qkv[:, :HQ * D].reshape(B, HQ, D)
    k_pre = qkv[:, HQ * D:(HQ + HKV) * D].reshape(B, HKV, D).contiguous()
    v = qkv[:, (HQ + HKV) * D:].reshape(B, HKV, D).contiguous()
    pos_d = torch.as_tensor(lens, dtype=torch.int32, device=dev)
    N.kv_append_rope_nvfp4(cache, k_pre, v, torch.arange(B, dtype=torch.int32, device=dev), pos_d, table)
    q = rope_torch(q_pre.float(), pos_d.long(), table).to(torch.bfloat16).contiguous()
    cache.seq_lens.copy_(torch.as_tensor(lens + 1, dtype=torch.int32))
    g_o_d = torch.tensor([g_o], dtype=torch.float32, device=dev)
    oc = torch.empty(B, HQ * D // 2, dtype=torch.uint8, device=dev)
    os_ = torch.empty(N.nvfp4_scales_bytes(B, HQ * D, 1), dtype=torch.uint8, device=dev)
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(B, HQ, CAP) // 4, dtype=torch.float32, device=dev)
    N.decode_attention_nvfp4_quantize(cache, q, scale, g_o_d, oc, os_, ws)
    o_proj = gpu_linear(N, (oc, os_, g_o_d), o_w, B, H, HQ * D)
    h = (xd.float() + o_proj.float()).to(torch.bfloat16)
    g_h_d = torch.tensor([gh], dtype=torch.float32, device=dev)
    hq_ = (torch.empty(B, H // 2, dtype=torch.uint8, device=dev),
           torch.empty(N.nvfp4_scales_bytes(B, H, 1), dtype=torch.uint8, device=dev), g_h_d)
    N.nvfp4_quantize(h, g_h_d, hq_[0], hq_[1], 1)
    g_m_d = torch.tensor([g_m], dtype=torch.float32, device=dev)
    mc = torch.empty(B, I // 2, dtype=torch.uint8, device=dev)
    ms = torch.empty(N.nvfp4_scales_bytes(B, I, 1), dtype=torch.uint8, device=dev)
    N.nvfp4_linear_swiglu_quantize(hq_[0], hq_[1], hq_[2], gu_w[0], gu_w[1], gu_w[2], B, I, H, g_m_d, mc, ms)
    y = gpu_linear(N, (mc, ms, g_m_d), d_w, B, H, I)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0

    # ---------------- the exact layer (fp64, nothing quantized)
    xf, group = f32(x).astype(np.float64), HQ // HKV
    qkv_t = xf @ f32(Wqkv).astype(np.float64).T
    q_t = O.rope(qkv_t[:, :HQ * D].reshape(B, HQ, D).transpose(1, 0, 2), lens).transpose(1, 0, 2)
    k_t = O.rope(qkv_t[:, HQ * D:(HQ + HKV) * D].reshape(B, HKV, D).transpose(1, 0, 2), lens).transpose(1, 0, 2)
    v_t = qkv_t[:, (HQ + HKV) * D:].reshape(B, HKV, D)
    k0 = O.rope(f32(k_pre0).astype(np.float64).transpose(1, 0, 2), pos0).transpose(1, 0, 2)
    o_t = np.zeros((B, HQ, D))
    for b in range(B):
        rows = np.nonzero(seq0 == b)[0]
        for hh in range(HQ):
            kv = hh // group
            Kb = np.concatenate([k0[rows, kv], k_t[b, kv][None]])
            Vb = np.concatenate([f32(v0)[rows, kv].astype(np.float64), v_t[b, kv][None]])
            o_t[b, hh] = O.attention_fp64(q_t[b, hh], Kb, Vb, scale)
    h_t = xf + o_t.reshape(B, HQ * D) @ f32(Wo).astype(np.float64).T
    a_t = O.silu(h_t @ f32(Wg).astype(np.float64).T) * (h_t @ f32(Wu).astype(np.float64).T)
    y_t = a_t @ f32(Wd).astype(np.float64).T

    def rel(got, ref):
        return float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
    e_gpu, e_orc, e_chain = rel(f32(y), y_t), rel(y_r, y_t), rel(f32(y), y_r)
    print(f"layer output vs the exact layer: GPU {e_gpu:.3e}, oracle {e_orc:.3e}; GPU vs oracle {e_chain:.3e}")
    assert rel(f32(qkv), qkv_r) < 5e-3                  # one GEMM from identical codes
    assert e_gpu <= 1.25 * e_orc + 5e-3
    assert e_chain < 0.25
