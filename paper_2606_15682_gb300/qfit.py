"""Q-FIT calibration on the GPU (Algorithm 1).

Chooses the paired pre-RoPE scale (S_Q, S_K) and the post-RoPE key shift m of
Eq. 2 by a grid search over (alpha_s, alpha_m): S = S0^alpha_s with S0 the
pair-shared key magnitudes, m = alpha_m * mu with mu the token mean of the
RoPE'd keys.  Each grid point is scored by the mean squared difference
between a reference attention (unscaled, unshifted, unquantized keys and
values) and the attention over the KV4 cache.  The KV4 side runs in this
library's kernels:
  * kv_append_rope_nvfp4 applies RoPE, subtracts m and quantizes;
  * decode_attention_nvfp4 attends over the quantized cache.
The rest is small tensor arithmetic in PyTorch on the device: the initial
scale, mu, the queries' RoPE, the fp32 reference attention and the error.

Calibration is an offline step.  Its result is applied at inference: S goes
into the query and key projection weights, and m into kv_append_rope_nvfp4's
k_shift.

The readings where the algorithm leaves a choice open are the oracle's:
  * RoPE in fp32 from the (cos, sin) table;
  * the scaled keys rounded to bf16;
  * each query at positions q_pos attends to all T tokens with scale
    1/sqrt(d);
  * a static tensor scale per grid point, amax / (qmax * 448).
"""
from __future__ import annotations

import math

import torch

from . import nvfp4 as N


def _rope(x, positions, table):
    """fp32 RoPE from a (cos, sin) table [n_pos, d/2, 2]: y1 = x1 c - x2 s, y2 = x1 s + x2 c,
    each product and sum a separate fp32 operation.  x [n, ..., d] with one row per position."""
    half = x.shape[-1] // 2
    cs = table[positions]                                   # [n, d/2, 2]
    shape = (x.shape[0],) + (1,) * (x.dim() - 2) + (half,)
    c, s = cs[..., 0].reshape(shape), cs[..., 1].reshape(shape)
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x1 * s + x2 * c], dim=-1)


def qfit_calibrate(q_pre, k_pre, v, rope_table, q_pos, grid_s, grid_m, eps=1e-6, kv_format=N.KV_E2M1):
    """q_pre [T, H_q, d], k_pre and v [T, H_kv, d] (bf16, device, pre-RoPE Q and K);
    rope_table fp32 [>= T, d/2, 2] on the device; q_pos: query positions (long tensor).
    Returns (s_q [H_q, d], s_k [H_kv, d], m [H_kv, d], errors [grid_s, grid_m]) in fp32."""
    dev = k_pre.device
    T, hkv, d = k_pre.shape
    hq = q_pre.shape[1]
    group = hq // hkv
    nq = int(q_pos.numel())
    half = d // 2
    qmax = 6.0 if kv_format == N.KV_E2M1 else 3.5
    pos = torch.arange(T, device=dev)
    kf, vf = k_pre.float(), v.float()

    # Algorithm 1: initial paired scale and its query-head replica, shift template, reference
    a = torch.maximum(kf[..., :half].abs().amax(0), kf[..., half:].abs().amax(0)).clamp_min(eps)
    s0_k = torch.cat([a, a], dim=-1)                        # [H_kv, d]
    s0_q = s0_k.repeat_interleave(group, dim=0)             # [H_q, d]
    k0 = _rope(kf, pos, rope_table)
    mu = k0.double().mean(0).float()
    q0 = _rope(q_pre[q_pos].float(), q_pos, rope_table)
    scale = 1.0 / math.sqrt(d)
    kv_of = torch.arange(hq, device=dev) // group
    logits = torch.einsum("qhd,thd->qht", q0.double(), k0.double()[:, kv_of]) * scale
    y_ref = torch.einsum("qht,thd->qhd", torch.softmax(logits, dim=-1), vf.double()[:, kv_of])

    # One cached sequence per query, each holding all T tokens (decode-form attention).
    cap = T + (T & 1)
    cache = N.KVCache(nq, hkv, cap, 1.0, 1.0, device=dev, kv_format=kv_format)
    cache.seq_lens.fill_(T)
    seq = torch.arange(nq, device=dev, dtype=torch.int32).repeat_interleave(T)
    tok = pos.to(torch.int32).repeat(nq)
    v_rep = v.repeat(nq, 1, 1).contiguous()
    g_v = float(vf.abs().max()) / (qmax * 448)
    out = torch.empty(nq, hq, d, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(N.decode_attention_nvfp4_workspace_size(nq, hq, cap) // 4, dtype=torch.float32, device=dev)
    table_rows = rope_table[:cap] if rope_table.shape[0] >= cap else None
    if table_rows is None:
        raise ValueError("rope_table must cover the cache capacity (T rounded up to even)")
    errors = torch.full((grid_s, grid_m), float("inf"), dtype=torch.float64)
    best = None
    for ia in range(grid_s):
        alpha_s = ia / grid_s
        s_k = (s0_k.double() ** alpha_s).float()
        s_q = (s0_q.double() ** alpha_s).float()
        k_in = (kf / s_k).to(torch.bfloat16)
        kr = _rope(k_in.float(), pos, rope_table)
        qt = _rope(q_pre[q_pos].float() * s_q, q_pos, rope_table).to(torch.bfloat16).contiguous()
        k_rep = k_in.repeat(nq, 1, 1).contiguous()
        for ib in range(grid_m):
            alpha_m = ib / grid_m
            m = (alpha_m * mu).contiguous()
            cache.k_gscale = float((kr - m).abs().max()) / (qmax * 448)
            cache.v_gscale = g_v
            N.kv_append_rope_nvfp4(cache, k_rep, v_rep, seq, tok, table_rows.contiguous(), m)
            N.decode_attention_nvfp4(cache, qt, scale, out, ws)
            e = float(((out.double() - y_ref) ** 2).mean())
            errors[ia, ib] = e
            if best is None or e < best[0]:
                best = (e, s_q.clone(), s_k.clone(), m.clone())
    if N.nvfp4_get_device_status() != 0:
        raise RuntimeError("device status set during calibration")
    return best[1], best[2], best[3], errors
