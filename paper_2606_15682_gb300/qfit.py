"""Q-FIT calibration on the GPU (Algorithm 1): a binding of nvfp4_qfit_calibrate.

Chooses the paired pre-RoPE scale (S_Q, S_K) and the post-RoPE key shift m of
Eq. 2 by a grid search over (alpha_s, alpha_m).  Every step runs in the
library (include/nvfp4.h documents the readings: B calibration sequences, the
causal attention scored at each sequence's last token, fp32 RoPE from the
table, bf16 scaled keys and queries, a static KV scale per grid point); this
module only allocates the outputs and the workspace and passes pointers.

Calibration is an offline step.  Its result is applied at inference: S goes
into the query and key projection weights, and m into kv_append_rope_nvfp4's
k_shift.
"""
from __future__ import annotations

import torch

from . import nvfp4 as N


def qfit_calibrate(q_pre, k_pre, v, rope_table, grid_s, grid_m, eps=1e-6, kv_format=N.KV_E2M1, stream=None):
    """q_pre [B, T, H_q, 128], k_pre and v [B, T, H_kv, 128] (bf16, device, pre-RoPE Q and K);
    rope_table fp32 [>= T rounded up to even, 64, 2] on the device.
    Returns (s_q [H_q, 128], s_k [H_kv, 128], m [H_kv, 128]) on the device and the fp64
    errors [grid_s, grid_m] on the host."""
    B, T, hq, d = q_pre.shape
    hkv = k_pre.shape[2]
    dev = k_pre.device
    ws_bytes = N.nvfp4_qfit_workspace_size(B, T, hq, hkv, grid_s, grid_m)
    if ws_bytes == 0:
        raise ValueError("unsupported calibration shape or grid")
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    s_q = torch.empty(hq, d, dtype=torch.float32, device=dev)
    s_k = torch.empty(hkv, d, dtype=torch.float32, device=dev)
    m = torch.empty(hkv, d, dtype=torch.float32, device=dev)
    errors = torch.empty(grid_s * grid_m, dtype=torch.float64)
    N.nvfp4_qfit_calibrate(q_pre, k_pre, v, rope_table, grid_s, grid_m, eps, kv_format, s_q, s_k, m, errors, ws,
                           stream)
    return s_q, s_k, m, errors.view(grid_s, grid_m)
