"""Seeded synthetic inputs shaped like the paper's R1-Distill-Qwen workloads.

The paper's models, calibration text and benchmarks are not available, so every
input is drawn from a fixed-seed generator with the shapes and value
distributions listed in WORKLOADS.  This module only draws numbers: it holds
no quantization or attention arithmetic, and both the CUDA path and the CPU
oracle consume what it produces.

Distributions (per workload):
  activations  N(0, 1); a seeded set of "outlier" channels (columns) is scaled
               by a constant (4 channels x20 for the single linear, 1% of the
               channels x30 elsewhere), as LLM activations have a few large
               channels;
  weights      N(0, 0.02^2);
  K / V        N(0, 1) times a per-(KV head, channel) lognormal factor exp(z),
               z ~ N(0, 1) (channel-wise scale spread), then multiplied by a
               seeded per-KV-head orthogonal 128x128 matrix R (QR of a Gaussian,
               sign-fixed); queries N(0, 1), rotated by the R of their KV head
               so that q.k is preserved.
Everything is rounded once to bf16 at the end.  Generation runs on the device
given (CPU for small cases, the GPU for full-size workloads); the same seed
gives the same values on the same device type.
"""
from __future__ import annotations

import hashlib

import torch

WORKLOADS = {
    # Single NVFP4 W4A4 linear.
    "w4a4_linear_m16_k1536_n1536": dict(
        index=0, M=16, linears={"linear": (1536, 1536)}, outlier_count=4, outlier_mult=20.0),
    # Qwen-1.5B-shaped prefill linears (hidden 1536, 12 q / 2 kv heads, head_dim 128, intermediate 8960).
    "qwen1.5b_prefill_linears_m2048": dict(
        index=1, M=2048, outlier_frac=0.01, outlier_mult=30.0,
        linears={"qkv": (2048, 1536), "o": (1536, 1536), "gate_up": (17920, 1536), "down": (1536, 8960)}),
    # Qwen-14B-shaped decode-batch linears (hidden 5120, 40 q / 8 kv heads, intermediate 13824) + K/V append.
    "qwen14b_decode_linears_m256": dict(
        index=2, M=256, outlier_frac=0.01, outlier_mult=30.0,
        linears={"qkv": (7168, 5120), "o": (5120, 5120), "gate_up": (27648, 5120), "down": (5120, 13824)},
        kv_append=dict(n_new=256, num_kv_heads=8, head_dim=128)),
    # Qwen-14B-shaped decode attention over the NVFP4 KV cache.
    "qwen14b_decode_attention_b64_t16384": dict(
        index=3, batch=64, num_q_heads=40, num_kv_heads=8, head_dim=128, context=16384, lognormal_sigma=1.0),
    # Qwen-32B-shaped full-layer prefill linears (hidden 5120, 64 q / 8 kv heads, intermediate 27648).
    "qwen32b_prefill_linears_m8192": dict(
        index=4, M=8192, outlier_frac=0.01, outlier_mult=30.0,
        linears={"qkv": (10240, 5120), "o": (5120, 8192), "gate_up": (55296, 5120), "down": (5120, 27648)}),
}


def seed_for(workload: str, tensor: str) -> int:
    """Seed of one tensor: 1000 + workload index, mixed with the tensor's name."""
    base = 1000 + WORKLOADS[workload]["index"] if workload in WORKLOADS else 1000
    h = hashlib.sha256(f"{base}:{tensor}".encode()).digest()
    return int.from_bytes(h[:8], "little") & ((1 << 63) - 1)


def _gen(seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def activation(rows, cols, seed, outlier_count=None, outlier_frac=None, outlier_mult=30.0, device="cpu"):
    """bf16 [rows, cols] ~ N(0,1) with seeded outlier channels scaled by outlier_mult."""
    g = _gen(seed, device)
    x = torch.randn(rows, cols, generator=g, device=device, dtype=torch.float32)
    n_out = outlier_count if outlier_count is not None else max(1, round((outlier_frac or 0.0) * cols))
    gc = _gen(seed ^ 0x5A5A5A5A, "cpu")
    idx = torch.randperm(cols, generator=gc)[:n_out].to(device)
    x[:, idx] *= outlier_mult
    return x.to(torch.bfloat16)


def weight(rows, cols, seed, sigma=0.02, device="cpu"):
    """bf16 [rows, cols] ~ N(0, sigma^2) (an nn.Linear weight [out, in])."""
    g = _gen(seed, device)
    return (torch.randn(rows, cols, generator=g, device=device, dtype=torch.float32) * sigma).to(torch.bfloat16)


def linear_inputs(workload, name, M=None, device="cpu"):
    """(activation [M, K], weight [N, K]) of one linear of a workload."""
    w = WORKLOADS[workload]
    N, K = w["linears"][name]
    M = w["M"] if M is None else M
    a = activation(M, K, seed_for(workload, f"act:{name}"), outlier_count=w.get("outlier_count"),
                   outlier_frac=w.get("outlier_frac"), outlier_mult=w["outlier_mult"], device=device)
    W = weight(N, K, seed_for(workload, f"weight:{name}"), device=device)
    return a, W


def orthogonal(n, seed, device="cpu"):
    """Seeded Haar-like orthogonal n x n matrix: QR of a Gaussian with sign-fixed R."""
    g = _gen(seed, "cpu")
    a = torch.randn(n, n, generator=g, dtype=torch.float64)
    q, r = torch.linalg.qr(a)
    q = q * torch.sign(torch.diagonal(r))[None, :]
    return q.to(device)


class KVRecipe:
    """Per-(KV head, channel) lognormal spread and per-KV-head rotations of a workload."""

    def __init__(self, num_kv_heads, head_dim=128, sigma=1.0, seed=1003, device="cpu"):
        self.num_kv_heads, self.head_dim, self.seed, self.device = num_kv_heads, head_dim, seed, device
        g = _gen(seed, "cpu")
        self.k_spread = torch.exp(sigma * torch.randn(num_kv_heads, head_dim, generator=g, dtype=torch.float64))
        self.v_spread = torch.exp(sigma * torch.randn(num_kv_heads, head_dim, generator=g, dtype=torch.float64))
        self.R = torch.stack([orthogonal(head_dim, seed * 131 + h) for h in range(num_kv_heads)])  # [H, d, d]
        self.k_spread = self.k_spread.to(device, torch.float32)
        self.v_spread = self.v_spread.to(device, torch.float32)
        self.R32 = self.R.to(device, torch.float32)

    def kv(self, n_tokens, seed):
        """K, V bf16 [n_tokens, H_kv, d] for one sequence (or batch of rows)."""
        g = _gen(seed, self.device)
        k = torch.randn(n_tokens, self.num_kv_heads, self.head_dim, generator=g, device=self.device) * self.k_spread
        v = torch.randn(n_tokens, self.num_kv_heads, self.head_dim, generator=g, device=self.device) * self.v_spread
        k = torch.einsum("thc,hcd->thd", k, self.R32)
        v = torch.einsum("thc,hcd->thd", v, self.R32)
        return k.to(torch.bfloat16).contiguous(), v.to(torch.bfloat16).contiguous()

    def queries(self, batch, num_q_heads, seed):
        """q bf16 [batch, H_q, d], rotated by the R of each head's KV head (contiguous groups)."""
        g = _gen(seed, self.device)
        q = torch.randn(batch, num_q_heads, self.head_dim, generator=g, device=self.device)
        group = num_q_heads // self.num_kv_heads
        R = self.R32.repeat_interleave(group, dim=0)  # [H_q, d, d]
        return torch.einsum("bhc,hcd->bhd", q, R).to(torch.bfloat16).contiguous()


def kv_recipe(workload="qwen14b_decode_attention_b64_t16384", device="cpu"):
    w = WORKLOADS[workload]
    return KVRecipe(w["num_kv_heads"], w["head_dim"], w["lognormal_sigma"], seed=seed_for(workload, "kv_recipe") % (1 << 31),
                    device=device)
