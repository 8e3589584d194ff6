"""GPU parity of nvfp4_linear_dynamic (a1 + a2 + a3 in one launch for an
activation of at most 32 rows): g_a and the bf16 output must be
bit-identical to nvfp4_quantize_dynamic (MMA scales) followed by
nvfp4_linear, and, on the single W4A4 linear, match the oracle's tensor
scale and fp64 product of its own quantized operands."""
import numpy as np
import pytest
import torch

from _util import assert_close, f32
from oracle import nvfp4_oracle as O
from paper_2606_15682_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from _util import lib
    return lib()


def quantized_weight(N, W):
    g = torch.empty(1, dtype=torch.float32, device="cuda")
    N.nvfp4_tensor_scale(W, g)
    codes = torch.empty(W.shape[0], W.shape[1] // 2, dtype=torch.uint8, device="cuda")
    scales = torch.empty(N.nvfp4_scales_bytes(W.shape[0], W.shape[1], N.SCALES_MMA), dtype=torch.uint8,
                         device="cuda")
    N.nvfp4_quantize(W, g, codes, scales, N.SCALES_MMA)
    return codes, scales, g


def two_call(N, x, wc, wsf, gw, Nn, ldo):
    """The reference path: nvfp4_quantize_dynamic, then nvfp4_linear."""
    M, K = x.shape
    state = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device="cuda")
    ga = torch.empty(1, dtype=torch.float32, device="cuda")
    ac = torch.empty(M, K // 2, dtype=torch.uint8, device="cuda")
    asf = torch.empty(N.nvfp4_scales_bytes(M, K, N.SCALES_MMA), dtype=torch.uint8, device="cuda")
    N.nvfp4_quantize_dynamic(x, state, ga, ac, asf, N.SCALES_MMA)
    out = torch.full((M, ldo), float("nan"), dtype=torch.bfloat16, device="cuda")
    N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K, ldo=ldo)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return out, ga


def fused(N, x, wc, wsf, gw, Nn, ldo, with_g=True):
    M = x.shape[0]
    ga = torch.full((1,), float("nan"), dtype=torch.float32, device="cuda") if with_g else None
    out = torch.full((M, ldo), float("nan"), dtype=torch.bfloat16, device="cuda")
    N.nvfp4_linear_dynamic(x, wc, wsf, gw, out, Nn, ldo=ldo, g_a=ga)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return out, ga


def activation(M, K, seed, ld=None, scale=1.0):
    x = synth.activation(M, K, seed, outlier_count=3, outlier_mult=25.0, device="cuda") * scale
    x = x.to(torch.bfloat16)
    if ld is not None and ld != K:
        buf = torch.full((M, ld), float("nan"), dtype=torch.bfloat16, device="cuda")
        buf[:, :K] = x
        x = buf[:, :K]
    return x


@pytest.mark.parametrize("M,Nn,K", [(1, 16, 256), (16, 1536, 1536), (7, 144, 512), (25, 1024, 1280),
                                    (31, 272, 768), (32, 640, 1536), (32, 128, 256), (32, 5120, 1024),
                                    (2, 1536, 1536),
                                    # more 128-column tiles than SMs: a second round per CTA through
                                    # the double-buffered accumulator and the W ring
                                    (16, 20480, 512), (17, 39936, 256)])
def test_bit_identical_to_two_calls(N, M, Nn, K):
    W = synth.weight(Nn, K, 7 * Nn + K, device="cuda")
    wc, wsf, gw = quantized_weight(N, W)
    x = activation(M, K, 1000 + M * 7 + K)
    ref, ga_ref = two_call(N, x, wc, wsf, gw, Nn, Nn)
    out, ga = fused(N, x, wc, wsf, gw, Nn, Nn)
    assert torch.equal(ga, ga_ref)
    assert torch.equal(out.view(torch.int16), ref.view(torch.int16))


@pytest.mark.parametrize("M,Nn,K,ld_x,ldo", [(16, 1536, 1536, 1544, 1536), (30, 400, 768, 1024, 408),
                                             (32, 256, 1536, 1536, 264)])
def test_padded_rows_and_output_pitch(N, M, Nn, K, ld_x, ldo):
    """Row pitch of x above K, output pitch above N: the padding is neither
    read into the result nor written."""
    W = synth.weight(Nn, K, 3 * Nn + K, device="cuda")
    wc, wsf, gw = quantized_weight(N, W)
    x = activation(M, K, 77 + M, ld=ld_x)
    assert x.stride(0) == ld_x
    ref, ga_ref = two_call(N, x.contiguous(), wc, wsf, gw, Nn, ldo)
    out, ga = fused(N, x, wc, wsf, gw, Nn, ldo, with_g=False)
    assert ga is None
    assert torch.equal(out[:, :Nn].view(torch.int16), ref[:, :Nn].view(torch.int16))
    assert torch.isnan(out[:, Nn:].float()).all()


def test_zero_activation_gives_unit_scale_and_zero_output(N):
    Nn, K = 256, 512
    W = synth.weight(Nn, K, 5, device="cuda")
    wc, wsf, gw = quantized_weight(N, W)
    x = torch.zeros(16, K, dtype=torch.bfloat16, device="cuda")
    out, ga = fused(N, x, wc, wsf, gw, Nn, Nn)
    assert ga.item() == 1.0
    assert (out.float() == 0).all()


def test_tiny_and_huge_magnitudes(N):
    """Activations whose amax sits near the bf16 extremes: the tensor scale and
    the block scales take the same rounding and saturation as the two calls."""
    Nn, K = 384, 768
    W = synth.weight(Nn, K, 9, device="cuda")
    wc, wsf, gw = quantized_weight(N, W)
    for scale in (2.0 ** -120, 2.0 ** 100):
        x = activation(24, K, 31, scale=scale)
        ref, ga_ref = two_call(N, x, wc, wsf, gw, Nn, Nn)
        out, ga = fused(N, x, wc, wsf, gw, Nn, Nn)
        assert torch.equal(ga, ga_ref)
        assert torch.equal(out.view(torch.int16), ref.view(torch.int16))


def test_single_linear_against_oracle(N):
    """The single W4A4 linear (16 x 1536 x 1536) at full size: g_a equals the
    oracle's tensor scale and the output matches the oracle's fp64 product of
    the oracle-quantized operands within the GEMM tolerance."""
    wl = "w4a4_linear_m16_k1536_n1536"
    a, W = synth.linear_inputs(wl, "linear", device="cuda")
    Nn = W.shape[0]
    wc, wsf, gw = quantized_weight(N, W)
    out, ga = fused(N, a, wc, wsf, gw, Nn, Nn)
    g_a, g_w = O.tensor_scale(f32(a)), O.tensor_scale(f32(W))
    assert np.float32(ga.item()) == g_a and np.float32(gw.item()) == g_w
    ra_c, ra_s = O.quantize(f32(a), g_a)
    rw_c, rw_s = O.quantize(f32(W), g_w)
    assert_close(f32(out), O.linear(ra_c, ra_s, g_a, rw_c, rw_s, g_w), what=wl)


def test_unsupported_shapes_are_rejected(N):
    x = torch.zeros(33, 256, dtype=torch.bfloat16, device="cuda")
    wc = torch.zeros(16, 128, dtype=torch.uint8, device="cuda")
    wsf = torch.zeros(N.nvfp4_scales_bytes(16, 256, N.SCALES_MMA), dtype=torch.uint8, device="cuda")
    gw = torch.ones(1, dtype=torch.float32, device="cuda")
    out = torch.zeros(33, 16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(N.NVFP4Error) as e:
        N.nvfp4_linear_dynamic(x, wc, wsf, gw, out, 16)
    assert e.value.code == 4
