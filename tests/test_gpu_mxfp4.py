"""GPU parity of the MXFP4 format variant: the quantizer (with and without the
32-element block rotation) bit-exact against the CPU oracle, and the MXFP4
linear against the oracle's fp64 product of identical dequantized operands."""
import numpy as np
import pytest
import torch

from _util import assert_close, assert_mxfp4_within, f32, lib, rotated_tolerance, swiglu_tolerance, u8
from oracle import mxfp4_oracle as X
from oracle import nvfp4_oracle as O
from paper_2606_15682_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return lib()


def gpu_mx_quantize(N, x, layout, rotate):
    rows, cols = x.shape
    codes = torch.full((rows, cols // 2), 0xEE, dtype=torch.uint8, device="cuda")
    scales = torch.full((N.mxfp4_scales_bytes(rows, cols, layout),), 0xEE, dtype=torch.uint8, device="cuda")
    N.mxfp4_quantize(x, codes, scales, layout=layout, rotate=rotate)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return codes, scales


def check_mx_quantize(N, x_bf16, layout, rotate, rows_sample=None, ld=None):
    rows, cols = x_bf16.shape
    if ld is None:
        x = x_bf16.cuda()
    else:
        buf = torch.zeros(rows, ld, dtype=torch.bfloat16, device="cuda")
        buf[:, :cols] = x_bf16.cuda()
        x = buf[:, :cols]
    codes, scales = gpu_mx_quantize(N, x, layout, rotate)
    sel = np.arange(rows) if rows_sample is None else np.asarray(rows_sample)
    assert sel.min() >= 0 and sel.max() < rows
    rc, rs = X.quantize_mx(f32(x_bf16[torch.as_tensor(sel)]), rotate=rotate)
    gc = u8(codes)[sel]
    gs = u8(scales)
    gs = gs.reshape(rows, cols // 32)[sel] if layout == 0 else X.mx_scales_from_mma(gs, rows, cols)[sel]
    bad = np.argwhere(gc != rc)
    assert bad.size == 0, f"{len(bad)} code bytes differ, first at {bad[:3].tolist()}"
    assert np.array_equal(gs, rs)
    if layout == 1 and rows % 128:
        pad = np.setdiff1d(np.arange(O.mma_scale_bytes(rows, cols)), O._mma_offsets(rows, cols // 16).ravel())
        assert not u8(scales)[pad].any(), "padding rows of the MMA scale layout must be zero"
    return codes, scales


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
@pytest.mark.parametrize("layout", [0, 1], ids=["rowmajor", "mma"])
@pytest.mark.parametrize("rows,cols", [(1, 64), (130, 256), (257, 1536), (64, 8960)])
def test_mx_quantize_matches_oracle(N, rows, cols, layout, rotate):
    x = synth.activation(rows, cols, 7000 + rows + cols, outlier_frac=0.01)
    check_mx_quantize(N, x, layout, rotate)


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
def test_mx_quantize_padded_rows_and_rowmajor_32(N, rotate):
    x = synth.activation(33, 96, 7101, outlier_frac=0.05)
    check_mx_quantize(N, x, 0, rotate, ld=136)          # cols % 64 != 0: row-major only; padded leading dim
    x = synth.activation(200, 512, 7102, outlier_frac=0.02)
    check_mx_quantize(N, x, 1, rotate, ld=520)


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
def test_mx_quantize_edge_values(N, rotate):
    """Zero blocks, signed zeros, bf16 subnormals, huge and tiny magnitudes,
    exact E2M1 grid values and ties, saturation between 6 and 8 scales."""
    g = torch.Generator().manual_seed(7200)
    x = torch.randn(16, 256, generator=g)
    x[0] = 0.0
    x[1] = -0.0
    x[2] = torch.randn(256, generator=g) * 1e-39            # bf16 subnormals
    x[3] = torch.randn(256, generator=g) * 1e36            # large, and a rotated block sum stays finite
    x[4, :32] = torch.tensor([6.0, 0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0] * 4)
    x[5, :32] = torch.tensor([7.5, -7.9, 1.0, -0.0] * 8)
    x[6] = torch.randn(256, generator=g) * 1e-38
    x[6, ::32] = 1e-37                                     # amax near the bottom of E8M0's range
    x[7, :32] = 2.0 ** -127
    x[8, ::2] = 0.0
    x = x.to(torch.bfloat16)
    for layout in (0, 1):
        check_mx_quantize(N, x, layout, rotate)


def test_mx_quantize_full_size_sampled(N):
    """The 32B prefill down projection's input (8192 x 27648), in the launch
    configuration of the bench: sampled rows against the oracle."""
    M, K = 8192, 27648
    x = synth.activation(M, K, 7300, outlier_frac=0.01, device="cuda")
    rows = np.unique(np.r_[0:16, 4096:4112, M - 16:M])
    for rotate in (False, True):
        codes, scales = gpu_mx_quantize(N, x, 1, rotate)
        rc, rs = X.quantize_mx(f32(x[torch.as_tensor(rows, device="cuda")]), rotate=rotate)
        assert np.array_equal(u8(codes[torch.as_tensor(rows, device="cuda")]), rc)
        assert np.array_equal(X.mx_scales_from_mma(u8(scales), M, K)[rows], rs)


def test_mx_quantize_empty_is_noop(N):
    x = torch.empty(0, 64, dtype=torch.bfloat16, device="cuda")
    N.mxfp4_quantize(x, None, None)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0


def run_mx_linear(N, a_codes, a_scales_rm, w_codes, w_scales_rm, M, Nn, K, ldo=None):
    dev = "cuda"
    ac = torch.from_numpy(a_codes).to(dev)
    wc = torch.from_numpy(w_codes).to(dev)
    asf = torch.from_numpy(X.mx_scales_to_mma(a_scales_rm)).to(dev)
    wsf = torch.from_numpy(X.mx_scales_to_mma(w_scales_rm)).to(dev)
    ldo = Nn if ldo is None else ldo
    out = torch.full((M, ldo), float("nan"), dtype=torch.bfloat16, device=dev)
    N.mxfp4_linear(ac, asf, wc, wsf, out, M, Nn, K, ldo=ldo)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return out


@pytest.mark.parametrize("M,Nn,K", [(128, 128, 256), (1, 16, 256), (130, 144, 512), (257, 384, 1024),
                                    # N % 256 == 0: 256 x 256 CTA-pair tiles (enough of them)
                                    (2048, 1280, 1024),
                                    # more pair tiles than pairs with 6 k-blocks: the W-resident form
                                    (2048, 2560, 1536),
                                    # too few pair tiles with a long K: split-K clusters (S = 4, 2)
                                    (256, 768, 4096), (200, 7168, 4608)])
def test_mx_linear_random_operands(N, M, Nn, K):
    """Seeded random codes and E8M0 scales (isolates the GEMM from the quantizer)."""
    gen = torch.Generator().manual_seed(7400 + M + Nn + K)
    ac = torch.randint(0, 256, (M, K // 2), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    wc = torch.randint(0, 256, (Nn, K // 2), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    asf = torch.randint(118, 134, (M, K // 32), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    wsf = torch.randint(110, 126, (Nn, K // 32), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    out = run_mx_linear(N, ac, asf, wc, wsf, M, Nn, K)
    assert_close(f32(out), X.linear_mx(ac, asf, wc, wsf), what=f"mxfp4 linear {M}x{Nn}x{K}")


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
def test_mx_linear_on_workload_operands(N, rotate):
    """The 1.5B prefill qkv shape (2048 x 2048 x 1536) from bf16 activations and
    weights quantized by the oracle (rotated along K on both sides when asked):
    the GPU product matches the oracle's, and with the rotation both stay as
    close to the unquantized product as the oracle's pipeline is."""
    a, w = synth.linear_inputs("qwen1.5b_prefill_linears_m2048", "qkv")
    ac, asf = X.quantize_mx(f32(a), rotate=rotate)
    wc, wsf = X.quantize_mx(f32(w), rotate=rotate)
    M, K = a.shape
    Nn = w.shape[0]
    out = run_mx_linear(N, ac, asf, wc, wsf, M, Nn, K)
    ref = X.linear_mx(ac, asf, wc, wsf)
    assert_close(f32(out), ref, what="mxfp4 qkv")
    exact = f32(a).astype(np.float64) @ f32(w).astype(np.float64).T
    e_orc = np.abs(ref - exact).max() / np.abs(exact).max()
    e_gpu = np.abs(f32(out) - exact).max() / np.abs(exact).max()
    assert e_gpu <= 1.05 * e_orc + 4e-3


def test_mx_linear_padded_output(N):
    gen = torch.Generator().manual_seed(7500)
    M, Nn, K = 130, 144, 512
    ac = torch.randint(0, 256, (M, K // 2), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    wc = torch.randint(0, 256, (Nn, K // 2), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    asf = torch.randint(120, 130, (M, K // 32), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    wsf = torch.randint(120, 130, (Nn, K // 32), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    out = run_mx_linear(N, ac, asf, wc, wsf, M, Nn, K, ldo=168)
    assert_close(f32(out[:, :Nn]), X.linear_mx(ac, asf, wc, wsf), what="mxfp4 padded ldo")
    assert torch.isnan(out[:, Nn:].float()).all(), "columns beyond N must be left untouched"


def mx_random_operand(rows, K, gen, lo, hi):
    codes = torch.randint(0, 256, (rows, K // 2), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    scales = torch.randint(lo, hi, (rows, K // 32), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    return codes, scales


def mx_swiglu_case(N, M, I, K, seed, rotate, rows=None):
    gen = torch.Generator().manual_seed(seed)
    a_c, a_s = mx_random_operand(M, K, gen, 121, 129)
    wg_c, wg_s = mx_random_operand(I, K, gen, 116, 122)
    wu_c, wu_s = mx_random_operand(I, K, gen, 116, 122)
    rows = np.arange(M) if rows is None else np.asarray(rows)
    h, rc, rs = X.linear_swiglu_quantize_mx(a_c, a_s, wg_c, wg_s, wu_c, wu_s, rotate=rotate, rows=rows)
    G = X.linear_mx_rows(a_c, a_s, wg_c, wg_s, rows)
    U = X.linear_mx_rows(a_c, a_s, wu_c, wu_s, rows)
    tol = swiglu_tolerance(G, U, h)
    w_c = O.interleave_gate_up(wg_c, wu_c)
    w_s = O.interleave_gate_up(wg_s, wu_s)
    dev = "cuda"
    out_c = torch.full((M, I // 2), 0xEE, dtype=torch.uint8, device=dev)
    out_s = torch.full((N.mxfp4_scales_bytes(M, I, 1),), 0xEE, dtype=torch.uint8, device=dev)
    N.mxfp4_linear_swiglu_quantize(torch.from_numpy(a_c).to(dev), torch.from_numpy(X.mx_scales_to_mma(a_s)).to(dev),
                                   torch.from_numpy(w_c).to(dev), torch.from_numpy(X.mx_scales_to_mma(w_s)).to(dev),
                                   M, I, K, out_c, out_s, rotate=rotate)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return h, rc, rs, rows, u8(out_c), u8(out_s), tol


def check_mx_swiglu(h, rc, rs, rows, out_c, out_s, M, I, rotate, tol):
    """The kernel's SiLU uses the hardware tanh approximation: every E8M0 scale
    and code must be one the recipe gives for some h' within that
    approximation's error of the exact fp64 h (rotated by the exact
    H_32 / sqrt(32) when asked, the bound spread by the rotation); no other
    difference is allowed.  Most equal the oracle's; padding scales are zero."""
    gs = X.mx_scales_from_mma(out_s, M, I)[rows]
    target = X.rotate_blocks(h) if rotate else h
    tol_t = rotated_tolerance(h, tol) if rotate else tol
    assert_mxfp4_within(out_c[rows], gs, target, tol_t, what=f"mx swiglu rotate={rotate}")
    assert (gs == rs).mean() > 0.99 and (out_c[rows] == rc).mean() > 0.99
    pad = np.setdiff1d(np.arange(O.mma_scale_bytes(M, I)), O._mma_offsets(M, I // 16).ravel())
    assert not out_s[pad].any(), "padding rows of the output scales must be zero"


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
@pytest.mark.parametrize("M,I,K", [(256, 128, 256), (129, 384, 512), (640, 512, 768)])
def test_mx_linear_swiglu_quantize(N, M, I, K, rotate):
    h, rc, rs, rows, out_c, out_s, tol = mx_swiglu_case(N, M, I, K, seed=M + I + K + rotate, rotate=rotate)
    check_mx_swiglu(h, rc, rs, rows, out_c, out_s, M, I, rotate, tol)


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
def test_mx_linear_swiglu_quantize_prefill_shape_then_down(N, rotate):
    """The 1.5B-prefill MLP shape (M=2048, I=8960, K=1536; the W-resident form)
    on sampled rows, then fed to the MXFP4 down projection as its A operand."""
    M, I, K, Hd = 2048, 8960, 1536, 1536
    rows = np.sort(np.r_[np.random.default_rng(3).choice(M - 1, 40, replace=False), M - 1])
    h, rc, rs, rows, out_c, out_s, tol = mx_swiglu_case(N, M, I, K, seed=123 + rotate, rotate=rotate, rows=rows)
    check_mx_swiglu(h, rc, rs, rows, out_c, out_s, M, I, rotate, tol)
    gen = torch.Generator().manual_seed(8)
    wd_c, wd_s = mx_random_operand(Hd, I, gen, 116, 122)
    out = torch.empty(M, Hd, dtype=torch.bfloat16, device="cuda")
    N.mxfp4_linear(torch.from_numpy(out_c).cuda(), torch.from_numpy(out_s).cuda(), torch.from_numpy(wd_c).cuda(),
                   torch.from_numpy(X.mx_scales_to_mma(wd_s)).cuda(), out, M, Hd, I)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    ref = X.linear_mx_rows(out_c, X.mx_scales_from_mma(out_s, M, I), wd_c, wd_s, rows)
    assert_close(f32(out[torch.as_tensor(rows, device="cuda")]), ref, what="mx down(swiglu)")


@pytest.mark.parametrize("rotate", [False, True], ids=["plain", "rotated"])
def test_mx_mlp_chain_tracks_the_exact_mlp(N, rotate):
    """x -> mxfp4_quantize -> fused gate_up (SwiGLU + MXFP4 h) -> mxfp4_linear
    against W_down, with every operand rotated along its K when asked: the GPU
    chain is as close to the exact fp64 MLP as the oracle's chain is (the
    rotation preserves each product only if both operands are rotated)."""
    M, H, I = 256, 1536, 1024
    dev = "cuda"
    x = synth.activation(M, H, 7600, outlier_frac=0.01)
    wg, wu = synth.weight(I, H, 7601), synth.weight(I, H, 7602)
    wd = synth.weight(H, I, 7603)
    exact_h = O.silu(f32(x).astype(np.float64) @ f32(wg).astype(np.float64).T) * (
        f32(x).astype(np.float64) @ f32(wu).astype(np.float64).T)
    exact = exact_h @ f32(wd).astype(np.float64).T

    def q(t):
        c = torch.empty(t.shape[0], t.shape[1] // 2, dtype=torch.uint8, device=dev)
        s = torch.empty(N.mxfp4_scales_bytes(t.shape[0], t.shape[1], 1), dtype=torch.uint8, device=dev)
        N.mxfp4_quantize(t.to(dev).contiguous(), c, s, 1, rotate=rotate)
        return c, s
    wi = torch.empty(2 * I, H, dtype=torch.bfloat16, device=dev)
    N.nvfp4_interleave_gate_up(wg.to(dev), wu.to(dev), wi)
    (xc, xs), (wc, ws), (dc, ds) = q(x), q(wi), q(wd)
    hc = torch.empty(M, I // 2, dtype=torch.uint8, device=dev)
    hs = torch.empty(N.mxfp4_scales_bytes(M, I, 1), dtype=torch.uint8, device=dev)
    N.mxfp4_linear_swiglu_quantize(xc, xs, wc, ws, M, I, H, hc, hs, rotate=rotate)
    y = torch.empty(M, H, dtype=torch.bfloat16, device=dev)
    N.mxfp4_linear(hc, hs, dc, ds, y, M, H, I)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0

    oc, os_ = X.quantize_mx(f32(x), rotate=rotate)
    gc, gs = X.quantize_mx(f32(wg), rotate=rotate)
    uc, us = X.quantize_mx(f32(wu), rotate=rotate)
    odc, ods = X.quantize_mx(f32(wd), rotate=rotate)
    _, ohc, ohs = X.linear_swiglu_quantize_mx(oc, os_, gc, gs, uc, us, rotate=rotate)
    y_orc = X.linear_mx(ohc, ohs, odc, ods)
    scale = np.abs(exact).max()
    e_orc = np.abs(y_orc - exact).max() / scale
    e_gpu = np.abs(f32(y).astype(np.float64) - exact).max() / scale
    print(f"MXFP4 MLP ({'rotated' if rotate else 'plain'}): GPU {e_gpu:.3e}, oracle {e_orc:.3e}")
    assert e_orc < 0.5
    assert e_gpu <= 1.25 * e_orc + 5e-3


WL = [w for w in synth.WORKLOADS if "linears" in synth.WORKLOADS[w]]


@pytest.mark.parametrize("workload", WL)
def test_mx_workload_linears(N, workload):
    """Every linear of every workload at full size in the MXFP4 W4A4 launch
    configuration the bench times (activation and weight rotated and
    quantized on the GPU, then mxfp4_linear), on seeded samples of output
    rows and columns; the sampled operands' codes and scales are bit-exact."""
    dev = "cuda"
    for name, (Nn, K) in synth.WORKLOADS[workload]["linears"].items():
        a, W = synth.linear_inputs(workload, name, device=dev)
        M = a.shape[0]
        ac, asf = gpu_mx_quantize(N, a, 1, True)
        wc, wsf = gpu_mx_quantize(N, W, 1, True)
        out = torch.empty(M, Nn, dtype=torch.bfloat16, device=dev)
        N.mxfp4_linear(ac, asf, wc, wsf, out, M, Nn, K)
        torch.cuda.synchronize()
        assert N.nvfp4_get_device_status() == 0
        rng = np.random.default_rng(2)
        rows = np.arange(M) if M * K <= 2048 * 8960 else np.sort(np.r_[rng.choice(M - 1, 64, replace=False), M - 1])
        cols = np.arange(Nn) if Nn * K <= 17920 * 1536 else np.sort(np.r_[rng.choice(Nn - 1, 192, replace=False), Nn - 1])
        assert rows.max() < M and cols.max() < Nn
        tr, tc = torch.as_tensor(rows, device=dev), torch.as_tensor(cols, device=dev)
        ra_c, ra_s = X.quantize_mx(f32(a[tr]), rotate=True)
        rw_c, rw_s = X.quantize_mx(f32(W[tc]), rotate=True)
        assert np.array_equal(u8(ac[tr]), ra_c) and np.array_equal(X.mx_scales_from_mma(u8(asf), M, K)[rows], ra_s)
        assert np.array_equal(u8(wc[tc]), rw_c) and np.array_equal(X.mx_scales_from_mma(u8(wsf), Nn, K)[cols], rw_s)
        ref = X.linear_mx(ra_c, ra_s, rw_c, rw_s)
        assert_close(f32(out[tr][:, tc]), ref, what=f"mxfp4 {workload}/{name}")
        del a, W, ac, asf, wc, wsf, out
