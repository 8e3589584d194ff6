"""GPU parity of a3 (block-scaled NVFP4 linear, tcgen05): outputs against the
oracle's fp64 product of identical dequantized operands.

Two kinds of inputs: (1) seeded random codes and scales handed to both sides
(isolates the GEMM from the quantizer), (2) the workloads' bf16 activations
and weights quantized by each side (codes are bit-exact, checked in
test_gpu_quantize), so the dequantized operands are identical."""
import numpy as np
import pytest
import torch

from _util import TOL, assert_close, assert_nvfp4_within, errors, f32, lib, swiglu_tolerance, u8
from oracle import nvfp4_oracle as O
from paper_2606_15682_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return lib()


def random_operand(rows, K, gen, scale_lo=0x30, scale_hi=0x48):
    """Seeded random NVFP4 operand: packed codes, row-major scales (all codes, moderate scales)."""
    codes = torch.randint(0, 256, (rows, K // 2), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    scales = torch.randint(scale_lo, scale_hi, (rows, K // 16), generator=gen, dtype=torch.int32).to(torch.uint8).numpy()
    return codes, scales


def run_linear(N, a_codes, a_scales_rm, g_a, w_codes, w_scales_rm, g_w, M, Nn, K, ldo=None):
    dev = "cuda"
    ac = torch.from_numpy(a_codes).to(dev)
    wc = torch.from_numpy(w_codes).to(dev)
    asf = torch.from_numpy(O.scales_to_mma(a_scales_rm)).to(dev)
    wsf = torch.from_numpy(O.scales_to_mma(w_scales_rm)).to(dev)
    ga = torch.tensor([g_a], dtype=torch.float32, device=dev)
    gw = torch.tensor([g_w], dtype=torch.float32, device=dev)
    ldo = Nn if ldo is None else ldo
    out = torch.full((M, ldo), float("nan"), dtype=torch.bfloat16, device=dev)
    N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K, ldo=ldo)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return out


@pytest.mark.parametrize("M,Nn,K", [(128, 128, 256), (1, 16, 256), (16, 128, 512), (130, 144, 512),
                                    (257, 384, 1024), (300, 272, 2304), (128, 1024, 256),
                                    # N % 256 == 0 with too few 256 x 256 tiles for the pairs and a short
                                    # K: single CTAs
                                    (256, 256, 512), (300, 512, 1024), (640, 768, 768), (129, 1280, 2048),
                                    (16, 1536, 1536), (256, 5120, 3584),
                                    # ... and with K >= 4096: split-K clusters of 2, 3 or 4 pairs, even
                                    # and uneven K ranges, M tails, a spare CTA per pair when M <= 128
                                    (256, 512, 4096), (16, 1536, 4608), (1, 256, 4096), (300, 768, 5120),
                                    (100, 512, 6400), (256, 7168, 4096), (256, 5120, 4352),
                                    # CTA-pair path (enough 256 x 256 tiles to occupy the pairs):
                                    # M tails with a spare CTA, odd super-tile counts, one-row tail
                                    (256, 10240, 512), (300, 10240, 1024), (640, 5120, 768), (129, 12800, 256),
                                    # more 256 x 256 tiles than pairs: a second round of tiles (K = 1024), and
                                    # the W-resident form (K = 1280, 1536): runs of two units per pair, an M
                                    # tail, runs that cross a W tile
                                    (512, 10240, 1024), (300, 15360, 1536), (640, 7680, 1280),
                                    # N % 256 != 0 with K >= 2048 (single CTAs), and a pair shape with K = 4096
                                    # and a one-row M tail
                                    (640, 10112, 2048), (512, 10576, 2048), (257, 15360, 4096)])
def test_random_codes(N, M, Nn, K):
    gen = torch.Generator().manual_seed(M * 1000 + Nn * 10 + K)
    a_c, a_s = random_operand(M, K, gen)
    w_c, w_s = random_operand(Nn, K, gen)
    g_a, g_w = np.float32(0.0173), np.float32(0.00091)
    out = run_linear(N, a_c, a_s, g_a, w_c, w_s, g_w, M, Nn, K)
    ref = O.linear(a_c, a_s, g_a, w_c, w_s, g_w)
    assert_close(f32(out), ref, what=f"{M}x{Nn}x{K}")


@pytest.mark.parametrize("M,Nn,K,ldo", [(200, 160, 512, 200),     # single CTAs
                                        (200, 512, 4096, 520),    # split-K clusters
                                        (640, 10240, 1024, 10248)])  # CTA pairs
def test_ldo_padding_untouched(N, M, Nn, K, ldo):
    gen = torch.Generator().manual_seed(5)
    a_c, a_s = random_operand(M, K, gen)
    w_c, w_s = random_operand(Nn, K, gen)
    out = run_linear(N, a_c, a_s, 1.0, w_c, w_s, 1.0, M, Nn, K, ldo=ldo)
    ref = O.linear(a_c, a_s, 1.0, w_c, w_s, 1.0)
    assert_close(f32(out[:, :Nn]), ref)
    assert torch.isnan(out[:, Nn:].float()).all(), "columns beyond N must not be written"


def test_single_block_structure(N):
    # Only one nonzero 16-block per row: each output is one scaled block dot product,
    # so a misplaced scale (row, k-block) shows up as a wrong value.
    M, Nn, K = 128, 128, 512
    rng = np.random.default_rng(9)
    a_c = np.zeros((M, K // 2), np.uint8); w_c = np.zeros((Nn, K // 2), np.uint8)
    kb_a = rng.integers(0, K // 16, M); kb_w = rng.integers(0, K // 16, Nn)
    for r in range(M):
        a_c[r, kb_a[r] * 8:(kb_a[r] + 1) * 8] = rng.integers(0, 256, 8)
    for r in range(Nn):
        w_c[r, kb_w[r] * 8:(kb_w[r] + 1) * 8] = rng.integers(0, 256, 8)
    a_s = rng.integers(0x28, 0x50, (M, K // 16)).astype(np.uint8)
    w_s = rng.integers(0x28, 0x50, (Nn, K // 16)).astype(np.uint8)
    out = run_linear(N, a_c, a_s, 1.0, w_c, w_s, 1.0, M, Nn, K)
    ref = O.linear(a_c, a_s, 1.0, w_c, w_s, 1.0)
    assert_close(f32(out), ref)


@pytest.mark.parametrize("M,Nn,K", [(256, 256, 1024),    # single CTAs
                                    (256, 5120, 4352)])  # split-K clusters: partials summed in split order
def test_deterministic(N, M, Nn, K):
    gen = torch.Generator().manual_seed(11)
    # Wide scale range: partial sums that round in fp32, so a change of
    # summation order would show.
    a_c, a_s = random_operand(M, K, gen, 0x20, 0x58)
    w_c, w_s = random_operand(Nn, K, gen, 0x20, 0x58)
    o1 = run_linear(N, a_c, a_s, 1.0, w_c, w_s, 1.0, M, Nn, K)
    o2 = run_linear(N, a_c, a_s, 1.0, w_c, w_s, 1.0, M, Nn, K)
    assert torch.equal(o1, o2)


def quantize_gpu(N, x):
    g = torch.empty(1, dtype=torch.float32, device="cuda")
    N.nvfp4_tensor_scale(x, g)
    codes = torch.empty(x.shape[0], x.shape[1] // 2, dtype=torch.uint8, device="cuda")
    scales = torch.empty(N.nvfp4_scales_bytes(x.shape[0], x.shape[1], 1), dtype=torch.uint8, device="cuda")
    N.nvfp4_quantize(x, g, codes, scales, 1)
    return codes, scales, g


WL = [w for w in synth.WORKLOADS if "linears" in synth.WORKLOADS[w]]


@pytest.mark.parametrize("workload", WL)
def test_workload_linears(N, workload):
    """Every linear of every workload at full size, in the launch configuration the bench times.
    Large outputs are compared on seeded samples of rows and columns."""
    w = synth.WORKLOADS[workload]
    report = []
    for name, (Nn, K) in w["linears"].items():
        a, W = synth.linear_inputs(workload, name, device="cuda")
        M = a.shape[0]
        ac, asf, ga = quantize_gpu(N, a)
        wc, wsf, gw = quantize_gpu(N, W)
        out = torch.empty(M, Nn, dtype=torch.bfloat16, device="cuda")
        N.nvfp4_linear(ac, asf, ga, wc, wsf, gw, out, M, Nn, K)
        torch.cuda.synchronize()
        assert N.nvfp4_get_device_status() == 0
        rng = np.random.default_rng(1)
        rows = np.arange(M) if M * K <= 2048 * 8960 else np.sort(np.r_[rng.choice(M, 96, replace=False), M - 1])
        cols = np.arange(Nn) if Nn * K <= 17920 * 1536 else np.sort(np.r_[rng.choice(Nn, 256, replace=False), Nn - 1])
        g_a, g_w = O.tensor_scale(f32(a)), O.tensor_scale(f32(W))
        assert np.float32(ga.item()) == g_a and np.float32(gw.item()) == g_w
        ra_c, ra_s = O.quantize(f32(a[torch.as_tensor(rows, device="cuda")]), g_a)
        rw_c, rw_s = O.quantize(f32(W[torch.as_tensor(cols, device="cuda")]), g_w)
        ref = O.linear(ra_c, ra_s, g_a, rw_c, rw_s, g_w)
        got = f32(out[torch.as_tensor(rows, device="cuda")][:, torch.as_tensor(cols, device="cuda")])
        report.append((name,) + assert_close(got, ref, what=f"{workload}/{name}"))
    print(workload, report)


def test_injected_missing_stage_times_out_and_next_call_is_exact(N):
    """Failure detection of the GEMM without a GPU fault: the test-only fault
    knob makes both CTAs of the first CTA pair leave their first ring stage
    unissued.  The MMA issuer's and scale copiers' bounded waits run out after
    ~2 s, the pair drains its MMAs, frees TMEM and exits, the call reports
    NVFP4_ERR_TIMEOUT, and the next call is exact again."""
    import time
    M, Nn, K = 640, 10240, 2048  # a CTA-pair shape with more tiles than resident pairs
    gen = torch.Generator().manual_seed(31)
    a_c, a_s = random_operand(M, K, gen)
    w_c, w_s = random_operand(Nn, K, gen)
    dev = "cuda"
    args = (torch.from_numpy(a_c).to(dev), torch.from_numpy(O.scales_to_mma(a_s)).to(dev),
            torch.ones(1, device=dev), torch.from_numpy(w_c).to(dev),
            torch.from_numpy(O.scales_to_mma(w_s)).to(dev), torch.ones(1, device=dev))
    out = torch.full((M, Nn), float("nan"), dtype=torch.bfloat16, device=dev)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    N.nvfp4_debug_inject_fault(N.FAULT_GEMM_SKIP_STAGE)
    try:
        t0 = time.time()
        N.nvfp4_linear(*args, out, M, Nn, K)
        torch.cuda.synchronize()
        waited = time.time() - t0
    finally:
        N.nvfp4_debug_inject_fault(N.FAULT_NONE)
    assert N.nvfp4_get_device_status() == 6
    assert 1.0 < waited < 20.0, f"bounded wait expected (~2-4 s), took {waited:.1f} s"
    out.fill_(float("nan"))
    N.nvfp4_linear(*args, out, M, Nn, K)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    assert_close(f32(out), O.linear(a_c, a_s, 1.0, w_c, w_s, 1.0), what="after the injected timeout")


def test_injected_missing_stage_in_split_k_cluster_times_out(N):
    """The same fault in the split-K cluster kernel (a decode-sized shape with
    three CTA pairs per tile): the first pair of the first cluster leaves its
    first stage unissued; the other pairs of that cluster finish and wait at
    the cluster barrier, the faulted pair's bounded waits run out, the call
    reports NVFP4_ERR_TIMEOUT and the next call is exact."""
    import time
    M, Nn, K = 256, 5120, 4352
    gen = torch.Generator().manual_seed(37)
    a_c, a_s = random_operand(M, K, gen)
    w_c, w_s = random_operand(Nn, K, gen)
    dev = "cuda"
    args = (torch.from_numpy(a_c).to(dev), torch.from_numpy(O.scales_to_mma(a_s)).to(dev),
            torch.ones(1, device=dev), torch.from_numpy(w_c).to(dev),
            torch.from_numpy(O.scales_to_mma(w_s)).to(dev), torch.ones(1, device=dev))
    out = torch.full((M, Nn), float("nan"), dtype=torch.bfloat16, device=dev)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    N.nvfp4_debug_inject_fault(N.FAULT_GEMM_SKIP_STAGE)
    try:
        t0 = time.time()
        N.nvfp4_linear(*args, out, M, Nn, K)
        torch.cuda.synchronize()
        waited = time.time() - t0
    finally:
        N.nvfp4_debug_inject_fault(N.FAULT_NONE)
    assert N.nvfp4_get_device_status() == 6
    assert 1.0 < waited < 20.0, f"bounded wait expected (~2-4 s), took {waited:.1f} s"
    out.fill_(float("nan"))
    N.nvfp4_linear(*args, out, M, Nn, K)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    assert_close(f32(out), O.linear(a_c, a_s, 1.0, w_c, w_s, 1.0), what="after the injected timeout")


# ------------------------------------ gate_up with SwiGLU + quantize fused ---

def test_interleave_gate_up_matches_oracle(N):
    gen = torch.Generator().manual_seed(12)
    I, K = 96, 200
    g = torch.randn(I, K, generator=gen).to(torch.bfloat16)
    u = torch.randn(I, K, generator=gen).to(torch.bfloat16)
    out = torch.empty(2 * I, K, dtype=torch.bfloat16, device="cuda")
    N.nvfp4_interleave_gate_up(g.cuda(), u.cuda(), out)
    torch.cuda.synchronize()
    ref = O.interleave_gate_up(g.view(torch.int16).numpy(), u.view(torch.int16).numpy())
    assert np.array_equal(out.cpu().view(torch.int16).numpy(), ref)


def swiglu_case(N, M, I, K, seed, rows=None):
    gen = torch.Generator().manual_seed(seed)
    a_c, a_s = random_operand(M, K, gen)
    wg_c, wg_s = random_operand(I, K, gen, 0x30, 0x40)
    wu_c, wu_s = random_operand(I, K, gen, 0x30, 0x40)
    g_a, g_w = np.float32(0.0173), np.float32(0.0021)
    rows = np.arange(M) if rows is None else rows
    G = O.linear_rows(a_c, a_s, g_a, wg_c, wg_s, g_w, rows)
    U = O.linear_rows(a_c, a_s, g_a, wu_c, wu_s, g_w, rows)
    h = O.silu(G) * U
    g_out = O.tensor_scale(h.astype(np.float32))            # a calibrated static scale
    w_c = O.interleave_gate_up(wg_c, wu_c)
    w_s = O.interleave_gate_up(wg_s, wu_s)
    dev = "cuda"
    out_c = torch.full((M, I // 2), 0xEE, dtype=torch.uint8, device=dev)
    out_s = torch.full((N.nvfp4_scales_bytes(M, I, 1),), 0xEE, dtype=torch.uint8, device=dev)
    N.nvfp4_linear_swiglu_quantize(torch.from_numpy(a_c).to(dev), torch.from_numpy(O.scales_to_mma(a_s)).to(dev),
                                   torch.tensor([g_a], device=dev), torch.from_numpy(w_c).to(dev),
                                   torch.from_numpy(O.scales_to_mma(w_s)).to(dev), torch.tensor([g_w], device=dev),
                                   M, I, K, torch.tensor([g_out], device=dev), out_c, out_s)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    return h, g_out, rows, u8(out_c), u8(out_s), swiglu_tolerance(G, U, h)


@pytest.mark.parametrize("M,I,K", [(256, 128, 256), (129, 384, 512), (300, 256, 1024), (640, 512, 768)])
def test_linear_swiglu_quantize(N, M, I, K):
    """h = SiLU(gate) * up from the fp32 accumulators, quantized with a static
    scale.  The kernel's SiLU uses the hardware tanh approximation, so every
    block scale and code must be one the recipe gives for some h' within that
    approximation's error of the exact fp64 h; no other difference is allowed.
    Most equal the oracle's quantization of h; padding scales are zero."""
    h, g_out, rows, out_c, out_s, tol = swiglu_case(N, M, I, K, seed=M + I + K)
    rc, rs = O.quantize(h.astype(np.float32), g_out)
    gs = O.scales_from_mma(out_s, M, I)
    assert_nvfp4_within(out_c, gs, h, tol, g_out, what=f"swiglu {M}x{I}x{K}")
    assert (gs == rs).mean() > 0.99 and (out_c == rc).mean() > 0.99
    pad = np.setdiff1d(np.arange(O.mma_scale_bytes(M, I)), O._mma_offsets(M, I // 16).ravel())
    assert not out_s[pad].any(), "padding rows of the output scales must be zero"


def test_linear_swiglu_quantize_prefill_shape_then_down(N):
    """The 1.5B-prefill MLP shape (M=2048, I=8960, K=1536) checked on sampled rows,
    then fed to the down projection as its A operand."""
    M, I, K, Hd = 2048, 8960, 1536, 1536
    rows = np.sort(np.r_[np.random.default_rng(2).choice(M, 48, replace=False), M - 1])
    h, g_out, rows, out_c, out_s, tol = swiglu_case(N, M, I, K, seed=99, rows=rows)
    gs = O.scales_from_mma(out_s, M, I)[rows]
    assert_nvfp4_within(out_c[rows], gs, h, tol, g_out, what="swiglu 1.5B prefill")
    # down projection straight from the fused output
    gen = torch.Generator().manual_seed(7)
    wd_c, wd_s = random_operand(Hd, I, gen)
    g_wd = np.float32(0.003)
    out = torch.empty(M, Hd, dtype=torch.bfloat16, device="cuda")
    N.nvfp4_linear(torch.from_numpy(out_c).cuda(), torch.from_numpy(out_s).cuda(),
                   torch.tensor([g_out], device="cuda"), torch.from_numpy(wd_c).cuda(),
                   torch.from_numpy(O.scales_to_mma(wd_s)).cuda(), torch.tensor([g_wd], device="cuda"), out, M, Hd, I)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    ref = O.linear_rows(out_c, O.scales_from_mma(out_s, M, I), g_out, wd_c, wd_s, g_wd, rows)
    assert_close(f32(out[torch.as_tensor(rows, device="cuda")]), ref, what="down(swiglu)")


def test_linear_swiglu_quantize_invalid_g_out_zeroes_and_reports(N):
    M, I, K = 256, 128, 256
    gen = torch.Generator().manual_seed(3)
    a_c, a_s = random_operand(M, K, gen)
    w_c, w_s = random_operand(2 * I, K, gen)
    dev = "cuda"
    out_c = torch.full((M, I // 2), 0xEE, dtype=torch.uint8, device=dev)
    out_s = torch.full((N.nvfp4_scales_bytes(M, I, 1),), 0xEE, dtype=torch.uint8, device=dev)
    N.nvfp4_get_device_status()
    N.nvfp4_linear_swiglu_quantize(torch.from_numpy(a_c).to(dev), torch.from_numpy(O.scales_to_mma(a_s)).to(dev),
                                   torch.ones(1, device=dev), torch.from_numpy(w_c).to(dev),
                                   torch.from_numpy(O.scales_to_mma(w_s)).to(dev), torch.ones(1, device=dev),
                                   M, I, K, torch.tensor([-1.0], device=dev), out_c, out_s)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 1
    assert not u8(out_c).any() and not u8(out_s).any()
