"""GPU parity of a1 (tensor scale) and a2 (NVFP4 quantize): bit-exact against
the CPU oracle on the same seeded inputs."""
import os

import numpy as np
import pytest
import torch

from _util import f32, lib, u8
from oracle import nvfp4_oracle as O
from paper_2606_15682_gb300 import synth

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def N():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return lib()


def gpu_quantize(N, x, g, layout):
    rows, cols = x.shape
    codes = torch.empty(rows, cols // 2, dtype=torch.uint8, device="cuda")
    scales = torch.full((N.nvfp4_scales_bytes(rows, cols, layout),), 0xEE, dtype=torch.uint8, device="cuda")
    N.nvfp4_quantize(x, g, codes, scales, layout)
    return codes, scales


def check_quantize(N, x_bf16, g_np=None, layout=1, rows_sample=None):
    """Quantize on the GPU with a GPU tensor scale (or a given g) and compare with the oracle."""
    x = x_bf16.cuda()
    g = torch.empty(1, dtype=torch.float32, device="cuda")
    if g_np is None:
        N.nvfp4_tensor_scale(x, g)
        g_ref = O.tensor_scale(f32(x_bf16))
        assert np.float32(g.item()) == g_ref
    else:
        g.fill_(float(g_np))
        g_ref = np.float32(g_np)
    codes, scales = gpu_quantize(N, x, g, layout)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    rows, cols = x.shape
    sel = np.arange(rows) if rows_sample is None else np.asarray(rows_sample)
    xc = f32(x_bf16[torch.as_tensor(sel)])
    rc, rs = O.quantize(xc, g_ref)
    gc = u8(codes)[sel]
    gs = u8(scales)
    gs = gs.reshape(rows, cols // 16)[sel] if layout == 0 else O.scales_from_mma(gs, rows, cols)[sel]
    bad = np.argwhere(gc != rc)
    assert bad.size == 0, f"{len(bad)} code bytes differ, first at {bad[:3].tolist()}: gpu {gc[tuple(bad[0])]:#x} oracle {rc[tuple(bad[0])]:#x}"
    assert np.array_equal(gs, rs)
    if layout == 1 and rows % 128:
        pad = np.setdiff1d(np.arange(O.mma_scale_bytes(rows, cols)), O._mma_offsets(rows, cols // 16).ravel())
        assert not u8(scales)[pad].any(), "padding rows of the MMA scale layout must be zero"
    return codes, scales, g


def _golden_blocks():
    rows = []
    for line in open(os.path.join(GOLDEN, "nvfp4_blocks.txt")):
        line = line.split("#", 1)[0].strip()
        if line:
            g, vals, sc, packed = [p.strip() for p in line.split("|")]
            rows.append((np.float32(float(g)), np.array([float(t) for t in vals.split()], np.float32),
                         int(sc, 16), [int(t, 16) for t in packed.split()]))
    return rows


def test_golden_blocks_on_gpu(N):
    # Hand-worked ties, saturation, signed zeros, scale underflow, subnormal scales.
    for g, vals, sc, packed in _golden_blocks():
        x = torch.from_numpy(np.tile(vals, 4)[None, :]).to(torch.bfloat16)
        assert np.array_equal(f32(x)[0, :16], vals)
        codes, scales = gpu_quantize(N, x.cuda(), torch.tensor([g], device="cuda"), 0)
        assert u8(scales)[0] == sc
        assert list(u8(codes)[0, :8]) == packed


def test_signed_zero_and_tie_sweep(N):
    # Every E2M1 midpoint, its float32 neighbours and tiny negatives, in blocks with S = 1, g = 1.
    mids = [0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0]
    vals = []
    for m in mids:
        for v in (m, float(np.nextafter(np.float32(m), 0)), float(np.nextafter(np.float32(m), 10))):
            vals += [v, -v]
    vals += [-0.1, -0.0, 0.0, -1e-3, 1e-3, 6.0, -6.0]
    vals = np.array(vals, np.float32)
    vals = vals[np.abs(vals) <= 6]
    x = np.zeros((len(vals), 16), np.float32)
    x[:, 0] = 6.0
    x[:, 1] = vals
    xb = torch.from_numpy(x).to(torch.bfloat16)  # neighbours round to bf16 values near the ties
    check_quantize(N, xb, g_np=1.0, layout=0)


@pytest.mark.parametrize("layout", [0, 1])
@pytest.mark.parametrize("rows,cols,ld", [(1, 64, 64), (3, 16, 16), (130, 192, 192), (257, 512, 520), (64, 1536, 1536)])
def test_random_blocks(N, rows, cols, ld, layout):
    if layout == 1 and cols % 64:
        pytest.skip("MMA layout needs cols % 64")
    gen = torch.Generator().manual_seed(rows * 7919 + cols)
    base = torch.randn(rows, ld, generator=gen)
    # Per-block magnitudes over ~40 binades: exercises subnormal and saturated scales.
    mag = torch.exp2(torch.randint(-30, 12, (rows, (ld + 15) // 16), generator=gen).float())
    x = (base * mag.repeat_interleave(16, dim=1)[:, :ld]).to(torch.bfloat16)
    x[0, :16] = 0
    xv = x.cuda()[:, :cols] if ld != cols else x.cuda()
    g = torch.empty(1, dtype=torch.float32, device="cuda")
    N.nvfp4_tensor_scale(xv, g)
    gref = O.tensor_scale(f32(x[:, :cols]))
    assert np.float32(g.item()) == gref
    codes, scales = gpu_quantize(N, xv, g, layout)
    rc, rs = O.quantize(f32(x[:, :cols]), gref)
    assert np.array_equal(u8(codes), rc)
    gs = u8(scales).reshape(rows, cols // 16) if layout == 0 else O.scales_from_mma(u8(scales), rows, cols)
    assert np.array_equal(gs, rs)


def test_tensor_scale_all_zero_and_empty(N):
    x = torch.zeros(5, 64, dtype=torch.bfloat16, device="cuda")
    g = torch.full((1,), 7.0, device="cuda")
    N.nvfp4_tensor_scale(x, g)
    assert g.item() == 1.0
    codes, scales = gpu_quantize(N, x, g, 1)
    assert not u8(codes).any() and not u8(scales).any()
    e = torch.zeros(0, 64, dtype=torch.bfloat16, device="cuda")
    N.nvfp4_tensor_scale(e, g)
    assert g.item() == 1.0


def test_invalid_tensor_scale_sets_device_status(N):
    x = torch.randn(4, 64, device="cuda").to(torch.bfloat16)
    N.nvfp4_get_device_status()
    codes, scales = gpu_quantize(N, x, torch.tensor([-1.0], device="cuda"), 0)
    assert N.nvfp4_get_device_status() == 1
    assert not u8(codes).any() and not u8(scales).any()
    assert N.nvfp4_get_device_status() == 0


def test_relayout_roundtrip(N):
    rows, cols = 300, 320
    s = torch.randint(0, 255, (rows, cols // 16), dtype=torch.uint8)
    dst = torch.full((N.nvfp4_scales_bytes(rows, cols, 1),), 0xEE, dtype=torch.uint8, device="cuda")
    N.nvfp4_scales_relayout(s.cuda(), dst, rows, cols, 0, 1)
    assert np.array_equal(u8(dst), O.scales_to_mma(s.numpy()))
    back = torch.zeros(rows * cols // 16, dtype=torch.uint8, device="cuda")
    N.nvfp4_scales_relayout(dst, back, rows, cols, 1, 0)
    assert np.array_equal(u8(back).reshape(rows, -1), s.numpy())


WL = [w for w in synth.WORKLOADS if "linears" in synth.WORKLOADS[w]]


@pytest.mark.parametrize("workload", WL)
def test_workload_tensors_bit_exact(N, workload):
    """Activations and weights of every linear of every workload, at full size."""
    w = synth.WORKLOADS[workload]
    big = w["M"] >= 8192
    for name in w["linears"]:
        a, W = synth.linear_inputs(workload, name, device="cuda")
        rs = np.random.default_rng(0)
        a_rows = np.sort(rs.choice(a.shape[0], 192, replace=False)) if big else None
        w_rows = np.sort(rs.choice(W.shape[0], 384, replace=False)) if W.shape[0] * W.shape[1] > 5e7 else None
        if big:
            a_rows = np.concatenate([a_rows, [a.shape[0] - 1]])
        for t, rows in ((a, a_rows), (W, w_rows)):
            g_ref = O.tensor_scale(f32(t)) if rows is not None else None
            if rows is not None:
                # Same g as the GPU's own tensor-scale kernel, checked on the full tensor.
                g = torch.empty(1, dtype=torch.float32, device="cuda")
                N.nvfp4_tensor_scale(t, g)
                assert np.float32(g.item()) == g_ref
            check_quantize(N, t.cpu() if rows is None else t, g_np=g_ref, layout=1, rows_sample=rows)


# ------------------------------------------------ one-launch a1 + a2 ---

def dynamic(N, x, state, layout=1):
    rows, cols = x.shape
    g = torch.full((1,), float("nan"), dtype=torch.float32, device="cuda")
    codes = torch.empty(rows, cols // 2, dtype=torch.uint8, device="cuda")
    scales = torch.full((N.nvfp4_scales_bytes(rows, cols, layout),), 0xEE, dtype=torch.uint8, device="cuda")
    N.nvfp4_quantize_dynamic(x, state, g, codes, scales, layout)
    return codes, scales, g


def test_dynamic_matches_oracle_and_two_call_path(N):
    """Different shapes (so different grid sizes) and both layouts on one state:
    each call starts a new epoch of the state without clearing it."""
    state = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device="cuda")
    gen = torch.Generator().manual_seed(77)
    for i, (rows, cols, ld, layout) in enumerate([(130, 192, 192, 1), (3, 64, 64, 0), (2048, 1536, 1536, 1),
                                                  (257, 512, 520, 0), (1, 64, 64, 1), (700, 8960, 8960, 1)]):
        base = torch.randn(rows, ld, generator=gen)
        mag = torch.exp2(torch.randint(-20, 8, (rows, (ld + 15) // 16), generator=gen).float())
        x = (base * mag.repeat_interleave(16, dim=1)[:, :ld]).to(torch.bfloat16)
        xv = x.cuda()[:, :cols] if ld != cols else x.cuda()
        codes, scales, g = dynamic(N, xv, state, layout)
        g2 = torch.empty(1, dtype=torch.float32, device="cuda")
        N.nvfp4_tensor_scale(xv, g2)
        c2, s2 = gpu_quantize(N, xv, g2, layout)
        torch.cuda.synchronize()
        assert N.nvfp4_get_device_status() == 0
        gref = O.tensor_scale(f32(x[:, :cols]))
        assert np.float32(g.item()) == gref == np.float32(g2.item()), f"call {i}"
        assert torch.equal(codes, c2) and torch.equal(scales, s2), f"call {i}: differs from the two-call path"
        sel = np.arange(rows) if rows <= 300 else np.r_[0:64, rows - 64:rows]
        rc, rs = O.quantize(f32(x[:, :cols][torch.as_tensor(sel)]), gref)
        assert np.array_equal(u8(codes)[sel], rc), f"call {i}"
        gs = u8(scales).reshape(rows, cols // 16) if layout == 0 else O.scales_from_mma(u8(scales), rows, cols)
        assert np.array_equal(gs[sel], rs), f"call {i}"
    # Ten calls in a row (ten epochs), the last one checked.
    x = torch.randn(512, 1024, generator=gen).to(torch.bfloat16).cuda()
    for _ in range(10):
        codes, scales, g = dynamic(N, x, state)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    assert np.float32(g.item()) == O.tensor_scale(f32(x))


def test_dynamic_all_zero_and_empty(N):
    state = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device="cuda")
    codes, scales, g = dynamic(N, torch.zeros(5, 64, dtype=torch.bfloat16, device="cuda"), state)
    assert g.item() == 1.0 and not u8(codes).any() and not u8(scales).any()
    # An empty tensor: g = 1, the state is untouched, and the next call still works.
    e = torch.zeros(0, 64, dtype=torch.bfloat16, device="cuda")
    g = torch.full((1,), 3.0, device="cuda")
    N.nvfp4_quantize_dynamic(e, state, g, None, None, 1)
    assert g.item() == 1.0
    x = torch.randn(64, 128, device="cuda").to(torch.bfloat16)
    codes, scales, g = dynamic(N, x, state)
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    assert np.float32(g.item()) == O.tensor_scale(f32(x))


@pytest.mark.parametrize("workload", WL)
def test_dynamic_workload_activations(N, workload):
    """Every activation of every workload at full size, as the bench step quantizes it."""
    state = torch.zeros(N.DYNAMIC_STATE_BYTES, dtype=torch.uint8, device="cuda")
    for name in synth.WORKLOADS[workload]["linears"]:
        a, _ = synth.linear_inputs(workload, name, device="cuda")
        codes, scales, g = dynamic(N, a, state)
        g2 = torch.empty(1, dtype=torch.float32, device="cuda")
        N.nvfp4_tensor_scale(a, g2)
        c2, s2 = gpu_quantize(N, a, g2, 1)
        torch.cuda.synchronize()
        assert N.nvfp4_get_device_status() == 0
        assert g.item() == g2.item() and np.float32(g.item()) == O.tensor_scale(f32(a))
        assert torch.equal(codes, c2) and torch.equal(scales, s2), name
        M = a.shape[0]
        rows = np.unique(np.r_[0:min(32, M), max(M - 32, 0):M])
        assert rows.min() >= 0 and rows.max() < M  # checked on the host before indexing on the device
        rc, rs = O.quantize(f32(a[torch.as_tensor(rows, device="cuda")]), np.float32(g.item()))
        assert np.array_equal(u8(codes)[rows], rc)
        assert np.array_equal(O.scales_from_mma(u8(scales), a.shape[0], a.shape[1])[rows], rs)


def test_dynamic_barrier_wait_runs_out_and_reports_timeout(N):
    """A state whose arrival count can never reach the grid size (a flag that
    nothing sets): every block's bounded barrier wait expires after ~2 s, the
    kernel returns without writing, NVFP4_ERR_TIMEOUT is reported, and the
    device stays usable -- a zero-filled state works again afterwards."""
    x = torch.randn(256, 1024, device="cuda").to(torch.bfloat16)
    state = torch.zeros(N.DYNAMIC_STATE_BYTES // 8, dtype=torch.int64, device="cuda")
    state[0] = 0x7FFFFF00          # epoch 0, an arrival count far beyond any grid
    N.nvfp4_get_device_status()
    codes, scales, g = dynamic(N, x, state.view(torch.uint8))
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 6
    assert np.isnan(g.item()), "g must stay unwritten after a timeout"
    state.zero_()
    codes, scales, g = dynamic(N, x, state.view(torch.uint8))
    torch.cuda.synchronize()
    assert N.nvfp4_get_device_status() == 0
    assert np.float32(g.item()) == O.tensor_scale(f32(x))
