"""Pins for the MXFP4 oracle (oracle/mxfp4_oracle.py).

Sources of truth: the MXFP4 format (Appendix A: E2M1 elements, one E8M0 scale
per 32 elements, no global scale), a library decoder of E8M0
(torch.float8_e8m0fnu), a library Hadamard matrix (scipy.linalg.hadamard),
closed forms of the shared exponent, hand-worked blocks, exact round trips,
the algebra of H_32 (symmetric, H H = 32 I) and brute force on tiny inputs.
"""
import numpy as np
import pytest
import scipy.linalg
import torch

from oracle import mxfp4_oracle as X
from oracle import nvfp4_oracle as O


def _f32(a):
    return np.asarray(a, dtype=np.float32)


# ----------------------------------------------------------------- E8M0 ---

def test_e8m0_decode_matches_torch_for_every_code():
    codes = np.arange(256)
    ref = torch.from_numpy(codes.astype(np.uint8)).view(torch.float8_e8m0fnu).double().numpy()
    got = X.e8m0_decode(codes)
    assert np.isnan(got[255]) and np.isnan(ref[255])
    assert np.array_equal(got[:255], ref[:255])
    assert got[127] == 1.0 and got[0] == 2.0 ** -127 and got[254] == 2.0 ** 127


# ------------------------------------------------------- shared exponent ---

def test_shared_exponent_closed_form():
    rng = np.random.default_rng(1)
    # Magnitudes across the whole bf16 normal range: amax / 2**e lands in [4, 8).
    amax = np.ldexp(rng.uniform(1.0, 2.0, 4000), rng.integers(-120, 120, 4000))
    e = X.shared_exponent(amax)
    r = amax / np.ldexp(1.0, e)
    assert np.all((r >= 4.0) & (r < 8.0))
    # Powers of two: e = log2(amax) - 2 exactly; the largest element maps onto 4.
    k = np.arange(-100, 101)
    assert np.array_equal(X.shared_exponent(np.ldexp(1.0, k)), k - 2)
    # Just below a power of two the exponent drops by one.
    assert X.shared_exponent(np.nextafter(8.0, 0.0)) == 0
    assert X.shared_exponent(8.0) == 1


def test_shared_exponent_clamps_and_zero():
    assert X.shared_exponent(0.0) == -127
    assert X.shared_exponent(2.0 ** -140) == -127          # below E8M0's range: clamped
    assert X.shared_exponent(2.0 ** -125) == -127          # floor(log2) - 2 = -127
    assert X.shared_exponent(2.0 ** -124) == -126
    big = float(np.float32(3.0e38))                        # near the bf16 / fp32 maximum
    assert X.shared_exponent(big) == 125                   # floor(log2) = 127


# ---------------------------------------------------------- quantization ---

def test_hand_worked_block():
    # amax = 6: e = floor(log2 6) - 2 = 0, X = 1, so the codes are plain E2M1 RNE
    # of the values: ties go to the even mantissa (0.25 -> 0, 0.75 -> 1,
    # 1.25 -> 1, 1.75 -> 2, 2.5 -> 2, 3.5 -> 4, 5 -> 4), the sign is kept.
    vals = [6.0, 0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, -0.25, -0.75, -1.25, -1.75, -2.5, -3.5, -5.0, -6.0]
    x = _f32([vals + [0.0] * 16])
    codes, scales = X.quantize_mx(x)
    assert scales.tolist() == [[127]]
    c = O.unpack_codes(codes)[0].tolist()
    assert c[:16] == [7, 0, 2, 2, 4, 4, 6, 6, 8, 10, 10, 12, 12, 14, 14, 15]
    assert c[16:] == [0] * 16


def test_clipping_between_6_and_8_scales():
    # amax = 7.5: e = 0 still, so 7.5 saturates to 6 (the format's clipping);
    # amax = 8: e = 1, X = 2, 8 -> 4 exactly and 7.5 -> 3.75 -> 4 (RNE between 3 and 4).
    x = _f32([[7.5, 1.0] + [0.0] * 30, [8.0, 7.5] + [0.0] * 30])
    codes, scales = X.quantize_mx(x)
    assert scales[:, 0].tolist() == [127, 128]
    c = O.unpack_codes(codes)
    assert c[0, :2].tolist() == [7, 2]
    assert c[1, :2].tolist() == [6, 6]
    xh = X.dequantize_mx(codes, scales)
    assert xh[0, 0] == 6.0 and xh[1, 0] == 8.0 and xh[1, 1] == 8.0


def test_every_code_round_trips_at_every_binade():
    # A block whose amax is 4 * 2**E or 6 * 2**E has e = E, so every element
    # that is an E2M1 value times 2**E is reproduced exactly.
    rng = np.random.default_rng(2)
    grid = O.e2m1_decode(np.arange(16))
    for E in [-120, -30, -3, 0, 5, 60, 120]:
        for lead in (4.0, 6.0):
            codes_in = rng.integers(0, 16, size=(8, 31))
            vals = np.ldexp(grid[codes_in], E)
            x = np.concatenate([np.full((8, 1), np.ldexp(lead, E)), vals], axis=1)
            q, s = X.quantize_mx(_f32(x))
            assert np.all(s == E + 127)
            assert np.array_equal(X.dequantize_mx(q, s), x)


def test_error_bound_property():
    rng = np.random.default_rng(3)
    x = _f32(rng.standard_normal((64, 256)) * np.exp(rng.standard_normal((64, 1)) * 3))
    q, s = X.quantize_mx(x)
    xh = X.dequantize_mx(q, s)
    scale = np.repeat(X.e8m0_decode(s), 32, axis=1)
    v = np.abs(x.astype(np.float64)) / scale
    # half the E2M1 gap at |v| (gaps 0.5 up to 2, 1 up to 4, 2 up to 6); beyond 6 the clipping error
    half_gap = np.where(v < 2, 0.25, np.where(v < 4, 0.5, 1.0))
    bound = np.where(v <= 6, half_gap, v - 6) * scale
    assert np.all(np.abs(xh - x) <= bound * (1 + 1e-12))


def test_zero_and_signed_zero_blocks():
    x = _f32([[0.0] * 32, [-0.0] + [0.0] * 31, [-1e-30] + [1.0] + [0.0] * 30])
    q, s = X.quantize_mx(x)
    assert s[:, 0].tolist() == [0, 0, 125]            # all-zero blocks: 2**-127; amax 1 -> e = -2
    c = O.unpack_codes(q)
    assert c[0].tolist() == [0] * 32
    assert c[1, 0] == 8                                 # -0 keeps its sign
    assert c[2, 0] == 8 and c[2, 1] == 6                # a tiny negative rounds to -0; 1.0 / 0.25 = 4 is code 6


def test_brute_force_tiny():
    # Each element independently: the nearest of the 16 E2M1 values times X
    # (ties to the even code), with X = 2**e from the block's amax.
    rng = np.random.default_rng(4)
    x = _f32(rng.standard_normal((3, 64)) * 5)
    q, s = X.quantize_mx(x)
    c = O.unpack_codes(q)
    grid = O.e2m1_decode(np.arange(8))
    for r in range(3):
        for j in range(64):
            b = j // 32
            blk = x[r, 32 * b: 32 * b + 32].astype(np.float64)
            e = int(np.floor(np.log2(np.max(np.abs(blk))))) - 2
            v = abs(float(x[r, j])) / 2.0 ** e
            d = np.abs(grid - min(v, 6.0))
            best = np.flatnonzero(d == d.min())
            k = best[0] if len(best) == 1 else [i for i in best if i % 2 == 0][0]
            assert s[r, b] == e + 127
            assert c[r, j] == (k | (8 if x[r, j] < 0 else 0))


# -------------------------------------------------------------- rotation ---

def test_hadamard_is_sylvester_and_orthogonal():
    h = X.hadamard(32)
    assert np.array_equal(h, scipy.linalg.hadamard(32))
    assert np.array_equal(h, h.T)
    assert np.array_equal(h @ h, 32 * np.eye(32))


def test_rotation_definition_is_orthogonal_and_involutive():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((4, 128))
    y = X.rotate_blocks(x)
    assert np.allclose(np.linalg.norm(y.reshape(4, 4, 32), axis=2), np.linalg.norm(x.reshape(4, 4, 32), axis=2),
                       rtol=1e-13)
    assert np.allclose(X.rotate_blocks(y), x, rtol=0, atol=1e-13)


def test_rotation_fp32_matches_definition():
    rng = np.random.default_rng(6)
    x = _f32(rng.standard_normal((16, 256)) * np.exp(rng.standard_normal((16, 1))))
    got = X.rotate_blocks_f32(x).astype(np.float64)
    ref = X.rotate_blocks(x)
    # Five butterfly stages and one scaling, each rounded to fp32: the error
    # stays below 8 ulp of the block's l1 norm / sqrt(32).
    l1 = np.repeat(np.abs(x.astype(np.float64)).reshape(16, 8, 32).sum(axis=2), 32, axis=1)
    assert np.all(np.abs(got - ref) <= 8 * 2.0 ** -24 * l1 / np.sqrt(32))
    # Unit vectors: row j of H_32 times fp32(1/sqrt(32)), exactly.
    e = np.eye(32, dtype=np.float32)
    inv = np.float32(1 / np.sqrt(32))
    assert np.array_equal(X.rotate_blocks_f32(e), (scipy.linalg.hadamard(32) * inv).astype(np.float32))
    # Small integers: the butterflies are exact, only the final scaling rounds.
    xi = _f32(rng.integers(-50, 50, size=(4, 64)))
    exact = (xi.astype(np.float64).reshape(4, 2, 32) @ scipy.linalg.hadamard(32)).reshape(4, 64)
    assert np.array_equal(X.rotate_blocks_f32(xi), (_f32(exact) * inv).astype(np.float32))


def test_rotated_quantization_uses_the_rotated_values():
    rng = np.random.default_rng(7)
    x = _f32(rng.standard_normal((8, 64)))
    assert all(np.array_equal(a, b) for a, b in zip(X.quantize_mx(x, rotate=True),
                                                    X.quantize_mx(X.rotate_blocks_f32(x))))


# ---------------------------------------------------------------- linear ---

def test_mx_linear_brute_force_and_rotation_invariance():
    rng = np.random.default_rng(8)
    a = _f32(rng.standard_normal((5, 64)))
    w = _f32(rng.standard_normal((7, 64)) * 0.05)
    ac, asf = X.quantize_mx(a)
    wc, wsf = X.quantize_mx(w)
    ref = X.linear_mx(ac, asf, wc, wsf)
    ah, wh = X.dequantize_mx(ac, asf), X.dequantize_mx(wc, wsf)
    brute = np.array([[sum(ah[i, k] * wh[j, k] for k in range(64)) for j in range(7)] for i in range(5)])
    assert np.allclose(ref, brute, rtol=1e-12, atol=1e-15)
    # Rotating both operands along K (exact fp64) leaves the product unchanged.
    assert np.allclose(X.rotate_blocks(ah) @ X.rotate_blocks(wh).T, ref, rtol=1e-12, atol=1e-12)
    rows = np.array([4, 0, 2])
    assert np.array_equal(X.linear_mx_rows(ac, asf, wc, wsf, rows), ref[rows])


def test_mx_scales_mma_layout_duplicates_each_block_scale():
    rng = np.random.default_rng(9)
    s = rng.integers(0, 255, size=(130, 8)).astype(np.uint8)      # 130 rows, 256 columns
    flat = X.mx_scales_to_mma(s)
    assert flat.size == O.mma_scale_bytes(130, 256)
    s16 = O.scales_from_mma(flat, 130, 256)
    assert np.array_equal(s16[:, 0::2], s) and np.array_equal(s16[:, 1::2], s)
    assert np.array_equal(X.mx_scales_from_mma(flat, 130, 256), s)
    bad = flat.copy()
    bad[O._mma_offsets(130, 16)[0, 1]] ^= 1
    with pytest.raises(ValueError):
        X.mx_scales_from_mma(bad, 130, 256)


def test_swiglu_quantize_mx_composes_library_silu_and_the_quantizer():
    # SiLU against scipy's logistic function; the fused form is SiLU(G) * U of
    # the fp64 products, quantized from fp32 (brute-force products here).
    import scipy.special
    x = np.linspace(-30, 30, 1001)
    assert np.allclose(O.silu(x), x * scipy.special.expit(x), rtol=1e-14, atol=1e-300)
    rng = np.random.default_rng(10)
    a = _f32(rng.standard_normal((6, 64)))
    wg = _f32(rng.standard_normal((64, 64)) * 0.1)
    wu = _f32(rng.standard_normal((64, 64)) * 0.1)
    (ac, asf), (gc, gsf), (uc, usf) = X.quantize_mx(a), X.quantize_mx(wg), X.quantize_mx(wu)
    ah, gh, uh = X.dequantize_mx(ac, asf), X.dequantize_mx(gc, gsf), X.dequantize_mx(uc, usf)
    G = np.array([[sum(ah[i, k] * gh[j, k] for k in range(64)) for j in range(64)] for i in range(6)])
    U = np.array([[sum(ah[i, k] * uh[j, k] for k in range(64)) for j in range(64)] for i in range(6)])
    h_ref = G * scipy.special.expit(G) * U
    for rotate in (False, True):
        h, c, s = X.linear_swiglu_quantize_mx(ac, asf, gc, gsf, uc, usf, rotate=rotate)
        assert np.allclose(h, h_ref, rtol=1e-12, atol=1e-15)
        rc, rs = X.quantize_mx(h_ref.astype(np.float32), rotate=rotate)
        assert np.array_equal(c, rc) and np.array_equal(s, rs)
        hr, cr, sr = X.linear_swiglu_quantize_mx(ac, asf, gc, gsf, uc, usf, rotate=rotate, rows=[5, 1])
        assert np.array_equal(cr, c[[5, 1]]) and np.array_equal(sr, s[[5, 1]])
