"""Pins for the CPU oracle: each check ties it to something other than itself.

Sources of truth used here: the NVFP4 format (Appendix A: E2M1 elements, E4M3
block scale per 16 elements, FP32 tensor scale), hand-worked values in
tests/golden/, closed forms, a library routine (torch's float8_e4m3fn cast),
brute force on tiny inputs, and the exact invariances of attention stated in
Sec. 2.1 / Eq. 2 (softmax shift invariance under the post-RoPE key shift,
logit preservation under paired pre-RoPE scaling).
"""
import math
import os

import numpy as np
import pytest
import torch

from oracle import nvfp4_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                yield line


# ----------------------------------------------------------------- E2M1 ---

def test_e2m1_decode_exhaustive_table():
    # Appendix A: E2M1, the eight magnitudes 0, .5, 1, 1.5, 2, 3, 4, 6 and a sign bit.
    expect = [0, .5, 1, 1.5, 2, 3, 4, 6, -0.0, -.5, -1, -1.5, -2, -3, -4, -6]
    got = O.e2m1_decode(np.arange(16))
    assert np.array_equal(got, np.array(expect))
    assert np.signbit(got[8])


def test_e2m1_roundtrip_all_codes():
    for c in range(16):
        assert O.e2m1_encode(O.e2m1_decode(c)) == c


def test_e2m1_golden_ties_and_saturation():
    for row in _golden_rows("e2m1_rne.txt"):
        v, c = row.split()
        assert O.e2m1_encode(np.float64(float(v))) == int(c, 16), row


def test_e2m1_neighbours_of_midpoints():
    # Just off a tie the nearest grid point decides, whatever the tie rule.
    grid = O.E2M1_GRID
    for i in range(7):
        mid = np.float32((grid[i] + grid[i + 1]) / 2)
        lo = np.nextafter(mid, np.float32(0)); hi = np.nextafter(mid, np.float32(10))
        assert O.e2m1_encode(lo) == i and O.e2m1_encode(hi) == i + 1
        assert O.e2m1_encode(-lo) == 8 | i and O.e2m1_encode(-hi) == 8 | (i + 1)


def test_e2m1_is_nearest_point_dense_sweep():
    # Independent check of "nearest": the decoded value is never farther from v
    # than any other grid magnitude.
    v = np.linspace(-7, 7, 20001)
    c = O.e2m1_encode(v)
    dec = np.abs(O.e2m1_decode(c))
    dist = np.abs(np.abs(np.minimum(np.abs(v), 6.0))[:, None] - O.E2M1_GRID[None, :]).min(axis=1)
    assert np.allclose(np.abs(np.minimum(np.abs(v), 6.0) - dec), dist, atol=0)


# ----------------------------------------------------------------- E4M3 ---

def test_e4m3_decode_matches_library_all_codes():
    lib = torch.arange(256, dtype=torch.int32).to(torch.uint8).view(torch.float8_e4m3fn).double().numpy()
    ours = O.e4m3_decode(np.arange(256))
    assert np.array_equal(np.isnan(lib), np.isnan(ours))
    fin = ~np.isnan(lib)
    assert np.array_equal(lib[fin], ours[fin])


def test_e4m3_encode_identity_on_all_finite_nonneg_codes():
    codes = np.arange(0x7F)  # 0x00..0x7E: every finite non-negative value
    assert np.array_equal(O.e4m3_encode_nonneg(O.e4m3_decode(codes)), codes.astype(np.uint8))


def test_e4m3_encode_matches_library_rne_in_range():
    rng = np.random.default_rng(7)
    v = np.concatenate([rng.uniform(0, 448, 20000), np.exp(rng.uniform(-16, 6, 20000)),
                        (O.e4m3_decode(np.arange(0x7E)) + O.e4m3_decode(np.arange(1, 0x7F))) / 2])
    v = v.astype(np.float32)
    lib = torch.from_numpy(v).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(O.e4m3_encode_nonneg(v), lib)


def test_e4m3_golden_and_saturation():
    for row in _golden_rows("e4m3_rne.txt"):
        v, c = row.split()
        assert O.e4m3_encode_nonneg(np.float64(float(v))) == int(c, 16), row
    assert O.e4m3_encode_nonneg(np.inf) == 0x7E


# ------------------------------------------------------------- quantize ---

def _parse_block(row):
    g, vals, sc, packed = [p.strip() for p in row.split("|")]
    vals = [float(t) for t in vals.split()]
    return np.float32(float(g)), np.array(vals, np.float32), int(sc, 16), [int(t, 16) for t in packed.split()]


def test_quantize_golden_blocks():
    n = 0
    for row in _golden_rows("nvfp4_blocks.txt"):
        g, x, sc, packed = _parse_block(row)
        codes, scales = O.quantize(x[None, :], g)
        assert scales[0, 0] == sc, row
        assert list(codes[0]) == packed, row
        n += 1
    assert n == 6


def test_quantize_scale_closed_form_and_error_bound():
    rng = np.random.default_rng(1)
    x = (rng.standard_normal((64, 256)) * np.exp(rng.uniform(-3, 3, (64, 1)))).astype(np.float32)
    g = O.tensor_scale(x)
    codes, S = O.quantize(x, g)
    s_true = np.abs(x.reshape(64, 16, 16)).max(axis=2) / (6.0 * float(g))
    s_val = O.e4m3_decode(S)
    normal = s_true >= 2 ** -6
    # RNE onto 3 mantissa bits: relative error at most 2**-4 in the normal range.
    assert np.all(np.abs(s_val[normal] - s_true[normal]) <= 2 ** -4 * s_true[normal] * (1 + 1e-6))
    # The block holding the tensor amax maps to the largest scale, 448.
    r, b = np.unravel_index(np.argmax(np.abs(x)), x.shape)
    assert S[r, b // 16] == 0x7E
    # Element error: half the local grid spacing times S*g, plus saturation.
    xh = O.dequantize(codes, S, g)
    Sg = np.repeat(s_val, 16, axis=1) * float(g)
    v = np.abs(x) / np.where(Sg > 0, Sg, 1)
    gap = np.where(v < 2, 0.5, np.where(v < 4, 1.0, 2.0))
    bound = 0.5 * gap * Sg + np.maximum(v - 6, 0) * Sg + 1e-6 * np.abs(x)
    assert np.all(np.abs(x - xh) <= bound)


def test_quantize_roundtrip_of_representable_blocks():
    # Every code, both signs, in blocks whose amax pins S exactly: quantize(dequant) == id.
    rng = np.random.default_rng(3)
    for _ in range(20):
        g = np.float32(2.0 ** rng.integers(-20, 5))
        S = int(rng.integers(0x08, 0x7F))                  # normal E4M3 scale
        codes = rng.integers(0, 16, 16).astype(np.uint8)
        codes[0] = 7                                        # amax element = 6 * S * g
        packed = (codes[0::2] | (codes[1::2] << 4)).astype(np.uint8)[None, :]
        x = O.dequantize(packed, np.array([[S]], np.uint8), g).astype(np.float32)
        c2, s2 = O.quantize(x, g)
        assert s2[0, 0] == S and np.array_equal(c2, packed)


def test_pack_order_low_nibble_first():
    x = np.zeros((1, 16), np.float32)
    x[0, 0] = 6.0  # code 7 in the low nibble of byte 0
    x[0, 3] = -3.0  # code 0xD in the high nibble of byte 1
    codes, _ = O.quantize(x, np.float32(1.0))
    assert codes[0, 0] == 0x07 and codes[0, 1] == 0xD0


def test_tensor_scale_closed_form():
    x = np.array([[0.5, -2688.0, 3.0]], np.float32)
    assert O.tensor_scale(x) == np.float32(1.0)
    assert O.tensor_scale(np.zeros((2, 16), np.float32)) == np.float32(1.0)


# ----------------------------------------------------------- MMA layout ---

def test_mma_layout_golden_offsets():
    rows, cols = 256, 128
    S = np.zeros((rows, cols // 16), np.uint8)
    for row in _golden_rows("mma_scale_layout.txt"):
        r, kb, off = (int(t) for t in row.split())
        S[:] = 0
        S[r, kb] = 0xA5
        flat = O.scales_to_mma(S)
        assert flat.size == 2048 and np.flatnonzero(flat).tolist() == [off], row


def test_mma_layout_roundtrip_and_padding():
    rng = np.random.default_rng(5)
    for rows, cols in [(1, 64), (130, 192), (256, 128), (17, 1536)]:
        S = rng.integers(1, 255, (rows, cols // 16)).astype(np.uint8)
        flat = O.scales_to_mma(S)
        assert flat.size == ((rows + 127) // 128) * 128 * cols // 16
        assert np.array_equal(O.scales_from_mma(flat, rows, cols), S)
        assert np.count_nonzero(flat) == S.size  # padding rows are zero


# ----------------------------------------------------------------- GEMM ---

def _brute_linear(a, w):
    M, K = a.shape
    N = w.shape[0]
    out = [[0.0] * N for _ in range(M)]
    for m in range(M):
        for n in range(N):
            acc = 0.0
            for k in range(K):
                acc += float(a[m, k]) * float(w[n, k])
            out[m][n] = acc
    return np.array(out)


@pytest.mark.parametrize("M,N,K", [(3, 5, 16), (7, 4, 32), (2, 9, 64), (5, 3, 256)])
def test_linear_brute_force(M, N, K):
    rng = np.random.default_rng(M * 100 + N)
    a = rng.standard_normal((M, K)).astype(np.float32)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    ga, gw = O.tensor_scale(a), O.tensor_scale(w)
    ac, as_ = O.quantize(a, ga)
    wc, ws = O.quantize(w, gw)
    ref = O.linear(ac, as_, ga, wc, ws, gw)
    brute = _brute_linear(O.dequantize(ac, as_, ga), O.dequantize(wc, ws, gw))
    assert ref.shape == (M, N)
    assert np.allclose(ref, brute, rtol=1e-12, atol=1e-300)
    # Rows subset agrees with the full product.
    assert np.allclose(O.linear_rows(ac, as_, ga, wc, ws, gw, [M - 1, 0]), ref[[M - 1, 0]], rtol=1e-13, atol=0)


def test_linear_k16_is_outer_product_and_identity_codes():
    a = np.array([[1, 2, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0]], np.float32) * 3.0
    w = np.zeros((16, 16), np.float32)
    for i in range(16):
        w[i, i] = 6.0                                       # W = 6 * I, exact in NVFP4 with S = 1, g = 1
    ac, as_ = O.quantize(a, np.float32(1.0))
    wc, ws = O.quantize(w, np.float32(1.0))
    out = O.linear(ac, as_, 1.0, wc, ws, 1.0)
    assert np.array_equal(out, 6.0 * O.dequantize(ac, as_, 1.0))
    # K = 16, single block: the result is an outer product of (dequantized) vectors.
    u = O.dequantize(*O.quantize(np.ones((4, 16), np.float32) * np.arange(1, 5, dtype=np.float32)[:, None], 1.0), 1.0)
    v = O.dequantize(*O.quantize(np.ones((3, 16), np.float32) * np.float32(0.5), 1.0), 1.0)
    assert np.array_equal(O.linear(*O.quantize(np.ones((4, 16), np.float32) * np.arange(1, 5, dtype=np.float32)[:, None], 1.0), 1.0,
                                   *O.quantize(np.ones((3, 16), np.float32) * np.float32(0.5), 1.0), 1.0),
                          16 * np.outer(u[:, 0], v[:, 0]))


# ------------------------------------------------------------ attention ---

def _cache(rng, B, Hkv, T, d=128, cap=None):
    cap = cap or T
    kc = np.zeros((B, Hkv, cap, d // 2), np.uint8); ks = np.zeros((B, Hkv, cap, d // 16), np.uint8)
    vc = np.zeros_like(kc); vs = np.zeros_like(ks)
    k = rng.standard_normal((B * T, Hkv, d)).astype(np.float32)
    v = rng.standard_normal((B * T, Hkv, d)).astype(np.float32)
    gk, gv = O.tensor_scale(k), O.tensor_scale(v)
    seq = np.repeat(np.arange(B), T); pos = np.tile(np.arange(T), B)
    O.kv_append(kc, ks, vc, vs, k, v, seq, pos, gk, gv)
    return kc, ks, vc, vs, gk, gv


def test_attention_single_token_returns_v():
    rng = np.random.default_rng(11)
    kc, ks, vc, vs, gk, gv = _cache(rng, 2, 2, 1)
    q = rng.standard_normal((2, 6, 128)).astype(np.float32)
    out = O.decode_attention(q, kc, ks, vc, vs, [1, 1], gk, gv, 1 / math.sqrt(128))
    for b in range(2):
        for h in range(6):
            assert np.array_equal(out[b, h], O.dequantize(vc[b, h // 3, :1], vs[b, h // 3, :1], gv)[0])


def test_attention_empty_sequence_is_zero():
    rng = np.random.default_rng(10)
    kc, ks, vc, vs, gk, gv = _cache(rng, 2, 1, 3)
    q = rng.standard_normal((2, 2, 128)).astype(np.float32)
    out = O.decode_attention(q, kc, ks, vc, vs, [0, 3], gk, gv, 0.1)
    assert not out[0].any() and out[1].any()


def test_attention_equal_keys_or_zero_query_is_mean_of_v():
    rng = np.random.default_rng(12)
    kc, ks, vc, vs, gk, gv = _cache(rng, 1, 1, 37)
    V = O.dequantize(vc[0, 0], vs[0, 0], gv)
    q0 = np.zeros((1, 2, 128), np.float32)
    out = O.decode_attention(q0, kc, ks, vc, vs, [37], gk, gv, 0.1)
    assert np.allclose(out[0, 0], V.mean(axis=0), rtol=1e-13, atol=1e-15)
    kc[0, 0, :] = kc[0, 0, 5]; ks[0, 0, :] = ks[0, 0, 5]      # all keys equal
    q = rng.standard_normal((1, 2, 128)).astype(np.float32)
    out = O.decode_attention(q, kc, ks, vc, vs, [37], gk, gv, 0.1)
    assert np.allclose(out[0, 1], V.mean(axis=0), rtol=1e-13, atol=1e-15)


def test_attention_brute_force_and_gqa_map():
    rng = np.random.default_rng(13)
    kc, ks, vc, vs, gk, gv = _cache(rng, 2, 2, 9)
    q = rng.standard_normal((2, 10, 128)).astype(np.float32)
    out = O.decode_attention(q, kc, ks, vc, vs, [9, 4], gk, gv, 0.125)
    for b, T in [(0, 9), (1, 4)]:
        for h in range(10):
            kv = h // 5                                       # contiguous groups of 5 query heads
            K = O.dequantize(kc[b, kv, :T], ks[b, kv, :T], gk)
            V = O.dequantize(vc[b, kv, :T], vs[b, kv, :T], gv)
            logits = [0.125 * sum(float(q[b, h, i]) * K[t, i] for i in range(128)) for t in range(T)]
            mx = max(logits)
            e = [math.exp(l - mx) for l in logits]
            ref = sum(e[t] / sum(e) * V[t] for t in range(T))
            assert np.allclose(out[b, h], ref, rtol=1e-12, atol=1e-14)


def test_attention_invariant_to_key_shift():
    # Softmax shift invariance behind the post-RoPE shift K~ = R(K) - m (Sec. 2.1, Eq. 2):
    # subtracting the same vector from every key changes all logits of a query by a constant.
    rng = np.random.default_rng(14)
    K = rng.standard_normal((50, 128)); V = rng.standard_normal((50, 128)); q = rng.standard_normal(128)
    m = rng.standard_normal(128) * 3
    a = O.attention_fp64(q, K, V, 0.09)
    b = O.attention_fp64(q, K - m[None, :], V, 0.09)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-13)
    assert not np.allclose(O.attention_fp64(q, K * 1.5, V, 0.09), a)  # the check can fail


def test_paired_scaling_commutes_with_rope_and_preserves_logits():
    # Eq. 2 / Sec. 2.1: with s_r = s_{r+d/2}, R(q*s) . R(k/s) == R(q) . R(k).
    rng = np.random.default_rng(15)
    d, T = 128, 20
    q_pre = rng.standard_normal((T, d)); k_pre = rng.standard_normal((T, d))
    half = np.exp(rng.standard_normal(d // 2))
    s = np.concatenate([half, half])
    pos = np.arange(T) * 37
    qt, kt = O.qfit_transform(q_pre, k_pre, s, np.zeros(d), pos)
    q0, k0 = O.rope(q_pre, pos), O.rope(k_pre, pos)
    assert np.allclose(qt @ kt.T, q0 @ k0.T, rtol=1e-10, atol=1e-10)
    # An unpaired scale breaks it (so the check can fail).
    s_bad = np.exp(rng.standard_normal(d))
    qb, kb = O.qfit_transform(q_pre, k_pre, s_bad, np.zeros(d), pos)
    assert not np.allclose(qb @ kb.T, q0 @ k0.T, rtol=1e-6)
    # RoPE preserves norms (a rotation of channel pairs).
    assert np.allclose(np.linalg.norm(q0, axis=1), np.linalg.norm(q_pre, axis=1))


def test_kv_append_shift_is_subtracted_before_quantization():
    rng = np.random.default_rng(16)
    B, Hkv, d = 1, 2, 128
    k = rng.standard_normal((3, Hkv, d)).astype(np.float32) + 4.0
    v = rng.standard_normal((3, Hkv, d)).astype(np.float32)
    m = np.full((Hkv, d), 4.0, np.float32)
    kc = np.zeros((B, Hkv, 8, 64), np.uint8); ks = np.zeros((B, Hkv, 8, 8), np.uint8)
    vc = np.zeros_like(kc); vs = np.zeros_like(ks)
    O.kv_append(kc, ks, vc, vs, k, v, [0, 0, 0], [5, 1, 2], np.float32(0.01), np.float32(0.02), k_shift=m)
    c, s = O.quantize((k[0] - m).astype(np.float32), np.float32(0.01))
    assert np.array_equal(kc[0, :, 5], c) and np.array_equal(ks[0, :, 5], s)
    c, s = O.quantize(v[1], np.float32(0.02))
    assert np.array_equal(vc[0, :, 1], c) and np.array_equal(vs[0, :, 1], s)
    assert not kc[0, :, 0].any() and not kc[0, :, 3:5].any()


# ------------------------------------------------- RoPE from a table (fp32) ---

def test_rope_table_matches_closed_form_angles():
    t = O.rope_table(5, head_dim=8, theta=10000.0)
    assert t.dtype == np.float32 and t.shape == (5, 4, 2)
    assert np.array_equal(t[0, :, 0], np.ones(4, np.float32)) and np.array_equal(t[0, :, 1], np.zeros(4, np.float32))
    # channel 0 has frequency 1: angle = position exactly
    assert np.array_equal(t[:, 0, 0], np.cos(np.arange(5.0)).astype(np.float32))
    assert np.array_equal(t[:, 0, 1], np.sin(np.arange(5.0)).astype(np.float32))
    # last pair: theta^(-2*3/8) = 10000^-0.75 = 0.001
    assert np.allclose(t[3, 3, 1], np.sin(3 * 1e-3), rtol=1e-6)


def test_rope_f32_position_zero_is_identity_and_matches_fp64_rope():
    rng = np.random.default_rng(21)
    x = rng.standard_normal((6, 3, 128)).astype(np.float32)
    pos = np.array([0, 1, 7, 100, 4095, 16383])
    tab = O.rope_table(16384)
    y = O.rope_f32(x, pos, tab)
    assert np.array_equal(y[0], x[0])                       # cos = 1, sin = 0 exactly
    ref = O.rope(np.moveaxis(x, 0, -2), pos)                # fp64 closed form, [3, 6, 128]
    ref = np.moveaxis(ref, -2, 0)
    # fp32 table (|error| <= 2^-25) plus three fp32 roundings: a few ulps of the inputs' scale
    assert np.abs(y - ref).max() <= 8 * np.finfo(np.float32).eps * np.abs(x).max()
    # a rotation: each (i, i + 64) pair keeps its length
    n_in = x[..., :64] ** 2 + x[..., 64:] ** 2
    n_out = y.astype(np.float64)[..., :64] ** 2 + y.astype(np.float64)[..., 64:] ** 2
    assert np.allclose(n_out, n_in, rtol=1e-5, atol=1e-6)


def test_rope_f32_quarter_turn_swaps_halves():
    # A table whose angle is pi/2 exactly in fp32 terms (cos 0, sin 1): y1 = -x2, y2 = x1.
    tab = np.zeros((1, 64, 2), np.float32); tab[..., 1] = 1.0
    x = np.random.default_rng(3).standard_normal((1, 2, 128)).astype(np.float32)
    y = O.rope_f32(x, np.array([0]), tab)
    assert np.array_equal(y[..., :64], -x[..., 64:]) and np.array_equal(y[..., 64:], x[..., :64])


def test_kv_append_rope_equals_rope_then_shifted_append():
    rng = np.random.default_rng(8)
    B, H, T, n = 2, 2, 16, 5
    tab = O.rope_table(T)
    k = (rng.standard_normal((n, H, 128)) * 3).astype(np.float32)
    v = rng.standard_normal((n, H, 128)).astype(np.float32)
    m = rng.standard_normal((H, 128)).astype(np.float32)
    seq = np.array([0, 1, 1, 0, 1]); pos = np.array([3, 0, 15, 9, 4])
    bufs = lambda: [np.zeros((B, H, T, 64), np.uint8), np.zeros((B, H, T, 8), np.uint8),
                    np.zeros((B, H, T, 64), np.uint8), np.zeros((B, H, T, 8), np.uint8)]
    a, b = bufs(), bufs()
    O.kv_append_rope(*a, k, v, seq, pos, np.float32(0.01), np.float32(0.02), tab, k_shift=m)
    O.kv_append(*b, O.rope_f32(k, pos, tab), v, seq, pos, np.float32(0.01), np.float32(0.02), k_shift=m)
    for u, w in zip(a, b):
        assert np.array_equal(u, w)
    # the shift is applied after RoPE: dequantized K~ + m is close to RoPE(K)
    kc = a[0][seq, :, pos]; ks = a[1][seq, :, pos]
    kh = O.dequantize(kc.reshape(n * H, 64), ks.reshape(n * H, 8), np.float32(0.01)).reshape(n, H, 128)
    ref = np.moveaxis(O.rope(np.moveaxis(k, 0, -2), pos), -2, 0) - m
    assert np.abs(kh - ref).max() <= 0.01 * 448 * 6 / 4 + 1e-3


# ------------------------------------------- SwiGLU + quantize after gate_up ---

def test_silu_closed_forms():
    assert O.silu(0.0) == 0.0
    assert np.isclose(O.silu(1.0), 1.0 / (1.0 + np.exp(-1.0)), rtol=1e-15)
    x = np.linspace(-30, 30, 61)
    assert np.allclose(O.silu(-x), O.silu(x) - x, atol=1e-12)       # sigmoid(-x) = 1 - sigmoid(x)
    assert np.allclose(O.silu(np.array([50.0, 100.0])), [50.0, 100.0])
    assert np.abs(O.silu(np.array([-50.0, -100.0]))).max() < 1e-18
    assert np.isclose(O.silu(-1.2784645), -0.2784645, atol=1e-6)    # the minimum of x*sigmoid(x)


def test_interleave_gate_up_row_order():
    I, K = 48, 3
    g = np.arange(I * K).reshape(I, K); u = -np.arange(I * K).reshape(I, K) - 1
    w = O.interleave_gate_up(g, u)
    assert w.shape == (2 * I, K)
    assert np.array_equal(w[0:16], g[0:16]) and np.array_equal(w[16:32], u[0:16])
    assert np.array_equal(w[64:80], g[32:48]) and np.array_equal(w[80:96], u[32:48])
    assert sorted(map(tuple, w.tolist())) == sorted(map(tuple, np.concatenate([g, u]).tolist()))


def test_linear_swiglu_quantize_brute_force():
    rng = np.random.default_rng(4)
    M, I, K = 3, 16, 32
    a_c = rng.integers(0, 256, (M, K // 2)).astype(np.uint8); a_s = rng.integers(0x30, 0x40, (M, K // 16)).astype(np.uint8)
    g_c = rng.integers(0, 256, (I, K // 2)).astype(np.uint8); g_s = rng.integers(0x30, 0x40, (I, K // 16)).astype(np.uint8)
    u_c = rng.integers(0, 256, (I, K // 2)).astype(np.uint8); u_s = rng.integers(0x30, 0x40, (I, K // 16)).astype(np.uint8)
    ga, gw = np.float32(0.25), np.float32(0.5)
    h, codes, scales = O.linear_swiglu_quantize(a_c, a_s, ga, g_c, g_s, u_c, u_s, gw, np.float32(0.01))
    A = O.dequantize(a_c, a_s, ga); Wg = O.dequantize(g_c, g_s, gw); Wu = O.dequantize(u_c, u_s, gw)
    for m in range(M):
        for i in range(I):
            gs = sum(A[m, k] * Wg[i, k] for k in range(K)); us = sum(A[m, k] * Wu[i, k] for k in range(K))
            assert np.isclose(h[m, i], gs / (1 + np.exp(-gs)) * us, rtol=1e-12, atol=1e-12)
    rc, rs = O.quantize(h.astype(np.float32), np.float32(0.01))
    assert np.array_equal(codes, rc) and np.array_equal(scales, rs)


# ------------------------------------------------------- E1M2 KV elements ---

def test_e1m2_decode_exhaustive_table():
    # two's-complement nibbles 0..7 -> 0..3.5, 8 -> -4 (never written), 9..15 -> -3.5..-0.5
    want = [0, .5, 1, 1.5, 2, 2.5, 3, 3.5, -4, -3.5, -3, -2.5, -2, -1.5, -1, -.5]
    assert np.array_equal(O.e1m2_decode(np.arange(16)), np.array(want))


def test_e1m2_grid_is_the_bias0_minifloat():
    # 1 exponent bit (bias 0), 2 mantissa bits: e=0 -> m/2, e=1 -> 2 + m/2
    mags = [(m / 2.0 if e == 0 else 2.0 + m / 2.0) for e in (0, 1) for m in range(4)]
    assert np.array_equal(np.sort(np.unique(np.abs(O.e1m2_decode(np.arange(16)))))[:8], np.array(mags))


def test_e1m2_encode_ties_saturation_and_roundtrip():
    # ties of 2|v| go to the even integer; beyond 3.5 saturates
    v = np.array([0.25, 0.75, 1.25, 1.75, 2.25, 3.25, 3.75, 100.0, -0.25, -0.75, -1e-9, 0.0])
    got = O.e1m2_decode(O.e1m2_encode(v))
    assert np.array_equal(got, [0.0, 1.0, 1.0, 2.0, 2.0, 3.0, 3.5, 3.5, 0.0, -1.0, 0.0, 0.0])
    codes = np.array([c for c in range(16) if c != 8])
    assert np.array_equal(O.e1m2_encode(O.e1m2_decode(codes)), codes.astype(np.uint8))


def test_e1m2_quantize_scale_closed_form_and_error_bound():
    rng = np.random.default_rng(14)
    x = (rng.standard_normal((40, 64)) * np.exp2(rng.integers(-4, 4, (40, 1)))).astype(np.float32)
    g = np.float32(np.abs(x).max() / (3.5 * 448))
    codes, S = O.quantize(x, g, "e1m2")
    blocks = np.abs(x).reshape(40, 4, 16).max(axis=2)
    # the block scale is the E4M3 rounding of amax / (3.5 g)
    want = O.e4m3_encode_nonneg((blocks / np.float32(np.float32(3.5) * g)).astype(np.float32))
    assert np.array_equal(S, want)
    xh = O.dequantize(codes, S, g, "e1m2")
    Sv = np.repeat(O.e4m3_decode(S), 16, axis=1) * np.float64(g)
    # uniform grid with step 0.5: error <= 0.25 scale units inside the range, plus E4M3's
    # rounding of the scale below amax (at most 1/16 of 3.5 units) at the block maximum
    assert np.all(np.abs(xh - x) <= (0.25 + 3.5 / 16) * Sv + 1e-12)


# -------------------------------------------------- Q-FIT calibration (Alg. 1) ---

def test_qfit_init_scale_pairs_and_floor():
    k = np.zeros((3, 1, 8)); k[0, 0, 1] = -5.0; k[2, 0, 5] = 7.0; k[1, 0, 3] = 2.0
    s0 = O.qfit_init_scale(k, eps=0.5)
    # pairs (r, r+4): (0,4) -> eps, (1,5) -> max(5, 7) = 7, (2,6) -> eps, (3,7) -> 2
    assert np.array_equal(s0[0], [0.5, 7, 0.5, 2, 0.5, 7, 0.5, 2])


def _qfit_data(B=3, T=64, hq=4, hkv=2, d=128, seed=3, offset=3.0):
    """B calibration sequences [B, T, heads, d] with per-channel outliers and a common key offset."""
    rng = np.random.default_rng(seed)
    spread = np.exp(rng.standard_normal((hkv, d)))                 # channel outliers (paired scaling helps)
    k = (rng.standard_normal((B, T, hkv, d)) * spread + offset).astype(np.float32)   # a mean (the shift helps)
    q = rng.standard_normal((B, T, hq, d)).astype(np.float32)
    v = rng.standard_normal((B, T, hkv, d)).astype(np.float32)
    return _bf(q), _bf(k), _bf(v)


def _bf(x):
    return O._bf16_round(x)


def _inverse_rope(c, positions, theta=1.0e6):
    """Keys whose RoPE at each position is the fixed vector c: rotate c by minus
    the RoPE angle pos * theta^(-2i/d) of each pair (i, i + d/2), in fp64."""
    c = np.asarray(c, np.float64)
    d = c.shape[-1]
    half = d // 2
    ang = -np.asarray(positions, np.float64)[:, None] * theta ** (-np.arange(half) * 2.0 / d)[None, :]
    cs, sn = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]       # [T, 1, half] over heads
    c1, c2 = c[None, ..., :half], c[None, ..., half:]
    return np.concatenate([c1 * cs - c2 * sn, c1 * sn + c2 * cs], axis=-1)


def test_qfit_shift_template_is_the_mean_of_the_post_rope_keys():
    # Keys built so that RoPE maps every token to the same vector c: the
    # template must be c, while the pre-RoPE keys (rotating with position)
    # average to something else.
    rng = np.random.default_rng(21)
    B, T, hkv, d = 2, 48, 2, 128
    c = rng.standard_normal((hkv, d)) * 2.0 + 1.0
    k = np.stack([_inverse_rope(c, np.arange(T)) for _ in range(B)]).astype(np.float32)
    mu = O.qfit_shift_template(k, O.rope_table(T))
    assert mu.shape == (hkv, d)
    assert np.abs(mu - c).max() < 1e-5 * np.abs(c).max()
    assert np.abs(k.astype(np.float64).reshape(-1, hkv, d).mean(axis=0) - c).max() > 0.1


def test_qfit_shift_template_at_position_zero_is_the_plain_mean():
    # One token per sequence, at position 0 where RoPE is the identity.
    rng = np.random.default_rng(22)
    k = _bf(rng.standard_normal((5, 1, 2, 128)).astype(np.float32))
    mu = O.qfit_shift_template(k, O.rope_table(1))
    assert np.array_equal(mu, k.astype(np.float64)[:, 0].mean(axis=0))


def test_qfit_reference_is_the_last_token_over_its_own_sequence():
    q, k, v = _qfit_data(B=2, T=9)
    tab = O.rope_table(9)
    y = O.qfit_reference(q, k, v, tab)
    # a single cached token: the output is that token's value (softmax of one logit)
    y1 = O.qfit_reference(q[:, :1], k[:, :1], v[:, :1], tab)
    assert np.allclose(y1, np.repeat(v[:, 0], 2, axis=1), rtol=0, atol=0)
    # each sequence attends to its own tokens only: changing sequence 1 leaves sequence 0
    k2, v2 = k.copy(), v.copy()
    k2[1] += 1.0
    v2[1] *= -1.0
    y2 = O.qfit_reference(q, k2, v2, tab)
    assert np.array_equal(y2[0], y[0]) and not np.allclose(y2[1], y[1])
    # causal: the last token's output depends on every earlier token of its sequence
    v3 = v.copy()
    v3[0, 0] += 1.0
    assert not np.array_equal(O.qfit_reference(q, k, v3, tab)[0], y[0])


def test_qfit_identity_point_is_plain_kv4_attention():
    # alpha_s = alpha_m = 0: the error is that of RoPE'd keys and values in the
    # KV4 cache, with the cache and the attention taken from the separately
    # pinned kv_append and decode_attention.
    q, k, v = _qfit_data(B=2, T=40)
    B, T, hq, d = q.shape
    hkv = k.shape[2]
    tab = O.rope_table(T)
    ones_k, ones_q, zero = np.ones((hkv, d), np.float32), np.ones((hq, d), np.float32), np.zeros((hkv, d), np.float32)
    e = O.qfit_attention_error(q, k, v, tab, ones_k, ones_q, zero)
    kr = np.stack([O.rope_f32(k[b], np.arange(T), tab) for b in range(B)])
    g_k = np.float32(np.abs(kr).max() / np.float32(2688.0))
    g_v = np.float32(np.abs(v).max() / np.float32(2688.0))
    kc = np.zeros((B, hkv, T, 64), np.uint8); ks = np.zeros((B, hkv, T, 8), np.uint8)
    vc, vs = kc.copy(), ks.copy()
    seq = np.repeat(np.arange(B), T); pos = np.tile(np.arange(T), B)
    O.kv_append(kc, ks, vc, vs, kr.reshape(-1, hkv, d), v.reshape(-1, hkv, d), seq, pos, g_k, g_v)
    qt = _bf(O.rope_f32(q[:, T - 1], np.full(B, T - 1), tab))
    y = O.decode_attention(qt, kc, ks, vc, vs, np.full(B, T), g_k, g_v, 1.0 / np.sqrt(d))
    expect = np.mean((y - O.qfit_reference(q, k, v, tab)) ** 2)
    # decode_attention takes the softmax scale as an fp32 argument (1/sqrt(128)
    # rounded to fp32); the calibration uses it in fp64: a ~1e-8 relative effect
    assert np.isclose(e, expect, rtol=1e-6, atol=0)


def test_qfit_grid_points_preserve_attention_without_quantization(monkeypatch):
    q, k, v = _qfit_data()
    tab = O.rope_table(k.shape[1])
    # With the quantizer replaced by the identity, every grid point reproduces the
    # reference (paired scaling and the shift leave attention unchanged), up to the
    # bf16 rounding of the scaled inputs.
    e_q = O.qfit_attention_error(q, k, v, tab, np.ones((2, 128), np.float32), np.ones((4, 128), np.float32),
                                 np.zeros((2, 128), np.float32))     # with the KV4 quantizer
    monkeypatch.setattr(O, "quantize", lambda x, g, element="e2m1": (np.asarray(x, np.float32), g))
    monkeypatch.setattr(O, "dequantize", lambda c, s, g, element="e2m1": np.asarray(c, np.float64))
    s0 = O.qfit_init_scale(k, 1e-6)
    mu = O.qfit_shift_template(k, tab)
    for alpha_s, alpha_m in [(0.0, 0.0), (0.5, 0.5), (0.8, 0.8)]:
        e = O.qfit_attention_error(q, k, v, tab, (s0 ** alpha_s).astype(np.float32),
                                   np.repeat(s0 ** alpha_s, 2, axis=0).astype(np.float32),
                                   (alpha_m * mu).astype(np.float32))
        # bf16 rounding of the scaled q and k (relative 2^-9) is all that remains
        assert e < 1e-4 and e < 1e-2 * e_q, (alpha_s, alpha_m, e, e_q)


def test_qfit_calibration_prefers_the_shift_for_offset_keys():
    q, k, v = _qfit_data(offset=6.0)
    tab = O.rope_table(k.shape[1])
    s_q, s_k, m, err = O.qfit_calibrate(q, k, v, tab, grid_s=3, grid_m=4)
    assert err.shape == (3, 4) and np.isfinite(err).all()
    # keys with a large common offset: some shift beats none at alpha_s = 0
    assert err[0, 1:].min() < err[0, 0]
    # the returned transformation is the first least-error grid point's:
    # S = S0^alpha_s (paired, replicated to the query heads), m = alpha_m * mu
    a, b = np.unravel_index(err.argmin(), err.shape)
    s0 = O.qfit_init_scale(k, 1e-6)
    assert np.array_equal(s_k, (s0 ** (a / 3)).astype(np.float32))
    assert np.array_equal(s_q, np.repeat(s_k, 2, axis=0))
    assert np.array_equal(m, ((b / 4) * O.qfit_shift_template(k, tab)).astype(np.float32))
    assert b > 0


def test_qfit_calibration_avoids_the_shift_for_centred_keys():
    # Without a common offset the template is ~0 and shifting buys nothing: the
    # errors along alpha_m stay within the KV4 noise of the alpha_m = 0 column.
    q, k, v = _qfit_data(offset=0.0, seed=9)
    tab = O.rope_table(k.shape[1])
    _, _, _, err = O.qfit_calibrate(q, k, v, tab, grid_s=2, grid_m=3)
    assert np.all(err[:, 1:] > 0.8 * err[:, :1])
