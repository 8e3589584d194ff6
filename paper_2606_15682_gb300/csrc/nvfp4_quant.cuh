// NVFP4 block quantization in registers (Appendix A format; the library's
// rounding recipe is stated in include/nvfp4.h).  One thread holds 8
// consecutive elements; the two lanes (2i, 2i+1) of a warp together hold one
// 16-element block and exchange their partial amax with one shuffle.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace nvfp4 {

// Exact value of an unsigned E4M3 code (bias 7, 3 mantissa bits;
// subnormals m * 2^-9).  Codes produced by the quantizer never exceed 0x7E.
__device__ __forceinline__ float e4m3_value(uint32_t c) {
  const uint32_t e = (c >> 3) & 0xFu, m = c & 7u;
  return e ? __uint_as_float(((e + 120u) << 23) | (m << 20)) : __fmul_rn(static_cast<float>(m), 0.001953125f);
}

// RNE + saturate-to-finite conversion of a non-negative fp32 to E4M3 (hardware cvt).
__device__ __forceinline__ uint32_t e4m3_rne_sat(float s) {
  uint16_t p;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(p) : "f"(0.0f), "f"(s));
  return p & 0xFFu;
}

// Block scale from the block amax: S = E4M3(amax / (6 g)); the element
// multiplier is 1 / (S g), or 0 for a zero scale so the codes become signed zeros.
struct BlockScale {
  uint32_t code;
  float mult;
};
__device__ __forceinline__ BlockScale block_scale(float amax, float g, float six_g) {
  BlockScale b;
  const float s = __fdiv_rn(amax, six_g);
  b.code = e4m3_rne_sat(s);
  const float d = __fmul_rn(e4m3_value(b.code), g);
  b.mult = b.code ? __frcp_rn(d) : 0.0f;
  return b;
}

// 8 fp32 -> 8 E2M1 codes packed into 32 bits, element 0 in the lowest nibble.
// cvt.e2m1x2 puts its first source in the high nibble, its second in the low one.
__device__ __forceinline__ uint32_t e2m1x8(const float v[8]) {
  uint32_t out;
  asm("{\n .reg .b8 b0, b1, b2, b3;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b0, %2, %1;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b1, %4, %3;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b2, %6, %5;\n"
      " cvt.rn.satfinite.e2m1x2.f32 b3, %8, %7;\n"
      " mov.b32 %0, {b0, b1, b2, b3};\n}"
      : "=r"(out)
      : "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]));
  return out;
}

// 8 fp32 -> 8 E1M2 elements (the KV variant), element 0 in the lowest nibble:
// k = RNE(2|v|) saturated at 7, stored as the two's-complement nibble of
// sign * k (a negative value that rounds to zero is stored as 0).
__device__ __forceinline__ uint32_t e1m2x8(const float v[8]) {
  uint32_t out = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int k = min(__float2int_rn(fabsf(v[i]) * 2.0f), 7);
    const int n = signbit(v[i]) ? -k : k;
    out |= (static_cast<uint32_t>(n) & 0xFu) << (4 * i);
  }
  return out;
}

// bf16 -> fp32 (exact) for the low / high half of a 32-bit pair.
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ void unpack_bf16x8(const uint4 v, float x[8]) {
  x[0] = bf16_lo(v.x); x[1] = bf16_hi(v.x);
  x[2] = bf16_lo(v.y); x[3] = bf16_hi(v.y);
  x[4] = bf16_lo(v.z); x[5] = bf16_hi(v.z);
  x[6] = bf16_lo(v.w); x[7] = bf16_hi(v.w);
}

// |x| maximum of 8 bf16 as a bf16 bit pattern: non-negative bf16 patterns
// compare like their values, so the sign bit is masked and halves compared
// as unsigned 16-bit integers.
__device__ __forceinline__ uint32_t amax_bits_bf16x8(const uint4 v) {
  const uint32_t a = __vmaxu2(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu);
  const uint32_t b = __vmaxu2(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu);
  const uint32_t m = __vmaxu2(a, b);
  return max(m & 0xFFFFu, m >> 16);
}

// Quantize 8 fp32 values whose block partner lane holds the other 8.  All 32
// lanes of the warp must call this together.  Returns packed codes; *scale
// receives the block's E4M3 code (identical in both lanes).
// kE1M2: E1M2 elements; qmax_g is then 3.5 g instead of 6 g.
template <bool kE1M2 = false>
__device__ __forceinline__ uint32_t quantize8_pair(const float x[8], float amax_own, float g, float qmax_g,
                                                   uint32_t* scale) {
  const float amax = fmaxf(amax_own, __shfl_xor_sync(0xffffffffu, amax_own, 1));
  const BlockScale b = block_scale(amax, g, qmax_g);
  float v[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __fmul_rn(x[i], b.mult);
  *scale = b.code;
  return kE1M2 ? e1m2x8(v) : e2m1x8(v);
}

// ---- MXFP4 (Appendix A: E8M0 scale per 32 elements, no global scale) ----
constexpr uint32_t kInvSqrt32Bits = 0x3E3504F3u;  // fp32(1 / sqrt(32)), round to nearest

// In-register fast Walsh-Hadamard transform of 32 values: butterflies
// (a + b, a - b) at strides 1, 2, 4, 8, 16, each rounded to fp32, then one
// fp32 multiplication by 1/sqrt(32) (Sylvester order: the result is x H_32 / sqrt(32)).
__device__ __forceinline__ void hadamard32(float x[32]) {
#pragma unroll
  for (int h = 1; h < 32; h <<= 1) {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      if ((i & h) == 0) {
        const float a = x[i], b = x[i + h];
        x[i] = __fadd_rn(a, b);
        x[i + h] = __fsub_rn(a, b);
      }
    }
  }
  const float inv = __uint_as_float(kInvSqrt32Bits);
#pragma unroll
  for (int i = 0; i < 32; ++i) x[i] = __fmul_rn(x[i], inv);
}

// E8M0 code of a 32-element block with this amax: e = floor(log2 amax) - 2,
// clamped to [-127, 127], read off the binary exponent field E (zero and
// subnormal amax have E = 0 and clamp), so the code e + 127 is max(E - 2, 0);
// a finite amax < 2^128 keeps e <= 125.
__device__ __forceinline__ uint32_t mx_scale_code(float amax) {
  const uint32_t E = __float_as_uint(amax) >> 23;
  return E > 2u ? E - 2u : 0u;
}
// 1 / 2^e = 2^(127 - code), a normal fp32 for every code the quantizer makes (<= 252).
__device__ __forceinline__ float mx_inv_scale(uint32_t code) { return __uint_as_float((254u - code) << 23); }

// Byte offset of block scale (row r, k-block kb) in the tensor-core storage
// order: 128-row tiles, groups of 4 k-blocks, 512-byte atoms k-group fastest,
// inside an atom (r%32)*16 + ((r%128)/32)*4 + kb%4.
__host__ __device__ __forceinline__ uint64_t mma_scale_offset(uint64_t r, uint32_t kb, uint32_t kgroups) {
  return ((r >> 7) * kgroups + (kb >> 2)) * 512u + (r & 31u) * 16u + ((r >> 5) & 3u) * 4u + (kb & 3u);
}

// Round-up fast division of 32-bit unsigned integers by a runtime constant.
struct FastDiv {
  uint32_t d, m, s;
  FastDiv() = default;
  __host__ explicit FastDiv(uint32_t div) : d(div) {
    s = 0;
    while ((1ull << s) < div) ++s;
    m = static_cast<uint32_t>((((1ull << 32) * ((1ull << s) - div)) / div) + 1);
  }
  __device__ __forceinline__ uint32_t div(uint32_t n) const {
    return static_cast<uint32_t>((static_cast<uint64_t>(__umulhi(n, m)) + n) >> s);
  }
};

}  // namespace nvfp4
