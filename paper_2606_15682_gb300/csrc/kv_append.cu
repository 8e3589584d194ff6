// a4: quantize new K/V rows (optionally shifted by the Q-FIT post-RoPE vector
// m, Eq. 2) and write them into the NVFP4 KV cache; optionally rotate K by
// RoPE first (the fused RoPE -> shift -> quantize -> append step).
//
// Work item = one 8-element chunk of one 128-channel row; the 16 lanes that
// hold a row cover its 8 blocks.  Item order (token, kv head, K|V, chunk) keeps
// each warp's 512-byte bf16 read contiguous in the [n_new, H_kv, 128] inputs.
#include <cfloat>

#include "common.cuh"
#include "nvfp4_quant.cuh"

namespace nvfp4 {
namespace {

constexpr int kThreads = 256;

// kRope: K arrives before RoPE and is rotated here (rotate-half pairing,
// channel i with i + 64) with the (cos, sin) table row of its position, in
// fp32: y_i = x_i c_i - x_{i+64} s_i, y_{i+64} = x_i s_i + x_{i+64} c_i.
template <bool kRope, bool kE1M2>
__global__ void __launch_bounds__(kThreads) kv_append_kernel(
    const uint16_t* __restrict__ k_in, const uint16_t* __restrict__ v_in, const int32_t* __restrict__ seq_idx,
    const int32_t* __restrict__ pos, const float* __restrict__ k_shift, const float* __restrict__ rope,
    uint32_t n_rows /* n_new*H_kv */, FastDiv hkv, uint32_t batch, uint32_t capacity, uint8_t* __restrict__ kc,
    uint8_t* __restrict__ ks, uint8_t* __restrict__ vc, uint8_t* __restrict__ vs, float gk, float gv, int* status) {
  griddep_wait_and_release();
  const uint32_t total = n_rows * 32u;  // 2 tensors x 16 chunks per row: a multiple of the warp
  const uint32_t lane = threadIdx.x & 31;
  const float qmax = kE1M2 ? 3.5f : 6.0f;  // largest element magnitude of the grid
  const float six_gk = __fmul_rn(qmax, gk), six_gv = __fmul_rn(qmax, gv);
  for (uint32_t c0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31u); c0 < total; c0 += gridDim.x * blockDim.x) {
    const uint32_t c = c0 + lane;
    const bool live = c < total;
    const uint32_t j = c & 15u;          // chunk within the 128-channel row
    const bool is_v = (c >> 4) & 1u;
    const uint32_t rr = c >> 5;          // token * H_kv + head
    const uint32_t tok = hkv.div(rr);
    const uint32_t h = rr - tok * hkv.d;
    uint4 raw = make_uint4(0, 0, 0, 0);
    if (live) raw = __ldg(reinterpret_cast<const uint4*>((is_v ? v_in : k_in) + static_cast<uint64_t>(rr) * 128 + j * 8));
    float x[8];
    unpack_bf16x8(raw, x);
    if (kRope) {
      // The partner chunk (channels 64 apart) is held by lane ^ 8; the whole warp is live.
      uint4 pr;
      pr.x = __shfl_xor_sync(0xffffffffu, raw.x, 8);
      pr.y = __shfl_xor_sync(0xffffffffu, raw.y, 8);
      pr.z = __shfl_xor_sync(0xffffffffu, raw.z, 8);
      pr.w = __shfl_xor_sync(0xffffffffu, raw.w, 8);
      if (live && !is_v) {
        float xp[8];
        unpack_bf16x8(pr, xp);
        int32_t p = __ldg(pos + tok);
        if (p < 0 || static_cast<uint32_t>(p) >= capacity) p = 0;  // reported as CAPACITY below
        const float4* cs = reinterpret_cast<const float4*>(rope + (static_cast<uint64_t>(p) * 64 + (j & 7u) * 8) * 2);
        float cv[8], sv[8];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 t = __ldg(cs + q);
          cv[2 * q] = t.x; sv[2 * q] = t.y; cv[2 * q + 1] = t.z; sv[2 * q + 1] = t.w;
        }
#pragma unroll
        for (int e = 0; e < 8; ++e)
          x[e] = j < 8 ? __fsub_rn(__fmul_rn(x[e], cv[e]), __fmul_rn(xp[e], sv[e]))
                       : __fadd_rn(__fmul_rn(xp[e], sv[e]), __fmul_rn(x[e], cv[e]));
      }
    }
    if (live && !is_v && k_shift) {
      const float4* m4 = reinterpret_cast<const float4*>(k_shift + h * 128u + j * 8u);
      const float4 m0 = __ldg(m4), m1 = __ldg(m4 + 1);
      x[0] = __fsub_rn(x[0], m0.x); x[1] = __fsub_rn(x[1], m0.y);
      x[2] = __fsub_rn(x[2], m0.z); x[3] = __fsub_rn(x[3], m0.w);
      x[4] = __fsub_rn(x[4], m1.x); x[5] = __fsub_rn(x[5], m1.y);
      x[6] = __fsub_rn(x[6], m1.z); x[7] = __fsub_rn(x[7], m1.w);
    }
    float amax = 0.0f;
#pragma unroll
    for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(x[i]));
    uint32_t sc;
    const uint32_t packed = quantize8_pair<kE1M2>(x, amax, is_v ? gv : gk, is_v ? six_gv : six_gk, &sc);
    if (!live) continue;
    const int32_t b = __ldg(seq_idx + tok), p = __ldg(pos + tok);
    if (b < 0 || static_cast<uint32_t>(b) >= batch || p < 0 || static_cast<uint32_t>(p) >= capacity) {
      if (j == 0 && !is_v) set_status(status, NVFP4_ERR_CAPACITY);
      continue;
    }
    const uint64_t row = (static_cast<uint64_t>(b) * hkv.d + h) * capacity + static_cast<uint32_t>(p);
    if (!in_bounds(status, row < static_cast<uint64_t>(batch) * hkv.d * capacity && j < 16u)) continue;
    uint8_t* codes = is_v ? vc : kc;
    uint8_t* scales = is_v ? vs : ks;
    reinterpret_cast<uint32_t*>(codes + row * 64)[j] = packed;
    if ((j & 1u) == 0) scales[row * 8 + (j >> 1)] = static_cast<uint8_t>(sc);
  }
}

nvfp4_status append(const nvfp4_kv_cache* cache, const void* k_bf16, const void* v_bf16, const int32_t* seq_idx,
                    const int32_t* pos, int64_t n_new, const float* k_shift, const float* rope, void* stream) {
  if (!cache || !k_bf16 || !v_bf16 || !seq_idx || !pos) return NVFP4_ERR_INVALID_ARG;
  if (!cache->k_codes || !cache->k_scales || !cache->v_codes || !cache->v_scales) return NVFP4_ERR_INVALID_ARG;
  if (!(cache->k_gscale > 0.0f && cache->k_gscale <= FLT_MAX) || !(cache->v_gscale > 0.0f && cache->v_gscale <= FLT_MAX))
    return NVFP4_ERR_INVALID_ARG;
  if (cache->kv_format != NVFP4_KV_E2M1 && cache->kv_format != NVFP4_KV_E1M2) return NVFP4_ERR_INVALID_ARG;
  if (cache->head_dim != 128 || cache->batch <= 0 || cache->num_kv_heads <= 0 || cache->capacity <= 0 || n_new < 0)
    return NVFP4_ERR_SHAPE;
  if (n_new * cache->num_kv_heads * 32 >= (1ll << 32)) return NVFP4_ERR_SHAPE;
  if (!aligned(k_bf16, 16) || !aligned(v_bf16, 16) || !aligned(cache->k_codes, 16) || !aligned(cache->v_codes, 16) ||
      !aligned(cache->k_scales, 8) || !aligned(cache->v_scales, 8) || (k_shift && !aligned(k_shift, 16)) ||
      (rope && !aligned(rope, 16)))
    return NVFP4_ERR_ALIGN;
  if (n_new == 0) return NVFP4_OK;
  const uint32_t n_rows = static_cast<uint32_t>(n_new * cache->num_kv_heads);
  const uint64_t items = static_cast<uint64_t>(n_rows) * 32;
  uint64_t grid = (items + kThreads - 1) / kThreads;
  const uint64_t cap = static_cast<uint64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  const bool e1m2 = cache->kv_format == NVFP4_KV_E1M2;
  const auto kernel = rope ? (e1m2 ? kv_append_kernel<true, true> : kv_append_kernel<true, false>)
                           : (e1m2 ? kv_append_kernel<false, true> : kv_append_kernel<false, false>);
  const cudaError_t e =
      launch_pdl(kernel, dim3(static_cast<int>(grid)), dim3(kThreads),
                 0, static_cast<cudaStream_t>(stream), static_cast<const uint16_t*>(k_bf16),
                 static_cast<const uint16_t*>(v_bf16), seq_idx, pos, k_shift, rope, n_rows,
                 FastDiv(static_cast<uint32_t>(cache->num_kv_heads)), static_cast<uint32_t>(cache->batch),
                 static_cast<uint32_t>(cache->capacity), cache->k_codes, cache->k_scales, cache->v_codes,
                 cache->v_scales, cache->k_gscale, cache->v_gscale, status_word_dev());
  if (e != cudaSuccess) return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

// table[p][i] = (cos, sin) of p * theta^(-2i/d): angle, sine and cosine in
// fp64, each of the two results rounded once to fp32.
__global__ void rope_table_kernel(float2* __restrict__ table, uint32_t n_pos, uint32_t half, double theta, double d) {
  griddep_wait_and_release();
  const uint64_t n = static_cast<uint64_t>(n_pos) * half;
  for (uint64_t k = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; k < n;
       k += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint32_t p = static_cast<uint32_t>(k / half), i = static_cast<uint32_t>(k % half);
    const double inv = pow(theta, -2.0 * static_cast<double>(i) / d);
    double sn, cs;
    sincos(static_cast<double>(p) * inv, &sn, &cs);
    table[k] = make_float2(static_cast<float>(cs), static_cast<float>(sn));
  }
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API nvfp4_status kv_append_nvfp4(const nvfp4_kv_cache* cache, const void* k_bf16, const void* v_bf16,
                                       const int32_t* seq_idx, const int32_t* pos, int64_t n_new,
                                       const float* k_shift, void* stream) {
  NVFP4_TRACE("kv_append_nvfp4");
  return append(cache, k_bf16, v_bf16, seq_idx, pos, n_new, k_shift, nullptr, stream);
}

NVFP4_API nvfp4_status kv_append_rope_nvfp4(const nvfp4_kv_cache* cache, const void* k_pre_bf16, const void* v_bf16,
                                            const int32_t* seq_idx, const int32_t* pos, int64_t n_new,
                                            const float* rope_table, int64_t rope_positions, const float* k_shift,
                                            void* stream) {
  NVFP4_TRACE("kv_append_rope_nvfp4");
  if (!cache || !rope_table) return NVFP4_ERR_INVALID_ARG;
  if (rope_positions < cache->capacity) return NVFP4_ERR_SHAPE;
  return append(cache, k_pre_bf16, v_bf16, seq_idx, pos, n_new, k_shift, rope_table, stream);
}

NVFP4_API nvfp4_status nvfp4_rope_table(float* table, int64_t n_pos, int32_t head_dim, float theta, void* stream) {
  NVFP4_TRACE("nvfp4_rope_table");
  if (n_pos < 0 || head_dim <= 0 || head_dim % 2 || n_pos * (head_dim / 2) >= (1ll << 40)) return NVFP4_ERR_SHAPE;
  if (!(theta > 1.0f && theta <= FLT_MAX)) return NVFP4_ERR_INVALID_ARG;
  if (n_pos == 0) return NVFP4_OK;
  if (!table) return NVFP4_ERR_INVALID_ARG;
  if (!aligned(table, 8)) return NVFP4_ERR_ALIGN;
  const uint64_t n = static_cast<uint64_t>(n_pos) * (head_dim / 2);
  uint64_t grid = (n + 255) / 256;
  const uint64_t cap = static_cast<uint64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  if (launch_pdl(rope_table_kernel, dim3(static_cast<int>(grid)), dim3(256), 0, static_cast<cudaStream_t>(stream),
                 reinterpret_cast<float2*>(table), static_cast<uint32_t>(n_pos), static_cast<uint32_t>(head_dim / 2),
                 static_cast<double>(theta), static_cast<double>(head_dim)) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}
