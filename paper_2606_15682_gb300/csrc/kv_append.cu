// a4: quantize new K/V rows (optionally shifted by the Q-FIT post-RoPE vector
// m, Eq. 2) and write them into the NVFP4 KV cache.
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

__global__ void __launch_bounds__(kThreads) kv_append_kernel(
    const uint16_t* __restrict__ k_in, const uint16_t* __restrict__ v_in, const int32_t* __restrict__ seq_idx,
    const int32_t* __restrict__ pos, const float* __restrict__ k_shift, uint32_t n_rows /* n_new*H_kv */,
    FastDiv hkv, uint32_t batch, uint32_t capacity, uint8_t* __restrict__ kc, uint8_t* __restrict__ ks,
    uint8_t* __restrict__ vc, uint8_t* __restrict__ vs, float gk, float gv, int* status) {
  const uint32_t total = n_rows * 32u;  // 2 tensors x 16 chunks per row
  const uint32_t lane = threadIdx.x & 31;
  const float six_gk = __fmul_rn(6.0f, gk), six_gv = __fmul_rn(6.0f, gv);
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
    const uint32_t packed = quantize8_pair(x, amax, is_v ? gv : gk, is_v ? six_gv : six_gk, &sc);
    if (!live) continue;
    const int32_t b = __ldg(seq_idx + tok), p = __ldg(pos + tok);
    if (b < 0 || static_cast<uint32_t>(b) >= batch || p < 0 || static_cast<uint32_t>(p) >= capacity) {
      if (j == 0 && !is_v) set_status(status, NVFP4_ERR_CAPACITY);
      continue;
    }
    const uint64_t row = (static_cast<uint64_t>(b) * hkv.d + h) * capacity + static_cast<uint32_t>(p);
    uint8_t* codes = is_v ? vc : kc;
    uint8_t* scales = is_v ? vs : ks;
    reinterpret_cast<uint32_t*>(codes + row * 64)[j] = packed;
    if ((j & 1u) == 0) scales[row * 8 + (j >> 1)] = static_cast<uint8_t>(sc);
  }
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API nvfp4_status kv_append_nvfp4(const nvfp4_kv_cache* cache, const void* k_bf16, const void* v_bf16,
                                       const int32_t* seq_idx, const int32_t* pos, int64_t n_new,
                                       const float* k_shift, void* stream) {
  if (!cache || !k_bf16 || !v_bf16 || !seq_idx || !pos) return NVFP4_ERR_INVALID_ARG;
  if (!cache->k_codes || !cache->k_scales || !cache->v_codes || !cache->v_scales) return NVFP4_ERR_INVALID_ARG;
  if (!(cache->k_gscale > 0.0f && cache->k_gscale <= FLT_MAX) || !(cache->v_gscale > 0.0f && cache->v_gscale <= FLT_MAX))
    return NVFP4_ERR_INVALID_ARG;
  if (cache->head_dim != 128 || cache->batch <= 0 || cache->num_kv_heads <= 0 || cache->capacity <= 0 || n_new < 0)
    return NVFP4_ERR_SHAPE;
  if (n_new * cache->num_kv_heads * 32 >= (1ll << 32)) return NVFP4_ERR_SHAPE;
  if (!aligned(k_bf16, 16) || !aligned(v_bf16, 16) || !aligned(cache->k_codes, 16) || !aligned(cache->v_codes, 16) ||
      !aligned(cache->k_scales, 8) || !aligned(cache->v_scales, 8) || (k_shift && !aligned(k_shift, 16)))
    return NVFP4_ERR_ALIGN;
  if (n_new == 0) return NVFP4_OK;
  const uint32_t n_rows = static_cast<uint32_t>(n_new * cache->num_kv_heads);
  const uint64_t items = static_cast<uint64_t>(n_rows) * 32;
  uint64_t grid = (items + kThreads - 1) / kThreads;
  const uint64_t cap = static_cast<uint64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  if (launch_pdl(kv_append_kernel, dim3(static_cast<int>(grid)), dim3(kThreads), 0, static_cast<cudaStream_t>(stream),
                 static_cast<const uint16_t*>(k_bf16), static_cast<const uint16_t*>(v_bf16), seq_idx, pos, k_shift,
                 n_rows, FastDiv(static_cast<uint32_t>(cache->num_kv_heads)), static_cast<uint32_t>(cache->batch),
                 static_cast<uint32_t>(cache->capacity), cache->k_codes, cache->k_scales, cache->v_codes,
                 cache->v_scales, cache->k_gscale, cache->v_gscale, status_word_dev()) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}
