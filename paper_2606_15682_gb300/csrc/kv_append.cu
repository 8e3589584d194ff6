// a4: quantize new K/V rows (optionally shifted by the Q-FIT post-RoPE vector
// m, Eq. 2) and write them into the NVFP4 KV cache; optionally rotate K by
// RoPE first (the fused RoPE -> shift -> quantize -> append step).
//
// Work item = one 16-element block of one 128-channel row (one thread per
// block: the block scale is computed once).  Item order (token, kv head, K|V,
// block) keeps each warp's reads contiguous in the [n_new, H_kv, 128] inputs.
#include <cfloat>

#include "common.cuh"
#include "nvfp4_quant.cuh"

namespace nvfp4 {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;  // items (16-element blocks) per thread per pass

// kRope: K arrives before RoPE and is rotated here (rotate-half pairing,
// channel i with i + 64) with the (cos, sin) table row of its position, in
// fp32: y_i = x_i c_i - x_{i+64} s_i, y_{i+64} = x_i s_i + x_{i+64} c_i.
//
// Work item = one 16-element block of one row (row = token, KV head, K or V):
// 16 items per (token, head), so a warp covers two.  Lane l of a warp takes
// (token-head 2w + l/16, K or V by bit 3, block l % 8); the RoPE partner block
// (channels 64 apart) is on lane l ^ 4.  kUnroll items per thread per pass,
// all their loads issued first.
template <bool kRope, bool kE1M2>
__global__ void __launch_bounds__(kThreads) kv_append_kernel(
    const uint16_t* __restrict__ k_in, const uint16_t* __restrict__ v_in, const int32_t* __restrict__ seq_idx,
    const int32_t* __restrict__ pos, const float* __restrict__ k_shift, const float* __restrict__ rope,
    uint32_t n_rows /* n_new*H_kv */, FastDiv hkv, uint32_t batch, uint32_t capacity, uint8_t* __restrict__ kc,
    uint8_t* __restrict__ ks, uint8_t* __restrict__ vc, uint8_t* __restrict__ vs, float gk, float gv, int* status) {
  griddep_wait_and_release();
  const uint32_t total = n_rows * 16u;  // 2 tensors x 8 blocks per row: a multiple of the warp
  const uint32_t lane = threadIdx.x & 31;
  const float qmax = kE1M2 ? 3.5f : 6.0f;  // largest element magnitude of the grid
  const float six_gk = __fmul_rn(qmax, gk), six_gv = __fmul_rn(qmax, gv);
  const uint32_t stride = gridDim.x * blockDim.x;
  // Item indices are formed in 64 bits: a pass may reach past 2^32 near the end.
  for (uint64_t c00 = blockIdx.x * blockDim.x + (threadIdx.x & ~31u); c00 < total;
       c00 += static_cast<uint64_t>(stride) * kUnroll) {
    uint4 lo[kUnroll], hi[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint64_t c = c00 + static_cast<uint64_t>(u) * stride + lane;
      const uint32_t rr = static_cast<uint32_t>(c >> 4);
      const bool is_v = (c >> 3) & 1u;
      const uint4* src = reinterpret_cast<const uint4*>((is_v ? v_in : k_in) + static_cast<uint64_t>(rr) * 128 +
                                                        (c & 7u) * 16);
      const bool in = c < total;
      lo[u] = in ? __ldg(src) : make_uint4(0, 0, 0, 0);
      hi[u] = in ? __ldg(src + 1) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint64_t c0 = c00 + static_cast<uint64_t>(u) * stride;
      if (c0 >= total) continue;  // warp-uniform: c0 is the warp's first item
      const uint32_t c = static_cast<uint32_t>(c0) + lane;  // c0 < total < 2^32
      const bool live = c < total;         // an odd row count leaves half of the last warp idle
      const uint32_t blk = c & 7u;         // block within the 128-channel row
      const bool is_v = (c >> 3) & 1u;
      const uint32_t rr = c >> 4;          // token * H_kv + head
      const uint32_t tok = hkv.div(rr);
      const uint32_t h = rr - tok * hkv.d;
      float x[16];
      unpack_bf16x8(lo[u], x);
      unpack_bf16x8(hi[u], x + 8);
      if (kRope) {
        // The partner block (channels 64 apart) is on lane ^ 4; every lane of the warp is live.
        uint4 plo, phi;
        plo.x = __shfl_xor_sync(0xffffffffu, lo[u].x, 4);
        plo.y = __shfl_xor_sync(0xffffffffu, lo[u].y, 4);
        plo.z = __shfl_xor_sync(0xffffffffu, lo[u].z, 4);
        plo.w = __shfl_xor_sync(0xffffffffu, lo[u].w, 4);
        phi.x = __shfl_xor_sync(0xffffffffu, hi[u].x, 4);
        phi.y = __shfl_xor_sync(0xffffffffu, hi[u].y, 4);
        phi.z = __shfl_xor_sync(0xffffffffu, hi[u].z, 4);
        phi.w = __shfl_xor_sync(0xffffffffu, hi[u].w, 4);
        if (live && !is_v) {
          float xp[16];
          unpack_bf16x8(plo, xp);
          unpack_bf16x8(phi, xp + 8);
          int32_t p = __ldg(pos + tok);
          if (p < 0 || static_cast<uint32_t>(p) >= capacity) p = 0;  // reported as CAPACITY below
          const float4* cs =
              reinterpret_cast<const float4*>(rope + (static_cast<uint64_t>(p) * 64 + (blk & 3u) * 16) * 2);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float4 t = __ldg(cs + q);
            const float cv0 = t.x, sv0 = t.y, cv1 = t.z, sv1 = t.w;
            const int e = 2 * q;
            x[e] = blk < 4 ? __fsub_rn(__fmul_rn(x[e], cv0), __fmul_rn(xp[e], sv0))
                           : __fadd_rn(__fmul_rn(xp[e], sv0), __fmul_rn(x[e], cv0));
            x[e + 1] = blk < 4 ? __fsub_rn(__fmul_rn(x[e + 1], cv1), __fmul_rn(xp[e + 1], sv1))
                               : __fadd_rn(__fmul_rn(xp[e + 1], sv1), __fmul_rn(x[e + 1], cv1));
          }
        }
      }
      if (live && !is_v && k_shift) {
        const float4* m4 = reinterpret_cast<const float4*>(k_shift + h * 128u + blk * 16u);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 m = __ldg(m4 + q);
          x[4 * q] = __fsub_rn(x[4 * q], m.x);
          x[4 * q + 1] = __fsub_rn(x[4 * q + 1], m.y);
          x[4 * q + 2] = __fsub_rn(x[4 * q + 2], m.z);
          x[4 * q + 3] = __fsub_rn(x[4 * q + 3], m.w);
        }
      }
      float amax = 0.0f;
#pragma unroll
      for (int i = 0; i < 16; ++i) amax = fmaxf(amax, fabsf(x[i]));
      const BlockScale bs = block_scale(amax, is_v ? gv : gk, is_v ? six_gv : six_gk);
#pragma unroll
      for (int i = 0; i < 16; ++i) x[i] = __fmul_rn(x[i], bs.mult);
      const uint2 packed = kE1M2 ? make_uint2(e1m2x8(x), e1m2x8(x + 8)) : make_uint2(e2m1x8(x), e2m1x8(x + 8));
      if (!live) continue;
      const int32_t b = __ldg(seq_idx + tok), p = __ldg(pos + tok);
      if (b < 0 || static_cast<uint32_t>(b) >= batch || p < 0 || static_cast<uint32_t>(p) >= capacity) {
        if (blk == 0 && !is_v) set_status(status, NVFP4_ERR_CAPACITY);
        continue;
      }
      const uint64_t row = (static_cast<uint64_t>(b) * hkv.d + h) * capacity + static_cast<uint32_t>(p);
      if (!in_bounds(status, row < static_cast<uint64_t>(batch) * hkv.d * capacity && blk < 8u)) continue;
      reinterpret_cast<uint2*>((is_v ? vc : kc) + row * 64)[blk] = packed;
      (is_v ? vs : ks)[row * 8 + blk] = static_cast<uint8_t>(bs.code);
    }
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
  const uint64_t items = static_cast<uint64_t>(n_rows) * 16;
  uint64_t grid = (items + kThreads * kUnroll - 1) / (kThreads * kUnroll);
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
