// a5: decode attention straight from the NVFP4 KV cache (Sec. 2.1:
// z = softmax(Q K_hat^T / sqrt(d)) V_hat with quantized K and V).
//
// Split-KV ("flash-decoding"): CTA (split, kv_head, seq) owns a contiguous
// chunk of tokens; its 4 warps take interleaved 16-token tiles.  Each lane
// loads its FP4 codes with 128/64-bit coalesced loads, dequantizes them in
// registers (cvt e2m1x2 -> f16x2, times the E4M3 block scale, exact in f16)
// and feeds mma.sync m16n8k16 with fp32 accumulation:
//   S^T[16 tok x 8 head] = K_hat[16 tok x 128] . Q^T[128 x 8]   (8 MMAs)
//   O^T[128 x 8 head]   += V_hat^T[128 x 16 tok] . P^T[16 x 8]  (8 MMAs)
// The up to 8 query heads that share a KV head (grouped-query attention) fill
// the MMA's N = 8.  Softmax is online, in fp32, in the log2 domain.  The
// combine kernel merges the per-chunk (max, sum, O) partials.
//
// Lane roles (g = lane/4, t = lane%4), fixed by the m16n8k16 fragment layouts:
//   K: lane holds tokens g and g+8, channels 32t..32t+31 (16 bytes, blocks 2t, 2t+1)
//   V: lane holds tokens 2t, 2t+1, 2t+8, 2t+9, channels 16g..16g+15 (8 bytes, block g)
//   Q: lane holds head g, channels 32t..32t+31
// The contraction order of channels inside an MMA is permuted to match, which
// leaves the dot products unchanged.
#include <cfloat>

#include "common.cuh"

namespace nvfp4 {
namespace {

constexpr int kWarps = 4;
constexpr int kChunk = 1024;  // tokens per CTA
constexpr int kD = 128;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void mma16816(float c[4], const uint32_t a[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Four packed e2m1x2 bytes -> four f16x2 (low nibble -> low half).
__device__ __forceinline__ void e2m1x8_to_f16x2(uint32_t w, uint32_t h[4]) {
  asm("{\n .reg .b8 b0, b1, b2, b3;\n mov.b32 {b0, b1, b2, b3}, %4;\n"
      " cvt.rn.f16x2.e2m1x2 %0, b0;\n cvt.rn.f16x2.e2m1x2 %1, b1;\n"
      " cvt.rn.f16x2.e2m1x2 %2, b2;\n cvt.rn.f16x2.e2m1x2 %3, b3;\n}"
      : "=r"(h[0]), "=r"(h[1]), "=r"(h[2]), "=r"(h[3])
      : "r"(w));
}

// Two E4M3 bytes (low byte -> low half) -> f16x2, exact.
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two_bytes) {
  uint32_t h;
  asm("{\n .reg .b16 s;\n cvt.u16.u32 s, %1;\n cvt.rn.f16x2.e4m3x2 %0, s;\n}" : "=r"(h) : "r"(two_bytes));
  return h;
}

__device__ __forceinline__ uint32_t hmul2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

__device__ __forceinline__ uint32_t f32x2_to_f16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t bcast_lo(uint32_t x) { return __byte_perm(x, x, 0x1010); }
__device__ __forceinline__ uint32_t bcast_hi(uint32_t x) { return __byte_perm(x, x, 0x3232); }

struct TileData {
  uint4 ka, kb;        // K codes: token g, token g+8 (channels 32t..32t+31)
  uint32_t ksa, ksb;   // K scales (blocks 2t, 2t+1) of those tokens
  uint2 v[4];          // V codes: tokens 2t, 2t+1, 2t+8, 2t+9 (channels 16g..16g+15)
  uint32_t vs01, vs89; // V scales (block g): tokens (2t | 2t+1 << 8), (2t+8 | 2t+9 << 8)
};

__device__ __forceinline__ void load_tile(TileData& d, const uint8_t* __restrict__ kc, const uint8_t* __restrict__ ks,
                                          const uint8_t* __restrict__ vc, const uint8_t* __restrict__ vs, int tile,
                                          int t_end, int g, int t) {
  const int ta = tile + g, tb = tile + g + 8;
  const uint4 z4 = make_uint4(0, 0, 0, 0);
  d.ka = ta < t_end ? __ldg(reinterpret_cast<const uint4*>(kc + static_cast<size_t>(ta) * 64) + t) : z4;
  d.kb = tb < t_end ? __ldg(reinterpret_cast<const uint4*>(kc + static_cast<size_t>(tb) * 64) + t) : z4;
  d.ksa = ta < t_end ? __ldg(reinterpret_cast<const uint16_t*>(ks + static_cast<size_t>(ta) * 8) + t) : 0u;
  d.ksb = tb < t_end ? __ldg(reinterpret_cast<const uint16_t*>(ks + static_cast<size_t>(tb) * 8) + t) : 0u;
  const int toks[4] = {tile + 2 * t, tile + 2 * t + 1, tile + 2 * t + 8, tile + 2 * t + 9};
  uint32_t s[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const bool ok = toks[i] < t_end;
    d.v[i] = ok ? __ldg(reinterpret_cast<const uint2*>(vc + static_cast<size_t>(toks[i]) * 64) + g) : make_uint2(0, 0);
    s[i] = ok ? __ldg(vs + static_cast<size_t>(toks[i]) * 8 + g) : 0u;
  }
  d.vs01 = s[0] | (s[1] << 8);
  d.vs89 = s[2] | (s[3] << 8);
}

__global__ void __launch_bounds__(kWarps * 32) attn_partial_kernel(
    const uint8_t* __restrict__ k_codes, const uint8_t* __restrict__ k_scales, const uint8_t* __restrict__ v_codes,
    const uint8_t* __restrict__ v_scales, const int32_t* __restrict__ seq_lens, int hkv, int capacity,
    const uint16_t* __restrict__ q, int hq, int group, float logit_mult /* softmax_scale*g_K*log2(e) */,
    int n_splits, float* __restrict__ o_ws, float* __restrict__ ml_ws, int* status) {
  const int split = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;

  int seq_len = __ldg(seq_lens + b);
  if (seq_len > capacity) {
    if (split == 0 && kvh == 0 && threadIdx.x == 0) set_status(status, NVFP4_ERR_CAPACITY);
    seq_len = capacity;
  }
  if (seq_len < 0) seq_len = 0;
  const int t_begin = split * kChunk;
  const int t_end = min(t_begin + kChunk, seq_len);

  const size_t row0 = (static_cast<size_t>(b) * hkv + kvh) * capacity;
  const uint8_t* kc = k_codes + row0 * 64;
  const uint8_t* ks = k_scales + row0 * 8;
  const uint8_t* vc = v_codes + row0 * 64;
  const uint8_t* vs = v_scales + row0 * 8;

  // Queries of head slot g: f16 after an exact power-of-two scaling that keeps
  // |q| < 1; the scaling is undone in the logit multiplier.
  const bool head_live = g < group;
  const int hq_idx = kvh * group + g;
  float qv[32];
  {
    const uint4* qp = reinterpret_cast<const uint4*>(q + (static_cast<size_t>(b) * hq + hq_idx) * kD + 32 * t);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint4 w = head_live ? __ldg(qp + i) : make_uint4(0, 0, 0, 0);
      const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        qv[8 * i + 2 * k] = __uint_as_float(ws[k] << 16);
        qv[8 * i + 2 * k + 1] = __uint_as_float(ws[k] & 0xFFFF0000u);
      }
    }
  }
  float qmax = 0.0f;
#pragma unroll
  for (int i = 0; i < 32; ++i) qmax = fmaxf(qmax, fabsf(qv[i]));
  qmax = fmaxf(qmax, __shfl_xor_sync(0xffffffffu, qmax, 1));
  qmax = fmaxf(qmax, __shfl_xor_sync(0xffffffffu, qmax, 2));
  // 2^-(e+1) with qmax in [2^e, 2^(e+1)): scaled |q| < 1.
  const int qexp = qmax > 0.0f ? static_cast<int>((__float_as_uint(qmax) >> 23) & 0xFF) - 126 : 0;
  const float qscale = ldexpf(1.0f, -qexp);
  uint32_t qf[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) qf[i] = f32x2_to_f16x2(qv[2 * i] * qscale, qv[2 * i + 1] * qscale);
  // Logit multipliers of this lane's two S columns (head slots 2t, 2t+1).
  const float mult_self = logit_mult / qscale;
  const float mult0 = __shfl_sync(0xffffffffu, mult_self, (2 * t) * 4);
  const float mult1 = __shfl_sync(0xffffffffu, mult_self, (2 * t + 1) * 4);

  float o[8][4];
#pragma unroll
  for (int i = 0; i < 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.0f;
  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.0f, 0.0f};

  int tile = t_begin + warp * 16;
  TileData cur;
  if (tile < t_end) load_tile(cur, kc, ks, vc, vs, tile, t_end, g, t);
  for (; tile < t_end; tile += kWarps * 16) {
    TileData nxt;
    const int ntile = tile + kWarps * 16;
    if (ntile < t_end) load_tile(nxt, kc, ks, vc, vs, ntile, t_end, g, t);

    // ---- S^T = K_hat Q^T: 8 k-steps of 16 channels --------------------------
    const uint32_t ksa = e4m3x2_to_f16x2(cur.ksa), ksb = e4m3x2_to_f16x2(cur.ksb);
    const uint32_t sa_lo = bcast_lo(ksa), sa_hi = bcast_hi(ksa);
    const uint32_t sb_lo = bcast_lo(ksb), sb_hi = bcast_hi(ksb);
    float s[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    const uint32_t kaw[4] = {cur.ka.x, cur.ka.y, cur.ka.z, cur.ka.w};
    const uint32_t kbw[4] = {cur.kb.x, cur.kb.y, cur.kb.z, cur.kb.w};
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      uint32_t ha[4], hb[4];
      e2m1x8_to_f16x2(kaw[w], ha);
      e2m1x8_to_f16x2(kbw[w], hb);
      const uint32_t sa = w < 2 ? sa_lo : sa_hi, sb = w < 2 ? sb_lo : sb_hi;
#pragma unroll
      for (int h = 0; h < 2; ++h) {  // k-step j = 2w + h uses bytes 2j (low dims) and 2j+1
        const uint32_t a[4] = {hmul2(ha[2 * h], sa), hmul2(hb[2 * h], sb), hmul2(ha[2 * h + 1], sa),
                               hmul2(hb[2 * h + 1], sb)};
        const int j = 2 * w + h;
        mma16816(s, a, qf[2 * j], qf[2 * j + 1]);
      }
    }
    // ---- online softmax over this tile (log2 domain) ----------------------
    const bool va = tile + g < t_end, vb = tile + g + 8 < t_end;
    float x0 = va ? s[0] * mult0 : -INFINITY;  // token g,   head 2t
    float x1 = va ? s[1] * mult1 : -INFINITY;  // token g,   head 2t+1
    float x2 = vb ? s[2] * mult0 : -INFINITY;  // token g+8, head 2t
    float x3 = vb ? s[3] * mult1 : -INFINITY;  // token g+8, head 2t+1
    float mx0 = fmaxf(x0, x2), mx1 = fmaxf(x1, x3);
#pragma unroll
    for (int sh = 4; sh < 32; sh <<= 1) {
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, sh));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, sh));
    }
    const float mn0 = fmaxf(m_run[0], mx0), mn1 = fmaxf(m_run[1], mx1);  // finite: tile has a live token
    const float al0 = fast_exp2(m_run[0] - mn0), al1 = fast_exp2(m_run[1] - mn1);
    m_run[0] = mn0; m_run[1] = mn1;
    const float p0 = fast_exp2(x0 - mn0), p1 = fast_exp2(x1 - mn1);
    const float p2 = fast_exp2(x2 - mn0), p3 = fast_exp2(x3 - mn1);
    l_run[0] = l_run[0] * al0 + (p0 + p2);
    l_run[1] = l_run[1] * al1 + (p1 + p3);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      o[i][0] *= al0; o[i][1] *= al1; o[i][2] *= al0; o[i][3] *= al1;
    }
    // P^T fragments for the PV product: transpose the two 8x8 (token, head) blocks.
    const uint32_t pb0 = movmatrix_trans(f32x2_to_f16x2(p0, p1));
    const uint32_t pb1 = movmatrix_trans(f32x2_to_f16x2(p2, p3));

    // ---- O^T += V_hat^T P^T: 8 m-tiles, m-tile i = channels 16g+2i, 16g+2i+1
    const uint32_t vs01 = e4m3x2_to_f16x2(cur.vs01), vs89 = e4m3x2_to_f16x2(cur.vs89);
#pragma unroll
    for (int half = 0; half < 2; ++half) {  // bytes 0-3, then 4-7 of each token's 8-byte slice
      const uint32_t wa = half ? cur.v[0].y : cur.v[0].x, wb = half ? cur.v[1].y : cur.v[1].x;
      const uint32_t wc = half ? cur.v[2].y : cur.v[2].x, wd = half ? cur.v[3].y : cur.v[3].x;
      // Pair the same channel of two tokens in one e2m1x2 byte (token 2t in the low nibble).
      const uint32_t lo_ab = (wa & 0x0F0F0F0Fu) | ((wb << 4) & 0xF0F0F0F0u);
      const uint32_t hi_ab = ((wa >> 4) & 0x0F0F0F0Fu) | (wb & 0xF0F0F0F0u);
      const uint32_t lo_cd = (wc & 0x0F0F0F0Fu) | ((wd << 4) & 0xF0F0F0F0u);
      const uint32_t hi_cd = ((wc >> 4) & 0x0F0F0F0Fu) | (wd & 0xF0F0F0F0u);
      uint32_t f_lo_ab[4], f_hi_ab[4], f_lo_cd[4], f_hi_cd[4];
      e2m1x8_to_f16x2(lo_ab, f_lo_ab);
      e2m1x8_to_f16x2(hi_ab, f_hi_ab);
      e2m1x8_to_f16x2(lo_cd, f_lo_cd);
      e2m1x8_to_f16x2(hi_cd, f_hi_cd);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t a[4] = {hmul2(f_lo_ab[k], vs01), hmul2(f_hi_ab[k], vs01), hmul2(f_lo_cd[k], vs89),
                               hmul2(f_hi_cd[k], vs89)};
        mma16816(o[4 * half + k], a, pb0, pb1);
      }
    }
    if (ntile < t_end) cur = nxt;
  }

  // ---- merge the 4 warps of the CTA, write this chunk's partial -----------
  l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 4);
  l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 4);
  l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 8);
  l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 8);
  l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 16);
  l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 16);

  __shared__ float sh_o[kWarps][8][kD];
  __shared__ float sh_m[kWarps][8], sh_l[kWarps][8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int c0 = 16 * g + 2 * i;  // channel of accumulator rows g / g+8 of m-tile i
    sh_o[warp][2 * t][c0] = o[i][0];
    sh_o[warp][2 * t + 1][c0] = o[i][1];
    sh_o[warp][2 * t][c0 + 1] = o[i][2];
    sh_o[warp][2 * t + 1][c0 + 1] = o[i][3];
  }
  if (g == 0) {
    sh_m[warp][2 * t] = m_run[0]; sh_m[warp][2 * t + 1] = m_run[1];
    sh_l[warp][2 * t] = l_run[0]; sh_l[warp][2 * t + 1] = l_run[1];
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < group * kD; idx += kWarps * 32) {
    const int h = idx / kD, c = idx % kD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sh_m[w][h]);
    float acc = 0.0f, L = 0.0f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const float wt = fast_exp2(sh_m[w][h] - M);
        acc += wt * sh_o[w][h][c];
        L += wt * sh_l[w][h];
      }
    }
    const size_t rec = (static_cast<size_t>(b) * hq + kvh * group + h) * n_splits + split;
    o_ws[rec * kD + c] = acc;
    if (c == 0) {
      ml_ws[rec * 2] = M;
      ml_ws[rec * 2 + 1] = L;
    }
  }
}

// out[b, h] = g_V * sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s
__global__ void __launch_bounds__(kD) attn_combine_kernel(const float* __restrict__ o_ws,
                                                         const float* __restrict__ ml_ws, int n_splits, float gv,
                                                         uint16_t* __restrict__ out) {
  const size_t bh = static_cast<size_t>(blockIdx.y) * gridDim.x + blockIdx.x;
  const float* ml = ml_ws + bh * n_splits * 2;
  float M = -INFINITY;
  for (int s = 0; s < n_splits; ++s) M = fmaxf(M, __ldg(ml + 2 * s));
  float acc = 0.0f, L = 0.0f;
  if (M != -INFINITY) {
    for (int s = 0; s < n_splits; ++s) {
      const float w = fast_exp2(__ldg(ml + 2 * s) - M);
      L += w * __ldg(ml + 2 * s + 1);
      acc += w * __ldg(o_ws + (bh * n_splits + s) * kD + threadIdx.x);
    }
  }
  const float r = L > 0.0f ? __fdiv_rn(acc, L) * gv : 0.0f;
  uint16_t bits;
  asm("cvt.rn.bf16.f32 %0, %1;" : "=h"(bits) : "f"(r));
  out[bh * kD + threadIdx.x] = bits;
}

int splits_for(int capacity) { return (capacity + kChunk - 1) / kChunk; }

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API size_t decode_attention_nvfp4_workspace_size(int32_t batch, int32_t num_q_heads, int32_t capacity) {
  if (batch <= 0 || num_q_heads <= 0 || capacity <= 0) return 0;
  return static_cast<size_t>(batch) * num_q_heads * splits_for(capacity) * (kD + 2) * sizeof(float);
}

NVFP4_API nvfp4_status decode_attention_nvfp4(const nvfp4_kv_cache* cache, const void* q_bf16, int32_t num_q_heads,
                                              float softmax_scale, void* out_bf16, void* workspace,
                                              size_t workspace_bytes, void* stream) {
  if (!cache || !q_bf16 || !out_bf16 || !workspace || !cache->seq_lens) return NVFP4_ERR_INVALID_ARG;
  if (!cache->k_codes || !cache->k_scales || !cache->v_codes || !cache->v_scales) return NVFP4_ERR_INVALID_ARG;
  if (!(cache->k_gscale > 0.0f && cache->k_gscale <= FLT_MAX) || !(cache->v_gscale > 0.0f && cache->v_gscale <= FLT_MAX) ||
      !(softmax_scale > 0.0f && softmax_scale <= FLT_MAX))
    return NVFP4_ERR_INVALID_ARG;
  if (cache->head_dim != kD || cache->batch <= 0 || cache->num_kv_heads <= 0 || cache->capacity <= 0 ||
      num_q_heads <= 0 || num_q_heads % cache->num_kv_heads || num_q_heads / cache->num_kv_heads > 8)
    return NVFP4_ERR_SHAPE;
  if (static_cast<int64_t>(cache->batch) > 65535 || cache->num_kv_heads > 65535) return NVFP4_ERR_SHAPE;
  if (workspace_bytes < decode_attention_nvfp4_workspace_size(cache->batch, num_q_heads, cache->capacity))
    return NVFP4_ERR_SHAPE;
  if (!aligned(q_bf16, 16) || !aligned(out_bf16, 16) || !aligned(workspace, 16) || !aligned(cache->k_codes, 16) ||
      !aligned(cache->v_codes, 16) || !aligned(cache->k_scales, 8) || !aligned(cache->v_scales, 8))
    return NVFP4_ERR_ALIGN;
  const int group = num_q_heads / cache->num_kv_heads;
  const int n_splits = splits_for(cache->capacity);
  float* o_ws = static_cast<float*>(workspace);
  float* ml_ws = o_ws + static_cast<size_t>(cache->batch) * num_q_heads * n_splits * kD;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const dim3 grid(n_splits, cache->num_kv_heads, cache->batch);
  attn_partial_kernel<<<grid, kWarps * 32, 0, s>>>(
      cache->k_codes, cache->k_scales, cache->v_codes, cache->v_scales, cache->seq_lens, cache->num_kv_heads,
      cache->capacity, static_cast<const uint16_t*>(q_bf16), num_q_heads, group,
      softmax_scale * cache->k_gscale * kLog2e, n_splits, o_ws, ml_ws, status_word_dev());
  attn_combine_kernel<<<dim3(num_q_heads, cache->batch), kD, 0, s>>>(o_ws, ml_ws, n_splits, cache->v_gscale,
                                                                     static_cast<uint16_t*>(out_bf16));
  count_launches(2);
  return launch_status();
}
