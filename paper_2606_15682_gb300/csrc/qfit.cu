// f4: Q-FIT calibration (Algorithm 1) on the GPU.
//
// Chooses the paired pre-RoPE scale S (S_Q for the query heads, S_K for the
// KV heads) and the post-RoPE key shift m of Eq. 2 by a grid search over
// (alpha_s, alpha_m): S = S0^alpha_s, S0 the pair-shared key magnitudes;
// m = alpha_m * mu, mu the token mean of RoPE(K_pre).  Each grid point is
// scored by the mean squared difference between the unquantized attention
// Y_ref and the attention over the KV4 cache.  The calibration set is B
// sequences of T tokens; the causal attention is scored at the last token of
// every sequence (it attends to the whole sequence: one decode step over the
// cached sequence).  Per grid point the library's own kernels build the KV4
// cache (kv_append_rope_nvfp4: RoPE, minus m, NVFP4 or E1M2 quantization) and
// attend over it (decode_attention_nvfp4); the kernels below compute S0, mu,
// Y_ref, the grid point's keys and queries, and the error.
//
// Arithmetic that decides a quantized code follows the oracle's order in fp32
// (round to nearest even, no fused multiply-add): K_pre / S_K rounded to bf16,
// RoPE from the (cos, sin) table as y1 = x1 c - x2 s, y2 = x1 s + x2 c, then
// minus m; the static scale amax / (qmax * 448).  Y_ref and the error are
// accumulated in fp32 and fp64.
#include <cuda_bf16.h>

#include <cfloat>
#include <cmath>
#include <cstring>
#include <vector>

#include "common.cuh"

namespace nvfp4 {
namespace {

constexpr int kD = 128, kHalf = 64;
constexpr int kMaxTokens = 8192;  // logits of one sequence in shared memory (32 KB)
constexpr int kMaxGrid = 64;

__device__ __forceinline__ float bf16_bits_to_f32(uint16_t b) { return __uint_as_float(static_cast<uint32_t>(b) << 16); }
__device__ __forceinline__ uint16_t f32_to_bf16_bits(float x) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

// RoPE of the channel pair (r, r + 64) at position p from the fp32 (cos, sin) table.
__device__ __forceinline__ void rope_pair(float x1, float x2, const float* __restrict__ table, int p, int r,
                                          float* y1, float* y2) {
  const float2 cs = *reinterpret_cast<const float2*>(table + (static_cast<size_t>(p) * kHalf + r) * 2);
  *y1 = __fsub_rn(__fmul_rn(x1, cs.x), __fmul_rn(x2, cs.y));
  *y2 = __fadd_rn(__fmul_rn(x1, cs.y), __fmul_rn(x2, cs.x));
}

// Algorithm 1's initialization, one block per KV head, one thread per channel
// pair r: S0[h, r] = S0[h, r + 64] = max(max_t |K[t,h,r]|, max_t |K[t,h,r+64]|, eps)
// and mu[h, c] = mean_t RoPE(K_pre)[t, h, c] over all n_tok tokens (token i of
// the flattened [B, T] set sits at position i % T).
__global__ void qfit_init_kernel(const uint16_t* __restrict__ k, int n_tok, int T, int hkv,
                                 const float* __restrict__ table, double eps, double* __restrict__ s0,
                                 double* __restrict__ mu) {
  griddep_wait_and_release();
  const int h = blockIdx.x, r = threadIdx.x;
  float amax = 0.0f;
  double sum1 = 0.0, sum2 = 0.0;
  for (int i = 0; i < n_tok; ++i) {
    const size_t base = (static_cast<size_t>(i) * hkv + h) * kD;
    const float x1 = bf16_bits_to_f32(k[base + r]), x2 = bf16_bits_to_f32(k[base + r + kHalf]);
    amax = fmaxf(amax, fmaxf(fabsf(x1), fabsf(x2)));
    float y1, y2;
    rope_pair(x1, x2, table, i % T, r, &y1, &y2);
    sum1 += y1;
    sum2 += y2;
  }
  const double s = fmax(static_cast<double>(amax), eps);
  s0[h * kD + r] = s;
  s0[h * kD + r + kHalf] = s;
  mu[h * kD + r] = sum1 / n_tok;
  mu[h * kD + r + kHalf] = sum2 / n_tok;
}

// Y_ref[b, h] = softmax(scale * q0 . RoPE(K_b)^T) V_b for the last token of
// sequence b (fp32), q0 = RoPE(Q_pre[b, T-1, h]).  One block of 128 threads
// per (query head, sequence); the T logits live in shared memory.
__global__ void __launch_bounds__(kD) qfit_reference_kernel(const uint16_t* __restrict__ q,
                                                            const uint16_t* __restrict__ k,
                                                            const uint16_t* __restrict__ v, int T, int hq, int hkv,
                                                            const float* __restrict__ table, float scale,
                                                            float* __restrict__ y_ref) {
  griddep_wait_and_release();
  extern __shared__ float logits[];
  __shared__ float q0[kD];
  __shared__ float red[kD / 32];
  const int h = blockIdx.x, b = blockIdx.y, kv = h / (hq / hkv);
  const int c = threadIdx.x, warp = c >> 5, lane = c & 31;
  {
    const size_t qb = ((static_cast<size_t>(b) * T + (T - 1)) * hq + h) * kD;
    const int r = c & (kHalf - 1);
    float y1, y2;
    rope_pair(bf16_bits_to_f32(q[qb + r]), bf16_bits_to_f32(q[qb + r + kHalf]), table, T - 1, r, &y1, &y2);
    q0[c] = c < kHalf ? y1 : y2;
  }
  __syncthreads();
  // Logits: one warp per token, each lane the pairs (lane, lane + 64) and (lane + 32, lane + 96).
  for (int t = warp; t < T; t += kD / 32) {
    const size_t kb = ((static_cast<size_t>(b) * T + t) * hkv + kv) * kD;
    float dot = 0.0f;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int r = lane + 32 * j;
      float y1, y2;
      rope_pair(bf16_bits_to_f32(k[kb + r]), bf16_bits_to_f32(k[kb + r + kHalf]), table, t, r, &y1, &y2);
      dot = fmaf(q0[r], y1, dot);
      dot = fmaf(q0[r + kHalf], y2, dot);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    if (lane == 0) logits[t] = dot * scale;
  }
  __syncthreads();
  float mx = -FLT_MAX;
  for (int t = c; t < T; t += kD) mx = fmaxf(mx, logits[t]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if (lane == 0) red[warp] = mx;
  __syncthreads();
  mx = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
  __syncthreads();
  float sum = 0.0f;
  for (int t = c; t < T; t += kD) {
    const float p = __expf(logits[t] - mx);
    logits[t] = p;
    sum += p;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  if (lane == 0) red[warp] = sum;
  __syncthreads();
  sum = red[0] + red[1] + red[2] + red[3];
  float acc = 0.0f;
  for (int t = 0; t < T; ++t)
    acc = fmaf(logits[t], bf16_bits_to_f32(v[((static_cast<size_t>(b) * T + t) * hkv + kv) * kD + c]), acc);
  y_ref[(static_cast<size_t>(b) * hq + h) * kD + c] = acc / sum;
}

// amax |x| over n bf16 values, max-reduced into *amax_bits (fp32 bits, non-negative).
__global__ void qfit_amax_kernel(const uint16_t* __restrict__ x, size_t n, uint32_t* __restrict__ amax_bits) {
  griddep_wait_and_release();
  float m = 0.0f;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x)
    m = fmaxf(m, fabsf(bf16_bits_to_f32(x[i])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0 && m > 0.0f) atomicMax(amax_bits, __float_as_uint(m));
}

// One grid point's transformation: S_K = fp32(S0^alpha_s), S_Q its copy for
// each query head of the group, m = fp32(alpha_m * mu).
__global__ void qfit_params_kernel(const double* __restrict__ s0, const double* __restrict__ mu, double alpha_s,
                                   double alpha_m, int hq, int hkv, float* __restrict__ s_q, float* __restrict__ s_k,
                                   float* __restrict__ m) {
  griddep_wait_and_release();
  const int group = hq / hkv;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < hq * kD; i += gridDim.x * blockDim.x) {
    const int h = i / kD, c = i % kD, kvc = (h / group) * kD + c;
    const float s = static_cast<float>(pow(s0[kvc], alpha_s));
    s_q[i] = s;
    if (h % group == 0) {
      s_k[kvc] = s;
      m[kvc] = static_cast<float>(alpha_m * mu[kvc]);
    }
  }
}

// The grid point's cached keys before RoPE, bf16(K_pre / S_K), and the amax of
// RoPE(bf16(K_pre / S_K)) - m over all of them (for the static key scale).
// One thread per (token, KV head, channel pair).
__global__ void qfit_keys_kernel(const uint16_t* __restrict__ k, int n_tok, int T, int hkv,
                                 const float* __restrict__ table, const float* __restrict__ s_k,
                                 const float* __restrict__ m, uint16_t* __restrict__ k_in,
                                 uint32_t* __restrict__ amax_bits) {
  griddep_wait_and_release();
  const size_t n = static_cast<size_t>(n_tok) * hkv * kHalf;
  float amax = 0.0f;
  for (size_t j = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; j < n;
       j += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int r = static_cast<int>(j % kHalf);
    const size_t th = j / kHalf;  // token * hkv + head
    const int h = static_cast<int>(th % hkv), i = static_cast<int>(th / hkv);
    const size_t base = th * kD;
    const uint16_t b1 = f32_to_bf16_bits(__fdiv_rn(bf16_bits_to_f32(k[base + r]), s_k[h * kD + r]));
    const uint16_t b2 = f32_to_bf16_bits(__fdiv_rn(bf16_bits_to_f32(k[base + r + kHalf]), s_k[h * kD + r + kHalf]));
    k_in[base + r] = b1;
    k_in[base + r + kHalf] = b2;
    float y1, y2;
    rope_pair(bf16_bits_to_f32(b1), bf16_bits_to_f32(b2), table, i % T, r, &y1, &y2);
    amax = fmaxf(amax, fmaxf(fabsf(__fsub_rn(y1, m[h * kD + r])), fabsf(__fsub_rn(y2, m[h * kD + r + kHalf]))));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  if ((threadIdx.x & 31) == 0 && amax > 0.0f) atomicMax(amax_bits, __float_as_uint(amax));
}

// The grid point's queries: bf16(RoPE(Q_pre[b, T-1, h] * S_Q[h])) at position T - 1.
__global__ void qfit_queries_kernel(const uint16_t* __restrict__ q, int B, int T, int hq,
                                    const float* __restrict__ table, const float* __restrict__ s_q,
                                    uint16_t* __restrict__ q_t) {
  griddep_wait_and_release();
  const int n = B * hq * kHalf;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < n; j += gridDim.x * blockDim.x) {
    const int r = j % kHalf, bh = j / kHalf, h = bh % hq, b = bh / hq;
    const size_t src = ((static_cast<size_t>(b) * T + (T - 1)) * hq + h) * kD;
    const float x1 = __fmul_rn(bf16_bits_to_f32(q[src + r]), s_q[h * kD + r]);
    const float x2 = __fmul_rn(bf16_bits_to_f32(q[src + r + kHalf]), s_q[h * kD + r + kHalf]);
    float y1, y2;
    rope_pair(x1, x2, table, T - 1, r, &y1, &y2);
    q_t[static_cast<size_t>(bh) * kD + r] = f32_to_bf16_bits(y1);
    q_t[static_cast<size_t>(bh) * kD + r + kHalf] = f32_to_bf16_bits(y2);
  }
}

// *err = mean((out - y_ref)^2) over n values, accumulated in fp64 (one block).
__global__ void __launch_bounds__(1024) qfit_mse_kernel(const uint16_t* __restrict__ out,
                                                        const float* __restrict__ y_ref, int n,
                                                        double* __restrict__ err) {
  griddep_wait_and_release();
  __shared__ double red[32];
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const double d = static_cast<double>(bf16_bits_to_f32(out[i])) - static_cast<double>(y_ref[i]);
    s += d * d;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    s = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (threadIdx.x == 0) *err = s / n;
  }
}

__global__ void qfit_fill_indices_kernel(int B, int T, int32_t* __restrict__ seq_idx, int32_t* __restrict__ pos,
                                         int32_t* __restrict__ seq_lens) {
  griddep_wait_and_release();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < B * T; i += gridDim.x * blockDim.x) {
    seq_idx[i] = i / T;
    pos[i] = i % T;
    if (i < B) seq_lens[i] = T;
  }
}

// Workspace carve-up (every part 256-byte aligned).
struct QfitWorkspace {
  uint8_t *kc, *ks, *vc, *vs;
  int32_t *seq_lens, *seq_idx, *pos;
  uint16_t *k_in, *q_t, *out;
  float* y_ref;
  double *s0, *mu;
  float *s_q, *s_k, *m;
  uint32_t* amax;  // [0] keys of the current grid point, [1] values
  double* err;
  void* attn_ws;
  size_t attn_ws_bytes;
  size_t total;
};

QfitWorkspace qfit_layout(uint8_t* base, int B, int T, int hq, int hkv, int grid_points) {
  QfitWorkspace w{};
  const int cap = T + (T & 1);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    uint8_t* p = base ? base + off : nullptr;
    off += (bytes + 255) & ~static_cast<size_t>(255);
    return p;
  };
  const size_t rows = static_cast<size_t>(B) * hkv * cap;
  w.kc = take(rows * 64);
  w.ks = take(rows * 8);
  w.vc = take(rows * 64);
  w.vs = take(rows * 8);
  w.seq_lens = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * B));
  w.seq_idx = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * B * T));
  w.pos = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * B * T));
  w.k_in = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * B * T * hkv * kD));
  w.q_t = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * B * hq * kD));
  w.out = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * B * hq * kD));
  w.y_ref = reinterpret_cast<float*>(take(sizeof(float) * B * hq * kD));
  w.s0 = reinterpret_cast<double*>(take(sizeof(double) * hkv * kD));
  w.mu = reinterpret_cast<double*>(take(sizeof(double) * hkv * kD));
  w.s_q = reinterpret_cast<float*>(take(sizeof(float) * hq * kD));
  w.s_k = reinterpret_cast<float*>(take(sizeof(float) * hkv * kD));
  w.m = reinterpret_cast<float*>(take(sizeof(float) * hkv * kD));
  w.amax = reinterpret_cast<uint32_t*>(take(2 * sizeof(uint32_t)));
  w.err = reinterpret_cast<double*>(take(sizeof(double) * grid_points));
  w.attn_ws_bytes = decode_attention_nvfp4_workspace_size(B, hq, cap);
  w.attn_ws = take(w.attn_ws_bytes);
  w.total = off;
  return w;
}

bool qfit_shape_ok(int B, int T, int hq, int hkv, int head_dim) {
  return B > 0 && T > 0 && T <= kMaxTokens && hq > 0 && hkv > 0 && hq % hkv == 0 && hq / hkv <= 8 &&
         head_dim == kD && static_cast<int64_t>(B) * T <= (1 << 24) && B <= 65535 && hq <= 65535;
}

int blocks_for(size_t n, int threads) {
  const size_t want = (n + threads - 1) / threads, cap = static_cast<size_t>(sm_count()) * 8;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API size_t nvfp4_qfit_workspace_size(int32_t batch, int32_t tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                           int32_t grid_s, int32_t grid_m) {
  if (!qfit_shape_ok(batch, tokens, num_q_heads, num_kv_heads, kD) || grid_s <= 0 || grid_m <= 0 ||
      grid_s > kMaxGrid || grid_m > kMaxGrid)
    return 0;
  return qfit_layout(nullptr, batch, tokens, num_q_heads, num_kv_heads, grid_s * grid_m).total;
}

NVFP4_API nvfp4_status nvfp4_qfit_calibrate(const void* q_pre_bf16, const void* k_pre_bf16, const void* v_bf16,
                                            int32_t batch, int32_t tokens, int32_t num_q_heads,
                                            int32_t num_kv_heads, int32_t head_dim, const float* rope_table,
                                            int64_t rope_positions, int32_t grid_s, int32_t grid_m, double eps,
                                            int32_t kv_format, float* s_q, float* s_k, float* m,
                                            double* errors_host, void* workspace, size_t workspace_bytes,
                                            void* stream) {
  NVFP4_TRACE("nvfp4_qfit_calibrate");
  if (!q_pre_bf16 || !k_pre_bf16 || !v_bf16 || !rope_table || !s_q || !s_k || !m || !workspace)
    return NVFP4_ERR_INVALID_ARG;
  if (kv_format != NVFP4_KV_E2M1 && kv_format != NVFP4_KV_E1M2) return NVFP4_ERR_INVALID_ARG;
  if (!(eps > 0.0) || !std::isfinite(eps)) return NVFP4_ERR_INVALID_ARG;
  if (!qfit_shape_ok(batch, tokens, num_q_heads, num_kv_heads, head_dim)) return NVFP4_ERR_SHAPE;
  if (grid_s <= 0 || grid_m <= 0 || grid_s > kMaxGrid || grid_m > kMaxGrid) return NVFP4_ERR_SHAPE;
  const int B = batch, T = tokens, hq = num_q_heads, hkv = num_kv_heads, cap = T + (T & 1);
  if (rope_positions < cap) return NVFP4_ERR_SHAPE;
  const int points = grid_s * grid_m;
  if (workspace_bytes < qfit_layout(nullptr, B, T, hq, hkv, points).total) return NVFP4_ERR_SHAPE;
  if (!aligned(q_pre_bf16, 16) || !aligned(k_pre_bf16, 16) || !aligned(v_bf16, 16) || !aligned(rope_table, 16) ||
      !aligned(workspace, 256) || !aligned(s_q, 4) || !aligned(s_k, 4) || !aligned(m, 4))
    return NVFP4_ERR_ALIGN;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const QfitWorkspace w = qfit_layout(static_cast<uint8_t*>(workspace), B, T, hq, hkv, points);
  const auto* q = static_cast<const uint16_t*>(q_pre_bf16);
  const auto* k = static_cast<const uint16_t*>(k_pre_bf16);
  const auto* v = static_cast<const uint16_t*>(v_bf16);
  const int n_tok = B * T;
  const float qmax_448 = kv_format == NVFP4_KV_E2M1 ? 6.0f * 448.0f : 3.5f * 448.0f;
  const float scale = 1.0f / sqrtf(static_cast<float>(kD));
  uint64_t launches = 0;
  auto ok = [&](cudaError_t e) {
    ++launches;
    return e == cudaSuccess;
  };

  // Algorithm 1's initialization, the reference attention, the value scale and the cache indices.
  if (cudaMemsetAsync(w.amax, 0, 2 * sizeof(uint32_t), st) != cudaSuccess ||
      !ok(launch_pdl(qfit_init_kernel, dim3(hkv), dim3(kHalf), 0, st, k, n_tok, T, hkv, rope_table, eps, w.s0,
                     w.mu)) ||
      !ok(launch_pdl(qfit_reference_kernel, dim3(hq, B), dim3(kD), static_cast<size_t>(T) * sizeof(float), st, q, k,
                     v, T, hq, hkv, rope_table, scale, w.y_ref)) ||
      !ok(launch_pdl(qfit_amax_kernel, dim3(blocks_for(static_cast<size_t>(n_tok) * hkv * kD, 256)), dim3(256), 0,
                     st, v, static_cast<size_t>(n_tok) * hkv * kD, w.amax + 1)) ||
      !ok(launch_pdl(qfit_fill_indices_kernel, dim3(blocks_for(n_tok, 256)), dim3(256), 0, st, B, T, w.seq_idx,
                     w.pos, w.seq_lens)))
    return NVFP4_ERR_CUDA;
  uint32_t amax_v = 0;
  if (cudaMemcpyAsync(&amax_v, w.amax + 1, sizeof(amax_v), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  auto gscale = [&](uint32_t bits) {
    float a;
    std::memcpy(&a, &bits, sizeof(a));
    return a > 0.0f ? a / qmax_448 : 1.0f;  // an all-zero tensor gets scale 1, as nvfp4_tensor_scale
  };
  nvfp4_kv_cache cache{w.kc, w.ks, w.vc, w.vs, w.seq_lens, B, hkv, kD, cap, 1.0f, gscale(amax_v), kv_format};

  for (int a = 0; a < grid_s; ++a) {
    const double alpha_s = static_cast<double>(a) / grid_s;
    for (int b = 0; b < grid_m; ++b) {
      const double alpha_m = static_cast<double>(b) / grid_m;
      if (cudaMemsetAsync(w.amax, 0, sizeof(uint32_t), st) != cudaSuccess ||
          !ok(launch_pdl(qfit_params_kernel, dim3(blocks_for(static_cast<size_t>(hq) * kD, 256)), dim3(256), 0, st,
                         w.s0, w.mu, alpha_s, alpha_m, hq, hkv, w.s_q, w.s_k, w.m)) ||
          !ok(launch_pdl(qfit_keys_kernel, dim3(blocks_for(static_cast<size_t>(n_tok) * hkv * kHalf, 256)), dim3(256),
                         0, st, k, n_tok, T, hkv, rope_table, w.s_k, w.m, w.k_in, w.amax)) ||
          !ok(launch_pdl(qfit_queries_kernel, dim3(blocks_for(static_cast<size_t>(B) * hq * kHalf, 256)), dim3(256),
                         0, st, q, B, T, hq, rope_table, w.s_q, w.q_t)))
        return NVFP4_ERR_CUDA;
      // The static key scale of this grid point is a host argument of the cache.
      uint32_t amax_k = 0;
      if (cudaMemcpyAsync(&amax_k, w.amax, sizeof(amax_k), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
          cudaStreamSynchronize(st) != cudaSuccess)
        return NVFP4_ERR_CUDA;
      cache.k_gscale = gscale(amax_k);
      nvfp4_status s2 = kv_append_rope_nvfp4(&cache, w.k_in, v, w.seq_idx, w.pos, n_tok, rope_table, rope_positions,
                                             w.m, stream);
      if (s2 != NVFP4_OK) return s2;
      s2 = decode_attention_nvfp4(&cache, w.q_t, hq, scale, w.out, w.attn_ws, w.attn_ws_bytes, stream);
      if (s2 != NVFP4_OK) return s2;
      if (!ok(launch_pdl(qfit_mse_kernel, dim3(1), dim3(1024), 0, st, w.out, w.y_ref, B * hq * kD,
                         w.err + a * grid_m + b)))
        return NVFP4_ERR_CUDA;
    }
  }
  // The first grid point (alpha_s-major order) with the least error wins.
  std::vector<double> err(points);
  if (cudaMemcpyAsync(err.data(), w.err, sizeof(double) * points, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  int best = 0;
  for (int i = 1; i < points; ++i)
    if (err[i] < err[best]) best = i;
  if (errors_host)
    for (int i = 0; i < points; ++i) errors_host[i] = err[i];
  if (!ok(launch_pdl(qfit_params_kernel, dim3(blocks_for(static_cast<size_t>(hq) * kD, 256)), dim3(256), 0, st,
                     w.s0, w.mu, static_cast<double>(best / grid_m) / grid_s,
                     static_cast<double>(best % grid_m) / grid_m, hq, hkv, s_q, s_k, m)) ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(launches);
  return launch_status();
}
