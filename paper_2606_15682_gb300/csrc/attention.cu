// a5: decode attention straight from the NVFP4 KV cache (Sec. 2.1:
// z = softmax(Q K_hat^T / sqrt(d)) V_hat with quantized K and V).
//
// Split-KV ("flash-decoding") with persistent CTAs.  A work item is one
// (sequence, KV head, 1024-token chunk).  Each CTA has a producer warp that
// streams the items' FP4 K/V codes and E4M3 scales into a 2-stage ring of
// 128-token stages with 1-D bulk copies (the ring runs on across items), and
// four consumer warps that each take two 16-token tiles of every stage (one
// barrier hand-off per two tiles; measured faster than 4 x 64-token stages).  A consumer
// dequantizes in registers (cvt e2m1x2 -> f16x2, times the E4M3 block scale:
// exact in f16) and runs mma.sync m16n8k16 with fp32 accumulation:
//   S^T[16 tok x 8 head] = K_hat[16 tok x 128] . Q^T[128 x 8]   (8 MMAs)
//   O^T[128 x 8 head]   += V_hat^T[128 x 16 tok] . P^T[16 x 8]  (8 MMAs)
// The up to 8 query heads that share a KV head (grouped-query attention) fill
// the MMA's N = 8.  Softmax is online, in fp32, in the log2 domain, with lazy
// rescaling (the running max moves only when a tile exceeds it by 2^8).  At
// the end of an item the four warps merge their partial (max, sum, O) and
// write one record; a combine kernel merges the records of all chunks.
//
// Lane roles (g = lane/4, t = lane%4), fixed by the m16n8k16 fragment layouts:
//   K: rows g and g+8 of the S tile, channels 32t..32t+31 (16 bytes, blocks 2t, 2t+1)
//   V: k-indices 2t, 2t+1, 2t+8, 2t+9, channels 16g..16g+15 (8 bytes, block g)
//   Q: head slot g, channels 32t..32t+31
// Row/k index m of a 16-token tile is token TOK(m) = (m&1)*4 + (m>>1&3) +
// (m&8): the V rows each lane reads are then t, t+4, t+8, t+12, so a V load
// instruction covers four consecutive token rows (measured faster on GB300
// than the orders that favour the K loads instead).  The channel order inside
// an MMA is permuted to match the lanes' contiguous bytes; neither
// permutation changes the dot products.
#include <cfloat>
#include <map>
#include <mutex>

#include "common.cuh"
#include "nvfp4_quant.cuh"

namespace nvfp4 {
namespace {

constexpr int kD = 128;
constexpr int kChunk = 1024;          // tokens per work item
constexpr int kStageTok = 128;        // tokens per ring stage
#ifndef NVFP4_ATTN_STAGES
#define NVFP4_ATTN_STAGES 2
#endif
#ifndef NVFP4_ATTN_MIN_CTAS
#define NVFP4_ATTN_MIN_CTAS 4
#endif
constexpr int kStages = NVFP4_ATTN_STAGES;  // 2 x 18 KiB ring + merge buffer: 4 CTAs per SM
constexpr int kConsumers = 4;         // consumer warps, 16 tokens of a stage each
constexpr int kThreads = 32 * (1 + kConsumers);
constexpr uint32_t kStageBytes = kStageTok * (64 + 8) * 2;  // K, V codes + scales: 18 KiB
static_assert(kChunk % kStageTok == 0 && kStageTok % (16 * kConsumers) == 0, "stage tiling");
constexpr uint32_t kOffKc = 0, kOffVc = kStageTok * 64, kOffKs = 2 * kStageTok * 64, kOffVs = kOffKs + kStageTok * 8;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleLog2 = 8.0f;  // lazy rescale threshold (P stays <= 2^8 in f16)

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

// E1M2 nibbles (two's complement n, value n/2) decode to f16 n; the 1/2 goes
// into the block scale.  The nibble XOR 8 in the low mantissa bits of 1024.0
// (0x6400) reads as 1032 + n, and one f16x2 subtraction of 1032 leaves n.  A
// nibble in bits 4-7 of a half is decoded where it stands: 1024 + 16 (n + 8)
// minus 1152 leaves 16 n, and its block scale carries a further 1/16.  Both
// are exact, and the product with the scale is the same f16 either way
// (16 n times s / 16 is n times s, and s / 16 is exact in f16 for every E4M3
// scale), so the tensor-core operands are those of the shifted decode.
__device__ __forceinline__ uint32_t hsub2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
// K side: the eight nibbles n0..n7 of w (n0 lowest) -> h[i] = (n_i, n_{i+4}),
// with h[1] and h[3] holding 16 n (their scales carry the 1/16): one
// mask-and-xor and one subtraction per pair, one shift per word.  The channel
// order inside each group of eight differs from the E2M1 path; the queries
// are paired the same way, so every logit is the same sum.
__device__ __forceinline__ void e1m2x8_to_f16x2_paired(uint32_t w, uint32_t h[4]) {
  const uint32_t t = w >> 8;
  h[0] = hsub2((w & 0x000F000Fu) ^ 0x64086408u, 0x64086408u);
  h[1] = hsub2((w & 0x00F000F0u) ^ 0x64806480u, 0x64806480u);
  h[2] = hsub2((t & 0x000F000Fu) ^ 0x64086408u, 0x64086408u);
  h[3] = hsub2((t & 0x00F000F0u) ^ 0x64806480u, 0x64806480u);
}
// V side: byte k of two tokens' words a and b -> lo = (a, b) of the byte's
// low-nibble channel, hi = 16 (a, b) of its high-nibble channel (its scale
// carries the 1/16).
__device__ __forceinline__ void e1m2_token_pair(uint32_t wa, uint32_t wb, int k, uint32_t* lo, uint32_t* hi) {
  const uint32_t x = __byte_perm(wa, wb, 0x4400u + 0x1111u * k);  // bytes: a_k, a_k, b_k, b_k
  *lo = hsub2((x & 0x000F000Fu) ^ 0x64086408u, 0x64086408u);
  *hi = hsub2((x & 0x00F000F0u) ^ 0x64806480u, 0x64806480u);
}

template <bool kE1M2>
__device__ __forceinline__ void decode8(uint32_t w, uint32_t h[4]) {
  if (kE1M2) e1m2x8_to_f16x2_paired(w, h);
  else e2m1x8_to_f16x2(w, h);
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

__device__ __forceinline__ void named_barrier_consumers() {
  asm volatile("bar.sync 1, %0;" ::"n"(32 * kConsumers) : "memory");
}

// Token of row / k index m (0..15) of a 16-token tile.
__device__ __forceinline__ int tile_tok(int m) { return (m & 1) * 4 + ((m >> 1) & 3) + (m & 8); }

struct Item {
  int b, kvh, split, t_begin, t_end;
};

__device__ __forceinline__ Item decode_item(int item, int n_splits, int hkv, const int32_t* __restrict__ seq_lens,
                                            int capacity) {
  Item it;
  it.split = item % n_splits;
  const int rest = item / n_splits;
  it.kvh = rest % hkv;
  it.b = rest / hkv;
  int len = __ldg(seq_lens + it.b);
  len = max(0, min(len, capacity));
  it.t_begin = it.split * kChunk;
  it.t_end = min(it.t_begin + kChunk, len);
  return it;
}

struct Params {
  const uint8_t* k_codes;
  const uint8_t* k_scales;
  const uint8_t* v_codes;
  const uint8_t* v_scales;
  const int32_t* seq_lens;
  const uint16_t* q;
  float* o_ws;
  float* ml_ws;
  int* status;
  int hkv, capacity, hq, group, n_splits, n_items;
  float logit_mult;  // softmax_scale * g_K * log2(e)
  int fault_skip_stage;  // test-only: CTA 0's producer leaves its first stage unissued
};

// kE1M2: the cache holds E1M2 elements (decoded to n, the scale carries 1/2).
template <bool kE1M2>
__global__ void __launch_bounds__(kThreads, NVFP4_ATTN_MIN_CTAS) attn_partial_kernel(const Params p) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* ring = smem;
  float* sh_o = reinterpret_cast<float*>(smem + kStages * kStageBytes);  // [kConsumers][8][128]
  float* sh_m = sh_o + kConsumers * 8 * kD;                              // [kConsumers][8]
  float* sh_l = sh_m + kConsumers * 8;
  uint64_t* full = reinterpret_cast<uint64_t*>(sh_l + kConsumers * 8);
  uint64_t* empty = full + kStages;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumers);
    }
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  griddep_wait_and_release();
  if (p.capacity > 0 && blockIdx.x == 0 && threadIdx.x == 0) {
    for (int b = 0; b < p.n_items / (p.n_splits * p.hkv); ++b)
      if (__ldg(p.seq_lens + b) > p.capacity) { set_status(p.status, NVFP4_ERR_CAPACITY); break; }
  }

  if (warp == 0) {
    // ------------------------------------------------------------ producer ---
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_parity[kStages];
      bool issued[kStages];
      for (int s = 0; s < kStages; ++s) issued[s] = false;
      bool skip_stage = p.fault_skip_stage && blockIdx.x == 0;
      for (int item = blockIdx.x; item < p.n_items && !abort_flag; item += gridDim.x) {
        const Item it = decode_item(item, p.n_splits, p.hkv, p.seq_lens, p.capacity);
        const size_t row0 = (static_cast<size_t>(it.b) * p.hkv + it.kvh) * p.capacity;
        for (int t0 = it.t_begin; t0 < it.t_end; t0 += kStageTok) {
          const int n = min(kStageTok, it.t_end - t0);
          const int n_even = (n + 1) & ~1;  // scale rows copied in 16-byte units (capacity is even)
          if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, &abort_flag)) {
            set_status(p.status, NVFP4_ERR_TIMEOUT);
            abort_flag = 1;
            break;
          }
          if (skip_stage) {
            // Injected fault: the stage is neither armed nor loaded, so the
            // consumers' bounded wait on it runs out (NVFP4_ERR_TIMEOUT).
            skip_stage = false;
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
            continue;
          }
          uint8_t* st = ring + stage * kStageBytes;
          mbar_arrive_expect_tx(&full[stage], 2u * (n * 64 + n_even * 8));
          const size_t tok = row0 + t0;
          bulk_load(st + kOffKc, p.k_codes + tok * 64, n * 64, &full[stage]);
          bulk_load(st + kOffVc, p.v_codes + tok * 64, n * 64, &full[stage]);
          bulk_load(st + kOffKs, p.k_scales + tok * 8, n_even * 8, &full[stage]);
          bulk_load(st + kOffVs, p.v_scales + tok * 8, n_even * 8, &full[stage]);
          issued[stage] = true;
          issued_parity[stage] = phase;
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
      }
      if (abort_flag)
        for (int s = 0; s < kStages; ++s)
          if (issued[s]) mbar_wait_bounded(&full[s], issued_parity[s], nullptr);
    }
    return;
  }

  // -------------------------------------------------------------- consumers ---
  const int cw = warp - 1;  // consumer index: tiles cw, cw + 4, ... of each stage
  const int g = lane >> 2, t = lane & 3;
  const int rk0 = tile_tok(g), rk1 = tile_tok(g + 8);                    // K rows of this lane
  const int rv[4] = {tile_tok(2 * t), tile_tok(2 * t + 1), tile_tok(2 * t + 8), tile_tok(2 * t + 9)};  // V rows
  int stage = 0;
  uint32_t phase = 0;
  for (int item = blockIdx.x; item < p.n_items; item += gridDim.x) {
    const Item it = decode_item(item, p.n_splits, p.hkv, p.seq_lens, p.capacity);
    // Queries of head slot g: f16 after an exact power-of-two scaling that
    // keeps |q| < 1; the scaling is undone in the logit multiplier.
    const bool head_live = g < p.group;
    float qv[32];
    {
      const uint4* qp = reinterpret_cast<const uint4*>(
          p.q + (static_cast<size_t>(it.b) * p.hq + it.kvh * p.group + (head_live ? g : 0)) * kD + 32 * t);
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
    const int qexp = qmax > 0.0f ? static_cast<int>((__float_as_uint(qmax) >> 23) & 0xFF) - 126 : 0;
    const float qscale = ldexpf(1.0f, -qexp);
    uint32_t qf[16];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      // k-step j = 2w + h.  E2M1 keys hold channel pairs (4j, 4j+1), (4j+2, 4j+3);
      // E1M2 keys (decoded in pairs i, i+4 of each word) hold (8w+2h, 8w+2h+4), (8w+2h+1, 8w+2h+5).
      const int c0 = kE1M2 ? 8 * (j >> 1) + 2 * (j & 1) : 4 * j;
      const int c1 = kE1M2 ? c0 + 4 : c0 + 1, c2 = kE1M2 ? c0 + 1 : c0 + 2, c3 = kE1M2 ? c0 + 5 : c0 + 3;
      qf[2 * j] = f32x2_to_f16x2(qv[c0] * qscale, qv[c1] * qscale);
      qf[2 * j + 1] = f32x2_to_f16x2(qv[c2] * qscale, qv[c3] * qscale);
    }
    const float mult_self = p.logit_mult / qscale;
    const float mult0 = __shfl_sync(0xffffffffu, mult_self, (2 * t) * 4);
    const float mult1 = __shfl_sync(0xffffffffu, mult_self, (2 * t + 1) * 4);

    float o[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.0f;
    float m_run[2] = {-INFINITY, -INFINITY};
    float l_run[2] = {0.0f, 0.0f};

    for (int t0 = it.t_begin; t0 < it.t_end; t0 += kStageTok) {
      int ok = 1;
      if (lane == 0) {
        ok = !abort_flag && mbar_wait_bounded(&full[stage], phase, &abort_flag);
        if (!ok && !abort_flag) {
          set_status(p.status, NVFP4_ERR_TIMEOUT);
          abort_flag = 1;
        }
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) return;
      const uint8_t* st = ring + stage * kStageBytes;
      // The warp's two tiles of the stage, unrolled: the second tile's loads,
      // decode and score MMAs interleave with the first tile's softmax and
      // value MMAs (same 96 registers, same 4 CTAs per SM): B=64, T=16384
      // 248.4 -> 241.3 us, bit-identical.
#pragma unroll
      for (int sub = 0; sub < kStageTok / (16 * kConsumers); ++sub) {
      const int r0 = 16 * (cw + kConsumers * sub);  // this warp's tile within the stage
      const int tile = t0 + r0;
      const int valid = it.t_end - tile;  // tokens of this warp's tile inside the item (may be <= 0)
      if (valid > 0) {
        // ---- S^T = K_hat Q^T: 8 k-steps of 16 channels ---------------------
        const uint4 ka = *reinterpret_cast<const uint4*>(st + kOffKc + (r0 + rk0) * 64 + 16 * t);
        const uint4 kb = *reinterpret_cast<const uint4*>(st + kOffKc + (r0 + rk1) * 64 + 16 * t);
        uint32_t ksa = e4m3x2_to_f16x2(*reinterpret_cast<const uint16_t*>(st + kOffKs + (r0 + rk0) * 8 + 2 * t));
        uint32_t ksb = e4m3x2_to_f16x2(*reinterpret_cast<const uint16_t*>(st + kOffKs + (r0 + rk1) * 8 + 2 * t));
        if (kE1M2) { ksa = hmul2(ksa, 0x38003800u); ksb = hmul2(ksb, 0x38003800u); }  // times 1/2, exact
        const uint32_t sa_lo = bcast_lo(ksa), sa_hi = bcast_hi(ksa);
        const uint32_t sb_lo = bcast_lo(ksb), sb_hi = bcast_hi(ksb);
        float s[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        const uint32_t kaw[4] = {ka.x, ka.y, ka.z, ka.w};
        const uint32_t kbw[4] = {kb.x, kb.y, kb.z, kb.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          uint32_t ha[4], hb[4];
          decode8<kE1M2>(kaw[w], ha);
          decode8<kE1M2>(kbw[w], hb);
          const uint32_t sa = w < 2 ? sa_lo : sa_hi, sb = w < 2 ? sb_lo : sb_hi;
          // E1M2: the scales of the pairs decoded as 16 n (times 1/16, exact).
          const uint32_t sa1 = kE1M2 ? hmul2(sa, 0x2C002C00u) : sa, sb1 = kE1M2 ? hmul2(sb, 0x2C002C00u) : sb;
#pragma unroll
          for (int h = 0; h < 2; ++h) {  // k-step j = 2w + h uses bytes 2j and 2j+1
            const uint32_t a[4] = {hmul2(ha[2 * h], sa), hmul2(hb[2 * h], sb), hmul2(ha[2 * h + 1], sa1),
                                   hmul2(hb[2 * h + 1], sb1)};
            const int j = 2 * w + h;
            mma16816(s, a, qf[2 * j], qf[2 * j + 1]);
          }
        }
        // ---- online softmax over this tile (log2 domain) -------------------
        float x0 = s[0] * mult0, x1 = s[1] * mult1, x2 = s[2] * mult0, x3 = s[3] * mult1;
        uint32_t vs01_raw, vs89_raw;
        {
          const uint32_t s0 = st[kOffVs + (r0 + rv[0]) * 8 + g], s1 = st[kOffVs + (r0 + rv[1]) * 8 + g];
          const uint32_t s2 = st[kOffVs + (r0 + rv[2]) * 8 + g], s3 = st[kOffVs + (r0 + rv[3]) * 8 + g];
          vs01_raw = s0 | (s1 << 8);
          vs89_raw = s2 | (s3 << 8);
        }
        if (valid < 16) {  // ragged end of the item: mask keys, zero the scales of absent values
          if (rk0 >= valid) x0 = x1 = -INFINITY;
          if (rk1 >= valid) x2 = x3 = -INFINITY;
          if (rv[0] >= valid) vs01_raw &= 0xFF00u;
          if (rv[1] >= valid) vs01_raw &= 0x00FFu;
          if (rv[2] >= valid) vs89_raw &= 0xFF00u;
          if (rv[3] >= valid) vs89_raw &= 0x00FFu;
        }
        float mx0 = fmaxf(x0, x2), mx1 = fmaxf(x1, x3);
        // The tile maximum is needed only when some logit exceeds the running
        // maximum by more than the lazy threshold: vote first, reduce then.
        if (__any_sync(0xffffffffu, mx0 > m_run[0] + kRescaleLog2 || mx1 > m_run[1] + kRescaleLog2)) {
#pragma unroll
          for (int sh = 4; sh < 32; sh <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, sh));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, sh));
          }
          const bool up0 = mx0 > m_run[0] + kRescaleLog2, up1 = mx1 > m_run[1] + kRescaleLog2;
          const float al0 = up0 ? fast_exp2(m_run[0] - mx0) : 1.0f;
          const float al1 = up1 ? fast_exp2(m_run[1] - mx1) : 1.0f;
          if (up0) m_run[0] = mx0;
          if (up1) m_run[1] = mx1;
          l_run[0] *= al0;
          l_run[1] *= al1;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            o[i][0] *= al0; o[i][1] *= al1; o[i][2] *= al0; o[i][3] *= al1;
          }
        }
        const float p0 = fast_exp2(x0 - m_run[0]), p1 = fast_exp2(x1 - m_run[1]);
        const float p2 = fast_exp2(x2 - m_run[0]), p3 = fast_exp2(x3 - m_run[1]);
        l_run[0] += p0 + p2;
        l_run[1] += p1 + p3;
        // P^T fragments for the PV product: transpose the two 8x8 (token, head) blocks.
        const uint32_t pb0 = movmatrix_trans(f32x2_to_f16x2(p0, p1));
        const uint32_t pb1 = movmatrix_trans(f32x2_to_f16x2(p2, p3));

        // ---- O^T += V_hat^T P^T: 8 m-tiles, m-tile i = channels 16g+2i, 16g+2i+1
        uint32_t vs01 = e4m3x2_to_f16x2(vs01_raw), vs89 = e4m3x2_to_f16x2(vs89_raw);
        if (kE1M2) { vs01 = hmul2(vs01, 0x38003800u); vs89 = hmul2(vs89, 0x38003800u); }
        // E1M2: the high-nibble channels are decoded as 16 n; their scales carry 1/16 (exact).
        const uint32_t vs01_hi = kE1M2 ? hmul2(vs01, 0x2C002C00u) : vs01;
        const uint32_t vs89_hi = kE1M2 ? hmul2(vs89, 0x2C002C00u) : vs89;
        const uint2 va = *reinterpret_cast<const uint2*>(st + kOffVc + (r0 + rv[0]) * 64 + 8 * g);
        const uint2 vb = *reinterpret_cast<const uint2*>(st + kOffVc + (r0 + rv[1]) * 64 + 8 * g);
        const uint2 vc = *reinterpret_cast<const uint2*>(st + kOffVc + (r0 + rv[2]) * 64 + 8 * g);
        const uint2 vd = *reinterpret_cast<const uint2*>(st + kOffVc + (r0 + rv[3]) * 64 + 8 * g);
#pragma unroll
        for (int half = 0; half < 2; ++half) {  // bytes 0-3, then 4-7 of each token's 8-byte slice
          const uint32_t wa = half ? va.y : va.x, wb = half ? vb.y : vb.x;
          const uint32_t wc = half ? vc.y : vc.x, wd = half ? vd.y : vd.x;
          uint32_t f_lo_ab[4], f_hi_ab[4], f_lo_cd[4], f_hi_cd[4];
          if (kE1M2) {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              e1m2_token_pair(wa, wb, k, &f_lo_ab[k], &f_hi_ab[k]);
              e1m2_token_pair(wc, wd, k, &f_lo_cd[k], &f_hi_cd[k]);
            }
          } else {
            // Pair the same channel of two tokens in one e2m1x2 byte (first token in the low nibble).
            const uint32_t lo_ab = (wa & 0x0F0F0F0Fu) | ((wb << 4) & 0xF0F0F0F0u);
            const uint32_t hi_ab = ((wa >> 4) & 0x0F0F0F0Fu) | (wb & 0xF0F0F0F0u);
            const uint32_t lo_cd = (wc & 0x0F0F0F0Fu) | ((wd << 4) & 0xF0F0F0F0u);
            const uint32_t hi_cd = ((wc >> 4) & 0x0F0F0F0Fu) | (wd & 0xF0F0F0F0u);
            e2m1x8_to_f16x2(lo_ab, f_lo_ab);
            e2m1x8_to_f16x2(hi_ab, f_hi_ab);
            e2m1x8_to_f16x2(lo_cd, f_lo_cd);
            e2m1x8_to_f16x2(hi_cd, f_hi_cd);
          }
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t a[4] = {hmul2(f_lo_ab[k], vs01), hmul2(f_hi_ab[k], vs01_hi), hmul2(f_lo_cd[k], vs89),
                                   hmul2(f_hi_cd[k], vs89_hi)};
            mma16816(o[4 * half + k], a, pb0, pb1);
          }
        }
      }
      }  // tiles of the stage
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[stage]);
      if (++stage == kStages) { stage = 0; phase ^= 1u; }
    }

    // ---- merge the consumer warps, write this item's partial --------------
    l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 4);
    l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 4);
    l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 8);
    l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 8);
    l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 16);
    l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 16);
    float* my_o = sh_o + cw * 8 * kD;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int c0 = 16 * g + 2 * i;  // channel of accumulator rows g / g+8 of m-tile i
      my_o[(2 * t) * kD + c0] = o[i][0];
      my_o[(2 * t + 1) * kD + c0] = o[i][1];
      my_o[(2 * t) * kD + c0 + 1] = o[i][2];
      my_o[(2 * t + 1) * kD + c0 + 1] = o[i][3];
    }
    if (g == 0) {
      sh_m[cw * 8 + 2 * t] = m_run[0]; sh_m[cw * 8 + 2 * t + 1] = m_run[1];
      sh_l[cw * 8 + 2 * t] = l_run[0]; sh_l[cw * 8 + 2 * t + 1] = l_run[1];
    }
    named_barrier_consumers();
    for (int idx = threadIdx.x - 32; idx < p.group * kD; idx += 32 * kConsumers) {
      const int h = idx / kD, c = idx % kD;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kConsumers; ++w) M = fmaxf(M, sh_m[w * 8 + h]);
      float acc = 0.0f, L = 0.0f;
      if (M != -INFINITY) {
#pragma unroll
        for (int w = 0; w < kConsumers; ++w) {
          const float wt = fast_exp2(sh_m[w * 8 + h] - M);
          acc += wt * sh_o[(w * 8 + h) * kD + c];
          L += wt * sh_l[w * 8 + h];
        }
      }
      const size_t rec = (static_cast<size_t>(it.b) * p.hq + it.kvh * p.group + h) * p.n_splits + it.split;
      p.o_ws[rec * kD + c] = acc;
      if (c == 0) {
        p.ml_ws[rec * 2] = M;
        p.ml_ws[rec * 2 + 1] = L;
      }
    }
    named_barrier_consumers();  // the merge buffer is rewritten by the next item
  }
}

// out[b, h] = g_V * sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s
// Where the combine kernel puts o: bf16 [batch, heads, 128], or (kQuant) the
// NVFP4 A operand of the output projection: the bf16-rounded o of each query
// head's 128 channels quantized in 8 blocks of 16 with the static tensor scale
// g_out by the library's recipe, codes [batch, heads * 64] bytes and MMA-layout
// scales of the [batch, heads * 128] matrix (padding rows zero).
struct CombineOut {
  uint16_t* bf16;
  uint8_t* codes;
  uint8_t* scales;
  const float* g_out;
  int* status;
  int rows;
  uint32_t kgroups;
};

template <bool kQuant>
__global__ void __launch_bounds__(kD) attn_combine_kernel(const float* __restrict__ o_ws,
                                                         const float* __restrict__ ml_ws, int n_splits, float gv,
                                                         const CombineOut out) {
  griddep_wait_and_release();
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
  if (!kQuant) {
    out.bf16[bh * kD + threadIdx.x] = bits;
    return;
  }
  // Lanes 16j..16j+15 of a warp hold one 16-channel block of this head.
  const float g_in = __ldg(out.g_out);
  const bool g_ok = g_in > 0.0f && g_in <= FLT_MAX;
  if (!g_ok && bh == 0 && threadIdx.x == 0) set_status(out.status, NVFP4_ERR_INVALID_ARG);
  const float g = g_ok ? g_in : 1.0f;
  const float x = __uint_as_float(static_cast<uint32_t>(bits) << 16);
  float amax = fabsf(x);
#pragma unroll
  for (int sh = 1; sh < 16; sh <<= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, sh));
  const BlockScale bs = block_scale(amax, g, __fmul_rn(6.0f, g));
  // Lane pairs (2i, 2i+1) form one code byte, element 2i in the low nibble.
  const float mine = __fmul_rn(x, bs.mult);
  const float other = __shfl_xor_sync(0xffffffffu, mine, 1);
  uint32_t pair;  // the first source of the conversion goes to the high nibble
  asm("{\n .reg .b8 t;\n cvt.rn.satfinite.e2m1x2.f32 t, %1, %2;\n cvt.u32.u8 %0, t;\n}"
      : "=r"(pair)
      : "f"(other), "f"(mine));
  const uint32_t row = blockIdx.y, head = blockIdx.x, c = threadIdx.x;
  const uint32_t padded = (static_cast<uint32_t>(out.rows) + 127u) & ~127u;
  const uint64_t code_bytes = static_cast<uint64_t>(out.rows) * gridDim.x * (kD / 2);
  const uint64_t scale_bytes = static_cast<uint64_t>(padded) * out.kgroups * 4;
  const uint64_t code_off = static_cast<uint64_t>(row) * (gridDim.x * (kD / 2)) + head * (kD / 2) + c / 2;
  if ((c & 1) == 0 && in_bounds(out.status, code_off < code_bytes))
    out.codes[code_off] = g_ok ? static_cast<uint8_t>(pair & 0xFFu) : 0;
  const uint32_t kb = head * (kD / 16) + c / 16;
  const uint64_t sc_off = mma_scale_offset(row, kb, out.kgroups);
  if ((c & 15) == 0 && in_bounds(out.status, sc_off < scale_bytes))
    out.scales[sc_off] = g_ok ? static_cast<uint8_t>(bs.code) : 0;
  // Rows from batch up to the next multiple of 128 hold zero scales.
  if (row == 0 && c < kD / 16) {
    for (uint32_t pr = out.rows; pr < padded; ++pr) {
      const uint64_t off = mma_scale_offset(pr, head * (kD / 16) + c, out.kgroups);
      if (in_bounds(out.status, off < scale_bytes)) out.scales[off] = 0;
    }
  }
}

int splits_for(int capacity) { return (capacity + kChunk - 1) / kChunk; }

constexpr size_t kSmemBytes =
    kStages * kStageBytes + (kConsumers * 8 * kD + 2 * kConsumers * 8) * sizeof(float) + 2 * kStages * 8;

template <bool kE1M2>
int resident_ctas() {
  static std::mutex mu;
  static std::map<int, int> cache;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(d);
  if (it != cache.end()) return it->second;
  if (cudaFuncSetAttribute(attn_partial_kernel<kE1M2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kSmemBytes)) != cudaSuccess)
    return 0;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attn_partial_kernel<kE1M2>, kThreads, kSmemBytes) !=
          cudaSuccess ||
      per_sm <= 0)
    return 0;
  cache[d] = per_sm * sm_count();
  return cache[d];
}

// The partial kernel for the cache's element format, and its resident CTAs.
using PartialKernel = void (*)(const Params);
PartialKernel partial_kernel(const nvfp4_kv_cache* cache) {
  return cache->kv_format == NVFP4_KV_E1M2 ? attn_partial_kernel<true> : attn_partial_kernel<false>;
}
int resident_ctas(const nvfp4_kv_cache* cache) {
  return cache->kv_format == NVFP4_KV_E1M2 ? resident_ctas<true>() : resident_ctas<false>();
}
bool kv_format_ok(const nvfp4_kv_cache* cache) {
  return cache->kv_format == NVFP4_KV_E2M1 || cache->kv_format == NVFP4_KV_E1M2;
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API size_t decode_attention_nvfp4_workspace_size(int32_t batch, int32_t num_q_heads, int32_t capacity) {
  if (batch <= 0 || num_q_heads <= 0 || capacity <= 0) return 0;
  return static_cast<size_t>(batch) * num_q_heads * splits_for(capacity) * (kD + 2) * sizeof(float);
}

namespace nvfp4 {
namespace {

// Checks shared by the decode-attention entry points (all but the output
// buffers and the split-KV partials).
nvfp4_status attention_validate(const nvfp4_kv_cache* cache, const void* q_bf16, int32_t num_q_heads,
                                float softmax_scale) {
  if (!cache || !q_bf16 || !cache->seq_lens) return NVFP4_ERR_INVALID_ARG;
  if (!cache->k_codes || !cache->k_scales || !cache->v_codes || !cache->v_scales) return NVFP4_ERR_INVALID_ARG;
  if (!kv_format_ok(cache)) return NVFP4_ERR_INVALID_ARG;
  if (!(cache->k_gscale > 0.0f && cache->k_gscale <= FLT_MAX) || !(cache->v_gscale > 0.0f && cache->v_gscale <= FLT_MAX) ||
      !(softmax_scale > 0.0f && softmax_scale <= FLT_MAX))
    return NVFP4_ERR_INVALID_ARG;
  if (cache->head_dim != kD || cache->batch <= 0 || cache->num_kv_heads <= 0 || cache->capacity <= 0 ||
      cache->capacity % 2 || num_q_heads <= 0 || num_q_heads % cache->num_kv_heads ||
      num_q_heads / cache->num_kv_heads > 8)
    return NVFP4_ERR_SHAPE;
  if (static_cast<int64_t>(cache->batch) > 65535 || num_q_heads > 65535) return NVFP4_ERR_SHAPE;
  const int64_t n_items = static_cast<int64_t>(cache->batch) * cache->num_kv_heads * splits_for(cache->capacity);
  if (n_items >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  return NVFP4_OK;
}

// Alignment of the query and cache arrays, then the partial kernel's
// parameters with its partials at `partials` and its grid size.
nvfp4_status attention_params(const nvfp4_kv_cache* cache, const void* q_bf16, int32_t num_q_heads,
                              float softmax_scale, float* partials, Params* prm, int* grid) {
  if (!aligned(q_bf16, 16) || !aligned(cache->k_codes, 16) || !aligned(cache->v_codes, 16) ||
      !aligned(cache->k_scales, 16) || !aligned(cache->v_scales, 16))
    return NVFP4_ERR_ALIGN;
  const int ctas_max = resident_ctas(cache);
  if (ctas_max <= 0) return NVFP4_ERR_CUDA;
  const int64_t n_items = static_cast<int64_t>(cache->batch) * cache->num_kv_heads * splits_for(cache->capacity);
  prm->k_codes = cache->k_codes;
  prm->k_scales = cache->k_scales;
  prm->v_codes = cache->v_codes;
  prm->v_scales = cache->v_scales;
  prm->seq_lens = cache->seq_lens;
  prm->q = static_cast<const uint16_t*>(q_bf16);
  prm->status = status_word_dev();
  prm->hkv = cache->num_kv_heads;
  prm->capacity = cache->capacity;
  prm->hq = num_q_heads;
  prm->group = num_q_heads / cache->num_kv_heads;
  prm->n_splits = splits_for(cache->capacity);
  prm->n_items = static_cast<int>(n_items);
  prm->logit_mult = softmax_scale * cache->k_gscale * kLog2e;
  prm->fault_skip_stage = take_fault(NVFP4_FAULT_ATTN_SKIP_STAGE) ? 1 : 0;
  // Every record the combine kernel reads is written by the partial kernel of
  // the same call, so nothing left from an earlier call needs clearing.
  prm->o_ws = partials;
  prm->ml_ws = prm->o_ws + static_cast<size_t>(cache->batch) * num_q_heads * prm->n_splits * kD;
  *grid = static_cast<int>(n_items < ctas_max ? n_items : ctas_max);
  return NVFP4_OK;
}

}  // namespace
}  // namespace nvfp4

NVFP4_API nvfp4_status decode_attention_nvfp4(const nvfp4_kv_cache* cache, const void* q_bf16, int32_t num_q_heads,
                                              float softmax_scale, void* out_bf16, void* workspace,
                                              size_t workspace_bytes, void* stream) {
  NVFP4_TRACE("decode_attention_nvfp4");
  if (!out_bf16 || !workspace) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = attention_validate(cache, q_bf16, num_q_heads, softmax_scale);
  if (st != NVFP4_OK) return st;
  if (workspace_bytes < decode_attention_nvfp4_workspace_size(cache->batch, num_q_heads, cache->capacity))
    return NVFP4_ERR_SHAPE;
  if (!aligned(out_bf16, 16) || !aligned(workspace, 16)) return NVFP4_ERR_ALIGN;
  Params prm;
  int grid = 0;
  st = attention_params(cache, q_bf16, num_q_heads, softmax_scale, static_cast<float*>(workspace), &prm, &grid);
  if (st != NVFP4_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (launch_pdl(partial_kernel(cache), dim3(grid), dim3(kThreads), kSmemBytes, s, prm) != cudaSuccess ||
      launch_pdl(attn_combine_kernel<false>, dim3(num_q_heads, cache->batch), dim3(kD), 0, s,
                 static_cast<const float*>(prm.o_ws), static_cast<const float*>(prm.ml_ws), prm.n_splits,
                 cache->v_gscale, CombineOut{static_cast<uint16_t*>(out_bf16)}) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(2);
  return launch_status();
}

NVFP4_API nvfp4_status decode_attention_nvfp4_quantize(const nvfp4_kv_cache* cache, const void* q_bf16,
                                                       int32_t num_q_heads, float softmax_scale, const float* g_out,
                                                       uint8_t* out_codes, uint8_t* out_scales, void* workspace,
                                                       size_t workspace_bytes, void* stream) {
  NVFP4_TRACE("decode_attention_nvfp4_quantize");
  if (!g_out || !out_codes || !out_scales || !workspace) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = attention_validate(cache, q_bf16, num_q_heads, softmax_scale);
  if (st != NVFP4_OK) return st;
  if (workspace_bytes < decode_attention_nvfp4_workspace_size(cache->batch, num_q_heads, cache->capacity))
    return NVFP4_ERR_SHAPE;
  if (!aligned(out_codes, 16) || !aligned(out_scales, 4) || !aligned(g_out, 4) || !aligned(workspace, 16))
    return NVFP4_ERR_ALIGN;
  Params prm;
  int grid = 0;
  st = attention_params(cache, q_bf16, num_q_heads, softmax_scale, static_cast<float*>(workspace), &prm, &grid);
  if (st != NVFP4_OK) return st;
  CombineOut o{};
  o.codes = out_codes;
  o.scales = out_scales;
  o.g_out = g_out;
  o.status = status_word_dev();
  o.rows = cache->batch;
  o.kgroups = static_cast<uint32_t>(num_q_heads) * (kD / 64);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (launch_pdl(partial_kernel(cache), dim3(grid), dim3(kThreads), kSmemBytes, s, prm) != cudaSuccess ||
      launch_pdl(attn_combine_kernel<true>, dim3(num_q_heads, cache->batch), dim3(kD), 0, s,
                 static_cast<const float*>(prm.o_ws), static_cast<const float*>(prm.ml_ws), prm.n_splits,
                 cache->v_gscale, o) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(2);
  return launch_status();
}

// ---------------------------------------------------------------------------
// Decode attention for callers that cannot allocate device memory.  The
// split-KV partials live in one file-scope device array instead of a caller
// workspace; every GPU that loads the library holds it until the process
// exits, and all calls share it.
namespace nvfp4 {
namespace {

static __device__ __align__(256) float g_attn_static_scratch[NVFP4_ATTN_STATIC_SCRATCH_BYTES / sizeof(float)];

// Device address of the static scratch for the current device, looked up once
// per device with that device current.  Host code must not hand the symbol
// itself to a kernel: on the host it is only a stand-in for the device array.
float* attn_static_scratch_dev() {
  static std::mutex mu;
  static std::map<int, float*> addr;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  auto it = addr.find(d);
  if (it != addr.end()) return it->second;
  float* p = nullptr;
  if (cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_attn_static_scratch) != cudaSuccess || !p) return nullptr;
  addr[d] = p;
  return p;
}

}  // namespace
}  // namespace nvfp4

NVFP4_API nvfp4_status decode_attention_nvfp4_static_scratch(const nvfp4_kv_cache* cache, const void* q_bf16,
                                                             int32_t num_q_heads, float softmax_scale,
                                                             void* out_bf16, void* stream) {
  NVFP4_TRACE("decode_attention_nvfp4_static_scratch");
  if (!out_bf16) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = attention_validate(cache, q_bf16, num_q_heads, softmax_scale);
  if (st != NVFP4_OK) return st;
  // The partials must fit in the static scratch; larger problems are refused.
  if (decode_attention_nvfp4_workspace_size(cache->batch, num_q_heads, cache->capacity) >
      NVFP4_ATTN_STATIC_SCRATCH_BYTES)
    return NVFP4_ERR_SHAPE;
  if (!aligned(out_bf16, 16)) return NVFP4_ERR_ALIGN;
  float* scratch = attn_static_scratch_dev();
  if (!scratch) return NVFP4_ERR_CUDA;
  Params prm;
  int grid = 0;
  st = attention_params(cache, q_bf16, num_q_heads, softmax_scale, scratch, &prm, &grid);
  if (st != NVFP4_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (launch_pdl(partial_kernel(cache), dim3(grid), dim3(kThreads), kSmemBytes, s, prm) != cudaSuccess ||
      launch_pdl(attn_combine_kernel<false>, dim3(num_q_heads, cache->batch), dim3(kD), 0, s,
                 static_cast<const float*>(prm.o_ws), static_cast<const float*>(prm.ml_ws), prm.n_splits,
                 cache->v_gscale, CombineOut{static_cast<uint16_t*>(out_bf16)}) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(2);
  return launch_status();
}
