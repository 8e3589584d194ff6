// a1 tensor scale and a2 NVFP4 quantization (Appendix A format).
// All kernels are launched with programmatic dependent launch.
//
// Both kernels stream bf16 with 128-bit loads.  The tensor-scale reduction
// takes one 8-element chunk per lane per step; the quantizer one 16-element
// block per lane.  They are HBM-bound: the quantizer moves 2 B in and
// 0.5625 B out per element.
#include <cfloat>
#include <map>
#include <mutex>

#include "common.cuh"
#include "nvfp4_quant.cuh"

namespace nvfp4 {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;
// Timeline build (-DNVFP4_TIMELINE): quantize_dynamic_kernel records, per
// block, the globaltimer at entry, when its phase-1 loads are done, when it
// has arrived at the grid barrier, when the barrier released it and when its
// stores are issued.  The release build compiles the stamps away.
#ifdef NVFP4_TIMELINE
constexpr int kTimelineBlocks = 2048;
__device__ unsigned long long g_quantize_timeline[kTimelineBlocks][5];
__device__ __forceinline__ void timeline_stamp(int event) {
  if (threadIdx.x == 0 && blockIdx.x < kTimelineBlocks) g_quantize_timeline[blockIdx.x][event] = globaltimer_ns();
}
#else
__device__ __forceinline__ void timeline_stamp(int) {}
#endif

#ifndef NVFP4_BARRIER_POLL_NS
#define NVFP4_BARRIER_POLL_NS 100  // sleep between polls of the one-launch quantizer's grid barrier
#endif

// Chunk c (8 elements) of a [rows, cols] tensor with leading dimension ld.
struct ChunkMap {
  FastDiv cpr;   // chunks per row
  uint32_t total;
  int64_t ld;
  bool dense;    // ld == cols: chunk c starts at element 8c
  __device__ __forceinline__ int64_t elem(uint32_t c, uint32_t* row, uint32_t* chunk_in_row) const {
    const uint32_t r = cpr.div(c);
    *row = r;
    *chunk_in_row = c - r * cpr.d;
    return dense ? static_cast<int64_t>(c) * 8 : static_cast<int64_t>(r) * ld + static_cast<int64_t>(*chunk_in_row) * 8;
  }
};

__global__ void __launch_bounds__(kThreads) amax_kernel(const uint16_t* __restrict__ x, ChunkMap map,
                                                        uint32_t* __restrict__ amax_bits) {
  griddep_wait_and_release();
  const uint32_t stride = gridDim.x * blockDim.x;
  uint32_t m = 0;
  for (uint32_t c0 = blockIdx.x * blockDim.x; c0 < map.total; c0 += stride * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint32_t c = c0 + u * stride + threadIdx.x;
      uint32_t r, j;
      v[u] = c < map.total ? __ldg(reinterpret_cast<const uint4*>(x + map.elem(c, &r, &j))) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) m = max(m, amax_bits_bf16x8(v[u]));
  }
  m = __reduce_max_sync(0xffffffffu, m);
  __shared__ uint32_t warp_max[kThreads / 32];
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x < 32) {
    m = threadIdx.x < kThreads / 32 ? warp_max[threadIdx.x] : 0u;
    m = __reduce_max_sync(0xffffffffu, m);
    if (threadIdx.x == 0 && m) atomicMax(amax_bits, m);
  }
}

// The amax accumulator (the bits of *g) starts at zero.
__global__ void tensor_scale_init(float* g) {
  griddep_wait_and_release();
  *reinterpret_cast<uint32_t*>(g) = 0u;
}

// g of an empty tensor.
__global__ void tensor_scale_finalize_empty(float* g) {
  griddep_wait_and_release();
  *g = 1.0f;
}

// g = amax / (6 * 448) in fp32, or 1 for an all-zero tensor.
__global__ void tensor_scale_finalize(float* g) {
  griddep_wait_and_release();
  const uint32_t bits = *reinterpret_cast<uint32_t*>(g);
  const float amax = __uint_as_float(bits << 16);
  *g = amax > 0.0f ? __fdiv_rn(amax, 2688.0f) : 1.0f;
}

// One thread quantizes one 16-element block: two 128-bit loads (the second
// half of the 32 bytes is in L1 after the first load of the warp), one scale
// computation, one 64-bit code store.  A warp covers 32 consecutive blocks.
// Where one pass of the quantizer reads: the thread's kUnroll 16-element
// blocks of the iteration that starts at the warp-uniform block index bidx0
// (block bidx0 + u * stride + lane).
struct BlockSlots {
  uint4 v0[kUnroll], v1[kUnroll];
  uint32_t row[kUnroll], kb[kUnroll];
};

__device__ __forceinline__ void load_blocks(const uint16_t* __restrict__ x, FastDiv kblocks_div, uint32_t total_blocks,
                                            int64_t ld, bool dense, uint32_t bidx0, uint32_t stride, uint32_t lane,
                                            BlockSlots& sl) {
  const uint32_t kblocks = kblocks_div.d;
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const uint32_t b = bidx0 + u * stride + lane;
    sl.row[u] = kblocks_div.div(b);
    sl.kb[u] = b - sl.row[u] * kblocks;
    const int64_t off = dense ? static_cast<int64_t>(b) * 16 : static_cast<int64_t>(sl.row[u]) * ld + sl.kb[u] * 16;
    const uint4* src = reinterpret_cast<const uint4*>(x + off);
    const bool live = b < total_blocks;
    sl.v0[u] = live ? __ldg(src) : make_uint4(0, 0, 0, 0);
    sl.v1[u] = live ? __ldg(src + 1) : make_uint4(0, 0, 0, 0);
  }
}

__device__ __forceinline__ uint32_t amax_bits_of(const BlockSlots& sl) {
  uint32_t m = 0;
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) m = max(m, max(amax_bits_bf16x8(sl.v0[u]), amax_bits_bf16x8(sl.v1[u])));
  return m;
}

// Quantize the loaded blocks with tensor scale g.  Every lane of the warp
// takes part (the MMA-layout scale gather shuffles across lanes).
template <bool kMMA>
__device__ __forceinline__ void quantize_loaded(const BlockSlots& sl, uint32_t total_blocks, uint32_t kblocks,
                                                uint32_t bidx0, uint32_t stride, uint32_t lane, float g, float six_g,
                                                bool g_ok, uint2* __restrict__ codes, uint8_t* __restrict__ scales, int* status) {
  const uint32_t kgroups = kblocks >> 2;
  // Scale bytes the kernel may write: padded rows in the MMA layout.
  const uint64_t scale_bytes =
      kMMA ? static_cast<uint64_t>((total_blocks / kblocks + 127u) & ~127u) * kblocks : total_blocks;
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const uint32_t b = bidx0 + u * stride + lane;
    const bool live = b < total_blocks;
    float xf[16];
    unpack_bf16x8(sl.v0[u], xf);
    unpack_bf16x8(sl.v1[u], xf + 8);
    const float amax = __uint_as_float(max(amax_bits_bf16x8(sl.v0[u]), amax_bits_bf16x8(sl.v1[u])) << 16);
    const BlockScale bs = block_scale(amax, g, six_g);
    float q[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) q[i] = __fmul_rn(xf[i], bs.mult);
    uint2 packed = make_uint2(e2m1x8(q), e2m1x8(q + 8));
    uint32_t sc = bs.code;
    if (!g_ok) { packed = make_uint2(0, 0); sc = 0; }
    if (live) codes[b] = packed;
    if (kMMA) {
      // Lanes 4j..4j+3 hold the four k-blocks of one MMA scale group (kblocks % 4 == 0,
      // so a group never straddles rows): assemble them into one 32-bit store.
      uint32_t w = sc << (8 * (lane & 3));
      w |= __shfl_xor_sync(0xffffffffu, w, 1);
      w |= __shfl_xor_sync(0xffffffffu, w, 2);
      const uint64_t off = mma_scale_offset(sl.row[u], sl.kb[u], kgroups);
      if (live && (lane & 3) == 0 && in_bounds(status, off % 4 == 0 && off + 4 <= scale_bytes))
        *reinterpret_cast<uint32_t*>(scales + off) = w;
    } else if (live) {
      const uint64_t off = static_cast<uint64_t>(sl.row[u]) * kblocks + sl.kb[u];
      if (in_bounds(status, off < scale_bytes)) scales[off] = static_cast<uint8_t>(sc);
    }
  }
}

// Zero the MMA-layout scales of the padding rows up to the next multiple of 128.
__device__ __forceinline__ void zero_scale_padding(uint32_t rows, uint32_t kblocks, uint8_t* __restrict__ scales,
                                                   int* status) {
  const uint32_t kgroups = kblocks >> 2;
  const uint32_t padded = (rows + 127u) & ~127u;
  const uint32_t pad = (padded - rows) * kblocks;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < pad; i += gridDim.x * blockDim.x) {
    const uint32_t r = rows + i / kblocks, k = i % kblocks;
    const uint64_t off = mma_scale_offset(r, k, kgroups);
    if (in_bounds(status, off < static_cast<uint64_t>(padded) * kblocks)) scales[off] = 0;
  }
}

// One thread quantizes one 16-element block per slot: two 128-bit loads (the
// second half of the 32 bytes is in L1 after the first load of the warp), one
// scale computation, one 64-bit code store.  A warp covers 32 consecutive
// blocks per slot.
template <bool kMMA>
__device__ __forceinline__ void quantize_blocks(const uint16_t* __restrict__ x, FastDiv kblocks_div,
                                                uint32_t total_blocks, int64_t ld, bool dense, uint32_t rows,
                                                float g, bool g_ok, uint2* __restrict__ codes,
                                                uint8_t* __restrict__ scales, int* status) {
  const float six_g = __fmul_rn(6.0f, g);
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t stride = gridDim.x * blockDim.x;
  // bidx0 is warp-uniform so every lane takes part in the scale gather.
  for (uint32_t bidx0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31u); bidx0 < total_blocks; bidx0 += stride * kUnroll) {
    BlockSlots sl;
    load_blocks(x, kblocks_div, total_blocks, ld, dense, bidx0, stride, lane, sl);
    quantize_loaded<kMMA>(sl, total_blocks, kblocks_div.d, bidx0, stride, lane, g, six_g, g_ok, codes, scales,
                          status);
  }
  if (kMMA) zero_scale_padding(rows, kblocks_div.d, scales, status);
}

template <bool kMMA>
__global__ void __launch_bounds__(kThreads) quantize_kernel(const uint16_t* __restrict__ x, FastDiv kblocks_div,
                                                            uint32_t total_blocks, int64_t ld, bool dense,
                                                            uint32_t rows, const float* __restrict__ g_ptr,
                                                            uint2* __restrict__ codes, uint8_t* __restrict__ scales,
                                                            int* status) {
  griddep_wait_and_release();
  const float g_in = *g_ptr;
  const bool g_ok = g_in > 0.0f && g_in <= FLT_MAX;
  if (!g_ok && blockIdx.x == 0 && threadIdx.x == 0) set_status(status, NVFP4_ERR_INVALID_ARG);
  quantize_blocks<kMMA>(x, kblocks_div, total_blocks, ld, dense, rows, g_ok ? g_in : 1.0f, g_ok, codes, scales,
                        status);
}

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// The waiting blocks need only the value of the word they poll (the release
// store carries the new epoch and the amax together), so they poll with
// relaxed loads: no acquire per poll.
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned long long atom_add_acq_rel_u64(unsigned long long* p, unsigned long long v) {
  unsigned long long old;
  asm volatile("atom.acq_rel.gpu.global.add.u64 %0, [%1], %2;" : "=l"(old) : "l"(p), "l"(v) : "memory");
  return old;
}
__device__ __forceinline__ void red_max_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("red.relaxed.gpu.global.max.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// a1 + a2 in one cooperative launch.  Phase 1 reduces amax(|x|) over the
// same 16-element blocks phase 2 quantizes; a grid-wide barrier separates
// them.  Caller-owned state (two 64-bit words, zero before the first call):
//   state[0] = (call epoch << 32) | (previous call's amax bits << 16) | blocks arrived
//   state[1] = (epoch << 32) | amax bits, combined with a max reduction
// A newer epoch's tag dominates any older value, so nothing is cleared
// between calls.  Each block max-reduces its amax into state[1], then counts
// itself into state[0] with an acquire-release add (the release orders the
// reduction before the count).  The last block to arrive reads the total
// amax (its acquire made every reduction visible) and opens the next epoch
// with one release store that also carries the amax, so the waiting blocks
// learn both from the load that ends their wait.  The epoch is read before
// the loads of phase 1: it cannot change until every block has arrived.
template <bool kMMA>
__global__ void __launch_bounds__(kThreads) quantize_dynamic_kernel(
    const uint16_t* __restrict__ x, FastDiv kblocks_div, uint32_t total_blocks, int64_t ld, bool dense, uint32_t rows,
    unsigned long long* state, float* __restrict__ g_out, uint2* __restrict__ codes, uint8_t* __restrict__ scales,
    int* status, int stash_iters) {
  // Shared-memory stash: the blocks of the first stash_iters phase-1
  // iterations, [iteration * kUnroll + slot][half][thread] as 16-byte words.
  extern __shared__ uint4 stash[];
  griddep_wait_and_release();
  timeline_stamp(0);
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t stride = gridDim.x * blockDim.x;
  unsigned long long epoch = 0;
  if (threadIdx.x == 0) epoch = ld_acquire_u64(&state[0]) >> 32;
  // Resident: one pass covers the tensor, so the loaded blocks stay in
  // registers across the barrier and x is read once.  Otherwise the blocks
  // of the last phase-1 iteration stay in registers, those of the first
  // stash_iters iterations in shared memory, and phase 2 reads from x again
  // only the iterations in between.
  const uint32_t bidx_first = blockIdx.x * blockDim.x + (threadIdx.x & ~31u);
  BlockSlots sl;
  uint32_t m = 0, bidx_last = bidx_first;
  int it = 0;
  for (uint32_t bidx0 = bidx_first; bidx0 < total_blocks || bidx0 == bidx_first; bidx0 += stride * kUnroll, ++it) {
    load_blocks(x, kblocks_div, total_blocks, ld, dense, bidx0, stride, lane, sl);
    m = max(m, amax_bits_of(sl));
    if (it < stash_iters) {
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        stash[((it * kUnroll + u) * 2) * kThreads + threadIdx.x] = sl.v0[u];
        stash[((it * kUnroll + u) * 2 + 1) * kThreads + threadIdx.x] = sl.v1[u];
      }
    }
    bidx_last = bidx0;
  }
  m = __reduce_max_sync(0xffffffffu, m);
  __shared__ uint32_t warp_max[kThreads / 32];
  __shared__ uint32_t s_amax;
#ifdef NVFP4_TIMELINE
  __syncthreads();
  timeline_stamp(1);
#endif
  __shared__ int s_ok;
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x < 32) {
    m = threadIdx.x < kThreads / 32 ? warp_max[threadIdx.x] : 0u;
    m = __reduce_max_sync(0xffffffffu, m);
    if (threadIdx.x == 0) {
      red_max_u64(&state[1], (epoch << 32) | m);
      const unsigned long long old = atom_add_acq_rel_u64(&state[0], 1ull);
      timeline_stamp(2);
      int ok = (old >> 32) == epoch;
      uint32_t amax_bits = 0;
      if (ok && static_cast<uint32_t>(old & 0xFFFFu) == gridDim.x - 1) {
        const unsigned long long a = ld_acquire_u64(&state[1]);
        ok = (a >> 32) == epoch;
        amax_bits = static_cast<uint32_t>(a) & 0xFFFFu;
        if (ok) st_release_u64(&state[0], ((epoch + 1) << 32) | (static_cast<unsigned long long>(amax_bits) << 16));
      } else if (ok) {
        // Every waiting block polls the one word the last arrival will
        // release; a short sleep between polls keeps the polls from queueing
        // ahead of the arrivals' atomics and the release store at L2.
        const uint64_t t0 = globaltimer_ns();
        unsigned long long v;
        for (uint32_t it = 0; ((v = ld_relaxed_u64(&state[0])) >> 32) == epoch; ++it) {
          __nanosleep(NVFP4_BARRIER_POLL_NS);
          if ((it & 63u) == 63u && globaltimer_ns() - t0 > kWaitLimitNs) { ok = 0; break; }
        }
        if (ok && (v >> 32) != epoch + 1) ok = 0;
        amax_bits = static_cast<uint32_t>(v >> 16) & 0xFFFFu;
      }
      if (!ok) set_status(status, NVFP4_ERR_TIMEOUT);
      s_amax = amax_bits;
      s_ok = ok;
    }
  }
  __syncthreads();
  timeline_stamp(3);
  if (!s_ok) return;
  const float amax = __uint_as_float(s_amax << 16);
  const float g = amax > 0.0f ? __fdiv_rn(amax, 2688.0f) : 1.0f;
  const float six_g = __fmul_rn(6.0f, g);
  if (blockIdx.x == 0 && threadIdx.x == 0) *g_out = g;
  if (bidx_last < total_blocks)
    quantize_loaded<kMMA>(sl, total_blocks, kblocks_div.d, bidx_last, stride, lane, g, six_g, true, codes, scales,
                          status);
  // The iterations between the stashed ones and the last are read from x
  // again, most recent first: when x does not fit in L2, phase 1 left the
  // latest of them in L2.  The stashed ones come from shared memory.
  const int n_iter = it;
  for (int k = n_iter - 2; k >= 0; --k) {
    const uint32_t bidx0 = bidx_first + static_cast<uint32_t>(k) * stride * kUnroll;
    BlockSlots t;
    if (k < stash_iters) {
      const uint32_t kblocks = kblocks_div.d;
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const uint32_t b = bidx0 + u * stride + lane;
        t.row[u] = kblocks_div.div(b);
        t.kb[u] = b - t.row[u] * kblocks;
        t.v0[u] = stash[((k * kUnroll + u) * 2) * kThreads + threadIdx.x];
        t.v1[u] = stash[((k * kUnroll + u) * 2 + 1) * kThreads + threadIdx.x];
      }
    } else {
      load_blocks(x, kblocks_div, total_blocks, ld, dense, bidx0, stride, lane, t);
    }
    quantize_loaded<kMMA>(t, total_blocks, kblocks_div.d, bidx0, stride, lane, g, six_g, true, codes, scales, status);
  }
  if (kMMA) zero_scale_padding(rows, kblocks_div.d, scales, status);
#ifdef NVFP4_TIMELINE
  __syncthreads();
  timeline_stamp(4);
#endif
}

// Blocks of quantize_dynamic_kernel that fit on the device at once (a
// cooperative launch must not exceed it).
// Shared-memory stash per block for one phase-1 iteration (kUnroll slots of
// two 16-byte words per thread), and the most iterations stashed.
constexpr size_t kStashIterBytes = static_cast<size_t>(kUnroll) * 2 * kThreads * 16;
constexpr int kMaxStashIters = 2;

template <bool kMMA>
int dynamic_capacity(int stash_iters) {
  static std::mutex mu;
  static std::map<std::pair<int, int>, int> cache;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find({d, stash_iters});
  if (it != cache.end()) return it->second;
  const size_t smem = stash_iters * kStashIterBytes;
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(quantize_dynamic_kernel<kMMA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kMaxStashIters * kStashIterBytes)) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, quantize_dynamic_kernel<kMMA>, kThreads, smem) !=
          cudaSuccess ||
      per_sm <= 0) {
    cudaGetLastError();
    return 0;
  }
  cache[{d, stash_iters}] = per_sm * sm_count();
  return cache[{d, stash_iters}];
}

// ---------------------------------------------------------------------------
// MXFP4 (Appendix A): E2M1 elements, one E8M0 scale per 32 elements, no
// global scale; optionally each 32-element block is first rotated by
// H_32 / sqrt(32) (the block-wise rotation applied before MXFP4 quantization,
// Sec. 4).  One thread quantizes one block per slot; no tensor-wide pass.
// ---------------------------------------------------------------------------
// Block index b (of rows * cols/32) -> its 32 bf16 elements as fp32, the row and block-in-row.
// U blocks per thread per pass: 1 when one pass covers the tensor (more CTAs
// to hide the load latency of small tensors), 2 for large ones.
template <bool kMMA, bool kRotate, int U>
__global__ void __launch_bounds__(kThreads) mx_quantize_kernel(const uint16_t* __restrict__ x, FastDiv nb_div,
                                                               uint32_t total_blocks, int64_t ld, bool dense,
                                                               uint32_t rows, uint4* __restrict__ codes,
                                                               uint8_t* __restrict__ scales, int* status) {
  griddep_wait_and_release();
  const uint32_t nb = nb_div.d;           // 32-element blocks per row
  const uint32_t kgroups = nb >> 1;       // 64-element scale groups per row (MMA layout)
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t stride = gridDim.x * blockDim.x;
  for (uint32_t b0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31u); b0 < total_blocks; b0 += stride * U) {
    uint4 v[U][4];
    uint32_t row[U], j[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t b = b0 + u * stride + lane;
      row[u] = nb_div.div(b);
      j[u] = b - row[u] * nb;
      const int64_t off = dense ? static_cast<int64_t>(b) * 32 : static_cast<int64_t>(row[u]) * ld + j[u] * 32;
      const uint4* src = reinterpret_cast<const uint4*>(x + off);
      const bool live = b < total_blocks;
#pragma unroll
      for (int q = 0; q < 4; ++q) v[u][q] = live ? __ldg(src + q) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint32_t b = b0 + u * stride + lane;
      const bool live = b < total_blocks;
      float xf[32];
#pragma unroll
      for (int q = 0; q < 4; ++q) unpack_bf16x8(v[u][q], xf + 8 * q);
      if (kRotate) hadamard32(xf);
      float amax = 0.0f;
#pragma unroll
      for (int i = 0; i < 32; ++i) amax = fmaxf(amax, fabsf(xf[i]));
      const uint32_t code = mx_scale_code(amax);
      const float inv_scale = mx_inv_scale(code);
#pragma unroll
      for (int i = 0; i < 32; ++i) xf[i] = __fmul_rn(xf[i], inv_scale);
      const uint4 packed = make_uint4(e2m1x8(xf), e2m1x8(xf + 8), e2m1x8(xf + 16), e2m1x8(xf + 24));
      if (live) codes[b] = packed;
      if (kMMA) {
        // The 16-element-block MMA layout with each E8M0 scale stored for both
        // halves of its block: lanes 2i, 2i+1 hold the two blocks of one
        // 64-element group (nb is even, so a group never straddles rows).
        uint32_t w = (code | (code << 8)) << (16 * (lane & 1));
        w |= __shfl_xor_sync(0xffffffffu, w, 1);
        const uint64_t off = mma_scale_offset(row[u], 2 * j[u], kgroups);
        if (live && (lane & 1) == 0 &&
            in_bounds(status, off % 4 == 0 && off + 4 <= static_cast<uint64_t>((rows + 127u) & ~127u) * 2 * nb))
          *reinterpret_cast<uint32_t*>(scales + off) = w;
      } else if (live) {
        const uint64_t off = static_cast<uint64_t>(row[u]) * nb + j[u];
        if (in_bounds(status, off < total_blocks)) scales[off] = static_cast<uint8_t>(code);
      }
    }
  }
  if (kMMA) zero_scale_padding(rows, nb * 2, scales, status);
}

template <bool kToMMA>
__global__ void relayout_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst, uint32_t rows,
                                uint32_t kblocks) {
  griddep_wait_and_release();
  const uint32_t kgroups = kblocks >> 2;
  const uint32_t padded = (rows + 127u) & ~127u;
  const uint32_t n = padded * kblocks;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const uint32_t r = i / kblocks, kb = i % kblocks;
    const uint64_t m = mma_scale_offset(r, kb, kgroups);
    if (kToMMA) {
      dst[m] = r < rows ? src[i] : 0;
    } else if (r < rows) {
      dst[i] = src[m];
    }
  }
}

int grid_for(uint64_t work_items, int threads) {
  const uint64_t want = (work_items + threads - 1) / threads;
  const uint64_t cap = static_cast<uint64_t>(sm_count()) * 8;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

nvfp4_status check_bf16_matrix(const void* x, int64_t rows, int64_t cols, int64_t ld, int64_t col_mult) {
  if (!x && rows * cols != 0) return NVFP4_ERR_INVALID_ARG;
  if (rows < 0 || cols < 0 || ld < cols || cols % col_mult) return NVFP4_ERR_SHAPE;
  if (rows * (cols / 8) >= (1ll << 32) || rows >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(x, 16) || ld % 8) return NVFP4_ERR_ALIGN;
  return NVFP4_OK;
}

ChunkMap make_map(int64_t rows, int64_t cols, int64_t ld) {
  ChunkMap m;
  m.cpr = FastDiv(static_cast<uint32_t>(cols / 8 > 0 ? cols / 8 : 1));
  m.total = static_cast<uint32_t>(rows * (cols / 8));
  m.ld = ld;
  m.dense = (ld == cols);
  return m;
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API size_t nvfp4_scales_bytes(int64_t rows, int64_t cols, nvfp4_scale_layout layout) {
  if (rows < 0 || cols < 0) return 0;
  const int64_t r = layout == NVFP4_SCALES_MMA ? ((rows + 127) / 128) * 128 : rows;
  return static_cast<size_t>(r * (cols / 16));
}

NVFP4_API nvfp4_status nvfp4_tensor_scale(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld,
                                          float* g_dev, void* stream) {
  NVFP4_TRACE("nvfp4_tensor_scale");
  if (!g_dev) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = check_bf16_matrix(x_bf16, rows, cols, ld, 8);
  if (st != NVFP4_OK) return st;
  if (!aligned(g_dev, 4)) return NVFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (launch_pdl(tensor_scale_init, dim3(1), dim3(1), 0, s, g_dev) != cudaSuccess) return NVFP4_ERR_CUDA;
  count_launches(1);
  const ChunkMap map = make_map(rows, cols, ld);
  if (map.total) {
    if (launch_pdl(amax_kernel, dim3(grid_for(map.total, kThreads * kUnroll)), dim3(kThreads), 0, s,
                   static_cast<const uint16_t*>(x_bf16), map, reinterpret_cast<uint32_t*>(g_dev)) != cudaSuccess)
      return NVFP4_ERR_CUDA;
    count_launches(1);
  }
  if (launch_pdl(tensor_scale_finalize, dim3(1), dim3(1), 0, s, g_dev) != cudaSuccess) return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

NVFP4_API nvfp4_status nvfp4_quantize(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld,
                                      const float* g_dev, uint8_t* codes, uint8_t* scales,
                                      nvfp4_scale_layout layout, void* stream) {
  NVFP4_TRACE("nvfp4_quantize");
  if (layout != NVFP4_SCALES_ROWMAJOR && layout != NVFP4_SCALES_MMA) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = check_bf16_matrix(x_bf16, rows, cols, ld, layout == NVFP4_SCALES_MMA ? 64 : 16);
  if (st != NVFP4_OK) return st;
  if (rows == 0 || cols == 0) return NVFP4_OK;
  if (!g_dev || !codes || !scales) return NVFP4_ERR_INVALID_ARG;
  if (!aligned(codes, 8) || !aligned(g_dev, 4)) return NVFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const uint32_t kblocks = static_cast<uint32_t>(cols / 16);
  const uint32_t total_blocks = static_cast<uint32_t>(rows * kblocks);
  const int grid = grid_for(total_blocks, kThreads * kUnroll);
  const bool dense = (ld == cols);
  cudaError_t e = launch_pdl(layout == NVFP4_SCALES_MMA ? quantize_kernel<true> : quantize_kernel<false>, dim3(grid),
                             dim3(kThreads), 0, s, static_cast<const uint16_t*>(x_bf16), FastDiv(kblocks),
                             total_blocks, ld, dense, static_cast<uint32_t>(rows), g_dev,
                             reinterpret_cast<uint2*>(codes), scales, status_word_dev());
  if (e != cudaSuccess) return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

NVFP4_API nvfp4_status nvfp4_quantize_dynamic(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld,
                                              void* state_dev, float* g_dev, uint8_t* codes, uint8_t* scales,
                                              nvfp4_scale_layout layout, void* stream) {
  NVFP4_TRACE("nvfp4_quantize_dynamic");
  if (layout != NVFP4_SCALES_ROWMAJOR && layout != NVFP4_SCALES_MMA) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = check_bf16_matrix(x_bf16, rows, cols, ld, layout == NVFP4_SCALES_MMA ? 64 : 16);
  if (st != NVFP4_OK) return st;
  if (!state_dev || !g_dev) return NVFP4_ERR_INVALID_ARG;
  if (!aligned(state_dev, 16) || !aligned(g_dev, 4)) return NVFP4_ERR_ALIGN;
  if (rows == 0 || cols == 0) {
    // Nothing to quantize; the tensor scale of an empty tensor is 1.
    if (launch_pdl(tensor_scale_finalize_empty, dim3(1), dim3(1), 0, static_cast<cudaStream_t>(stream), g_dev) !=
        cudaSuccess)
      return NVFP4_ERR_CUDA;
    count_launches(1);
    return launch_status();
  }
  if (!codes || !scales) return NVFP4_ERR_INVALID_ARG;
  if (!aligned(codes, 8)) return NVFP4_ERR_ALIGN;
  const bool mma = layout == NVFP4_SCALES_MMA;
  const uint32_t kblocks = static_cast<uint32_t>(cols / 16);
  const uint32_t total_blocks = static_cast<uint32_t>(rows * kblocks);
  // kUnroll blocks per thread per pass, as few CTAs as that allows (each CTA
  // is one arrival at the grid barrier); x stays in registers across the
  // barrier when one pass covers it, and up to kMaxStashIters more passes
  // wait in shared memory.
  int grid = grid_for(total_blocks, kThreads * kUnroll);
  int cap = mma ? dynamic_capacity<true>(0) : dynamic_capacity<false>(0);
  if (cap <= 0) return NVFP4_ERR_CUDA;
  int stash_iters = 0;
  if (grid > cap) {
    const int cap_stash = mma ? dynamic_capacity<true>(kMaxStashIters) : dynamic_capacity<false>(kMaxStashIters);
    if (cap_stash > 0) {
      const uint64_t per_iter = static_cast<uint64_t>(cap_stash) * kThreads * kUnroll;
      const uint64_t iters = (total_blocks + per_iter - 1) / per_iter;
      stash_iters = static_cast<int>(iters - 1 < kMaxStashIters ? iters - 1 : kMaxStashIters);
      cap = cap_stash;
    }
  }
  if (grid > cap) grid = cap;
  if (grid > 0xFFFF) grid = 0xFFFF;  // the barrier counts arrivals in 16 bits
  // Cooperative: every block is resident at once, so the grid barrier can
  // complete.  A plain launch with programmatic dependent launch (the grid is
  // capped at the co-resident blocks anyway) was measured too: 2-4 us faster
  // per four back-to-back quantizations, but slower inside a step that
  // alternates quantizations and GEMMs (32B prefill layer: 1697 vs 1658-1679
  // us graph-replayed), so the cooperative launch stays.
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = stash_iters * kStashIterBytes;
  cfg.stream = static_cast<cudaStream_t>(stream);
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e =
      cudaLaunchKernelEx(&cfg, mma ? quantize_dynamic_kernel<true> : quantize_dynamic_kernel<false>,
                         static_cast<const uint16_t*>(x_bf16), FastDiv(kblocks), total_blocks, ld, ld == cols,
                         static_cast<uint32_t>(rows), static_cast<unsigned long long*>(state_dev), g_dev,
                         reinterpret_cast<uint2*>(codes), scales, status_word_dev(), stash_iters);
  if (e != cudaSuccess) return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

NVFP4_API nvfp4_status nvfp4_scales_relayout(const uint8_t* src, uint8_t* dst, int64_t rows, int64_t cols,
                                             nvfp4_scale_layout from, nvfp4_scale_layout to, void* stream) {
  NVFP4_TRACE("nvfp4_scales_relayout");
  if (!src || !dst) return NVFP4_ERR_INVALID_ARG;
  if ((from != NVFP4_SCALES_ROWMAJOR && from != NVFP4_SCALES_MMA) ||
      (to != NVFP4_SCALES_ROWMAJOR && to != NVFP4_SCALES_MMA))
    return NVFP4_ERR_INVALID_ARG;
  if (rows < 0 || cols < 0 || cols % 64 || rows >= (1ll << 24)) return NVFP4_ERR_SHAPE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t bytes = nvfp4_scales_bytes(rows, cols, from);
  if (from == to) {
    if (bytes && cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, s) != cudaSuccess) return NVFP4_ERR_CUDA;
    return NVFP4_OK;
  }
  if (rows == 0 || cols == 0) return NVFP4_OK;
  const uint32_t kblocks = static_cast<uint32_t>(cols / 16);
  const uint64_t n = static_cast<uint64_t>((rows + 127) / 128 * 128) * kblocks;
  if (launch_pdl(to == NVFP4_SCALES_MMA ? relayout_kernel<true> : relayout_kernel<false>, dim3(grid_for(n, 256)),
                 dim3(256), 0, s, src, dst, static_cast<uint32_t>(rows), kblocks) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

NVFP4_API size_t mxfp4_scales_bytes(int64_t rows, int64_t cols, nvfp4_scale_layout layout) {
  if (rows < 0 || cols < 0) return 0;
  if (layout == NVFP4_SCALES_MMA) return nvfp4_scales_bytes(rows, cols, layout);
  return static_cast<size_t>(rows * (cols / 32));
}

NVFP4_API nvfp4_status mxfp4_quantize(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld, int rotate,
                                      uint8_t* codes, uint8_t* scales, nvfp4_scale_layout layout, void* stream) {
  NVFP4_TRACE("mxfp4_quantize");
  if (layout != NVFP4_SCALES_ROWMAJOR && layout != NVFP4_SCALES_MMA) return NVFP4_ERR_INVALID_ARG;
  if (rotate != 0 && rotate != 1) return NVFP4_ERR_INVALID_ARG;
  nvfp4_status st = check_bf16_matrix(x_bf16, rows, cols, ld, layout == NVFP4_SCALES_MMA ? 64 : 32);
  if (st != NVFP4_OK) return st;
  if (rows == 0 || cols == 0) return NVFP4_OK;
  if (!codes || !scales) return NVFP4_ERR_INVALID_ARG;
  if (!aligned(codes, 16)) return NVFP4_ERR_ALIGN;
  const uint32_t nb = static_cast<uint32_t>(cols / 32);
  const uint32_t total_blocks = static_cast<uint32_t>(rows * nb);
  const bool mma = layout == NVFP4_SCALES_MMA;
  const bool one_pass = total_blocks <= static_cast<uint64_t>(sm_count()) * 8 * kThreads;
  const int grid = grid_for(total_blocks, kThreads * (one_pass ? 1 : 2));
  auto kernel = one_pass ? (mma ? (rotate ? mx_quantize_kernel<true, true, 1> : mx_quantize_kernel<true, false, 1>)
                                : (rotate ? mx_quantize_kernel<false, true, 1> : mx_quantize_kernel<false, false, 1>))
                         : (mma ? (rotate ? mx_quantize_kernel<true, true, 2> : mx_quantize_kernel<true, false, 2>)
                                : (rotate ? mx_quantize_kernel<false, true, 2> : mx_quantize_kernel<false, false, 2>));
  const cudaError_t e = launch_pdl(kernel, dim3(grid), dim3(kThreads), 0, static_cast<cudaStream_t>(stream),
                                   static_cast<const uint16_t*>(x_bf16), FastDiv(nb), total_blocks, ld, ld == cols,
                                   static_cast<uint32_t>(rows), reinterpret_cast<uint4*>(codes), scales,
                                   status_word_dev());
  if (e != cudaSuccess) return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

#ifdef NVFP4_TIMELINE
// Timeline build only (not part of the C ABI of include/nvfp4.h): copy the
// per-block stamps of the last nvfp4_quantize_dynamic launch to host memory
// ([2048][5] uint64, nanoseconds, zero where a block did not run), then clear
// them.  Synchronizes the device.
extern "C" __attribute__((visibility("default"))) int nvfp4_timeline_quantize_dynamic(unsigned long long* host) {
  if (cudaDeviceSynchronize() != cudaSuccess) return 1;
  if (cudaMemcpyFromSymbol(host, nvfp4::g_quantize_timeline, sizeof(nvfp4::g_quantize_timeline)) != cudaSuccess)
    return 1;
  static unsigned long long zero[nvfp4::kTimelineBlocks * 5];
  return cudaMemcpyToSymbol(nvfp4::g_quantize_timeline, zero, sizeof(zero)) == cudaSuccess ? 0 : 1;
}
#endif
