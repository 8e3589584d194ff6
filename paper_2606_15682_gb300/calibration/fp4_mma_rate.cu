// Calibration: the rate at which one SM retires block-scaled NVFP4 MMAs
// (tcgen05.mma kind::mxf4nvf4, scale_vec::4X, E2M1 operands, UE4M3 scales),
// the ceiling for the linear-layer GEMM.  Not part of the library.
//
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -std=c++17 \
//        -o fp4_mma_rate paper_2606_15682_gb300/calibration/fp4_mma_rate.cu && ./fp4_mma_rate
//
// One thread per CTA (one CTA per SM) issues ITERS x 4 back-to-back MMAs of
// 128 x 256 x 64 (or, for the CTA pair, 256 x 256 x 64 over two SMs) into one
// TMEM accumulator, from operands resident in shared memory, then waits for
// their completion on an mbarrier (bounded by 2 s).  Reported: SM cycles per
// MMA, FP4 FLOP per cycle per SM, the SM clock (clock64 against globaltimer),
// and the whole-GPU rate from CUDA events.  Operand bytes are filled with a
// hash so the tensor cores see random codes; scales are 1.0.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>

namespace {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t gtimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}
// K-major operand tile with the 128-byte swizzle: rows of 128 B, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (1ull << 16) | (static_cast<uint64_t>(1024 >> 4) << 32) |
         (1ull << 46) | (2ull << 61);
}

constexpr int kIters = 100000;
constexpr size_t kSmem = 120 * 1024;  // operands use 49 KB; the rest keeps one CTA per SM

// PAIR = false: cta_group::1, M = 128, N = 256.  PAIR = true: cta_group::2, M = 256, N = 256.
template <bool PAIR>
__global__ void __launch_bounds__(128, 1) mma_rate(unsigned long long* out, int* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t slot;
  const int warp = threadIdx.x >> 5;
  uint32_t rank = 0;
  if (PAIR) asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const uint32_t m = PAIR ? 256 : 128;
  const uint32_t idesc = (1u << 7) | (1u << 10) | (256u >> 3 << 17) | ((m >> 4) << 24);
  for (int i = threadIdx.x; i < (16384 + 32768) / 4; i += blockDim.x) {
    uint32_t x = static_cast<uint32_t>(i) * 2654435761u + blockIdx.x * 97u;
    x ^= x >> 15;
    x *= 2246822519u;
    x ^= x >> 13;
    reinterpret_cast<uint32_t*>(smem)[i] = x;
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&bar)));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    if (PAIR) {
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(smem_u32(&slot)) : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(smem_u32(&slot)) : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  if (PAIR) asm volatile("barrier.cluster.arrive.release.aligned; barrier.cluster.wait.acquire.aligned;" ::: "memory");
  else __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = slot;
  {  // scales 1.0 (E4M3 0x38) in columns 256..303; each warp writes its own TMEM lane quadrant
    const uint32_t v = 0x38383838u;
    for (int c = 0; c < 48; c += 16)
      asm volatile(
          "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1,%1};" ::"r"(
              tmem + (static_cast<uint32_t>(warp * 32) << 16) + 256 + c),
          "r"(v)
          : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  if (PAIR) asm volatile("barrier.cluster.arrive.release.aligned; barrier.cluster.wait.acquire.aligned;" ::: "memory");
  else __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

  const uint64_t t0 = gtimer();
  const unsigned long long c0 = clock64();
  if (threadIdx.x == 0 && rank == 0) {
    const uint32_t sA = smem_u32(smem), sB = sA + 16384;
    const uint32_t sf = tmem + 256;
    for (int i = 0; i < kIters; ++i) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t a = desc_sw128(sA + kk * 32), b = desc_sw128(sB + kk * 32);
        const uint32_t acc = (i | kk) != 0;
        if (PAIR)
          asm volatile(
              "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
              " tcgen05.mma.cta_group::2.kind::mxf4nvf4.block_scale.scale_vec::4X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(
                  tmem),
              "l"(a), "l"(b), "r"(idesc), "r"(acc), "r"(sf + kk * 4), "r"(sf + 16 + kk * 8)
              : "memory");
        else
          asm volatile(
              "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
              " tcgen05.mma.cta_group::1.kind::mxf4nvf4.block_scale.scale_vec::4X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(
                  tmem),
              "l"(a), "l"(b), "r"(idesc), "r"(acc), "r"(sf + kk * 4), "r"(sf + 16 + kk * 8)
              : "memory");
      }
    }
    if (PAIR)
      asm volatile(
          "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
              smem_u32(&bar)),
          "h"(static_cast<uint16_t>(3))
          : "memory");
    else
      asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(&bar))
                   : "memory");
  }
  if (threadIdx.x == 0) {
    uint32_t ok = 0;
    for (uint32_t it = 0; !ok; ++it) {
      asm volatile(
          "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
          : "=r"(ok)
          : "r"(smem_u32(&bar))
          : "memory");
      if ((it & 1023u) == 0 && gtimer() - t0 > 2000000000ull) break;
    }
    if (!ok) atomicExch(err, 1);
    if (blockIdx.x == 0) {
      out[0] = clock64() - c0;
      out[1] = gtimer() - t0;
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  if (PAIR) asm volatile("barrier.cluster.arrive.release.aligned; barrier.cluster.wait.acquire.aligned;" ::: "memory");
  else __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 0) {
    if (PAIR) asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
    else asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem) : "memory");
  }
}

template <bool PAIR>
int run(int sms) {
  if (cudaFuncSetAttribute(mma_rate<PAIR>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kSmem)) !=
      cudaSuccess)
    return 1;
  unsigned long long* out = nullptr;
  int* err = nullptr;
  if (cudaMalloc(&out, 16) != cudaSuccess || cudaMalloc(&err, 4) != cudaSuccess) return 1;
  cudaMemset(err, 0, 4);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = PAIR ? 2 : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(sms & ~1);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = kSmem;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaEvent_t e0, e1;
  cudaEventCreate(&e0);
  cudaEventCreate(&e1);
  cudaLaunchKernelEx(&cfg, mma_rate<PAIR>, out, err);  // warm-up
  cudaEventRecord(e0);
  cudaLaunchKernelEx(&cfg, mma_rate<PAIR>, out, err);
  cudaEventRecord(e1);
  const cudaError_t ce = cudaDeviceSynchronize();
  unsigned long long h[2] = {0, 0};
  int he = 0;
  cudaMemcpy(h, out, 16, cudaMemcpyDeviceToHost);
  cudaMemcpy(&he, err, 4, cudaMemcpyDeviceToHost);
  float ms = 0.0f;
  cudaEventElapsedTime(&ms, e0, e1);
  const double mmas = 4.0 * kIters;
  const double flop_per_sm_per_mma = 2.0 * 128 * 256 * 64;  // each SM's share, both forms
  const int ctas = sms & ~1;
  std::printf("%-32s %6.1f cycles/MMA  %6.0f FP4 FLOP/cycle/SM  SM clock %4.0f MHz  %5.2f PFLOP/s (%d SMs)  %s%s\n",
              PAIR ? "cta_group::2, 256x256x64" : "cta_group::1, 128x256x64", h[0] / mmas,
              flop_per_sm_per_mma * mmas / h[0], h[0] / static_cast<double>(h[1]) * 1e3,
              flop_per_sm_per_mma * mmas * ctas / (ms * 1e-3) / 1e15, ctas, cudaGetErrorString(ce),
              he ? "  (wait timed out)" : "");
  cudaFree(out);
  cudaFree(err);
  return ce != cudaSuccess || he;
}

}  // namespace

int main() {
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0) != cudaSuccess) return 1;
  return run<false>(sms) | run<true>(sms);
}
