// a3: block-scaled NVFP4 x NVFP4 linear layer with bf16 output, on the
// 5th-generation tensor cores (tcgen05.mma kind::mxf4nvf4, 16-element blocks
// with UE4M3 scales, fp32 accumulation in tensor memory).
//
//   out[m, n] = bf16( g_a g_w sum_k a[m,k] w[n,k] )      (all linears, Appendix D.1)
//
// Persistent, warp-specialized CTA (one per SM), tile 128 x 128 x 256:
//   warp 0      TMA producer: codes via 2-D tensor maps (128-byte swizzle),
//               block-scale atoms via 1-D bulk copies, into a 5-stage ring.
//   warp 1      allocates 512 TMEM columns; one lane copies the stage's scales
//               smem -> TMEM (tcgen05.cp) and issues 4 MMAs of K = 64 per stage.
//   warps 2..5  epilogue: tcgen05.ld the accumulator (double-buffered in TMEM so
//               the next tile's MMAs overlap it), scale by g_a g_w, round to
//               bf16, store.
// Every wait is bounded (NVFP4_ERR_TIMEOUT on expiry); the CTA then drains
// its copies and MMAs and frees TMEM before returning.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cfloat>
#include <mutex>

#include "common.cuh"

namespace nvfp4 {
namespace {

constexpr int BM = 128;
constexpr int BN = 128;
constexpr int BK = 256;                  // elements per k-block = 128 bytes per row
constexpr int kStages = 5;
constexpr int kThreads = 192;
constexpr uint32_t kTileBytesA = BM * BK / 2;  // 16 KiB
constexpr uint32_t kTileBytesB = BN * BK / 2;  // 16 KiB
constexpr uint32_t kSfBytes = 128 * (BK / 16); // 2 KiB: four 512-byte scale atoms
constexpr uint32_t kStageBytes = kTileBytesA + kTileBytesB + 2 * kSfBytes;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSfTmemCol = 2 * BN;        // scale slots after the two accumulators
constexpr size_t kSmemBytes = 1024 /*align slack*/ + kStages * kStageBytes + 256 /*barriers*/;

static_assert(kSfTmemCol + kStages * 32 <= kTmemCols, "TMEM budget");

// Instruction descriptor, kind::mxf4nvf4: A and B are packed E2M1 (format 1),
// both K-major, scale type UE4M3 (bit 23 = 0), N >> 3 at bit 17, M >> 4 at bit 24.
constexpr uint32_t kIdesc = (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
                            (static_cast<uint32_t>(BM >> 4) << 24);

// Shared-memory matrix descriptor of a K-major operand tile stored with the
// 128-byte swizzle: rows of 128 B, 8-row groups 1024 B apart (SBO).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (1ull << 16) | (static_cast<uint64_t>(1024 >> 4) << 32) |
         (1ull << 46) | (2ull << 61);
}
// Descriptor of one 512-byte scale atom: 32 rows of 16 B, no swizzle, 8-row
// core matrices 128 B apart.
__device__ __forceinline__ uint64_t desc_sf(uint32_t saddr) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) | (static_cast<uint64_t>(128 >> 4) << 16) |
         (static_cast<uint64_t>(128 >> 4) << 32) | (1ull << 46);
}

__device__ __forceinline__ void mma_fp4(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t sfa, uint32_t sfb,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::mxf4nvf4.block_scale.scale_vec::4X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate), "r"(sfa), "r"(sfb)
      : "memory");
}

__device__ __forceinline__ void copy_sf_to_tmem(uint32_t taddr, uint64_t desc) {
  asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(desc) : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t r[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
      "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

struct GemmArgs {
  const uint8_t* sfa;
  const uint8_t* sfb;
  const float* ga;
  const float* gb;
  uint16_t* out;
  int64_t ldo;
  int M, N, K;
  int tiles_m, tiles_n;
  int* status;
};

__global__ void __launch_bounds__(kThreads, 1)
    nvfp4_gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                      const GemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + kStages * kTileBytesA;
  uint8_t* sSFA = sB + kStages * kTileBytesB;
  uint8_t* sSFB = sSFA + kStages * kSfBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sSFB + kStages * kSfBytes);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kblocks = args.K / BK;
  const int kgroups = args.K / 64;
  const int total_tiles = args.tiles_m * args.tiles_n;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 4);
    }
    mbar_init(drain, 1);
    abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmap_a);
    prefetch_tmap(&tmap_b);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  auto fail = [&]() {
    set_status(args.status, NVFP4_ERR_TIMEOUT);
    abort_flag = 1;
  };

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------ TMA producer ---
    int stage = 0;
    uint32_t phase = 0;
    uint32_t issued_parity[kStages];
    bool issued[kStages];
    for (int s = 0; s < kStages; ++s) issued[s] = false;
    for (int tile = blockIdx.x; tile < total_tiles && !abort_flag; tile += gridDim.x) {
      const int mb = tile % args.tiles_m, nb = tile / args.tiles_m;
      const uint8_t* sfa_tile = args.sfa + (static_cast<size_t>(mb) * kgroups) * 512;
      const uint8_t* sfb_tile = args.sfb + (static_cast<size_t>(nb) * kgroups) * 512;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, &abort_flag)) { fail(); break; }
        mbar_arrive_expect_tx(&full[stage], kStageBytes);
        tma_load_2d(sA + stage * kTileBytesA, &tmap_a, &full[stage], kb * (BK / 2), mb * BM);
        tma_load_2d(sB + stage * kTileBytesB, &tmap_b, &full[stage], kb * (BK / 2), nb * BN);
        bulk_load(sSFA + stage * kSfBytes, sfa_tile + static_cast<size_t>(kb) * kSfBytes, kSfBytes, &full[stage]);
        bulk_load(sSFB + stage * kSfBytes, sfb_tile + static_cast<size_t>(kb) * kSfBytes, kSfBytes, &full[stage]);
        issued[stage] = true;
        issued_parity[stage] = phase;
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
    }
    if (abort_flag) {
      // Let every copy this thread started land before the CTA exits.
      for (int s = 0; s < kStages; ++s)
        if (issued[s]) mbar_wait_bounded(&full[s], issued_parity[s], nullptr);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------- MMA issuer ---
    int stage = 0;
    uint32_t phase = 0;
    int local = 0;
    const uint32_t sA0 = smem_u32(sA), sB0 = smem_u32(sB), sSFA0 = smem_u32(sSFA), sSFB0 = smem_u32(sSFB);
    for (int tile = blockIdx.x; tile < total_tiles && !abort_flag; tile += gridDim.x, ++local) {
      const int acc = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      if (!mbar_wait_bounded(&tempty[acc], acc_phase ^ 1u, &abort_flag)) { fail(); break; }
      tc_fence_after();
      const uint32_t d_tmem = tmem + acc * BN;
      bool ok = true;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&full[stage], phase, &abort_flag)) { fail(); ok = false; break; }
        tc_fence_after();
        const uint32_t sf_col = tmem + kSfTmemCol + stage * 32;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          copy_sf_to_tmem(sf_col + kk * 4, desc_sf(sSFA0 + stage * kSfBytes + kk * 512));
          copy_sf_to_tmem(sf_col + 16 + kk * 4, desc_sf(sSFB0 + stage * kSfBytes + kk * 512));
        }
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          mma_fp4(d_tmem, desc_sw128(sA0 + stage * kTileBytesA + kk * 32), desc_sw128(sB0 + stage * kTileBytesB + kk * 32),
                  sf_col + kk * 4, sf_col + 16 + kk * 4, (kb | kk) != 0);
        }
        tc_commit(&empty[stage]);
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      tc_commit(&tfull[acc]);
    }
    // Wait until every MMA issued above has retired before TMEM is freed.
    tc_commit(drain);
    mbar_wait_bounded(drain, 0, nullptr);
  } else if (warp >= 2) {
    // --------------------------------------------------------- epilogue ---
    const int quarter = warp & 3;  // TMEM lanes this warp may access
    const float scale = __fmul_rn(__ldg(args.ga), __ldg(args.gb));
    int local = 0;
    for (int tile = blockIdx.x; tile < total_tiles; tile += gridDim.x, ++local) {
      const int mb = tile % args.tiles_m, nb = tile / args.tiles_m;
      const int acc = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      // Lane 0 waits and broadcasts, so the warp stays converged for the
      // .sync.aligned TMEM loads below even on the timeout path.
      int ok = 1;
      if (lane == 0) {
        ok = !abort_flag && mbar_wait_bounded(&tfull[acc], acc_phase, &abort_flag);
        if (!ok && !abort_flag) fail();
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
      tc_fence_after();
      const int row = mb * BM + quarter * 32 + lane;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(taddr + c * 32, r);
        const int col0 = nb * BN + c * 32;
        if (row < args.M) {
          uint16_t* dst = args.out + static_cast<int64_t>(row) * args.ldo + col0;
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            if (col0 + v * 8 < args.N) {
              uint4 w;
              w.x = pack_bf16x2(__uint_as_float(r[8 * v + 0]) * scale, __uint_as_float(r[8 * v + 1]) * scale);
              w.y = pack_bf16x2(__uint_as_float(r[8 * v + 2]) * scale, __uint_as_float(r[8 * v + 3]) * scale);
              w.z = pack_bf16x2(__uint_as_float(r[8 * v + 4]) * scale, __uint_as_float(r[8 * v + 5]) * scale);
              w.w = pack_bf16x2(__uint_as_float(r[8 * v + 6]) * scale, __uint_as_float(r[8 * v + 7]) * scale);
              reinterpret_cast<uint4*>(dst)[v] = w;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ------------------------------------------------------------------- host ---

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Row-major [rows, K/2] byte matrix, box of 128 bytes x box_rows rows, 128-B swizzle.
bool make_code_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t K, uint32_t box_rows) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K / 2), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(K / 2)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK / 2), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool ensure_smem_attr() {
  static bool done[64] = {};
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= 64) return false;
  if (!done[d]) {
    if (cudaFuncSetAttribute(nvfp4_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kSmemBytes)) != cudaSuccess)
      return false;
    done[d] = true;
  }
  return true;
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API nvfp4_status nvfp4_linear(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a,
                                    const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w, int64_t M,
                                    int64_t N, int64_t K, void* out_bf16, int64_t ldo, void* stream) {
  if (!a_codes || !a_scales || !g_a || !w_codes || !w_scales || !g_w || !out_bf16) return NVFP4_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0 || K % BK || N % 16 || ldo < N || ldo % 8) return NVFP4_ERR_SHAPE;
  if (M >= (1ll << 31) || N >= (1ll << 31) || K >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(a_scales, 16) || !aligned(w_scales, 16) ||
      !aligned(out_bf16, 16) || !aligned(g_a, 4) || !aligned(g_w, 4))
    return NVFP4_ERR_ALIGN;
  const int64_t tiles_m = (M + BM - 1) / BM, tiles_n = (N + BN - 1) / BN;
  if (tiles_m * tiles_n >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  CUtensorMap ma, mb;
  if (!make_code_map(&ma, a_codes, M, K, BM) || !make_code_map(&mb, w_codes, N, K, BN)) return NVFP4_ERR_CUDA;
  if (!ensure_smem_attr()) return NVFP4_ERR_CUDA;
  GemmArgs args;
  args.sfa = a_scales;
  args.sfb = w_scales;
  args.ga = g_a;
  args.gb = g_w;
  args.out = static_cast<uint16_t*>(out_bf16);
  args.ldo = ldo;
  args.M = static_cast<int>(M);
  args.N = static_cast<int>(N);
  args.K = static_cast<int>(K);
  args.tiles_m = static_cast<int>(tiles_m);
  args.tiles_n = static_cast<int>(tiles_n);
  args.status = status_word_dev();
  const int64_t tiles = tiles_m * tiles_n;
  const int grid = static_cast<int>(tiles < sm_count() ? tiles : sm_count());
  nvfp4_gemm_kernel<<<grid, kThreads, kSmemBytes, static_cast<cudaStream_t>(stream)>>>(ma, mb, args);
  count_launches(1);
  return launch_status();
}
