// a3: block-scaled NVFP4 x NVFP4 linear layer with bf16 output, on the
// 5th-generation tensor cores (tcgen05.mma kind::mxf4nvf4, 16-element blocks
// with UE4M3 scales, fp32 accumulation in tensor memory).
//
//   out[m, n] = bf16( g_a g_w sum_k a[m,k] w[n,k] )      (all linears, Appendix D.1)
//
// Persistent, warp-specialized CTAs (one per SM), tile 128 x BN x 256:
//   warp 0      TMA producer: the A and W tiles (codes via 2-D tensor maps
//               with the 128-byte swizzle) and their block scales (1-D bulk
//               copies).
//   warp 1      allocates 512 TMEM columns; one lane issues 4 MMAs of K = 64
//               per stage; its commit releases the stage.
//   warp 2      one lane copies each stage's block scales smem -> TMEM
//               (tcgen05.cp) as soon as the stage lands, so the copies run
//               ahead of, and in a different issue stream from, the MMAs.
//   warps 3..   epilogue: drain 128 accumulator columns into registers, hand
//               the accumulator back, scale by g_a g_w, round to bf16, stage in
//               swizzled shared memory and write with TMA stores.
// Every wait is bounded (NVFP4_ERR_TIMEOUT on expiry); the CTA then drains
// its copies and MMAs and frees TMEM before returning.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cfloat>
#include <map>
#include <mutex>

#include "common.cuh"
#include "nvfp4_quant.cuh"

namespace nvfp4 {
namespace {

#ifndef NVFP4_GEMM_COPY_WARPS
#define NVFP4_GEMM_COPY_WARPS 2
#endif
#ifndef NVFP4_GEMM_PAIR_STAGES
#define NVFP4_GEMM_PAIR_STAGES 5
#endif

constexpr int BM = 128;
constexpr int BK = 256;  // elements per k-block = 128 bytes per row
constexpr uint32_t kTmemCols = 512;
constexpr int kEpiRows = 32, kEpiCols = 64;                 // one TMA store box (bf16)
constexpr uint32_t kEpiBufBytes = kEpiRows * kEpiCols * 2;  // 4 KiB per epilogue warp

// BN = 128: double-buffered TMEM accumulator, 4 epilogue warps.  BN = 256:
// one accumulator (TMEM also holds the scale slots) and 8 epilogue warps that
// drain it into registers and release it before storing.
template <int BN_, int STAGES_>
struct Cfg {
  static constexpr int BN = BN_;
  static constexpr int kStages = STAGES_;
  static constexpr int kAccBufs = BN == 128 ? 2 : 1;
  static constexpr int kEpiWarps = BN / 32;  // 128 accumulator columns each
  static constexpr int kThreads = 96 + 32 * kEpiWarps;  // producer, MMA, scale copier, epilogue
  static constexpr uint32_t kTileBytesA = BM * BK / 2;  // 16 KiB
  static constexpr uint32_t kTileBytesB = BN * BK / 2;
  static constexpr uint32_t kSfaBytes = 128 * (BK / 16);  // four 512-byte scale atoms
  static constexpr uint32_t kSfbBytes = kSfaBytes * (BN / 128);
  static constexpr uint32_t kStageBytes = kTileBytesA + kTileBytesB + kSfaBytes + kSfbBytes;
  static constexpr uint32_t kSfbColsPerMma = 4 * (BN / 128);
  static constexpr uint32_t kSfCols = 16 + 4 * kSfbColsPerMma;  // TMEM columns of one stage's scales
  static constexpr uint32_t kSfTmemCol = kAccBufs * BN;
  static constexpr size_t kSmemBytes =
      1024 /*align slack*/ + kStages * kStageBytes + kEpiWarps * kEpiBufBytes + 512 /*barriers*/;
  // Instruction descriptor, kind::mxf4nvf4: A and B packed E2M1 (format 1),
  // both K-major, UE4M3 scales (bit 23 = 0), N >> 3 at bit 17, M >> 4 at bit 24.
  static constexpr uint32_t kIdesc = (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
                                     (static_cast<uint32_t>(BM >> 4) << 24);
  static_assert(kSfTmemCol + kStages * kSfCols <= kTmemCols, "TMEM budget");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

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

__device__ __forceinline__ void mma_fp4(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t sfa,
                                        uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::mxf4nvf4.block_scale.scale_vec::4X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate), "r"(sfa), "r"(sfb)
      : "memory");
}

__device__ __forceinline__ void copy_sf_to_tmem(uint32_t taddr, uint64_t desc) {
  asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(desc) : "memory");
}

// 32 lanes x 32 consecutive fp32 columns; completion via tmem_ld_wait().
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
      "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr)
               : "memory");
  return v;
}

// The CTA-pair epilogue writes its staged boxes with coalesced st.global
// rather than TMA stores, leaving the TMA unit to the operand loads that bound
// the kernel: 32B prefill gate_up 731 -> 721 us, qkv 147.5 -> 145.4 us, the
// other shapes unchanged (bit-identical outputs).  0: TMA stores.
#ifndef NVFP4_GEMM_LSU_STORE
#define NVFP4_GEMM_LSU_STORE 1
#endif

// Write one staged 32 x 64 bf16 box (rows of 128 B whose 16-byte chunks sit at
// chunk ^ (row % 8)) to out[y.., x..] with coalesced 16-byte stores: per
// instruction the warp writes 4 rows x 128 B; rows at or past M are skipped.
// (In the bounds-checked build each store is also checked against [M, N].)
__device__ __forceinline__ void store_box_lsu(uint32_t buf, uint16_t* out, int64_t ldo, int x, int y, int M, int N,
                                              int lane, int* status) {
  const int cc = lane & 7;
#pragma unroll
  for (int it = 0; it < 8; ++it) {
    const int rr = 4 * it + (lane >> 3);
    const uint4 v = ld_shared_v4(buf + rr * 128 + ((cc ^ (rr & 7)) << 4));
    if (y + rr < M && in_bounds(status, x + cc * 8 + 8 <= N))
      *reinterpret_cast<uint4*>(out + static_cast<int64_t>(y + rr) * ldo + x + cc * 8) = v;
  }
}

// Work-unit order: units walk the N tiles within groups of `group_m` row
// super-tiles, so the CTAs running at the same time share a few A and W
// tiles that stay in L2 instead of streaming all of A for every column.
__device__ __forceinline__ void unit_coords(int u, int msup, int tiles_n, int group_m, int* ms, int* nb) {
  const int per_group = group_m * tiles_n;
  const int group = u / per_group, r = u - group * per_group;
  const int rows = min(group_m, msup - group * group_m);
  *ms = group * group_m + r % rows;
  *nb = r / rows;
}

// Timeline build (-DNVFP4_TIMELINE): the 1-CTA kernel records, per CTA, the
// globaltimer at kernel entry (0), after its set-up (barriers, TMEM, the
// previous kernel's completion) (1), when the producer issued the first stage
// (2), when the first stage's data had landed for the MMA issuer (3), when the
// last MMA was issued (4), when the first epilogue warp saw the last tile's
// accumulator (5), when its stores had completed (6) and at exit (7).  The
// split-K kernel uses the same slots: 3 and 4 in the pair's leader only, 5
// when the first epilogue warp has drained the partial into shared memory,
// 6 when it has reduced and stored its box (CTAs that store one).
#ifdef NVFP4_TIMELINE
constexpr int kGemmTimelineCtas = 1024;
__device__ unsigned long long g_gemm_timeline[kGemmTimelineCtas][8];
__device__ __forceinline__ void gemm_stamp(int event) {
  if (blockIdx.x < kGemmTimelineCtas) g_gemm_timeline[blockIdx.x][event] = globaltimer_ns();
}
#else
__device__ __forceinline__ void gemm_stamp(int) {}
#endif

// Scale-format bit of the block-scaled MMA instruction descriptor (bit 23: UE8M0).
constexpr uint32_t kScaleE8M0 = 1u << 23;

struct GemmArgs {
  const uint8_t* sfa;
  const uint8_t* sfb;
  const float* ga;
  const float* gb;
  int M, N, K;
  int tiles_m, tiles_n;
  int* status;
  // OR-ed into the MMA instruction descriptor: 0 for UE4M3 block scales
  // (NVFP4), kScaleE8M0 for UE8M0 (MXFP4).  With ga == nullptr the epilogue
  // applies no global scale (MXFP4 has none).
  uint32_t idesc_fmt;
  // Fused SwiGLU + quantization epilogue (pair kernel, kSwiGLU): outputs.
  uint8_t* q_codes;   // [M, N/4] bytes: N/2 SwiGLU outputs per row
  uint8_t* q_scales;  // MMA layout for [M, N/2]
  const float* g_out;
  // Quantization of the fused output: 0 NVFP4 with the static scale g_out,
  // 1 MXFP4, 2 MXFP4 after the H_32 block rotation.
  uint32_t q_mode;
  // Test-only (nvfp4_debug_inject_fault): both CTAs of pair 0 leave their
  // first stage unissued (CTA-pair kernel).
  int fault_skip_stage;
  // Row super-tiles per raster group (unit_coords).
  int group_m;
  // Split-K kernel: CTA pairs per cluster, each taking one range of K.
  int splits;
  // bf16 output [M, N] with row pitch ldo elements (the stores that do not
  // go through the output tensor map).
  uint16_t* out;
  int64_t ldo;
};

// Raster group for a GEMM with this K: with K <= 5120 the whole of A (M x K
// FP4) stays in L2 beside the W tiles in flight, so one group covers every
// row super-tile and W streams from DRAM once; longer K keeps groups of 8
// (measured on the 32B prefill shapes: gate_up 735 -> 715 us, qkv 147.5 ->
// 145.3 us with one group; down 362.5 us with 8 against 380.9 with one).
int raster_group(int64_t K, int64_t msup) {
  return static_cast<int>(K <= 5120 ? (msup < 1 ? 1 : msup) : 8);
}

template <class C>
__global__ void __launch_bounds__(C::kThreads, 1)
    nvfp4_gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                      const __grid_constant__ CUtensorMap tmap_out, const GemmArgs args) {
  constexpr int BN = C::BN;
  constexpr int kStages = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + kStages * C::kTileBytesA;
  uint8_t* sEpi = sB + kStages * C::kTileBytesB;  // 1024-aligned: every tile above is a multiple of 1 KiB
  uint8_t* sSFA = sEpi + C::kEpiWarps * kEpiBufBytes;
  uint8_t* sSFB = sSFA + kStages * C::kSfaBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sSFB + kStages * C::kSfbBytes);
  uint64_t* empty = full + kStages;
  uint64_t* sfready = empty + kStages;
  uint64_t* tfull = sfready + kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* drain_cp = drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_cp + 1);
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kblocks = args.K / BK;
  const int kgroups = args.K / 64;
  // Work unit: one 128-row tile x one BN-column tile.
  const int msup = args.tiles_m;
  const int total_units = msup * args.tiles_n;
  const int cta_id = blockIdx.x, n_ctas = gridDim.x;
  if (threadIdx.x == 0) gemm_stamp(0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);  // the MMA commit that retires the stage
      mbar_init(&sfready[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], C::kEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(drain_cp, 1);
    abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmap_a);
    prefetch_tmap(&tmap_b);
    prefetch_tmap(&tmap_out);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait_and_release();
  if (threadIdx.x == 0) gemm_stamp(1);
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
#ifdef NVFP4_TIMELINE
    bool first_issue = true;
#endif
    for (int u = cta_id; u < total_units && !abort_flag; u += n_ctas) {
      int ms, nb;
      unit_coords(u, msup, args.tiles_n, args.group_m, &ms, &nb);
      const int mb = ms;
      const uint8_t* sfa_tile = args.sfa + (static_cast<size_t>(mb) * kgroups) * 512;
      const uint8_t* sfb_tiles = args.sfb + (static_cast<size_t>(nb) * (BN / 128) * kgroups) * 512;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, &abort_flag)) { fail(); break; }
        mbar_arrive_expect_tx(&full[stage], C::kStageBytes);
        tma_load_2d(sA + stage * C::kTileBytesA, &tmap_a, &full[stage], kb * (BK / 2), mb * BM);
        bulk_load(sSFA + stage * C::kSfaBytes, sfa_tile + static_cast<size_t>(kb) * C::kSfaBytes, C::kSfaBytes,
                  &full[stage]);
        // The stage's W scales: BN/128 row tiles of 2 KiB each.
#pragma unroll
        for (int j = 0; j < BN / 128; ++j)
          bulk_load(sSFB + stage * C::kSfbBytes + j * C::kSfaBytes,
                    sfb_tiles + (static_cast<size_t>(j) * kgroups) * 512 + static_cast<size_t>(kb) * C::kSfaBytes,
                    C::kSfaBytes, &full[stage]);
        tma_load_2d(sB + stage * C::kTileBytesB, &tmap_b, &full[stage], kb * (BK / 2), nb * BN);
#ifdef NVFP4_TIMELINE
        if (first_issue) gemm_stamp(2);
        first_issue = false;
#endif
        issued[stage] = true;
        issued_parity[stage] = phase;
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
    }
    if (abort_flag) {
      // Let every copy destined for this CTA land before it exits.
      for (int s = 0; s < kStages; ++s)
        if (issued[s]) mbar_wait_bounded(&full[s], issued_parity[s], nullptr);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------- MMA issuer ---
    int stage = 0;
    uint32_t phase = 0;
    int local = 0;
    const uint32_t sA0 = smem_u32(sA), sB0 = smem_u32(sB), sSFA0 = smem_u32(sSFA), sSFB0 = smem_u32(sSFB);
    for (int u = cta_id; u < total_units && !abort_flag; u += n_ctas, ++local) {
      const int acc = local % C::kAccBufs;
      const uint32_t acc_phase = (local / C::kAccBufs) & 1;
      if (!mbar_wait_bounded(&tempty[acc], acc_phase ^ 1u, &abort_flag)) { fail(); break; }
      tc_fence_after();
      const uint32_t d_tmem = tmem + acc * BN;
      bool ok = true;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&sfready[stage], phase, &abort_flag)) { fail(); ok = false; break; }
        if (local == 0 && kb == 0) gemm_stamp(3);
        tc_fence_after();
        const uint32_t sfa_col = tmem + C::kSfTmemCol + stage * C::kSfCols;
        const uint32_t sfb_col = sfa_col + 16;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          mma_fp4(d_tmem, desc_sw128(sA0 + stage * C::kTileBytesA + kk * 32),
                  desc_sw128(sB0 + stage * C::kTileBytesB + kk * 32), C::kIdesc | args.idesc_fmt, sfa_col + kk * 4,
                  sfb_col + kk * C::kSfbColsPerMma, (kb | kk) != 0);
        }
        tc_commit(&empty[stage]);
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      tc_commit(&tfull[acc]);
      gemm_stamp(4);
    }
    // Wait until every MMA issued above has retired before TMEM is freed.
    tc_commit(drain);
    mbar_wait_bounded(drain, 0, nullptr);
  } else if (warp == 2 && lane == 0) {
    // ---------------------------------------------- block scales -> TMEM ---
    // Slot `stage` is rewritten only after the stage's next `full` phase, which
    // the producer starts only after the MMAs that read the slot have retired.
    int stage = 0;
    uint32_t phase = 0;
    const uint32_t sSFA0 = smem_u32(sSFA), sSFB0 = smem_u32(sSFB);
    for (int u = cta_id; u < total_units && !abort_flag; u += n_ctas) {
      bool ok = true;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&full[stage], phase, &abort_flag)) { fail(); ok = false; break; }
        tc_fence_after();
        const uint32_t sfa_col = tmem + C::kSfTmemCol + stage * C::kSfCols;
        const uint32_t sfb_col = sfa_col + 16;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          copy_sf_to_tmem(sfa_col + kk * 4, desc_sf(sSFA0 + stage * C::kSfaBytes + kk * 512));
#pragma unroll
          for (int j = 0; j < BN / 128; ++j)
            copy_sf_to_tmem(sfb_col + kk * C::kSfbColsPerMma + j * 4,
                            desc_sf(sSFB0 + stage * C::kSfbBytes + j * C::kSfaBytes + kk * 512));
        }
        tc_commit(&sfready[stage]);
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
    }
    tc_commit(drain_cp);
    mbar_wait_bounded(drain_cp, 0, nullptr);
  } else if (warp >= 3) {
    // --------------------------------------------------------- epilogue ---
    const int quarter = warp & 3;                 // TMEM lanes this warp may access
    const int colbase = ((warp - 3) >> 2) * 128;  // accumulator columns this warp drains
    uint8_t* buf_ptr = sEpi + (warp - 3) * kEpiBufBytes;
    const uint32_t buf = smem_u32(buf_ptr);
    const float scale = args.ga ? __fmul_rn(__ldg(args.ga), __ldg(args.gb)) : 1.0f;
    int local = 0;
    for (int u = cta_id; u < total_units; u += n_ctas, ++local) {
      int ms, nb;
      unit_coords(u, msup, args.tiles_n, args.group_m, &ms, &nb);
      const int mb = ms;
      const int acc = local % C::kAccBufs;
      const uint32_t acc_phase = (local / C::kAccBufs) & 1;
      // Lane 0 waits and broadcasts, so the warp stays converged for the
      // .sync.aligned TMEM loads below even on the timeout path.
      int ok = 1;
      if (lane == 0) {
        ok = !abort_flag && mbar_wait_bounded(&tfull[acc], acc_phase, &abort_flag);
        if (!ok && !abort_flag) fail();
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
      if (warp == 3 && lane == 0) gemm_stamp(5);
      tc_fence_after();
      // Drain 128 columns into registers, then hand the accumulator back.
      uint32_t r[128];
      const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN + colbase;
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(taddr + c * 32, r + 32 * c);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);

      // Two 32 x 64 bf16 boxes; row `lane` of a box is 8 chunks of 16 B stored
      // at chunk position (c ^ lane%8): the 128-byte swizzle the store expects.
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (lane == 0) bulk_wait_read_all();  // the previous box has left the buffer
        __syncwarp();
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint32_t* v = r + 64 * h + 8 * c;
          st_shared_v4(buf + lane * 128 + ((c ^ (lane & 7)) << 4),
                       pack_bf16x2(__uint_as_float(v[0]) * scale, __uint_as_float(v[1]) * scale),
                       pack_bf16x2(__uint_as_float(v[2]) * scale, __uint_as_float(v[3]) * scale),
                       pack_bf16x2(__uint_as_float(v[4]) * scale, __uint_as_float(v[5]) * scale),
                       pack_bf16x2(__uint_as_float(v[6]) * scale, __uint_as_float(v[7]) * scale));
        }
        fence_proxy_async_smem();
        __syncwarp();
        const int x = nb * BN + colbase + h * kEpiCols, y = mb * BM + quarter * 32;
        if (lane == 0 && x < args.N && y < args.M) {  // boxes reaching past M or N are clipped by the TMA unit
          tma_store_2d(&tmap_out, buf_ptr, x, y);
          bulk_commit_group();
        }
      }
    }
    if (lane == 0) bulk_wait_all();
    if (warp == 3 && lane == 0) gemm_stamp(6);
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x == 0) gemm_stamp(7);
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ------------------------------------------------------ CTA-pair kernel ---
// A pair of CTAs (a cluster of 2 on neighbouring SMs) computes a 256 x 256
// tile with tcgen05.mma.cta_group::2: each CTA holds its own 128 rows of A and
// its own 128-row half of the W tile in shared memory, and its 128 x 256 slice
// of the accumulator in its own TMEM.  Per SM this halves the W bytes loaded
// and the scale copies issued for the same FLOPs.  W scales (all 256 rows) are
// loaded by both CTAs so that each TMEM receives the full set.  The leader
// (rank 0) issues the copies and the MMAs; the peer issues its own loads with
// the pair form of TMA, whose completion is counted on the leader's barrier.

__device__ __forceinline__ void mma_fp4_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                             uint32_t sfa, uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::mxf4nvf4.block_scale.scale_vec::4X [%0], %1, %2, %3, [%5], [%6], p;\n}" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate), "r"(sfa), "r"(sfb)
      : "memory");
}
__device__ __forceinline__ void copy_sf_to_tmem_pair(uint32_t taddr, uint64_t desc) {
  asm volatile("tcgen05.cp.cta_group::2.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(desc) : "memory");
}
// Arrive on the barrier at this offset in every CTA of `mask` once all
// tcgen05 operations this thread issued for the pair have completed.
__device__ __forceinline__ void tc_commit_pair(uint64_t* bar, uint16_t mask) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
                   smem_u32(bar)),
               "h"(mask)
               : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* smem_slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(smem_slot)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// 2-D TMA load into this CTA's shared memory whose completion is counted on
// the barrier at offset `bar` in the leader CTA of the pair.
__device__ __forceinline__ void tma_load_2d_to_leader(void* smem_dst, const void* tmap, uint64_t* bar, int x, int y) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(bar)), "r"(0));
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(remote), "r"(x), "r"(y)
      : "memory");
}
// Arrive on the barrier at this shared-memory offset in CTA `rank` of the
// cluster, without release semantics.  Used only to hand the accumulator back:
// the arriving warp's TMEM loads have completed (tcgen05.wait::ld) and are
// ordered before the arrive by tcgen05.fence::before_thread_sync; no memory
// written by this thread is read by the waiter.  (A release.cluster arrive
// costs about a microsecond here, which stalled the MMAs at every tile.)
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint64_t* bar, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote) : "memory");
}

// RES_: the W-resident form for 1024 <= K <= 1536.  A pair walks a run of
// consecutive units that share one W tile.  The run's first unit loads the W
// tile's codes for the whole K into shared memory and copies its block scales
// for the whole K into TMEM (8 columns per 64-deep k group); the run's later
// units stream only A and its scales (18 KB per k-block and CTA instead of
// 38 KB).  The A ring keeps 4 stages.
template <int STAGES_, bool RES_ = false>
struct PairCfg {
  static constexpr int BN = 256;                 // MMA N (both halves of the pair)
  static constexpr int kStages = STAGES_;
  static constexpr bool kRes = RES_;
  static constexpr int kResKblocks = 6;                          // K <= 1536 in the resident form
  static constexpr int kBTiles = kRes ? kResKblocks : kStages;   // W tiles held in shared memory
  static constexpr uint32_t kSfbResCol = BN;                     // resident W scales
  static constexpr uint32_t kSfaResCol = BN + 32 * kResKblocks;  // per-stage A scales, 16 columns each
  static constexpr int kEpiWarps = 8;            // 128 rows x 256 accumulator columns per CTA
  static constexpr int kCopyWarps = NVFP4_GEMM_COPY_WARPS;  // warps issuing the scale copies (1, 2 or 4)
  static constexpr int kThreads = 64 + 32 * kCopyWarps + 32 * kEpiWarps;
  static constexpr uint32_t kTileBytesA = BM * BK / 2;   // own 128 rows
  static constexpr uint32_t kTileBytesB = 128 * BK / 2;  // own half of the 256-row W tile
  static constexpr uint32_t kSfaBytes = 128 * (BK / 16);
  static constexpr uint32_t kSfbBytes = 2 * kSfaBytes;   // all 256 W rows
  static constexpr uint32_t kStageBytes = kTileBytesA + kTileBytesB + kSfaBytes + kSfbBytes;
  static constexpr uint32_t kSfCols = 16 + 32;
  static constexpr uint32_t kSfTmemCol = BN;
  static constexpr size_t kSmemBytes = 1024 + kStages * (kStageBytes - kTileBytesB) + kBTiles * kTileBytesB +
                                       kEpiWarps * kEpiBufBytes + 512 /*barriers*/;
  static constexpr uint32_t kIdesc = (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
                                     (static_cast<uint32_t>(256 >> 4) << 24);
  static_assert(kRes ? kSfaResCol + kStages * 16 <= kTmemCols : kSfTmemCol + kStages * kSfCols <= kTmemCols,
                "TMEM budget");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

template <class C, bool kSwiGLU>
__global__ void __launch_bounds__(C::kThreads, 1)
    nvfp4_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                           const __grid_constant__ CUtensorMap tmap_sfa, const __grid_constant__ CUtensorMap tmap_sfb,
                           const __grid_constant__ CUtensorMap tmap_out, const GemmArgs args) {
  constexpr int BN = C::BN;
  constexpr int kStages = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + kStages * C::kTileBytesA;
  uint8_t* sEpi = sB + C::kBTiles * C::kTileBytesB;
  uint8_t* sSFA = sEpi + C::kEpiWarps * kEpiBufBytes;
  uint8_t* sSFB = sSFA + kStages * C::kSfaBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sSFB + kStages * C::kSfbBytes);  // codes landed
  uint64_t* empty = full + kStages;
  uint64_t* sfready = empty + kStages;
  uint64_t* sffull = sfready + kStages;  // block scales landed (loaded first, so copies overlap the codes)
  uint64_t* tfull = sffull + kStages;
  uint64_t* tempty = tfull + 1;
  uint64_t* drain = tempty + 1;
  uint64_t* drain_cp = drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_cp + 1);
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kblocks = args.K / BK;
  const int kgroups = args.K / 64;
  if (C::kRes && (kblocks < kStages || kblocks > C::kResKblocks)) {
    // Outside the resident form's K range (the host never launches it so):
    // the whole grid returns before touching any barrier or TMEM.
    if (blockIdx.x == 0 && threadIdx.x == 0) set_status(args.status, NVFP4_ERR_SHAPE);
    return;
  }
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int msup = (args.tiles_m + 1) / 2;
  const int total_units = msup * args.tiles_n;
  const int pair_id = blockIdx.x / 2, n_pairs = gridDim.x / 2;
  // Units of this pair: every n_pairs-th one, or (resident form) a
  // contiguous run in W-tile-major order, so that consecutive units share nb.
  const int run = C::kRes ? (total_units + n_pairs - 1) / n_pairs : 0;
  const int u_first = C::kRes ? pair_id * run : pair_id;
  const int u_end = C::kRes ? min(total_units, u_first + run) : total_units;
  const int u_step = C::kRes ? 1 : n_pairs;
  auto coords = [&](int u, int* ms, int* nb) {
    if (C::kRes) {
      // Within a W tile the row super-tiles start at a rotation of nb, so
      // that the pairs running at the same time read different A tiles.
      *nb = u / msup;
      *ms = (u - *nb * msup + *nb) % msup;
    } else {
      unit_coords(u, msup, args.tiles_n, args.group_m, ms, nb);
    }
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);  // leader: its expect_tx covers both CTAs' bytes; unused in the peer
      mbar_init(&empty[s], 1);
      mbar_init(&sfready[s], C::kCopyWarps);  // one commit per copy warp
      mbar_init(&sffull[s], 1);
    }
    mbar_init(tfull, 1);
    mbar_init(tempty, 2 * C::kEpiWarps);
    mbar_init(drain, 1);
    mbar_init(drain_cp, C::kCopyWarps);
    abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmap_a);
    prefetch_tmap(&tmap_b);
    prefetch_tmap(&tmap_sfa);
    prefetch_tmap(&tmap_sfb);
    prefetch_tmap(&tmap_out);
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  griddep_wait_and_release();
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
    int prev_nb = -1;
    int g = 0;  // k-blocks this pair has passed so far
    for (int u = u_first; u < u_end && !abort_flag; u += u_step) {
      int ms, nb;
      coords(u, &ms, &nb);
      // W codes and scales: every unit, or (resident form) a run's first.
      // Resident W tile kb is rewritten only after the MMAs of k-block kb of
      // the previous unit completed: this stage's empty barrier covers the
      // MMAs up to kStages k-blocks back, and kblocks >= kStages.
      const bool load_w = !C::kRes || nb != prev_nb;
      prev_nb = nb;
      const int mb = min(ms * 2 + static_cast<int>(rank), args.tiles_m - 1);  // a spare CTA redoes the last tile
      // Scale atoms through a [bytes / 256, 256] view: one (128-row tile,
      // k-block) group of four 512-byte atoms is 8 rows of that view.
      const int sfa_row = mb * kgroups * 2;
      const int sfb_row = nb * 2 * kgroups * 2;
      for (int kb = 0; kb < kblocks; ++kb, ++g) {
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, &abort_flag)) { fail(); break; }
        if (args.fault_skip_stage && pair_id == 0 && g == 0) {
          // Test-only injected fault: both CTAs of pair 0 leave their first
          // stage neither armed nor loaded, so no copy is ever in flight for
          // it and the consumers' bounded waits on it run out.
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
          continue;
        }
        uint8_t* a_dst = sA + stage * C::kTileBytesA;
        uint8_t* b_dst = sB + (C::kRes ? kb : stage) * C::kTileBytesB;
        uint8_t* sfa_dst = sSFA + stage * C::kSfaBytes;
        uint8_t* sfb_dst = sSFB + stage * C::kSfbBytes;
        const int kx = kb * (BK / 2), b_row = nb * BN + static_cast<int>(rank) * 128;
        constexpr uint32_t kSfStage = C::kSfaBytes + C::kSfbBytes;
        if (leader) {
          // Both CTAs' loads land on the leader's barriers.
          mbar_arrive_expect_tx(&sffull[stage], 2 * (load_w ? kSfStage : C::kSfaBytes));
          mbar_arrive_expect_tx(&full[stage], 2 * (C::kTileBytesA + (load_w ? C::kTileBytesB : 0u)));
          tma_load_2d(sfa_dst, &tmap_sfa, &sffull[stage], 0, sfa_row + kb * 8);
          if (load_w) {
            tma_load_2d(sfb_dst, &tmap_sfb, &sffull[stage], 0, sfb_row + kb * 8);
            tma_load_2d(sfb_dst + C::kSfaBytes, &tmap_sfb, &sffull[stage], 0, sfb_row + kgroups * 2 + kb * 8);
          }
          tma_load_2d(a_dst, &tmap_a, &full[stage], kx, mb * BM);
          if (load_w) tma_load_2d(b_dst, &tmap_b, &full[stage], kx, b_row);
        } else {
          tma_load_2d_to_leader(sfa_dst, &tmap_sfa, &sffull[stage], 0, sfa_row + kb * 8);
          if (load_w) {
            tma_load_2d_to_leader(sfb_dst, &tmap_sfb, &sffull[stage], 0, sfb_row + kb * 8);
            tma_load_2d_to_leader(sfb_dst + C::kSfaBytes, &tmap_sfb, &sffull[stage], 0,
                                  sfb_row + kgroups * 2 + kb * 8);
          }
          tma_load_2d_to_leader(a_dst, &tmap_a, &full[stage], kx, mb * BM);
          if (load_w) tma_load_2d_to_leader(b_dst, &tmap_b, &full[stage], kx, b_row);
        }
        issued[stage] = true;
        issued_parity[stage] = phase;
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
    }
    if (abort_flag && leader) {
      // Both CTAs' copies complete on the leader's barriers: wait for them here.
      for (int s = 0; s < kStages; ++s)
        if (issued[s]) {
          mbar_wait_bounded(&sffull[s], issued_parity[s], nullptr);
          mbar_wait_bounded(&full[s], issued_parity[s], nullptr);
        }
    }
  } else if (warp == 1 && lane == 0 && leader) {
    // ------------------------------------------------ MMA issuer (leader) ---
    int stage = 0;
    uint32_t phase = 0;
    int local = 0;
    const uint32_t sA0 = smem_u32(sA), sB0 = smem_u32(sB);
    for (int u = u_first; u < u_end && !abort_flag; u += u_step, ++local) {
      if (!mbar_wait_bounded(tempty, (local & 1) ^ 1u, &abort_flag)) { fail(); break; }
      tc_fence_after();
      bool ok = true;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&full[stage], phase, &abort_flag) ||
            !mbar_wait_bounded(&sfready[stage], phase, &abort_flag)) { fail(); ok = false; break; }
        tc_fence_after();
        const uint32_t sfa_col = tmem + (C::kRes ? C::kSfaResCol + stage * 16 : C::kSfTmemCol + stage * C::kSfCols);
        const uint32_t sfb_col = C::kRes ? tmem + C::kSfbResCol + kb * 32 : sfa_col + 16;
        const uint32_t b_tile = sB0 + (C::kRes ? kb : stage) * C::kTileBytesB;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_fp4_pair(tmem, desc_sw128(sA0 + stage * C::kTileBytesA + kk * 32), desc_sw128(b_tile + kk * 32),
                       C::kIdesc | args.idesc_fmt, sfa_col + kk * 4, sfb_col + kk * 8, (kb | kk) != 0);
        tc_commit_pair(&empty[stage], 0x3);
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      tc_commit_pair(tfull, 0x3);
    }
    tc_commit_pair(drain, 0x1);
    mbar_wait_bounded(drain, 0, nullptr);
  } else if (warp >= 2 && warp < 2 + C::kCopyWarps && lane == 0 && leader) {
    // ------------------------------------- leader: block scales -> TMEM ---
    // The K=64 steps of a stage are spread over the copy warps: copies issued
    // from different warps proceed concurrently, copies from one thread do not.
    constexpr int kPerWarp = 4 / C::kCopyWarps;
    const int kk0 = (warp - 2) * kPerWarp;
    int stage = 0;
    uint32_t phase = 0;
    const uint32_t sSFA0 = smem_u32(sSFA), sSFB0 = smem_u32(sSFB);
    int prev_nb = -1;
    for (int u = u_first; u < u_end && !abort_flag; u += u_step) {
      bool ok = true;
      int ms, nb;
      coords(u, &ms, &nb);
      // Resident form: a run's first unit copies the W scales for the whole
      // K.  The copy of k-block kb's columns waited (through the producer's
      // empty barrier) for the MMAs of the previous unit's k-block kb.
      const bool copy_w = !C::kRes || nb != prev_nb;
      prev_nb = nb;
      for (int kb = 0; kb < kblocks; ++kb) {
        if (!mbar_wait_bounded(&sffull[stage], phase, &abort_flag)) { fail(); ok = false; break; }
        {
          tc_fence_after();
          const uint32_t sfa_col =
              tmem + (C::kRes ? C::kSfaResCol + stage * 16 : C::kSfTmemCol + stage * C::kSfCols);
          const uint32_t sfb_col = C::kRes ? tmem + C::kSfbResCol + kb * 32 : sfa_col + 16;
#pragma unroll
          for (int kk = kk0; kk < kk0 + kPerWarp; ++kk) {
            copy_sf_to_tmem_pair(sfa_col + kk * 4, desc_sf(sSFA0 + stage * C::kSfaBytes + kk * 512));
            if (copy_w) {
#pragma unroll
              for (int j = 0; j < 2; ++j)
                copy_sf_to_tmem_pair(sfb_col + kk * 8 + j * 4,
                                     desc_sf(sSFB0 + stage * C::kSfbBytes + j * C::kSfaBytes + kk * 512));
            }
          }
          tc_commit_pair(&sfready[stage], 0x1);
        }
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
    }
    tc_commit_pair(drain_cp, 0x1);
    mbar_wait_bounded(drain_cp, 0, nullptr);
  } else if (kSwiGLU && warp >= 2 + C::kCopyWarps) {
    // ------------------------------------- epilogue: SwiGLU + NVFP4 output ---
    // W rows are interleaved in blocks of 16 (gate, then the matching up), so
    // each 32-column TMEM load gives a thread 16 gate and 16 up values of its
    // row: one 16-element block of h = SiLU(gate) * up, quantized here with
    // the static scale g_out by the library's recipe.  A warp's 128 columns
    // are 64 outputs = 4 blocks = 32 code bytes and one 32-bit scale word.
    constexpr int kEpi0 = 2 + C::kCopyWarps;
    const int quarter = warp & 3;
    const int colbase = ((warp - kEpi0) >> 2) * 128;
    const float scale = args.ga ? __fmul_rn(__ldg(args.ga), __ldg(args.gb)) : 1.0f;
    const float g_in = args.q_mode == 0 ? __ldg(args.g_out) : 1.0f;
    const bool g_ok = g_in > 0.0f && g_in <= FLT_MAX;
    if (!g_ok && blockIdx.x == 0 && threadIdx.x == 32 * kEpi0) set_status(args.status, NVFP4_ERR_INVALID_ARG);
    const float g = g_ok ? g_in : 1.0f, six_g = __fmul_rn(6.0f, g);
    const uint32_t q_cols = static_cast<uint32_t>(args.N) >> 1;  // SwiGLU outputs per row
    const uint32_t q_kgroups = q_cols >> 6;
    int local = 0;
    for (int u = u_first; u < u_end; u += u_step, ++local) {
      int ms, nb;
      coords(u, &ms, &nb);
      const int mb = ms * 2 + static_cast<int>(rank);  // mb >= tiles_m: nothing is stored
      int ok = 1;
      if (lane == 0) {
        ok = !abort_flag && mbar_wait_bounded(tfull, local & 1, &abort_flag);
        if (!ok && !abort_flag) fail();
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
      tc_fence_after();
      uint32_t r[128];
      const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + colbase;
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(taddr + c * 32, r + 32 * c);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster_relaxed(tempty, 0);
      // The MMAs of the next tile run while this warp computes and stores.
      const uint32_t row = static_cast<uint32_t>(mb * BM + quarter * 32 + lane);
      const uint32_t oc0 = static_cast<uint32_t>(nb) * (BN / 2) + static_cast<uint32_t>(colbase / 2);
      uint32_t codes[8], sc = 0;
      if (args.q_mode == 0) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float h[16];
          float amax = 0.0f;
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            // SiLU(x) = x sigmoid(x) = x/2 (1 + tanh(x/2)): one MUFU operation.
            const float half_g = __uint_as_float(r[32 * c + i]) * (0.5f * scale);
            const float up = __uint_as_float(r[32 * c + 16 + i]) * scale;
            h[i] = fmaf(half_g, tanh_approx(half_g), half_g) * up;
            amax = fmaxf(amax, fabsf(h[i]));
          }
          const BlockScale bs = block_scale(amax, g, six_g);
#pragma unroll
          for (int i = 0; i < 16; ++i) h[i] = __fmul_rn(h[i], bs.mult);
          codes[2 * c] = g_ok ? e2m1x8(h) : 0u;
          codes[2 * c + 1] = g_ok ? e2m1x8(h + 8) : 0u;
          sc |= (g_ok ? bs.code : 0u) << (8 * c);
        }
      } else {
        // MXFP4: two TMEM loads give 32 consecutive outputs, one 32-element
        // block (optionally rotated by H_32 / sqrt(32)) with one E8M0 scale,
        // stored for both 16-element halves in the MMA scale word.
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          float h[32];
#pragma unroll
          for (int cc = 0; cc < 2; ++cc) {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float half_g = __uint_as_float(r[32 * (2 * j + cc) + i]) * (0.5f * scale);
              const float up = __uint_as_float(r[32 * (2 * j + cc) + 16 + i]) * scale;
              h[16 * cc + i] = fmaf(half_g, tanh_approx(half_g), half_g) * up;
            }
          }
          if (args.q_mode == 2) hadamard32(h);
          float amax = 0.0f;
#pragma unroll
          for (int i = 0; i < 32; ++i) amax = fmaxf(amax, fabsf(h[i]));
          const uint32_t code = mx_scale_code(amax);
          const float inv = mx_inv_scale(code);
#pragma unroll
          for (int i = 0; i < 32; ++i) h[i] = __fmul_rn(h[i], inv);
          codes[4 * j] = e2m1x8(h);
          codes[4 * j + 1] = e2m1x8(h + 8);
          codes[4 * j + 2] = e2m1x8(h + 16);
          codes[4 * j + 3] = e2m1x8(h + 24);
          sc |= (code | (code << 8)) << (16 * j);
        }
      }
      if (mb < args.tiles_m) {
        // Scales for every row of the 128-row tile (rows past M hold zeros: A's
        // missing rows load as zeros), codes for rows < M.
        const uint64_t sc_off = mma_scale_offset(row, oc0 / 16, q_kgroups);
        const uint64_t sc_bytes = static_cast<uint64_t>((args.M + 127) & ~127) * (q_cols / 16);
        if (in_bounds(args.status, sc_off % 4 == 0 && sc_off + 4 <= sc_bytes))
          *reinterpret_cast<uint32_t*>(args.q_scales + sc_off) = sc;
        const uint64_t code_off = static_cast<uint64_t>(row) * (q_cols / 2) + oc0 / 2;
        if (row < static_cast<uint32_t>(args.M) &&
            in_bounds(args.status, code_off + 32 <= static_cast<uint64_t>(args.M) * (q_cols / 2))) {
          uint4* dst = reinterpret_cast<uint4*>(args.q_codes + code_off);
          dst[0] = make_uint4(codes[0], codes[1], codes[2], codes[3]);
          dst[1] = make_uint4(codes[4], codes[5], codes[6], codes[7]);
        }
      }
    }
  } else if (warp >= 2 + C::kCopyWarps) {
    // --------------------------------------------------------- epilogue ---
    constexpr int kEpi0 = 2 + C::kCopyWarps;
    const int quarter = warp & 3;
    const int colbase = ((warp - kEpi0) >> 2) * 128;
    uint8_t* buf_ptr = sEpi + (warp - kEpi0) * kEpiBufBytes;
    const uint32_t buf = smem_u32(buf_ptr);
    const float scale = args.ga ? __fmul_rn(__ldg(args.ga), __ldg(args.gb)) : 1.0f;
    int local = 0;
    for (int u = u_first; u < u_end; u += u_step, ++local) {
      int ms, nb;
      coords(u, &ms, &nb);
      const int mb = ms * 2 + static_cast<int>(rank);  // mb >= tiles_m: nothing is stored
      int ok = 1;
      if (lane == 0) {
        ok = !abort_flag && mbar_wait_bounded(tfull, local & 1, &abort_flag);
        if (!ok && !abort_flag) fail();
      }
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
      tc_fence_after();
      uint32_t r[128];
      const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + colbase;
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(taddr + c * 32, r + 32 * c);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster_relaxed(tempty, 0);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (lane == 0) bulk_wait_read_all();
        __syncwarp();
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint32_t* v = r + 64 * h + 8 * c;
          st_shared_v4(buf + lane * 128 + ((c ^ (lane & 7)) << 4),
                       pack_bf16x2(__uint_as_float(v[0]) * scale, __uint_as_float(v[1]) * scale),
                       pack_bf16x2(__uint_as_float(v[2]) * scale, __uint_as_float(v[3]) * scale),
                       pack_bf16x2(__uint_as_float(v[4]) * scale, __uint_as_float(v[5]) * scale),
                       pack_bf16x2(__uint_as_float(v[6]) * scale, __uint_as_float(v[7]) * scale));
        }
        const int x = nb * BN + colbase + h * kEpiCols, y = mb * BM + quarter * 32;
        if (NVFP4_GEMM_LSU_STORE) {
          __syncwarp();
          if (x < args.N && y < args.M) store_box_lsu(buf, args.out, args.ldo, x, y, args.M, args.N, lane, args.status);
          __syncwarp();  // the next box overwrites the staging buffer
        } else {
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0 && x < args.N && y < args.M) {
            tma_store_2d(&tmap_out, buf_ptr, x, y);
            bulk_commit_group();
          }
        }
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, kTmemCols);
}

// ------------------------------------------------- split-K cluster kernel ---
// For decode-sized M the 256 x 256 pair tiles are too few to occupy the GPU,
// and 128 x 128 tiles on single CTAs make every SM receive all of A and a W
// tile for the whole K (the k-loop is bound by the bytes each SM must take
// in).  Here a cluster of 2S CTAs computes one 256 x 256 tile: its S CTA
// pairs (ranks 2s and 2s + 1) each run the pair kernel's pipeline over one
// contiguous range of the k-blocks, so each W byte is still read once and
// each SM takes in 1/S of the tile's operands.  The S fp32 partial
// accumulators are then summed across the cluster in distributed shared
// memory: every CTA drains its 128 x 256 partial from TMEM into its own
// (now idle) operand ring, and after a cluster barrier the S CTAs holding the
// same 128 rows each reduce a share of the 32 x 64 output boxes, reading the
// other partials remotely and adding them in split order (so the result does
// not depend on which CTA reduces), scale by g_a g_w, round to bf16 and store
// with TMA.  One tile per cluster; no persistent loop.

// 16-byte chunk j of partial-buffer row `row` (1 KiB rows of 256 fp32): the
// chunk index is XOR-ed with row % 8 so that both the row-per-lane drain and
// the row-contiguous reduction touch every bank once per 8 lanes.
__device__ __forceinline__ uint32_t part_offset(uint32_t row, uint32_t j) {
  return row * 1024u + ((j ^ (row & 7u)) << 4);
}

// Load from a shared::cluster address (a CTA's shared memory mapped with mapa).
__device__ __forceinline__ float4 ld_cluster_f4(uint32_t cluster_addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(cluster_addr)
               : "memory");
  return v;
}
__device__ __forceinline__ void st_shared_v2(uint32_t addr, uint32_t a, uint32_t b) {
  asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}
// The pair-form TMA load of the pair kernel, completing on the barrier at
// offset `bar` in cluster CTA `lead_rank` (the pair's even rank).
__device__ __forceinline__ void tma_load_2d_to(void* smem_dst, const void* tmap, uint64_t* bar, int x, int y,
                                               uint32_t lead_rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(bar)), "r"(lead_rank));
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(remote), "r"(x), "r"(y)
      : "memory");
}

// One 32 x 64 output box of the split-K reduction: rows 32q .. 32q + 31 of
// the CTA's slice, 16-byte column chunk j (lane & 15 picks the chunk, lane >> 4
// the row of a pair).  The S partials (cluster ranks 2t + half) are read in
// batches of B row pairs with all S x B loads of a batch in flight, added in
// split order (the result does not depend on which CTA reduces), scaled,
// rounded to bf16 and written to the 128-byte-swizzled staging box.
template <int S, int B>
__device__ __forceinline__ void reduce_box(uint32_t part0, uint32_t half, int q, uint32_t j, int lane, float scale,
                                           uint32_t buf) {
  uint32_t base[S];
#pragma unroll
  for (int t = 0; t < S; ++t)
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(base[t]) : "r"(part0), "r"(2u * t + half));
  const uint32_t cchunk = static_cast<uint32_t>((lane & 15) >> 1);
#pragma unroll 1
  for (int b = 0; b < 16 / B; ++b) {
    float4 v[S][B];
#pragma unroll
    for (int t = 0; t < S; ++t)
#pragma unroll
      for (int i = 0; i < B; ++i) {
        const uint32_t rr = static_cast<uint32_t>(2 * (b * B + i) + (lane >> 4));
        v[t][i] = ld_cluster_f4(base[t] + part_offset(static_cast<uint32_t>(q * 32) + rr, j));
      }
#pragma unroll
    for (int i = 0; i < B; ++i) {
      float4 acc = v[0][i];
#pragma unroll
      for (int t = 1; t < S; ++t) {
        acc.x += v[t][i].x;
        acc.y += v[t][i].y;
        acc.z += v[t][i].z;
        acc.w += v[t][i].w;
      }
      const uint32_t rr = static_cast<uint32_t>(2 * (b * B + i) + (lane >> 4));
      st_shared_v2(buf + rr * 128 + ((cchunk ^ (rr & 7u)) << 4) + (lane & 1) * 8,
                   pack_bf16x2(acc.x * scale, acc.y * scale), pack_bf16x2(acc.z * scale, acc.w * scale));
    }
  }
}

template <class C>
__global__ void __launch_bounds__(C::kThreads, 1)
    nvfp4_gemm_splitk_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                             const __grid_constant__ CUtensorMap tmap_sfa,
                             const __grid_constant__ CUtensorMap tmap_sfb,
                             const __grid_constant__ CUtensorMap tmap_out, const GemmArgs args) {
  constexpr int BN = C::BN;
  constexpr int kStages = C::kStages;
  constexpr int kEpi0 = 2 + C::kCopyWarps;
  static_assert(!C::kRes, "streaming form only");
  static_assert(C::kEpiWarps == 8, "eight reduction warps");
  static_assert(128u * 1024u <= kStages * (C::kTileBytesA + C::kTileBytesB), "the partial fits in the ring");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + kStages * C::kTileBytesA;
  uint8_t* sEpi = sB + kStages * C::kTileBytesB;
  uint8_t* sSFA = sEpi + C::kEpiWarps * kEpiBufBytes;
  uint8_t* sSFB = sSFA + kStages * C::kSfaBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sSFB + kStages * C::kSfbBytes);
  uint64_t* empty = full + kStages;
  uint64_t* sfready = empty + kStages;
  uint64_t* sffull = sfready + kStages;
  uint64_t* tfull = sffull + kStages;
  uint64_t* drain = tfull + 1;
  uint64_t* drain_cp = drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_cp + 1);
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = args.splits;
  const int kblocks = args.K / BK;
  const int kgroups = args.K / 64;
  const uint32_t rank = cluster_ctarank();
  const uint32_t half = rank & 1u, split = rank >> 1, lead = rank & ~1u;
  const bool leader = half == 0;
  const int tile = blockIdx.x / (2 * S);
  const int msup = (args.tiles_m + 1) / 2;
  int ms, nb;
  unit_coords(tile, msup, args.tiles_n, args.group_m, &ms, &nb);
  const int k0 = static_cast<int>(split) * kblocks / S, k1 = (static_cast<int>(split) + 1) * kblocks / S;
  const int mb = ms * 2 + static_cast<int>(half);  // mb >= tiles_m: a spare CTA, nothing is stored
  if (threadIdx.x == 0) gemm_stamp(0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&sfready[s], C::kCopyWarps);
      mbar_init(&sffull[s], 1);
    }
    mbar_init(tfull, 1);
    mbar_init(drain, 1);
    mbar_init(drain_cp, C::kCopyWarps);
    abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmap_a);
    prefetch_tmap(&tmap_b);
    prefetch_tmap(&tmap_sfa);
    prefetch_tmap(&tmap_sfb);
    prefetch_tmap(&tmap_out);
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  griddep_wait_and_release();
  if (threadIdx.x == 0) gemm_stamp(1);
  const uint32_t tmem = *tmem_slot;

  auto fail = [&]() {
    set_status(args.status, NVFP4_ERR_TIMEOUT);
    abort_flag = 1;
  };

  bool have_partial = false;  // epilogue warps: this CTA's partial is in shared memory
  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------ TMA producer ---
    int stage = 0;
    uint32_t phase = 0;
    uint32_t issued_parity[kStages];
    bool issued[kStages];
    for (int s = 0; s < kStages; ++s) issued[s] = false;
    const int a_row = min(mb, args.tiles_m - 1) * BM;  // a spare CTA reloads the last tile
    const int sfa_row = min(mb, args.tiles_m - 1) * kgroups * 2;
    const int sfb_row = nb * 2 * kgroups * 2;
    const int b_row = nb * BN + static_cast<int>(half) * 128;
    for (int kb = k0; kb < k1; ++kb) {
      if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, &abort_flag)) { fail(); break; }
      if (args.fault_skip_stage && tile == 0 && split == 0 && kb == k0) {
        // Test-only injected fault, as in the pair kernel: the first stage of
        // the first pair is neither armed nor loaded.
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
        continue;
      }
      uint8_t* a_dst = sA + stage * C::kTileBytesA;
      uint8_t* b_dst = sB + stage * C::kTileBytesB;
      uint8_t* sfa_dst = sSFA + stage * C::kSfaBytes;
      uint8_t* sfb_dst = sSFB + stage * C::kSfbBytes;
      const int kx = kb * (BK / 2);
      if (leader) {
        // Both CTAs' loads land on the leader's barriers.
        mbar_arrive_expect_tx(&sffull[stage], 2 * (C::kSfaBytes + C::kSfbBytes));
        mbar_arrive_expect_tx(&full[stage], 2 * (C::kTileBytesA + C::kTileBytesB));
        tma_load_2d(sfa_dst, &tmap_sfa, &sffull[stage], 0, sfa_row + kb * 8);
        tma_load_2d(sfb_dst, &tmap_sfb, &sffull[stage], 0, sfb_row + kb * 8);
        tma_load_2d(sfb_dst + C::kSfaBytes, &tmap_sfb, &sffull[stage], 0, sfb_row + kgroups * 2 + kb * 8);
        tma_load_2d(a_dst, &tmap_a, &full[stage], kx, a_row);
        tma_load_2d(b_dst, &tmap_b, &full[stage], kx, b_row);
      } else {
        tma_load_2d_to(sfa_dst, &tmap_sfa, &sffull[stage], 0, sfa_row + kb * 8, lead);
        tma_load_2d_to(sfb_dst, &tmap_sfb, &sffull[stage], 0, sfb_row + kb * 8, lead);
        tma_load_2d_to(sfb_dst + C::kSfaBytes, &tmap_sfb, &sffull[stage], 0, sfb_row + kgroups * 2 + kb * 8,
                       lead);
        tma_load_2d_to(a_dst, &tmap_a, &full[stage], kx, a_row, lead);
        tma_load_2d_to(b_dst, &tmap_b, &full[stage], kx, b_row, lead);
      }
      if (kb == k0) gemm_stamp(2);
      issued[stage] = true;
      issued_parity[stage] = phase;
      if (++stage == kStages) { stage = 0; phase ^= 1u; }
    }
    if (abort_flag && leader) {
      for (int s = 0; s < kStages; ++s)
        if (issued[s]) {
          mbar_wait_bounded(&sffull[s], issued_parity[s], nullptr);
          mbar_wait_bounded(&full[s], issued_parity[s], nullptr);
        }
    }
  } else if (warp == 1 && lane == 0 && leader) {
    // ------------------------------------------------ MMA issuer (leader) ---
    int stage = 0;
    uint32_t phase = 0;
    const uint32_t sA0 = smem_u32(sA), sB0 = smem_u32(sB);
    bool ok = true;
    for (int kb = k0; kb < k1; ++kb) {
      if (!mbar_wait_bounded(&full[stage], phase, &abort_flag) ||
          !mbar_wait_bounded(&sfready[stage], phase, &abort_flag)) { fail(); ok = false; break; }
      if (kb == k0) gemm_stamp(3);
      tc_fence_after();
      const uint32_t sfa_col = tmem + C::kSfTmemCol + stage * C::kSfCols;
      const uint32_t sfb_col = sfa_col + 16;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        mma_fp4_pair(tmem, desc_sw128(sA0 + stage * C::kTileBytesA + kk * 32),
                     desc_sw128(sB0 + stage * C::kTileBytesB + kk * 32), C::kIdesc | args.idesc_fmt,
                     sfa_col + kk * 4, sfb_col + kk * 8, (kb != k0) | (kk != 0));
      tc_commit_pair(&empty[stage], static_cast<uint16_t>(3u << lead));
      if (++stage == kStages) { stage = 0; phase ^= 1u; }
    }
    if (ok) tc_commit_pair(tfull, static_cast<uint16_t>(3u << lead));
    gemm_stamp(4);
    tc_commit_pair(drain, static_cast<uint16_t>(1u << lead));
    mbar_wait_bounded(drain, 0, nullptr);
  } else if (warp >= 2 && warp < kEpi0 && lane == 0 && leader) {
    // ------------------------------------- leader: block scales -> TMEM ---
    constexpr int kPerWarp = 4 / C::kCopyWarps;
    const int kk0 = (warp - 2) * kPerWarp;
    int stage = 0;
    uint32_t phase = 0;
    const uint32_t sSFA0 = smem_u32(sSFA), sSFB0 = smem_u32(sSFB);
    for (int kb = k0; kb < k1; ++kb) {
      if (!mbar_wait_bounded(&sffull[stage], phase, &abort_flag)) { fail(); break; }
      tc_fence_after();
      const uint32_t sfa_col = tmem + C::kSfTmemCol + stage * C::kSfCols;
      const uint32_t sfb_col = sfa_col + 16;
#pragma unroll
      for (int kk = kk0; kk < kk0 + kPerWarp; ++kk) {
        copy_sf_to_tmem_pair(sfa_col + kk * 4, desc_sf(sSFA0 + stage * C::kSfaBytes + kk * 512));
#pragma unroll
        for (int j = 0; j < 2; ++j)
          copy_sf_to_tmem_pair(sfb_col + kk * 8 + j * 4,
                               desc_sf(sSFB0 + stage * C::kSfbBytes + j * C::kSfaBytes + kk * 512));
      }
      tc_commit_pair(&sfready[stage], static_cast<uint16_t>(1u << lead));
      if (++stage == kStages) { stage = 0; phase ^= 1u; }
    }
    tc_commit_pair(drain_cp, static_cast<uint16_t>(1u << lead));
    mbar_wait_bounded(drain_cp, 0, nullptr);
  } else if (warp >= kEpi0) {
    // ------------------------------- drain the partial into shared memory ---
    // The last MMA has completed (tfull), so every operand copy has landed
    // and been read: the ring is free for the partial.
    const int quarter = warp & 3;
    const int colbase = ((warp - kEpi0) >> 2) * 128;
    int ok = 1;
    if (lane == 0) {
      ok = !abort_flag && mbar_wait_bounded(tfull, 0, &abort_flag);
      if (!ok && !abort_flag) fail();
    }
    if (__shfl_sync(0xffffffffu, ok, 0)) {
      tc_fence_after();
      uint32_t r[128];
      const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + colbase;
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(taddr + c * 32, r + 32 * c);
      tmem_ld_wait();
      const uint32_t row = static_cast<uint32_t>(quarter * 32 + lane);
      const uint32_t part0 = smem_u32(smem);
#pragma unroll
      for (int c = 0; c < 32; ++c)
        st_shared_v4(part0 + part_offset(row, static_cast<uint32_t>(colbase / 4 + c)), r[4 * c], r[4 * c + 1],
                     r[4 * c + 2], r[4 * c + 3]);
      have_partial = true;
      if (warp == kEpi0 && lane == 0) gemm_stamp(5);
    }
  }

  // Every CTA's partial is written (or its CTA gave up) before any is read.
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();

  if (warp >= kEpi0 && !abort_flag) {
    // ------------------------------------------ reduce and store (one box) ---
    // Box p (0..15) covers rows 32 (p % 4) .. +31 and columns 64 (p / 4) .. +63
    // of this CTA's 128 x 256 slice; split s reduces boxes s, s + S, ...
    const int p = static_cast<int>(split) + (warp - kEpi0) * S;
    const bool all_ok = __all_sync(0xffffffffu, have_partial ? 1 : 0);
    if (p < 16 && mb < args.tiles_m && all_ok) {
      const int q = p & 3, pc = p >> 2;
      const float scale = args.ga ? __fmul_rn(__ldg(args.ga), __ldg(args.gb)) : 1.0f;
      uint8_t* buf_ptr = sEpi + (warp - kEpi0) * kEpiBufBytes;
      const uint32_t buf = smem_u32(buf_ptr), part0 = smem_u32(smem);
      const uint32_t j = static_cast<uint32_t>(pc * 16 + (lane & 15));
      if (S == 2) reduce_box<2, 8>(part0, half, q, j, lane, scale, buf);
      else if (S == 3) reduce_box<3, 4>(part0, half, q, j, lane, scale, buf);
      else reduce_box<4, 4>(part0, half, q, j, lane, scale, buf);
      fence_proxy_async_smem();
      __syncwarp();
      const int x = nb * BN + pc * 64, y = mb * BM + q * 32;
      if (lane == 0 && x < args.N && y < args.M) {
        tma_store_2d(&tmap_out, buf_ptr, x, y);
        bulk_commit_group();
        bulk_wait_all();
        if (warp == kEpi0) gemm_stamp(6);
      }
    }
  }

  // No CTA leaves while another may still read its partial.
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  if (threadIdx.x == 0) gemm_stamp(7);
  if (warp == 1) tmem_dealloc_pair(tmem, kTmemCols);
}

// ------------------------------------- quantize-in-prologue linear kernel ---
// a1 + a2 + a3 in one launch for an activation of at most 32 rows and K of
// at most 1536: every CTA reads the whole bf16 activation x (at most 96 KB,
// an L2 hit after the first CTA), reduces its amax, forms the tensor scale g_a
// and quantizes x into its own shared memory in the MMA layout (codes in the
// 128-byte-swizzled K-major tiles the tensor core reads, block scales in
// 512-byte atoms), exactly as nvfp4_quantize_dynamic would; no grid barrier
// is needed because each CTA does the reduction itself.  A and its scales then
// stay resident (A scales in TMEM for the whole K) while the producer streams
// only W through a 5-stage ring, from the kernel's first instruction on.
//   warp 0      TMA producer for W codes and scales (skips the prologue)
//   warps 1-11  prologue (amax, then quantization), then:
//   warp 1      TMEM allocation; one lane issues the MMAs
//   warp 2      one lane copies the A scales once, then each stage's W scales
//   warps 3-6   epilogue (double-buffered 128-column accumulator)
struct DynCfg {
  static constexpr int BN = 128;
  static constexpr int kStages = 5;
  static constexpr int kMaxKb = 6;                          // K <= 1536
  static constexpr int kMaxRows = 32;                       // M <= 32
  static constexpr int kEpiWarps = 4;
  // Warps 7-11 only help with the prologue, whose per-block arithmetic
  // (E4M3 scale, reciprocal, 16 conversions) is latency-bound with few warps.
  static constexpr int kThreads = 384;
  static constexpr int kProThreads = kThreads - 32;          // warps 1-11
  static constexpr uint32_t kTileBytesA = BM * BK / 2;       // 16 KiB per k-block
  static constexpr uint32_t kTileBytesB = BN * BK / 2;       // 16 KiB per stage
  static constexpr uint32_t kSfaBytes = 128 * (BK / 16);     // 2 KiB per k-block: four 512-byte atoms
  static constexpr uint32_t kSfbBytes = kSfaBytes;
  static constexpr uint32_t kSfaResCol = 2 * BN;             // A scales: 16 columns per k-block
  static constexpr uint32_t kSfbCol = kSfaResCol + 16 * kMaxKb;  // W scales: 16 columns per stage
  static constexpr size_t kSmemBytes = 1024 + kMaxKb * (kTileBytesA + kSfaBytes) +
                                       kStages * (kTileBytesB + kSfbBytes) + kEpiWarps * kEpiBufBytes + 512;
  static constexpr uint32_t kIdesc = (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
                                     (static_cast<uint32_t>(BM >> 4) << 24);
  static_assert(kSfbCol + kStages * 16 <= kTmemCols, "TMEM budget");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

struct DynArgs {
  const uint16_t* x;  // bf16 [M, K], row pitch ldx elements
  int64_t ldx;
  const uint8_t* sfb;
  const float* gb;
  float* g_out;  // optional: g_a
  int M, N, K;
  int tiles_n;
  int* status;
};

__device__ __forceinline__ void named_barrier(uint32_t id, uint32_t threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}
__device__ __forceinline__ void st_shared_v2_u32(uint32_t addr, uint32_t a, uint32_t b) {
  asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}
__device__ __forceinline__ void st_shared_u32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ void st_shared_u8(uint32_t addr, uint32_t v) {
  asm volatile("st.shared.u8 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

template <class C>
__global__ void __launch_bounds__(C::kThreads, 1)
    nvfp4_linear_dyn_kernel(const __grid_constant__ CUtensorMap tmap_b, const __grid_constant__ CUtensorMap tmap_out,
                            const DynArgs args) {
  constexpr int BN = C::BN;
  constexpr int kStages = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;                                        // resident A, one 16 KiB tile per k-block
  uint8_t* sB = sA + C::kMaxKb * C::kTileBytesA;
  uint8_t* sEpi = sB + kStages * C::kTileBytesB;
  uint8_t* sSFA = sEpi + C::kEpiWarps * kEpiBufBytes;        // resident A scale atoms
  uint8_t* sSFB = sSFA + C::kMaxKb * C::kSfaBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sSFB + kStages * C::kSfbBytes);
  uint64_t* empty = full + kStages;
  uint64_t* sfready = empty + kStages;
  uint64_t* tfull = sfready + kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* aready = tempty + 2;
  uint64_t* drain = aready + 1;
  uint64_t* drain_cp = drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_cp + 1);
  __shared__ volatile int abort_flag;
  __shared__ uint32_t warp_max[C::kThreads / 32];
  __shared__ float s_g;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kblocks = args.K / BK;
  const int kgroups = args.K / 64;
  const int total_units = args.tiles_n;
  const int cta_id = blockIdx.x, n_ctas = gridDim.x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&sfready[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], C::kEpiWarps);
    }
    mbar_init(aready, 1);
    mbar_init(drain, 1);
    mbar_init(drain_cp, 1);
    abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmap_b);
    prefetch_tmap(&tmap_out);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait_and_release();
  const uint32_t tmem = *tmem_slot;

  auto fail = [&]() {
    set_status(args.status, NVFP4_ERR_TIMEOUT);
    abort_flag = 1;
  };

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer ---
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_parity[kStages];
      bool issued[kStages];
      for (int s = 0; s < kStages; ++s) issued[s] = false;
      for (int u = cta_id; u < total_units && !abort_flag; u += n_ctas) {
        const uint8_t* sfb_tile = args.sfb + (static_cast<size_t>(u) * kgroups) * 512;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, &abort_flag)) { fail(); break; }
          mbar_arrive_expect_tx(&full[stage], C::kTileBytesB + C::kSfbBytes);
          bulk_load(sSFB + stage * C::kSfbBytes, sfb_tile + static_cast<size_t>(kb) * C::kSfbBytes, C::kSfbBytes,
                    &full[stage]);
          tma_load_2d(sB + stage * C::kTileBytesB, &tmap_b, &full[stage], kb * (BK / 2), u * BN);
          issued[stage] = true;
          issued_parity[stage] = phase;
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
      }
      if (abort_flag)
        for (int s = 0; s < kStages; ++s)
          if (issued[s]) mbar_wait_bounded(&full[s], issued_parity[s], nullptr);
    }
  } else {
    // ------------------------------- prologue: g_a and A into shared memory ---
    // Thread pt owns the 16-element blocks pt, pt + 352, ... of x in row-major
    // block order; they stay in registers from the amax pass to the
    // quantization pass, so x is read once.
    constexpr int kKeep = 10;
    static_assert(kKeep * C::kProThreads >= C::kMaxRows * C::kMaxKb * (BK / 16), "x fits in registers");
    const uint32_t pt = threadIdx.x - 32;
    const uint32_t kb16 = static_cast<uint32_t>(args.K) / 16;
    const uint32_t M = static_cast<uint32_t>(args.M);
    const uint32_t live = M * kb16;
    auto block_src = [&](uint32_t b) {
      const uint32_t r = b / kb16, j = b - r * kb16;
      return reinterpret_cast<const uint4*>(args.x + static_cast<int64_t>(r) * args.ldx + j * 16);
    };
    uint4 lo[kKeep], hi[kKeep];
#pragma unroll
    for (int i = 0; i < kKeep; ++i) {
      const uint32_t b = pt + i * C::kProThreads;
      lo[i] = hi[i] = make_uint4(0, 0, 0, 0);
      if (b < live) {
        const uint4* src = block_src(b);
        lo[i] = __ldg(src);
        hi[i] = __ldg(src + 1);
      }
    }
    const uint32_t sA0 = smem_u32(sA), sSFA0 = smem_u32(sSFA);
    // Rows M..127 of the tile: zero codes and zero scales, as the two-call
    // path gets from the TMA fill and the quantizer's padding rows.
    {
      const uint32_t pad_chunks = (128u - M) * 8u;  // 16-byte chunks per k-block
      for (uint32_t i = pt; i < static_cast<uint32_t>(kblocks) * pad_chunks; i += C::kProThreads) {
        const uint32_t kb = i / pad_chunks, c = i - kb * pad_chunks;
        st_shared_v4(sA0 + kb * C::kTileBytesA + M * 128u + c * 16u, 0u, 0u, 0u, 0u);
      }
      const uint32_t pad_rows = 128u - M;
      for (uint32_t i = pt; i < static_cast<uint32_t>(kgroups) * pad_rows; i += C::kProThreads) {
        const uint32_t jg = i / pad_rows, r = M + (i - jg * pad_rows);
        st_shared_u32(sSFA0 + jg * 512u + (r & 31u) * 16u + ((r >> 5) & 3u) * 4u, 0u);
      }
    }
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < kKeep; ++i) m = max(m, max(amax_bits_bf16x8(lo[i]), amax_bits_bf16x8(hi[i])));
    m = __reduce_max_sync(0xffffffffu, m);
    if (lane == 0) warp_max[warp] = m;
    named_barrier(1, C::kProThreads);
    if (pt == 0) {
      uint32_t mm = 0;
      for (int w = 1; w < C::kThreads / 32; ++w) mm = max(mm, warp_max[w]);
      // g_a = amax / (6 * 448), or 1 for an all-zero tensor: the dynamic
      // quantizer's tensor scale, bit for bit.
      const float amax = __uint_as_float(mm << 16);
      const float gv = amax > 0.0f ? __fdiv_rn(amax, 2688.0f) : 1.0f;
      s_g = gv;
      if (blockIdx.x == 0 && args.g_out) *args.g_out = gv;
    }
    named_barrier(1, C::kProThreads);
    const float g = s_g, six_g = __fmul_rn(6.0f, g);
    // One 16-element block: E4M3 scale and 16 E2M1 codes, stored where the
    // TMA load of the two-call path would have put them (row r at r * 128 in
    // its k-block tile, 16-byte chunk c at (c ^ r % 8) * 16) and the scale
    // byte at its place in the 512-byte atom of its 64-element group.
    auto quantize_block = [&](uint32_t b, const uint4 v0, const uint4 v1) {
      const uint32_t r = b / kb16, j = b - r * kb16;
      float xf[16];
      unpack_bf16x8(v0, xf);
      unpack_bf16x8(v1, xf + 8);
      const float amax = __uint_as_float(max(amax_bits_bf16x8(v0), amax_bits_bf16x8(v1)) << 16);
      const BlockScale bs = block_scale(amax, g, six_g);
      float q[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) q[i] = __fmul_rn(xf[i], bs.mult);
      const uint32_t kb = j >> 4, e = j & 15u;
      st_shared_v2_u32(sA0 + kb * C::kTileBytesA + r * 128u + (((e >> 1) ^ (r & 7u)) << 4) + (e & 1u) * 8u,
                       e2m1x8(q), e2m1x8(q + 8));
      st_shared_u8(sSFA0 + (j >> 2) * 512u + (r & 31u) * 16u + ((r >> 5) & 3u) * 4u + (j & 3u), bs.code);
    };
#pragma unroll
    for (int i = 0; i < kKeep; ++i) {
      const uint32_t b = pt + i * C::kProThreads;
      if (b < live) quantize_block(b, lo[i], hi[i]);
    }
    fence_proxy_async_smem();  // the tensor core reads A and its scales through the async proxy
    named_barrier(1, C::kProThreads);

    if (warp == 1 && lane == 0) {
      // ------------------------------------------------------- MMA issuer ---
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      const uint32_t sB0 = smem_u32(sB);
      bool ok = mbar_wait_bounded(aready, 0, &abort_flag);
      if (!ok) fail();
      for (int u = cta_id; ok && u < total_units && !abort_flag; u += n_ctas, ++local) {
        const int acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!mbar_wait_bounded(&tempty[acc], acc_phase ^ 1u, &abort_flag)) { fail(); break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem + acc * BN;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_bounded(&sfready[stage], phase, &abort_flag)) { fail(); ok = false; break; }
          tc_fence_after();
          const uint32_t sfa_col = tmem + C::kSfaResCol + kb * 16;
          const uint32_t sfb_col = tmem + C::kSfbCol + stage * 16;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_fp4(d_tmem, desc_sw128(sA0 + kb * C::kTileBytesA + kk * 32),
                    desc_sw128(sB0 + stage * C::kTileBytesB + kk * 32), C::kIdesc, sfa_col + kk * 4,
                    sfb_col + kk * 4, (kb | kk) != 0);
          tc_commit(&empty[stage]);
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        tc_commit(&tfull[acc]);
      }
      tc_commit(drain);
      mbar_wait_bounded(drain, 0, nullptr);
    } else if (warp == 2 && lane == 0) {
      // ------------------------------------------- block scales -> TMEM ---
      for (int kb = 0; kb < kblocks; ++kb)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          copy_sf_to_tmem(tmem + C::kSfaResCol + kb * 16 + kk * 4, desc_sf(sSFA0 + kb * C::kSfaBytes + kk * 512));
      tc_commit(aready);
      int stage = 0;
      uint32_t phase = 0;
      const uint32_t sSFB0 = smem_u32(sSFB);
      bool ok = true;
      for (int u = cta_id; ok && u < total_units && !abort_flag; u += n_ctas) {
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_bounded(&full[stage], phase, &abort_flag)) { fail(); ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            copy_sf_to_tmem(tmem + C::kSfbCol + stage * 16 + kk * 4, desc_sf(sSFB0 + stage * C::kSfbBytes + kk * 512));
          tc_commit(&sfready[stage]);
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
      }
      tc_commit(drain_cp);
      mbar_wait_bounded(drain_cp, 0, nullptr);
    } else if (warp >= 3 && warp < 3 + C::kEpiWarps) {
      // --------------------------------------------------------- epilogue ---
      const int quarter = warp & 3;
      uint8_t* buf_ptr = sEpi + (warp - 3) * kEpiBufBytes;
      const uint32_t buf = smem_u32(buf_ptr);
      const float scale = __fmul_rn(g, __ldg(args.gb));
      int local = 0;
      for (int u = cta_id; u < total_units; u += n_ctas, ++local) {
        const int acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        int ok = 1;
        if (lane == 0) {
          ok = !abort_flag && mbar_wait_bounded(&tfull[acc], acc_phase, &abort_flag);
          if (!ok && !abort_flag) fail();
        }
        if (!__shfl_sync(0xffffffffu, ok, 0)) break;
        tc_fence_after();
        uint32_t r[128];
        const uint32_t taddr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(taddr + c * 32, r + 32 * c);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (lane == 0) bulk_wait_read_all();
          __syncwarp();
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint32_t* v = r + 64 * h + 8 * c;
            st_shared_v4(buf + lane * 128 + ((c ^ (lane & 7)) << 4),
                         pack_bf16x2(__uint_as_float(v[0]) * scale, __uint_as_float(v[1]) * scale),
                         pack_bf16x2(__uint_as_float(v[2]) * scale, __uint_as_float(v[3]) * scale),
                         pack_bf16x2(__uint_as_float(v[4]) * scale, __uint_as_float(v[5]) * scale),
                         pack_bf16x2(__uint_as_float(v[6]) * scale, __uint_as_float(v[7]) * scale));
          }
          fence_proxy_async_smem();
          __syncwarp();
          const int x = u * BN + h * kEpiCols, y = quarter * 32;
          if (lane == 0 && x < args.N && y < args.M) {
            tma_store_2d(&tmap_out, buf_ptr, x, y);
            bulk_commit_group();
          }
        }
      }
      if (lane == 0) bulk_wait_all();
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

// MMA-layout block scales of a [rows, K] operand viewed as [bytes / 256, 256]
// bytes; a box of 8 rows is one (128-row tile, k-block) group of four atoms.
bool make_scale_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t K) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const int64_t bytes = ((rows + 127) / 128) * 128 * (K / 16);
  cuuint64_t dims[2] = {256, static_cast<cuuint64_t>(bytes / 256)};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {256, 8};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// bf16 [M, N] output with row pitch ldo, stored in 32 x 64 boxes, 128-B swizzle.
bool make_out_map(CUtensorMap* map, void* base, int64_t M, int64_t N, int64_t ldo) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(N), static_cast<cuuint64_t>(M)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ldo * 2)};
  cuuint32_t box[2] = {kEpiCols, kEpiRows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Per-device, per-configuration launch set-up: the shared-memory opt-in and
// the number of clusters resident on the GPU at once (persistent grid).
template <class C>
int resident_ctas() {
  static std::mutex mu;
  static std::map<int, int> cache;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(d);
  if (it != cache.end()) return it->second;
  if (cudaFuncSetAttribute(nvfp4_gemm_kernel<C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(C::kSmemBytes)) != cudaSuccess)
    return 0;
  const int n = sm_count();  // one CTA per SM (launch bounds and shared memory allow no more)
  cache[d] = n;
  return n;
}

template <class C>
nvfp4_status launch(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a, const uint8_t* w_codes,
                    const uint8_t* w_scales, const float* g_w, int64_t M, int64_t N, int64_t K, void* out_bf16,
                    int64_t ldo, cudaStream_t stream, uint32_t idesc_fmt) {
  const int64_t tiles_m = (M + BM - 1) / BM, tiles_n = (N + C::BN - 1) / C::BN;
  const int64_t units = tiles_m * tiles_n;
  if (units >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  CUtensorMap ma, mb, mo;
  if (!make_code_map(&ma, a_codes, M, K, BM) || !make_code_map(&mb, w_codes, N, K, C::BN) ||
      !make_out_map(&mo, out_bf16, M, N, ldo))
    return NVFP4_ERR_CUDA;
  const int ctas_max = resident_ctas<C>();
  if (ctas_max <= 0) return NVFP4_ERR_CUDA;
  GemmArgs args = {};
  args.idesc_fmt = idesc_fmt;
  args.sfa = a_scales;
  args.sfb = w_scales;
  args.ga = g_a;
  args.gb = g_w;
  args.M = static_cast<int>(M);
  args.N = static_cast<int>(N);
  args.K = static_cast<int>(K);
  args.tiles_m = static_cast<int>(tiles_m);
  args.tiles_n = static_cast<int>(tiles_n);
  args.group_m = raster_group(K, units / tiles_n);
  args.status = status_word_dev();
  const int ctas = static_cast<int>(units < ctas_max ? units : ctas_max);
  if (launch_pdl(nvfp4_gemm_kernel<C>, dim3(ctas), dim3(C::kThreads), C::kSmemBytes, stream, ma, mb, mo, args) !=
      cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

template <class C, bool kSwiGLU>
int resident_pairs() {
  static std::mutex mu;
  static std::map<int, int> cache;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(d);
  if (it != cache.end()) return it->second;
  if (cudaFuncSetAttribute(nvfp4_gemm_pair_kernel<C, kSwiGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(C::kSmemBytes)) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(2 * (sm_count() / 2), 1, 1);
  cfg.blockDim = dim3(C::kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, nvfp4_gemm_pair_kernel<C, kSwiGLU>, &cfg) != cudaSuccess ||
      clusters <= 0) {
    cudaGetLastError();
    return 0;
  }
  cache[d] = clusters;
  return clusters;
}

// kSwiGLU: out_bf16 is unused (no output map); the fused outputs go through
// args.q_codes / q_scales / g_out, which the caller fills in `extra`.
template <class C, bool kSwiGLU = false>
nvfp4_status launch_pair(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a, const uint8_t* w_codes,
                         const uint8_t* w_scales, const float* g_w, int64_t M, int64_t N, int64_t K, void* out_bf16,
                         int64_t ldo, cudaStream_t stream, const GemmArgs* extra = nullptr,
                         uint32_t idesc_fmt = 0) {
  const int64_t tiles_m = (M + BM - 1) / BM, tiles_n = N / C::BN;
  const int64_t units = ((tiles_m + 1) / 2) * tiles_n;
  if (units >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  CUtensorMap ma, mb, msa, msb, mo;
  if (!make_code_map(&ma, a_codes, M, K, BM) || !make_code_map(&mb, w_codes, N, K, 128) ||
      !make_scale_map(&msa, a_scales, M, K) || !make_scale_map(&msb, w_scales, N, K))
    return NVFP4_ERR_CUDA;
  if (kSwiGLU) mo = ma;  // not read by the fused epilogue
  else if (!make_out_map(&mo, out_bf16, M, N, ldo)) return NVFP4_ERR_CUDA;
  const int pairs_max = resident_pairs<C, kSwiGLU>();
  if (pairs_max <= 0) return NVFP4_ERR_CUDA;
  GemmArgs args = {};
  if (extra) args = *extra;
  args.idesc_fmt = idesc_fmt;
  args.sfa = a_scales;
  args.sfb = w_scales;
  args.ga = g_a;
  args.gb = g_w;
  args.M = static_cast<int>(M);
  args.N = static_cast<int>(N);
  args.K = static_cast<int>(K);
  args.tiles_m = static_cast<int>(tiles_m);
  args.tiles_n = static_cast<int>(tiles_n);
  args.group_m = raster_group(K, units / tiles_n);
  args.status = status_word_dev();
  args.fault_skip_stage = take_fault(NVFP4_FAULT_GEMM_SKIP_STAGE) ? 1 : 0;
  args.out = static_cast<uint16_t*>(out_bf16);
  args.ldo = ldo;
  const int pairs = static_cast<int>(units < pairs_max ? units : pairs_max);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  cfg.blockDim = dim3(C::kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (cudaLaunchKernelEx(&cfg, nvfp4_gemm_pair_kernel<C, kSwiGLU>, ma, mb, msa, msb, mo, args) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

using SplitCfg = PairCfg<NVFP4_GEMM_PAIR_STAGES>;

// Clusters of `size` CTAs of the split-K kernel that are resident on the GPU
// at once (0 if that cluster shape cannot be launched).
int resident_split_clusters(int size) {
  static std::mutex mu;
  static std::map<std::pair<int, int>, int> cache;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find({d, size});
  if (it != cache.end()) return it->second;
  int clusters = 0;
  if (cudaFuncSetAttribute(nvfp4_gemm_splitk_kernel<SplitCfg>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(SplitCfg::kSmemBytes)) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = size;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(size * (sm_count() / size), 1, 1);
    cfg.blockDim = dim3(SplitCfg::kThreads, 1, 1);
    cfg.dynamicSmemBytes = SplitCfg::kSmemBytes;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&clusters, nvfp4_gemm_splitk_kernel<SplitCfg>, &cfg) != cudaSuccess)
      clusters = 0;
  }
  cudaGetLastError();
  cache[{d, size}] = clusters;
  return clusters;
}

// Pairs per tile for the split-K kernel: among S = 2..4 with every tile's
// cluster of 2S CTAs resident at once, the one with the fewest k-blocks per
// pair (ties: the smaller S, less to reduce); 0 if none.  On GB300 clusters
// of 4, 6 and 8 CTAs of this kernel fit about 36, 24 and 16 at a time, so the
// 14B decode qkv (28 tiles) takes S = 2 and the o and down GEMMs (20 tiles)
// S = 3.  The cross-CTA reduction costs ~3-4 us, which only pays with a long
// K: measured back to back on GB300, 256 x 7168 x 5120 11.9 -> 11.1 us,
// 256 x 5120 x 5120 11.8 -> 10.7 us, 256 x 5120 x 13824 24.8 -> 15.2 us, but
// 16 x 1536 x 1536 (6 k-blocks) 5.7 -> 7.2 us; so K needs 16 k-blocks.
constexpr int64_t kSplitMinKblocks = 16;
int choose_splits(int64_t tiles, int64_t kblocks) {
  if (kblocks < kSplitMinKblocks) return 0;
  int best = 0;
  int64_t best_kb = kblocks;
  for (int S = 2; S <= 4; ++S) {
    if (kblocks < S || tiles > resident_split_clusters(2 * S)) continue;
    const int64_t kb = (kblocks + S - 1) / S;
    if (kb < best_kb) { best = S; best_kb = kb; }
  }
  return best;
}

nvfp4_status launch_splitk(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a, const uint8_t* w_codes,
                           const uint8_t* w_scales, const float* g_w, int64_t M, int64_t N, int64_t K, void* out_bf16,
                           int64_t ldo, cudaStream_t stream, uint32_t idesc_fmt, int splits) {
  using C = SplitCfg;
  const int64_t tiles_m = (M + BM - 1) / BM, tiles_n = N / C::BN;
  const int64_t tiles = ((tiles_m + 1) / 2) * tiles_n;
  if (tiles * 2 * splits >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  CUtensorMap ma, mb, msa, msb, mo;
  if (!make_code_map(&ma, a_codes, M, K, BM) || !make_code_map(&mb, w_codes, N, K, 128) ||
      !make_scale_map(&msa, a_scales, M, K) || !make_scale_map(&msb, w_scales, N, K) ||
      !make_out_map(&mo, out_bf16, M, N, ldo))
    return NVFP4_ERR_CUDA;
  GemmArgs args = {};
  args.idesc_fmt = idesc_fmt;
  args.sfa = a_scales;
  args.sfb = w_scales;
  args.ga = g_a;
  args.gb = g_w;
  args.M = static_cast<int>(M);
  args.N = static_cast<int>(N);
  args.K = static_cast<int>(K);
  args.tiles_m = static_cast<int>(tiles_m);
  args.tiles_n = static_cast<int>(tiles_n);
  args.group_m = raster_group(K, tiles / tiles_n);
  args.splits = splits;
  args.status = status_word_dev();
  args.fault_skip_stage = take_fault(NVFP4_FAULT_GEMM_SKIP_STAGE) ? 1 : 0;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2 * splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(tiles * 2 * splits), 1, 1);
  cfg.blockDim = dim3(C::kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (cudaLaunchKernelEx(&cfg, nvfp4_gemm_splitk_kernel<C>, ma, mb, msa, msb, mo, args) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

// nvfp4_linear_dynamic: one persistent CTA per 128-column tile of W, at most
// one per SM.
nvfp4_status launch_dynamic(const uint16_t* x, int64_t M, int64_t K, int64_t ldx, const uint8_t* w_codes,
                            const uint8_t* w_scales, const float* g_w, int64_t N, void* out_bf16, int64_t ldo,
                            float* g_out, cudaStream_t stream) {
  using C = DynCfg;
  static std::mutex mu;
  static std::map<int, bool> ready;
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess) return NVFP4_ERR_CUDA;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (!ready[d]) {
      if (cudaFuncSetAttribute(nvfp4_linear_dyn_kernel<C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(C::kSmemBytes)) != cudaSuccess)
        return NVFP4_ERR_CUDA;
      ready[d] = true;
    }
  }
  const int64_t tiles_n = (N + C::BN - 1) / C::BN;
  CUtensorMap mb, mo;
  if (!make_code_map(&mb, w_codes, N, K, C::BN) || !make_out_map(&mo, out_bf16, M, N, ldo)) return NVFP4_ERR_CUDA;
  DynArgs args = {};
  args.x = x;
  args.ldx = ldx;
  args.sfb = w_scales;
  args.gb = g_w;
  args.g_out = g_out;
  args.M = static_cast<int>(M);
  args.N = static_cast<int>(N);
  args.K = static_cast<int>(K);
  args.tiles_n = static_cast<int>(tiles_n);
  args.status = status_word_dev();
  const int sms = sm_count();
  if (sms <= 0) return NVFP4_ERR_CUDA;
  const int ctas = static_cast<int>(tiles_n < sms ? tiles_n : sms);
  if (launch_pdl(nvfp4_linear_dyn_kernel<C>, dim3(ctas), dim3(C::kThreads), C::kSmemBytes, stream, mb, mo, args) !=
      cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

#ifndef NVFP4_GEMM_BN
#define NVFP4_GEMM_BN 0  // 0: choose per shape
#endif
#ifndef NVFP4_GEMM_SPLITK
#define NVFP4_GEMM_SPLITK 1  // 0: never use the split-K kernel
#endif
#ifndef NVFP4_GEMM_PAIR
#define NVFP4_GEMM_PAIR 1  // 0: never use the CTA-pair kernel
#endif
#ifndef NVFP4_GEMM_RES
#define NVFP4_GEMM_RES 1  // 0: never use the W-resident form
#endif

using PairRes = PairCfg<4, true>;

// The W-resident form pays when a pair gets runs of two or more units (more
// units than pairs); K must fit its shared-memory and TMEM budget, and its
// copy-after-read order needs at least as many k-blocks as ring stages.
// Measured on GB300 (graph-replayed, L2 flushed): gate_up of the 1.5B
// prefill (2048 x 17920 x 1536) 38.0 -> 35.7 us; with 4 k-blocks
// (8192 x 5120 x 1024) it was slower, so it starts at 5.
bool use_w_resident(int64_t pair_units, int64_t K, int pairs) {
  const int64_t kblocks = K / BK;
  return NVFP4_GEMM_RES && pairs > 0 && pair_units > pairs && kblocks >= PairRes::kStages + 1 &&
         kblocks <= PairRes::kResKblocks;
}

}  // namespace
}  // namespace nvfp4

using namespace nvfp4;

namespace nvfp4 {
namespace {
// Kernel choice for one block-scaled linear (arguments already validated).
nvfp4_status linear_dispatch(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a,
                             const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w, int64_t M, int64_t N,
                             int64_t K, void* out_bf16, int64_t ldo, cudaStream_t s, uint32_t idesc_fmt) {
  const int64_t tiles_m = (M + BM - 1) / BM;
  // The CTA pair, unless its 256 x 256 tiles would leave most pairs idle
  // (decode-sized M): then, with a long K, the split-K clusters, else 128 x
  // 128 tiles on single CTAs, which spread the W stream over more SMs than
  // the pairs would (measured faster at M = 256 with N = 5120 or 7168, slower
  // with N = 27648).
  using Pair = PairCfg<NVFP4_GEMM_PAIR_STAGES>;
  if (NVFP4_GEMM_PAIR && N % 256 == 0 && tiles_m >= 2) {
    const int64_t pair_units = ((tiles_m + 1) / 2) * (N / 256);
    if (use_w_resident(pair_units, K, resident_pairs<PairRes, false>()))
      return launch_pair<PairRes>(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, N, K, out_bf16, ldo, s,
                                  nullptr, idesc_fmt);
    if (2 * pair_units >= resident_pairs<Pair, false>())
      return launch_pair<Pair>(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, N, K, out_bf16, ldo, s, nullptr,
                               idesc_fmt);
  }
  // Too few pair tiles for the GPU: split K across clusters of CTA pairs.
  if (NVFP4_GEMM_SPLITK && N % 256 == 0) {
    const int splits = choose_splits(((tiles_m + 1) / 2) * (N / 256), K / BK);
    if (splits)
      return launch_splitk(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, N, K, out_bf16, ldo, s, idesc_fmt,
                           splits);
  }
  // Single CTAs: BN = 128 (measured faster than 256 at M <= 256 on GB300).
  const int bn = NVFP4_GEMM_BN ? NVFP4_GEMM_BN : 128;
  if (bn == 256)
    return launch<Cfg<256, 3>>(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, N, K, out_bf16, ldo, s, idesc_fmt);
  return launch<Cfg<128, 5>>(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, N, K, out_bf16, ldo, s, idesc_fmt);
}

}  // namespace
}  // namespace nvfp4

NVFP4_API nvfp4_status nvfp4_linear(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a,
                                    const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w, int64_t M,
                                    int64_t N, int64_t K, void* out_bf16, int64_t ldo, void* stream) {
  NVFP4_TRACE("nvfp4_linear");
  if (!a_codes || !a_scales || !g_a || !w_codes || !w_scales || !g_w || !out_bf16) return NVFP4_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0 || K % BK || N % 16 || ldo < N || ldo % 8) return NVFP4_ERR_SHAPE;
  if (M >= (1ll << 31) || N >= (1ll << 31) || K >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(a_scales, 16) || !aligned(w_scales, 16) ||
      !aligned(out_bf16, 16) || !aligned(g_a, 4) || !aligned(g_w, 4))
    return NVFP4_ERR_ALIGN;
  return linear_dispatch(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, N, K, out_bf16, ldo,
                         static_cast<cudaStream_t>(stream), 0);
}

NVFP4_API nvfp4_status nvfp4_linear_dynamic(const void* x_bf16, int64_t M, int64_t K, int64_t ld_x,
                                            const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w,
                                            int64_t N, void* out_bf16, int64_t ldo, float* g_a_out, void* stream) {
  NVFP4_TRACE("nvfp4_linear_dynamic");
  if (!x_bf16 || !w_codes || !w_scales || !g_w || !out_bf16) return NVFP4_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0 || K % BK || N % 16 || ldo < N || ldo % 8 || ld_x < K) return NVFP4_ERR_SHAPE;
  if (M > DynCfg::kMaxRows || K > static_cast<int64_t>(DynCfg::kMaxKb) * BK) return NVFP4_ERR_UNSUPPORTED;
  if (N >= (1ll << 31) || ld_x >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(x_bf16, 16) || ld_x % 8 || !aligned(w_codes, 16) || !aligned(w_scales, 16) || !aligned(out_bf16, 16) ||
      !aligned(g_w, 4) || !aligned(g_a_out, 4))
    return NVFP4_ERR_ALIGN;
  return launch_dynamic(static_cast<const uint16_t*>(x_bf16), M, K, ld_x, w_codes, w_scales, g_w, N, out_bf16, ldo,
                        g_a_out, static_cast<cudaStream_t>(stream));
}

NVFP4_API nvfp4_status mxfp4_linear(const uint8_t* a_codes, const uint8_t* a_scales, const uint8_t* w_codes,
                                    const uint8_t* w_scales, int64_t M, int64_t N, int64_t K, void* out_bf16,
                                    int64_t ldo, void* stream) {
  NVFP4_TRACE("mxfp4_linear");
  if (!a_codes || !a_scales || !w_codes || !w_scales || !out_bf16) return NVFP4_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0 || K % BK || N % 16 || ldo < N || ldo % 8) return NVFP4_ERR_SHAPE;
  if (M >= (1ll << 31) || N >= (1ll << 31) || K >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(a_scales, 16) || !aligned(w_scales, 16) ||
      !aligned(out_bf16, 16))
    return NVFP4_ERR_ALIGN;
  return linear_dispatch(a_codes, a_scales, nullptr, w_codes, w_scales, nullptr, M, N, K, out_bf16, ldo,
                         static_cast<cudaStream_t>(stream), kScaleE8M0);
}

NVFP4_API nvfp4_status nvfp4_linear_swiglu_quantize(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a,
                                                    const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w,
                                                    int64_t M, int64_t I, int64_t K, const float* g_out,
                                                    uint8_t* out_codes, uint8_t* out_scales, void* stream) {
  NVFP4_TRACE("nvfp4_linear_swiglu_quantize");
  if (!a_codes || !a_scales || !g_a || !w_codes || !w_scales || !g_w || !g_out || !out_codes || !out_scales)
    return NVFP4_ERR_INVALID_ARG;
  if (M <= 0 || I <= 0 || K <= 0 || K % BK || I % 128) return NVFP4_ERR_SHAPE;
  if (M >= (1ll << 31) || 2 * I >= (1ll << 31) || K >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(a_scales, 16) || !aligned(w_scales, 16) ||
      !aligned(out_codes, 16) || !aligned(out_scales, 4) || !aligned(g_a, 4) || !aligned(g_w, 4) || !aligned(g_out, 4))
    return NVFP4_ERR_ALIGN;
  GemmArgs extra = {};
  extra.q_codes = out_codes;
  extra.q_scales = out_scales;
  extra.g_out = g_out;
  const int64_t pair_units = ((M + 2 * BM - 1) / (2 * BM)) * (2 * I / 256);
  if (use_w_resident(pair_units, K, resident_pairs<PairRes, true>()))
    return launch_pair<PairRes, true>(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, 2 * I, K, nullptr, 0,
                                      static_cast<cudaStream_t>(stream), &extra);
  return launch_pair<PairCfg<NVFP4_GEMM_PAIR_STAGES>, true>(a_codes, a_scales, g_a, w_codes, w_scales, g_w, M, 2 * I,
                                                           K, nullptr, 0, static_cast<cudaStream_t>(stream), &extra);
}

NVFP4_API nvfp4_status mxfp4_linear_swiglu_quantize(const uint8_t* a_codes, const uint8_t* a_scales,
                                                    const uint8_t* w_codes, const uint8_t* w_scales, int64_t M,
                                                    int64_t I, int64_t K, int rotate, uint8_t* out_codes,
                                                    uint8_t* out_scales, void* stream) {
  NVFP4_TRACE("mxfp4_linear_swiglu_quantize");
  if (!a_codes || !a_scales || !w_codes || !w_scales || !out_codes || !out_scales) return NVFP4_ERR_INVALID_ARG;
  if (rotate != 0 && rotate != 1) return NVFP4_ERR_INVALID_ARG;
  if (M <= 0 || I <= 0 || K <= 0 || K % BK || I % 128) return NVFP4_ERR_SHAPE;
  if (M >= (1ll << 31) || 2 * I >= (1ll << 31) || K >= (1ll << 31)) return NVFP4_ERR_SHAPE;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(a_scales, 16) || !aligned(w_scales, 16) ||
      !aligned(out_codes, 16) || !aligned(out_scales, 4))
    return NVFP4_ERR_ALIGN;
  GemmArgs extra = {};
  extra.q_codes = out_codes;
  extra.q_scales = out_scales;
  extra.q_mode = rotate ? 2u : 1u;
  const int64_t pair_units = ((M + 2 * BM - 1) / (2 * BM)) * (2 * I / 256);
  if (use_w_resident(pair_units, K, resident_pairs<PairRes, true>()))
    return launch_pair<PairRes, true>(a_codes, a_scales, nullptr, w_codes, w_scales, nullptr, M, 2 * I, K, nullptr,
                                      0, static_cast<cudaStream_t>(stream), &extra, kScaleE8M0);
  return launch_pair<PairCfg<NVFP4_GEMM_PAIR_STAGES>, true>(a_codes, a_scales, nullptr, w_codes, w_scales, nullptr, M,
                                                           2 * I, K, nullptr, 0, static_cast<cudaStream_t>(stream),
                                                           &extra, kScaleE8M0);
}

namespace nvfp4 {
namespace {
// out row 32j + t = gate row 16j + t, out row 32j + 16 + t = up row 16j + t
// (t < 16); one thread moves 16 bytes.
__global__ void interleave_gate_up_kernel(const uint4* __restrict__ gate, const uint4* __restrict__ up,
                                          uint4* __restrict__ out, uint64_t row_chunks, uint64_t n) {
  griddep_wait_and_release();
  for (uint64_t k = blockIdx.x * static_cast<uint64_t>(blockDim.x) + threadIdx.x; k < n;
       k += static_cast<uint64_t>(gridDim.x) * blockDim.x) {
    const uint64_t orow = k / row_chunks, c = k - orow * row_chunks;
    const uint64_t j = orow >> 5, t = orow & 31u;
    const uint64_t irow = 16 * j + (t & 15u);
    out[k] = __ldg((t < 16 ? gate : up) + irow * row_chunks + c);
  }
}
}  // namespace
}  // namespace nvfp4

NVFP4_API nvfp4_status nvfp4_interleave_gate_up(const void* w_gate, const void* w_up, int64_t I, int64_t row_bytes,
                                                void* w_out, void* stream) {
  NVFP4_TRACE("nvfp4_interleave_gate_up");
  if (!w_gate || !w_up || !w_out) return NVFP4_ERR_INVALID_ARG;
  if (I <= 0 || I % 16 || row_bytes <= 0 || row_bytes % 16) return NVFP4_ERR_SHAPE;
  if (!aligned(w_gate, 16) || !aligned(w_up, 16) || !aligned(w_out, 16)) return NVFP4_ERR_ALIGN;
  const uint64_t row_chunks = static_cast<uint64_t>(row_bytes) / 16, n = 2 * static_cast<uint64_t>(I) * row_chunks;
  uint64_t grid = (n + 255) / 256;
  const uint64_t cap = static_cast<uint64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  if (launch_pdl(interleave_gate_up_kernel, dim3(static_cast<int>(grid)), dim3(256), 0,
                 static_cast<cudaStream_t>(stream), static_cast<const uint4*>(w_gate), static_cast<const uint4*>(w_up),
                 static_cast<uint4*>(w_out), row_chunks, n) != cudaSuccess)
    return NVFP4_ERR_CUDA;
  count_launches(1);
  return launch_status();
}

#ifdef NVFP4_TIMELINE
// Timeline build only (not part of the C ABI of include/nvfp4.h): copy the
// per-CTA stamps of the last 1-CTA GEMM launch ([1024][8] uint64, ns, zero
// where a CTA or event did not occur) to host memory, then clear them.
// Synchronizes the device.
extern "C" __attribute__((visibility("default"))) int nvfp4_timeline_gemm(unsigned long long* host) {
  if (cudaDeviceSynchronize() != cudaSuccess) return 1;
  if (cudaMemcpyFromSymbol(host, nvfp4::g_gemm_timeline, sizeof(nvfp4::g_gemm_timeline)) != cudaSuccess) return 1;
  static unsigned long long zero[nvfp4::kGemmTimelineCtas * 8];
  return cudaMemcpyToSymbol(nvfp4::g_gemm_timeline, zero, sizeof(zero)) == cudaSuccess ? 0 : 1;
}
#endif
