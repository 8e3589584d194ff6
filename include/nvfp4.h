/*
 * nvfp4.h -- C ABI of the GB300 (sm_103a) NVFP4 W4A4KV4 hot path.
 *
 * The library implements the data-parallel inference path behind the paper's
 * deployment speedup: fully quantized NVFP4 execution of a transformer layer
 * ("W4A4KV4": 4-bit weights, activations and KV cache; Sec. 2.1, Sec. 5.3,
 * Appendix D.3).  NVFP4 is defined in Appendix A (table "Quantization
 * configurations of MXFP4 and NVFP4"): E2M1 elements, one FP8-E4M3 scale per
 * block of 16 elements, one FP32 scale per tensor.
 *
 * Conventions shared by every call
 *   - All pointers are DEVICE pointers unless a parameter says "host".  The
 *     caller owns every buffer; the library never allocates or frees memory.
 *   - Every call is asynchronous on `stream` (a cudaStream_t passed as void*,
 *     NULL = the legacy default stream) and never synchronizes, except
 *     nvfp4_get_device_status.  Calls are safe to capture in a CUDA graph.
 *   - bf16 tensors are row-major with a leading dimension in elements.
 *   - Host-side argument errors return a status before anything is launched.
 *     Faults only visible on the device (capacity overflow, a bad tensor
 *     scale, a bounded wait that timed out) set a per-device status word that
 *     nvfp4_get_device_status reads and clears; the kernel skips the affected
 *     writes and returns instead of trapping.
 *   - No C++ exceptions cross this boundary.
 *
 * Number formats
 *   codes  : packed E2M1, two per byte, element 2j in bits 0-3 and element
 *            2j+1 in bits 4-7 of byte j; a row of K elements is K/2 bytes.
 *   scales : unsigned E4M3 (OCP E4M3FN bit layout, sign always 0), one byte per
 *            16 consecutive elements of a row, in one of two storage orders
 *            (nvfp4_scale_layout).
 *   g      : FP32 tensor scale; an element dequantizes to e2m1 * e4m3 * g.
 *
 * Quantization recipe (the paper fixes the format, not the rounding; this is
 * the library's reading, identical in every kernel): per block of 16,
 *   s = amax / (6 g) in fp32; S = E4M3(s) round-to-nearest-even, saturating
 *   at 448; if S == 0 the block's codes are signed zeros, else each element
 *   becomes E2M1(x * (1 / (S g))) round-to-nearest-even, saturating at 6,
 *   sign kept.
 */
#ifndef NVFP4_H
#define NVFP4_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  NVFP4_OK = 0,
  NVFP4_ERR_INVALID_ARG = 1, /* null pointer, bad enum, non-finite scale      */
  NVFP4_ERR_SHAPE = 2,       /* unsupported or inconsistent sizes             */
  NVFP4_ERR_ALIGN = 3,       /* pointer / leading dimension not 16-B aligned  */
  NVFP4_ERR_UNSUPPORTED = 4, /* no sm_103a device, or device lacks a feature  */
  NVFP4_ERR_CUDA = 5,        /* a CUDA runtime/driver call or launch failed   */
  NVFP4_ERR_TIMEOUT = 6,     /* a bounded on-device wait gave up              */
  NVFP4_ERR_CAPACITY = 7,    /* KV append position beyond the cache capacity  */
  NVFP4_ERR_BOUNDS = 8       /* bounds-checked build only: a computed store   */
                             /* index left its buffer; the store was skipped  */
} nvfp4_status;

typedef enum {
  /* scales[r * (cols/16) + kb]: plain row-major [rows, cols/16].            */
  NVFP4_SCALES_ROWMAJOR = 0,
  /* The order the tensor core reads block scales in: rows grouped in tiles  *
   * of 128, K-blocks in groups of 4; each (row tile, k group) owns 512      *
   * contiguous bytes, k group fastest; inside, row r / k-block kb is at     *
   * (r%32)*16 + ((r%128)/32)*4 + kb%4.  Needs cols % 64 == 0; the buffer    *
   * holds ceil(rows/128)*128*(cols/16) bytes and padding rows are zeroed.   */
  NVFP4_SCALES_MMA = 1
} nvfp4_scale_layout;

/* Bytes of a scale buffer for a [rows, cols] tensor in the given layout. */
size_t nvfp4_scales_bytes(int64_t rows, int64_t cols, nvfp4_scale_layout layout);

/*
 * a1. FP32 tensor scale  g = amax(|x|) / (6 * 448)   (Appendix A: the FP32
 * global scale; with it the tensor's largest element maps onto the largest
 * NVFP4 value, E2M1 6 times E4M3 448).  An all-zero tensor gets g = 1.
 *   x_bf16 : [rows, cols] bf16, leading dimension ld >= cols (elements).
 *   g_dev  : one float, written on the device (never read first).
 * Three stream operations (clear, reduce, finalize).  Errors: null pointers
 * -> INVALID_ARG (x may be NULL when rows*cols == 0); rows or cols < 0,
 * ld < cols, cols % 8 != 0 -> SHAPE; x not 16-B aligned or ld % 8 != 0 ->
 * ALIGN.  rows*cols == 0 gives g = 1.
 */
nvfp4_status nvfp4_tensor_scale(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld,
                                float* g_dev, void* stream);

/*
 * a2. NVFP4 quantization of a bf16 tensor along its rows (Appendix A format,
 * recipe above).  Used for activations on the fly and, once, for weights.
 *   x_bf16  : [rows, cols] bf16, leading dimension ld (elements, ld % 8 == 0).
 *   g_dev   : device float, the tensor scale (from nvfp4_tensor_scale or a
 *             static calibration value).  g <= 0 or non-finite: the kernel
 *             writes zero codes and scales and sets INVALID_ARG on the device.
 *   codes   : [rows, cols/2] bytes, row pitch cols/2.
 *   scales  : nvfp4_scales_bytes(rows, cols, layout) bytes.
 * cols % 16 == 0 (ROWMAJOR) or cols % 64 == 0 (MMA), else SHAPE.  x must be
 * 16-B aligned, codes 8-B aligned (ALIGN).  rows*cols == 0 is a no-op (any
 * pointer may then be NULL); other null pointers -> INVALID_ARG.
 */
nvfp4_status nvfp4_quantize(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld,
                            const float* g_dev, uint8_t* codes, uint8_t* scales,
                            nvfp4_scale_layout layout, void* stream);

/* Bytes of caller-owned state used by nvfp4_quantize_dynamic. */
#define NVFP4_DYNAMIC_STATE_BYTES 16

/*
 * a1 + a2 in one kernel launch: the tensor scale g of x (exactly as
 * nvfp4_tensor_scale computes it) is stored in *g_dev and x is quantized
 * with it (exactly as nvfp4_quantize does); codes, scales and g are
 * bit-identical to the two calls in sequence.
 *   state_dev : NVFP4_DYNAMIC_STATE_BYTES of device memory, 16-B aligned,
 *               zero-filled once before its first use (the fill must be
 *               ordered before the call: same stream, or synchronized with
 *               it; a call that reads a stale state can report TIMEOUT) and
 *               left alone by the caller afterwards.  Calls that may run concurrently (other
 *               streams) need separate states; calls in one stream may share.
 *   g_dev     : device float, written (never read first).
 *   x, codes, scales, layout : as nvfp4_quantize.
 * A cooperative launch: a grid-wide barrier separates the amax reduction
 * from the quantization, and the second pass over x hits L2 when x fits in
 * it.  A barrier that does not complete within 2 s sets NVFP4_ERR_TIMEOUT
 * on the device and leaves the outputs unwritten; zero-fill the state again
 * before reusing it.  rows*cols == 0 writes g = 1 and nothing else.
 * Errors as nvfp4_quantize, plus: state_dev or g_dev NULL -> INVALID_ARG,
 * state_dev not 16-B aligned -> ALIGN.
 */
nvfp4_status nvfp4_quantize_dynamic(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld,
                                    void* state_dev, float* g_dev, uint8_t* codes, uint8_t* scales,
                                    nvfp4_scale_layout layout, void* stream);

/*
 * Reorder block scales between the two storage orders (both directions).
 * src and dst must not overlap.  cols % 64 == 0.
 */
nvfp4_status nvfp4_scales_relayout(const uint8_t* src, uint8_t* dst, int64_t rows, int64_t cols,
                                   nvfp4_scale_layout from, nvfp4_scale_layout to, void* stream);

/*
 * a3. Block-scaled FP4 x FP4 linear layer with bf16 output (every linear of
 * the decoder is quantized, Appendix D.1; the 4-bit GEMM is where the
 * paper's compute speedup comes from, Sec. 5.3):
 *   out[m, n] = bf16_rne( (g_a * g_w) * sum_k a[m,k] * w[n,k] )
 * with a[m,k] = e2m1 * e4m3 of A (no g) and likewise for W; the sum is
 * accumulated in fp32 by the tensor core (tcgen05 block-scaled MMA).  When
 * N % 256 == 0, K >= 4096 and the 256 x 256 tiles are too few to occupy the
 * GPU (decode-sized M), K is split into 2-4 contiguous ranges whose fp32 partial
 * sums are added in range order in the cluster's shared memory: the result
 * is deterministic for a given shape.
 *   a_codes  : [M, K/2] bytes (K-major), 16-B aligned.
 *   a_scales : MMA layout for [M, K].
 *   w_codes  : [N, K/2] bytes (K-major, i.e. the nn.Linear weight [N, K]).
 *   w_scales : MMA layout for [N, K].
 *   g_a,g_w  : device floats.
 *   out_bf16 : [M, N] bf16 with leading dimension ldo >= N (elements).
 * Requires K % 256 == 0, N % 16 == 0, ldo % 8 == 0, M,N,K > 0 (SHAPE),
 * pointers 16-B aligned (ALIGN).
 */
nvfp4_status nvfp4_linear(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a,
                          const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w,
                          int64_t M, int64_t N, int64_t K, void* out_bf16, int64_t ldo,
                          void* stream);

/*
 * a1 + a2 + a3 in one launch for a small activation: the tensor scale of x,
 * its NVFP4 quantization and the linear layer with W (Appendix A format,
 * Appendix D.1 linears; the tensor-scale reduction fused into the GEMM's
 * prologue).  Every CTA reduces the amax of the whole of x and quantizes it
 * into its own shared memory, so no grid barrier is needed.  g_a, the
 * quantized A and out are bit-identical to nvfp4_quantize_dynamic (MMA
 * scales) followed by nvfp4_linear; the quantized A is not written to
 * global memory.
 *   x_bf16   : [M, K] bf16, leading dimension ld_x >= K (elements), 16-B
 *              aligned, ld_x % 8 == 0.
 *   w_codes, w_scales, g_w, out_bf16, ldo : as nvfp4_linear.
 *   g_a_out  : device float that receives g_a, or NULL.
 * 1 <= M <= 32 and K <= 1536 (UNSUPPORTED otherwise: each CTA holds all of
 * x in registers and all of A in shared memory, and quantizes it itself;
 * measured on GB300 at N = K = 1536, one launch is faster than the two calls
 * up to M = 16, on par at M = 32 and 1.7x slower at M = 64); K % 256 == 0, N % 16 == 0, ldo >= N, ldo % 8 == 0
 * (SHAPE); pointers 16-B aligned, g_w and g_a_out 4-B aligned (ALIGN).  A
 * bounded on-device wait that expires sets NVFP4_ERR_TIMEOUT and leaves out
 * undefined.
 */
nvfp4_status nvfp4_linear_dynamic(const void* x_bf16, int64_t M, int64_t K, int64_t ld_x,
                                  const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w,
                                  int64_t N, void* out_bf16, int64_t ldo, float* g_a_out,
                                  void* stream);

/*
 * a3 for the gate_up projection, with the down projection's input produced in
 * the epilogue: h[m, i] = SiLU(G[m, i]) * U[m, i], where G and U are the gate
 * and up halves of the block-scaled product exactly as nvfp4_linear forms them
 * (fp32, scaled by g_a g_w, not rounded to bf16).  h is then NVFP4-quantized
 * with the static tensor scale g_out by the recipe of nvfp4_quantize and
 * written as the A operand of the down projection.  Every linear of the layer
 * is quantized (Appendix D.1); the paper's Q-FIT appendix notes that SwiGLU
 * makes the down projection's input the outlier-heavy activation.
 *   w_codes, w_scales : the [2I, K] gate/up weight, rows interleaved in blocks
 *                       of 16 (gate rows 16j..16j+15, then up rows 16j..16j+15;
 *                       nvfp4_interleave_gate_up on the bf16 weights, then
 *                       nvfp4_quantize with MMA scales).
 *   g_out             : device float, static scale of h (e.g. calibrated).
 *   out_codes         : [M, I/2] bytes, 16-B aligned.
 *   out_scales        : nvfp4_scales_bytes(M, I, NVFP4_SCALES_MMA) bytes, 4-B
 *                       aligned; padding rows are written as zeros.
 * SiLU is evaluated as x/2 (1 + tanh(x/2)) with the hardware tanh
 * approximation (relative error ~2^-11): h may differ from an exact SiLU by
 * that much, which changes a code only where h sits near a rounding boundary.  I % 128 == 0, K % 256 == 0, M, I, K > 0 (SHAPE).  g_out <= 0 or
 * non-finite: zero codes and scales, INVALID_ARG set on the device.
 */
nvfp4_status nvfp4_linear_swiglu_quantize(const uint8_t* a_codes, const uint8_t* a_scales, const float* g_a,
                                          const uint8_t* w_codes, const uint8_t* w_scales, const float* g_w,
                                          int64_t M, int64_t I, int64_t K, const float* g_out,
                                          uint8_t* out_codes, uint8_t* out_scales, void* stream);

/*
 * Row order for nvfp4_linear_swiglu_quantize: w_out row 32j + t = w_gate row
 * 16j + t and w_out row 32j + 16 + t = w_up row 16j + t (t < 16).  w_gate,
 * w_up: [I, *] rows of row_bytes bytes; w_out: [2I, *].  I % 16 == 0,
 * row_bytes % 16 == 0 (SHAPE); pointers 16-B aligned (ALIGN).
 */
nvfp4_status nvfp4_interleave_gate_up(const void* w_gate, const void* w_up, int64_t I, int64_t row_bytes,
                                      void* w_out, void* stream);

/*
 * MXFP4 format variant (Appendix A, table "Quantization configurations of
 * MXFP4 and NVFP4"): E2M1 elements, one E8M0 (power-of-two) scale per block
 * of 32 elements, no global scale; Sec. 5 evaluates MXFP4 W4A4 deployments.
 *
 * Bytes of an MXFP4 scale buffer for a [rows, cols] tensor: ROWMAJOR holds
 * one E8M0 byte per 32-element block ([rows, cols/32]); MMA holds the byte
 * order nvfp4_linear reads (nvfp4_scales_bytes(rows, cols, MMA) bytes), with
 * each block's scale stored for both of its 16-element halves.
 */
size_t mxfp4_scales_bytes(int64_t rows, int64_t cols, nvfp4_scale_layout layout);

/*
 * MXFP4-quantize a [rows, cols] bf16 tensor along its rows.  Per block of 32
 * consecutive elements (the paper fixes the format; the recipe is the OCP
 * Microscaling rule it cites):
 *   e = floor(log2(max |x_i|)) - 2, clamped to [-127, 127] (-127 for an
 *   all-zero block); scale code = e + 127;
 *   code_i = E2M1_RNE_satfinite(x_i / 2^e), sign kept (also for a value that
 *   rounds to zero); values in [6, 8) 2^e saturate to 6 2^e.
 * rotate = 1 first multiplies every 32-element block by H_32 / sqrt(32)
 * (Sylvester-Hadamard; the block-wise rotation applied before MXFP4
 * quantization, Sec. 4), computed in fp32 as butterflies (a + b, a - b) at
 * strides 1, 2, 4, 8, 16 and one multiplication by fp32(1/sqrt(32)); rotate
 * W's K dimension the same way so that the linear's product is unchanged.
 *   codes  : [rows, cols/2] bytes, element 2j in the low nibble of byte j,
 *            16-B aligned.
 *   scales : mxfp4_scales_bytes(rows, cols, layout) bytes; MMA padding rows
 *            are written as zeros.
 * cols % 32 == 0 (ROWMAJOR) or cols % 64 == 0 (MMA), else SHAPE; x 16-B
 * aligned and ld % 8 == 0 (ALIGN); rotate not 0/1 -> INVALID_ARG.
 * rows*cols == 0 is a no-op.  Inputs must be finite.
 */
nvfp4_status mxfp4_quantize(const void* x_bf16, int64_t rows, int64_t cols, int64_t ld, int rotate,
                            uint8_t* codes, uint8_t* scales, nvfp4_scale_layout layout, void* stream);

/*
 * a3 with MXFP4 operands: out[m, n] = bf16_rne( sum_k a[m,k] * w[n,k] ), a
 * and w the dequantized MXFP4 values (e2m1 * 2^e), accumulated in fp32 by the
 * tensor core (block-scaled MMA with UE8M0 scales).  Operands as
 * nvfp4_linear with MMA-layout MXFP4 scales (mxfp4_quantize(..., MMA)) and
 * no g.  Same shape and alignment rules as nvfp4_linear.
 */
nvfp4_status mxfp4_linear(const uint8_t* a_codes, const uint8_t* a_scales, const uint8_t* w_codes,
                          const uint8_t* w_scales, int64_t M, int64_t N, int64_t K, void* out_bf16,
                          int64_t ldo, void* stream);

/*
 * nvfp4_linear_swiglu_quantize for MXFP4 operands: the gate_up projection
 * with h[m, i] = SiLU(G[m, i]) * U[m, i] (the fp32 accumulators; SiLU as in
 * nvfp4_linear_swiglu_quantize) MXFP4-quantized in the epilogue by the recipe
 * of mxfp4_quantize, as the down projection's A operand.  E8M0 scales are
 * local to each 32-element block, so no output scale is needed.  rotate = 1
 * rotates each 32-element block of h by H_32 / sqrt(32) first (the down
 * weight's K dimension must be rotated the same way).
 *   a_codes, a_scales : MXFP4 A operand, MMA-layout scales.
 *   w_codes, w_scales : the [2I, K] MXFP4 gate/up weight, rows interleaved in
 *                       blocks of 16 as for nvfp4_linear_swiglu_quantize.
 *   out_codes         : [M, I/2] bytes, 16-B aligned.
 *   out_scales        : mxfp4_scales_bytes(M, I, NVFP4_SCALES_MMA) bytes, 4-B
 *                       aligned; padding rows are written as zeros.
 * I % 128 == 0, K % 256 == 0, M, I, K > 0 (SHAPE); rotate not 0/1 -> INVALID_ARG.
 */
nvfp4_status mxfp4_linear_swiglu_quantize(const uint8_t* a_codes, const uint8_t* a_scales,
                                          const uint8_t* w_codes, const uint8_t* w_scales, int64_t M,
                                          int64_t I, int64_t K, int rotate, uint8_t* out_codes,
                                          uint8_t* out_scales, void* stream);

/* Element grid of the KV cache (the block scales are E4M3 per 16 either way). */
typedef enum {
  /* E2M1, the NVFP4 element {0, 0.5, 1, 1.5, 2, 3, 4, 6} (the B200 deployment's
   * native 4-bit KV cache, Appendix D.3).  Nibble = sign | E2M1 magnitude.  */
  NVFP4_KV_E2M1 = 0,
  /* E1M2, the KV element of the paper's QAT runs (Q-FIT section): read as the
   * bias-0 grid {0, 0.5, ..., 3.5}; block scale E4M3(amax / (3.5 g)), element
   * RNE(2|v|) saturated at 7, stored as the two's-complement nibble of
   * sign * k.  Decode attention reads it through integer tricks (no hardware
   * conversion), so it is slower than E2M1.                                 */
  NVFP4_KV_E1M2 = 1
} nvfp4_kv_format;

/*
 * NVFP4 KV cache (W4A4KV4; the B200 deployment uses a native 4-bit KV cache,
 * Appendix D.3).  One row per (sequence, KV head, position); the 16-element
 * blocks run along head_dim, so an appended token never touches older rows.
 *   k_codes, v_codes   : [batch, num_kv_heads, capacity, head_dim/2] bytes
 *   k_scales, v_scales : [batch, num_kv_heads, capacity, head_dim/16] bytes
 *   seq_lens           : device int32 [batch], valid tokens per sequence
 *                        (maintained by the caller; read by attention).
 *   k_gscale, v_gscale : static per-layer FP32 tensor scales (an append-only
 *                        cache cannot re-scale rows it already holds).
 *   kv_format          : nvfp4_kv_format of both K and V (0 = E2M1 when a
 *                        caller zero-initializes the struct).
 * head_dim must be 128.  Buffers 16-B aligned.  A kv_format other than the
 * enum's values -> INVALID_ARG in every call that takes the cache.
 */
typedef struct {
  uint8_t* k_codes;
  uint8_t* k_scales;
  uint8_t* v_codes;
  uint8_t* v_scales;
  const int32_t* seq_lens;
  int32_t batch;
  int32_t num_kv_heads;
  int32_t head_dim;
  int32_t capacity;
  float k_gscale;
  float v_gscale;
  int32_t kv_format;
} nvfp4_kv_cache;

/*
 * a4. Quantize n_new K/V rows and append them to the cache.  With k_shift the
 * Q-FIT post-RoPE shift is applied first, K~ = R(K) - m (Eq. 2; the paper
 * applies it after an unfused RoPE, Appendix D.3), in fp32.
 *   k_bf16, v_bf16 : [n_new, num_kv_heads, head_dim] bf16 (K already rotated).
 *   seq_idx, pos   : device int32 [n_new]: destination sequence and position.
 *   k_shift        : device float [num_kv_heads, head_dim] or NULL.
 * A row whose seq_idx is outside [0, batch) or pos outside [0, capacity) is
 * skipped and sets CAPACITY on the device.
 */
nvfp4_status kv_append_nvfp4(const nvfp4_kv_cache* cache, const void* k_bf16, const void* v_bf16,
                             const int32_t* seq_idx, const int32_t* pos, int64_t n_new,
                             const float* k_shift, void* stream);

/*
 * The fused step before decode attention (a4 with RoPE): K~ = RoPE(K_pre, pos)
 * - m, then quantize and store K~ and V exactly as kv_append_nvfp4 does (Eq. 2:
 * K~ = R(K_pre / s) - m, with the pre-RoPE scaling s folded into the key
 * projection weights offline, as the paired Q/K scaling allows).
 *   k_pre_bf16 : [n_new, num_kv_heads, 128] bf16 keys before RoPE.
 *   rope_table : fp32 [rope_positions, 64, 2], (cos, sin) of p * theta^(-2i/128)
 *                for position p and pair i (nvfp4_rope_table writes one);
 *                16-B aligned; rope_positions >= cache->capacity, else SHAPE.
 * RoPE pairs channel i with i + 64 (rotate-half form) and is evaluated in fp32
 * as y_i = x_i c_i - x_{i+64} s_i, y_{i+64} = x_i s_i + x_{i+64} c_i, each
 * product and sum rounded to nearest even (no fused multiply-add).  Other
 * arguments, errors and device-side checks as kv_append_nvfp4.
 */
nvfp4_status kv_append_rope_nvfp4(const nvfp4_kv_cache* cache, const void* k_pre_bf16, const void* v_bf16,
                                  const int32_t* seq_idx, const int32_t* pos, int64_t n_new,
                                  const float* rope_table, int64_t rope_positions, const float* k_shift,
                                  void* stream);

/*
 * RoPE (cos, sin) table for kv_append_rope_nvfp4: table[p][i] = (cos, sin) of
 * p * theta^(-2i/head_dim), p < n_pos, i < head_dim/2 (Sec. 2.1 RoPE; the
 * evaluated models use theta = 1e6).  The angle and both functions are
 * evaluated in fp64 and rounded once to fp32.  table: fp32 [n_pos,
 * head_dim/2, 2], 8-B aligned.  Errors: head_dim odd or <= 0, n_pos < 0 ->
 * SHAPE; theta <= 1 or not finite, table NULL with n_pos > 0 -> INVALID_ARG.
 */
nvfp4_status nvfp4_rope_table(float* table, int64_t n_pos, int32_t head_dim, float theta, void* stream);

/*
 * a5. Decode attention straight from the NVFP4 cache (Sec. 2.1):
 *   out[b, h] = softmax(softmax_scale * q[b,h] . K_hat[b,kv,t]) V_hat[b,kv,t],
 *   t < seq_lens[b], kv = h / (num_q_heads / num_kv_heads) (contiguous
 *   grouped-query replication, as in Algorithm 1's Replicate step).
 * Softmax in fp32; K/V are dequantized in registers and multiplied on the
 * tensor cores.  Split-KV partials go to `workspace`, then a combine kernel
 * writes out.
 *   q_bf16   : [batch, num_q_heads, head_dim] bf16.
 *   out_bf16 : [batch, num_q_heads, head_dim] bf16.
 *   workspace: at least decode_attention_nvfp4_workspace_size(...) bytes, 16-B
 *              aligned; contents on entry are ignored.
 * num_q_heads % num_kv_heads == 0, num_q_heads/num_kv_heads <= 8 and an even
 * capacity (scale rows are streamed in 16-byte units) are required (SHAPE);
 * the four cache arrays must be 16-B aligned (ALIGN).
 * A sequence with seq_lens[b] == 0 gets zeros; seq_lens[b] > capacity sets
 * CAPACITY on the device and is clamped to capacity.
 */
size_t decode_attention_nvfp4_workspace_size(int32_t batch, int32_t num_q_heads, int32_t capacity);
nvfp4_status decode_attention_nvfp4(const nvfp4_kv_cache* cache, const void* q_bf16,
                                    int32_t num_q_heads, float softmax_scale, void* out_bf16,
                                    void* workspace, size_t workspace_bytes, void* stream);

/*
 * Decode attention whose output is written as the output projection's NVFP4
 * A operand (every linear of the layer, the o projection included, runs
 * W4A4: Appendix D.1).  The same attention as decode_attention_nvfp4; its
 * bf16 output o, viewed as the [batch, num_q_heads * 128] matrix, is then
 * quantized with the static tensor scale g_out by the recipe of
 * nvfp4_quantize (MMA scale layout).  codes and scales are bit-identical to
 * decode_attention_nvfp4 followed by nvfp4_quantize(o, g_out, MMA layout);
 * the bf16 o itself is never stored.
 *   g_out      : device float, static scale of o (e.g. calibrated).
 *   out_codes  : [batch, num_q_heads * 64] bytes, 16-B aligned.
 *   out_scales : nvfp4_scales_bytes(batch, num_q_heads * 128, NVFP4_SCALES_MMA)
 *                bytes, 4-B aligned; padding rows are written as zeros.
 *   workspace, errors: as decode_attention_nvfp4.  g_out <= 0 or non-finite:
 *   zero codes and scales, INVALID_ARG set on the device.
 */
nvfp4_status decode_attention_nvfp4_quantize(const nvfp4_kv_cache* cache, const void* q_bf16,
                                             int32_t num_q_heads, float softmax_scale, const float* g_out,
                                             uint8_t* out_codes, uint8_t* out_scales, void* workspace,
                                             size_t workspace_bytes, void* stream);

/*
 * Decode attention without a caller workspace (no counterpart in the paper).
 *
 * Same computation and arguments as decode_attention_nvfp4, but the split-KV
 * partials go to a scratch array that the library itself holds in device
 * memory, so the call allocates nothing and needs no workspace pointer.  It is
 * for callers that cannot obtain device memory at the point of the call: a
 * runtime that reserves all GPU memory at start-up and forbids later
 * allocations, a plug-in that is handed device pointers by a host framework
 * that owns the allocator, or a code path where an allocation would
 * synchronize the device or break a latency budget.
 *
 * Limits and sharing:
 *   - The scratch holds NVFP4_ATTN_STATIC_SCRATCH_BYTES (24 MiB); a problem
 *     whose decode_attention_nvfp4_workspace_size exceeds it returns SHAPE
 *     without launching anything.  Every GPU that loads the library keeps
 *     this array until the process exits.
 *   - All calls share the one array and it keeps the last call's contents;
 *     every value a call reads is written earlier in the same call, so no
 *     clearing is needed.  Calls that can overlap on the GPU (different
 *     streams, or concurrent host threads) race on the scratch and must be
 *     serialized by the caller.
 *   - The first call on a device looks up the device address of the array
 *     (a one-time host-side query); make that first call before capturing
 *     stream work into a CUDA graph.
 *   - The looked-up address is kept per device ordinal until the process
 *     exits.  Resetting the device (cudaDeviceReset) after the first call is
 *     not supported: the kept address, like that of the device status word,
 *     would then point into a freed context.
 * Errors: as decode_attention_nvfp4.
 */
#define NVFP4_ATTN_STATIC_SCRATCH_BYTES (24u << 20)
nvfp4_status decode_attention_nvfp4_static_scratch(const nvfp4_kv_cache* cache, const void* q_bf16,
                                                   int32_t num_q_heads, float softmax_scale, void* out_bf16,
                                                   void* stream);

/*
 * f4. Q-FIT calibration (Algorithm 1; Eq. 2): choose the paired pre-RoPE
 * scale S (S_Q for the query heads, S_K for the KV heads, equal on each RoPE
 * pair) and the post-RoPE key shift m by a grid search over (alpha_s,
 * alpha_m) = (a / grid_s, b / grid_m): S = S0^alpha_s with S0[h, r] =
 * max(max_t |K_pre[t,h,r]|, max_t |K_pre[t,h,r+64]|, eps); m = alpha_m * mu
 * with mu the mean over tokens of RoPE(K_pre).  A grid point's error is the
 * mean squared difference between the unquantized attention and the
 * attention over the KV4 cache of Q_KV4(RoPE(bf16(K_pre / S_K)) - m) and
 * Q_KV4(V) (static scales amax / (qmax * 448); kv_format as the cache's),
 * with queries bf16(RoPE(Q_pre * S_Q)).  The calibration set is `batch`
 * sequences of `tokens` tokens at positions 0..tokens-1; the causal
 * attention is scored at the last token of each sequence, which attends to
 * its whole sequence.  The KV4 side runs kv_append_rope_nvfp4 and
 * decode_attention_nvfp4.  The first grid point (alpha_s-major) with the
 * least error wins.
 *   q_pre_bf16 : [batch, tokens, num_q_heads, 128] bf16 (pre-RoPE queries).
 *   k_pre_bf16, v_bf16 : [batch, tokens, num_kv_heads, 128] bf16.
 *   rope_table : nvfp4_rope_table output with rope_positions >= tokens
 *                rounded up to even, 16-B aligned.
 *   s_q [num_q_heads, 128], s_k [num_kv_heads, 128], m [num_kv_heads, 128]:
 *                fp32 device outputs (S_Q, S_K, m of the chosen point).
 *   errors_host: NULL or host fp64 [grid_s, grid_m], every point's error.
 *   workspace  : nvfp4_qfit_workspace_size(...) bytes, 256-B aligned.
 * Offline: the call synchronizes `stream` once per grid point (the key scale
 * of a point is a host argument of the cache).  1 <= grid_s, grid_m <= 64,
 * tokens <= 8192, head_dim == 128, num_q_heads % num_kv_heads == 0 with a
 * group of at most 8 (SHAPE otherwise); eps > 0 and finite (INVALID_ARG).
 * Device-side errors of the append and the attention set the status word.
 */
size_t nvfp4_qfit_workspace_size(int32_t batch, int32_t tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                 int32_t grid_s, int32_t grid_m);
nvfp4_status nvfp4_qfit_calibrate(const void* q_pre_bf16, const void* k_pre_bf16, const void* v_bf16, int32_t batch,
                                  int32_t tokens, int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                  const float* rope_table, int64_t rope_positions, int32_t grid_s, int32_t grid_m,
                                  double eps, int32_t kv_format, float* s_q, float* s_k, float* m,
                                  double* errors_host, void* workspace, size_t workspace_bytes, void* stream);

/* Synchronize `stream`, copy the device status word of the current device to
 * *status_host (an nvfp4_status value) and clear it. */
nvfp4_status nvfp4_get_device_status(int32_t* status_host, void* stream);

/*
 * Test-only fault injection for the failure-detection tests: arms one fault
 * for the next call of the kind it names, then disarms itself.
 *   NVFP4_FAULT_ATTN_SKIP_STAGE: in the next decode-attention launch, CTA 0's
 *     producer leaves its first ring stage neither armed nor loaded, so the
 *     consumers' bounded wait on it runs out after ~2 s: the call reports
 *     NVFP4_ERR_TIMEOUT through nvfp4_get_device_status, its output is
 *     undefined, and the device stays usable.
 *   NVFP4_FAULT_GEMM_SKIP_STAGE: in the next launch of a CTA-pair GEMM kernel
 *     (the 256 x 256 tiles that nvfp4_linear / mxfp4_linear use when N % 256
 *     == 0, with or without a split of K across a cluster, and the fused
 *     SwiGLU calls), both CTAs of the first pair leave their first ring stage
 *     of their K range neither armed nor loaded; the MMA
 *     issuer's and the scale copiers' bounded waits run out after ~2 s, every
 *     role of the pair stops, the MMAs issued so far drain and TMEM is freed.
 *     The call reports NVFP4_ERR_TIMEOUT, its output is undefined, and the
 *     device stays usable.
 *   NVFP4_FAULT_NONE disarms.  Other values -> INVALID_ARG.
 */
#define NVFP4_FAULT_NONE 0
#define NVFP4_FAULT_ATTN_SKIP_STAGE 1
#define NVFP4_FAULT_GEMM_SKIP_STAGE 2
nvfp4_status nvfp4_debug_inject_fault(int what);

/* Static, human-readable name of a status. */
const char* nvfp4_status_string(nvfp4_status s);

/* Number of kernels this library has launched in this process (host counter). */
uint64_t nvfp4_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* NVFP4_H */
