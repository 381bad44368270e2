/*
 * qlin -- FP8 / NVFP4 quantized linear layer for NVIDIA GB300 (sm_103a).
 *
 * The paper (Sec. 4, paragraph "Quantization") speeds up the denoising
 * transformer with post-training quantization: weights are quantized once,
 * offline (a smaller memory footprint), and activations are quantized at run
 * time so the linear layers run on the FP8 / NVFP4 tensor cores (less compute
 * time).  This C ABI follows that split:
 *
 *   qlin_quantize_weight       offline weight quantization (NVFP4 or FP8)
 *   qlin_quantize_act_nvfp4    run-time activation quantization to NVFP4
 *   qlin_quantize_act_fp8      run-time activation quantization to FP8
 *   qlin_gemm_nvfp4 / _fp8     block-scaled GEMM, fp32 accumulation, bf16 out
 *   qlin_linear_fused          NVFP4 GEMM whose epilogue also re-quantizes the
 *                              bf16 output to NVFP4 for the next layer
 *
 * Formats (the paper names them and cites their definitions; it fixes no block
 * size or rounding rule, so the readings taken here are stated per call):
 *   - E4M3: FP8 with exponent bias 7, max 448, NaN = S.1111.111, no infinity
 *     (Micikevicius et al. 2022, cited in Sec. 4).
 *   - NVFP4: e2m1 elements (+-{0, .5, 1, 1.5, 2, 3, 4, 6}), one unsigned E4M3
 *     scale per 16 consecutive elements along K, one FP32 tensor scale
 *     (NVIDIA 2025, cited in Sec. 4).
 *   - All conversions round to nearest, ties to even, and saturate to the
 *     largest finite value.
 *
 * Conventions for every call:
 *   - All data pointers are DEVICE pointers owned by the caller.  The library
 *     allocates no memory during a call.  Output buffers are written, never
 *     freed or resized.
 *   - Matrices are row-major.  Activations x are [M, K] (K contiguous);
 *     weights W are [N, K] (the nn.Linear layout), and y = x W^T is [M, N].
 *   - bf16 data is passed as raw 16-bit patterns (void*).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Every call is asynchronous and stream-ordered.
 *   - Argument errors are detected on the host before anything is launched
 *     and returned synchronously; nothing is written in that case.
 *     Device-side failures (a bounded wait that expired) are recorded in a
 *     device status word that qlin_sync_status() returns and clears.
 *   - Shapes: K must be a positive multiple of 64; N a positive multiple of
 *     64; M >= 1 (any value: partial tiles are masked).
 *   - Alignment: every code, scale and bf16 buffer 16-byte aligned; fp32
 *     scalars 4-byte aligned.
 */
#ifndef QLIN_H
#define QLIN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  QLIN_OK = 0,
  QLIN_ERR_INVALID_ARG = 1, /* null pointer, bad shape or inconsistent sizes */
  QLIN_ERR_UNSUPPORTED = 2, /* format, shape or device this build does not handle */
  QLIN_ERR_MISALIGNED = 3,  /* a pointer violates the alignment rule above */
  QLIN_ERR_CUDA = 4,        /* a CUDA runtime/driver call failed */
  QLIN_ERR_TIMEOUT = 5,     /* a device-side bounded wait expired */
  QLIN_ERR_WORKSPACE = 6    /* workspace missing or smaller than required */
} qlin_status;

typedef enum { QLIN_FMT_NVFP4 = 1, QLIN_FMT_FP8 = 2 } qlin_format;

/*
 * NVFP4 operand [rows, K].
 *  codes:  rows x K/2 bytes, row stride K/2; byte j of a row holds element 2j
 *          in its low nibble and element 2j+1 in its high nibble.
 *  scales: the E4M3 block scales in the tensor-core layout: 128-row x
 *          4-scale atoms of 512 bytes, atom (i, j) covering rows 128i..128i+127
 *          and scale columns 4j..4j+3 (elements 64j..64j+63), atoms ordered
 *          i-major; inside an atom, row r / scale column c sits at byte
 *          (r % 32) * 16 + (r / 32) * 4 + c.  Size: qlin_nvfp4_scale_bytes().
 *          Bytes of padding rows (rows..ceil(rows/128)*128-1) are don't-care.
 *  tensor_scale: one fp32 decode scale S_dec, x ~= e2m1 * e4m3 * S_dec.
 */
typedef struct {
  uint8_t *codes;
  uint8_t *scales;
  float *tensor_scale;
  int64_t rows;
  int64_t K;
} qlin_nvfp4_t;

/*
 * FP8 (E4M3) operand [rows, K].
 *  codes: rows x K bytes, row stride K.
 *  scale: fp32 decode scale(s): one value (per_channel == 0, activations) or
 *         one per row (per_channel != 0, weights: one per output channel).
 */
typedef struct {
  uint8_t *codes;
  float *scale;
  int64_t rows;
  int64_t K;
  int32_t per_channel;
} qlin_fp8_t;

/* Bytes of the swizzled NVFP4 scale array for a [rows, K] operand:
 * ceil(rows / 128) * (K / 64) * 512.  Returns 0 for invalid shapes. */
size_t qlin_nvfp4_scale_bytes(int64_t rows, int64_t K);

/* Workspace bytes the dynamic-scale quantizers need (a device amax word);
 * the same for every shape.  Returns 256. */
size_t qlin_workspace_size(int64_t M, int64_t K);

/*
 * Run-time NVFP4 activation quantization (Sec. 4, "Quantization": activation
 * quantization so the layer runs on the NVFP4 tensor cores).
 *  x:            bf16 [M, K], 16-byte aligned.
 *  static_scale: device fp32 S_dec from calibration (post-training
 *                quantization, Sec. 4); NULL selects the dynamic tensor
 *                scale S_dec = amax(|x|) / (6 * 448) (1 if amax == 0), which
 *                first runs an amax pass over x.
 *  out:          rows == M, K == K; codes, scales and tensor_scale are written
 *                (tensor_scale receives S_dec in both modes).
 *  workspace:    device memory of >= qlin_workspace_size() bytes, 8-byte
 *                aligned, zero-filled before its first use; every call leaves
 *                it zero-filled again (its words carry a grid-wide amax and
 *                arrival counts inside one call).  Used only in dynamic mode,
 *                may be NULL in static mode.  Calls whose work overlaps on
 *                the GPU must not share one workspace.
 * Per 16-element block b (READING of the op order, each fp32 op rounded once):
 *   S_enc = 1 / S_dec (FLT_MAX if that overflows);
 *   s_b = E4M3((amax_b * S_enc) / 6);  r_b = s_b == 0 ? 0 : S_enc / s_b;
 *   code_i = e2m1(x_i * r_b).
 * Errors: INVALID_ARG (null/shape), MISALIGNED, WORKSPACE, CUDA.
 */
qlin_status qlin_quantize_act_nvfp4(const void *x_bf16, int64_t M, int64_t K,
                                    const float *static_scale, qlin_nvfp4_t *out,
                                    void *workspace, size_t ws_bytes, void *stream);

/*
 * Run-time FP8 activation quantization with one tensor scale (Sec. 4).
 *  static_scale: device S_dec, or NULL for the dynamic S_dec = amax / 448.
 *  out:          per_channel must be 0; codes [M, K] and scale[0] = S_dec.
 *  code = E4M3(x * S_enc), S_enc = 1 / S_dec.
 *  Workspace as for qlin_quantize_act_nvfp4.
 */
qlin_status qlin_quantize_act_fp8(const void *x_bf16, int64_t M, int64_t K,
                                  const float *static_scale, qlin_fp8_t *out,
                                  void *workspace, size_t ws_bytes, void *stream);

/*
 * Offline weight quantization (Sec. 4: "lowering weight precision reduces
 * VRAM"; post-training, applied once to a checkpoint).
 *  w:      bf16 [N, K].
 *  fmt:    QLIN_FMT_NVFP4 -> out_desc is a qlin_nvfp4_t* (rows N), quantized
 *          exactly as an activation with its own dynamic tensor scale;
 *          QLIN_FMT_FP8   -> out_desc is a qlin_fp8_t* with per_channel != 0:
 *          scale[n] = amax(|w_n|) / 448 (1 for an all-zero row) and
 *          code = E4M3(w * (1 / scale[n])).
 *  workspace: as for the activation quantizers (needed for NVFP4).
 */
qlin_status qlin_quantize_weight(const void *w_bf16, int64_t N, int64_t K,
                                 qlin_format fmt, void *out_desc, void *workspace,
                                 size_t ws_bytes, void *stream);

/*
 * NVFP4 x NVFP4 GEMM on the tensor cores (Sec. 4: NVFP4 tensor cores cut
 * compute time; Table 2's NVFP4 row).
 *  y[m, n] = bf16( alpha * sum_k e2m1(a)*e4m3(sa) * e2m1(w)*e4m3(sw) ),
 *  alpha = S_dec,A * S_dec,W (fp32), fp32 accumulation, bf16 round-to-nearest-
 *  even output [M, N] (row stride N).  A->K == W->K.
 */
qlin_status qlin_gemm_nvfp4(const qlin_nvfp4_t *A, const qlin_nvfp4_t *W,
                            void *y_bf16, void *stream);

/*
 * FP8 x FP8 GEMM (Sec. 4: FP8 tensor cores; Table 2's FP8 row).
 *  A: per_channel == 0; W: per_channel != 0 (scale per output channel) or 0.
 *  y[m, n] = bf16( (S_A * S_W[n]) * sum_k e4m3(a) * e4m3(w) ).
 */
qlin_status qlin_gemm_fp8(const qlin_fp8_t *A, const qlin_fp8_t *W, void *y_bf16,
                          void *stream);

/*
 * NVFP4 linear with a fused re-quantizing epilogue: the bf16 output is also
 * quantized to NVFP4 for the next layer, so the activation never makes an
 * extra HBM round trip (the chained linears of the denoiser, Sec. 4).
 *  y_bf16:      [M, N] output, or NULL when only the quantized output is needed.
 *  next_scale:  device fp32 S_dec of the next layer's input (a static,
 *               calibrated scale, as in post-training quantization); NULL
 *               disables the re-quantization (then y_bf16 must be non-NULL).
 *  y_q:         receives NVFP4 of y's columns [rq_col0, rq_col0 + y_q->K):
 *               rows == M, y_q->K % 64 == 0, rq_col0 % 64 == 0,
 *               rq_col0 + y_q->K <= N.  The input of the re-quantization is the
 *               bf16-rounded output, quantized as qlin_quantize_act_nvfp4 does
 *               with static_scale = next_scale; *y_q->tensor_scale receives
 *               *next_scale.
 */
qlin_status qlin_linear_fused(const qlin_nvfp4_t *A, const qlin_nvfp4_t *W,
                              void *y_bf16, const float *next_scale,
                              qlin_nvfp4_t *y_q, int64_t rq_col0, void *stream);

/* Bytes of device scratch that qlin_quantize_act_nvfp4_noalloc keeps in the
 * library's own static device array (per GPU that loads the library). */
#define QLIN_NOALLOC_SCRATCH_BYTES 256

/*
 * qlin_quantize_act_nvfp4 with the dynamic tensor scale, for callers that
 * cannot allocate device memory.  The paper has no counterpart: it is an
 * integration aid.  Some callers own no allocator of their own -- a plugin
 * running inside an inference runtime that hands out all device memory, or a
 * real-time loop that must never stall on cudaMalloc.  They can still pass x
 * and the output buffers, but not the workspace the dynamic amax pass needs.
 *
 * This entry point takes no workspace: its scratch (the amax and arrival
 * words) lives in a static device array of QLIN_NOALLOC_SCRATCH_BYTES bytes
 * that the library holds on every GPU that loads it, until the process exits.  It calls no
 * cudaMalloc, cudaFree or other allocating routine.
 *  - x, M, K, out: as for qlin_quantize_act_nvfp4 (out->tensor_scale receives
 *    the dynamic S_dec = amax / 2688).
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture.
 *  - Every call shares the one array and clears the part it uses before use.
 *    Calls whose work overlaps on the GPU (different streams, no ordering)
 *    race on it: order them on one stream or serialise them.
 *  - Returns QLIN_ERR_WORKSPACE if the scratch a shape needs
 *    (qlin_workspace_size(M, K)) exceeds QLIN_NOALLOC_SCRATCH_BYTES; other
 *    errors as for qlin_quantize_act_nvfp4.
 */
qlin_status qlin_quantize_act_nvfp4_noalloc(const void *x_bf16, int64_t M, int64_t K,
                                            qlin_nvfp4_t *out, void *stream);

/*
 * FP8 linear with the next layer's FP8 input written by the epilogue (Sec. 4:
 * W8A8 layers in a chain, post-training static activation scale): as
 * qlin_gemm_fp8, and columns [rq_col0, rq_col0 + y_q->K) of bf16(y) are
 * quantized to E4M3 with the static S_dec *next_scale:
 *   code = E4M3_rn_sat(bf16(y) * S_enc), S_enc = 1 / S_dec (FLT_MAX if that
 *   overflows) -- the FP8 activation quantizer's arithmetic.
 *  y_bf16:     may be NULL (only the quantized output is written).
 *  next_scale: device fp32 S_dec, required.
 *  y_q:        per-tensor FP8 operand, rows == A->rows, K % 64 == 0; its
 *              scale receives S_dec.  rq_col0 % 64 == 0.
 * Errors: INVALID_ARG, MISALIGNED, UNSUPPORTED, CUDA.
 */
qlin_status qlin_linear_fused_fp8(const qlin_fp8_t *A, const qlin_fp8_t *W, void *y_bf16,
                                  const float *next_scale, qlin_fp8_t *y_q, int64_t rq_col0,
                                  void *stream);

/*
 * Unquantized bf16 linear on the same tensor-core skeleton (tcgen05
 * kind::f16), the reference precision of Table 2 (BF16 / FP8 / NVFP4 step
 * latencies): y = a w^T, fp32 accumulation, bf16 out.
 *  a_bf16: bf16 [M, K] with row stride lda (elements, lda >= K, lda * 2 a
 *          multiple of 16), 16-byte aligned.  A strided view serves, e.g. the
 *          value columns of a QKV output.
 *  w_bf16: bf16 [N, K] row-major; y_bf16: bf16 [M, N].
 *  K % 64 == 0, N % 64 == 0.
 * Errors: INVALID_ARG, MISALIGNED, UNSUPPORTED, CUDA.
 */
qlin_status qlin_gemm_bf16(const void *a_bf16, int64_t lda, const void *w_bf16, int64_t M,
                           int64_t N, int64_t K, void *y_bf16, void *stream);

/*
 * Unquantized fp16 linear: qlin_gemm_bf16 with fp16 operands and an fp16
 * output, y = fp16_rn(a w^T), fp32 accumulation (Sec. 4: the FP16 engines of
 * the precision comparison; values beyond 65504 become infinities, as in
 * any fp16 engine).  Same arguments, layouts and errors as qlin_gemm_bf16.
 */
qlin_status qlin_gemm_fp16(const void *a_fp16, int64_t lda, const void *w_fp16, int64_t M,
                           int64_t N, int64_t K, void *y_fp16, void *stream);

/*
 * Dynamic per-tensor scaling inside a chain of linears (Sec. 4, "Quantization":
 * run-time activation quantization, here with the tensor scale of the layer's
 * own output instead of a calibrated one):
 *   y = A W^T (bf16, as qlin_gemm_nvfp4), while the GEMM epilogue reduces
 *   amax(|y|) into a workspace word and the GEMM's last CTA turns it into
 *   the dynamic S_dec = amax / 2688 (1 if amax == 0), written to
 *   y_q->tensor_scale; then y_q = NVFP4(y) with that scale, exactly as
 *   qlin_quantize_act_nvfp4(y, NULL) would produce it, without its amax pass
 *   over y.  y is stored with an L2 keep hint, since the quantizer reads it
 *   right after.
 *  A, W:      NVFP4 operands as for qlin_gemm_nvfp4.
 *  y_bf16:    bf16 [A->rows, W->rows], 16-byte aligned (required: the
 *             quantizer reads it).
 *  y_q:       rows == A->rows, K == W->rows; codes, scales and tensor_scale
 *             are written.
 *  workspace: as for qlin_quantize_act_nvfp4: zero-filled before its first
 *             use, left zero-filled by every call (two of its words count
 *             within a call); calls that share one workspace must not
 *             overlap on the GPU.
 * Errors: INVALID_ARG, MISALIGNED, WORKSPACE, CUDA.
 */
qlin_status qlin_linear_dynamic(const qlin_nvfp4_t *A, const qlin_nvfp4_t *W, void *y_bf16,
                                qlin_nvfp4_t *y_q, void *workspace, size_t ws_bytes,
                                void *stream);

/*
 * Waits for `stream`, then returns and clears the device status word:
 * QLIN_ERR_TIMEOUT if a kernel's bounded wait expired since the last call,
 * QLIN_ERR_CUDA if the stream reports an error, else QLIN_OK.
 */
qlin_status qlin_sync_status(void *stream);

/*
 * Diagnostic for the bounded-wait machinery used inside the GEMM kernels:
 * launches one CTA that waits on an mbarrier phase that nothing completes,
 * with the given limit (nanoseconds, clamped to [1 us, 2 s]).  The kernel
 * gives up, records QLIN_ERR_TIMEOUT in the status word and exits normally;
 * qlin_sync_status() then returns QLIN_ERR_TIMEOUT.
 */
qlin_status qlin_selftest_bounded_wait(uint64_t timeout_ns, void *stream);

/* Wait limit used by every device-side spin (default 2 s), in ns. */
void qlin_set_wait_timeout_ns(uint64_t ns);

/* Short text for a status code (static storage). */
const char *qlin_status_str(qlin_status s);

/* Text of the last CUDA error seen by this thread's calls (static storage). */
const char *qlin_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* QLIN_H */
