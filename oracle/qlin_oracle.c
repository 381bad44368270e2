/*
 * qlin CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct restatement of what the quantized linear
 * layer computes, written from the format definitions that the paper's
 * quantization recipe relies on (Sec. 4, paragraph "Quantization": FP8 and
 * NVFP4 post-training quantization of the denoising transformer's linears;
 * FP8 E4M3 as defined by Micikevicius et al. 2022 and NVFP4 as introduced by
 * NVIDIA 2025, both cited there).  The paper itself fixes no block size,
 * scale formula or rounding rule; every reading taken where it is silent is
 * marked READING below and listed in the design notes.
 *
 * Only tests/, the smoke check and the CPU-baseline leg of the benchmark may
 * load this library.  It shares no code, header or table with the CUDA
 * library; the product path never calls it.
 *
 * Arithmetic conventions:
 *  - "fp32 operation" means the exact result rounded once to binary32.  It is
 *    written as a binary64 operation on binary32 inputs followed by one
 *    conversion: for +, -, *, / this equals the correctly rounded binary32
 *    result because 53 >= 2*24 + 2.
 *  - Element codes are found from the grid definition itself (nearest
 *    representable value, ties to the even code, saturation to the largest
 *    finite magnitude), never from hardware conversions.
 *  - Build with -O2 -ffp-contract=off and no fast-math.
 *
 * Parity status: every function here is pinned by tests/test_oracle_*.py
 * (exhaustive code round trips, an independent library's rounding, hand-worked
 * blocks from tests/golden/, closed forms and brute-force tiny matmuls).
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ */
/* helpers                                                             */
/* ------------------------------------------------------------------ */

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void oracle_set_num_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* Round half to even on an fp64 value (exact: q is a short dyadic here). */
static double round_half_even(double q) {
  double f = floor(q);
  double r = q - f;
  if (r > 0.5) return f + 1.0;
  if (r < 0.5) return f;
  return (fmod(f, 2.0) == 0.0) ? f : f + 1.0;
}

static float f32_mul(float a, float b) { return (float)((double)a * (double)b); }
static float f32_div(float a, float b) { return (float)((double)a / (double)b); }

/* bf16 is the upper half of a binary32: widening is exact. */
float oracle_bf16_to_f32(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return f;
}

/* Nearest bf16 (8-bit significand, binary32 exponent range) to an fp64
 * value, ties to even; used to state the expected bf16 output of the linear
 * (the layer writes bf16).  Finite inputs; overflow gives +-inf. */
uint16_t oracle_round_bf16(double v) {
  uint16_t sign = signbit(v) ? 0x8000 : 0;
  double a = fabs(v);
  if (a == 0.0) return sign;
  int e2;
  frexp(a, &e2);               /* a in [2^(e2-1), 2^e2) */
  int E = e2 - 1;
  if (E < -126) E = -126;      /* subnormal range: fixed step 2^-133 */
  double q = round_half_even(ldexp(a, 7 - E));   /* significand in units of 2^(E-7) */
  if (q >= 256.0) { q /= 2.0; E += 1; }          /* carried into the next binade */
  if (E > 127) return sign | 0x7F80;
  uint32_t mant = (uint32_t)q;                   /* 128..255 normal, < 128 subnormal */
  uint32_t bits = (mant >= 128) ? ((uint32_t)(E + 127) << 7) | (mant - 128) : mant;
  return sign | (uint16_t)bits;
}

/* ------------------------------------------------------------------ */
/* e2m1 (FP4) -- the element type of NVFP4 (NVIDIA 2025, cited in Sec. 4)  */
/* code bits: s | e1 e0 | m, exponent bias 1, no inf/NaN.              */
/* ------------------------------------------------------------------ */

double oracle_e2m1_decode(int code) {
  int s = (code >> 3) & 1, e = (code >> 1) & 3, m = code & 1;
  double mag = (e == 0) ? 0.5 * m : ldexp(1.0 + 0.5 * m, e - 1);
  return s ? -mag : mag;
}

/* Nearest of the 8 magnitudes, ties to the even code, saturating at 6.
 * The sign bit is kept, so a negative value that rounds to zero gives 0x8
 * (READING: signed zero is preserved). */
int oracle_e2m1_encode(double v) {
  int s = signbit(v) ? 8 : 0;
  double a = fabs(v);
  if (a >= 6.0) return s | 7;
  int best = 0;
  double bestd = INFINITY;
  for (int c = 0; c < 8; ++c) {
    double d = fabs(a - oracle_e2m1_decode(c));
    if (d < bestd || (d == bestd && (c & 1) == 0)) {
      best = c;
      bestd = d;
    }
  }
  return s | best;
}

/* ------------------------------------------------------------------ */
/* E4M3 ("fn" variant) -- Micikevicius et al. 2022, cited in Sec. 4     */
/* bias 7, max normal 448, min normal 2^-6, subnormal step 2^-9,       */
/* NaN = S.1111.111, no infinities.                                    */
/* ------------------------------------------------------------------ */

double oracle_e4m3_decode(int code) {
  int s = (code >> 7) & 1, e = (code >> 3) & 15, m = code & 7;
  if (e == 15 && m == 7) return NAN;
  double mag = (e == 0) ? ldexp((double)m, -9) : ldexp((double)(8 + m), e - 10);
  return s ? -mag : mag;
}

/* Round to nearest, ties to even mantissa, saturating to +-448
 * (READING: saturate-to-finite, as the scale and element encoders need a
 * finite result; NaN maps to NaN). */
int oracle_e4m3_encode(double v) {
  if (isnan(v)) return signbit(v) ? 0xFF : 0x7F;
  int s = signbit(v) ? 0x80 : 0;
  double a = fabs(v);
  if (a >= 448.0) return s | 0x7E;
  if (a < ldexp(1.0, -6)) {
    /* subnormal range: value = m * 2^-9; m == 8 is the min normal 0x08 */
    double m = round_half_even(a * 512.0);
    return s | (int)m;
  }
  int e2;
  frexp(a, &e2);      /* a = f * 2^e2, f in [0.5, 1) */
  int E = e2 - 1;     /* floor(log2 a) */
  double m = round_half_even((ldexp(a, -E) - 1.0) * 8.0);
  if (m == 8.0) {
    m = 0.0;
    E += 1;
  }
  return s | ((E + 7) << 3) | (int)m;
}

/* ------------------------------------------------------------------ */
/* Tensor scales (Sec. 4 "Quantization": FP8 with a per-tensor scale,   */
/* NVFP4 with an FP32 tensor scale over E4M3 block scales).            */
/* READING: S_dec = amax / (6*448) for NVFP4, amax / 448 for FP8;       */
/* S_dec = 1 when amax == 0; S_enc = 1/S_dec, +inf replaced by FLT_MAX. */
/* ------------------------------------------------------------------ */

float oracle_amax_bf16(const uint16_t *x, int64_t n) {
  float amax = 0.0f;
  for (int64_t i = 0; i < n; ++i) {
    float a = fabsf(oracle_bf16_to_f32(x[i]));
    if (a > amax) amax = a;
  }
  return amax;
}

float oracle_nvfp4_tensor_scale(float amax) {
  return (amax == 0.0f) ? 1.0f : f32_div(amax, 2688.0f);
}

float oracle_fp8_tensor_scale(float amax) {
  return (amax == 0.0f) ? 1.0f : f32_div(amax, 448.0f);
}

float oracle_encode_scale(float s_dec) {
  float s_enc = f32_div(1.0f, s_dec);
  if (isinf(s_enc)) s_enc = FLT_MAX;
  return s_enc;
}

/* ------------------------------------------------------------------ */
/* NVFP4 quantization of a row-major bf16 [rows, K] matrix.            */
/* Blocks are 16 consecutive elements of one row along K.              */
/*   amax_b = max |x_i|                                                */
/*   s_b    = E4M3( (amax_b * S_enc) / 6 )          (block scale)       */
/*   r_b    = s_b == 0 ? 0 : S_enc / s_b                               */
/*   code_i = e2m1( x_i * r_b )                                        */
/* READING: this op order (one divide per block, one multiply per       */
/* element).  Codes: byte j of a row holds element 2j in the low       */
/* nibble and element 2j+1 in the high nibble.  scales_canon is the    */
/* row-major [rows, K/16] byte array of block scales.                  */
/* ------------------------------------------------------------------ */

void oracle_quant_nvfp4(const uint16_t *x, int64_t rows, int64_t K, float s_dec,
                        uint8_t *codes, uint8_t *scales_canon) {
  const float s_enc = oracle_encode_scale(s_dec);
  const int64_t nb = K / 16;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    const uint16_t *xr = x + r * K;
    for (int64_t b = 0; b < nb; ++b) {
      float amax_b = 0.0f;
      for (int i = 0; i < 16; ++i) {
        float a = fabsf(oracle_bf16_to_f32(xr[b * 16 + i]));
        if (a > amax_b) amax_b = a;
      }
      float t = f32_mul(amax_b, s_enc);
      int sb = oracle_e4m3_encode((double)f32_div(t, 6.0f));
      float sbf = (float)oracle_e4m3_decode(sb);
      float rb = (sb == 0) ? 0.0f : f32_div(s_enc, sbf);
      scales_canon[r * nb + b] = (uint8_t)sb;
      for (int i = 0; i < 16; i += 2) {
        float v0 = f32_mul(oracle_bf16_to_f32(xr[b * 16 + i]), rb);
        float v1 = f32_mul(oracle_bf16_to_f32(xr[b * 16 + i + 1]), rb);
        int c0 = oracle_e2m1_encode((double)v0);
        int c1 = oracle_e2m1_encode((double)v1);
        codes[r * (K / 2) + (b * 16 + i) / 2] = (uint8_t)(c0 | (c1 << 4));
      }
    }
  }
}

/* FP8 quantization with one tensor scale: code = E4M3(x * S_enc). */
void oracle_quant_fp8(const uint16_t *x, int64_t rows, int64_t K, float s_dec,
                      uint8_t *codes) {
  const float s_enc = oracle_encode_scale(s_dec);
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k)
      codes[r * K + k] = (uint8_t)oracle_e4m3_encode(
          (double)f32_mul(oracle_bf16_to_f32(x[r * K + k]), s_enc));
}

/* FP8 weights with one scale per output channel (row n):
 * s_n = amax_n / 448 (1 when the row is all zero), code = E4M3(w * 1/s_n). */
void oracle_quant_fp8_rows(const uint16_t *w, int64_t rows, int64_t K,
                           uint8_t *codes, float *s_dec_rows) {
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    float s_dec = oracle_fp8_tensor_scale(oracle_amax_bf16(w + r * K, K));
    float s_enc = oracle_encode_scale(s_dec);
    s_dec_rows[r] = s_dec;
    for (int64_t k = 0; k < K; ++k)
      codes[r * K + k] = (uint8_t)oracle_e4m3_encode(
          (double)f32_mul(oracle_bf16_to_f32(w[r * K + k]), s_enc));
  }
}

/* ------------------------------------------------------------------ */
/* Block-scale layout for the tensor-core operand: 128-row x 4-scale   */
/* atoms of 512 bytes.  Atom (i, j) covers rows 128i..128i+127 and      */
/* scale columns 4j..4j+3; inside it row r, column c sits at byte       */
/* (r % 32) * 16 + (r / 32) * 4 + c.  Atoms are ordered i-major.        */
/* Rows are padded to a multiple of 128 with zero scales.              */
/* ------------------------------------------------------------------ */

int64_t oracle_swizzled_scale_bytes(int64_t rows, int64_t K) {
  return ((rows + 127) / 128) * (K / 64) * 512;
}

int64_t oracle_swizzle_offset(int64_t r, int64_t c, int64_t K) {
  int64_t i = r / 128, rr = r % 128, j = c / 4, cc = c % 4;
  return (i * (K / 64) + j) * 512 + (rr % 32) * 16 + (rr / 32) * 4 + cc;
}

void oracle_swizzle_scales(const uint8_t *canon, int64_t rows, int64_t K,
                           uint8_t *swz) {
  memset(swz, 0, (size_t)oracle_swizzled_scale_bytes(rows, K));
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t c = 0; c < K / 16; ++c)
      swz[oracle_swizzle_offset(r, c, K)] = canon[r * (K / 16) + c];
}

void oracle_unswizzle_scales(const uint8_t *swz, int64_t rows, int64_t K,
                             uint8_t *canon) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t c = 0; c < K / 16; ++c)
      canon[r * (K / 16) + c] = swz[oracle_swizzle_offset(r, c, K)];
}

/* ------------------------------------------------------------------ */
/* Dequantization to fp64 (values are exact in fp64).                   */
/* sel: list of row indices to decode (NULL = all rows, nsel = rows).   */
/* ------------------------------------------------------------------ */

void oracle_dequant_nvfp4(const uint8_t *codes, const uint8_t *scales_canon,
                          float s_dec, int64_t rows, int64_t K,
                          const int64_t *sel, int64_t nsel, double *out) {
  (void)rows;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < nsel; ++t) {
    int64_t r = sel ? sel[t] : t;
    for (int64_t k = 0; k < K; ++k) {
      int byte = codes[r * (K / 2) + k / 2];
      int code = (k % 2 == 0) ? (byte & 15) : (byte >> 4);
      double sb = oracle_e4m3_decode(scales_canon[r * (K / 16) + k / 16]);
      out[t * K + k] = oracle_e2m1_decode(code) * sb * (double)s_dec;
    }
  }
}

/* s_dec has one entry (per_row == 0) or one per row (per_row != 0). */
void oracle_dequant_fp8(const uint8_t *codes, const float *s_dec, int per_row,
                        int64_t rows, int64_t K, const int64_t *sel,
                        int64_t nsel, double *out) {
  (void)rows;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < nsel; ++t) {
    int64_t r = sel ? sel[t] : t;
    double s = (double)(per_row ? s_dec[r] : s_dec[0]);
    for (int64_t k = 0; k < K; ++k)
      out[t * K + k] = oracle_e4m3_decode(codes[r * K + k]) * s;
  }
}

/* ------------------------------------------------------------------ */
/* The linear layer's exact result: y[m, n] = sum_k a[m, k] * w[n, k]   */
/* in fp64 over dequantized, scaled operands (y = x W^T, nn.Linear      */
/* layout).  Also returns ||a_m||_2 and ||w_n||_2, the normaliser of    */
/* the GEMM tolerance.                                                 */
/* ------------------------------------------------------------------ */

void oracle_gemm_f64(const double *a, const double *w, int64_t M, int64_t N,
                     int64_t K, double *y, double *norm_a, double *norm_w) {
#pragma omp parallel for schedule(static)
  for (int64_t m = 0; m < M; ++m) {
    const double *am = a + m * K;
    for (int64_t n = 0; n < N; ++n) {
      const double *wn = w + n * K;
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k) acc += am[k] * wn[k];
      y[m * N + n] = acc;
    }
  }
  if (norm_a)
    for (int64_t m = 0; m < M; ++m) {
      double s = 0.0;
      for (int64_t k = 0; k < K; ++k) s += a[m * K + k] * a[m * K + k];
      norm_a[m] = sqrt(s);
    }
  if (norm_w)
    for (int64_t n = 0; n < N; ++n) {
      double s = 0.0;
      for (int64_t k = 0; k < K; ++k) s += w[n * K + k] * w[n * K + k];
      norm_w[n] = sqrt(s);
    }
}

void oracle_round_bf16_array(const double *v, int64_t n, uint16_t *out) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) out[i] = oracle_round_bf16(v[i]);
}
