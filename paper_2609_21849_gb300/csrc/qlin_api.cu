// The C ABI of libqlin (declared in include/qlin.h): argument validation on
// the host, then launches on the caller's stream.  No call allocates memory.
#include <atomic>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "qlin_internal.h"

namespace qlin {
namespace {

// Device status word: kernels record device-side failures here.
__device__ unsigned g_status_word;

constexpr int kMaxDevices = 64;
std::mutex g_dev_mutex;
unsigned* g_status_ptr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};
std::atomic<uint64_t> g_timeout_ns{2000000000ull};
thread_local char g_last_error[256] = "";

qlin_status cuda_fail(cudaError_t e) {
  std::snprintf(g_last_error, sizeof g_last_error, "%s: %s", cudaGetErrorName(e),
                cudaGetErrorString(e));
  return QLIN_ERR_CUDA;
}

// Per-device state, set up on the first call made on that device: the
// address of the status word and the SM count.
qlin_status device_state(unsigned** status, int* num_sms) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= kMaxDevices) return QLIN_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_dev_mutex);
  if (g_status_ptr[dev] == nullptr) {
    int major = 0, minor = 0, sms = 0;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_fail(e);
    if (major != 10 || minor != 3) {
      std::snprintf(g_last_error, sizeof g_last_error,
                    "libqlin is built for sm_103a; device %d is sm_%d%d", dev, major, minor);
      return QLIN_ERR_UNSUPPORTED;
    }
    void* p = nullptr;
    if ((e = cudaGetSymbolAddress(&p, g_status_word)) != cudaSuccess) return cuda_fail(e);
    g_status_ptr[dev] = static_cast<unsigned*>(p);
    g_num_sms[dev] = sms;
  }
  *status = g_status_ptr[dev];
  *num_sms = g_num_sms[dev];
  return QLIN_OK;
}

// Scratch of qlin_quantize_act_nvfp4_noalloc: a static device array, so the
// entry point needs no allocation.  Host code may only use its device address
// (looked up once per device), never the symbol itself.
static __device__ __align__(256) unsigned char g_noalloc_scratch[QLIN_NOALLOC_SCRATCH_BYTES];
unsigned char* g_noalloc_ptr[kMaxDevices] = {};

qlin_status noalloc_scratch(unsigned char** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= kMaxDevices) return QLIN_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_dev_mutex);
  if (g_noalloc_ptr[dev] == nullptr) {
    void* p = nullptr;
    if ((e = cudaGetSymbolAddress(&p, g_noalloc_scratch)) != cudaSuccess) return cuda_fail(e);
    g_noalloc_ptr[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_noalloc_ptr[dev];
  return QLIN_OK;
}

uint64_t timeout() { return g_timeout_ns.load(std::memory_order_relaxed); }

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool shape_ok(int64_t rows, int64_t K) { return rows >= 1 && K >= 64 && K % 64 == 0; }

qlin_status check_nvfp4(const qlin_nvfp4_t* t, int64_t rows, int64_t K) {
  if (t == nullptr || t->codes == nullptr || t->scales == nullptr || t->tensor_scale == nullptr)
    return QLIN_ERR_INVALID_ARG;
  if (t->rows != rows || t->K != K || !shape_ok(rows, K)) return QLIN_ERR_INVALID_ARG;
  if (!aligned(t->codes, 16) || !aligned(t->scales, 16) || !aligned(t->tensor_scale, 4))
    return QLIN_ERR_MISALIGNED;
  return QLIN_OK;
}

qlin_status check_fp8(const qlin_fp8_t* t, int64_t rows, int64_t K) {
  if (t == nullptr || t->codes == nullptr || t->scale == nullptr) return QLIN_ERR_INVALID_ARG;
  if (t->rows != rows || t->K != K || !shape_ok(rows, K)) return QLIN_ERR_INVALID_ARG;
  if (!aligned(t->codes, 16) || !aligned(t->scale, 4)) return QLIN_ERR_MISALIGNED;
  return QLIN_OK;
}

qlin_status check_workspace(void* ws, size_t ws_bytes) {
  if (ws == nullptr || ws_bytes < qlin_workspace_size(0, 0)) return QLIN_ERR_WORKSPACE;
  // 8-byte aligned: the one-read quantizer reads its amax and arrival words
  // as one 64-bit load
  if (!aligned(ws, 8)) return QLIN_ERR_MISALIGNED;
  return QLIN_OK;
}

#define QLIN_TRY(expr)                 \
  do {                                 \
    qlin_status st__ = (expr);         \
    if (st__ != QLIN_OK) return st__;  \
  } while (0)

#define QLIN_CUDA(expr)                          \
  do {                                           \
    cudaError_t e__ = (expr);                    \
    if (e__ != cudaSuccess) return cuda_fail(e__); \
  } while (0)

}  // namespace
// Workspace words of the dynamic tensor scale: the one-read route's amax,
// arrival and departure counts (zero between calls), and the amax word of the
// two-pass route (cleared before each use).
constexpr int kWsOnePass = 0;
constexpr int kWsTwoPassAmax = 4;
// qlin_linear_dynamic: max |y| from the GEMM epilogue and the epilogue's
// departure count (words 5 and 6; zero between calls)
constexpr int kWsChainAmax = 5;

// Dynamic NVFP4 activation quantization: one read of x when it fits on chip,
// else the amax pass then the quantizer.  clear: zero the one-read words first.
cudaError_t quant_nvfp4_dynamic(const void* x, int64_t M, int64_t K, const qlin_nvfp4_t& out,
                                unsigned* ws, bool clear, cudaStream_t s, int sms,
                                unsigned* status) {
  cudaError_t e =
      launch_quant_nvfp4_onepass(x, M, K, out, ws + kWsOnePass, clear, s, sms, status, timeout());
  if (e != cudaErrorNotSupported) return e;
  unsigned* amax = ws + kWsTwoPassAmax;
  if ((e = launch_amax(x, M * K, amax, s, sms, status, timeout())) != cudaSuccess) return e;
  return launch_quant_nvfp4(x, M, K, reinterpret_cast<const float*>(amax), true, out, s, sms,
                            status, timeout());
}

}  // namespace qlin

using namespace qlin;

extern "C" {

size_t qlin_nvfp4_scale_bytes(int64_t rows, int64_t K) {
  if (!shape_ok(rows, K)) return 0;
  return (size_t)(((rows + 127) / 128) * (K / 64) * 512);
}

size_t qlin_workspace_size(int64_t M, int64_t K) {
  (void)M;
  (void)K;
  return 256;
}

qlin_status qlin_quantize_act_nvfp4(const void* x_bf16, int64_t M, int64_t K,
                                    const float* static_scale, qlin_nvfp4_t* out,
                                    void* workspace, size_t ws_bytes, void* stream) {
  if (x_bf16 == nullptr || !shape_ok(M, K)) return QLIN_ERR_INVALID_ARG;
  QLIN_TRY(check_nvfp4(out, M, K));
  if (!aligned(x_bf16, 16)) return QLIN_ERR_MISALIGNED;
  if (static_scale != nullptr && !aligned(static_scale, 4)) return QLIN_ERR_MISALIGNED;
  if (static_scale == nullptr) QLIN_TRY(check_workspace(workspace, ws_bytes));
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (static_scale == nullptr) {
    QLIN_CUDA(quant_nvfp4_dynamic(x_bf16, M, K, *out, static_cast<unsigned*>(workspace), false, s,
                                  sms, status));
  } else {
    QLIN_CUDA(launch_quant_nvfp4(x_bf16, M, K, static_scale, false, *out, s, sms, status, timeout()));
  }
  return QLIN_OK;
}

qlin_status qlin_quantize_act_nvfp4_noalloc(const void* x_bf16, int64_t M, int64_t K,
                                            qlin_nvfp4_t* out, void* stream) {
  if (x_bf16 == nullptr || !shape_ok(M, K)) return QLIN_ERR_INVALID_ARG;
  QLIN_TRY(check_nvfp4(out, M, K));
  if (!aligned(x_bf16, 16)) return QLIN_ERR_MISALIGNED;
  if (qlin_workspace_size(M, K) > QLIN_NOALLOC_SCRATCH_BYTES) {
    std::snprintf(g_last_error, sizeof g_last_error,
                  "shape [%lld, %lld] needs more than %d bytes of static scratch",
                  (long long)M, (long long)K, QLIN_NOALLOC_SCRATCH_BYTES);
    return QLIN_ERR_WORKSPACE;
  }
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  unsigned char* scratch = nullptr;
  QLIN_TRY(noalloc_scratch(&scratch));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the scratch words are cleared by the launch that uses them
  QLIN_CUDA(quant_nvfp4_dynamic(x_bf16, M, K, *out, reinterpret_cast<unsigned*>(scratch), true, s,
                                sms, status));
  return QLIN_OK;
}

qlin_status qlin_quantize_act_fp8(const void* x_bf16, int64_t M, int64_t K,
                                  const float* static_scale, qlin_fp8_t* out, void* workspace,
                                  size_t ws_bytes, void* stream) {
  if (x_bf16 == nullptr || !shape_ok(M, K)) return QLIN_ERR_INVALID_ARG;
  QLIN_TRY(check_fp8(out, M, K));
  if (out->per_channel) return QLIN_ERR_INVALID_ARG;
  if (!aligned(x_bf16, 16)) return QLIN_ERR_MISALIGNED;
  if (static_scale != nullptr && !aligned(static_scale, 4)) return QLIN_ERR_MISALIGNED;
  if (static_scale == nullptr) QLIN_TRY(check_workspace(workspace, ws_bytes));
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (static_scale == nullptr) {
    unsigned* ws = static_cast<unsigned*>(workspace);
    cudaError_t e = launch_quant_fp8_onepass(x_bf16, M, K, *out, ws + kWsOnePass, false, s, sms,
                                             status, timeout());
    if (e == cudaErrorNotSupported) {   // x does not fit on chip: amax pass, then quantize
      unsigned* amax = ws + kWsTwoPassAmax;
      QLIN_CUDA(launch_amax(x_bf16, M * K, amax, s, sms, status, timeout()));
      e = launch_quant_fp8(x_bf16, M, K, reinterpret_cast<const float*>(amax), true, *out, s, sms,
                           status, timeout());
    }
    QLIN_CUDA(e);
  } else {
    QLIN_CUDA(launch_quant_fp8(x_bf16, M, K, static_scale, false, *out, s, sms, status, timeout()));
  }
  return QLIN_OK;
}

qlin_status qlin_quantize_weight(const void* w_bf16, int64_t N, int64_t K, qlin_format fmt,
                                 void* out_desc, void* workspace, size_t ws_bytes, void* stream) {
  if (w_bf16 == nullptr || out_desc == nullptr || !shape_ok(N, K)) return QLIN_ERR_INVALID_ARG;
  if (!aligned(w_bf16, 16)) return QLIN_ERR_MISALIGNED;
  if (fmt == QLIN_FMT_NVFP4) {
    return qlin_quantize_act_nvfp4(w_bf16, N, K, nullptr, static_cast<qlin_nvfp4_t*>(out_desc),
                                   workspace, ws_bytes, stream);
  }
  if (fmt != QLIN_FMT_FP8) return QLIN_ERR_UNSUPPORTED;
  qlin_fp8_t* out = static_cast<qlin_fp8_t*>(out_desc);
  QLIN_TRY(check_fp8(out, N, K));
  if (!out->per_channel) return QLIN_ERR_INVALID_ARG;
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  QLIN_CUDA(launch_quant_fp8_rows(w_bf16, N, K, *out, static_cast<cudaStream_t>(stream), sms));
  return QLIN_OK;
}

static qlin_status gemm_common(bool fp4, const void* Aany, const void* Wany, void* y,
                               const float* next_scale, qlin_nvfp4_t* y_q, int64_t rq_col0,
                               void* stream, unsigned* y_amax = nullptr,
                               qlin_fp8_t* y_q8 = nullptr, float* y_sdec = nullptr) {
  GemmArgs a{};
  a.y_amax = y_amax;
  a.y_departures = y_amax != nullptr ? y_amax + 1 : nullptr;
  a.y_sdec = y_sdec;
  a.fp4 = fp4;
  if (fp4) {
    const qlin_nvfp4_t* A = static_cast<const qlin_nvfp4_t*>(Aany);
    const qlin_nvfp4_t* W = static_cast<const qlin_nvfp4_t*>(Wany);
    if (A == nullptr || W == nullptr) return QLIN_ERR_INVALID_ARG;
    QLIN_TRY(check_nvfp4(A, A->rows, A->K));
    QLIN_TRY(check_nvfp4(W, W->rows, A->K));
    a.a_codes = A->codes;
    a.w_codes = W->codes;
    a.sfa = A->scales;
    a.sfb = W->scales;
    a.sdec_a = A->tensor_scale;
    a.sdec_w = W->tensor_scale;
    a.M = A->rows;
    a.N = W->rows;
    a.K = A->K;
  } else {
    const qlin_fp8_t* A = static_cast<const qlin_fp8_t*>(Aany);
    const qlin_fp8_t* W = static_cast<const qlin_fp8_t*>(Wany);
    if (A == nullptr || W == nullptr) return QLIN_ERR_INVALID_ARG;
    QLIN_TRY(check_fp8(A, A->rows, A->K));
    QLIN_TRY(check_fp8(W, W->rows, A->K));
    if (A->per_channel) return QLIN_ERR_INVALID_ARG;
    a.a_codes = A->codes;
    a.w_codes = W->codes;
    a.sdec_a = A->scale;
    a.sdec_w = W->scale;
    a.w_per_channel = W->per_channel ? 1 : 0;
    a.M = A->rows;
    a.N = W->rows;
    a.K = A->K;
  }
  if (a.N % 64 != 0) return QLIN_ERR_INVALID_ARG;
  if (a.M > (int64_t)1 << 31 || a.N > (int64_t)1 << 31) return QLIN_ERR_UNSUPPORTED;
  if (y != nullptr && !aligned(y, 16)) return QLIN_ERR_MISALIGNED;
  a.y = y;
  if (next_scale != nullptr) {
    // the re-quantized operand: NVFP4 after an NVFP4 GEMM, FP8 after an FP8 one
    const int64_t rq_cols = fp4 ? (y_q ? y_q->K : 0) : (y_q8 ? y_q8->K : 0);
    if ((fp4 ? y_q == nullptr : y_q8 == nullptr) || !aligned(next_scale, 4))
      return QLIN_ERR_INVALID_ARG;
    if (rq_cols < 64 || rq_cols % 64 != 0 || rq_col0 < 0 || rq_col0 % 64 != 0 ||
        rq_col0 + rq_cols > a.N)
      return QLIN_ERR_INVALID_ARG;
    if (fp4) {
      QLIN_TRY(check_nvfp4(y_q, a.M, y_q->K));
      a.rq_codes = y_q->codes;
      a.rq_scales = y_q->scales;
      a.rq_tensor_scale = y_q->tensor_scale;
    } else {
      QLIN_TRY(check_fp8(y_q8, a.M, y_q8->K));
      if (y_q8->per_channel) return QLIN_ERR_INVALID_ARG;
      a.rq_codes = y_q8->codes;
      a.rq_tensor_scale = y_q8->scale;
    }
    a.next_scale = next_scale;
    a.rq_col0 = rq_col0;
    a.rq_cols = rq_cols;
  } else if (y == nullptr) {
    return QLIN_ERR_INVALID_ARG;  // nothing to write
  }
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  cudaError_t e = launch_gemm(a, static_cast<cudaStream_t>(stream), sms, status,
                              g_timeout_ns.load(std::memory_order_relaxed));
  if (e != cudaSuccess) return cuda_fail(e);
  return QLIN_OK;
}

qlin_status qlin_gemm_nvfp4(const qlin_nvfp4_t* A, const qlin_nvfp4_t* W, void* y_bf16,
                            void* stream) {
  if (y_bf16 == nullptr) return QLIN_ERR_INVALID_ARG;
  return gemm_common(true, A, W, y_bf16, nullptr, nullptr, 0, stream);
}

qlin_status qlin_gemm_fp8(const qlin_fp8_t* A, const qlin_fp8_t* W, void* y_bf16, void* stream) {
  if (y_bf16 == nullptr) return QLIN_ERR_INVALID_ARG;
  return gemm_common(false, A, W, y_bf16, nullptr, nullptr, 0, stream);
}

qlin_status qlin_linear_fused(const qlin_nvfp4_t* A, const qlin_nvfp4_t* W, void* y_bf16,
                              const float* next_scale, qlin_nvfp4_t* y_q, int64_t rq_col0,
                              void* stream) {
  return gemm_common(true, A, W, y_bf16, next_scale, y_q, rq_col0, stream);
}

// The unquantized 16-bit linear (bf16 or fp16 operands and output).
static qlin_status gemm16(const void* a16, int64_t lda, const void* w16, int64_t M, int64_t N,
                          int64_t K, void* y16, void* stream, bool fp16) {
  if (a16 == nullptr || w16 == nullptr || y16 == nullptr) return QLIN_ERR_INVALID_ARG;
  if (M < 1 || K < 64 || K % 64 != 0 || N < 64 || N % 64 != 0 || lda < K)
    return QLIN_ERR_INVALID_ARG;
  if (M > (int64_t)1 << 31 || N > (int64_t)1 << 31) return QLIN_ERR_UNSUPPORTED;
  if (!aligned(a16, 16) || !aligned(w16, 16) || !aligned(y16, 16) || (lda * 2) % 16 != 0)
    return QLIN_ERR_MISALIGNED;
  GemmArgs a{};
  a.bf16 = true;
  a.fp16 = fp16;
  a.a_codes = a16;
  a.a_row_bytes = lda * 2;
  a.w_codes = w16;
  a.y = y16;
  a.M = M;
  a.N = N;
  a.K = K;
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  cudaError_t e = launch_gemm(a, static_cast<cudaStream_t>(stream), sms, status, timeout());
  if (e != cudaSuccess) return cuda_fail(e);
  return QLIN_OK;
}

qlin_status qlin_gemm_bf16(const void* a_bf16, int64_t lda, const void* w_bf16, int64_t M,
                           int64_t N, int64_t K, void* y_bf16, void* stream) {
  return gemm16(a_bf16, lda, w_bf16, M, N, K, y_bf16, stream, false);
}

qlin_status qlin_gemm_fp16(const void* a_fp16, int64_t lda, const void* w_fp16, int64_t M,
                           int64_t N, int64_t K, void* y_fp16, void* stream) {
  return gemm16(a_fp16, lda, w_fp16, M, N, K, y_fp16, stream, true);
}

qlin_status qlin_linear_dynamic(const qlin_nvfp4_t* A, const qlin_nvfp4_t* W, void* y_bf16,
                                qlin_nvfp4_t* y_q, void* workspace, size_t ws_bytes,
                                void* stream) {
  if (A == nullptr || W == nullptr || y_bf16 == nullptr || y_q == nullptr)
    return QLIN_ERR_INVALID_ARG;
  QLIN_TRY(check_nvfp4(y_q, A->rows, W->rows));
  QLIN_TRY(check_workspace(workspace, ws_bytes));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned* amax = static_cast<unsigned*>(workspace) + kWsChainAmax;
  // y and its tensor scale in one GEMM (its last CTA writes S_dec into y_q's
  // tensor scale and resets the scratch words), then the quantizer of y with
  // that scale
  QLIN_TRY(gemm_common(true, A, W, y_bf16, nullptr, nullptr, 0, stream, amax, nullptr,
                       y_q->tensor_scale));
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  QLIN_CUDA(launch_quant_nvfp4(y_bf16, A->rows, W->rows, y_q->tensor_scale, false, *y_q, s, sms,
                               status, timeout()));
  return QLIN_OK;
}

qlin_status qlin_linear_fused_fp8(const qlin_fp8_t* A, const qlin_fp8_t* W, void* y_bf16,
                                  const float* next_scale, qlin_fp8_t* y_q, int64_t rq_col0,
                                  void* stream) {
  if (next_scale == nullptr) return QLIN_ERR_INVALID_ARG;
  return gemm_common(false, A, W, y_bf16, next_scale, nullptr, rq_col0, stream, nullptr, y_q);
}

qlin_status qlin_sync_status(void* stream) {
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  QLIN_CUDA(cudaStreamSynchronize(s));
  unsigned word = 0;
  QLIN_CUDA(cudaMemcpy(&word, status, sizeof word, cudaMemcpyDeviceToHost));
  if (word != 0) {
    const unsigned zero = 0;
    QLIN_CUDA(cudaMemcpy(status, &zero, sizeof zero, cudaMemcpyHostToDevice));
    return word == kErrTimeout ? QLIN_ERR_TIMEOUT : QLIN_ERR_CUDA;
  }
  return QLIN_OK;
}

qlin_status qlin_selftest_bounded_wait(uint64_t timeout_ns, void* stream) {
  unsigned* status;
  int sms;
  QLIN_TRY(device_state(&status, &sms));
  timeout_ns = std::min<uint64_t>(std::max<uint64_t>(timeout_ns, 1000ull), 2000000000ull);
  QLIN_CUDA(launch_wait_selftest(timeout_ns, static_cast<cudaStream_t>(stream), status));
  return QLIN_OK;
}

void qlin_set_wait_timeout_ns(uint64_t ns) {
  g_timeout_ns.store(std::max<uint64_t>(ns, 1000ull), std::memory_order_relaxed);
}

const char* qlin_status_str(qlin_status s) {
  switch (s) {
    case QLIN_OK: return "ok";
    case QLIN_ERR_INVALID_ARG: return "invalid argument";
    case QLIN_ERR_UNSUPPORTED: return "unsupported";
    case QLIN_ERR_MISALIGNED: return "misaligned pointer";
    case QLIN_ERR_CUDA: return "CUDA error";
    case QLIN_ERR_TIMEOUT: return "device wait timed out";
    case QLIN_ERR_WORKSPACE: return "workspace missing or too small";
  }
  return "unknown status";
}

const char* qlin_last_error(void) { return g_last_error; }

}  // extern "C"
