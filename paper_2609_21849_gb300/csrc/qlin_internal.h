// Internal declarations shared by the translation units of libqlin.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "qlin.h"
#include "qlin_device.cuh"

namespace qlin {

// ---- quantizers (qlin_quant.cu) ----
// err / timeout_ns: device status word and limit of the bounded waits.
cudaError_t launch_amax(const void* x, int64_t n_elems, unsigned* amax_bits, cudaStream_t s,
                        int num_sms, unsigned* err, uint64_t timeout_ns);
cudaError_t launch_quant_nvfp4(const void* x, int64_t M, int64_t K, const float* scale_src,
                               bool dynamic, const qlin_nvfp4_t& out, cudaStream_t s,
                               int num_sms, unsigned* err, uint64_t timeout_ns);
cudaError_t launch_quant_fp8(const void* x, int64_t M, int64_t K, const float* scale_src,
                             bool dynamic, const qlin_fp8_t& out, cudaStream_t s, int num_sms,
                             unsigned* err, uint64_t timeout_ns);
// Dynamic tensor scale in one read of x (x held on chip across the grid).
// sync: three device words of scratch, zero at launch (clear = zero them
// first) and zero again when the kernel ends.  Returns cudaErrorNotSupported,
// having launched nothing, when x does not fit; the caller then runs amax +
// quant.
cudaError_t launch_quant_nvfp4_onepass(const void* x, int64_t M, int64_t K,
                                       const qlin_nvfp4_t& out, unsigned* sync, bool clear,
                                       cudaStream_t s, int num_sms, unsigned* err,
                                       uint64_t timeout_ns);
cudaError_t launch_quant_fp8_onepass(const void* x, int64_t M, int64_t K, const qlin_fp8_t& out,
                                     unsigned* sync, bool clear, cudaStream_t s, int num_sms,
                                     unsigned* err, uint64_t timeout_ns);
cudaError_t launch_quant_fp8_rows(const void* w, int64_t N, int64_t K, const qlin_fp8_t& out,
                                  cudaStream_t s, int num_sms);

// ---- GEMMs (qlin_gemm.cu) ----
struct GemmArgs {
  bool fp4;                 // NVFP4 (true) or FP8
  bool bf16;                // 16-bit float operands (fp4 false), no scales
  bool fp16;                // with bf16: the operands and y are fp16, not bf16
  const void* a_codes;      // [M, K/2] or [M, K] bytes, or bf16 [M, K]
  int64_t a_row_bytes;      // row stride of A in bytes (0: packed rows)
  const void* w_codes;      // [N, K/2] or [N, K] bytes
  const uint8_t* sfa;       // swizzled block scales (NVFP4)
  const uint8_t* sfb;
  const float* sdec_a;      // tensor scale of A
  const float* sdec_w;      // tensor scale of W (NVFP4) / per-channel or single (FP8)
  int w_per_channel;        // FP8: 1 if sdec_w has N entries
  void* y;                  // bf16 [M, N] or null
  int64_t M, N, K;
  // fused NVFP4 re-quantization of y's columns [rq_col0, rq_col0 + rq_cols)
  const float* next_scale;  // null = off
  uint8_t* rq_codes;
  uint8_t* rq_scales;
  float* rq_tensor_scale;
  int64_t rq_col0, rq_cols;
  // optional max |bf16 y| (fp32 bits, atomicMax), with a departure count;
  // both are zero at launch and reset by the last CTA, which writes
  // S_dec = amax / (6 * 448) to y_sdec
  unsigned* y_amax;
  unsigned* y_departures;
  float* y_sdec;
};
cudaError_t launch_gemm(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                        uint64_t timeout_ns);
cudaError_t launch_wait_selftest(uint64_t timeout_ns, cudaStream_t s, unsigned* err);

// Resolves cuTensorMapEncodeTiled through the runtime (no libcuda link).
CUresult encode_tensor_map_out_bf16(CUtensorMap* map, void* base, uint64_t cols, uint64_t rows,
                                    bool fp16 = false);
CUresult encode_tensor_map_2d_u8(CUtensorMap* map, const void* base, uint64_t inner_bytes,
                                 uint64_t rows, uint32_t box_inner, uint32_t box_rows);

}  // namespace qlin
