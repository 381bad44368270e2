// Activation and weight quantizers (Sec. 4, "Quantization": FP8 / NVFP4
// post-training quantization; activations are quantized at run time, weights
// once).  All kernels here are HBM-bandwidth bound streaming kernels:
//
//   amax_bf16_kernel      max |x| over a tensor (the dynamic tensor scale)
//   quant_nvfp4_kernel    bf16 -> packed e2m1 codes + E4M3 block scales in the
//                         tensor-core scale layout + FP32 tensor scale
//   quant_fp8_kernel      bf16 -> E4M3 codes with one tensor scale
//   quant_fp8_rows_kernel bf16 weights -> E4M3 codes with one scale per row
//
// Data layout of the streaming kernels: the [M, K] input is viewed as a flat
// array of 8-element (16-byte) chunks.  A warp covers 32 consecutive chunks
// (512 contiguous bytes) per load instruction; two neighbouring lanes hold
// one 16-element block, eight neighbouring lanes one 64-element group whose
// four block scales form one 32-bit word of the scale layout.  Because
// K % 64 == 0, a group never straddles a row.
#include "qlin_internal.h"

namespace qlin {

namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;  // 16-byte chunks in flight per lane

// Largest |bf16| in a 16-byte chunk, as the bit pattern of a bf16 magnitude.
__device__ __forceinline__ uint32_t chunk_abs_max_bits(const uint4 v) {
  const uint32_t m = __vmaxu2(__vmaxu2(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu),
                              __vmaxu2(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu));
  return max(m & 0xFFFFu, m >> 16);
}

__device__ __forceinline__ void unpack8(const uint4 v, float (&f)[8]) {
  f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
  f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
  f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
  f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

// amax over n_chunks 16-byte chunks, folded into *amax_bits (fp32 bits;
// must be zero before the launch).
__global__ void __launch_bounds__(kThreads) amax_bf16_kernel(const uint4* __restrict__ x,
                                                             int64_t n_chunks,
                                                             unsigned* __restrict__ amax_bits) {
  __shared__ uint32_t warp_max[kThreads / 32];
  uint32_t m = 0;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  int64_t c = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  for (; c + (kUnroll - 1) * stride < n_chunks; c += kUnroll * stride) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) v[u] = __ldg(x + c + u * stride);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) m = max(m, chunk_abs_max_bits(v[u]));
  }
  for (; c < n_chunks; c += stride) m = max(m, chunk_abs_max_bits(__ldg(x + c)));
  m = __reduce_max_sync(0xFFFFFFFFu, m);
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t b = 0;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) b = max(b, warp_max[w]);
    if (b) atomicMax(amax_bits, b << 16);
  }
}

// NVFP4 quantizer.  kDynamic: scale_src holds amax (fp32) and
// S_dec = amax / 2688 (1 if amax == 0); otherwise scale_src holds S_dec.
template <bool kDynamic>
__global__ void __launch_bounds__(kThreads) quant_nvfp4_kernel(
    const uint4* __restrict__ x, int64_t n_chunks, int64_t K, const float* scale_src,
    float* sdec_out, uint32_t* __restrict__ codes, uint8_t* __restrict__ scales) {
  float s_dec;
  if (kDynamic) {
    const float amax = *scale_src;
    s_dec = (amax == 0.0f) ? 1.0f : __fdiv_rn(amax, 2688.0f);
  } else {
    s_dec = *scale_src;
  }
  const float s_enc = encode_scale(s_dec);
  if (blockIdx.x == 0 && threadIdx.x == 0 && sdec_out != scale_src) *sdec_out = s_dec;

  const int lane = threadIdx.x & 31;
  const int g0 = lane & ~7;
  const int64_t chunks_per_row = K >> 3;
  const int64_t warp = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
  for (int64_t base = warp * 32 * kUnroll; base < n_chunks; base += nwarps * 32 * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t c = base + u * 32 + lane;
      v[u] = (c < n_chunks) ? __ldg(x + c) : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t c = base + u * 32 + lane;
      // block amax over the lane pair holding the 16-element block
      uint32_t mb = chunk_abs_max_bits(v[u]);
      mb = max(mb, __shfl_xor_sync(0xFFFFFFFFu, mb, 1));
      float r_b;
      const uint32_t sb = nvfp4_block_scale(__uint_as_float(mb << 16), s_enc, &r_b);
      float f[8];
      unpack8(v[u], f);
#pragma unroll
      for (int i = 0; i < 8; ++i) f[i] = __fmul_rn(f[i], r_b);
      const uint32_t code = e2m1x8(f);
      const uint32_t s0 = __shfl_sync(0xFFFFFFFFu, sb, g0);
      const uint32_t s1 = __shfl_sync(0xFFFFFFFFu, sb, g0 + 2);
      const uint32_t s2 = __shfl_sync(0xFFFFFFFFu, sb, g0 + 4);
      const uint32_t s3 = __shfl_sync(0xFFFFFFFFu, sb, g0 + 6);
      if (c < n_chunks) {
        codes[c] = code;
        if ((lane & 7) == 0) {
          const int64_t row = c / chunks_per_row;
          const int64_t col = (c - row * chunks_per_row) << 3;
          *reinterpret_cast<uint32_t*>(scales + scale_offset(row, col >> 4, K)) =
              s0 | (s1 << 8) | (s2 << 16) | (s3 << 24);
        }
      }
    }
  }
}

// FP8 quantizer with one tensor scale (dynamic: S_dec = amax / 448).
template <bool kDynamic>
__global__ void __launch_bounds__(kThreads) quant_fp8_kernel(const uint4* __restrict__ x,
                                                             int64_t n_chunks,
                                                             const float* scale_src,
                                                             float* sdec_out,
                                                             uint2* __restrict__ codes) {
  float s_dec;
  if (kDynamic) {
    const float amax = *scale_src;
    s_dec = (amax == 0.0f) ? 1.0f : __fdiv_rn(amax, 448.0f);
  } else {
    s_dec = *scale_src;
  }
  const float s_enc = encode_scale(s_dec);
  if (blockIdx.x == 0 && threadIdx.x == 0 && sdec_out != scale_src) *sdec_out = s_dec;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t c = (int64_t)blockIdx.x * kThreads + threadIdx.x; c < n_chunks; c += stride) {
    float f[8];
    unpack8(__ldg(x + c), f);
#pragma unroll
    for (int i = 0; i < 8; ++i) f[i] = __fmul_rn(f[i], s_enc);
    codes[c] = make_uint2(e4m3x4(f[0], f[1], f[2], f[3]), e4m3x4(f[4], f[5], f[6], f[7]));
  }
}

// FP8 weights, one scale per row: one warp per row, two passes over the row
// (the second hits L1/L2).
__global__ void __launch_bounds__(kThreads) quant_fp8_rows_kernel(const uint4* __restrict__ w,
                                                                  int64_t rows, int64_t K,
                                                                  float* __restrict__ s_rows,
                                                                  uint2* __restrict__ codes) {
  const int lane = threadIdx.x & 31;
  const int64_t cpr = K >> 3;
  const int64_t warp = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * kThreads) >> 5;
  for (int64_t r = warp; r < rows; r += nwarps) {
    const uint4* wr = w + r * cpr;
    uint32_t m = 0;
    for (int64_t c = lane; c < cpr; c += 32) m = max(m, chunk_abs_max_bits(__ldg(wr + c)));
    m = __reduce_max_sync(0xFFFFFFFFu, m);
    const float amax = __uint_as_float(m << 16);
    const float s_dec = (amax == 0.0f) ? 1.0f : __fdiv_rn(amax, 448.0f);
    const float s_enc = encode_scale(s_dec);
    if (lane == 0) s_rows[r] = s_dec;
    for (int64_t c = lane; c < cpr; c += 32) {
      float f[8];
      unpack8(__ldg(wr + c), f);
#pragma unroll
      for (int i = 0; i < 8; ++i) f[i] = __fmul_rn(f[i], s_enc);
      codes[r * cpr + c] =
          make_uint2(e4m3x4(f[0], f[1], f[2], f[3]), e4m3x4(f[4], f[5], f[6], f[7]));
    }
  }
}

int grid_for(int64_t work_items, int items_per_block, int num_sms) {
  const int64_t want = (work_items + items_per_block - 1) / items_per_block;
  const int64_t cap = (int64_t)num_sms * (2048 / kThreads);
  return (int)std::max<int64_t>(1, std::min(want, cap));
}

}  // namespace

cudaError_t launch_amax(const void* x, int64_t n_elems, unsigned* amax_bits, cudaStream_t s,
                        int num_sms) {
  cudaError_t e = cudaMemsetAsync(amax_bits, 0, sizeof(unsigned), s);
  if (e != cudaSuccess) return e;
  const int64_t n_chunks = n_elems / 8;
  amax_bf16_kernel<<<grid_for(n_chunks, kThreads * kUnroll, num_sms), kThreads, 0, s>>>(
      static_cast<const uint4*>(x), n_chunks, amax_bits);
  return cudaGetLastError();
}

cudaError_t launch_quant_nvfp4(const void* x, int64_t M, int64_t K, const float* scale_src,
                               bool dynamic, const qlin_nvfp4_t& out, cudaStream_t s,
                               int num_sms) {
  const int64_t n_chunks = M * K / 8;
  const int grid = grid_for(n_chunks, kThreads * kUnroll, num_sms);
  auto* xin = static_cast<const uint4*>(x);
  auto* codes = reinterpret_cast<uint32_t*>(out.codes);
  if (dynamic)
    quant_nvfp4_kernel<true><<<grid, kThreads, 0, s>>>(xin, n_chunks, K, scale_src,
                                                        out.tensor_scale, codes, out.scales);
  else
    quant_nvfp4_kernel<false><<<grid, kThreads, 0, s>>>(xin, n_chunks, K, scale_src,
                                                         out.tensor_scale, codes, out.scales);
  return cudaGetLastError();
}

cudaError_t launch_quant_fp8(const void* x, int64_t M, int64_t K, const float* scale_src,
                             bool dynamic, const qlin_fp8_t& out, cudaStream_t s, int num_sms) {
  const int64_t n_chunks = M * K / 8;
  const int grid = grid_for(n_chunks, kThreads * kUnroll, num_sms);
  auto* xin = static_cast<const uint4*>(x);
  auto* codes = reinterpret_cast<uint2*>(out.codes);
  if (dynamic)
    quant_fp8_kernel<true><<<grid, kThreads, 0, s>>>(xin, n_chunks, scale_src, out.scale, codes);
  else
    quant_fp8_kernel<false><<<grid, kThreads, 0, s>>>(xin, n_chunks, scale_src, out.scale, codes);
  return cudaGetLastError();
}

cudaError_t launch_quant_fp8_rows(const void* w, int64_t N, int64_t K, const qlin_fp8_t& out,
                                  cudaStream_t s, int num_sms) {
  const int grid = grid_for(N, kThreads / 32, num_sms);
  quant_fp8_rows_kernel<<<grid, kThreads, 0, s>>>(static_cast<const uint4*>(w), N, K, out.scale,
                                                  reinterpret_cast<uint2*>(out.codes));
  return cudaGetLastError();
}

}  // namespace qlin
