// Exhaustive check of qlin::e4m3_code_div6 (the NVFP4 block-scale code
// E4M3(t / 6) of Sec. 4's two-level scaling, computed without a division)
// against the E4M3 code of the correctly rounded fp32 quotient __fdiv_rn(t, 6)
// for every fp32 t in [0, 4096], every 1021st pattern above it, and +inf.
// NaN must stay NaN.  Prints one line: "mismatches N nan_ok B".
#include <cstdio>
#include <cstdint>
#include "qlin_device.cuh"

__device__ unsigned long long g_bad;
__device__ unsigned g_nan_ok;

__global__ void check(uint32_t lo, uint32_t hi, uint32_t step) {
  const uint64_t n = ((uint64_t)hi - lo) / step + 1;
  for (uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; i < n;
       i += (uint64_t)gridDim.x * blockDim.x) {
    const float t = __uint_as_float(lo + (uint32_t)(i * step));
    if (qlin::e4m3_code_div6(t) != qlin::e4m3_code(__fdiv_rn(t, 6.0f))) atomicAdd(&g_bad, 1ull);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    const uint32_t c = qlin::e4m3_code_div6(__uint_as_float(0x7FC00000u));
    g_nan_ok = (c & 0x7Fu) == 0x7Fu;
  }
}

int main() {
  unsigned long long zero = 0;
  cudaMemcpyToSymbol(g_bad, &zero, sizeof zero);
  check<<<1216, 256>>>(0u, 0x45800000u, 1u);             // [0, 4096]
  check<<<1216, 256>>>(0x45800001u, 0x7F800000u, 1021u);  // (4096, +inf]
  check<<<1, 32>>>(0x7F800000u, 0x7F800000u, 1u);         // +inf itself
  const cudaError_t e = cudaDeviceSynchronize();
  unsigned long long bad = 0;
  unsigned nan_ok = 0;
  cudaMemcpyFromSymbol(&bad, g_bad, sizeof bad);
  cudaMemcpyFromSymbol(&nan_ok, g_nan_ok, sizeof nan_ok);
  printf("mismatches %llu nan_ok %u status %s\n", bad, nan_ok, cudaGetErrorString(e));
  return e == cudaSuccess ? 0 : 1;
}
