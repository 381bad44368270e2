// Tensor-core rate probe (measurement only, not part of the linear layer):
// back-to-back tcgen05.mma instructions of one kind and shape from one thread
// per CTA (or CTA pair), on every SM at once, operands resident in shared
// memory.  It gives the MMA ceiling that the GEMMs' roofline fractions are
// also reported against, in FLOP per SM cycle (clock-independent) and in
// FLOP/s at the clock the probe ran at.
//
// The instruction kinds are the ones the GEMMs issue: kind::mxf4nvf4
// block_scale scale_vec::4X (NVFP4), kind::f8f6f4 (E4M3) and kind::f16
// (bf16), each as cta_group::1 (M = 128) and cta_group::2 (M = 256), with A
// in shared memory (as in the GEMMs) or in TMEM (the A-from-tensor-memory
// form, A written there by tcgen05.st), which shows whether operand reads
// from shared memory bound the rate.
#include <cstdio>

#include "qlin_device.cuh"
#include "qlin_probe.h"

namespace qlin {
namespace {

constexpr int kProbeThreads = 128;
constexpr int kASmem = 128 * 128;       // 128 rows x 128 bytes of K
constexpr int kBSmemMax = 256 * 128;    // up to 256 rows x 128 bytes
constexpr int kSfSmem = 4096;           // scale atoms (NVFP4)
// Requested shared memory: more than half an SM's, so that no SM holds two
// probe CTAs (each allocates all 512 TMEM columns; two CTA pairs sharing SMs
// could otherwise wait on each other's allocations).
constexpr int kProbeSmem = 160 * 1024;
static_assert(1024 + kASmem + kBSmemMax + kSfSmem <= kProbeSmem, "probe buffers");

__device__ __forceinline__ uint32_t hash32(uint32_t x) {
  x ^= x >> 16;
  x *= 0x7FEB352Du;
  x ^= x >> 15;
  x *= 0x846CA68Bu;
  x ^= x >> 16;
  return x;
}

// Bounded wait on an mbarrier phase (iteration limit of a few seconds at the
// try_wait suspend hint; records an error flag).
__device__ __forceinline__ bool probe_wait(uint64_t* bar, uint32_t parity, unsigned* err) {
  for (uint32_t i = 0; i < (1u << 17); ++i)
    if (mbar_try_wait(smem_u32(bar), parity)) return true;
  atomicExch(err, kErrTimeout);
  return false;
}

// A operand in TMEM: D[tmem] (+)= A[tmem] * B[smem]^T.
__device__ __forceinline__ void mma_ts(int kind, bool pair, uint32_t d, uint32_t a_t, uint64_t b,
                                       uint32_t idesc, uint32_t sfa, uint32_t sfb, uint32_t acc) {
  if (kind == 4 && pair)
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::2.kind::mxf4nvf4.block_scale.scale_vec::4X"
                 " [%0], [%1], %2, %3, [%5], [%6], p;\n\t}" ::"r"(d),
                 "r"(a_t), "l"(b), "r"(idesc), "r"(acc), "r"(sfa), "r"(sfb) : "memory");
  else if (kind == 4)
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::mxf4nvf4.block_scale.scale_vec::4X"
                 " [%0], [%1], %2, %3, [%5], [%6], p;\n\t}" ::"r"(d),
                 "r"(a_t), "l"(b), "r"(idesc), "r"(acc), "r"(sfa), "r"(sfb) : "memory");
  else if (kind == 8 && pair)
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
                 "r"(a_t), "l"(b), "r"(idesc), "r"(acc) : "memory");
  else if (kind == 8)
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
                 "r"(a_t), "l"(b), "r"(idesc), "r"(acc) : "memory");
  else if (pair)
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::2.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
                 "r"(a_t), "l"(b), "r"(idesc), "r"(acc) : "memory");
  else
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
                 "r"(a_t), "l"(b), "r"(idesc), "r"(acc) : "memory");
}

// Write 32 consecutive TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0],"
      " {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16,"
      " %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// kKind: 4 = NVFP4 (mxf4nvf4, K = 64), 8 = FP8 (f8f6f4, K = 32), 16 = bf16
// (f16, K = 16); every instruction reads 32 bytes of K per operand row.
// kATmem: A from TMEM columns [384, 416) (8 columns per instruction).
template <int kKind, bool kPair, int kN, bool kATmem = false>
__global__ void __launch_bounds__(kProbeThreads, 1)
    mma_probe_kernel(int iters, unsigned long long* out, unsigned* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = base;
  uint8_t* sB = base + kASmem;
  uint8_t* sSF = sB + kBSmemMax;
  __shared__ uint64_t bar;
  __shared__ uint32_t tmem_slot;
  // operands: hashed bytes (typical bit toggling), finite in every format
  // (bf16 / E4M3 exponent fields kept below all-ones); scales 1.0 (0x38)
  for (int i = threadIdx.x; i < (kASmem + kBSmemMax) / 4; i += kProbeThreads) {
    uint32_t v = hash32((uint32_t)i * 2654435761u + blockIdx.x);
    if (kKind == 8) v &= 0xBFBFBFBFu;          // E4M3: no NaN codes
    if (kKind == 16) v &= 0xBFFFBFFFu;         // bf16: exponent below all-ones
    reinterpret_cast<uint32_t*>(base)[i] = v;
  }
  for (int i = threadIdx.x; i < kSfSmem / 4; i += kProbeThreads)
    reinterpret_cast<uint32_t*>(sSF)[i] = 0x38383838u;
  const uint32_t rank = kPair ? cluster_ctarank() : 0;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    mbar_fence_init();
  }
  if ((threadIdx.x >> 5) == 1) {
    if (kPair)
      tmem_alloc_pair(&tmem_slot, 512);
    else
      tmem_alloc(&tmem_slot, 512);
  }
  fence_proxy_async_smem();
  tc_fence_before();
  if (kPair)
    cluster_sync();
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tb = tmem_slot;
  if (kATmem) {
    // A in TMEM: each warp writes its lane quarter's 32 columns
    uint32_t r[32];
    for (int i = 0; i < 32; ++i) {
      uint32_t v = hash32((uint32_t)(threadIdx.x * 32 + i) * 2246822519u + blockIdx.x);
      if (kKind == 8) v &= 0xBFBFBFBFu;
      if (kKind == 16) v &= 0xBFFFBFFFu;
      r[i] = v;
    }
    tmem_st32(tb + ((uint32_t)((threadIdx.x >> 5) * 32) << 16) + 384, r);
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    tc_fence_before();
    if (kPair)
      cluster_sync();
    else
      __syncthreads();
    tc_fence_after();
  }
  if (threadIdx.x == 0 && rank == 0) {
    constexpr int kM = kPair ? 256 : 128;
    const uint32_t idesc = kKind == 4 ? idesc_nvfp4(kN, kM)
                           : kKind == 8 ? idesc_fp8(kN, kM)
                                        : idesc_bf16(kN, kM);
    const uint32_t a = smem_u32(sA), b = smem_u32(sB), sf = smem_u32(sSF);
    const uint32_t sf_t = tb + 256;   // scale columns: A at +0, B atoms at +4, +8
    if (kKind == 4) {
      for (int r = 0; r < 3; ++r) {
        if (kPair)
          tc_cp_scales_pair(sf_t + 4 * r, sdesc_scales(sf + 512 * r));
        else
          tc_cp_scales(sf_t + 4 * r, sdesc_scales(sf + 512 * r));
      }
    }
    if (kPair)
      tc_commit_pair_mc(&bar, 1);
    else
      tc_commit(&bar);
    bool ok = probe_wait(&bar, 0, err);
    tc_fence_after();
    const unsigned long long c0 = clock64();
    const uint64_t t0 = global_timer_ns();
    for (int i = 0; ok && i < iters; ++i) {
      const uint32_t j = (uint32_t)(i & 3) * 32;
      const uint64_t ad = sdesc_k128(a + j), bd = sdesc_k128(b + j);
      const uint32_t acc = i > 0 ? 1u : 0u;
      if (kATmem) {
        mma_ts(kKind, kPair, tb, tb + 384 + (uint32_t)(i & 3) * 8, bd, idesc, sf_t, sf_t + 4, acc);
      } else if (kKind == 4) {
        if (kPair)
          mma_nvfp4_pair(tb, ad, bd, idesc, sf_t, sf_t + 4, acc);
        else
          mma_nvfp4(tb, ad, bd, idesc, sf_t, sf_t + 4, acc);
      } else if (kKind == 8) {
        if (kPair)
          mma_fp8_pair(tb, ad, bd, idesc, acc);
        else
          mma_fp8(tb, ad, bd, idesc, acc);
      } else {
        if (kPair)
          mma_bf16_pair(tb, ad, bd, idesc, acc);
        else
          mma_bf16(tb, ad, bd, idesc, acc);
      }
    }
    if (kPair)
      tc_commit_pair_mc(&bar, 1);
    else
      tc_commit(&bar);
    ok = ok && probe_wait(&bar, 1, err);
    const unsigned long long c1 = clock64();
    const uint64_t t1 = global_timer_ns();
    const int slot = (int)blockIdx.x / (kPair ? 2 : 1);
    out[2 * slot] = ok ? c1 - c0 : 0ull;
    out[2 * slot + 1] = ok ? t1 - t0 : 0ull;
  }
  tc_fence_before();
  if (kPair)
    cluster_sync();
  else
    __syncthreads();
  if ((threadIdx.x >> 5) == 1) {
    tc_fence_after();
    if (kPair)
      tmem_dealloc_pair(tb, 512);
    else
      tmem_dealloc(tb, 512);
  }
}

template <int kKind, bool kPair, int kN, bool kATmem = false>
cudaError_t launch_probe(int ctas, int iters, unsigned long long* out, unsigned* err,
                         cudaStream_t s) {
  auto kern = mma_probe_kernel<kKind, kPair, kN, kATmem>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kProbeSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kPair ? 2 : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3((unsigned)ctas, 1, 1);
  cfg.blockDim = dim3(kProbeThreads, 1, 1);
  cfg.dynamicSmemBytes = kProbeSmem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, iters, out, err);
}

// ------------------------------------------------- scale-copy issue rate ---
// One CTA pair: thread 0 of CTA 0 issues `mmas` NVFP4 pair MMAs (N = 256) per
// iteration while `warps` warps of CTA 0 (lane 0 each) issue `copies`
// tcgen05.cp.cta_group::2.32x128b.warpx4 per iteration between them, into
// TMEM columns away from the MMAs' (the accumulator and its scale columns).
// Per pair: out[0] the MMA thread's cycles, out[1] the first copy warp's
// cycles until all copies (every warp's) have completed.
constexpr int kCpThreads = 320;               // warp 0 MMA, warp 1 TMEM, warps 2-9 copies
constexpr int kCpSmem = 160 * 1024;
constexpr int kCpSrc = 65536;                 // copy sources: 16 slots of 4 KB
static_assert(1024 + kCpSrc + 16 * 4096 <= kCpSmem, "copy probe buffers");

__global__ void __launch_bounds__(kCpThreads, 1)
    cp_probe_kernel(int iters, int mmas, int copies, int warps, unsigned long long* out,
                    unsigned* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = base;
  uint8_t* sB = base + kASmem;
  uint8_t* sSF = base + 49152;
  uint8_t* sCp = base + kCpSrc;
  __shared__ uint64_t bar[3];
  __shared__ uint32_t tmem_slot;
  for (int i = threadIdx.x; i < (kCpSrc + 16 * 4096) / 4; i += kCpThreads) {
    uint32_t v = hash32((uint32_t)i * 2654435761u + blockIdx.x);
    // operands hashed; the scale region and the copy sources hold 1.0 (0x38)
    reinterpret_cast<uint32_t*>(base)[i] = (i >= 49152 / 4) ? 0x38383838u : v;
  }
  const uint32_t rank = cluster_ctarank();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    mbar_init(&bar[2], warps);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc_pair(&tmem_slot, 512);
  fence_proxy_async_smem();
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tb = tmem_slot;
  const uint32_t sf_t = tb + 256;   // the MMAs' scale columns (256..267)
  if (threadIdx.x == 0 && rank == 0) {
    for (int r = 0; r < 3; ++r) tc_cp_scales_pair(sf_t + 4 * r, sdesc_scales(smem_u32(sSF) + 512 * r));
    tc_commit_pair_mc(&bar[0], 1);
    (void)probe_wait(&bar[0], 0, err);
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  if (rank == 0 && warp == 0 && lane == 0) {
    const uint32_t idesc = idesc_nvfp4(256, 256);
    const uint32_t a = smem_u32(sA), b = smem_u32(sB);
    const unsigned long long c0 = clock64();
    for (int i = 0; i < iters; ++i)
      for (int j = 0; j < mmas; ++j)
        mma_nvfp4_pair(tb, sdesc_k128(a + (j & 3) * 32), sdesc_k128(b + (j & 3) * 32), idesc,
                       sf_t, sf_t + 4, (i | j) ? 1u : 0u);
    tc_commit_pair_mc(&bar[1], 1);
    const bool ok = probe_wait(&bar[1], 0, err);
    out[2 * (blockIdx.x / 2)] = ok ? clock64() - c0 : 0ull;
  }
  if (rank == 0 && lane == 0 && warp >= 2 && warp < 2 + warps) {
    const int per = copies / warps;
    const unsigned long long c0 = clock64();
    for (int i = 0; i < iters; ++i)
      for (int c = 0; c < per; ++c) {
        const int k = (i * per + c + 5 * (warp - 2)) & 15;
        tc_cp_scales_pair(tb + 320 + (uint32_t)((k & 7) * 8),
                          sdesc_scales(smem_u32(sCp) + (uint32_t)k * 4096));
      }
    tc_commit_pair_mc(&bar[2], 1);
    if (warp == 2) {
      const bool ok = probe_wait(&bar[2], 0, err);
      out[2 * (blockIdx.x / 2) + 1] = ok ? clock64() - c0 : 0ull;
    }
  }
  __syncwarp();
  tc_fence_before();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tb, 512);
  }
}

// ------------------------------------------- shared-memory fill rate ---
// One CTA per SM: `threads` issuing threads (lane 0 of warps 0..threads-1)
// each keep `depth` copies of 16 KB in flight into a ring of their own, for
// `iters` copies: mode 0 tiled 2-D tensor copies (a 128-row x 128-byte box,
// 128-byte swizzle, from a [rows, 1536-byte] view of src, as the GEMM's
// operand boxes), mode 1 plain bulk copies of 16 contiguous KB.  Box
// positions are pseudo-random over src.  out[cta] = the first thread's
// cycles until its last copy landed.
constexpr int kFillThreads = 256;
constexpr int kFillSmem = 200 * 1024;
constexpr int kFillBox = 16384;
constexpr int kFillRowBytes = 1536;

__global__ void __launch_bounds__(kFillThreads, 1)
    fill_probe_kernel(const __grid_constant__ CUtensorMap tm, const uint8_t* src,
                      unsigned long long src_bytes, int mode, int threads, int depth, int iters,
                      int rows, unsigned long long* out, unsigned* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t bar[8][8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int w = 0; w < 8; ++w)
      for (int d = 0; d < 8; ++d) mbar_init(&bar[w][d], 1);
    mbar_fence_init();
  }
  __syncthreads();
  if (lane == 0 && warp < threads) {
    uint8_t* ring = base + warp * depth * kFillBox;
    uint32_t ph[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    unsigned long long r = ((unsigned long long)blockIdx.x * 8 + warp) * 7919ull + 1ull;
    const unsigned long long c0 = clock64();
    int issued = 0;
    bool ok = true;
    for (int i = 0; i < iters; ++i) {
      const int sl = i % depth;
      if (i >= depth) {
        if (!probe_wait(&bar[warp][sl], ph[sl], err)) {
          ok = false;
          break;
        }
        ph[sl] ^= 1u;
      }
      mbar_arrive_expect_tx(&bar[warp][sl], kFillBox);
      r = r * 6364136223846793005ull + 1442695040888963407ull;
      if (mode == 0) {
        const int x = (int)((r >> 33) % (unsigned long long)(kFillRowBytes / 128)) * 128;
        const int y = (int)((r >> 13) % (unsigned long long)(rows / 128)) * 128;
        tma_load_2d(ring + sl * kFillBox, &tm, &bar[warp][sl], x, y);
      } else {
        const unsigned long long off = ((r >> 20) % (src_bytes / kFillBox)) * kFillBox;
        bulk_load(ring + sl * kFillBox, src + off, kFillBox, &bar[warp][sl]);
      }
      ++issued;
    }
    // the copies still in flight land before the CTA exits
    for (int k = 0; k < depth && k < issued; ++k) {
      const int sl = (issued - 1 - k) % depth;
      if (!probe_wait(&bar[warp][sl], ph[sl], err)) ok = false;
      ph[sl] ^= 1u;
    }
    if (warp == 0) out[blockIdx.x] = ok ? clock64() - c0 : 0ull;
  }
  __syncthreads();
}

}  // namespace
}  // namespace qlin

using namespace qlin;

extern "C" int qlin_probe_mma(int kind, int pair, int n, int ctas, int iters,
                              unsigned long long* out, unsigned* err, void* stream) {
  // kind + 100: the same kind with A in TMEM
  const bool a_tmem = kind > 100;
  if (a_tmem) kind -= 100;
  if (out == nullptr || err == nullptr || iters < 1 || ctas < 1) return 1;
  if (pair && ctas % 2 != 0) return 1;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSuccess;
  bool matched = false;
#define QLIN_PROBE_CASE(K, P, N)                                      \
  if (kind == K && (pair != 0) == P && n == N) {                      \
    matched = true;                                                   \
    e = a_tmem ? launch_probe<K, P, N, true>(ctas, iters, out, err, s) \
               : launch_probe<K, P, N, false>(ctas, iters, out, err, s); \
  }
  QLIN_PROBE_CASE(4, true, 256);
  QLIN_PROBE_CASE(4, false, 256);
  QLIN_PROBE_CASE(4, false, 128);
  QLIN_PROBE_CASE(8, true, 256);
  QLIN_PROBE_CASE(8, false, 256);
  QLIN_PROBE_CASE(16, true, 256);
#undef QLIN_PROBE_CASE
  if (!matched) return 1;
  return e == cudaSuccess ? 0 : 4;
}

extern "C" int qlin_probe_scale_copy(int warps, int copies, int mmas, int ctas, int iters,
                                     unsigned long long* out, unsigned* err, void* stream) {
  if (out == nullptr || err == nullptr || iters < 1 || ctas < 2 || ctas % 2 != 0) return 1;
  if (warps < 1 || warps > 8 || copies < 0 || copies % warps != 0 || mmas < 0 || mmas > 16)
    return 1;
  if (cudaFuncSetAttribute(cp_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kCpSmem) != cudaSuccess)
    return 4;
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3((unsigned)ctas, 1, 1);
  cfg.blockDim = dim3(kCpThreads, 1, 1);
  cfg.dynamicSmemBytes = kCpSmem;
  cfg.stream = static_cast<cudaStream_t>(stream);
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, cp_probe_kernel, iters, mmas, copies, warps, out, err) ==
                 cudaSuccess
             ? 0
             : 4;
}

extern "C" int qlin_probe_fill(int mode, int threads, int depth, int ctas, int iters,
                               const void* src, unsigned long long src_bytes,
                               unsigned long long* out, unsigned* err, void* stream) {
  if (out == nullptr || err == nullptr || src == nullptr || iters < 1 || ctas < 1) return 1;
  if ((mode != 0 && mode != 1) || threads < 1 || threads > 8 || depth < 1 || depth > 8 ||
      1024 + threads * depth * kFillBox > kFillSmem)
    return 1;
  const unsigned long long rows = src_bytes / kFillRowBytes / 128 * 128;
  if (rows < 128 || rows > (1ull << 30) || (reinterpret_cast<uintptr_t>(src) & 127u) != 0)
    return 1;
  using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                       &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || fn == nullptr)
    return 4;
  CUtensorMap tm;
  const cuuint64_t dims[2] = {(cuuint64_t)kFillRowBytes, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)kFillRowBytes};
  const cuuint32_t box[2] = {128, 128};
  const cuuint32_t es[2] = {1, 1};
  if (reinterpret_cast<EncodeFn>(fn)(&tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(src),
                                     dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return 1;
  if (cudaFuncSetAttribute(fill_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kFillSmem) != cudaSuccess)
    return 4;
  fill_probe_kernel<<<ctas, kFillThreads, kFillSmem, static_cast<cudaStream_t>(stream)>>>(
      tm, static_cast<const uint8_t*>(src), src_bytes, mode, threads, depth, iters, (int)rows,
      out, err);
  return cudaGetLastError() == cudaSuccess ? 0 : 4;
}
