// Block-scaled GEMMs on the 5th-generation tensor cores (tcgen05) of sm_103a:
// the NVFP4 and FP8 linear layers of Sec. 4 ("Quantization": activation
// quantization lets the linears run on the FP8 / NVFP4 tensor cores), with a
// fused epilogue that writes the bf16 output and, optionally, re-quantizes it
// to NVFP4 for the next layer.
//
// Kernel structure (one persistent CTA per SM, 320 threads):
//   warp 0      TMA producer: A/W code tiles (tensor maps, 128-byte swizzle)
//               and, for NVFP4, the 512-byte scale atoms (bulk copies) into a
//               ring of shared-memory stages.
//   warp 1      TMEM allocator and MMA issuer: per 32 bytes of K one
//               tcgen05.mma (NVFP4: kind::mxf4nvf4 with scale_vec::4X, K = 64;
//               FP8: kind::f8f6f4, K = 32) into an fp32 TMEM accumulator of
//               128 lanes x BN columns.  NVFP4 scales are first moved
//               shared -> TMEM with tcgen05.cp.
//   warps 2-9   epilogue: tcgen05.ld of the accumulator (each warp its 32-lane
//               quarter and one half of the columns), alpha scaling, bf16
//               rounding, global stores, and the optional NVFP4 re-quantization
//               of the bf16 values (one row per thread, so block amax is
//               thread-local).
// Tiles are 128 x BN output blocks, scheduled m-fastest so consecutive CTAs
// share a weight tile in L2.  Every wait is bounded (see WaitCtl).
#include <mutex>

#include "qlin_internal.h"

namespace qlin {

namespace {

constexpr int kBM = 128;
constexpr int kRowBytes = 128;      // bytes of K per stage and row: one swizzle row
constexpr int kStepsPerStage = 4;   // one MMA per 32 bytes of K
constexpr int kEpiWarps = 8;
constexpr int kThreads = (2 + kEpiWarps) * 32;
constexpr int kSmemBudget = 232448 - 2048;  // opt-in shared memory minus barriers/alignment

constexpr int pow2_at_least(int x) {
  int p = 32;
  while (p < x) p <<= 1;
  return p;
}

template <bool kFp4, int kBN>
struct Cfg {
  static constexpr int kSfbAtoms = kFp4 ? (kBN + 127) / 128 : 0;
  static constexpr int kABytes = kBM * kRowBytes;
  static constexpr int kBBytes = kBN * kRowBytes;
  static constexpr int kSfaBytes = kFp4 ? kStepsPerStage * 512 : 0;
  static constexpr int kSfbBytes = kFp4 ? kSfbAtoms * kStepsPerStage * 512 : 0;
  static constexpr int kStageBytes = kABytes + kBBytes + kSfaBytes + kSfbBytes;
  static constexpr int kStagesRaw = kSmemBudget / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kNumAcc = (kFp4 && kBN == 256) ? 1 : 2;
  static constexpr int kSfColsPerStep = kFp4 ? 4 + 4 * kSfbAtoms : 0;
  static constexpr int kSfColBase = kNumAcc * kBN;
  static constexpr int kTmemCols =
      pow2_at_least(kSfColBase + kStages * kStepsPerStage * kSfColsPerStep);
  static constexpr int kBarrierBytes = 256;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kBarrierBytes;
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
  static_assert(kTmemCols <= 512, "TMEM budget");
  static_assert(kSmemBytes <= 232448, "shared memory budget");
  static_assert(kStages >= 2, "pipeline depth");
};

struct KParams {
  const uint8_t* sfa;
  const uint8_t* sfb;
  const float* sdec_a;
  const float* sdec_w;
  int w_per_channel;
  uint16_t* y;
  int64_t M, N, K;
  const float* next_scale;
  uint8_t* rq_codes;
  uint8_t* rq_scales;
  float* rq_tensor_scale;
  int64_t rq_col0, rq_cols;
  unsigned* err;
  uint64_t timeout_ns;
};

// Bounded wait that ignores the abort flag: used to drain copies and MMAs in
// flight before the CTA releases TMEM and exits.
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity, uint64_t timeout_ns,
                                           unsigned* err) {
  const uint32_t a = smem_u32(bar);
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(a, parity)) {
    if (global_timer_ns() - t0 > timeout_ns) {
      atomicExch(err, kErrTimeout);
      return;
    }
  }
}

__device__ __forceinline__ void st_global_v4(void* p, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.global.v4.b32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

template <bool kFp4, int kBN, bool kRequant>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_a,
                const __grid_constant__ CUtensorMap tmap_b, const KParams p) {
  using C = Cfg<kFp4, kBN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* tmem_full = empty + C::kStages;
  uint64_t* tmem_empty = tmem_full + 2;
  uint64_t* mma_done = tmem_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tmem_full[a], 1);
      mbar_init(&tmem_empty[a], kEpiWarps);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmap_a);
    prefetch_tmap(&tmap_b);
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.err, p.timeout_ns};

  const int tiles_m = (int)((p.M + kBM - 1) / kBM);
  const int tiles_n = (int)((p.N + kBN - 1) / kBN);
  const int num_tiles = tiles_m * tiles_n;
  const int64_t k_bytes = kFp4 ? p.K / 2 : p.K;
  const int num_kb = (int)((k_bytes + kRowBytes - 1) / kRowBytes);
  const int k_steps = (int)(k_bytes / 32);
  const int64_t k_atoms = p.K / 64;  // 4-scale atom columns (NVFP4)

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer ---
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      const int n_atom_rows = (int)((p.N + 127) / 128);
      for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
        const int mb = tile % tiles_m, nb = tile / tiles_m;
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, ctl)) {
            ok = false;
            break;
          }
          uint8_t* sA = smem + stage * C::kStageBytes;
          uint8_t* sB = sA + C::kABytes;
          uint32_t bytes = C::kABytes + C::kBBytes;
          int nat = 0, nsfb = 0;
          if (kFp4) {
            nat = min(kStepsPerStage, k_steps - kb * kStepsPerStage);
            nsfb = min(C::kSfbAtoms, n_atom_rows - nb * (kBN / 128));
            bytes += (uint32_t)(nat * 512 * (1 + nsfb));
          }
          mbar_arrive_expect_tx(&full[stage], bytes);
          tma_load_2d(sA, &tmap_a, &full[stage], kb * kRowBytes, mb * kBM);
          tma_load_2d(sB, &tmap_b, &full[stage], kb * kRowBytes, nb * kBN);
          if (kFp4) {
            uint8_t* sSFA = sB + C::kBBytes;
            uint8_t* sSFB = sSFA + C::kSfaBytes;
            bulk_load(sSFA, p.sfa + ((int64_t)mb * k_atoms + kb * kStepsPerStage) * 512,
                      (uint32_t)nat * 512, &full[stage]);
            for (int r = 0; r < nsfb; ++r)
              bulk_load(sSFB + r * kStepsPerStage * 512,
                        p.sfb + ((int64_t)(nb * (kBN / 128) + r) * k_atoms +
                                 kb * kStepsPerStage) * 512,
                        (uint32_t)nat * 512, &full[stage]);
          }
          ++issued;
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      // Wait for the last copies issued (normally complete long ago) so none
      // is in flight when the CTA exits.
      const int n_drain = min(issued, C::kStages);
      for (int i = 0; i < n_drain; ++i) {
        if (--stage < 0) {
          stage = C::kStages - 1;
          phase ^= 1u;
        }
        mbar_drain(&full[stage], phase, p.timeout_ns, p.err);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------- MMA issuer ---
    if (lane == 0) {
      const uint32_t idesc = kFp4 ? idesc_nvfp4(kBN) : idesc_fp8(kBN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        if (!mbar_wait(&tmem_empty[acc], acc_phase ^ 1u, ctl)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kBN);
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&full[stage], phase, ctl)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sA = smem_u32(smem + stage * C::kStageBytes);
          const uint32_t sB = sA + C::kABytes;
          const int nsteps = min(kStepsPerStage, k_steps - kb * kStepsPerStage);
          for (int j = 0; j < nsteps; ++j) {
            const uint64_t adesc = sdesc_k128(sA + j * 32);
            const uint64_t bdesc = sdesc_k128(sB + j * 32);
            const uint32_t accumulate = (kb > 0 || j > 0) ? 1u : 0u;
            if (kFp4) {
              const uint32_t sSFA = sB + C::kBBytes;
              const uint32_t sSFB = sSFA + C::kSfaBytes;
              const uint32_t sfa_t = tmem_base + (uint32_t)(C::kSfColBase +
                                                            (stage * kStepsPerStage + j) *
                                                                C::kSfColsPerStep);
              const uint32_t sfb_t = sfa_t + 4;
              tc_cp_scales(sfa_t, sdesc_scales(sSFA + j * 512));
#pragma unroll
              for (int r = 0; r < C::kSfbAtoms; ++r)
                tc_cp_scales(sfb_t + 4 * r,
                             sdesc_scales(sSFB + r * kStepsPerStage * 512 + j * 512));
              mma_nvfp4(d_tmem, adesc, bdesc, idesc, sfa_t, sfb_t, accumulate);
            } else {
              mma_fp8(d_tmem, adesc, bdesc, idesc, accumulate);
            }
          }
          tc_commit(&empty[stage]);
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(&tmem_full[acc]);
        if (C::kNumAcc == 2) {
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1u;
        } else {
          acc_phase ^= 1u;
        }
      }
      // Every MMA / scale copy issued must finish before TMEM is released.
      tc_commit(mma_done);
      mbar_drain(mma_done, 0, p.timeout_ns, p.err);
    }
  } else {
    // --------------------------------------------------------- epilogue ---
    constexpr int kCols = kBN / 2;  // columns per thread
    constexpr int kChunks = kCols / 32;
    const int e = warp - 2;
    const int quarter = warp & 3;   // the TMEM lane quarter this warp may access
    const int half = e >> 2;
    const float sdec_a = *p.sdec_a;
    const float alpha = kFp4 ? __fmul_rn(sdec_a, *p.sdec_w) : 0.0f;
    float s_enc_next = 0.0f;
    if (kRequant) {
      const float s_next = *p.next_scale;
      s_enc_next = encode_scale(s_next);
      if (blockIdx.x == 0 && threadIdx.x == 64 && p.rq_tensor_scale != p.next_scale)
        *p.rq_tensor_scale = s_next;
    }
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      if (!mbar_wait(&tmem_full[acc], acc_phase, ctl)) break;
      tc_fence_after();
      const int mb = tile % tiles_m, nb = tile / tiles_m;
      const int64_t row = (int64_t)mb * kBM + quarter * 32 + lane;
      const int64_t col0 = (int64_t)nb * kBN + half * kCols;
      uint32_t packed[kCols / 2];
      const uint32_t taddr =
          tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * kBN + half * kCols);
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        uint32_t r[32];
        tmem_ld32(taddr + c * 32, r);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float a0 = alpha, a1 = alpha;
          if (!kFp4) {
            const int64_t n = col0 + c * 32 + 2 * i;
            const float w0 = p.w_per_channel ? (n < p.N ? __ldg(p.sdec_w + n) : 0.0f) : *p.sdec_w;
            const float w1 =
                p.w_per_channel ? (n + 1 < p.N ? __ldg(p.sdec_w + n + 1) : 0.0f) : *p.sdec_w;
            a0 = __fmul_rn(sdec_a, w0);
            a1 = __fmul_rn(sdec_a, w1);
          }
          packed[c * 16 + i] = pack_bf16x2(__fmul_rn(__uint_as_float(r[2 * i]), a0),
                                           __fmul_rn(__uint_as_float(r[2 * i + 1]), a1));
        }
      }
      // The accumulator is in registers: hand it back to the MMA warp.
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tmem_empty[acc]);
      if (C::kNumAcc == 2) {
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      } else {
        acc_phase ^= 1u;
      }

      if (row < p.M) {
        if (p.y != nullptr) {
          uint16_t* yr = p.y + row * p.N + col0;
#pragma unroll
          for (int v = 0; v < kCols / 8; ++v)
            if (col0 + v * 8 < p.N)
              st_global_v4(yr + v * 8, packed[4 * v], packed[4 * v + 1], packed[4 * v + 2],
                           packed[4 * v + 3]);
        }
        if (kRequant) {
#pragma unroll
          for (int g = 0; g < kCols / 64; ++g) {
            const int64_t c64 = col0 + g * 64;
            if (c64 < p.rq_col0 || c64 + 64 > p.rq_col0 + p.rq_cols || c64 >= p.N) continue;
            const int64_t lc = c64 - p.rq_col0;
            uint32_t words[8];
            uint32_t sw = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
              const uint32_t* pk = packed + g * 32 + b * 8;  // 16 bf16 of this block
              uint32_t m = 0;
#pragma unroll
              for (int i = 0; i < 8; ++i) m = __vmaxu2(m, pk[i] & 0x7FFF7FFFu);
              m = max(m & 0xFFFFu, m >> 16);
              float r_b;
              const uint32_t sb = nvfp4_block_scale(__uint_as_float(m << 16), s_enc_next, &r_b);
              sw |= sb << (8 * b);
#pragma unroll
              for (int h8 = 0; h8 < 2; ++h8) {
                float f[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  f[2 * i] = __fmul_rn(bf16_lo(pk[h8 * 4 + i]), r_b);
                  f[2 * i + 1] = __fmul_rn(bf16_hi(pk[h8 * 4 + i]), r_b);
                }
                words[b * 2 + h8] = e2m1x8(f);
              }
            }
            uint8_t* cp = p.rq_codes + row * (p.rq_cols / 2) + lc / 2;
            st_global_v4(cp, words[0], words[1], words[2], words[3]);
            st_global_v4(cp + 16, words[4], words[5], words[6], words[7]);
            *reinterpret_cast<uint32_t*>(p.rq_scales + scale_offset(row, lc / 16, p.rq_cols)) = sw;
          }
        }
      }
    }
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::kTmemCols);
  }
}

// One CTA waits on an mbarrier phase that nothing completes; the bounded wait
// expires, records the timeout and the kernel returns normally.
__global__ void wait_selftest_kernel(unsigned* err, uint64_t timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const WaitCtl ctl{&abort_flag, err, timeout_ns};
    (void)mbar_wait(&bar, 0, ctl);
  }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

template <bool kFp4, int kBN, bool kRequant>
cudaError_t launch_cfg(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                       uint64_t timeout_ns) {
  using C = Cfg<kFp4, kBN>;
  const uint64_t k_bytes = kFp4 ? (uint64_t)a.K / 2 : (uint64_t)a.K;
  CUtensorMap ta, tb;
  if (encode_tensor_map_2d_u8(&ta, a.a_codes, k_bytes, (uint64_t)a.M, kRowBytes, kBM) !=
          CUDA_SUCCESS ||
      encode_tensor_map_2d_u8(&tb, a.w_codes, k_bytes, (uint64_t)a.N, kRowBytes, kBN) !=
          CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  KParams p{};
  p.sfa = a.sfa;
  p.sfb = a.sfb;
  p.sdec_a = a.sdec_a;
  p.sdec_w = a.sdec_w;
  p.w_per_channel = a.w_per_channel;
  p.y = static_cast<uint16_t*>(a.y);
  p.M = a.M;
  p.N = a.N;
  p.K = a.K;
  p.next_scale = a.next_scale;
  p.rq_codes = a.rq_codes;
  p.rq_scales = a.rq_scales;
  p.rq_tensor_scale = a.rq_tensor_scale;
  p.rq_col0 = a.rq_col0;
  p.rq_cols = a.rq_cols;
  p.err = err;
  p.timeout_ns = timeout_ns;
  auto kern = gemm_kernel<kFp4, kBN, kRequant>;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    C::kSmemBytes);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const int64_t tiles = ((a.M + kBM - 1) / kBM) * ((a.N + kBN - 1) / kBN);
  const int grid = (int)std::min<int64_t>(tiles, num_sms);
  kern<<<grid, kThreads, C::kSmemBytes, s>>>(ta, tb, p);
  return cudaGetLastError();
}

template <bool kFp4>
cudaError_t dispatch_bn(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                        uint64_t timeout_ns) {
  // 128 x 256 tiles when they fill the machine, else 128 x 128 (small M).
  const int64_t tiles256 = ((a.M + kBM - 1) / kBM) * ((a.N + 255) / 256);
  const bool wide = tiles256 >= num_sms;
  if constexpr (kFp4) {
    if (a.next_scale != nullptr)
      return wide ? launch_cfg<true, 256, true>(a, s, num_sms, err, timeout_ns)
                  : launch_cfg<true, 128, true>(a, s, num_sms, err, timeout_ns);
  }
  return wide ? launch_cfg<kFp4, 256, false>(a, s, num_sms, err, timeout_ns)
              : launch_cfg<kFp4, 128, false>(a, s, num_sms, err, timeout_ns);
}

}  // namespace

CUresult encode_tensor_map_2d_u8(CUtensorMap* map, const void* base, uint64_t inner_bytes,
                                 uint64_t rows, uint32_t box_inner, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return CUDA_ERROR_NOT_FOUND;
  const cuuint64_t dims[2] = {inner_bytes, rows};
  const cuuint64_t strides[1] = {inner_bytes};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

cudaError_t launch_gemm(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                        uint64_t timeout_ns) {
  return a.fp4 ? dispatch_bn<true>(a, s, num_sms, err, timeout_ns)
               : dispatch_bn<false>(a, s, num_sms, err, timeout_ns);
}

cudaError_t launch_wait_selftest(uint64_t timeout_ns, cudaStream_t s, unsigned* err) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(err, timeout_ns);
  return cudaGetLastError();
}

}  // namespace qlin
