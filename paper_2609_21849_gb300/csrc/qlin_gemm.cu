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
#include <cstring>
#include <mutex>

#include "qlin_internal.h"

namespace qlin {

namespace {

constexpr int kBM = 128;
constexpr int kRowBytes = 128;      // bytes of K per stage and row: one swizzle row
constexpr int kStepsPerStage = 4;   // one MMA per 32 bytes of K
constexpr int kEpiWarps = 8;
constexpr int kEpiWarp0 = 4;   // warps 0-3: producer, MMA, two scale-copy warps
constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
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
  // epilogue staging: per epilogue warp two 32 x 32 bf16 boxes (2 KB each)
  static constexpr int kOutBytes = kEpiWarps * 2 * 2048;
  static constexpr int kStagesRaw = (kSmemBudget - kOutBytes) / kStageBytes;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kNumAcc = (kFp4 && kBN == 256) ? 1 : 2;
  static constexpr int kSfColsPerStep = kFp4 ? 4 + 4 * kSfbAtoms : 0;
  static constexpr int kSfColBase = kNumAcc * kBN;
  static constexpr int kTmemCols =
      pow2_at_least(kSfColBase + kStages * kStepsPerStage * kSfColsPerStep);
  static constexpr int kBarrierBytes = 512;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kOutBytes + kBarrierBytes;
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

template <bool kFp4, int kBN, int kCM, bool kRequant>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_a,
                const __grid_constant__ CUtensorMap tmap_b,
                const __grid_constant__ CUtensorMap tmap_y, const KParams p) {
  using C = Cfg<kFp4, kBN>;
  // kCM CTAs of a cluster take kCM consecutive M tiles of the same N tile;
  // each loads 1/kCM of the weight tile (and of its scales) and multicasts
  // it to all, so W is read from L2 once per cluster.
  constexpr int kBRows = kBN / kCM;
  constexpr uint16_t kMask = (uint16_t)((1u << kCM) - 1u);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* out_stage = smem + C::kStages * C::kStageBytes;   // epilogue staging boxes
  uint64_t* full = reinterpret_cast<uint64_t*>(out_stage + C::kOutBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* sf_ready = empty + C::kStages;   // NVFP4: the stage's scales are in TMEM
  uint64_t* sf_full = sf_ready + C::kStages;  // NVFP4: the stage's scale bytes landed
  uint64_t* tmem_full = sf_full + C::kStages;
  uint64_t* tmem_empty = tmem_full + 2;
  uint64_t* mma_done = tmem_empty + 2;
  uint64_t* sf_done = mma_done + 1;   // two barriers, one per scale-copy warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sf_done + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = kCM > 1 ? (int)cluster_ctarank() : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCM);   // one arrival from the MMA warp of each CTA
      mbar_init(&sf_ready[s], 2);   // one commit per scale-copy warp
      mbar_init(&sf_full[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tmem_full[a], 1);
      mbar_init(&tmem_empty[a], kEpiWarps);
    }
    mbar_init(mma_done, 1);
    mbar_init(&sf_done[0], 1);
    mbar_init(&sf_done[1], 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmap_a);
    prefetch_tmap(&tmap_b);
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  if (kCM > 1)
    cluster_sync();   // peers' barriers exist before any multicast reaches them
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.err, p.timeout_ns};

  const int tiles_m = (int)((p.M + kBM - 1) / kBM);
  const int tiles_n = (int)((p.N + kBN - 1) / kBN);
  const int groups_m = (tiles_m + kCM - 1) / kCM;
  const int num_ctiles = groups_m * tiles_n;
  const int cid = (int)blockIdx.x / kCM;
  const int ncl = (int)gridDim.x / kCM;
  const int64_t k_bytes = kFp4 ? p.K / 2 : p.K;
  const int num_kb = (int)((k_bytes + kRowBytes - 1) / kRowBytes);
  const int k_steps = (int)(k_bytes / 32);
  const int64_t k_atoms = p.K / 64;  // 4-scale atom columns (NVFP4)

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer ---
    // A TMA instruction occupies its issuing thread for hundreds of cycles,
    // so the stage's copies are issued by several lanes executing the SAME
    // instruction with per-lane operands: lanes 0 and 1 one tensor load (A
    // tile, W tile), lanes 2.. one bulk copy (A scales, W scale rows).
    const int nlanes = kFp4 ? 3 + C::kSfbAtoms : 2;
    if (lane < nlanes) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      const int n_atom_rows = (int)((p.N + 127) / 128);
      const uint16_t self_mask = (uint16_t)(1u << rank);
      for (int ct = cid; ct < num_ctiles; ct += ncl) {
        const int nb = ct / groups_m;
        const int mb = (ct % groups_m) * kCM + rank;
        const bool m_live = mb < tiles_m;   // the last group may be partly past M
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, ctl)) {
            ok = false;
            break;
          }
          uint8_t* sA = smem + stage * C::kStageBytes;
          uint8_t* sB = sA + C::kABytes;
          const int nat = min(kStepsPerStage, k_steps - kb * kStepsPerStage);
          const int nsfb = kFp4 ? min(C::kSfbAtoms, n_atom_rows - nb * (kBN / 128)) : 0;
          if (lane == 0) mbar_arrive_expect_tx(&full[stage], C::kABytes + C::kBBytes);
          if (kFp4 && lane == 2)   // the scales complete on their own barrier
            mbar_arrive_expect_tx(&sf_full[stage],
                                  (uint32_t)(nat * 512 * ((m_live ? 1 : 0) + nsfb)));
          __syncwarp((1u << nlanes) - 1u);
          // operand tiles
          if (lane < 2) {
            const bool is_a = lane == 0;
            const CUtensorMap* map = is_a ? &tmap_a : &tmap_b;
            const int32_t y = is_a ? mb * kBM : nb * kBN + rank * kBRows;
            uint8_t* dst = is_a ? sA : sB + rank * kBRows * kRowBytes;
            if (kCM == 1)
              tma_load_2d(dst, map, &full[stage], kb * kRowBytes, y);
            else
              tma_load_2d_mc(dst, map, &full[stage], kb * kRowBytes, y,
                             is_a ? self_mask : kMask);
          } else if (kFp4) {
            // block scales: lane 2 the A atoms, lane 3 + r the W atom row r
            const bool is_a = lane == 2;
            const int r = lane - 3;
            const bool live = is_a ? m_live : (r < nsfb && r % kCM == rank);
            const uint8_t* src =
                is_a ? p.sfa + ((int64_t)mb * k_atoms + kb * kStepsPerStage) * 512
                     : p.sfb + ((int64_t)(nb * (kBN / 128) + r) * k_atoms + kb * kStepsPerStage) *
                                   512;
            uint8_t* dst = is_a ? sB + C::kBBytes
                                : sB + C::kBBytes + C::kSfaBytes + r * kStepsPerStage * 512;
            if (live) {
              if (kCM == 1)
                bulk_load(dst, src, (uint32_t)nat * 512, &sf_full[stage]);
              else
                bulk_load_mc(dst, src, (uint32_t)nat * 512, &sf_full[stage],
                             is_a ? self_mask : kMask);
            }
          }
          ++issued;
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      // Wait for the last copies into this CTA (normally complete long ago)
      // so none is in flight when the CTA exits.
      if (lane == 0 || (kFp4 && lane == 2)) {
        uint64_t* bars = lane == 0 ? full : sf_full;
        const int n_drain = min(issued, C::kStages);
        for (int i = 0; i < n_drain; ++i) {
          if (--stage < 0) {
            stage = C::kStages - 1;
            phase ^= 1u;
          }
          mbar_drain(&bars[stage], phase, p.timeout_ns, p.err);
        }
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
      for (int ct = cid; ct < num_ctiles && ok; ct += ncl) {
        if (!mbar_wait(&tmem_empty[acc], acc_phase ^ 1u, ctl)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kBN);
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&full[stage], phase, ctl) ||
              (kFp4 && !mbar_wait(&sf_ready[stage], phase, ctl))) {
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
              const uint32_t sfa_t = tmem_base + (uint32_t)(C::kSfColBase +
                                                            (stage * kStepsPerStage + j) *
                                                                C::kSfColsPerStep);
              mma_nvfp4(d_tmem, adesc, bdesc, idesc, sfa_t, sfa_t + 4, accumulate);
            } else {
              mma_fp8(d_tmem, adesc, bdesc, idesc, accumulate);
            }
          }
          // the stage is free once this CTA's MMAs have read it: tell every
          // CTA of the cluster (their producers multicast into it)
          if (kCM == 1)
            tc_commit(&empty[stage]);
          else
            tc_commit_mc(&empty[stage], kMask);
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
  } else if (warp == 2 || warp == 3) {
    // --------------------------------------------- NVFP4 scale copies ---
    // Block scales move shared -> TMEM from two threads of their own (a
    // tcgen05.cp occupies its issuing thread ~50 cycles), beside the MMA
    // stream: warp 2 the A atoms and W atom row 0, warp 3 W atom row 1.
    if (kFp4 && lane == 0) {
      const int sw = warp - 2;
      int stage = 0;
      uint32_t phase = 0;
      for (int ct = cid; ct < num_ctiles; ct += ncl) {
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&sf_full[stage], phase, ctl)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sSFA = smem_u32(smem + stage * C::kStageBytes) + C::kABytes + C::kBBytes;
          const uint32_t sSFB = sSFA + C::kSfaBytes;
          const int nsteps = min(kStepsPerStage, k_steps - kb * kStepsPerStage);
          for (int j = 0; j < nsteps; ++j) {
            const uint32_t sfa_t = tmem_base + (uint32_t)(C::kSfColBase +
                                                          (stage * kStepsPerStage + j) *
                                                              C::kSfColsPerStep);
            if (sw == 0) {
              tc_cp_scales(sfa_t, sdesc_scales(sSFA + j * 512));
              tc_cp_scales(sfa_t + 4, sdesc_scales(sSFB + j * 512));
            } else if (C::kSfbAtoms > 1) {
              tc_cp_scales(sfa_t + 8, sdesc_scales(sSFB + kStepsPerStage * 512 + j * 512));
            }
          }
          tc_commit(&sf_ready[stage]);
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      tc_commit(&sf_done[sw]);
      mbar_drain(&sf_done[sw], 0, p.timeout_ns, p.err);
    }
  } else {
    // --------------------------------------------------------- epilogue ---
    constexpr int kCols = kBN / 2;  // columns per thread
    constexpr int kChunks = kCols / 32;
    const int e = warp - kEpiWarp0;
    const int quarter = warp & 3;   // the TMEM lane quarter this warp may access
    const int half = e >> 2;
    uint8_t* const out_buf = out_stage + e * 4096;   // this warp's two staging boxes
    const float sdec_a = *p.sdec_a;
    const float alpha = kFp4 ? __fmul_rn(sdec_a, *p.sdec_w) : 0.0f;
    float s_enc_next = 0.0f;
    if (kRequant) {
      const float s_next = *p.next_scale;
      s_enc_next = encode_scale(s_next);
      if (blockIdx.x == 0 && threadIdx.x == kEpiWarp0 * 32 && p.rq_tensor_scale != p.next_scale)
        *p.rq_tensor_scale = s_next;
    }
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int ct = cid; ct < num_ctiles; ct += ncl) {
      if (!mbar_wait(&tmem_full[acc], acc_phase, ctl)) break;
      tc_fence_after();
      const int nb = ct / groups_m;
      const int mb = (ct % groups_m) * kCM + rank;
      const int64_t row = (int64_t)mb * kBM + quarter * 32 + lane;
      const int64_t col0 = (int64_t)nb * kBN + half * kCols;
      uint32_t packed[kCols / 2];
      const uint32_t taddr =
          tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * kBN + half * kCols);
#pragma unroll
      for (int c2 = 0; c2 < kChunks; c2 += 2) {
        // two 32-column loads in flight per wait
        uint32_t r[2][32];
        tmem_ld32(taddr + c2 * 32, r[0]);
        tmem_ld32(taddr + c2 * 32 + 32, r[1]);
        tmem_ld_wait();
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int c = c2 + h;
          float a[32];
          if (kFp4) {
#pragma unroll
            for (int i = 0; i < 32; ++i) a[i] = alpha;
          } else {
            const int64_t n0 = col0 + c * 32;
            if (p.w_per_channel && n0 < p.N) {
              const float4* sw = reinterpret_cast<const float4*>(p.sdec_w + n0);
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const float4 v = __ldg(sw + i);
                a[4 * i] = __fmul_rn(sdec_a, v.x);
                a[4 * i + 1] = __fmul_rn(sdec_a, v.y);
                a[4 * i + 2] = __fmul_rn(sdec_a, v.z);
                a[4 * i + 3] = __fmul_rn(sdec_a, v.w);
              }
            } else {
              const float a0 = p.w_per_channel ? 0.0f : __fmul_rn(sdec_a, *p.sdec_w);
#pragma unroll
              for (int i = 0; i < 32; ++i) a[i] = a0;
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i)
            packed[c * 16 + i] =
                pack_bf16x2(__fmul_rn(__uint_as_float(r[h][2 * i]), a[2 * i]),
                            __fmul_rn(__uint_as_float(r[h][2 * i + 1]), a[2 * i + 1]));
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

      if (p.y != nullptr) {
        // bf16 output: each 32 x 32 box goes through a 64-byte-swizzled
        // staging buffer and one TMA store (rows >= M, cols >= N are clipped).
#pragma unroll
        for (int c = 0; c < kChunks; ++c) {
          uint8_t* const bufp = out_buf + (c & 1) * 2048;
          const uint32_t buf = smem_u32(bufp);
          if (lane == 0) bulk_wait_group_read<1>();   // this buffer's last store has read it
          __syncwarp();
#pragma unroll
          for (int k = 0; k < 4; ++k)
            st_shared_v4(buf + lane * 64 + ((k ^ ((lane >> 1) & 3)) << 4), packed[c * 16 + 4 * k],
                         packed[c * 16 + 4 * k + 1], packed[c * 16 + 4 * k + 2],
                         packed[c * 16 + 4 * k + 3]);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tmap_y, bufp, (int32_t)(col0 + c * 32), (int32_t)(row - lane));
            bulk_commit_group();
          }
        }
      }
      if (row < p.M) {
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
    if (lane == 0) bulk_wait_group_all();   // output stores complete before exit
  }

  // No CTA of the cluster may exit while a peer can still multicast into it
  // or arrive on its barriers.
  tc_fence_before();
  if (kCM > 1)
    cluster_sync();
  else
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

template <bool kFp4, int kBN, int kCM, bool kRequant>
cudaError_t launch_cfg(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                       uint64_t timeout_ns) {
  using C = Cfg<kFp4, kBN>;
  const uint64_t k_bytes = kFp4 ? (uint64_t)a.K / 2 : (uint64_t)a.K;
  CUtensorMap ta, tb, ty;
  std::memset(&ty, 0, sizeof ty);
  if (encode_tensor_map_2d_u8(&ta, a.a_codes, k_bytes, (uint64_t)a.M, kRowBytes, kBM) !=
          CUDA_SUCCESS ||
      encode_tensor_map_2d_u8(&tb, a.w_codes, k_bytes, (uint64_t)a.N, kRowBytes, kBN / kCM) !=
          CUDA_SUCCESS ||
      (a.y != nullptr && encode_tensor_map_out_bf16(&ty, a.y, (uint64_t)a.N, (uint64_t)a.M) !=
                             CUDA_SUCCESS))
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
  auto kern = gemm_kernel<kFp4, kBN, kCM, kRequant>;

  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCM;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;

  // one-time per instantiation: opt into the shared memory size and find how
  // many clusters fit at once (a persistent grid never exceeds that)
  static std::once_flag once;
  static cudaError_t setup_err = cudaSuccess;
  static int max_clusters = 0;
  std::call_once(once, [&] {
    setup_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     C::kSmemBytes);
    if (setup_err != cudaSuccess) return;
    cfg.gridDim = dim3((unsigned)(num_sms / kCM * kCM), 1, 1);
    setup_err = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
    if (setup_err == cudaSuccess && max_clusters < 1) setup_err = cudaErrorInvalidConfiguration;
  });
  if (setup_err != cudaSuccess) return setup_err;
  const int64_t tiles_m = (a.M + kBM - 1) / kBM;
  const int64_t ctiles = ((tiles_m + kCM - 1) / kCM) * ((a.N + kBN - 1) / kBN);
  const int clusters = (int)std::min<int64_t>(ctiles, std::min(max_clusters, num_sms / kCM));
  cfg.gridDim = dim3((unsigned)(clusters * kCM), 1, 1);
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, ty, p);
}

template <bool kFp4>
cudaError_t dispatch_bn(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                        uint64_t timeout_ns) {
  // 128 x 256 tiles in clusters of two along M (shared weight tile) when they
  // fill the machine, else 128 x 128 single-CTA tiles (small M).
  const int64_t tiles256 = ((a.M + kBM - 1) / kBM) * ((a.N + 255) / 256);
  const bool wide = tiles256 >= num_sms;
  if constexpr (kFp4) {
    if (a.next_scale != nullptr)
      return wide ? launch_cfg<true, 256, 2, true>(a, s, num_sms, err, timeout_ns)
                  : launch_cfg<true, 128, 1, true>(a, s, num_sms, err, timeout_ns);
  }
  return wide ? launch_cfg<kFp4, 256, 2, false>(a, s, num_sms, err, timeout_ns)
              : launch_cfg<kFp4, 128, 1, false>(a, s, num_sms, err, timeout_ns);
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

// bf16 [rows, cols] output map: 32 x 32 boxes, 64-byte swizzle (the layout of
// the epilogue's staging boxes).
CUresult encode_tensor_map_out_bf16(CUtensorMap* map, void* base, uint64_t cols, uint64_t rows) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return CUDA_ERROR_NOT_FOUND;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {32, 32};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
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
