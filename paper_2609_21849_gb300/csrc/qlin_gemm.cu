// Block-scaled GEMMs on the 5th-generation tensor cores (tcgen05) of sm_103a:
// the NVFP4 and FP8 linear layers of Sec. 4 ("Quantization": activation
// quantization lets the linears run on the FP8 / NVFP4 tensor cores), with a
// fused epilogue that writes the 16-bit output and, optionally, re-quantizes
// it for the next layer (NVFP4 or FP8) or reduces its tensor amax.  The same
// skeleton runs the unquantized bf16 / fp16 linears of Table 2's precision
// ladder (kind::f16).
//
// Two tile configurations share one kernel template:
//   pair   256 x 256 output tiles on a CTA pair (a cluster of two CTAs on two
//          SMs): one tcgen05 MMA of M = 256 (cta_group::2) issued by CTA 0
//          drives both SMs' tensor cores; each CTA holds its own 128 rows of A
//          and its own half of the W tile in shared memory.
//   single 128 x 128 tiles on one CTA, for small M (the translator's linears).
// Roles (one persistent CTA per SM; 12 warps, 15 for NVFP4 pair tiles):
//   warp 0      TMA producer: per pipeline stage one 4-D tensor copy per lane,
//               the A tile and the W tile as two row boxes each from four
//               lanes, as one instruction (and, except for NVFP4 pair tiles,
//               the A and W scale atoms from two more lanes).  In a pair,
//               CTA 1's copies complete on CTA 0's barriers (cta_group::2
//               form).
//   warp 1      TMEM allocation; MMA issue (per 32 bytes of K one tcgen05.mma:
//               NVFP4 kind::mxf4nvf4 scale_vec::4X with K = 64, FP8
//               kind::f8f6f4 with K = 32, bf16 / fp16 kind::f16 with K = 16)
//               into an fp32 TMEM accumulator.
//   warps 2..   NVFP4: block scales shared -> TMEM (tcgen05.cp), beside the
//               MMA stream (two warps, four for pair tiles), each warp the
//               atoms of an equal share of the stage's MMA steps.
//   next warp   NVFP4 pair tiles: TMA producer of the scale atoms.
//   last 8      epilogue: tcgen05.ld of the accumulator, alpha, 16-bit
//               rounding; pair tiles store y straight from registers (FP8 /
//               16-bit tiles use the freed staging memory for a seventh
//               stage), single-CTA tiles by TMA through swizzled staging;
//               optional re-quantization of the 16-bit values, one row per
//               thread, and optional output amax.
// Every wait is bounded (see WaitCtl).
#include <cstring>
#include <mutex>

#include "qlin_internal.h"

namespace qlin {

namespace {

constexpr int kBM = 128;
constexpr int kRowBytes = 128;      // bytes of K per stage and row: one swizzle row
constexpr int kStepsPerStage = 4;   // one MMA per 32 bytes of K
constexpr int kEpiWarps = 8;
// Build-time layout choices (the defaults measured fastest): scale-copy warps
// of NVFP4 pair tiles, a warp of its own for their scale boxes, and row boxes
// per operand tile and stage.
#ifndef QLIN_PAIR_CP_WARPS
#define QLIN_PAIR_CP_WARPS 4
#endif
#ifndef QLIN_SPLIT_SCALE_ISSUE
#define QLIN_SPLIT_SCALE_ISSUE 1
#endif
#ifndef QLIN_TMA_SPLIT
#define QLIN_TMA_SPLIT 2
#endif
// NVFP4 pair tiles store y straight from registers (no staging boxes and no
// TMA stores sharing the copy engine with the operand loads)
#ifndef QLIN_FP4_DIRECT_STORE
#define QLIN_FP4_DIRECT_STORE 1
#endif
// Tile order: cluster tiles are visited in groups of this many M tile groups
// (0: all of M, i.e. M fastest within each N tile; on the 4608 x 12288 x 3072
// NVFP4 GEMM groups of 1 to 9 measured 3-6% slower)
#ifndef QLIN_GROUP_M
#define QLIN_GROUP_M 0
#endif
constexpr int kSmemBudget = 232448 - 2048;  // opt-in shared memory minus barriers/alignment
constexpr int kSplit = QLIN_TMA_SPLIT;      // row boxes per operand tile and stage

constexpr int pow2_at_least(int x) {
  int p = 32;
  while (p < x) p <<= 1;
  return p;
}

// kPair: a CTA pair runs one tcgen05 MMA of M = 256 (cta_group::2); each CTA
// holds its own 128 rows of A and its own half of the W tile.
template <bool kFp4, int kBN, bool kPair = false>
struct Cfg {
  // warps: 0 producer, 1 MMA, then the scale-copy warps, then the epilogue
  // (an epilogue warp w reads TMEM lanes 32 (w % 4) and up, so any eight
  // consecutive warps cover the accumulator).  NVFP4 pair tiles need 12
  // scale copies per stage, shared between the scale-copy warps.
  static constexpr int kCpWarps = (kFp4 && kPair) ? QLIN_PAIR_CP_WARPS : 2;
  static_assert(kStepsPerStage % kCpWarps == 0, "each scale-copy warp takes whole MMA steps");
  // NVFP4 pair tiles: a warp of its own issues the scale boxes, so the
  // operand boxes' instruction has two lanes instead of four
  static constexpr int kScaleWarp = (kFp4 && kPair && QLIN_SPLIT_SCALE_ISSUE) ? 2 + kCpWarps : -1;
  static constexpr int kEpiWarp0 = 2 + kCpWarps + (kScaleWarp >= 0 ? 1 : 0);
  static constexpr int kThreads = (kEpiWarp0 + kEpiWarps) * 32;
  static constexpr int kSfbAtoms = kFp4 ? (kBN + 127) / 128 : 0;
  static constexpr int kABytes = kBM * kRowBytes;
  static constexpr int kBBytes = (kPair ? kBN / 2 : kBN) * kRowBytes;
  static constexpr int kSfaBytes = kFp4 ? kStepsPerStage * 512 : 0;
  static constexpr int kSfbBytes = kFp4 ? kSfbAtoms * kStepsPerStage * 512 : 0;
  static constexpr int kStageBytes = kABytes + kBBytes + kSfaBytes + kSfbBytes;
  // Pair tiles store y straight from registers (each thread its row's 64
  // bytes per 32 columns): for FP8 / 16-bit tiles the staging's shared memory
  // holds a seventh pipeline stage, and for NVFP4 tiles the operand loads
  // keep the copy engine to themselves (measured 70.1 -> 66.7 us on the
  // 4608 x 12288 x 3072 GEMM).  Otherwise per epilogue warp two 32 x 32 bf16
  // boxes (2 KB each) stage TMA stores.
  static constexpr bool kDirectStore = kPair && kBN == 256 && (!kFp4 || QLIN_FP4_DIRECT_STORE);
  static constexpr int kOutBytes = kDirectStore ? 0 : kEpiWarps * 2 * 2048;
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
  unsigned* y_amax;   // optional: max |bf16 y| over the output, as fp32 bits (atomicMax)
  unsigned* y_departures;   // with y_amax: CTAs done (the last one turns the amax into S_dec)
  float* y_sdec;            // with y_amax: where the last CTA writes S_dec = amax / 2688
  int fp16;           // 16-bit operand kernel only: fp16 operands and output (else bf16)
  int y_v8;           // y is 32-byte aligned: direct stores may use 32-byte vectors
  int rq_v8;          // the re-quantized codes are 32-byte aligned: one 32-byte store per group
  unsigned* err;
  uint64_t timeout_ns;
};

// Coordinates of cluster tile ct: its M tile group and its N tile.  Tiles are
// visited in groups of kGroup M tile groups (the last group may be smaller),
// M fastest within a group.
__device__ __forceinline__ void tile_coords(int ct, int groups_m, int tiles_n, int* mg, int* nb) {
  constexpr int kGroup = QLIN_GROUP_M;
  if (kGroup <= 0) {
    *nb = ct / groups_m;
    *mg = ct % groups_m;
    return;
  }
  const int per = kGroup * tiles_n;
  const int grp = ct / per;
  const int within = ct - grp * per;
  const int gm = min(kGroup, groups_m - grp * kGroup);
  *mg = grp * kGroup + within % gm;
  *nb = within / gm;
}

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

// 32-byte store (p 32-byte aligned): a whole L2 sector from one lane.
__device__ __forceinline__ void st_global_v8(void* p, const uint32_t* v) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(v[0]),
               "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
               : "memory");
}

// The same stores with an L2 cache-policy hint (createpolicy result).
__device__ __forceinline__ void st_global_v8_hint(void* p, const uint32_t* v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8}, %9;" ::"l"(
                   p),
               "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]),
               "r"(v[7]), "l"(pol)
               : "memory");
}
__device__ __forceinline__ void st_global_v4_hint(void* p, uint32_t a, uint32_t b, uint32_t c,
                                                  uint32_t d, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.v4.b32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "r"(a),
               "r"(b), "r"(c), "r"(d), "l"(pol)
               : "memory");
}

// kBf16 (with !kFp4): bf16 operands on the FP8 skeleton (the same 128-byte
// rows, 32 bytes of K per MMA), no scales.
template <bool kFp4, int kBN, bool kPair, bool kRequant, bool kBf16 = false>
__global__ void __launch_bounds__(Cfg<kFp4, kBN, kPair>::kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_a,
                const __grid_constant__ CUtensorMap tmap_b,
                const __grid_constant__ CUtensorMap tmap_sfa,
                const __grid_constant__ CUtensorMap tmap_sfb,
                const __grid_constant__ CUtensorMap tmap_y, const KParams p) {
  using C = Cfg<kFp4, kBN, kPair>;
  constexpr int kCM = kPair ? 2 : 1;          // CTAs per cluster (M tiles per cluster tile)
  constexpr uint16_t kMask = (uint16_t)((1u << kCM) - 1u);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* out_stage = smem + C::kStages * C::kStageBytes;   // epilogue staging boxes
  uint64_t* full = reinterpret_cast<uint64_t*>(out_stage + C::kOutBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* sf_full = empty + C::kStages;   // NVFP4: the stage's scale bytes landed
  uint64_t* tmem_full = sf_full + C::kStages;
  uint64_t* tmem_empty = tmem_full + 2;
  uint64_t* mma_done = tmem_empty + 2;
  uint64_t* sf_done = mma_done + 1;   // one barrier per scale-copy warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sf_done + C::kCpWarps);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = kPair ? (int)cluster_ctarank() : 0;
  const bool leader = rank == 0;   // a pair's MMA / scale-copy CTA

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      // NVFP4: the scale-copy warps' commits (one per warp) also arrive on
      // full, so the MMA issuer waits on one barrier per stage
      mbar_init(&full[s], kFp4 ? 1 + C::kCpWarps : 1);
      mbar_init(&empty[s], 1);
      mbar_init(&sf_full[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tmem_full[a], 1);
      mbar_init(&tmem_empty[a], kCM * kEpiWarps);   // every epilogue warp of the cluster
    }
    mbar_init(mma_done, 1);
    for (int w = 0; w < C::kCpWarps; ++w) mbar_init(&sf_done[w], 1);
    *abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 0 && lane < (kFp4 ? 4 : 2))
    prefetch_tmap(lane == 0 ? &tmap_a : lane == 1 ? &tmap_b : lane == 2 ? &tmap_sfa : &tmap_sfb);
  if (warp == 1) {
    if (kPair)
      tmem_alloc_pair(tmem_slot, C::kTmemCols);
    else
      tmem_alloc(tmem_slot, C::kTmemCols);
  }
  tc_fence_before();
  if (kPair)
    cluster_sync();   // the peer's barriers exist before any copy completes on them
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.err, p.timeout_ns};
  // the prologue above overlaps the previous kernel; global data only below
  grid_dep_wait();
  grid_dep_launch();

  const int tiles_m = (int)((p.M + kBM - 1) / kBM);
  const int tiles_n = (int)((p.N + kBN - 1) / kBN);
  const int groups_m = (tiles_m + kCM - 1) / kCM;
  const int num_ctiles = groups_m * tiles_n;
  const int cid = (int)blockIdx.x / kCM;
  const int ncl = (int)gridDim.x / kCM;
  const int64_t k_bytes = kFp4 ? p.K / 2 : kBf16 ? p.K * 2 : p.K;
  const int num_kb = (int)((k_bytes + kRowBytes - 1) / kRowBytes);
  const int k_steps = (int)(k_bytes / 32);

  if (warp == 0 || warp == C::kScaleWarp) {
    // ------------------------------------------------------ TMA producer ---
    // One 4-D tensor copy per lane (0: A tile, 1: W tile, 2: A scale atoms,
    // 3: W scale atoms), all four issued as ONE instruction: a TMA copy holds
    // its issuing thread for hundreds of cycles, so issuing them one by one
    // would starve the tensor cores.  Out-of-range boxes (rows past M or N, K
    // atoms past the end) are zero-filled and still count their full bytes,
    // so every stage expects the same byte counts.
    // Each operand tile is split into kSplit row boxes, one lane each, so
    // more copies run at once (lanes [0, kSplit): A parts, [kSplit, 2 kSplit):
    // W parts, then A scales, W scales): an SM's tensor copies fill shared
    // memory at ~15 B/cycle per issuing lane, up to ~72 B/cycle with six or
    // more lanes at once (measured), and a copy's rows split in two keep the
    // stage's bytes in more streams (4608 x 12288 x 3072 NVFP4: 64.5 -> 63.0
    // us; four boxes measured slower).
    // With a scale-issue warp, warp 0 takes the operand lanes and that warp
    // the two scale lanes; pl numbers the producer lanes across both.
    constexpr int kOpLanes = 2 * kSplit;
    const int pl = warp == 0 ? lane : kOpLanes + lane;
    const int nlanes = warp != 0 ? 2 : (kFp4 && C::kScaleWarp < 0) ? kOpLanes + 2 : kOpLanes;
    if (lane < nlanes) {
      const bool is_scale = pl >= kOpLanes;
      const int part = pl % kSplit;
      const CUtensorMap* map = pl < kSplit      ? &tmap_a
                               : pl < kOpLanes  ? &tmap_b
                               : pl == kOpLanes ? &tmap_sfa
                                                : &tmap_sfb;
      uint64_t* bars = is_scale ? sf_full : full;
      // barrier each copy completes on: this CTA's, or in a pair CTA 0's
      const uint32_t bar0 = kPair ? mapa_shared(bars, 0) : smem_u32(bars);
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      for (int ct = cid; ct < num_ctiles; ct += ncl) {
        int mg, nb;
        tile_coords(ct, groups_m, tiles_n, &mg, &nb);
        const int mb = mg * kCM + rank;
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, ctl)) {
            ok = false;
            break;
          }
          uint8_t* sA = smem + stage * C::kStageBytes;
          uint8_t* sB = sA + C::kABytes;
          uint8_t* sSF = sB + C::kBBytes;   // the stage's scale atoms: A's, then W's
          if (leader && pl == 0)
            mbar_arrive_expect_tx(&full[stage], kCM * (C::kABytes + C::kBBytes));
          if (kFp4 && leader && pl == kOpLanes)
            mbar_arrive_expect_tx(&sf_full[stage], kCM * (C::kSfaBytes + C::kSfbBytes));
          __syncwarp((1u << nlanes) - 1u);
          uint8_t* dst;
          int32_t c0, c1, c2, c3;
          constexpr int kARows = kBM / kSplit, kBRowsPart = kBN / kCM / kSplit;
          if (pl < kSplit) {                // A: part of this CTA's M tile
            dst = sA + part * kARows * kRowBytes;
            c0 = kb * kRowBytes; c1 = mb * kBM + part * kARows; c2 = 0; c3 = 0;
          } else if (pl < kOpLanes) {       // W: part of this CTA's rows of the N tile
            dst = sB + part * kBRowsPart * kRowBytes;
            c0 = kb * kRowBytes; c1 = nb * kBN + rank * (kBN / kCM) + part * kBRowsPart;
            c2 = 0; c3 = 0;
          } else if (pl == kOpLanes) {      // A scale atoms of this stage
            dst = sSF; c0 = kb * kStepsPerStage * 64; c1 = mb; c2 = 0; c3 = 0;
          } else {                          // W scale atoms (all atom rows of the N tile)
            dst = sSF + C::kSfaBytes; c0 = kb * kStepsPerStage * 64;
            c1 = (nb * kBN) >> 7; c2 = 0; c3 = 0;   // first 128-row atom of the N tile
          }
          const uint32_t bar = bar0 + (uint32_t)(stage * 8);
          if (kPair)
            tma_load_4d_pair(dst, map, bar, c0, c1, c2, c3);
          else
            tma_load_4d(dst, map, bar, c0, c1, c2, c3);
          ++issued;
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      // Let the last copies into this CTA land before it exits (the barriers
      // that count them live in CTA 0; its producer drains them).
      if (leader && (pl == 0 || (kFp4 && pl == kOpLanes))) {
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
    if (lane == 0 && leader) {
      constexpr int kMmaM = kPair ? 256 : 128;
      const uint32_t idesc = kFp4    ? idesc_nvfp4(kBN, kMmaM)
                             : kBf16 ? (p.fp16 ? idesc_fp16(kBN, kMmaM) : idesc_bf16(kBN, kMmaM))
                                     : idesc_fp8(kBN, kMmaM);
      // A stage is ready for its MMAs once its operands have landed and, for
      // NVFP4, its scales are in TMEM (one barrier counts both).
      auto wait_ready = [&](int st, uint32_t ph) { return mbar_wait(&full[st], ph, ctl); };
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int ct = cid; ct < num_ctiles && ok; ct += ncl) {
        // 64-wide tiles use one half of a 128-row W scale atom: its rows
        // 32 w + lane sit in TMEM column w, so the odd tile's half starts two
        // columns in
        int mg_, nb_;
        tile_coords(ct, groups_m, tiles_n, &mg_, &nb_);
        const uint32_t sfb_off = kBN < 128 ? 2u * (uint32_t)(nb_ & 1) : 0u;
        if (!mbar_wait(&tmem_empty[acc], acc_phase ^ 1u, ctl)) break;
        if (!wait_ready(stage, phase)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kBN);
        for (int kb = 0; kb < num_kb; ++kb) {
          const uint32_t sA = smem_u32(smem + stage * C::kStageBytes);
          const uint32_t sB = sA + C::kABytes;
          const int nsteps = min(kStepsPerStage, k_steps - kb * kStepsPerStage);
          // step j's operands start 32 j bytes in: the descriptors' start
          // address field (address / 16, 14 bits; shared addresses stay
          // below 256 KB, so it never carries) advances by 2 j
          const uint64_t adesc0 = sdesc_k128(sA), bdesc0 = sdesc_k128(sB);
          const uint32_t sfa0 = tmem_base + (uint32_t)(C::kSfColBase + stage * kStepsPerStage *
                                                                           C::kSfColsPerStep);
          auto issue = [&](int j, uint32_t accumulate) {
            const uint64_t adesc = adesc0 + (uint64_t)(2 * j);
            const uint64_t bdesc = bdesc0 + (uint64_t)(2 * j);
            if (kFp4) {
              const uint32_t sfa_t = sfa0 + (uint32_t)(j * C::kSfColsPerStep);
              if (kPair)
                mma_nvfp4_pair(d_tmem, adesc, bdesc, idesc, sfa_t, sfa_t + 4, accumulate);
              else
                mma_nvfp4(d_tmem, adesc, bdesc, idesc, sfa_t, sfa_t + 4 + sfb_off, accumulate);
            } else if (kBf16) {
              if (kPair)
                mma_bf16_pair(d_tmem, adesc, bdesc, idesc, accumulate);
              else
                mma_bf16(d_tmem, adesc, bdesc, idesc, accumulate);
            } else {
              if (kPair)
                mma_fp8_pair(d_tmem, adesc, bdesc, idesc, accumulate);
              else
                mma_fp8(d_tmem, adesc, bdesc, idesc, accumulate);
            }
          };
          // Full stages issue their MMAs unrolled, with no branch between
          // them: a runtime step loop around the MMA issue costs ~100 cycles
          // a stage (measured), a fifth of the stage's tensor work.  Only a
          // partial last stage (K % 256 != 0) takes the loop.
          if (nsteps == kStepsPerStage) {
            issue(0, kb > 0 ? 1u : 0u);
#pragma unroll
            for (int jj = 1; jj < kStepsPerStage; ++jj) issue(jj, 1u);
          } else {
            for (int jj = 0; jj < nsteps; ++jj) issue(jj, (jj > 0 || kb > 0) ? 1u : 0u);
          }
          // The stage is free once the MMAs have read it (both CTAs' halves).
          // The release comes right after the stage's last MMA: deferring it
          // under the next stage's first MMA (to shorten the gap between
          // issues) measured slower, the load pipeline being the bound.
          if (kPair)
            tc_commit_pair_mc(&empty[stage], kMask);
          else
            tc_commit(&empty[stage]);
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
          // the tile's next stage: one barrier test per stage (the scale
          // copies arrive on the same barrier as the operands; a second
          // barrier's test cost ~100 cycles a stage in shared memory this
          // busy, the MMA queue holding about one instruction)
          if (kb + 1 < num_kb) {
            if (!wait_ready(stage, phase)) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
        }
        if (!ok) break;
        if (kPair)
          tc_commit_pair_mc(&tmem_full[acc], kMask);   // both CTAs' epilogues
        else
          tc_commit(&tmem_full[acc]);
        if (C::kNumAcc == 2) {
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1u;
        } else {
          acc_phase ^= 1u;
        }
      }
      // Every MMA / scale copy issued must finish before TMEM is released.
      if (kPair)
        tc_commit_pair_mc(mma_done, 1);
      else
        tc_commit(mma_done);
      mbar_drain(mma_done, 0, p.timeout_ns, p.err);
    }
  } else if (warp < C::kEpiWarp0) {
    // --------------------------------------------- NVFP4 scale copies ---
    // Block scales move shared -> TMEM from threads of their own (one lane of
    // each scale-copy warp), beside the MMA stream: a tcgen05.cp occupies its
    // issuing thread ~80-120 cycles while the MMAs run, and a stage needs 12
    // (pair tiles), so each warp copies the atoms of an equal share of the
    // stage's MMA steps.  Copies issued from separate warps overlap (12 take
    // ~850 cycles from two warps, ~510 from four, with the MMAs running: the
    // MMAs' rate is unaffected), so pair tiles use four.  (A converged
    // instruction from several lanes of one warp does not issue one copy per
    // lane.)  In a pair, CTA 0's copies fill both SMs' TMEM from their own
    // shared memory.
    if (kFp4 && lane == 0 && leader) {
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
          // each warp copies all atoms (A, then each W atom row) of its share
          // of the stage's MMA steps
          constexpr int kShare = kStepsPerStage / C::kCpWarps;
          const int j_end = min(nsteps, (sw + 1) * kShare);
          for (int j = sw * kShare; j < j_end; ++j) {
            const uint32_t sfa_t = tmem_base + (uint32_t)(C::kSfColBase +
                                                          (stage * kStepsPerStage + j) *
                                                              C::kSfColsPerStep);
            if (kPair)
              tc_cp_scales_pair(sfa_t, sdesc_scales(sSFA + j * 512));
            else
              tc_cp_scales(sfa_t, sdesc_scales(sSFA + j * 512));
#pragma unroll
            for (int r = 0; r < C::kSfbAtoms; ++r) {
              const uint32_t src = sSFB + r * kStepsPerStage * 512 + j * 512;
              if (kPair)
                tc_cp_scales_pair(sfa_t + 4 + 4 * r, sdesc_scales(src));
              else
                tc_cp_scales(sfa_t + 4 + 4 * r, sdesc_scales(src));
            }
          }
          // the stage is ready for its MMAs once these copies and its
          // operands have landed: both arrive on its full barrier.  (Its
          // previous phase has completed: the scale boxes of this stage were
          // issued after the MMAs of the stage that last used it.)
          if (kPair)
            tc_commit_pair_mc(&full[stage], 1);
          else
            tc_commit(&full[stage]);
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      if (kPair)
        tc_commit_pair_mc(&sf_done[sw], 1);
      else
        tc_commit(&sf_done[sw]);
      mbar_drain(&sf_done[sw], 0, p.timeout_ns, p.err);
    }
  } else {
    // --------------------------------------------------------- epilogue ---
    constexpr int kCols = kBN / 2;  // columns per thread
    constexpr int kChunks = kCols / 32;
    const int e = warp - C::kEpiWarp0;
    const int quarter = warp & 3;   // the TMEM lane quarter this warp may access
    const int half = e >> 2;
    const float sdec_a = kBf16 ? 1.0f : *p.sdec_a;
    const float alpha = kFp4 ? __fmul_rn(sdec_a, *p.sdec_w) : kBf16 ? 1.0f : 0.0f;
    float s_enc_next = 0.0f;
    if (kRequant) {
      const float s_next = *p.next_scale;
      s_enc_next = encode_scale(s_next);
      if (blockIdx.x == 0 && threadIdx.x == C::kEpiWarp0 * 32 && p.rq_tensor_scale != p.next_scale)
        *p.rq_tensor_scale = s_next;
    }
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int ct = cid; ct < num_ctiles; ct += ncl) {
      int mg, nb;
      tile_coords(ct, groups_m, tiles_n, &mg, &nb);
      if (!kFp4 && !kBf16 && p.w_per_channel) {
        // FP8: this tile's per-channel weight scales into L1 while the
        // accumulator is still being computed (lane i: the 128-byte line of
        // chunk i), so that the epilogue's loads of them wait on L1 rather
        // than L2 -- the last tile's epilogue is on the kernel's critical path
        const int64_t cl = (int64_t)nb * kBN + half * kCols + 32 * lane;
        if (lane < kCols / 32 && cl < p.N)
          asm volatile("prefetch.global.L1 [%0];" ::"l"(p.sdec_w + cl));
      }
      if (!mbar_wait(&tmem_full[acc], acc_phase, ctl)) break;
      tc_fence_after();
      const int mb = mg * kCM + rank;
      const int64_t row = (int64_t)mb * kBM + quarter * 32 + lane;
      // chunk c (32 columns) of this thread starts at column ccol(c)
      const int64_t col0 = (int64_t)nb * kBN + half * kCols;
      auto ccol = [&](int c) -> int64_t { return col0 + c * 32; };
      uint32_t packed[kCols / 2];
      const uint32_t taddr =
          tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * kBN + half * kCols);
      // Accumulator columns in batches of tcgen05.ld per wait; TMEM goes back
      // to the MMA issuer right after the last batch has landed in registers.
      // With a single accumulator the next tile's MMAs wait for that, so all
      // columns form one batch where the register budget (168 a thread at
      // 12 warps, 128 above) allows.
      constexpr int kBatch =
          (C::kNumAcc == 1 && C::kThreads <= 384) ? kChunks : (kChunks < 2 ? kChunks : 2);
      static_assert(kChunks % kBatch == 0, "TMEM is released after the last batch");
#pragma unroll
      for (int cb = 0; cb < kChunks; cb += kBatch) {
        uint32_t r[kBatch][32];
#pragma unroll
        for (int b = 0; b < kBatch; ++b) tmem_ld32(taddr + (cb + b) * 32, r[b]);
        tmem_ld_wait();
        if (cb + kBatch == kChunks) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (kPair && rank == 1)
              mbar_arrive_cluster(mapa_shared(&tmem_empty[acc], 0));   // CTA 0 owns the MMA
            else
              mbar_arrive(&tmem_empty[acc]);
          }
          if (C::kNumAcc == 2) {
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1u;
          } else {
            acc_phase ^= 1u;
          }
        }
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
          const int c = cb + b;
          float a[32];
          if (kFp4 || kBf16) {
#pragma unroll
            for (int i = 0; i < 32; ++i) a[i] = alpha;
          } else {
            const int64_t n0 = ccol(c);
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
          if (kBf16 && p.fp16) {
#pragma unroll
            for (int i = 0; i < 16; ++i)
              packed[c * 16 + i] = pack_f16x2(__uint_as_float(r[b][2 * i]),
                                              __uint_as_float(r[b][2 * i + 1]));
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
              packed[c * 16 + i] =
                  pack_bf16x2(__fmul_rn(__uint_as_float(r[b][2 * i]), a[2 * i]),
                              __fmul_rn(__uint_as_float(r[b][2 * i + 1]), a[2 * i + 1]));
          }
        }
      }

      if (p.y_amax != nullptr) {
        // the output's tensor amax (for a dynamic scale of the next layer's
        // input): max over this thread's bf16 values, then the warp, then
        // one atomic per warp.  Rows past M and columns past N hold zeros
        // (zero-filled operands), which leave the maximum unchanged.
        uint32_t m = 0;
#pragma unroll
        for (int i = 0; i < kCols / 2; ++i) m = __vmaxu2(m, packed[i] & 0x7FFF7FFFu);
        m = max(m & 0xFFFFu, m >> 16);
        m = __reduce_max_sync(0xFFFFFFFFu, m);
        if (lane == 0 && m != 0u) atomicMax(p.y_amax, m << 16);
      }
      if constexpr (C::kDirectStore) {
        // 16-bit output straight from registers: the thread's row, 32
        // columns (64 bytes) per chunk; N % 64 == 0, so a chunk is wholly
        // inside or outside the matrix
        if (p.y != nullptr && row < p.M) {
          uint16_t* const yrow = p.y + row * p.N;
          // With an output amax (the dynamic chain), y is read back right
          // after this kernel by the quantizer: keep it in L2 if it can.
          const bool keep = p.y_amax != nullptr;
          const uint64_t pol = keep ? policy_evict_last() : 0ull;
#pragma unroll
          for (int c = 0; c < kChunks; ++c) {
            if (ccol(c) >= p.N) continue;
            uint32_t* const dst = reinterpret_cast<uint32_t*>(yrow + ccol(c));
            if (p.y_v8) {
              if (keep) {
                st_global_v8_hint(dst, &packed[c * 16], pol);
                st_global_v8_hint(dst + 8, &packed[c * 16 + 8], pol);
              } else {
                st_global_v8(dst, &packed[c * 16]);
                st_global_v8(dst + 8, &packed[c * 16 + 8]);
              }
            } else {
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                if (keep)
                  st_global_v4_hint(dst + 4 * k, packed[c * 16 + 4 * k], packed[c * 16 + 4 * k + 1],
                                    packed[c * 16 + 4 * k + 2], packed[c * 16 + 4 * k + 3], pol);
                else
                  st_global_v4(dst + 4 * k, packed[c * 16 + 4 * k], packed[c * 16 + 4 * k + 1],
                               packed[c * 16 + 4 * k + 2], packed[c * 16 + 4 * k + 3]);
              }
            }
          }
        }
      } else if (p.y != nullptr) {
        // bf16 output: each 32 x 32 box goes through a 64-byte-swizzled
        // staging buffer and one TMA store (rows >= M, cols >= N are clipped).
        uint8_t* const out_buf = out_stage + e * 4096;   // this warp's two staging boxes
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
            tma_store_2d(&tmap_y, bufp, (int32_t)ccol(c), (int32_t)(row - lane));
            bulk_commit_group();
          }
        }
      }
      if (row < p.M) {
        if (kRequant && !kFp4) {
          // FP8 re-quantization with the static next-layer scale: E4M3 of
          // bf16(y) * S_enc per element, 64 columns per group
#pragma unroll
          for (int g = 0; g < kCols / 64; ++g) {
            const int64_t c64 = ccol(2 * g);   // chunks 2g, 2g + 1: 64 contiguous columns
            if (c64 < p.rq_col0 || c64 + 64 > p.rq_col0 + p.rq_cols || c64 >= p.N) continue;
            uint8_t* cp = p.rq_codes + row * p.rq_cols + (c64 - p.rq_col0);
#pragma unroll
            for (int q2 = 0; q2 < 2; ++q2) {   // 32 columns per 32-byte store (or two 16-byte)
              uint32_t w8[8];
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const uint32_t* pk = packed + g * 32 + (2 * q2 + h) * 8;
#pragma unroll
                for (int i = 0; i < 4; ++i)
                  w8[4 * h + i] = e4m3x4(__fmul_rn(bf16_lo(pk[2 * i]), s_enc_next),
                                         __fmul_rn(bf16_hi(pk[2 * i]), s_enc_next),
                                         __fmul_rn(bf16_lo(pk[2 * i + 1]), s_enc_next),
                                         __fmul_rn(bf16_hi(pk[2 * i + 1]), s_enc_next));
              }
              if (p.rq_v8) {
                st_global_v8(cp + 32 * q2, w8);
              } else {
                st_global_v4(cp + 32 * q2, w8[0], w8[1], w8[2], w8[3]);
                st_global_v4(cp + 32 * q2 + 16, w8[4], w8[5], w8[6], w8[7]);
              }
            }
          }
        }
        if (kRequant && kFp4) {
#pragma unroll
          for (int g = 0; g < kCols / 64; ++g) {
            const int64_t c64 = ccol(2 * g);   // chunks 2g, 2g + 1: 64 contiguous columns
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
                  f[2 * i] = bf16_lo(pk[h8 * 4 + i]);
                  f[2 * i + 1] = bf16_hi(pk[h8 * 4 + i]);
                  mul2_rn(f[2 * i], f[2 * i + 1], r_b);
                }
                words[b * 2 + h8] = e2m1x8(f);
              }
            }
            uint8_t* cp = p.rq_codes + row * (p.rq_cols / 2) + lc / 2;
            // the group's 32 bytes of codes: one store where aligned (each
            // store instruction of the epilogue slows the mainloop beside it)
            if (p.rq_v8) {
              st_global_v8(cp, words);
            } else {
              st_global_v4(cp, words[0], words[1], words[2], words[3]);
              st_global_v4(cp + 16, words[4], words[5], words[6], words[7]);
            }
            *reinterpret_cast<uint32_t*>(p.rq_scales + scale_offset(row, lc / 16, p.rq_cols)) = sw;
          }
        }
      }
    }
    // The staging buffers must have been read out before the CTA exits; the
    // stores' global writes complete with the grid (as for any store), so
    // the CTA does not wait for them.
    if (lane == 0) bulk_wait_group_read<0>();
    if (p.y_amax != nullptr) {
      // The output's tensor scale: once every epilogue warp of the CTA has
      // added its maxima, the CTA departs; the last CTA of the grid to depart
      // turns the amax into S_dec = amax / (6 * 448) (1 for an all-zero
      // output), writes it where the quantizer of y reads its scale, and
      // resets both scratch words for the next call (so no clearing node
      // precedes the kernel).
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
      if (threadIdx.x == C::kEpiWarp0 * 32) {
        __threadfence();
        if (atomicAdd(p.y_departures, 1u) == gridDim.x - 1) {
          __threadfence();
          const unsigned bits = atomicExch(p.y_amax, 0u);
          const float amax = __uint_as_float(bits);
          *p.y_sdec = bits == 0u ? 1.0f : __fdiv_rn(amax, 2688.0f);
          atomicExch(p.y_departures, 0u);
        }
      }
    }
  }

  // No CTA of the cluster may exit while a peer can still multicast into it
  // or arrive on its barriers.  Each warp reconverges first: the cluster
  // barrier is a warp-aligned instruction, and most roles run on one lane.
  __syncwarp();
  tc_fence_before();
  if (kPair)
    cluster_sync();
  else
    __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (kPair)
      tmem_dealloc_pair(tmem_base, C::kTmemCols);
    else
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

// 4-D tensor map (dims innermost first, in elements; strides in bytes for
// dims 1-3).
CUresult encode_4d(CUtensorMap* map, CUtensorMapDataType type, const void* base,
                   const cuuint64_t (&dims)[4], const cuuint64_t (&strides)[3],
                   const cuuint32_t (&box)[4], CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return CUDA_ERROR_NOT_FOUND;
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, type, 4, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Codes [rows, k_bytes] (row stride row_stride bytes, 0 = packed) as a 4-D
// tensor with two unit dimensions, 128-byte x box_rows boxes with the
// 128-byte swizzle.
CUresult encode_codes(CUtensorMap* map, const void* base, uint64_t k_bytes, uint64_t rows,
                      uint32_t box_rows, uint64_t row_stride = 0) {
  const uint64_t st = row_stride ? row_stride : k_bytes;
  const cuuint64_t dims[4] = {k_bytes, rows, 1, 1};
  const cuuint64_t strides[3] = {st, st * rows, st * rows};
  const cuuint32_t box[4] = {kRowBytes, box_rows, 1, 1};
  return encode_4d(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, base, dims, strides, box,
                   CU_TENSOR_MAP_SWIZZLE_128B);
}

// Swizzled block scales: the atoms of one 128-row block are contiguous along
// K (512 bytes per 64 elements of K), so the scales are a [row blocks, K]
// tensor of 8-byte words.  A box of {256 words, n row blocks} is the four
// atoms of one pipeline stage for n row blocks (2 KB each, 16 rows of 128
// bytes per request stream instead of 128 of 16 bytes), laid out in shared
// memory exactly as in global memory.
CUresult encode_scales(CUtensorMap* map, const void* base, uint64_t rows, uint64_t K,
                       uint32_t row_blocks_per_box) {
  const cuuint64_t dims[4] = {K, (rows + 127) / 128, 1, 1};
  const cuuint64_t strides[3] = {K * 8, K * 8 * dims[1], K * 8 * dims[1]};
  const cuuint32_t box[4] = {(cuuint32_t)(kStepsPerStage * 64), row_blocks_per_box, 1, 1};
  return encode_4d(map, CU_TENSOR_MAP_DATA_TYPE_UINT64, base, dims, strides, box,
                   CU_TENSOR_MAP_SWIZZLE_NONE);
}

template <bool kFp4, int kBN, bool kPair, bool kRequant, bool kBf16 = false>
cudaError_t launch_cfg(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                       uint64_t timeout_ns) {
  using C = Cfg<kFp4, kBN, kPair>;
  constexpr int kCM = kPair ? 2 : 1;
  const uint64_t k_bytes = kFp4 ? (uint64_t)a.K / 2 : kBf16 ? (uint64_t)a.K * 2 : (uint64_t)a.K;
  CUtensorMap ta, tb, tsa, tsb, ty;
  std::memset(&tsa, 0, sizeof tsa);
  std::memset(&tsb, 0, sizeof tsb);
  std::memset(&ty, 0, sizeof ty);
  if (encode_codes(&ta, a.a_codes, k_bytes, (uint64_t)a.M, kBM / kSplit,
                   (uint64_t)a.a_row_bytes) != CUDA_SUCCESS ||
      encode_codes(&tb, a.w_codes, k_bytes, (uint64_t)a.N, kBN / kCM / kSplit) != CUDA_SUCCESS ||
      (kFp4 && (encode_scales(&tsa, a.sfa, (uint64_t)a.M, (uint64_t)a.K, 1) != CUDA_SUCCESS ||
                encode_scales(&tsb, a.sfb, (uint64_t)a.N, (uint64_t)a.K, C::kSfbAtoms) !=
                    CUDA_SUCCESS)) ||
      (a.y != nullptr &&
       encode_tensor_map_out_bf16(&ty, a.y, (uint64_t)a.N, (uint64_t)a.M, kBf16 && a.fp16) !=
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
  p.y_amax = a.y_amax;
  p.y_departures = a.y_departures;
  p.y_sdec = a.y_sdec;
  p.fp16 = kBf16 && a.fp16 ? 1 : 0;
  p.y_v8 = (reinterpret_cast<uintptr_t>(a.y) & 31u) == 0 ? 1 : 0;
  p.rq_v8 = (reinterpret_cast<uintptr_t>(a.rq_codes) & 31u) == 0 ? 1 : 0;
  p.err = err;
  p.timeout_ns = timeout_ns;
  auto kern = gemm_kernel<kFp4, kBN, kPair, kRequant, kBf16>;

  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCM;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(C::kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;   // the occupancy query below takes the cluster attribute only

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
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, tsa, tsb, ty, p);
}

template <bool kFp4>
cudaError_t dispatch_bn(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                        uint64_t timeout_ns) {
  // 256 x 256 tiles on CTA pairs when they fill the machine, else 128 x 128
  // single-CTA tiles (small M), or 128 x 64 when 128 x 128 tiles would leave
  // at least half the SMs idle (no fused re-quantization: its 64-column
  // groups need 128-column tiles).
  const int64_t tiles_m = (a.M + kBM - 1) / kBM;
  const bool wide = tiles_m * ((a.N + 255) / 256) >= num_sms;
  if (a.next_scale != nullptr) {
    return wide ? launch_cfg<kFp4, 256, true, true>(a, s, num_sms, err, timeout_ns)
                : launch_cfg<kFp4, 128, false, true>(a, s, num_sms, err, timeout_ns);
  }
  if (wide) return launch_cfg<kFp4, 256, true, false>(a, s, num_sms, err, timeout_ns);
  const bool narrow = 2 * tiles_m * ((a.N + 127) / 128) <= num_sms;
  return narrow ? launch_cfg<kFp4, 64, false, false>(a, s, num_sms, err, timeout_ns)
                : launch_cfg<kFp4, 128, false, false>(a, s, num_sms, err, timeout_ns);
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

// bf16 (or fp16) [rows, cols] output map: 32 x 32 boxes, 64-byte swizzle (the
// layout of the epilogue's staging boxes).
CUresult encode_tensor_map_out_bf16(CUtensorMap* map, void* base, uint64_t cols, uint64_t rows,
                                    bool fp16) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return CUDA_ERROR_NOT_FOUND;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {32, 32};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, fp16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
            base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

cudaError_t launch_gemm(const GemmArgs& a, cudaStream_t s, int num_sms, unsigned* err,
                        uint64_t timeout_ns) {
  if (a.bf16) {
    const int64_t tiles256 = ((a.M + kBM - 1) / kBM) * ((a.N + 255) / 256);
    return tiles256 >= num_sms
               ? launch_cfg<false, 256, true, false, true>(a, s, num_sms, err, timeout_ns)
               : launch_cfg<false, 128, false, false, true>(a, s, num_sms, err, timeout_ns);
  }
  return a.fp4 ? dispatch_bn<true>(a, s, num_sms, err, timeout_ns)
               : dispatch_bn<false>(a, s, num_sms, err, timeout_ns);
}

cudaError_t launch_wait_selftest(uint64_t timeout_ns, cudaStream_t s, unsigned* err) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(err, timeout_ns);
  return cudaGetLastError();
}

}  // namespace qlin
