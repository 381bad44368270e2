// Activation and weight quantizers (Sec. 4, "Quantization": FP8 / NVFP4
// post-training quantization; activations are quantized at run time, weights
// once).  All kernels here are HBM-bandwidth bound streaming kernels:
//
//   onepass_kernel<Op>    dynamic scale in one read of x: the grid holds x in
//                         shared memory, reduces amax across the grid, then
//                         quantizes from shared memory (when x fits on chip)
//   amax_kernel           max |x| over a tensor (the dynamic tensor scale)
//   quant_kernel<NVFP4>   bf16 -> packed e2m1 codes + E4M3 block scales in the
//                         tensor-core scale layout + FP32 tensor scale
//   quant_kernel<FP8>     bf16 -> E4M3 codes with one tensor scale
//   quant_fp8_rows_kernel bf16 weights -> E4M3 codes with one scale per row
//
// Streaming structure: the [M, K] input is a flat array of 16-byte chunks (8
// bf16), cut into 16 KB tiles.  A persistent grid (three CTAs per SM)
// streams tiles through a four-deep shared-memory ring filled by bulk copies,
// so ~192 KB per SM of input is in flight regardless of register pressure.
// Inside a tile, each thread takes consecutive units of chunks (NVFP4: one
// 16-element block per lane, so four neighbouring lanes hold one 64-element
// group, whose four block scales form one 32-bit word of the scale layout;
// because K % 64 == 0 a group never straddles a row).
#include "qlin_internal.h"

namespace qlin {

namespace {

constexpr int kThreads = 512;
constexpr int kTileChunks = 1024;             // 16 KB of input per tile
constexpr int kStages = 4;
constexpr int kSmem = kStages * kTileChunks * 16 + 64;
constexpr int kBlocksPerSm = 3;

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

__device__ __forceinline__ uint4 lds128(const uint4* p) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(smem_u32(p)));
  return v;
}

// The per-tile work of each kernel (called by every thread for each tile).
struct AmaxOp {
  static constexpr int kUnit = 1;   // chunks per thread and call
  uint32_t m = 0;
  __device__ __forceinline__ void bind(float*) {}
  __device__ __forceinline__ void init() {}
  __device__ __forceinline__ void unit(const uint4 (&v)[1], uint64_t, bool valid) {
    if (valid) m = max(m, chunk_abs_max_bits(v[0]));
  }
};

// One lane per 16-element block (two chunks); each lane stores its block's
// scale code as one byte of the atom layout (one store instruction per warp,
// instead of gathering a 64-element group's four codes by shuffles: measured
// 2-7% faster).  r_b = S_enc / s_b comes from a per-CTA table over the 127
// finite E4M3 codes, filled with the same fp32 division.
template <typename Idx>
struct Nvfp4Op {
  static constexpr int kUnit = 2;
  static constexpr bool kBlockMax = true;   // the one-read kernel keeps block maxima
  float s_enc;
  Idx chunks_per_row;
  // row = chunk / chunks_per_row without a division (32-bit indices):
  // t = umulhi(div_m, c), row = (t + ((c - t) >> div_s1)) >> div_s2
  // (Granlund and Montgomery, PLDI 1994, division by invariant integers)
  uint32_t div_m, div_s1, div_s2;
  int64_t K;
  uint32_t* codes;
  uint8_t* scales;
  float* r_table;   // shared memory, 128 entries
  __device__ __forceinline__ void bind(float* table) { r_table = table; }
  __device__ __forceinline__ void init() {
    if (threadIdx.x < 128) {
      const uint32_t c = threadIdx.x;
      r_table[c] = (c == 0u) ? 0.0f : __fdiv_rn(s_enc, e4m3_value(c));
    }
  }
  // The codes of one 16-element block (block amax bits mb) and its scale
  // code (in `word`).
  __device__ __forceinline__ void quantize_block(const uint4 (&v)[2], uint32_t mb,
                                                 uint32_t& code0, uint32_t& code1,
                                                 uint32_t& word) const {
    const float t = __fmul_rn(__uint_as_float(mb << 16), s_enc);
    const uint32_t sb = e4m3_code_div6(t);
    const float r_b = r_table[sb];
    float f[8];
    unpack8(v[0], f);
#pragma unroll
    for (int i = 0; i < 8; i += 2) mul2_rn(f[i], f[i + 1], r_b);
    code0 = e2m1x8(f);
    unpack8(v[1], f);
#pragma unroll
    for (int i = 0; i < 8; i += 2) mul2_rn(f[i], f[i + 1], r_b);
    code1 = e2m1x8(f);
    word = sb;
  }
  __device__ __forceinline__ void unit(const uint4 (&v)[2], uint64_t c, bool valid) {
    uint32_t code0, code1, word;
    quantize_block(v, max(chunk_abs_max_bits(v[0]), chunk_abs_max_bits(v[1])), code0, code1,
                   word);
    if (valid) {
      reinterpret_cast<uint2*>(codes)[c >> 1] = make_uint2(code0, code1);
      {
        if constexpr (sizeof(Idx) == 4) {
          const uint32_t ci = (uint32_t)c;
          const uint32_t t = __umulhi(div_m, ci);
          const uint32_t row = (t + ((ci - t) >> div_s1)) >> div_s2;
          const uint32_t colc = ci - row * (uint32_t)chunks_per_row;   // in chunks
          scales[((row >> 7) * (uint32_t)(K >> 6) + (colc >> 3)) * 512u +
                 (row & 31u) * 16u + ((row >> 5) & 3u) * 4u + ((colc >> 1) & 3u)] = (uint8_t)word;
        } else {
          const Idx ci = (Idx)c;
          const Idx row = ci / chunks_per_row;
          const Idx col = (ci - row * chunks_per_row) << 3;
          scales[scale_offset((int64_t)row, (int64_t)(col >> 4), K)] = (uint8_t)word;
        }
      }
    }
  }
  // A slice of n chunks held in shared memory, global chunks [c0, c0 + n)
  // (c0 and n multiples of 8): each thread takes units of two chunks at a
  // stride of the block, two units per step for instruction-level
  // parallelism, and tracks its row and column without dividing.  The
  // block amax bits of step s's two units are bm[s] (low, high halves), as
  // gathered by block_max_pass.
  template <int kThreadsPerBlock, int kSteps>
  __device__ __forceinline__ void run_slice(const uint4* buf, uint32_t n, uint64_t c0,
                                            const uint32_t (&bm)[kSteps]) const {
    constexpr uint32_t kStride = 2u * kThreadsPerBlock;          // chunks per step and unit
    const uint32_t cpr = (uint32_t)chunks_per_row;
    const uint32_t dq = (2u * kStride) / cpr, dr = (2u * kStride) % cpr;
    const uint32_t kq = kStride / cpr, kr = kStride % cpr;
    const uint64_t cg = c0 + 2u * threadIdx.x;
    uint32_t row = (uint32_t)(cg / cpr), col = (uint32_t)(cg % cpr);   // col in chunks
    const uint32_t kgroups = (uint32_t)(K >> 6);
    // the loop bound is block-uniform
#pragma unroll
    for (int s = 0; s < kSteps; ++s) {
      const uint32_t base = (uint32_t)s * 2u * kStride;
      if (base >= n) break;
      const uint32_t cl = base + 2u * threadIdx.x;
      uint4 va[2], vb[2];
      const bool ok_a = cl < n, ok_b = cl + kStride < n;   // units never straddle n
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        va[k] = ok_a ? lds128(buf + cl + k) : make_uint4(0u, 0u, 0u, 0u);
        vb[k] = ok_b ? lds128(buf + cl + kStride + k) : make_uint4(0u, 0u, 0u, 0u);
      }
      uint32_t a0, a1, aw, b0, b1, bw;
      quantize_block(va, bm[s] & 0xFFFFu, a0, a1, aw);
      quantize_block(vb, bm[s] >> 16, b0, b1, bw);
      uint32_t row_b = row + kq, col_b = col + kr;
      if (col_b >= cpr) {
        col_b -= cpr;
        ++row_b;
      }
      if (ok_a) {
        reinterpret_cast<uint2*>(codes)[(c0 + cl) >> 1] = make_uint2(a0, a1);
        scales[((row >> 7) * kgroups + (col >> 3)) * 512u + (row & 31u) * 16u +
               ((row >> 5) & 3u) * 4u + ((col >> 1) & 3u)] = (uint8_t)aw;
      }
      if (ok_b) {
        reinterpret_cast<uint2*>(codes)[(c0 + cl + kStride) >> 1] = make_uint2(b0, b1);
        scales[((row_b >> 7) * kgroups + (col_b >> 3)) * 512u + (row_b & 31u) * 16u +
               ((row_b >> 5) & 3u) * 4u + ((col_b >> 1) & 3u)] = (uint8_t)bw;
      }
      row += dq;
      col += dr;
      if (col >= cpr) {
        col -= cpr;
        ++row;
      }
    }
  }
};

struct Fp8Op {
  static constexpr int kUnit = 1;
  static constexpr bool kBlockMax = false;
  float s_enc;
  uint2* codes;
  __device__ __forceinline__ void bind(float*) {}
  __device__ __forceinline__ void init() {}
  __device__ __forceinline__ void unit(const uint4 (&v)[1], uint64_t c, bool valid) {
    if (!valid) return;
    float f[8];
    unpack8(v[0], f);
#pragma unroll
    for (int i = 0; i < 8; ++i) f[i] = __fmul_rn(f[i], s_enc);
    codes[c] = make_uint2(e4m3x4(f[0], f[1], f[2], f[3]), e4m3x4(f[4], f[5], f[6], f[7]));
  }
  template <int kThreadsPerBlock>
  __device__ __forceinline__ void run_slice(const uint4* buf, uint32_t n, uint64_t c0) const {
    for (uint32_t cl = threadIdx.x; cl < n; cl += kThreadsPerBlock) {
      float f[8];
      unpack8(lds128(buf + cl), f);
#pragma unroll
      for (int i = 0; i < 8; ++i) f[i] = __fmul_rn(f[i], s_enc);
      codes[c0 + cl] =
          make_uint2(e4m3x4(f[0], f[1], f[2], f[3]), e4m3x4(f[4], f[5], f[6], f[7]));
    }
  }
};

// Persistent tile loop: thread 0 keeps kStages bulk copies of 16 KB tiles in
// flight; every thread applies `op` to its chunks of each landed tile.
// `setup(op)` runs once the first copies are on their way (reads that only
// the arithmetic needs, such as the tensor scale, overlap the loads).
// kReverse visits the tiles last-first: a second pass over data that a
// first pass has just streamed forward starts on the lines still in L2
// (NVFP4 dynamic route at 18432 x 3072, amax pass then quantizer: 49.5 ->
// 48.2 us).  Returns false if a bounded wait expired (recorded in *err).
template <bool kReverse = false, typename Op, typename Setup>
__device__ __forceinline__ bool stream_tiles(const uint4* __restrict__ x, uint64_t n_chunks,
                                             Op& op, Setup setup, unsigned* err,
                                             uint64_t timeout_ns) {
  extern __shared__ __align__(128) uint8_t qsm[];
  uint4* buf = reinterpret_cast<uint4*>(qsm);
  uint64_t* full = reinterpret_cast<uint64_t*>(qsm + kStages * kTileChunks * 16);
  __shared__ int abort_flag;
  const uint64_t n_tiles = (n_chunks + kTileChunks - 1) / kTileChunks;
  const int tid = threadIdx.x;

  auto issue = [&](uint64_t t, int s) {
    const uint64_t c0 = (kReverse ? n_tiles - 1 - t : t) * kTileChunks;
    const uint64_t left = n_chunks - c0;
    const uint32_t nc = left < (uint64_t)kTileChunks ? (uint32_t)left : (uint32_t)kTileChunks;
    mbar_arrive_expect_tx(&full[s], nc * 16u);
    bulk_load(buf + s * kTileChunks, x + c0, nc * 16u, &full[s]);
  };

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
    abort_flag = 0;
    mbar_fence_init();
    for (int s = 0; s < kStages; ++s) {
      const uint64_t t = blockIdx.x + (uint64_t)s * gridDim.x;
      if (t < n_tiles) issue(t, s);
    }
  }
  setup(op);
  op.init();
  __syncthreads();
  int s = 0;
  uint32_t phase = 0;
  bool ok = true;
  uint64_t t_stop = 0;
  for (uint64_t t = blockIdx.x; t < n_tiles; t += gridDim.x) {
    if (tid == 0) {
      const WaitCtl ctl{&abort_flag, err, timeout_ns};
      if (!mbar_wait(&full[s], phase, ctl)) abort_flag = 1;
    }
    __syncthreads();
    if (abort_flag) {
      ok = false;
      t_stop = t;
      break;
    }
    const uint64_t c0 = (kReverse ? n_tiles - 1 - t : t) * kTileChunks;
    constexpr int kU = Op::kUnit;
#pragma unroll
    for (int u = 0; u < kTileChunks / (kU * kThreads); ++u) {
      const int cl = (u * kThreads + tid) * kU;   // first chunk of this thread's unit
      const uint64_t c = c0 + cl;
      const bool valid = c < n_chunks;           // units never straddle n_chunks
      uint4 v[kU];
#pragma unroll
      for (int k = 0; k < kU; ++k)
        v[k] = valid ? lds128(buf + s * kTileChunks + cl + k) : make_uint4(0u, 0u, 0u, 0u);
      op.unit(v, c, valid);
    }
    __syncthreads();   // every thread is done with this stage
    if (tid == 0) {
      const uint64_t nt = t + (uint64_t)kStages * gridDim.x;
      if (nt < n_tiles) issue(nt, s);
    }
    if (++s == kStages) {
      s = 0;
      phase ^= 1u;
    }
  }
  if (!ok && tid == 0) {
    // Let every copy already issued land before the CTA exits: the tiles
    // t_stop, t_stop + G, ... (at most kStages of them) sit in stages
    // s, s + 1, ... with the current phase, flipping on wrap-around.
    uint64_t tt = t_stop;
    for (int i = 0; i < kStages && tt < n_tiles; ++i, tt += gridDim.x) {
      const uint32_t a = smem_u32(&full[s]);
      const uint64_t t0 = global_timer_ns();
      while (!mbar_try_wait(a, phase) && global_timer_ns() - t0 < timeout_ns) {
      }
      if (++s == kStages) {
        s = 0;
        phase ^= 1u;
      }
    }
  }
  return ok;
}

// The CTA's first tile into L2 (one bulk prefetch from thread 0), issued
// before grid_dep_wait: a prefetch is a hint that returns no data, so it is
// correct even while the previous kernel still writes x, and the tile's DRAM
// read overlaps that kernel's tail.  NVFP4 4608 x 3072 static, measured:
// 9.1 -> 8.0 us in a chain of launches, 9.3 -> 8.3 us right after a fused
// GEMM, unchanged (15.0 us) alone after an L2 flush.  Prefetching all four
// ring tiles gained 0.1-0.8 us more in chains but cost 1.1 us alone.
__device__ __forceinline__ void l2_prefetch_first_tile(const uint4* x, uint64_t n_chunks) {
  if (threadIdx.x == 0 && (uint64_t)blockIdx.x * kTileChunks < n_chunks) {
    const uint64_t c0 = (uint64_t)blockIdx.x * kTileChunks;
    const uint64_t left = n_chunks - c0;
    const uint32_t nc = left < (uint64_t)kTileChunks ? (uint32_t)left : (uint32_t)kTileChunks;
    l2_prefetch_bulk(x + c0, nc * 16u);
  }
}

// amax over n_chunks 16-byte chunks, folded into *amax_bits (fp32 bits;
// cleared before the launch).
__global__ void __launch_bounds__(kThreads, kBlocksPerSm)
    amax_kernel(const uint4* __restrict__ x, uint64_t n_chunks, unsigned* __restrict__ amax_bits,
                unsigned* err, uint64_t timeout_ns) {
  l2_prefetch_first_tile(x, n_chunks);
  grid_dep_wait();
  grid_dep_launch();
  __shared__ uint32_t warp_max[kThreads / 32];
  AmaxOp op;
  stream_tiles(x, n_chunks, op, [](AmaxOp&) {}, err, timeout_ns);
  const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, op.m);
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t b = 0;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) b = max(b, warp_max[w]);
    if (b) atomicMax(amax_bits, b << 16);
  }
}

// Tensor scale: kDynamic -> scale_src holds amax, S_dec = amax / qmax (1 if
// amax == 0); otherwise scale_src holds S_dec.  Block 0 records S_dec.
template <bool kDynamic>
__device__ __forceinline__ float tensor_scale(const float* scale_src, float* sdec_out,
                                              float qmax) {
  float s_dec;
  if (kDynamic) {
    const float amax = *scale_src;
    s_dec = (amax == 0.0f) ? 1.0f : __fdiv_rn(amax, qmax);
  } else {
    s_dec = *scale_src;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0 && sdec_out != scale_src) *sdec_out = s_dec;
  return s_dec;
}

template <bool kDynamic, typename Idx>
__global__ void __launch_bounds__(kThreads, kBlocksPerSm)
    quant_nvfp4_kernel(const uint4* __restrict__ x, uint64_t n_chunks, int64_t K,
                       const float* scale_src, float* sdec_out, uint32_t* __restrict__ codes,
                       uint8_t* __restrict__ scales, uint3 row_div, unsigned* err,
                       uint64_t timeout_ns) {
  // The dynamic-scale instance is the second pass over x (after amax_kernel,
  // or over y after the GEMM that reduced its amax): it reads last-first, and
  // its first tiles are then the ones most recently in L2.
  if (!kDynamic) l2_prefetch_first_tile(x, n_chunks);
  grid_dep_wait();
  grid_dep_launch();
  __shared__ float r_table[128];
  Nvfp4Op<Idx> op;
  op.r_table = r_table;
  op.chunks_per_row = (Idx)(K >> 3);
  op.div_m = row_div.x;
  op.div_s1 = row_div.y;
  op.div_s2 = row_div.z;
  op.K = K;
  op.codes = codes;
  op.scales = scales;
  stream_tiles<kDynamic>(
      x, n_chunks, op,
      [&](Nvfp4Op<Idx>& o) {
        o.s_enc = encode_scale(tensor_scale<kDynamic>(scale_src, sdec_out, 2688.0f));
      },
      err, timeout_ns);
}

template <bool kDynamic>
__global__ void __launch_bounds__(kThreads, kBlocksPerSm)
    quant_fp8_kernel(const uint4* __restrict__ x, uint64_t n_chunks, const float* scale_src,
                     float* sdec_out, uint2* __restrict__ codes, unsigned* err,
                     uint64_t timeout_ns) {
  l2_prefetch_first_tile(x, n_chunks);
  grid_dep_wait();
  grid_dep_launch();
  Fp8Op op;
  op.codes = codes;
  stream_tiles(
      x, n_chunks, op,
      [&](Fp8Op& o) { o.s_enc = encode_scale(tensor_scale<kDynamic>(scale_src, sdec_out, 448.0f)); },
      err, timeout_ns);
}

// FP8 weights, one scale per row: one warp per row, two passes over the row
// (the second hits L1/L2).  Offline, once per layer.
__global__ void __launch_bounds__(kThreads) quant_fp8_rows_kernel(const uint4* __restrict__ w,
                                                                  int64_t rows, int64_t K,
                                                                  float* __restrict__ s_rows,
                                                                  uint2* __restrict__ codes) {
  grid_dep_wait();
  grid_dep_launch();
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

// ------------------------------------------------ one-pass dynamic scale ---
// The tensor scale depends on max |x| over the whole tensor (the amax pass),
// and the codes depend on the tensor scale, so a streaming quantizer reads x
// twice.  When x fits in the aggregate shared memory of the grid (one CTA per
// SM, launched cooperatively so every CTA is resident), each CTA loads its
// slice once, the grid combines the slice maxima through two words of
// global memory, and each CTA quantizes its slice from shared memory.
constexpr int kOnePassThreads = 1024;
constexpr int kOnePassSmem = 225 * 1024;
constexpr int kOnePassSliceMax = 14 * 1024;       // chunks: 224 KB of data at most
// NVFP4 steps of run_slice: two 2-chunk units per thread and step
constexpr int kOnePassSteps = (kOnePassSliceMax + 4 * kOnePassThreads - 1) / (4 * kOnePassThreads);

// The amax word and the arrival count as one 64-bit acquire load (they are
// adjacent words of one 8-byte-aligned pair, low word first).
__device__ __forceinline__ uint64_t ld_acquire_gpu_pair(const unsigned* p) {
  uint64_t v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

// Wait until at most `pending` (0-3) of this thread's cp.async groups are
// still in flight (the operand must be an immediate; a constant argument
// folds the switch).
__device__ __forceinline__ void cp_async_wait_pending(int pending) {
  switch (pending) {
    case 3: asm volatile("cp.async.wait_group 3;" ::: "memory"); break;
    case 2: asm volatile("cp.async.wait_group 2;" ::: "memory"); break;
    case 1: asm volatile("cp.async.wait_group 1;" ::: "memory"); break;
    default: asm volatile("cp.async.wait_group 0;" ::: "memory"); break;
  }
}

// sync[0]: amax bits (fp32), sync[1]: arrival count, sync[2]: departure
// count; all zero at launch, and the last CTA to depart zeroes them again, so
// back-to-back launches (graph replays included) need no clearing between.
template <typename Op>
__global__ void __launch_bounds__(kOnePassThreads, 1)
    onepass_kernel(const uint4* __restrict__ x, uint64_t n_chunks, uint32_t slice, Op op,
                   float qmax, float* sdec_out, unsigned* sync, unsigned* err,
                   uint64_t timeout_ns) {
  extern __shared__ __align__(128) uint8_t qsm[];
  uint4* buf = reinterpret_cast<uint4*>(qsm);
  __shared__ uint32_t warp_max[kOnePassThreads / 32];
  __shared__ float op_table[128];
  __shared__ float s_amax;
  __shared__ int abort_flag;
  grid_dep_wait();
  const int tid = threadIdx.x;
  const uint64_t c_begin = (uint64_t)blockIdx.x * slice;
  const uint32_t n = c_begin >= n_chunks ? 0u
                     : (uint32_t)(n_chunks - c_begin < slice ? n_chunks - c_begin : slice);
  // every thread copies its chunks (a dozen 16-byte asynchronous copies in
  // flight per thread), then takes their amax; it reads only the chunks it
  // copied itself, so waiting for its own copies suffices.  NVFP4 copies in
  // the units run_slice quantizes (two adjacent chunks, a warp covering 1 KB),
  // one copy group per step of block maxima, so that each step's maxima are
  // taken while the later steps' copies are still landing (4608 x 3072:
  // 12.46 -> 12.23 us)
  const uint4* xs = x + c_begin;
  if constexpr (Op::kBlockMax) {
#pragma unroll
    for (int s = 0; s < 2 * kOnePassSteps; ++s) {
      const uint32_t c = (uint32_t)s * 2u * kOnePassThreads + 2u * tid;
      if (c < n) {
        cp_async16(smem_u32(buf + c), xs + c);
        cp_async16(smem_u32(buf + c + 1), xs + c + 1);
      }
      if (s & 1) asm volatile("cp.async.commit_group;" ::: "memory");   // step s / 2
    }
  } else {
    for (uint32_t i = tid; i < n; i += kOnePassThreads) cp_async16(smem_u32(buf + i), xs + i);
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
    grid_dep_launch();   // x is on chip: the next kernel may begin launching
  }
  uint32_t m = 0;
  uint32_t bm[kOnePassSteps] = {};
  if constexpr (Op::kBlockMax) {
    // NVFP4: the amax of each 16-element block this thread will quantize
    // (the units of run_slice), kept for after the barrier
    static_assert(kOnePassSteps <= 4, "cp_async_wait_pending takes 0-3 groups");
#pragma unroll
    for (int s = 0; s < kOnePassSteps; ++s) {
      cp_async_wait_pending(kOnePassSteps - 1 - s);   // steps 0..s have landed
      if (s == kOnePassSteps - 1) grid_dep_launch();  // x is on chip
      const uint32_t ca = (uint32_t)s * 4u * kOnePassThreads + 2u * tid;
      const uint32_t cb = ca + 2u * kOnePassThreads;
      const uint32_t a =
          ca < n ? max(chunk_abs_max_bits(lds128(buf + ca)), chunk_abs_max_bits(lds128(buf + ca + 1)))
                 : 0u;
      const uint32_t b =
          cb < n ? max(chunk_abs_max_bits(lds128(buf + cb)), chunk_abs_max_bits(lds128(buf + cb + 1)))
                 : 0u;
      bm[s] = a | (b << 16);
      m = max(m, max(a, b));
    }
  } else {
    for (uint32_t i = tid; i < n; i += kOnePassThreads)
      m = max(m, chunk_abs_max_bits(lds128(buf + i)));
  }
  m = __reduce_max_sync(0xFFFFFFFFu, m);
  if ((tid & 31) == 0) warp_max[tid >> 5] = m;
  if (tid == 0) abort_flag = 0;
  __syncthreads();
  if (tid == 0) {
    uint32_t b = 0;
#pragma unroll
    for (int w = 0; w < kOnePassThreads / 32; ++w) b = max(b, warp_max[w]);
    // publish, arrive, and wait (bounded) for every CTA of the grid
    if (b) atomicMax(&sync[0], b << 16);
    // the arrival releases the maximum above to every CTA that sees it
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(&sync[1]) : "memory");
    // The count and the amax are read together: a load that sees every
    // CTA's arrival also sees every maximum released before it, which saves
    // the second round trip to L2 that reading the amax afterwards took.
    const uint64_t t0 = global_timer_ns();
    uint64_t pair = ld_acquire_gpu_pair(&sync[0]);
    while ((uint32_t)(pair >> 32) < gridDim.x) {
      if (global_timer_ns() - t0 > timeout_ns) {
        atomicExch(err, kErrTimeout);
        abort_flag = 1;
        break;
      }
      pair = ld_acquire_gpu_pair(&sync[0]);
    }
    s_amax = __uint_as_float((uint32_t)pair);
  }
  __syncthreads();
  if (tid == 0) {
    // depart (after a timeout too); the last CTA out resets the words.  The
    // other warps do not wait for this atomic's round trip.
    if (atomicAdd(&sync[2], 1u) == gridDim.x - 1u) {
      sync[0] = 0u;
      sync[1] = 0u;
      sync[2] = 0u;
    }
  }
  if (abort_flag) return;
  const float amax = s_amax;
  const float s_dec = (amax == 0.0f) ? 1.0f : __fdiv_rn(amax, qmax);
  if (blockIdx.x == 0 && tid == 0) *sdec_out = s_dec;
  op.s_enc = encode_scale(s_dec);
  op.bind(op_table);
  op.init();
  __syncthreads();
  if constexpr (Op::kBlockMax)
    op.template run_slice<kOnePassThreads, kOnePassSteps>(buf, n, c_begin, bm);
  else
    op.template run_slice<kOnePassThreads>(buf, n, c_begin);
}

// Opt each kernel into kSmem bytes of dynamic shared memory, once.
template <auto kKern>
cudaError_t set_smem() {
  static const cudaError_t e =
      cudaFuncSetAttribute(kKern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  return e;
}

// Launch with programmatic stream serialization (see grid_dep_wait).
template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kern)(Params...), int grid, int block, int smem, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3((unsigned)block, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

int stream_grid(uint64_t n_chunks, int num_sms) {
  const uint64_t tiles = (n_chunks + kTileChunks - 1) / kTileChunks;
  return (int)std::max<uint64_t>(1, std::min<uint64_t>(tiles, (uint64_t)num_sms * kBlocksPerSm));
}

}  // namespace

cudaError_t launch_amax(const void* x, int64_t n_elems, unsigned* amax_bits, cudaStream_t s,
                        int num_sms, unsigned* err, uint64_t timeout_ns) {
  cudaError_t e = cudaMemsetAsync(amax_bits, 0, sizeof(unsigned), s);
  if (e != cudaSuccess) return e;
  if ((e = set_smem<amax_kernel>()) != cudaSuccess) return e;
  const uint64_t n_chunks = (uint64_t)n_elems / 8;
  return launch_pdl(amax_kernel, stream_grid(n_chunks, num_sms), kThreads, kSmem, s,
                    static_cast<const uint4*>(x), n_chunks, amax_bits, err, timeout_ns);
}

// One-pass dynamic quantization when x fits on chip: returns
// cudaErrorNotSupported (nothing launched) when it does not, or when the
// device cannot hold the grid resident.
template <typename Op>
static cudaError_t launch_onepass(const void* x, uint64_t n_chunks, const Op& op, float qmax,
                                  float* sdec_out, unsigned* sync, bool clear, cudaStream_t s,
                                  int num_sms, unsigned* err, uint64_t timeout_ns) {
  // slices of whole 64-element groups (8 chunks), one per SM
  uint64_t slice = (n_chunks + num_sms - 1) / num_sms;
  slice = (slice + 7) / 8 * 8;
  if (slice > (uint64_t)kOnePassSliceMax || slice == 0) return cudaErrorNotSupported;
  const int grid = (int)((n_chunks + slice - 1) / slice);
  auto kern = onepass_kernel<Op>;
  static const cudaError_t attr =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kOnePassSmem);
  if (attr != cudaSuccess) return attr;
  static int resident = -1;   // CTAs of this kernel one SM can hold
  if (resident < 0) {
    int r = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, kern, kOnePassThreads, kOnePassSmem) !=
        cudaSuccess)
      r = 0;
    resident = r;
  }
  if (resident < 1 || grid > num_sms * resident) return cudaErrorNotSupported;
  if (clear) {
    const cudaError_t e = cudaMemsetAsync(sync, 0, 3 * sizeof(unsigned), s);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeCooperative;   // all CTAs resident: the grid waits on itself
  at[0].val.cooperative = 1;
  at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kOnePassThreads, 1, 1);
  cfg.dynamicSmemBytes = kOnePassSmem;
  cfg.stream = s;
  cfg.attrs = at;
  // with programmatic serialization where the driver accepts it alongside a
  // cooperative launch, else without
  static bool pdl_ok = true;
  cfg.numAttrs = pdl_ok ? 2 : 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, static_cast<const uint4*>(x), n_chunks,
                                     (uint32_t)slice, op, qmax, sdec_out, sync, err, timeout_ns);
  if (e != cudaSuccess && pdl_ok) {
    (void)cudaGetLastError();
    pdl_ok = false;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, static_cast<const uint4*>(x), n_chunks, (uint32_t)slice,
                           op, qmax, sdec_out, sync, err, timeout_ns);
  }
  return e;
}

cudaError_t launch_quant_nvfp4_onepass(const void* x, int64_t M, int64_t K,
                                       const qlin_nvfp4_t& out, unsigned* sync, bool clear,
                                       cudaStream_t s, int num_sms, unsigned* err,
                                       uint64_t timeout_ns) {
  const uint64_t n_chunks = (uint64_t)M * (uint64_t)K / 8;
  if (n_chunks >= (1ull << 32)) return cudaErrorNotSupported;
  Nvfp4Op<uint32_t> op;
  op.s_enc = 0.0f;   // set in the kernel once amax is known
  op.chunks_per_row = (uint32_t)(K >> 3);
  op.div_m = op.div_s1 = op.div_s2 = 0;   // run_slice tracks rows without dividing
  op.K = K;
  op.codes = reinterpret_cast<uint32_t*>(out.codes);
  op.scales = out.scales;
  op.r_table = nullptr;   // set in the kernel (shared memory)
  return launch_onepass(x, n_chunks, op, 2688.0f, out.tensor_scale, sync, clear, s, num_sms, err,
                        timeout_ns);
}

cudaError_t launch_quant_fp8_onepass(const void* x, int64_t M, int64_t K, const qlin_fp8_t& out,
                                     unsigned* sync, bool clear, cudaStream_t s, int num_sms,
                                     unsigned* err, uint64_t timeout_ns) {
  const uint64_t n_chunks = (uint64_t)M * (uint64_t)K / 8;
  Fp8Op op;
  op.s_enc = 0.0f;
  op.codes = reinterpret_cast<uint2*>(out.codes);
  return launch_onepass(x, n_chunks, op, 448.0f, out.scale, sync, clear, s, num_sms, err,
                        timeout_ns);
}

// Multiplier and shifts that divide a 32-bit index by d (1 <= d < 2^31)
// without a division instruction: the round-up form of Granlund and
// Montgomery (PLDI 1994), exact for every 32-bit dividend.
static uint3 invariant_divisor(uint32_t d) {
  int l = 0;
  while ((1ull << l) < d) ++l;   // ceil(log2 d)
  const uint64_t m = ((1ull << 32) * ((1ull << l) - d)) / d + 1;
  return make_uint3((uint32_t)m, (uint32_t)(l < 1 ? l : 1), (uint32_t)(l > 1 ? l - 1 : 0));
}

template <bool kDynamic>
static cudaError_t launch_nvfp4_t(const void* x, int64_t M, int64_t K, const float* scale_src,
                                  const qlin_nvfp4_t& out, cudaStream_t s, int num_sms,
                                  unsigned* err, uint64_t timeout_ns) {
  const uint64_t n_chunks = (uint64_t)M * (uint64_t)K / 8;
  const uint3 row_div = invariant_divisor((uint32_t)(K >> 3));
  const int grid = stream_grid(n_chunks, num_sms);
  auto* xin = static_cast<const uint4*>(x);
  auto* codes = reinterpret_cast<uint32_t*>(out.codes);
  cudaError_t e;
  if (n_chunks < (1ull << 32)) {   // 32-bit index math is enough
    if ((e = set_smem<quant_nvfp4_kernel<kDynamic, uint32_t>>()) != cudaSuccess) return e;
    e = launch_pdl(quant_nvfp4_kernel<kDynamic, uint32_t>, grid, kThreads, kSmem, s, xin,
                   n_chunks, K, scale_src, out.tensor_scale, codes, out.scales, row_div, err,
                   timeout_ns);
  } else {
    if ((e = set_smem<quant_nvfp4_kernel<kDynamic, uint64_t>>()) != cudaSuccess) return e;
    e = launch_pdl(quant_nvfp4_kernel<kDynamic, uint64_t>, grid, kThreads, kSmem, s, xin,
                   n_chunks, K, scale_src, out.tensor_scale, codes, out.scales, row_div, err,
                   timeout_ns);
  }
  return e;
}

cudaError_t launch_quant_nvfp4(const void* x, int64_t M, int64_t K, const float* scale_src,
                               bool dynamic, const qlin_nvfp4_t& out, cudaStream_t s,
                               int num_sms, unsigned* err, uint64_t timeout_ns) {
  return dynamic ? launch_nvfp4_t<true>(x, M, K, scale_src, out, s, num_sms, err, timeout_ns)
                 : launch_nvfp4_t<false>(x, M, K, scale_src, out, s, num_sms, err, timeout_ns);
}

cudaError_t launch_quant_fp8(const void* x, int64_t M, int64_t K, const float* scale_src,
                             bool dynamic, const qlin_fp8_t& out, cudaStream_t s, int num_sms,
                             unsigned* err, uint64_t timeout_ns) {
  const uint64_t n_chunks = (uint64_t)M * (uint64_t)K / 8;
  const int grid = stream_grid(n_chunks, num_sms);
  auto* xin = static_cast<const uint4*>(x);
  auto* codes = reinterpret_cast<uint2*>(out.codes);
  cudaError_t e;
  if (dynamic) {
    if ((e = set_smem<quant_fp8_kernel<true>>()) != cudaSuccess) return e;
    return launch_pdl(quant_fp8_kernel<true>, grid, kThreads, kSmem, s, xin, n_chunks, scale_src,
                      out.scale, codes, err, timeout_ns);
  }
  if ((e = set_smem<quant_fp8_kernel<false>>()) != cudaSuccess) return e;
  return launch_pdl(quant_fp8_kernel<false>, grid, kThreads, kSmem, s, xin, n_chunks, scale_src,
                    out.scale, codes, err, timeout_ns);
}

cudaError_t launch_quant_fp8_rows(const void* w, int64_t N, int64_t K, const qlin_fp8_t& out,
                                  cudaStream_t s, int num_sms) {
  const int64_t want = (N + kThreads / 32 - 1) / (kThreads / 32);
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)num_sms * 8));
  return launch_pdl(quant_fp8_rows_kernel, grid, kThreads, 0, s, static_cast<const uint4*>(w), N, K,
                    out.scale, reinterpret_cast<uint2*>(out.codes));
}

}  // namespace qlin
