/* qlin_probe.h -- tensor-core rate probe of the qlin measurement harness.
 *
 * Not part of the quantized linear layer: the paper has no counterpart.  It
 * measures the ceiling of the tcgen05 MMA forms that the GEMMs of libqlin
 * issue, so that their roofline fractions can be stated against a measured
 * tensor-core rate as well as against the nominal one, and the issue rates
 * of the copies that feed them (block-scale copies into TMEM, operand copies
 * into shared memory).  Built as its own library, libqlin_probe.so.
 */
#ifndef QLIN_PROBE_H
#define QLIN_PROBE_H

#ifdef __cplusplus
extern "C" {
#endif

/* Launch `ctas` CTAs (one per SM; an even count for CTA pairs), each issuing
 * `iters` back-to-back tcgen05.mma instructions from one thread, with its
 * operands resident in shared memory.
 *   kind  4 = NVFP4 (kind::mxf4nvf4, scale_vec::4X, K = 64 per instruction),
 *         8 = FP8 E4M3 (kind::f8f6f4, K = 32), 16 = bf16 (kind::f16, K = 16);
 *         kind + 100: the same with the A operand read from TMEM (written
 *         there first by tcgen05.st) instead of shared memory
 *   pair  0 = cta_group::1 (M = 128), 1 = cta_group::2 (M = 256 on two SMs)
 *   n     the instruction's N: 256 for every kind, or 128 for kind 4, pair 0
 *   out   device array of 2 x (number of MMA-issuing CTAs) uint64: per issuing
 *         CTA its SM cycles (clock64) and nanoseconds (globaltimer) from the
 *         first MMA to the completion of the last; 0 if its wait expired
 *   err   device word, set to 5 if a bounded wait expired
 *   stream  cudaStream_t (NULL = default stream); the call is asynchronous.
 * Returns 0 on launch, 1 for an invalid argument or an unsupported
 * (kind, pair, n), 4 for a CUDA launch error.  Allocates nothing. */
int qlin_probe_mma(int kind, int pair, int n, int ctas, int iters, unsigned long long *out,
                   unsigned *err, void *stream);

/* Issue rate of the block-scale copies the NVFP4 GEMM makes beside its MMA
 * stream (tcgen05.cp.cta_group::2.32x128b.warpx4, one 512-byte scale atom
 * into 4 TMEM columns of both SMs).  `ctas` CTAs as pairs (even count, one per
 * SM); in CTA 0 of each pair one thread issues `mmas` NVFP4 pair MMAs (N = 256,
 * 0..16) per iteration while `warps` warps (1..8, one lane each) issue
 * `copies` copies per iteration between them (copies % warps == 0), for
 * `iters` iterations.
 *   out   device array of `ctas` uint64: per pair, the MMA thread's SM cycles
 *         until its MMAs completed, then the first copy warp's cycles until
 *         every warp's copies completed; 0 if a wait expired
 *   err   device word, set to 5 if a bounded wait expired
 * Returns 0 on launch, 1 for an invalid argument, 4 for a CUDA error. */
int qlin_probe_scale_copy(int warps, int copies, int mmas, int ctas, int iters,
                          unsigned long long *out, unsigned *err, void *stream);

/* Shared-memory fill rate of an SM's asynchronous copies, per issuing
 * thread.  `ctas` CTAs (one per SM); in each, `threads` threads (1..8, one
 * per warp) keep `depth` (1..8) copies of 16 KB in flight each, `iters`
 * copies per thread; threads * depth * 16 KB must fit in 199 KB.
 *   mode  0 = tiled 2-D tensor copies of 128-row x 128-byte boxes with the
 *         128-byte swizzle (as the GEMMs' operand boxes) from a [rows, 1536
 *         bytes] view of src; 1 = plain bulk copies of 16 contiguous KB
 *   src, src_bytes  device buffer read at pseudo-random box positions
 *         (128-byte aligned; at least 128 rows of 1536 bytes)
 *   out   device array of `ctas` uint64: per CTA the first thread's SM
 *         cycles until its last copy landed; 0 if a wait expired
 *   err   device word, set to 5 if a bounded wait expired
 * Returns 0 on launch, 1 for an invalid argument, 4 for a CUDA error. */
int qlin_probe_fill(int mode, int threads, int depth, int ctas, int iters, const void *src,
                    unsigned long long src_bytes, unsigned long long *out, unsigned *err,
                    void *stream);

#ifdef __cplusplus
}
#endif

#endif /* QLIN_PROBE_H */
