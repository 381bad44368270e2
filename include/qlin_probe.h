/* qlin_probe.h -- tensor-core rate probe of the qlin measurement harness.
 *
 * Not part of the quantized linear layer: the paper has no counterpart.  It
 * measures the ceiling of the tcgen05 MMA forms that the GEMMs of libqlin
 * issue, so that their roofline fractions can be stated against a measured
 * tensor-core rate as well as against the nominal one.  Built as its own
 * library, libqlin_probe.so.
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

#ifdef __cplusplus
}
#endif

#endif /* QLIN_PROBE_H */
