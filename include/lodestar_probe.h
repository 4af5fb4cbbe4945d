/*
 * lodestar_probe.h -- measurement kernels for the roofline ceilings of the
 * routing path.  None of them is a step of the path; the benchmark runs them
 * to state, on the GPU at hand, the ceilings the path's kernels are judged
 * against where the plain copy bandwidth and the dense bf16 GEMM rate are not
 * the right denominators:
 *   - the prefix matcher's index probes are random 8-byte reads, so its
 *     ceiling is the rate of independent random 8-byte gathers from a table
 *     resident in L2 or in HBM;
 *   - the fp32 CUDA-core scorer is bound by fp32 FMA issue;
 *   - the tensor-core scorers stream weight tiles from L2.
 * Conventions are those of lodestar.h: device pointers, asynchronous on
 * `stream` (a cudaStream_t passed as void*), LS_OK or LS_ERR_ARG /
 * LS_ERR_CUDA returned, ls_last_error() for the message.
 */
#ifndef LODESTAR_PROBE_H
#define LODESTAR_PROBE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Random 8-byte gathers: every thread of `blocks` x 256 performs
 * `per_thread` loads table[mix64(seed + g) & (n_slots - 1)] (g its global
 * load number; eight independent loads in flight per thread) and writes the
 * XOR of what it read to out[thread] (so no load is dead).  table: DEVICE
 * uint64 [n_slots], n_slots a power of two >= 2; out: DEVICE uint64
 * [blocks * 256].  Useful bytes per launch: 8 * blocks * 256 * per_thread. */
int ls_probe_gather(const uint64_t *table, int64_t n_slots, int32_t blocks, int32_t per_thread, uint64_t seed,
                    uint64_t *out, void *stream);

/* fp32 FMA issue rate: every thread of `blocks` x 256 runs `iters` rounds of
 * eight independent fused multiply-adds and writes one float to out[thread].
 * FLOPs per launch: 2 * 8 * iters * blocks * 256. */
int ls_probe_fma(int32_t blocks, int64_t iters, float *out, void *stream);

/* Streaming read bandwidth: `passes` reads of buf (DEVICE, 16-byte aligned,
 * n16 16-byte words) by a grid of `blocks` x 256 threads, 16-byte loads; each
 * thread writes the XOR of its words to out[thread] (DEVICE uint32 x 4
 * [blocks * 256]).  A buffer well inside L2 measures L2 read bandwidth.
 * Bytes per launch: 16 * n16 * passes. */
int ls_probe_read(const void *buf, int64_t n16, int32_t passes, int32_t blocks, void *out, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* LODESTAR_PROBE_H */
