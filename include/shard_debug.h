/*
 * shard_debug.h -- test exports of libshard (not part of the serving path).
 *
 * They expose single pieces of the step so tests can check them bit by bit:
 * the private weight layout read back in natural order, and one projection
 * (the same GEMV kernel the step runs, with a plain fp32 store instead of the
 * fused epilogue).  The fused projections are numbered
 *   0 = q|k|v  (rows: the q rows, then k, then v; inputs H)
 *   1 = o      (rows H; inputs Hq*d)
 *   2 = gate|up (rows: the F gate rows, then the F up rows; inputs H)
 *   3 = down   (rows H; inputs F)
 * Same conventions as shard.h (0 / negative SHARD_E* codes, fp16 as uint16_t).
 */
#ifndef GB300_SHARD_DEBUG_H
#define GB300_SHARD_DEBUG_H

#include <stdint.h>

#include "shard.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Natural row count, input count K, and private-layout bytes of a fused
 * projection of one layer. */
int shard_debug_op_info(shard_t shard, int layer, int op, int* rows, int* K, long long* bytes);

/* Dequantises a fused projection from the library's private layout:
 * out (dev fp32, [rows][ld], ld >= K) receives (q - z) * s in natural order
 * (Section 3.2, Step 4).  Synchronous. */
int shard_debug_unpack(shard_t shard, int layer, int op, float* out, int ld);

/* y[m][r] = sum_k W[r][k] * x[m][k] for m < M (1..16) with the step's GEMV
 * kernel.  x: dev fp16 [M][K]; y: dev fp32 [M][y_ld], y_ld >= rows.  Uses the
 * shard's work buffers: do not overlap with shard_step.  Asynchronous on
 * cuda_stream. */
int shard_debug_gemv(shard_t shard, int layer, int op, const uint16_t* x, int M, float* y, int y_ld,
                     void* cuda_stream);

/* Phase durations of the last completed shard_step, from the GPU's global
 * timer read by one thread at each grid barrier of the step kernel: us[i] is
 * the time between barrier i and barrier i+1 (barrier 0 = kernel start;
 * order: prologue, then per layer: RMSNorm + q|k|v + attention, o,
 * RMSNorm + gate|up, down; the last layer's down phase
 * ends with the kernel and is not reported).  Returns the number of values
 * written (at most n), or a negative error.  Synchronises the device. */
int shard_debug_phase_times(shard_t shard, double* us, int n);

#ifdef __cplusplus
}
#endif

#endif /* GB300_SHARD_DEBUG_H */
