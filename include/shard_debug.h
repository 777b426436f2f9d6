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

/* y[n][r] = sum_k W[r][k] * x[n][k] for n < S (any S >= 1) with the
 * many-token tensor-core projection (tcgen05; the prefill path): x dev fp16
 * [S][x_ld], 16-byte aligned, x_ld a multiple of 128 and >= K rounded up to
 * 128, columns K .. x_ld - 1 zero; y dev fp32 [S][y_ld], y_ld >= rows,
 * natural row order.  Same W4A16 arithmetic as the step's projections (exact
 * q - z, fp32 sums, the fp16 group scale applied in fp32).  Asynchronous on
 * cuda_stream. */
int shard_debug_gemm(shard_t shard, int layer, int op, const uint16_t* x, int x_ld, int S, float* y, int y_ld,
                     void* cuda_stream);

/* Phase durations of the last completed shard_step, from the GPU's global
 * timer read by one thread at the end of each grid-barrier wait of the step
 * kernel: us[i] is the time between the end of wait i and the end of wait
 * i + 1 (time 0 = kernel start).  Order, 4 * n_layers + 1 values: the
 * prologue with the first RMSNorm and q|k|v projection; then per layer:
 * attention, o, RMSNorm + gate|up, down, and (except after the last layer)
 * the next layer's RMSNorm + q|k|v projection merged into its attention.
 * Returns the number of values written (at most n), or a negative error.
 * Synchronises the device. */
int shard_debug_phase_times(shard_t shard, double* us, int n);

/* Test knob for the step kernel's bounded waits (they must never hang the
 * GPU; the paper has no counterpart): limit = polls before a cross-CTA wait
 * gives up (default 2^22); skip_arrival >= 0 makes CTA 1 leave out its arrival at that grid barrier of every following
 * step (0 = the prologue's), so the other CTAs' waits run out; -1 = off.  A
 * wait that runs out makes the step report "pipeline wait timed out" (EINVAL)
 * through shard_sync_status or the next shard_step, and the KV states stay
 * rejected until kv_state_reset.  Takes effect at the next shard_step. */
int shard_debug_set_wait(shard_t shard, unsigned limit, int skip_arrival);

#ifdef __cplusplus
}
#endif

#endif /* GB300_SHARD_DEBUG_H */
