/*
 * head.h -- C ABI of the final pipeline stage's LM head with the top-1
 * epilogue (libshard.so).
 *
 * The last stage of the paper's pipeline turns its hidden states into
 * vocabulary logits; for greedy decoding the coordinator only needs the
 * argmax token and its probability, so the final stage sends back just that
 * pair instead of the 128256 fp32 logits (Section 6.7, "Top-1 Logits
 * Compression").  Here the whole head runs on the GPU and the logits never
 * leave it: per hidden row, RMSNorm with the final norm weight (rounded to
 * fp16 as the projection's activation operand), the INT4 group-quantised
 * lm_head projection to fp32 logits (the same W4A16 projection kernel as the
 * shard's layers), and a top-1 reduction: the greedy token (the largest
 * logit; the lowest token id among equal largest logits) and its softmax
 * probability p_max = 1 / sum_v exp(logit_v - logit_max).  The greedy
 * acceptance check of speculative decoding compares these token ids with
 * the drafts (Section 5.2).
 *
 * Conventions as in shard.h: 0 or a negative SHARD_E* code (message from
 * shard_last_error()); "dev" pointers live on the head's device; work is
 * ordered on the given CUDA stream (void* cudaStream_t; NULL = legacy
 * default stream); the caller owns every buffer it passes.  All calls on one
 * head must come from one host thread at a time and one stream at a time
 * (a head has one set of work buffers).
 */
#ifndef GB300_HEAD_H
#define GB300_HEAD_H

#include <stdint.h>

#include "shard.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Dimensions of the head.
 *   hidden   H, the width of the hidden states it reads
 *   vocab    V >= 1, rows of the lm_head (the logits per hidden row)
 *   group    uint4 quantisation group along the hidden dimension (32, 64 or
 *            128)
 *   rms_eps  epsilon of the final RMSNorm */
typedef struct head_config {
    int32_t hidden, vocab, group, reserved;
    double rms_eps;
} head_config;

/* lm_head [vocab][hidden] in the packed format of shard_matrix_host
 * (dequantised as (q - z) * s per row and group of inputs), and the final
 * RMSNorm weight (host fp16 [hidden]).  Copied by head_create. */
typedef struct head_weights_host {
    shard_matrix_host lm_head;
    const uint16_t* norm;
} head_weights_host;

typedef struct head_s* head_t;

/* Creates a head on the current CUDA device (weights copied and repacked
 * into the library's private layout).  Errors: EINVAL (dimensions or null
 * pointers), EUNSUPPORTED (group outside the supported set, or too many
 * weight units for this GPU's warp count), ENOMEM, ECUDA. */
int head_create(const head_config* cfg, const head_weights_host* weights, head_t* out);
int head_destroy(head_t head);

/* Top-1 of M hidden rows (1 <= M <= SHARD_MAX_TOKENS):
 *   hidden  dev fp16 [M][hidden] (e.g. a final shard's hidden_out)
 *   token   dev int32 [M]: the greedy token of each row
 *   p_max   dev fp32 [M]: its softmax probability, or NULL
 * Does not synchronise.  Errors: EINVAL (M out of range, null hidden or
 * token), ECUDA.  A bounded device wait of the projection that gave up
 * (never expected) makes every row's token -1 and p_max NaN, and leaves the
 * head's internal partial sums dirty: head_top1_host turns that into ECUDA
 * and clears them; a head_top1 caller that reads a -1 token should destroy
 * the head and create it again. */
int head_top1(head_t head, const uint16_t* hidden, int M, int32_t* token, float* p_max, void* cuda_stream);

/* head_top1 with host buffers: copies hidden (host fp16 [M][hidden]) to the
 * device, runs the head and copies token (host int32 [M]) and p_max (host
 * fp32 [M], or NULL) back, then synchronises the stream. */
int head_top1_host(head_t head, const uint16_t* hidden, int M, int32_t* token, float* p_max, void* cuda_stream);

/* Test export: the fp32 logits [M][ld] (ld >= vocab, dev) that head_top1
 * reduces, for element-wise comparison with a reference.  Does not
 * synchronise.  Errors as head_top1, plus EINVAL for ld < vocab. */
int head_debug_logits(head_t head, const uint16_t* hidden, int M, float* logits, int ld, void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* GB300_HEAD_H */
