/*
 * shard.h -- C ABI of the GB300 pipeline-shard decode library (libshard.so).
 *
 * One shard is a contiguous range of Llama-style decoder layers with INT4
 * (W4A16) group-quantised weights, as produced by the paper's per-stage export
 * (Section 3.2).  The library runs the decode-step forward of the shard over a
 * stateful fp16 KV cache (Section 3.4), reads cache rows indirectly through a
 * per-request beam_idx instead of reordering them (the Gather(ReadValue,
 * beam_idx) pattern of Section 4), and honours an attention_mask that hides
 * rejected speculative drafts instead of trimming them (Section 5.2).
 *
 * Conventions for every entry point:
 *  - Return 0 on success, a negative SHARD_E* code on failure; the message of
 *    the calling thread's last failure is available from shard_last_error().
 *    No C++ exception crosses the boundary.
 *  - "fp16" buffers hold IEEE binary16 values as uint16_t bit patterns.
 *  - "dev" pointers are CUDA device pointers on the shard's device; "host"
 *    pointers are ordinary host memory.  Device work is ordered on the CUDA
 *    stream passed in (a cudaStream_t as void*; NULL = legacy default
 *    stream).  shard_step does not synchronise.
 *  - The caller owns every buffer it passes; the library copies what it keeps.
 *    The library owns the shard's weights and the KV state's device memory.
 *  - All calls on one shard (and its KV states) must be issued from one host
 *    thread at a time and on one stream at a time: a shard has one set of
 *    per-step work buffers.
 *  - The shard lives on the CUDA device that is current when shard_create is
 *    called; later calls make that device current themselves.
 */
#ifndef GB300_SHARD_H
#define GB300_SHARD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    SHARD_OK = 0,
    SHARD_EINVAL = -1,       /* invalid argument (host check or device guard) */
    SHARD_ECAPACITY = -2,    /* KV capacity or a fixed limit exceeded */
    SHARD_ENOMEM = -3,       /* device or host allocation failed */
    SHARD_ECUDA = -4,        /* a CUDA runtime call failed */
    SHARD_EUNSUPPORTED = -5  /* valid request the library does not support */
};

/* Largest number of new tokens in one step (the sum of n_new over requests)
 * and largest number of requests. */
#define SHARD_MAX_TOKENS 16
#define SHARD_MAX_REQUESTS 16

/* Model dimensions of the shard (Llama family).
 *   hidden      H, the residual width
 *   n_heads     query heads Hq; n_kv_heads KV heads Hkv (Hq % Hkv == 0)
 *   head_dim    d (even; 64 or 128 supported)
 *   ffn         F, the SwiGLU inner width
 *   group       uint4 quantisation group along the input dimension
 *               (32, 64 or 128 supported)
 *   vocab       rows of the token embedding when the shard is a first stage
 *               (token ids accepted); 0 = hidden states only
 *   max_position  rotary tables cover positions [0, max_position)
 *   rms_eps     RMSNorm epsilon; rope_theta  RoPE base (frequencies
 *               theta^(-2i/d), rotate-half pairing (i, i + d/2)). */
typedef struct shard_config {
    int32_t n_layers, hidden, n_heads, n_kv_heads, head_dim, ffn, group, vocab, max_position, reserved;
    double rms_eps, rope_theta;
} shard_config;

/* One group-quantised matrix W [out][in] (PyTorch orientation), dequantised
 * as W[o][i] = (q[o][i] - z[o][i / group]) * s[o][i / group]  (Section 3.2,
 * Step 4, in its asymmetric form).  With G = ceil(in / group):
 *   codes   host uint8 [out][ceil(in/2)]; the low nibble holds the even input
 *   scales  host fp16  [out][G]
 *   zeros   host uint8 [out][ceil(G/2)]; the low nibble holds the even group
 * The last group of a row may be partial when in % group != 0. */
typedef struct shard_matrix_host {
    const uint8_t* codes;
    const uint16_t* scales;
    const uint8_t* zeros;
} shard_matrix_host;

/* Matrix order within a layer: q [Hq*d][H], k [Hkv*d][H], v [Hkv*d][H],
 * o [H][Hq*d], gate [F][H], up [F][H], down [H][F]. */
enum { SHARD_Q = 0, SHARD_K, SHARD_V, SHARD_O, SHARD_GATE, SHARD_UP, SHARD_DOWN, SHARD_N_MATRICES };

typedef struct shard_layer_host {
    shard_matrix_host w[SHARD_N_MATRICES];
    const uint16_t* attn_norm; /* host fp16 [H]: RMSNorm weight before attention */
    const uint16_t* ffn_norm;  /* host fp16 [H]: RMSNorm weight before the MLP */
} shard_layer_host;

typedef struct shard_weights_host {
    const shard_layer_host* layers; /* n_layers entries */
    const uint16_t* embedding;      /* host fp16 [vocab][H], or NULL when vocab == 0 */
} shard_weights_host;

typedef struct shard_s* shard_t;
typedef struct kvstate_s* kvstate_t;

/* Creates a shard on the current CUDA device from host weights (copied and
 * repacked into the library's private device layout; the caller may free its
 * buffers on return).  Errors: EINVAL (dimensions or pointers), EUNSUPPORTED
 * (group or head_dim outside the supported set), ENOMEM, ECUDA. */
int shard_create(const shard_config* cfg, const shard_weights_host* weights, shard_t* out);
int shard_destroy(shard_t shard);

/* KV state (Section 3.4): a device pool of fp16 K and V for n_rows request
 * rows of up to `capacity` cache entries per row and layer, plus a per-row
 * table of where each cache entry lives (the beam table).  Every row starts
 * empty.  Errors: EINVAL, ENOMEM. */
int kv_state_alloc(shard_t shard, int n_rows, int capacity, kvstate_t* out);
int kv_state_free(kvstate_t state);

/* Empties one row (row >= 0) or all rows (row == -1): the stateful cache of
 * Section 3.4 starts a new sequence.  Also clears a state that a rejected
 * step left unusable.  A single row can only be reset while no other row
 * shares its cache entries, i.e. before any step with a non-NULL beam_idx
 * since the last full reset (else EUNSUPPORTED).  Synchronous.  Errors:
 * EINVAL (row out of range), EUNSUPPORTED. */
int kv_state_reset(kvstate_t state, int row);

/* Sets one layer of one row to `len` cache entries from host fp16 K and V,
 * each [len][Hkv][d] (a prefilled cache, Section 3.4); the row's length
 * becomes len (load every layer with the same len).  Synchronous.  Errors: EINVAL, ECAPACITY (len > capacity),
 * EUNSUPPORTED (row entries shared through a beam gather; reset first). */
int kv_state_load(kvstate_t state, int row, int layer, const uint16_t* k, const uint16_t* v, int len);

/* Copies cache entries [start, start+len) of one row and layer, in the row's
 * own (logical) order -- through the beam table, as the step's attention
 * reads them (Section 4) -- into host fp16 K and V [len][Hkv][d]; what a
 * masked-rewind run is compared with against a physical trim (Section 5.2).  Synchronous
 * (waits for all work on the legacy default stream and the shard's streams
 * to finish by synchronising the device).  Errors: EINVAL. */
int kv_state_read(kvstate_t state, int row, int layer, int start, int len, uint16_t* k, uint16_t* v);

/* The row's current cache length (entries, including masked ones: mask-based
 * rewind, Section 5.2, never shortens a row).  Synchronous.  Errors: EINVAL. */
int kv_state_length(kvstate_t state, int row, int* len);

/* Physical trim (Section 5.1): removes the entries j < len with keep[j] == 0
 * from the row (len must equal the row's length; keep is host memory) and
 * shifts the rest down, in every layer.  This is the operation the mask-based
 * rewind replaces; it exists to compare against it.  Synchronous.
 * Errors: EINVAL, EUNSUPPORTED (entries shared through a beam gather). */
int kv_trim(kvstate_t state, int row, const uint8_t* keep, int len);

/* Prefix capture (Section 8.4, KV capture and warm-resume): copies the
 * row's cache entries j < len with keep[j] != 0 (keep host uint8 [len], or
 * NULL for all; len must equal the row's length), in cache order and for
 * every layer, to host k and v, each [n_layers][n_kept][Hkv][d] fp16, and
 * returns n_kept in *n_kept.  With keep = the request's attention-mask row,
 * the masked (rejected) entries are compacted away.  Entries are read
 * through the beam table, so rows that share entries after a gather export
 * correctly.  The buffers must hold the row's length.  Synchronous.
 * Errors: EINVAL. */
int kv_state_export(kvstate_t state, int row, const uint8_t* keep, int len, uint16_t* k, uint16_t* v, int* n_kept);

/* Warm resume: sets the row to len entries from host k and v, each
 * [n_layers][len][Hkv][d] fp16 (the layout kv_state_export writes), as
 * kv_state_load does for every layer.  Synchronous.  Errors: EINVAL,
 * ECAPACITY (len > capacity), EUNSUPPORTED (entries shared through a beam
 * gather; reset all rows first). */
int kv_state_import(kvstate_t state, int row, const uint16_t* k, const uint16_t* v, int len);

/* One decode step of the shard for B requests (B == the state's n_rows).
 *   n_new        host int32 [B], n_new[b] >= 1 new tokens of request b;
 *                M = sum(n_new) <= SHARD_MAX_TOKENS.  Tokens of request b
 *                are consecutive, request 0 first.
 *   hidden_in    dev fp16 [M][H] input hidden states, 16-byte aligned, or
 *                NULL when token_ids is given (exactly one of the two)
 *   token_ids    dev int32 [M], ids < vocab, looked up in the embedding
 *                (shards with vocab > 0 only; else EUNSUPPORTED)
 *   position_ids dev int32 [M], the RoPE positions (logical positions,
 *                independent of where entries sit in the cache), each in
 *                [0, max_position)
 *   attention_mask dev uint8 [B][mask_stride]; entry j of row b is used by
 *                attention iff mask[b][j] != 0 (Section 5.2).  It must cover
 *                the row's length after the step, P_b + n_b, and be 1 at the
 *                new entries P_b .. P_b + n_b - 1.
 *   beam_idx     dev int32 [B] or NULL (identity).  Before the step, row b
 *                takes over the cache entries and length of row beam_idx[b]
 *                (Gather(ReadValue, beam_idx, axis 0), Section 4); the cache
 *                itself is not moved -- only the per-row entry tables are.
 *   hidden_out   dev fp16 [M][H] output hidden states
 * Semantics: with P_b the row length after the gather, new token i of request
 * b is stored at entry P_b + i and attends to entries j <= P_b + i of row b
 * with mask[b][j] != 0; softmax scale 1/sqrt(d).  Host-side errors: EINVAL,
 * ECAPACITY (an append would exceed capacity), EUNSUPPORTED.  Values that
 * live on the device (beam_idx, positions, token ids, the mask) are checked
 * by the device; a violation makes the step write nothing further and is
 * reported as EINVAL by the next shard_step or by shard_sync_status.
 * Asynchronous on `cuda_stream`. */
int shard_step(shard_t shard, kvstate_t state, const uint16_t* hidden_in, const int32_t* token_ids,
               const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* attention_mask,
               int mask_stride, const int32_t* beam_idx, uint16_t* hidden_out, void* cuda_stream);

/* Packed step (Section 8.6, continuous batching by the mask layout): S new
 * tokens (1 <= S <= SHARD_MAX_TOKENS) on the single row of `state` (a state
 * with n_rows == 1), whose entries the caller partitions into regions -- for
 * example a shared prefix and one region per slot.  Token t is appended at
 * entry P + t (P the row's length before the step) and attends to exactly the
 * entries j < P + S with mask2d[t][j] != 0 (dev uint8 [S][mask_stride],
 * mask_stride >= P + S); it must open its own entry P + t (else the device
 * guard rejects the step, EINVAL).  Rows of one slot that open each other's
 * earlier entries form a causal chunk; rows of different slots are isolated;
 * an idle row opened only on its own entry affects nobody.  Other arguments
 * as shard_step (position_ids are each row's absolute RoPE positions).
 * Errors as shard_step. */
int shard_step_packed(shard_t shard, kvstate_t state, const uint16_t* hidden_in, const int32_t* token_ids, int S,
                      const int32_t* position_ids, const uint8_t* mask2d, int mask_stride, uint16_t* hidden_out,
                      void* cuda_stream);

/* Prefill of one row (Section 3.4: the prompt runs through the stage and
 * fills its stateful cache): S >= 1 new tokens of request `row`, any number,
 * appended at the row's entries P .. P + S - 1 (P its length).  The result
 * is the one shard_step gives for S tokens of one request -- the same
 * rounding points, causal attention among the new tokens and over the row's
 * entries with mask != 0 -- computed with the projections as dense
 * contractions on the tensor cores, in chunks of up to 256 tokens.
 *   hidden_in / token_ids  as shard_step (exactly one), [S] rows
 *   position_ids           dev int32 [S]
 *   attention_mask         dev uint8 [mask_len], the row's mask, mask_len >=
 *                          P + S, 1 at the new entries
 *   hidden_out             dev fp16 [S][H]
 * The row must hold its entries contiguously (no beam gather since the last
 * full reset; else EUNSUPPORTED).  The first call allocates the library's
 * prefill work buffers.  Device-side values (token ids, positions, the mask at
 * the new entries) are checked on the device; a violation is reported by
 * shard_sync_status or the next call as EINVAL.  Asynchronous on cuda_stream.
 * Errors: EINVAL, ECAPACITY, EUNSUPPORTED, ENOMEM, ECUDA. */
int shard_prefill(shard_t shard, kvstate_t state, int row, const uint16_t* hidden_in, const int32_t* token_ids, int S,
                  const int32_t* position_ids, const uint8_t* attention_mask, int mask_len, uint16_t* hidden_out,
                  void* cuda_stream);

/* shard_step on HOST buffers: copies the inputs to the device (through
 * library-owned pinned staging buffers), runs the step on `cuda_stream`,
 * copies hidden_out back and waits for it.  Arguments as in shard_step, but
 * every pointer is host memory. */
int shard_step_host(shard_t shard, kvstate_t state, const uint16_t* hidden_in, const int32_t* token_ids,
                    const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* attention_mask,
                    int mask_stride, const int32_t* beam_idx, uint16_t* hidden_out, void* cuda_stream);

/* Waits for `cuda_stream` and returns the device-side guard status of the
 * shard's steps since the last check: 0, or EINVAL (with a message naming the
 * violated condition).  Clears the status. */
int shard_sync_status(shard_t shard, void* cuda_stream);

/* One projection of the shard, y[m][r] = sum_k W[r][k] * x[m][k], without
 * any device allocation: for callers that must not allocate device memory
 * while they run (a runtime that has pre-reserved all of HBM in its own pool
 * and forbids outside cudaMalloc, a thread that may not take the allocator's
 * lock, or a loop where an allocation's implicit synchronisation is not
 * allowed).  It runs the same kernel as the step's projections; the kernel's
 * scratch (the row sums of row-blocks split between warps, in 64-bit fixed
 * point, the per-row-block counts of units added, and a zero-padded copy of
 * x) lives in one fixed 4 MiB device array inside the library, which every GPU
 * that loads the library holds until the process exits.  The paper has no
 * counterpart; this is a deployment convenience.
 *   op      0 = q|k|v, 1 = o, 2 = gate|up, 3 = down (row order as in
 *           shard_debug.h); layer in [0, n_layers)
 *   x       dev fp16 [M][K], K the op's input width, 1 <= M <= 16
 *   y       dev fp32 [M][y_ld], y_ld >= the op's natural row count
 * Calls larger than the fixed array (scratch for M tokens of K inputs and
 * of the op's rows) fail with ECAPACITY and a message giving the sizes.  The
 * kernel's own waits are bounded: one that runs out (never expected) sets the
 * shard's status word, which shard_sync_status then reports as EINVAL.
 * The first call on each device resolves the array's device address (with
 * that device made current); make that first call before any stream capture.
 * Every call on a device shares the one array and it keeps the last call's
 * contents (each call clears the counts, sums and padding on its stream before
 * its kernel runs): calls whose work
 * overlaps on the GPU -- different streams, or different host threads --
 * race and corrupt each other's results.  Asynchronous on cuda_stream; it
 * does not synchronise. */
int shard_gemv_noalloc(shard_t shard, int layer, int op, const uint16_t* x, int M, float* y, int y_ld,
                       void* cuda_stream);

/* Message of the calling thread's last failed call ("" if none). */
const char* shard_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* GB300_SHARD_H */
