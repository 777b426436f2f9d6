// Internal interface between the host side of libshard and its kernels.
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace shard {

constexpr int kMaxTokens = 16;    // SHARD_MAX_TOKENS
constexpr int kMaxRequests = 16;  // SHARD_MAX_REQUESTS

// ---------------------------------------------------------------------------
// Private INT4 weight layout ("unit stream").
//
// A fused projection with N output rows and K inputs is cut into row-blocks
// of 64 rows and units of 128 inputs.  Unit (rb, ku) is one contiguous run of
// unit_bytes(group) bytes at offset (rb * upr + ku) * unit_bytes, with
// upr = ceil(K / 128) units per row-block, so the whole matrix is one linear
// stream that bulk copies read front to back.
//
// Unit contents:
//  [0, 4096)   codes: 8 fragment tiles of 512 bytes, tile ft = kc * 4 + rt for
//              the 64-input half kc and the 16-row tile rt.  Lane l of a warp
//              reads 16 bytes at ft * 512 + 16 * l: four 32-bit words, word j
//              holding the 8 nibbles of that lane's m16n8k16 A fragment for
//              virtual k-block j.  With gid = l / 4, tig = l % 4, h = j / 2,
//              jj = j % 2 and k0 = 128 * ku + 64 * kc + 32 * h + 8 * tig + 4 * jj:
//                bits  0..3 / 16..19 : row gid,     inputs k0,   k0+1   (a0)
//                bits  4..7 / 20..23 : row gid + 8, inputs k0,   k0+1   (a1)
//                bits  8..11/ 24..27 : row gid,     inputs k0+2, k0+3   (a2)
//                bits 12..15/ 28..31 : row gid + 8, inputs k0+2, k0+3   (a3)
//              (rows relative to the tile).  The matching B fragment of
//              token n is then four consecutive activations x[n][k0..k0+3],
//              so a lane's activations for a (kc, h) pair are 8 contiguous
//              fp16 values: activations stay in natural [token][input] order.
//  [4096, ..)  per group of the unit (128 / group groups, group in 32/64/128):
//              64 fp16 scales then 64 uint8 zero points, each ordered
//              [gid 0..7][rt 0..3][lo, hi] so one lane reads its 8 scales with
//              one 16-byte load and its 8 zero points with one 8-byte load.
//              The zero point z of an upper row (hi: rows 8..15 of a tile) is
//              stored as 16 z, the low byte of the fp16 bits of -(64 + z), so
//              the dequantisation builds both offsets with one byte permute.
// Rows past the real ones and inputs past K carry code 0 / zero point 0 /
// scale 0, or (inputs of a real group past K) the group's zero point, so they
// contribute exactly 0.
// ---------------------------------------------------------------------------
constexpr int kRowsPerBlock = 64;
constexpr int kUnitK = 128;
constexpr int kCodeBytes = 4096;
constexpr int kMetaBytesPerGroup = 192;
inline int unit_bytes_for_group(int group) { return kCodeBytes + (kUnitK / group) * kMetaBytesPerGroup; }

enum OpKind { OP_QKV = 0, OP_O = 1, OP_GU = 2, OP_DOWN = 3, N_OPS = 4 };

// Row order inside the fused projections:
//  OP_QKV: q heads, then k heads, then v heads (d rows each).  Within a q or k
//          head, 16-row tile jt holds rotary pairs: rows 0..7 are dims
//          8*jt .. 8*jt+7 and rows 8..15 are dims d/2 + 8*jt .. +7.  v rows
//          are in natural order.
//  OP_GU:  16-row tile t holds gate rows 8t..8t+7 (rows 0..7) and up rows
//          8t..8t+7 (rows 8..15).
//  OP_O, OP_DOWN: natural order.
struct OpDims {
  int kind, Hq, Hkv, d, F, H;
};

// Natural output index of GPU row R of an op (q, k, v concatenated for QKV;
// gate then up for GU), or -1 for a padding row.
__host__ __device__ inline int natural_row(const OpDims& o, int R) {
  int T = R >> 4, r = R & 15;
  if (o.kind == OP_QKV) {
    int tph = o.d >> 4, nq = o.Hq * tph, nk = o.Hkv * tph;
    if (T < nq + nk) {
      int base = T < nq ? 0 : o.Hq * o.d;
      int t = T < nq ? T : T - nq;
      int head = t / tph, jt = t % tph;
      int dim = r < 8 ? 8 * jt + r : (o.d >> 1) + 8 * jt + (r - 8);
      return base + head * o.d + dim;
    }
    int Rv = R - (o.Hq + o.Hkv) * o.d;
    return Rv < o.Hkv * o.d ? (o.Hq + o.Hkv) * o.d + Rv : -1;
  }
  if (o.kind == OP_GU) {
    int j = 8 * T + (r & 7);
    if (j >= o.F) return -1;
    return r < 8 ? j : o.F + j;
  }
  return R < o.H ? R : -1;
}

struct PackedOp {
  uint8_t* units = nullptr;  // device
  int n_rb = 0, upr = 0, unit_bytes = 0, group = 0, K = 0, Kp = 0, rows = 0;
  size_t bytes = 0;
  OpDims dims{};
};

// Fixed-point accumulation.  Split projections add their partial sums with
// 64-bit integer atomics into accumulators holding round(value * 2^32):
// integer addition is associative, so a sum does not depend on the order in
// which contributions arrive -- results are deterministic and a request's
// rows are independent of what else is in the batch -- and the sum of the
// fp32 partials is exact (partials above 2^-9 in magnitude convert without
// rounding; the range is +-2^31).
constexpr float kFixOne = 4294967296.0f;             // 2^32
constexpr double kFixInv = 2.3283064365386962890625e-10;  // 2^-32

// Per-step request/token bookkeeping.  The step kernel derives it in every
// CTA from the step's arguments (the same values everywhere), so no CTA waits
// for another to publish it.
struct StepParams {
  int M, B, abort_step, pad0;
  int tok_req[kMaxTokens];
  int tok_idx[kMaxTokens];
  int tok_pos[kMaxTokens];
  int tok_slot[kMaxTokens];   // physical slot: phys_row * capacity + position in row
  int req_tok0[kMaxRequests + 1];
  int req_src[kMaxRequests];  // beam_idx[b] (the row whose entries row b continues)
  int req_P[kMaxRequests];    // row length after the gather, before the append
  int req_len[kMaxRequests];  // row length after the append
};

enum EpiKind { EPI_STORE = 0, EPI_QKV = 1, EPI_RESID = 2, EPI_SWIGLU = 3 };

// Where a projection's row-block sums go.
//   EPI_RESID   acc = the residual stream X [16][H] (fixed point): x += W a.
//   EPI_QKV     acc = q|k|v sums [16][acc_ld] in the op's row order; each
//               segment then adds its unit count to cnt[kv head of the
//               row-block] (release), which the attention items wait for.
//   EPI_SWIGLU  acc = gate|up sums [16][acc_ld]; cnt[row-block] counts the
//               units added; the contributor that completes a row-block reads
//               the sums, writes h = fp16(silu(gate) * up) and clears the
//               sums and the count.
//   EPI_STORE   as EPI_SWIGLU, but the completing contributor writes the fp32
//               sums to y[m][natural row].
struct EpiArgs {
  int kind;
  OpDims dims;
  long long* acc;
  int acc_ld;
  int* cnt;
  float* y;       // EPI_STORE: y[m][natural row], row stride y_ld
  int y_ld;
  uint16_t* h;    // EPI_SWIGLU: fp16 [M][h_ld]
  int h_ld;
};

struct GemvArgs {
  const uint8_t* units;
  int n_rb, upr;
  const uint16_t* act;  // fp16 activations [M][act_ld] (act_ld a multiple of 128, zero padded)
  int act_ld;
  int M;
  int* status;
  EpiArgs ep;           // EPI_STORE: acc [16][n_rb * 64] and cnt [n_rb] zero on entry (left zero)
};

// Launch geometry of the standalone projection for a given token bucket
// (nt = 1: M <= 8, nt = 2: M <= 16).
int gemv_grid(int nt, int num_sms);
cudaError_t launch_gemv(const GemvArgs& a, int nt, int group, int grid, cudaStream_t s, bool pdl);
// One-time per-device kernel attribute setup (dynamic shared memory limits).
cudaError_t gemv_setup();
int gemv_warps_per_cta();

// Many-token projection on the tensor cores (gemm_tc.cu): y[n][natural
// row] = sum_k W[r][k] act[n][k] for n < S.
struct GemmArgs {
  const uint8_t* units;
  int n_rb, upr;
  const uint16_t* act;  // fp16 [S][act_ld], act_ld a multiple of 128, zero padded past K
  int act_ld, S;
  float* y;             // fp32 [S][y_ld]
  int y_ld;
  OpDims dims;
  int* status;
};
cudaError_t gemm_tc_setup();
int gemm_tc_tile(int S);
cudaError_t launch_gemm_tc(const GemmArgs& a, int group, cudaStream_t s);

// Prefill (prefill.cu): per-token kernels around the tensor-core projections.
struct PrefillLayerArgs {
  const float* y;        // q|k|v projection outputs [S][y_ld], natural rows
  int y_ld, S, Hq, Hkv, d;
  const int* pos;        // [S] RoPE positions
  int max_position;
  const float2* rope;    // [max_position][d/2]
  float* q;              // [S][Hq*d] rotated queries
  uint16_t* kpool;       // this layer's K pool [n_rows][Hkv][cap][d]
  uint16_t* vpool;
  int row, cap, slot0;   // the row and the position in it of the first new entry
  const int* bt_row;     // the row's beam table
  const uint8_t* mask;   // the row's attention mask
  int P;                 // entries before the first token of this chunk
  uint16_t* attn;        // [S][attn_ld] fp16 attention output
  int attn_ld;
};
cudaError_t launch_prefill_check(const int* token_ids, int vocab, const int* pos, int max_position, const uint8_t* mask,
                                 int P, int S, int* status, cudaStream_t s);
cudaError_t launch_prefill_embed(const uint16_t* hidden_in, const int* token_ids, const uint16_t* embedding, int H,
                                 int S, int vocab, float* x, cudaStream_t s);
cudaError_t launch_prefill_norm(const float* x, int H, const uint16_t* w, float eps, uint16_t* act, int act_ld, int S,
                                cudaStream_t s);
cudaError_t launch_prefill_rope_append(const PrefillLayerArgs& a, cudaStream_t s);
cudaError_t launch_prefill_attention(const PrefillLayerArgs& a, cudaStream_t s);
cudaError_t launch_prefill_swiglu(const float* y, int y_ld, int S, int F, uint16_t* h, int h_ld, cudaStream_t s);
cudaError_t launch_prefill_residual(float* x, const float* y, int y_ld, int S, int H, uint16_t* out, cudaStream_t s);
cudaError_t launch_set_int(int* p, int v, cudaStream_t s);

struct PrologueArgs {
  int B, M;
  int n_new[kMaxRequests];
  int cursor[kMaxRequests];  // physical append position of each row
  const int* beam_idx;   // dev or nullptr
  const uint16_t* hidden_in;
  const int* token_ids;
  const int* position_ids;
  const uint8_t* mask;
  int mask_stride;
  int packed;            // the mask has one row per token (one request): shard_step_packed
  uint16_t* hidden_out;
  const int* bt_src;
  int* bt_dst;
  int* lens;             // [n_rows] row lengths (updated at the end of the step)
  int cap, max_position, vocab, H;
  const uint16_t* embedding;
  int* status;
};

// A projection's unit stream as the device code walks it.
struct OpDesc {
  const uint8_t* units;
  int n_rb, upr;
  // Work split.  q = 0: the unit stream is cut into one contiguous run per
  // warp of the grid.  q > 0 (whole-step kernel, gate|up): row-block rb
  // belongs to one CTA, whose q warps take its units in q contiguous K
  // ranges and reduce them in shared memory (set only when every row-block
  // of the projection finds its CTA in one round).
  int q;
};

// Arguments of the whole-step kernel (step_kernel.cu).
struct StepKernelArgs {
  PrologueArgs pro;          // per-step values
  const OpDesc* ops;         // [4 * L]: q|k|v, o, gate|up, down of each layer
  int L, H, Hq, Hkv, d, F, Kp_H, Kp_dq, Kp_F;
  float eps;
  const uint16_t* norms;     // [L][2][H]
  const float2* rope;        // [max_position][d/2]
  long long* X;              // residual [16][H], fixed point
  long long* acc_qkv;        // [16][qkv rows], zero between steps
  long long* acc_gu;         // [16][gate|up rows], zero between steps
  int* cnt_kv;               // [Hkv] q|k|v units finished per kv head, zero between steps
  int* cnt_gu;               // [gate|up row-blocks], zero between steps
  uint16_t* act_h;           // [16][Kp_H] (normalised rows, when they do not fit in shared memory)
  uint16_t* act_attn;        // [16][Kp_dq]
  uint16_t* act_f;           // [16][Kp_F]
  uint16_t* kpool;           // [L][n_rows][Hkv][cap][d]
  uint16_t* vpool;
  size_t layer_stride;
  int cap, n_chunks;         // items per row at kAttnChunkMin entries (the partials layout)
  const uint8_t* mask;
  int mask_stride;
  int packed;                // mask row per token (one request), no implicit causal bound
  float* attn_part;          // [B][Hkv][n_chunks][16*G][d+4]
  int* attn_cnt;             // [16][Hkv] finished chunks per (request, kv head); zero, self-resetting
  int* status;
  unsigned long long* barrier;         // grid-barrier counter (monotonic)
  unsigned long long barrier_base;     // its value when this launch starts
  unsigned long long* phase_clock;     // [step_barriers(L) + 1] globaltimer at each barrier
  int* status_out;           // host-mapped mirror: the last CTA to finish copies a nonzero status there
  int* exit_count;           // CTAs finished in this launch (zero between launches; the last resets it)
  int debug_skip_arrival;    // test knob: >= 0 makes CTA 1 skip that grid barrier's arrival
  unsigned wait_limit;       // polls before a cross-CTA wait gives up
  int gu_part;               // 1: shared memory holds the gate|up partial sums (OpDesc::q may be used)
};
// One-time attribute setup of the step kernel variants for a group size and
// head dim; number of grid barriers per step; launch (cooperative, one CTA
// per SM).
cudaError_t step_setup(int group, int head_dim);
// Warps per row-block for the shared-memory reduction of a gate|up
// projection of n_rb row-blocks of upr units on `grid` CTAs (0: the
// grid-wide split), when the kernel's shared memory for L layers leaves room
// for the partial sums.
int step_gu_split(int n_rb, int upr, int grid, int group, int L);
// Token count up to which the whole-step kernel uses that reduction.
int step_gu_cta_tokens();
// Whether the kernel's shared memory for L layers has room for the partial sums.
bool step_gu_part_fits(int group, int L);
int step_barriers(int n_layers);
cudaError_t launch_step(const StepKernelArgs& a, int nt, int group, int grid, cudaStream_t s);
size_t step_attention_part_floats(int B, int Hkv, int n_chunks, int G, int d);
constexpr int kAttnChunk = 64;     // most cache entries per attention item
constexpr int kAttnChunkMin = 32;  // fewest (partials are laid out for this many per item)

// Weight repacking (one fused op; all source pointers device).
// Source matrices of a fused op (q, k, v for OP_QKV; gate, up for OP_GU; one
// matrix otherwise), in the boundary's packed format, on the device.
struct RepackSrc {
  const uint8_t* codes[3];
  const uint16_t* scales[3];
  const uint8_t* zeros[3];
  int rows[3];
};
// rowmap: dev int [n_rb * 64]; entry = (source << 24) | source row, or -1.
cudaError_t launch_repack(const PackedOp& op, const int* rowmap, const RepackSrc& src, cudaStream_t s);
// Debug: dequantise an op back to natural order y[natural row][k] (fp32).
cudaError_t launch_unpack(const PackedOp& op, float* out, int ld, cudaStream_t s);

// KV utilities
cudaError_t launch_kv_gather(const uint16_t* pool, int n_layers, size_t layer_stride, int Hkv, int cap, int d,
                             const int* slots, int n, uint16_t* out /* [n_layers][n][Hkv][d] */, cudaStream_t s);
cudaError_t launch_kv_scatter(uint16_t* pool, int n_layers, size_t layer_stride, int Hkv, int cap, int d, int row,
                              const uint16_t* in /* [n_layers][n][Hkv][d] */, int n, cudaStream_t s);
cudaError_t launch_fill_identity(int* bt, int n_rows, int cap, int row /* -1 = all */, cudaStream_t s);

}  // namespace shard
