// Host side of libshard: the C ABI declared in include/shard.h and
// include/shard_debug.h.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <memory>
#include <string>
#include <vector>

#include "../../include/shard.h"
#include "../../include/shard_debug.h"
#include "common.cuh"

using namespace shard;

namespace {

thread_local std::string g_error;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_error = buf;
  return code;
}

#define CUDA_TRY(expr)                                                                        \
  do {                                                                                        \
    cudaError_t _e = (expr);                                                                  \
    if (_e != cudaSuccess)                                                                    \
      return fail(_e == cudaErrorMemoryAllocation ? SHARD_ENOMEM : SHARD_ECUDA, "%s: %s (%s:%d)", #expr, \
                  cudaGetErrorString(_e), __FILE__, __LINE__);                                \
  } while (0)

template <class T>
struct DevBuf {
  T* p = nullptr;
  size_t n = 0;
  ~DevBuf() {
    if (p) cudaFree(p);
  }
  cudaError_t alloc(size_t count) {
    n = count;
    return cudaMalloc(reinterpret_cast<void**>(&p), sizeof(T) * (count ? count : 1));
  }
};

std::string status_message(int bits) {
  std::string s;
  if (bits & ST_BEAM_IDX) s += "beam_idx entry outside [0, B); ";
  if (bits & ST_CAPACITY) s += "append would exceed the KV capacity; ";
  if (bits & ST_MASK_NEW) s += "attention_mask is 0 at a new entry; ";
  if (bits & ST_MASK_STRIDE) s += "mask_stride smaller than a row's length after the step; ";
  if (bits & ST_POSITION) s += "position id outside [0, max_position); ";
  if (bits & ST_TOKEN) s += "token id outside [0, vocab); ";
  if (bits & ST_WAIT_TIMEOUT) s += "pipeline wait timed out; ";
  return s;
}

}  // namespace

struct shard_s {
  int device = 0;
  shard_config cfg{};
  int num_sms = 0;
  int H = 0, Hq = 0, Hkv = 0, d = 0, F = 0, L = 0, dq = 0, dkv = 0;
  int Kp_H = 0, Kp_dq = 0, Kp_F = 0;
  std::vector<PackedOp> ops;      // [L][N_OPS]
  uint8_t* weight_pool = nullptr;  // all units of all layers
  size_t weight_bytes = 0;
  uint16_t* norms = nullptr;       // [L][2][H]
  uint16_t* embedding = nullptr;   // [V][H]
  float2* rope = nullptr;          // [max_position][d/2]
  // per-step work buffers (one set per shard); sums and counts are zero
  // between launches (each launch leaves them so)
  long long* X = nullptr;          // residual [16][H], fixed point
  long long* acc_qkv = nullptr;    // [16][qkv rows]
  long long* acc_gu = nullptr;     // [16][gate|up rows]
  long long* acc_store = nullptr;  // [16][max_rb * 64] (the standalone projection)
  int* cnt_kv = nullptr;           // [Hkv]
  int* cnt_gu = nullptr;           // [gate|up row-blocks]
  int* cnt_store = nullptr;        // [max_rb]
  int* attn_cnt = nullptr;         // [16][Hkv] attention chunks finished per (request, kv head)
  uint16_t* act_h = nullptr;       // [16][Kp_H]
  uint16_t* act_attn = nullptr;    // [16][Kp_dq]
  uint16_t* act_f = nullptr;       // [16][Kp_F]
  int max_rb = 0;
  size_t acc_qkv_n = 0, acc_gu_n = 0, acc_store_n = 0;
  int n_rb_gu = 0;
  // prefill work buffers, allocated at the first shard_prefill (chunks of kPrefillChunk tokens)
  float* pf_x = nullptr;           // [C][H] residual
  uint16_t* pf_act = nullptr;      // [C][Kp_H] normalised rows (padding zero)
  uint16_t* pf_attn = nullptr;     // [C][Kp_dq] attention output (padding zero)
  uint16_t* pf_h = nullptr;        // [C][Kp_F] SwiGLU output (padding zero)
  float* pf_y = nullptr;           // [C][max projection rows] projection outputs
  float* pf_q = nullptr;           // [C][dq] rotated queries
  int debug_skip_arrival = -1;     // test knob (shard_debug_set_wait)
  unsigned wait_limit = 1u << 22;  // polls before a cross-CTA wait gives up
  int* status = nullptr;           // device status word
  int* status_host = nullptr;      // host-mapped mirror the step kernel writes a nonzero status to
  int* status_host_dev = nullptr;  // its device address
  int* exit_count = nullptr;       // step kernel: CTAs finished (zero between launches)
  int grid[3] = {0, 0, 0};         // standalone GEMV grid per token bucket
  OpDesc* ops_dev = nullptr;       // [4L] op descriptors for the step kernel
  unsigned long long* barrier = nullptr;  // grid-barrier counter
  unsigned long long barrier_base = 0;    // its value at the next launch
  unsigned long long* phase_clock = nullptr;  // [8L + 1]
  int n_barriers = 0;
  // staging for shard_step_host
  void* pin = nullptr;
  size_t pin_bytes = 0;
  void* dstage = nullptr;
  size_t dstage_bytes = 0;
  std::vector<kvstate_s*> states;
};

struct kvstate_s {
  shard_s* sh = nullptr;
  int n_rows = 0, cap = 0;
  uint16_t* k = nullptr;  // [L][n_rows][Hkv][cap][d]
  uint16_t* v = nullptr;
  size_t layer_stride = 0;
  int* bt[2] = {nullptr, nullptr};
  int bt_cur = 0;
  int* lens = nullptr;    // device [n_rows]
  std::vector<int> cursor, len_host;
  bool shared = false;    // rows may share entries (a beam gather ran)
  bool poisoned = false;  // a step aborted on the device
  int n_chunks = 0;       // attention items per row at the smallest item size (kAttnChunkMin)
  float* attn_part = nullptr;
};

namespace {

void free_state(kvstate_s* st) {
  if (!st) return;
  cudaFree(st->k);
  cudaFree(st->v);
  cudaFree(st->bt[0]);
  cudaFree(st->bt[1]);
  cudaFree(st->lens);
  cudaFree(st->attn_part);
  delete st;
}

int round_up(int v, int m) { return (v + m - 1) / m * m; }

// Row maps of the fused projections (see kernels.h): entry = (source << 24) | row.
std::vector<int> build_rowmap(int kind, const shard_s& s, int n_rb) {
  std::vector<int> rm((size_t)n_rb * kRowsPerBlock, -1);
  if (kind == OP_QKV) {
    const int tph = s.d / 16, half = s.d / 2;
    int R = 0;
    for (int src = 0; src < 2; ++src) {
      const int heads = src == 0 ? s.Hq : s.Hkv;
      for (int h = 0; h < heads; ++h)
        for (int jt = 0; jt < tph; ++jt)
          for (int r = 0; r < 16; ++r, ++R) {
            const int dim = r < 8 ? 8 * jt + r : half + 8 * jt + (r - 8);
            rm[R] = (src << 24) | (h * s.d + dim);
          }
    }
    for (int e = 0; e < s.Hkv * s.d; ++e, ++R) rm[R] = (2 << 24) | e;
  } else if (kind == OP_GU) {
    const int tiles = (s.F + 7) / 8;
    for (int t = 0; t < tiles; ++t)
      for (int r = 0; r < 16; ++r) {
        const int j = 8 * t + (r & 7);
        if (j < s.F) rm[(size_t)t * 16 + r] = ((r < 8 ? 0 : 1) << 24) | j;
      }
  } else {
    for (int R = 0; R < s.H; ++R) rm[R] = R;
  }
  return rm;
}

int op_rows(int kind, const shard_s& s) {
  switch (kind) {
    case OP_QKV: return (s.Hq + 2 * s.Hkv) * s.d;
    case OP_GU: return ((s.F + 7) / 8) * 16;
    default: return s.H;
  }
}
int op_K(int kind, const shard_s& s) {
  switch (kind) {
    case OP_O: return s.dq;
    case OP_DOWN: return s.F;
    default: return s.H;
  }
}

int nt_for(int M) { return M <= 8 ? 1 : 2; }

// After a wait that gave up, the launch's sums, counts and grid-barrier
// count are left in an unknown state: put every work buffer back to zero.
cudaError_t reset_work_buffers(shard_s* sh) {
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemset(sh->acc_qkv, 0, sizeof(long long) * sh->acc_qkv_n);
  if (e == cudaSuccess) e = cudaMemset(sh->acc_gu, 0, sizeof(long long) * sh->acc_gu_n);
  if (e == cudaSuccess) e = cudaMemset(sh->acc_store, 0, sizeof(long long) * sh->acc_store_n);
  if (e == cudaSuccess) e = cudaMemset(sh->cnt_kv, 0, sizeof(int) * sh->Hkv);
  if (e == cudaSuccess) e = cudaMemset(sh->cnt_gu, 0, sizeof(int) * sh->n_rb_gu);
  if (e == cudaSuccess) e = cudaMemset(sh->cnt_store, 0, sizeof(int) * sh->max_rb);
  if (e == cudaSuccess) e = cudaMemset(sh->attn_cnt, 0, sizeof(int) * kMaxRequests * sh->Hkv);
  if (e == cudaSuccess) e = cudaMemset(sh->exit_count, 0, sizeof(int));
  if (e == cudaSuccess) e = cudaMemset(sh->barrier, 0, sizeof(unsigned long long));
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  sh->barrier_base = 0;
  return e;
}

// Frees everything a shard holds -- its kv states, device buffers and pinned
// staging -- and the shard itself, on the current device after its work has
// finished.  Buffers never allocated are null and skipped, so this also
// undoes a shard_create that failed part-way.
void release_shard(shard_s* sh) {
  cudaDeviceSynchronize();
  for (auto* st : sh->states) free_state(st);
  cudaFree(sh->weight_pool);
  cudaFree(sh->norms);
  cudaFree(sh->embedding);
  cudaFree(sh->rope);
  cudaFree(sh->pf_x);
  cudaFree(sh->pf_act);
  cudaFree(sh->pf_attn);
  cudaFree(sh->pf_h);
  cudaFree(sh->pf_y);
  cudaFree(sh->pf_q);
  cudaFree(sh->X);
  cudaFree(sh->acc_qkv);
  cudaFree(sh->acc_gu);
  cudaFree(sh->acc_store);
  cudaFree(sh->cnt_kv);
  cudaFree(sh->cnt_gu);
  cudaFree(sh->cnt_store);
  cudaFree(sh->attn_cnt);
  cudaFree(sh->act_h);
  cudaFree(sh->act_attn);
  cudaFree(sh->act_f);
  cudaFree(sh->status);
  cudaFree(sh->exit_count);
  cudaFree(sh->dstage);
  if (sh->pin) cudaFreeHost(sh->pin);
  if (sh->status_host) cudaFreeHost(sh->status_host);
  cudaFree(sh->ops_dev);
  cudaFree(sh->barrier);
  cudaFree(sh->phase_clock);
  delete sh;
}

struct ShardRelease {
  void operator()(shard_s* sh) const { release_shard(sh); }
};

int check_pending_status(shard_s* sh) {
  const int bits = *reinterpret_cast<volatile int*>(sh->status_host);
  if (bits) {
    *reinterpret_cast<volatile int*>(sh->status_host) = 0;
    for (auto* st : sh->states) st->poisoned = true;
    if (bits & ST_WAIT_TIMEOUT) reset_work_buffers(sh);
    return fail(SHARD_EINVAL, "an earlier step was rejected on the device: %s", status_message(bits).c_str());
  }
  return SHARD_OK;
}

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================

extern "C" {

const char* shard_last_error(void) { return g_error.c_str(); }

int shard_create(const shard_config* cfg, const shard_weights_host* w, shard_t* out) {
  if (!cfg || !w || !out || !w->layers) return fail(SHARD_EINVAL, "shard_create: null argument");
  *out = nullptr;
  const shard_config& c = *cfg;
  if (c.n_layers < 1 || c.hidden < 16 || c.n_heads < 1 || c.n_kv_heads < 1 || c.head_dim < 16 || c.ffn < 1 ||
      c.max_position < 1 || c.vocab < 0 || !(c.rms_eps >= 0) || !(c.rope_theta > 0))
    return fail(SHARD_EINVAL, "shard_create: invalid dimensions");
  if (c.n_heads % c.n_kv_heads) return fail(SHARD_EINVAL, "n_heads must be a multiple of n_kv_heads");
  if (c.head_dim % 16) return fail(SHARD_EUNSUPPORTED, "head_dim must be a multiple of 16");
  if (c.group != 32 && c.group != 64 && c.group != 128) return fail(SHARD_EUNSUPPORTED, "group must be 32, 64 or 128");
  if (c.hidden % 8 || (c.n_heads * c.head_dim) % 8) return fail(SHARD_EUNSUPPORTED, "hidden must be a multiple of 8");
  if (c.n_heads / c.n_kv_heads * kMaxTokens > 256) return fail(SHARD_EUNSUPPORTED, "n_heads / n_kv_heads must be <= 16");
  if (c.vocab > 0 && !w->embedding) return fail(SHARD_EINVAL, "vocab > 0 needs an embedding");

  // a failure below returns through the deleter, which frees what was allocated so far
  auto sh = std::unique_ptr<shard_s, ShardRelease>(new shard_s());
  CUDA_TRY(cudaGetDevice(&sh->device));
  CUDA_TRY(cudaDeviceGetAttribute(&sh->num_sms, cudaDevAttrMultiProcessorCount, sh->device));
  if (c.head_dim != 64 && c.head_dim != 128) return fail(SHARD_EUNSUPPORTED, "head_dim must be 64 or 128");
  CUDA_TRY(gemv_setup());
  CUDA_TRY(gemm_tc_setup());
  CUDA_TRY(step_setup(c.group, c.head_dim));
  sh->cfg = c;
  sh->H = c.hidden;
  sh->Hq = c.n_heads;
  sh->Hkv = c.n_kv_heads;
  sh->d = c.head_dim;
  sh->F = c.ffn;
  sh->L = c.n_layers;
  sh->dq = sh->Hq * sh->d;
  sh->dkv = sh->Hkv * sh->d;
  sh->Kp_H = round_up(sh->H, kUnitK);
  sh->Kp_dq = round_up(sh->dq, kUnitK);
  sh->Kp_F = round_up(sh->F, kUnitK);
  const int ub = unit_bytes_for_group(c.group);

  // Geometry of each op and the pool size.
  sh->ops.resize((size_t)sh->L * N_OPS);
  size_t total = 0;
  for (int l = 0; l < sh->L; ++l)
    for (int k = 0; k < N_OPS; ++k) {
      PackedOp& op = sh->ops[(size_t)l * N_OPS + k];
      op.rows = op_rows(k, *sh);
      op.K = op_K(k, *sh);
      op.Kp = round_up(op.K, kUnitK);
      op.n_rb = (op.rows + kRowsPerBlock - 1) / kRowsPerBlock;
      op.upr = op.Kp / kUnitK;
      op.unit_bytes = ub;
      op.group = c.group;
      op.bytes = (size_t)op.n_rb * op.upr * ub;
      op.dims = OpDims{k, sh->Hq, sh->Hkv, sh->d, sh->F, sh->H};
      // the device splits the unit stream with 32-bit arithmetic
      if (((uint64_t)op.n_rb * op.upr + 1) * ((uint64_t)sh->num_sms * gemv_warps_per_cta()) >= (1ull << 32))
        return fail(SHARD_EUNSUPPORTED, "a projection has too many units for this GPU's warp count");
      total += op.bytes;
      sh->max_rb = std::max(sh->max_rb, op.n_rb);
    }
  sh->weight_bytes = total;
  CUDA_TRY(cudaMalloc(&sh->weight_pool, total));
  {
    size_t off = 0;
    for (auto& op : sh->ops) {
      op.units = sh->weight_pool + off;
      off += op.bytes;
    }
  }

  // Upload and repack, op by op.
  {
    cudaStream_t s = nullptr;
    size_t max_src = 0;
    for (int k = 0; k < N_OPS; ++k) {
      const PackedOp& op = sh->ops[k];
      const int G = (op.K + c.group - 1) / c.group;
      const size_t per_row = (size_t)(op.K + 1) / 2 + (size_t)G * 2 + (size_t)(G + 1) / 2;
      max_src = std::max(max_src, per_row * (size_t)op.rows);
    }
    DevBuf<uint8_t> src;
    DevBuf<int> rowmap;
    CUDA_TRY(src.alloc(max_src + 3 * 256));
    CUDA_TRY(rowmap.alloc((size_t)sh->max_rb * kRowsPerBlock));
    for (int l = 0; l < sh->L; ++l) {
      const shard_layer_host& lw = w->layers[l];
      for (int k = 0; k < N_OPS; ++k) {
        PackedOp& op = sh->ops[(size_t)l * N_OPS + k];
        int mats[3] = {-1, -1, -1}, nm = 0;
        int rows[3] = {0, 0, 0};
        if (k == OP_QKV) {
          mats[0] = SHARD_Q; mats[1] = SHARD_K; mats[2] = SHARD_V; nm = 3;
          rows[0] = sh->dq; rows[1] = sh->dkv; rows[2] = sh->dkv;
        } else if (k == OP_GU) {
          mats[0] = SHARD_GATE; mats[1] = SHARD_UP; nm = 2;
          rows[0] = rows[1] = sh->F;
        } else {
          mats[0] = (k == OP_O) ? SHARD_O : SHARD_DOWN; nm = 1;
          rows[0] = sh->H;
        }
        const int G = (op.K + c.group - 1) / c.group;
        const size_t cb = (size_t)(op.K + 1) / 2, sb = (size_t)G * 2, zb = (size_t)(G + 1) / 2;
        RepackSrc rs{};
        size_t off = 0;
        for (int i = 0; i < nm; ++i) {
          const shard_matrix_host& m = lw.w[mats[i]];
          if (!m.codes || !m.scales || !m.zeros) return fail(SHARD_EINVAL, "layer %d matrix %d: null pointer", l, mats[i]);
          auto put = [&](const void* hp, size_t bytes) -> uint8_t* {
            off = (off + 255) / 256 * 256;
            uint8_t* dp = src.p + off;
            off += bytes;
            return cudaMemcpy(dp, hp, bytes, cudaMemcpyHostToDevice) == cudaSuccess ? dp : nullptr;
          };
          rs.codes[i] = put(m.codes, cb * rows[i]);
          rs.scales[i] = reinterpret_cast<const uint16_t*>(put(m.scales, sb * rows[i]));
          rs.zeros[i] = put(m.zeros, zb * rows[i]);
          rs.rows[i] = rows[i];
          if (!rs.codes[i] || !rs.scales[i] || !rs.zeros[i]) return fail(SHARD_ECUDA, "weight upload failed");
        }
        std::vector<int> rm = build_rowmap(k, *sh, op.n_rb);
        CUDA_TRY(cudaMemcpy(rowmap.p, rm.data(), rm.size() * sizeof(int), cudaMemcpyHostToDevice));
        CUDA_TRY(launch_repack(op, rowmap.p, rs, s));
        CUDA_TRY(cudaDeviceSynchronize());
      }
    }
  }

  // Norm weights, embedding, rotary table.
  CUDA_TRY(cudaMalloc(&sh->norms, sizeof(uint16_t) * (size_t)sh->L * 2 * sh->H));
  for (int l = 0; l < sh->L; ++l) {
    if (!w->layers[l].attn_norm || !w->layers[l].ffn_norm) return fail(SHARD_EINVAL, "layer %d: null norm", l);
    CUDA_TRY(cudaMemcpy(sh->norms + (size_t)l * 2 * sh->H, w->layers[l].attn_norm, sizeof(uint16_t) * sh->H,
                        cudaMemcpyHostToDevice));
    CUDA_TRY(cudaMemcpy(sh->norms + (size_t)l * 2 * sh->H + sh->H, w->layers[l].ffn_norm, sizeof(uint16_t) * sh->H,
                        cudaMemcpyHostToDevice));
  }
  if (c.vocab > 0) {
    CUDA_TRY(cudaMalloc(&sh->embedding, sizeof(uint16_t) * (size_t)c.vocab * sh->H));
    CUDA_TRY(cudaMemcpy(sh->embedding, w->embedding, sizeof(uint16_t) * (size_t)c.vocab * sh->H,
                        cudaMemcpyHostToDevice));
  }
  {
    // cos/sin of pos * theta^(-2i/d), computed in double, stored as fp32.
    const int pairs = sh->d / 2;
    std::vector<float2> tab((size_t)c.max_position * pairs);
    for (int p = 0; p < c.max_position; ++p)
      for (int i = 0; i < pairs; ++i) {
        const double ang = (double)p * std::pow(c.rope_theta, -2.0 * i / sh->d);
        tab[(size_t)p * pairs + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
      }
    CUDA_TRY(cudaMalloc(&sh->rope, sizeof(float2) * tab.size()));
    CUDA_TRY(cudaMemcpy(sh->rope, tab.data(), sizeof(float2) * tab.size(), cudaMemcpyHostToDevice));
  }

  // Work buffers.
  CUDA_TRY(cudaMalloc(&sh->X, sizeof(long long) * kMaxTokens * sh->H));
  sh->acc_qkv_n = (size_t)kMaxTokens * (sh->dq + 2 * sh->dkv);
  sh->n_rb_gu = sh->ops[OP_GU].n_rb;
  sh->acc_gu_n = (size_t)kMaxTokens * sh->n_rb_gu * kRowsPerBlock;
  sh->acc_store_n = (size_t)kMaxTokens * sh->max_rb * kRowsPerBlock;
  CUDA_TRY(cudaMalloc(&sh->acc_qkv, sizeof(long long) * sh->acc_qkv_n));
  CUDA_TRY(cudaMalloc(&sh->acc_gu, sizeof(long long) * sh->acc_gu_n));
  CUDA_TRY(cudaMalloc(&sh->acc_store, sizeof(long long) * sh->acc_store_n));
  CUDA_TRY(cudaMalloc(&sh->cnt_kv, sizeof(int) * sh->Hkv));
  CUDA_TRY(cudaMalloc(&sh->cnt_gu, sizeof(int) * sh->n_rb_gu));
  CUDA_TRY(cudaMalloc(&sh->cnt_store, sizeof(int) * sh->max_rb));
  CUDA_TRY(cudaMalloc(&sh->attn_cnt, sizeof(int) * kMaxRequests * sh->Hkv));
  CUDA_TRY(cudaMalloc(&sh->act_h, sizeof(uint16_t) * kMaxTokens * sh->Kp_H));
  CUDA_TRY(cudaMalloc(&sh->act_attn, sizeof(uint16_t) * kMaxTokens * sh->Kp_dq));
  CUDA_TRY(cudaMalloc(&sh->act_f, sizeof(uint16_t) * kMaxTokens * sh->Kp_F));
  CUDA_TRY(cudaMemset(sh->act_h, 0, sizeof(uint16_t) * kMaxTokens * sh->Kp_H));
  CUDA_TRY(cudaMemset(sh->act_attn, 0, sizeof(uint16_t) * kMaxTokens * sh->Kp_dq));
  CUDA_TRY(cudaMemset(sh->act_f, 0, sizeof(uint16_t) * kMaxTokens * sh->Kp_F));
  for (int nt = 1; nt <= 2; ++nt) sh->grid[nt] = gemv_grid(nt, sh->num_sms);
  CUDA_TRY(cudaMalloc(&sh->status, sizeof(int)));
  CUDA_TRY(cudaMemset(sh->status, 0, sizeof(int)));
  CUDA_TRY(cudaHostAlloc(&sh->status_host, sizeof(int), cudaHostAllocMapped));
  *sh->status_host = 0;
  CUDA_TRY(cudaHostGetDevicePointer(reinterpret_cast<void**>(&sh->status_host_dev), sh->status_host, 0));
  CUDA_TRY(cudaMalloc(&sh->exit_count, sizeof(int)));
  CUDA_TRY(cudaMemset(sh->exit_count, 0, sizeof(int)));
  {
    std::vector<OpDesc> od(sh->ops.size());
    for (size_t i = 0; i < od.size(); ++i) {
      const auto& o = sh->ops[i];
      // gate|up (op 2 of each layer): shared-memory reduction when it fits
      const int q = i % 4 == 2 ? step_gu_split(o.n_rb, o.upr, sh->num_sms, sh->cfg.group, sh->L) : 0;
      od[i] = OpDesc{o.units, o.n_rb, o.upr, q};
    }
    CUDA_TRY(cudaMalloc(&sh->ops_dev, sizeof(OpDesc) * od.size()));
    CUDA_TRY(cudaMemcpy(sh->ops_dev, od.data(), sizeof(OpDesc) * od.size(), cudaMemcpyHostToDevice));
  }
  sh->n_barriers = step_barriers(sh->L);
  CUDA_TRY(cudaMalloc(&sh->barrier, sizeof(unsigned long long)));
  CUDA_TRY(cudaMalloc(&sh->phase_clock, sizeof(unsigned long long) * (sh->n_barriers + 1)));
  CUDA_TRY(cudaMemset(sh->phase_clock, 0, sizeof(unsigned long long) * (sh->n_barriers + 1)));
  CUDA_TRY(reset_work_buffers(sh.get()));
  *out = sh.release();
  return SHARD_OK;
}

int shard_destroy(shard_t sh) {
  if (!sh) return fail(SHARD_EINVAL, "shard_destroy: null shard");
  cudaSetDevice(sh->device);
  release_shard(sh);
  return SHARD_OK;
}

int kv_state_alloc(shard_t sh, int n_rows, int capacity, kvstate_t* out) {
  if (!sh || !out) return fail(SHARD_EINVAL, "kv_state_alloc: null argument");
  if (n_rows < 1 || n_rows > SHARD_MAX_REQUESTS) return fail(SHARD_EINVAL, "n_rows must be in [1, %d]", SHARD_MAX_REQUESTS);
  if (capacity < 1 || (long long)n_rows * capacity >= (1LL << 31)) return fail(SHARD_EINVAL, "invalid capacity");
  CUDA_TRY(cudaSetDevice(sh->device));
  auto st = new kvstate_s();
  st->sh = sh;
  st->n_rows = n_rows;
  st->cap = capacity;
  st->layer_stride = (size_t)n_rows * sh->Hkv * capacity * sh->d;
  const size_t pool = st->layer_stride * sh->L;
  st->cursor.assign(n_rows, 0);
  st->len_host.assign(n_rows, 0);
  st->n_chunks = (capacity + kAttnChunkMin - 1) / kAttnChunkMin;
  int rc = SHARD_OK;
  auto chk = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == SHARD_OK)
      rc = fail(e == cudaErrorMemoryAllocation ? SHARD_ENOMEM : SHARD_ECUDA, "kv_state_alloc: %s", cudaGetErrorString(e));
  };
  chk(cudaMalloc(&st->k, sizeof(uint16_t) * pool));
  chk(cudaMalloc(&st->v, sizeof(uint16_t) * pool));
  chk(cudaMalloc(&st->bt[0], sizeof(int) * (size_t)n_rows * capacity));
  chk(cudaMalloc(&st->bt[1], sizeof(int) * (size_t)n_rows * capacity));
  chk(cudaMalloc(&st->lens, sizeof(int) * n_rows));
  const int G = sh->Hq / sh->Hkv;
  chk(cudaMalloc(&st->attn_part, sizeof(float) * step_attention_part_floats(n_rows, sh->Hkv, st->n_chunks, G, sh->d)));
  if (rc == SHARD_OK) {
    chk(cudaMemset(st->lens, 0, sizeof(int) * n_rows));
    chk(cudaMemset(st->k, 0, sizeof(uint16_t) * pool));
    chk(cudaMemset(st->v, 0, sizeof(uint16_t) * pool));
    chk(launch_fill_identity(st->bt[0], n_rows, capacity, -1, nullptr));
    chk(launch_fill_identity(st->bt[1], n_rows, capacity, -1, nullptr));
    chk(cudaDeviceSynchronize());
  }
  if (rc != SHARD_OK) {
    free_state(st);
    return rc;
  }
  sh->states.push_back(st);
  *out = st;
  return SHARD_OK;
}

int kv_state_free(kvstate_t st) {
  if (!st) return fail(SHARD_EINVAL, "null state");
  shard_s* sh = st->sh;
  cudaSetDevice(sh->device);
  cudaDeviceSynchronize();
  for (size_t i = 0; i < sh->states.size(); ++i)
    if (sh->states[i] == st) {
      sh->states.erase(sh->states.begin() + i);
      break;
    }
  free_state(st);
  return SHARD_OK;
}

int kv_state_reset(kvstate_t st, int row) {
  if (!st) return fail(SHARD_EINVAL, "null state");
  if (row < -1 || row >= st->n_rows) return fail(SHARD_EINVAL, "row %d out of range", row);
  CUDA_TRY(cudaSetDevice(st->sh->device));
  CUDA_TRY(cudaDeviceSynchronize());
  if (row == -1) {
    CUDA_TRY(cudaMemset(st->lens, 0, sizeof(int) * st->n_rows));
    CUDA_TRY(launch_fill_identity(st->bt[0], st->n_rows, st->cap, -1, nullptr));
    CUDA_TRY(launch_fill_identity(st->bt[1], st->n_rows, st->cap, -1, nullptr));
    st->cursor.assign(st->n_rows, 0);
    st->len_host.assign(st->n_rows, 0);
    st->bt_cur = 0;
    st->shared = false;
    st->poisoned = false;
  } else {
    if (st->shared) return fail(SHARD_EUNSUPPORTED, "rows share entries after a beam gather; reset all rows (-1)");
    CUDA_TRY(cudaMemset(st->lens + row, 0, sizeof(int)));
    CUDA_TRY(launch_fill_identity(st->bt[st->bt_cur], st->n_rows, st->cap, row, nullptr));
    st->cursor[row] = 0;
    st->len_host[row] = 0;
  }
  CUDA_TRY(cudaDeviceSynchronize());
  return SHARD_OK;
}

int kv_state_load(kvstate_t st, int row, int layer, const uint16_t* k, const uint16_t* v, int len) {
  if (!st || !k || !v) return fail(SHARD_EINVAL, "kv_state_load: null argument");
  shard_s* sh = st->sh;
  if (row < 0 || row >= st->n_rows || layer < 0 || layer >= sh->L || len < 0)
    return fail(SHARD_EINVAL, "kv_state_load: row/layer/len out of range");
  if (len > st->cap) return fail(SHARD_ECAPACITY, "kv_state_load: len %d > capacity %d", len, st->cap);
  if (st->shared) return fail(SHARD_EUNSUPPORTED, "rows share entries after a beam gather; reset all rows (-1) first");
  CUDA_TRY(cudaSetDevice(sh->device));
  CUDA_TRY(cudaDeviceSynchronize());
  const size_t d2 = sizeof(uint16_t) * sh->d;
  for (int h = 0; h < sh->Hkv; ++h) {
    const size_t off = (size_t)layer * st->layer_stride + (((size_t)row * sh->Hkv + h) * st->cap) * sh->d;
    if (len > 0) {
      CUDA_TRY(cudaMemcpy2D(st->k + off, d2, k + (size_t)h * sh->d, d2 * sh->Hkv, d2, len, cudaMemcpyHostToDevice));
      CUDA_TRY(cudaMemcpy2D(st->v + off, d2, v + (size_t)h * sh->d, d2 * sh->Hkv, d2, len, cudaMemcpyHostToDevice));
    }
  }
  CUDA_TRY(launch_fill_identity(st->bt[st->bt_cur], st->n_rows, st->cap, row, nullptr));
  CUDA_TRY(cudaMemcpy(st->lens + row, &len, sizeof(int), cudaMemcpyHostToDevice));
  st->cursor[row] = len;
  st->len_host[row] = len;
  CUDA_TRY(cudaDeviceSynchronize());
  return SHARD_OK;
}

int kv_state_length(kvstate_t st, int row, int* len) {
  if (!st || !len || row < 0 || row >= st->n_rows) return fail(SHARD_EINVAL, "kv_state_length: bad argument");
  CUDA_TRY(cudaSetDevice(st->sh->device));
  CUDA_TRY(cudaDeviceSynchronize());
  CUDA_TRY(cudaMemcpy(len, st->lens + row, sizeof(int), cudaMemcpyDeviceToHost));
  return SHARD_OK;
}

int kv_state_read(kvstate_t st, int row, int layer, int start, int len, uint16_t* k, uint16_t* v) {
  if (!st || !k || !v) return fail(SHARD_EINVAL, "kv_state_read: null argument");
  shard_s* sh = st->sh;
  if (row < 0 || row >= st->n_rows || layer < 0 || layer >= sh->L || start < 0 || len < 0)
    return fail(SHARD_EINVAL, "kv_state_read: row/layer/start/len out of range");
  int cur = 0;
  int rc = kv_state_length(st, row, &cur);
  if (rc) return rc;
  if ((long long)start + len > cur)
    return fail(SHARD_EINVAL, "kv_state_read: [%d, %d + %d) beyond row length %d", start, start, len, cur);
  if (len == 0) return SHARD_OK;
  DevBuf<uint16_t> tmp;
  CUDA_TRY(tmp.alloc((size_t)len * sh->Hkv * sh->d));
  const int* slots = st->bt[st->bt_cur] + (size_t)row * st->cap + start;
  for (int which = 0; which < 2; ++which) {
    const uint16_t* pool = (which == 0 ? st->k : st->v) + (size_t)layer * st->layer_stride;
    CUDA_TRY(launch_kv_gather(pool, 1, st->layer_stride, sh->Hkv, st->cap, sh->d, slots, len, tmp.p, nullptr));
    CUDA_TRY(cudaMemcpy(which == 0 ? k : v, tmp.p, sizeof(uint16_t) * tmp.n, cudaMemcpyDeviceToHost));
  }
  return SHARD_OK;
}

int kv_state_export(kvstate_t st, int row, const uint8_t* keep, int len, uint16_t* k, uint16_t* v, int* n_kept) {
  if (!st || !k || !v || !n_kept) return fail(SHARD_EINVAL, "kv_state_export: null argument");
  shard_s* sh = st->sh;
  if (row < 0 || row >= st->n_rows) return fail(SHARD_EINVAL, "kv_state_export: row out of range");
  int cur = 0;
  int rc = kv_state_length(st, row, &cur);
  if (rc) return rc;
  if (len != cur) return fail(SHARD_EINVAL, "kv_state_export: len %d != row length %d", len, cur);
  *n_kept = 0;
  if (len == 0) return SHARD_OK;
  // the row's slots (beam table), then the kept ones in cache order
  std::vector<int> all(len), slots;
  CUDA_TRY(cudaMemcpy(all.data(), st->bt[st->bt_cur] + (size_t)row * st->cap, sizeof(int) * len,
                      cudaMemcpyDeviceToHost));
  for (int j = 0; j < len; ++j)
    if (!keep || keep[j]) slots.push_back(all[j]);
  const int n = static_cast<int>(slots.size());
  if (n > 0) {
    DevBuf<int> dslots;
    DevBuf<uint16_t> tmp;
    CUDA_TRY(dslots.alloc(n));
    CUDA_TRY(cudaMemcpy(dslots.p, slots.data(), sizeof(int) * n, cudaMemcpyHostToDevice));
    CUDA_TRY(tmp.alloc((size_t)sh->L * n * sh->Hkv * sh->d));
    for (int which = 0; which < 2; ++which) {
      const uint16_t* pool = which == 0 ? st->k : st->v;
      CUDA_TRY(launch_kv_gather(pool, sh->L, st->layer_stride, sh->Hkv, st->cap, sh->d, dslots.p, n, tmp.p, nullptr));
      CUDA_TRY(cudaMemcpy(which == 0 ? k : v, tmp.p, sizeof(uint16_t) * tmp.n, cudaMemcpyDeviceToHost));
    }
  }
  *n_kept = n;
  return SHARD_OK;
}

int kv_state_import(kvstate_t st, int row, const uint16_t* k, const uint16_t* v, int len) {
  if (!st || ((!k || !v) && len > 0)) return fail(SHARD_EINVAL, "kv_state_import: null argument");
  shard_s* sh = st->sh;
  const size_t per_layer = (size_t)len * sh->Hkv * sh->d;
  for (int l = 0; l < sh->L; ++l) {
    int rc = kv_state_load(st, row, l, len > 0 ? k + (size_t)l * per_layer : k, len > 0 ? v + (size_t)l * per_layer : v,
                           len);
    if (rc) return rc;
  }
  return SHARD_OK;
}

int kv_trim(kvstate_t st, int row, const uint8_t* keep, int len) {
  if (!st || !keep) return fail(SHARD_EINVAL, "kv_trim: null argument");
  shard_s* sh = st->sh;
  if (row < 0 || row >= st->n_rows) return fail(SHARD_EINVAL, "kv_trim: row out of range");
  if (st->shared) return fail(SHARD_EUNSUPPORTED, "kv_trim: rows share entries after a beam gather");
  int cur = 0;
  int rc = kv_state_length(st, row, &cur);
  if (rc) return rc;
  if (len != cur) return fail(SHARD_EINVAL, "kv_trim: len %d != row length %d", len, cur);
  std::vector<int> slots;
  for (int j = 0; j < len; ++j)
    if (keep[j]) slots.push_back(row * st->cap + j);  // unshared rows map entry j to slot (row, j)
  const int n = static_cast<int>(slots.size());
  if (n > 0) {
    DevBuf<int> dslots;
    DevBuf<uint16_t> tmp;
    CUDA_TRY(dslots.alloc(n));
    CUDA_TRY(cudaMemcpy(dslots.p, slots.data(), sizeof(int) * n, cudaMemcpyHostToDevice));
    CUDA_TRY(tmp.alloc((size_t)sh->L * n * sh->Hkv * sh->d));
    for (int which = 0; which < 2; ++which) {
      uint16_t* pool = which == 0 ? st->k : st->v;
      CUDA_TRY(launch_kv_gather(pool, sh->L, st->layer_stride, sh->Hkv, st->cap, sh->d, dslots.p, n, tmp.p, nullptr));
      CUDA_TRY(launch_kv_scatter(pool, sh->L, st->layer_stride, sh->Hkv, st->cap, sh->d, row, tmp.p, n, nullptr));
    }
    CUDA_TRY(cudaDeviceSynchronize());
  }
  CUDA_TRY(launch_fill_identity(st->bt[st->bt_cur], st->n_rows, st->cap, row, nullptr));
  CUDA_TRY(cudaMemcpy(st->lens + row, &n, sizeof(int), cudaMemcpyHostToDevice));
  st->cursor[row] = n;
  st->len_host[row] = n;
  CUDA_TRY(cudaDeviceSynchronize());
  return SHARD_OK;
}

static int step_impl(shard_t sh, kvstate_t st, const uint16_t* hidden_in, const int32_t* token_ids,
                     const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* attention_mask,
                     int mask_stride, const int32_t* beam_idx, uint16_t* hidden_out, void* cuda_stream, int packed);

int shard_step(shard_t sh, kvstate_t st, const uint16_t* hidden_in, const int32_t* token_ids, const int32_t* n_new,
               int B, const int32_t* position_ids, const uint8_t* attention_mask, int mask_stride,
               const int32_t* beam_idx, uint16_t* hidden_out, void* cuda_stream) {
  return step_impl(sh, st, hidden_in, token_ids, n_new, B, position_ids, attention_mask, mask_stride, beam_idx,
                   hidden_out, cuda_stream, 0);
}

int shard_step_packed(shard_t sh, kvstate_t st, const uint16_t* hidden_in, const int32_t* token_ids, int S,
                      const int32_t* position_ids, const uint8_t* mask2d, int mask_stride, uint16_t* hidden_out,
                      void* cuda_stream) {
  if (!st || st->n_rows != 1) return fail(SHARD_EINVAL, "shard_step_packed: the state must have exactly one row");
  if (S < 1 || S > SHARD_MAX_TOKENS) return fail(SHARD_EINVAL, "shard_step_packed: S = %d outside [1, %d]", S, SHARD_MAX_TOKENS);
  const int32_t n_new[1] = {S};
  return step_impl(sh, st, hidden_in, token_ids, n_new, 1, position_ids, mask2d, mask_stride, nullptr, hidden_out,
                   cuda_stream, 1);
}

static int step_impl(shard_t sh, kvstate_t st, const uint16_t* hidden_in, const int32_t* token_ids,
                     const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* attention_mask,
                     int mask_stride, const int32_t* beam_idx, uint16_t* hidden_out, void* cuda_stream, int packed) {
  if (!sh || !st || st->sh != sh) return fail(SHARD_EINVAL, "shard_step: shard/state mismatch");
  if (!n_new || !position_ids || !attention_mask || !hidden_out) return fail(SHARD_EINVAL, "shard_step: null argument");
  if ((hidden_in == nullptr) == (token_ids == nullptr))
    return fail(SHARD_EINVAL, "shard_step: pass exactly one of hidden_in and token_ids");
  if (reinterpret_cast<uintptr_t>(hidden_in) % 16)
    return fail(SHARD_EINVAL, "shard_step: hidden_in must be 16-byte aligned");
  if (token_ids && sh->cfg.vocab <= 0) return fail(SHARD_EUNSUPPORTED, "shard_step: this shard has no embedding");
  if (B != st->n_rows) return fail(SHARD_EINVAL, "shard_step: B (%d) must equal the state's n_rows (%d)", B, st->n_rows);
  if (mask_stride < 1) return fail(SHARD_EINVAL, "shard_step: mask_stride must be >= 1");
  int M = 0, maxn = 0;
  for (int b = 0; b < B; ++b) {
    if (n_new[b] < 1 || n_new[b] > SHARD_MAX_TOKENS)
      return fail(SHARD_EINVAL, "shard_step: n_new[%d] = %d outside [1, %d]", b, n_new[b], SHARD_MAX_TOKENS);
    M += n_new[b];
    maxn = std::max(maxn, n_new[b]);
  }
  if (M > SHARD_MAX_TOKENS) return fail(SHARD_EINVAL, "shard_step: %d new tokens > %d", M, SHARD_MAX_TOKENS);
  if (st->poisoned) return fail(SHARD_EINVAL, "shard_step: the KV state was left inconsistent by a rejected step; reset it");
  int rc = check_pending_status(sh);
  if (rc) return rc;
  for (int b = 0; b < B; ++b) {
    if (st->cursor[b] + n_new[b] > st->cap)
      return fail(SHARD_ECAPACITY, "shard_step: row %d would hold %d entries > capacity %d", b, st->cursor[b] + n_new[b],
                  st->cap);
    if (!st->shared && !beam_idx) {
      if (st->len_host[b] + n_new[b] > mask_stride)
        return fail(SHARD_EINVAL, "shard_step: mask_stride %d < row %d length after the step %d", mask_stride, b,
                    st->len_host[b] + n_new[b]);
    }
  }
  CUDA_TRY(cudaSetDevice(sh->device));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);

  PrologueArgs pa{};
  pa.B = B;
  pa.M = M;
  for (int b = 0; b < B; ++b) {
    pa.n_new[b] = n_new[b];
    pa.cursor[b] = st->cursor[b];
  }
  pa.beam_idx = beam_idx;
  pa.hidden_in = hidden_in;
  pa.token_ids = token_ids;
  pa.position_ids = position_ids;
  pa.mask = attention_mask;
  pa.mask_stride = mask_stride;
  pa.packed = packed;
  pa.hidden_out = hidden_out;
  pa.bt_src = st->bt[st->bt_cur];
  pa.bt_dst = st->bt[beam_idx ? st->bt_cur ^ 1 : st->bt_cur];
  pa.lens = st->lens;
  pa.cap = st->cap;
  pa.max_position = sh->cfg.max_position;
  pa.vocab = sh->cfg.vocab;
  pa.H = sh->H;
  pa.embedding = sh->embedding;
  pa.status = sh->status;
  StepKernelArgs ka{};
  ka.pro = pa;
  ka.ops = sh->ops_dev;
  ka.L = sh->L;
  ka.H = sh->H;
  ka.Hq = sh->Hq;
  ka.Hkv = sh->Hkv;
  ka.d = sh->d;
  ka.F = sh->F;
  ka.Kp_H = sh->Kp_H;
  ka.Kp_dq = sh->Kp_dq;
  ka.Kp_F = sh->Kp_F;
  ka.eps = static_cast<float>(sh->cfg.rms_eps);
  ka.norms = sh->norms;
  ka.rope = sh->rope;
  ka.X = sh->X;
  ka.acc_qkv = sh->acc_qkv;
  ka.acc_gu = sh->acc_gu;
  ka.cnt_kv = sh->cnt_kv;
  ka.cnt_gu = sh->cnt_gu;
  ka.act_h = sh->act_h;
  ka.act_attn = sh->act_attn;
  ka.act_f = sh->act_f;
  ka.mask = attention_mask;
  ka.mask_stride = mask_stride;
  ka.packed = packed;
  ka.kpool = st->k;
  ka.vpool = st->v;
  ka.layer_stride = st->layer_stride;
  ka.cap = st->cap;
  ka.n_chunks = st->n_chunks;
  ka.attn_part = st->attn_part;
  ka.attn_cnt = sh->attn_cnt;
  ka.status = sh->status;
  ka.debug_skip_arrival = sh->debug_skip_arrival;
  ka.wait_limit = sh->wait_limit;
  ka.gu_part = step_gu_part_fits(sh->cfg.group, sh->L) ? 1 : 0;
  ka.barrier = sh->barrier;
  ka.barrier_base = sh->barrier_base;
  ka.phase_clock = sh->phase_clock;
  ka.status_out = sh->status_host_dev;
  ka.exit_count = sh->exit_count;
  const int grid = sh->num_sms;
  CUDA_TRY(launch_step(ka, M <= 8 ? 1 : 2, sh->cfg.group, grid, s));
  sh->barrier_base += (unsigned long long)sh->n_barriers * grid;

  for (int b = 0; b < B; ++b) st->cursor[b] += n_new[b];
  if (beam_idx) {
    st->bt_cur ^= 1;
    st->shared = true;
    int mx = 0;
    for (int b = 0; b < B; ++b) mx = std::max(mx, st->len_host[b]);
    for (int b = 0; b < B; ++b) st->len_host[b] = mx + n_new[b];  // upper bound
  } else {
    for (int b = 0; b < B; ++b) st->len_host[b] += n_new[b];
  }
  return SHARD_OK;
}

// Prefill chunk: tokens per pass through the layers (buffers scale with it).
constexpr int kPrefillChunk = 256;

int shard_prefill(shard_t sh, kvstate_t st, int row, const uint16_t* hidden_in, const int32_t* token_ids, int S,
                  const int32_t* position_ids, const uint8_t* attention_mask, int mask_len, uint16_t* hidden_out,
                  void* cuda_stream) {
  if (!sh || !st || st->sh != sh) return fail(SHARD_EINVAL, "shard_prefill: shard/state mismatch");
  if (!position_ids || !attention_mask || !hidden_out) return fail(SHARD_EINVAL, "shard_prefill: null argument");
  if ((hidden_in == nullptr) == (token_ids == nullptr))
    return fail(SHARD_EINVAL, "shard_prefill: pass exactly one of hidden_in and token_ids");
  if (token_ids && sh->cfg.vocab <= 0) return fail(SHARD_EUNSUPPORTED, "shard_prefill: this shard has no embedding");
  if (row < 0 || row >= st->n_rows || S < 1) return fail(SHARD_EINVAL, "shard_prefill: row or S out of range");
  if (st->poisoned) return fail(SHARD_EINVAL, "shard_prefill: the KV state was left inconsistent; reset it");
  if (st->shared) return fail(SHARD_EUNSUPPORTED, "shard_prefill: rows share entries after a beam gather; reset first");
  int rc = check_pending_status(sh);
  if (rc) return rc;
  const int P = st->len_host[row];
  if (st->cursor[row] != P) return fail(SHARD_EINVAL, "shard_prefill: row %d is not contiguous", row);
  if ((long long)P + S > st->cap)
    return fail(SHARD_ECAPACITY, "shard_prefill: %d + %d entries > capacity %d", P, S, st->cap);
  if (mask_len < P + S) return fail(SHARD_EINVAL, "shard_prefill: mask_len %d < %d", mask_len, P + S);
  CUDA_TRY(cudaSetDevice(sh->device));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  const int C = kPrefillChunk;
  const int y_rows = std::max(std::max(sh->dq + 2 * sh->dkv, 2 * sh->F), sh->H);
  if (!sh->pf_x) {
    // all or none: a call that fails here leaves no partial set behind for
    // the next call to mistake for a complete one
    float *x = nullptr, *y = nullptr, *q = nullptr;
    uint16_t *act = nullptr, *attn = nullptr, *hh = nullptr;
    cudaError_t e = cudaMalloc(&x, sizeof(float) * C * sh->H);
    if (e == cudaSuccess) e = cudaMalloc(&act, sizeof(uint16_t) * C * sh->Kp_H);
    if (e == cudaSuccess) e = cudaMalloc(&attn, sizeof(uint16_t) * C * sh->Kp_dq);
    if (e == cudaSuccess) e = cudaMalloc(&hh, sizeof(uint16_t) * C * sh->Kp_F);
    if (e == cudaSuccess) e = cudaMalloc(&y, sizeof(float) * C * y_rows);
    if (e == cudaSuccess) e = cudaMalloc(&q, sizeof(float) * C * sh->dq);
    if (e == cudaSuccess) e = cudaMemset(act, 0, sizeof(uint16_t) * C * sh->Kp_H);
    if (e == cudaSuccess) e = cudaMemset(attn, 0, sizeof(uint16_t) * C * sh->Kp_dq);
    if (e == cudaSuccess) e = cudaMemset(hh, 0, sizeof(uint16_t) * C * sh->Kp_F);
    if (e != cudaSuccess) {
      cudaFree(x);
      cudaFree(act);
      cudaFree(attn);
      cudaFree(hh);
      cudaFree(y);
      cudaFree(q);
      return fail(e == cudaErrorMemoryAllocation ? SHARD_ENOMEM : SHARD_ECUDA, "shard_prefill: work buffers: %s",
                  cudaGetErrorString(e));
    }
    sh->pf_x = x;
    sh->pf_act = act;
    sh->pf_attn = attn;
    sh->pf_h = hh;
    sh->pf_y = y;
    sh->pf_q = q;
  }
  CUDA_TRY(launch_prefill_check(token_ids, sh->cfg.vocab, position_ids, sh->cfg.max_position, attention_mask, P, S,
                                sh->status, s));
  const int* bt_row = st->bt[st->bt_cur] + (size_t)row * st->cap;
  const float eps = static_cast<float>(sh->cfg.rms_eps);
  for (int t0 = 0; t0 < S; t0 += C) {
    const int c = std::min(C, S - t0);
    CUDA_TRY(launch_prefill_embed(hidden_in ? hidden_in + (size_t)t0 * sh->H : nullptr,
                                  token_ids ? token_ids + t0 : nullptr, sh->embedding, sh->H, c, sh->cfg.vocab,
                                  sh->pf_x, s));
    for (int l = 0; l < sh->L; ++l) {
      const uint16_t* nrm = sh->norms + (size_t)l * 2 * sh->H;
      auto gemm = [&](int k, const uint16_t* act, int act_ld) -> cudaError_t {
        const PackedOp& p = sh->ops[(size_t)l * N_OPS + k];
        GemmArgs g{};
        g.units = p.units;
        g.n_rb = p.n_rb;
        g.upr = p.upr;
        g.act = act;
        g.act_ld = act_ld;
        g.S = c;
        g.y = sh->pf_y;
        g.y_ld = k == OP_QKV ? sh->dq + 2 * sh->dkv : k == OP_GU ? 2 * sh->F : sh->H;
        g.dims = p.dims;
        g.status = sh->status;
        return launch_gemm_tc(g, sh->cfg.group, s);
      };
      CUDA_TRY(launch_prefill_norm(sh->pf_x, sh->H, nrm, eps, sh->pf_act, sh->Kp_H, c, s));
      CUDA_TRY(gemm(OP_QKV, sh->pf_act, sh->Kp_H));
      PrefillLayerArgs pa{};
      pa.y = sh->pf_y;
      pa.y_ld = sh->dq + 2 * sh->dkv;
      pa.S = c;
      pa.Hq = sh->Hq;
      pa.Hkv = sh->Hkv;
      pa.d = sh->d;
      pa.pos = position_ids + t0;
      pa.max_position = sh->cfg.max_position;
      pa.rope = sh->rope;
      pa.q = sh->pf_q;
      pa.kpool = st->k + (size_t)l * st->layer_stride;
      pa.vpool = st->v + (size_t)l * st->layer_stride;
      pa.row = row;
      pa.cap = st->cap;
      pa.slot0 = P + t0;
      pa.bt_row = bt_row;
      pa.mask = attention_mask;
      pa.P = P + t0;
      pa.attn = sh->pf_attn;
      pa.attn_ld = sh->Kp_dq;
      CUDA_TRY(launch_prefill_rope_append(pa, s));
      CUDA_TRY(launch_prefill_attention(pa, s));
      CUDA_TRY(gemm(OP_O, sh->pf_attn, sh->Kp_dq));
      CUDA_TRY(launch_prefill_residual(sh->pf_x, sh->pf_y, sh->H, c, sh->H, nullptr, s));
      CUDA_TRY(launch_prefill_norm(sh->pf_x, sh->H, nrm + sh->H, eps, sh->pf_act, sh->Kp_H, c, s));
      CUDA_TRY(gemm(OP_GU, sh->pf_act, sh->Kp_H));
      CUDA_TRY(launch_prefill_swiglu(sh->pf_y, 2 * sh->F, c, sh->F, sh->pf_h, sh->Kp_F, s));
      CUDA_TRY(gemm(OP_DOWN, sh->pf_h, sh->Kp_F));
      CUDA_TRY(launch_prefill_residual(sh->pf_x, sh->pf_y, sh->H, c, sh->H,
                                       l + 1 == sh->L ? hidden_out + (size_t)t0 * sh->H : nullptr, s));
    }
  }
  CUDA_TRY(launch_set_int(st->lens + row, P + S, s));
  st->cursor[row] += S;
  st->len_host[row] += S;
  return SHARD_OK;
}

int shard_step_host(shard_t sh, kvstate_t st, const uint16_t* hidden_in, const int32_t* token_ids,
                    const int32_t* n_new, int B, const int32_t* position_ids, const uint8_t* attention_mask,
                    int mask_stride, const int32_t* beam_idx, uint16_t* hidden_out, void* cuda_stream) {
  if (!sh || !st || !n_new || !position_ids || !attention_mask || !hidden_out)
    return fail(SHARD_EINVAL, "shard_step_host: null argument");
  if (B < 1 || B > SHARD_MAX_REQUESTS || mask_stride < 1) return fail(SHARD_EINVAL, "shard_step_host: bad B or mask_stride");
  int M = 0;
  for (int b = 0; b < B; ++b) {
    if (n_new[b] < 1 || n_new[b] > SHARD_MAX_TOKENS)
      return fail(SHARD_EINVAL, "shard_step_host: n_new[%d] = %d outside [1, %d]", b, n_new[b], SHARD_MAX_TOKENS);
    M += n_new[b];
  }
  if (M > SHARD_MAX_TOKENS) return fail(SHARD_EINVAL, "shard_step_host: %d new tokens > %d", M, SHARD_MAX_TOKENS);
  CUDA_TRY(cudaSetDevice(sh->device));
  const size_t b_hid = hidden_in ? sizeof(uint16_t) * M * sh->H : 0;
  const size_t b_tok = token_ids ? sizeof(int32_t) * M : 0;
  const size_t b_pos = sizeof(int32_t) * M;
  const size_t b_mask = (size_t)B * mask_stride;
  const size_t b_beam = beam_idx ? sizeof(int32_t) * B : 0;
  const size_t b_out = sizeof(uint16_t) * M * sh->H;
  auto al = [](size_t v) { return (v + 255) / 256 * 256; };
  const size_t in_bytes = al(b_hid) + al(b_tok) + al(b_pos) + al(b_mask) + al(b_beam);
  const size_t need = in_bytes + al(b_out);
  if (sh->pin_bytes < need) {
    if (sh->pin) cudaFreeHost(sh->pin);
    sh->pin = nullptr;
    sh->pin_bytes = 0;  // a failed allocation leaves no stale size behind
    CUDA_TRY(cudaHostAlloc(&sh->pin, need, cudaHostAllocDefault));
    sh->pin_bytes = need;
  }
  if (sh->dstage_bytes < need) {
    cudaFree(sh->dstage);
    sh->dstage = nullptr;
    sh->dstage_bytes = 0;
    CUDA_TRY(cudaMalloc(&sh->dstage, need));
    sh->dstage_bytes = need;
  }
  uint8_t* hp = static_cast<uint8_t*>(sh->pin);
  uint8_t* dp = static_cast<uint8_t*>(sh->dstage);
  size_t off = 0;
  auto stage = [&](const void* src, size_t bytes) -> uint8_t* {
    if (!src || !bytes) return nullptr;
    memcpy(hp + off, src, bytes);
    uint8_t* d = dp + off;
    off += al(bytes);
    return d;
  };
  const uint16_t* d_hid = reinterpret_cast<const uint16_t*>(stage(hidden_in, b_hid));
  const int32_t* d_tok = reinterpret_cast<const int32_t*>(stage(token_ids, b_tok));
  const int32_t* d_pos = reinterpret_cast<const int32_t*>(stage(position_ids, b_pos));
  const uint8_t* d_mask = stage(attention_mask, b_mask);
  const int32_t* d_beam = reinterpret_cast<const int32_t*>(stage(beam_idx, b_beam));
  uint16_t* d_out = reinterpret_cast<uint16_t*>(dp + in_bytes);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  CUDA_TRY(cudaMemcpyAsync(dp, hp, off, cudaMemcpyHostToDevice, s));
  int rc = shard_step(sh, st, d_hid, d_tok, n_new, B, d_pos, d_mask, mask_stride, d_beam, d_out, cuda_stream);
  if (rc) {
    cudaStreamSynchronize(s);
    return rc;
  }
  CUDA_TRY(cudaMemcpyAsync(hp + in_bytes, d_out, b_out, cudaMemcpyDeviceToHost, s));
  CUDA_TRY(cudaStreamSynchronize(s));
  memcpy(hidden_out, hp + in_bytes, b_out);
  return SHARD_OK;
}

int shard_sync_status(shard_t sh, void* cuda_stream) {
  if (!sh) return fail(SHARD_EINVAL, "null shard");
  CUDA_TRY(cudaSetDevice(sh->device));
  CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(cuda_stream)));
  int bits = 0;
  CUDA_TRY(cudaMemcpy(&bits, sh->status, sizeof(int), cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemset(sh->status, 0, sizeof(int)));
  *reinterpret_cast<volatile int*>(sh->status_host) = 0;
  if (bits & ST_WAIT_TIMEOUT) CUDA_TRY(reset_work_buffers(sh));
  if (bits) {
    for (auto* st : sh->states) st->poisoned = true;
    return fail(SHARD_EINVAL, "device guard: %s", status_message(bits).c_str());
  }
  return SHARD_OK;
}

// ---------------------------------------------------------------------------
// Debug / test entry points (include/shard_debug.h)
// ---------------------------------------------------------------------------

int shard_debug_op_info(shard_t sh, int layer, int op, int* rows, int* K, long long* bytes) {
  if (!sh || layer < 0 || layer >= sh->L || op < 0 || op >= N_OPS) return fail(SHARD_EINVAL, "bad op");
  const PackedOp& p = sh->ops[(size_t)layer * N_OPS + op];
  const int nat[N_OPS] = {sh->dq + 2 * sh->dkv, sh->H, 2 * sh->F, sh->H};
  if (rows) *rows = nat[op];
  if (K) *K = p.K;
  if (bytes) *bytes = (long long)p.bytes;
  return SHARD_OK;
}

int shard_debug_unpack(shard_t sh, int layer, int op, float* out, int ld) {
  if (!sh || !out || layer < 0 || layer >= sh->L || op < 0 || op >= N_OPS) return fail(SHARD_EINVAL, "bad argument");
  const PackedOp& p = sh->ops[(size_t)layer * N_OPS + op];
  if (ld < p.K) return fail(SHARD_EINVAL, "ld < K");
  CUDA_TRY(cudaSetDevice(sh->device));
  CUDA_TRY(launch_unpack(p, out, ld, nullptr));
  CUDA_TRY(cudaDeviceSynchronize());
  return SHARD_OK;
}

int shard_debug_gemv(shard_t sh, int layer, int op, const uint16_t* x, int M, float* y, int y_ld, void* cuda_stream) {
  if (!sh || !x || !y || layer < 0 || layer >= sh->L || op < 0 || op >= N_OPS) return fail(SHARD_EINVAL, "bad argument");
  if (M < 1 || M > SHARD_MAX_TOKENS) return fail(SHARD_EINVAL, "M out of range");
  const PackedOp& p = sh->ops[(size_t)layer * N_OPS + op];
  CUDA_TRY(cudaSetDevice(sh->device));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  // x [M][K] -> zero-padded [M][Kp] in the shard's activation buffer
  uint16_t* act = (op == OP_O) ? sh->act_attn : (op == OP_DOWN) ? sh->act_f : sh->act_h;
  const int ld = (op == OP_O) ? sh->Kp_dq : (op == OP_DOWN) ? sh->Kp_F : sh->Kp_H;
  CUDA_TRY(cudaMemsetAsync(act, 0, sizeof(uint16_t) * ld * M, s));
  CUDA_TRY(cudaMemcpy2DAsync(act, sizeof(uint16_t) * ld, x, sizeof(uint16_t) * p.K, sizeof(uint16_t) * p.K, M,
                             cudaMemcpyDeviceToDevice, s));
  GemvArgs g{};
  g.units = p.units;
  g.n_rb = p.n_rb;
  g.upr = p.upr;
  g.act = act;
  g.act_ld = ld;
  g.M = M;
  g.status = sh->status;
  g.ep.kind = EPI_STORE;
  g.ep.dims = p.dims;
  g.ep.acc = sh->acc_store;
  g.ep.acc_ld = p.n_rb * kRowsPerBlock;
  g.ep.cnt = sh->cnt_store;
  g.ep.y = y;
  g.ep.y_ld = y_ld;
  const int nt = nt_for(M);
  CUDA_TRY(launch_gemv(g, nt, sh->cfg.group, std::min<long long>(sh->grid[nt], (long long)p.n_rb * p.upr), s, false));
  return SHARD_OK;
}

int shard_debug_gemm(shard_t sh, int layer, int op, const uint16_t* x, int x_ld, int S, float* y, int y_ld,
                     void* cuda_stream) {
  if (!sh || !x || !y || layer < 0 || layer >= sh->L || op < 0 || op >= N_OPS || S < 1)
    return fail(SHARD_EINVAL, "shard_debug_gemm: bad argument");
  const PackedOp& p = sh->ops[(size_t)layer * N_OPS + op];
  const int nat[N_OPS] = {sh->dq + 2 * sh->dkv, sh->H, 2 * sh->F, sh->H};
  if (y_ld < nat[op]) return fail(SHARD_EINVAL, "shard_debug_gemm: y_ld %d < rows %d", y_ld, nat[op]);
  if (x_ld < p.Kp || x_ld % kUnitK || reinterpret_cast<uintptr_t>(x) % 16)
    return fail(SHARD_EINVAL, "shard_debug_gemm: x_ld %d must be a multiple of 128 and >= %d; x 16-byte aligned", x_ld,
                p.Kp);
  CUDA_TRY(cudaSetDevice(sh->device));
  GemmArgs g{};
  g.units = p.units;
  g.n_rb = p.n_rb;
  g.upr = p.upr;
  g.act = x;
  g.act_ld = x_ld;
  g.S = S;
  g.y = y;
  g.y_ld = y_ld;
  g.dims = p.dims;
  g.status = sh->status;
  CUDA_TRY(launch_gemm_tc(g, sh->cfg.group, static_cast<cudaStream_t>(cuda_stream)));
  return SHARD_OK;
}

int shard_debug_set_wait(shard_t sh, unsigned limit, int skip_arrival) {
  if (!sh || limit < 1) return fail(SHARD_EINVAL, "shard_debug_set_wait: bad argument");
  sh->wait_limit = limit;
  sh->debug_skip_arrival = skip_arrival;
  return SHARD_OK;
}

int shard_debug_phase_times(shard_t sh, double* us, int n) {
  if (!sh || !us || n < 1) return fail(SHARD_EINVAL, "bad argument");
  CUDA_TRY(cudaSetDevice(sh->device));
  CUDA_TRY(cudaDeviceSynchronize());
  std::vector<unsigned long long> t(sh->n_barriers + 1);
  CUDA_TRY(cudaMemcpy(t.data(), sh->phase_clock, sizeof(unsigned long long) * t.size(), cudaMemcpyDeviceToHost));
  const int k = std::min(n, sh->n_barriers);
  for (int i = 0; i < k; ++i) us[i] = (double)(t[i + 1] - t[i]) * 1e-3;
  return k;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Support for shard_gemv_noalloc (noalloc.cu)
// ---------------------------------------------------------------------------
namespace shard {

struct NoAllocView {
  const PackedOp* op;
  int group, grid_nt1, grid_nt2, device, rows;
  int* status;  // the shard's device status word (shard_sync_status reports it)
};

int shard_noalloc_fail(int code, const char* msg) { return fail(code, "%s", msg); }
int shard_fail_msg(int code, const char* msg) { return fail(code, "%s", msg); }

int shard_noalloc_view(shard_t sh, int layer, int op, NoAllocView* v) {
  if (!sh || !v) return fail(SHARD_EINVAL, "shard_gemv_noalloc: null shard");
  if (layer < 0 || layer >= sh->L || op < 0 || op >= N_OPS)
    return fail(SHARD_EINVAL, "shard_gemv_noalloc: layer %d / op %d out of range", layer, op);
  v->op = &sh->ops[(size_t)layer * N_OPS + op];
  v->group = sh->cfg.group;
  v->grid_nt1 = sh->grid[1];
  v->grid_nt2 = sh->grid[2];
  v->device = sh->device;
  const int nat[N_OPS] = {sh->dq + 2 * sh->dkv, sh->H, 2 * sh->F, sh->H};
  v->rows = nat[op];
  v->status = sh->status;
  return SHARD_OK;
}

}  // namespace shard

