// The final stage's LM head with the top-1 epilogue (include/head.h,
// Section 6.7): per hidden row, the final RMSNorm, the INT4 lm_head
// projection to fp32 logits and a top-1 reduction to (greedy token, its
// softmax probability).  Three kernels on the caller's stream:
//   head_norm_kernel  one CTA per row: fp16 hidden -> fp16 normalised row in
//                     the zero-padded activation buffer;
//   gemv_kernel       the shard's W4A16 projection (gemv_core.cuh) with the
//                     plain store epilogue, launched with programmatic
//                     dependent launch so its weight ring fills while the
//                     norm finishes;
//   head_top1_kernel  (chunk, row) CTAs: each reduces a chunk of the row's
//                     logits to (max, lowest argmax, sum of exp relative to
//                     the max); the CTA that finishes a row last combines the
//                     chunks in chunk order (a fixed order: deterministic).
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <vector>

#include "../../include/head.h"
#include "common.cuh"

namespace shard {
// Sets the calling thread's last error (shard_api.cu) and returns code.
int shard_fail_msg(int code, const char* msg);
}  // namespace shard

using namespace shard;

namespace {

constexpr int kNormThreads = 512;
constexpr int kNormVec = 4;          // 8-element pieces per thread kept in registers (H <= 16384)
constexpr int kTopThreads = 256;
constexpr int kTopChunkMin = 512;    // logits per top-1 CTA, at least ...
constexpr int kTopChunkMax = 1024;   // ... and at most (four per thread, loaded at once)

int fail(int code, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  return shard_fail_msg(code, buf);
}

#define HEAD_CUDA_TRY(expr)                                                                         \
  do {                                                                                              \
    cudaError_t _e = (expr);                                                                        \
    if (_e != cudaSuccess)                                                                          \
      return fail(_e == cudaErrorMemoryAllocation ? SHARD_ENOMEM : SHARD_ECUDA, "%s: %s (%s:%d)", #expr, \
                  cudaGetErrorString(_e), __FILE__, __LINE__);                                      \
  } while (0)

__device__ __forceinline__ float2 h2f2(uint32_t u) {
  return make_float2(h2f(static_cast<uint16_t>(u & 0xFFFFu)), h2f(static_cast<uint16_t>(u >> 16)));
}

__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    float t = lane < nw ? red[lane] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) red[0] = t;
  }
  __syncthreads();
  const float r = red[0];
  __syncthreads();
  return r;
}

// x = hidden[m] / sqrt(mean(hidden[m]^2) + eps) * w, rounded to fp16.  One
// CTA per row; when H is a multiple of 8 and fits, every thread loads its
// 8-element pieces once (all loads in flight) and keeps them in registers.
__global__ void __launch_bounds__(kNormThreads) head_norm_kernel(const uint16_t* __restrict__ hidden, int H,
                                                                 const uint16_t* __restrict__ w, float eps,
                                                                 uint16_t* __restrict__ act, int act_ld) {
  __shared__ float red[kNormThreads / 32];
  pdl_launch_dependents();  // the projection may start streaming its weights
  const int m = blockIdx.x, tid = threadIdx.x;
  const uint16_t* h = hidden + (size_t)m * H;
  uint16_t* out = act + (size_t)m * act_ld;
  if (H % 8 == 0 && H <= kNormThreads * kNormVec * 8) {
    const int nv = H / 8;
    uint4 v[kNormVec], wv[kNormVec];
#pragma unroll
    for (int j = 0; j < kNormVec; ++j) {
      const int i = tid + j * kNormThreads;
      if (i < nv) {
        v[j] = __ldcg(reinterpret_cast<const uint4*>(h) + i);
        wv[j] = __ldg(reinterpret_cast<const uint4*>(w) + i);
      }
    }
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < kNormVec; ++j) {
      if (tid + j * kNormThreads < nv) {
        const uint32_t u[4] = {v[j].x, v[j].y, v[j].z, v[j].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = h2f2(u[q]);
          ss += f.x * f.x + f.y * f.y;
        }
      }
    }
    const float r = rsqrtf(block_sum(ss, red) / H + eps);
#pragma unroll
    for (int j = 0; j < kNormVec; ++j) {
      const int i = tid + j * kNormThreads;
      if (i < nv) {
        const uint32_t u[4] = {v[j].x, v[j].y, v[j].z, v[j].w};
        const uint32_t g[4] = {wv[j].x, wv[j].y, wv[j].z, wv[j].w};
        uint32_t o[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = h2f2(u[q]), gw = h2f2(g[q]);
          o[q] = (uint32_t)f2h(f.x * r * gw.x) | ((uint32_t)f2h(f.y * r * gw.y) << 16);
        }
        reinterpret_cast<uint4*>(out)[i] = make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
    return;
  }
  float ss = 0.f;
  for (int i = tid; i < H; i += blockDim.x) {
    const float x = h2f(h[i]);
    ss += x * x;
  }
  const float r = rsqrtf(block_sum(ss, red) / H + eps);
  for (int i = tid; i < H; i += blockDim.x) out[i] = f2h(h2f(h[i]) * r * h2f(w[i]));
}

struct Top1Part {
  float max, sum;  // the largest logit; sum of exp(logit - max)
  int idx, pad;    // the lowest id holding max
};

// Folds (bm, bs, bi) into (am, as, ai), a first: the larger maximum wins,
// equal maxima keep the lower id, the sums are rescaled to the new maximum.
// An empty side has max -inf and sum 0.
__device__ __forceinline__ void top1_combine(float& am, float& as, int& ai, float bm, float bs, int bi) {
  if (bm == -INFINITY) return;
  if (am == -INFINITY) {
    am = bm;
    as = bs;
    ai = bi;
    return;
  }
  const float nm = fmaxf(am, bm);
  as = as * expf(am - nm) + bs * expf(bm - nm);
  ai = am > bm ? ai : (bm > am ? bi : min(ai, bi));
  am = nm;
}

// Butterfly over the 32 lanes; both partners fold the lower lane's part
// first, so every lane ends with the same bits.
__device__ __forceinline__ void top1_warp(float& m, float& s, int& i) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, i, o);
    if ((lane & o) == 0) {
      top1_combine(m, s, i, m2, s2, i2);
    } else {
      float am = m2, as = s2;
      int ai = i2;
      top1_combine(am, as, ai, m, s, i);
      m = am;
      s = as;
      i = ai;
    }
  }
}

// (chunk, row) CTAs: one pass over the chunk's logits with an online
// (max, sum of exp) per thread, a fixed-order reduction over the CTA, and
// the row's last CTA folds the chunks.
__global__ void __launch_bounds__(kTopThreads) head_top1_kernel(const float* __restrict__ logits, int ld, int V,
                                                                int chunk, Top1Part* __restrict__ parts,
                                                                int* __restrict__ done, const int* status,
                                                                int32_t* __restrict__ token,
                                                                float* __restrict__ p_max) {
  __shared__ float s_m[kTopThreads / 32], s_s[kTopThreads / 32];
  __shared__ int s_i[kTopThreads / 32];
  __shared__ int s_last;
  const int c = blockIdx.x, m = blockIdx.y, nc = gridDim.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float* l = logits + (size_t)m * ld;
  const int b = c * chunk, e = min(V, b + chunk);
  float mx = -INFINITY, sm = 0.f;
  int ix = 0x7fffffff;
  constexpr int kPer = kTopChunkMax / kTopThreads;
  float x[kPer];
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    const int v = b + threadIdx.x + j * kTopThreads;
    x[j] = v < e ? __ldcg(l + v) : -INFINITY;
  }
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    const int v = b + threadIdx.x + j * kTopThreads;
    if (v < e) top1_combine(mx, sm, ix, x[j], 1.f, v);  // ids rise along a thread's walk
  }
  top1_warp(mx, sm, ix);
  if (lane == 0) {
    s_m[warp] = mx;
    s_s[warp] = sm;
    s_i[warp] = ix;
  }
  __syncthreads();
  if (warp == 0) {
    mx = lane < kTopThreads / 32 ? s_m[lane] : -INFINITY;
    sm = lane < kTopThreads / 32 ? s_s[lane] : 0.f;
    ix = lane < kTopThreads / 32 ? s_i[lane] : 0x7fffffff;
    top1_warp(mx, sm, ix);
    if (lane == 0) {
      parts[(size_t)m * nc + c] = Top1Part{mx, sm, ix, 0};
      __threadfence();
      s_last = atomicAdd(done + m, 1) == nc - 1;
    }
  }
  __syncthreads();
  if (!s_last || warp != 0) return;
  // the row's last CTA: lane L folds chunks L, L + 32, ... in order, then the
  // butterfly -- a fixed order, whatever the arrival order of the CTAs
  __threadfence();
  float gm = -INFINITY, gs = 0.f;
  int gi = 0x7fffffff;
  for (int k = lane; k < nc; k += 32)
    top1_combine(gm, gs, gi, __ldcg(&parts[(size_t)m * nc + k].max), __ldcg(&parts[(size_t)m * nc + k].sum),
                 __ldcg(&parts[(size_t)m * nc + k].idx));
  top1_warp(gm, gs, gi);
  if (lane == 0) {
    // a projection wait that gave up (never expected) marks the row failed
    const bool ok = __ldcg(status) == 0;
    token[m] = ok ? gi : -1;
    if (p_max) p_max[m] = ok ? 1.f / gs : __int_as_float(0x7fc00000);
    done[m] = 0;  // ready for the next call
  }
}

}  // namespace

struct head_s {
  int device = 0;
  head_config cfg{};
  int num_sms = 0;
  PackedOp op;
  uint8_t* units = nullptr;
  uint16_t* norm = nullptr;
  uint16_t* act = nullptr;      // fp16 [16][Kp], padding columns zero
  float* logits = nullptr;      // fp32 [16][ld]
  int ld = 0;
  long long* acc = nullptr;     // projection sums [16][n_rb * 64], fixed point, zero between calls
  int* cnt = nullptr;           // projection units finished per row-block, zero between calls
  int* status = nullptr;
  Top1Part* parts = nullptr;    // [16][max chunks]
  int* done = nullptr;          // [16] chunk arrivals per row (self-resetting)
  int max_chunks = 0;
  int grid[3] = {0, 0, 0};
  uint16_t* hidden_dev = nullptr;  // head_top1_host staging
  int32_t* token_dev = nullptr;
  float* p_dev = nullptr;
};

namespace {

void destroy(head_s* h) {
  if (!h) return;
  cudaSetDevice(h->device);
  cudaFree(h->units);
  cudaFree(h->norm);
  cudaFree(h->act);
  cudaFree(h->logits);
  cudaFree(h->acc);
  cudaFree(h->cnt);
  cudaFree(h->status);
  cudaFree(h->parts);
  cudaFree(h->done);
  cudaFree(h->hidden_dev);
  cudaFree(h->token_dev);
  cudaFree(h->p_dev);
  delete h;
}

int chunk_of(const head_s* h, int M, int* n_chunks) {
  // about one CTA per SM over the M rows, kTopChunkMin..kTopChunkMax logits each
  const int V = h->cfg.vocab;
  int nc = std::max(1, h->num_sms / M);
  nc = std::min(nc, std::max(1, (V + kTopChunkMin - 1) / kTopChunkMin));
  nc = std::max(nc, (V + kTopChunkMax - 1) / kTopChunkMax);
  const int chunk = (V + nc - 1) / nc;
  *n_chunks = (V + chunk - 1) / chunk;
  return chunk;
}

// norm -> projection -> top-1 (logits only, when token == nullptr).  No
// status copy per call: a copy-engine transfer between the calls' kernels
// measured ~9 us of stream time per call; the top-1 kernel reports a failed
// projection in the tokens instead.
int run(head_s* h, const uint16_t* hidden, int M, int32_t* token, float* p_max, float* logits, int ld,
        cudaStream_t s) {
  const head_config& c = h->cfg;
  head_norm_kernel<<<M, kNormThreads, 0, s>>>(hidden, c.hidden, h->norm, (float)c.rms_eps, h->act, h->op.Kp);
  HEAD_CUDA_TRY(cudaGetLastError());
  GemvArgs g{};
  g.units = h->op.units;
  g.n_rb = h->op.n_rb;
  g.upr = h->op.upr;
  g.act = h->act;
  g.act_ld = h->op.Kp;
  g.M = M;
  g.status = h->status;
  g.ep.kind = EPI_STORE;
  g.ep.dims = h->op.dims;
  g.ep.acc = h->acc;
  g.ep.acc_ld = h->op.n_rb * kRowsPerBlock;
  g.ep.cnt = h->cnt;
  g.ep.y = logits;
  g.ep.y_ld = ld;
  const int nt = M <= 8 ? 1 : 2;
  HEAD_CUDA_TRY(launch_gemv(g, nt, c.group, std::min<long long>(h->grid[nt], (long long)h->op.n_rb * h->op.upr), s,
                            true));
  if (token) {
    // a plain launch: with programmatic dependent launch this kernel measured
    // ~8 us slower per call
    int nc = 0;
    const int chunk = chunk_of(h, M, &nc);
    head_top1_kernel<<<dim3(nc, M), kTopThreads, 0, s>>>(logits, ld, c.vocab, chunk, h->parts, h->done, h->status,
                                                        token, p_max);
    HEAD_CUDA_TRY(cudaGetLastError());
  }
  return SHARD_OK;
}

}  // namespace

extern "C" {

int head_create(const head_config* cfg, const head_weights_host* w, head_t* out) {
  if (!cfg || !w || !out) return fail(SHARD_EINVAL, "head_create: null argument");
  *out = nullptr;
  const head_config c = *cfg;
  if (c.hidden < 1 || c.vocab < 1 || !(c.rms_eps >= 0.0))
    return fail(SHARD_EINVAL, "head_create: hidden %d / vocab %d / rms_eps out of range", c.hidden, c.vocab);
  if (c.group != 32 && c.group != 64 && c.group != 128)
    return fail(SHARD_EUNSUPPORTED, "head_create: group %d (supported: 32, 64, 128)", c.group);
  if (!w->lm_head.codes || !w->lm_head.scales || !w->lm_head.zeros || !w->norm)
    return fail(SHARD_EINVAL, "head_create: null weight pointer");
  head_s* h = new head_s();
  h->cfg = c;
  auto bail = [&](int rc) {
    destroy(h);
    return rc;
  };
  int rc;
  if ((rc = [&]() -> int {
         HEAD_CUDA_TRY(cudaGetDevice(&h->device));
         HEAD_CUDA_TRY(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device));
         HEAD_CUDA_TRY(gemv_setup());
         PackedOp& op = h->op;
         op.rows = c.vocab;
         op.K = c.hidden;
         op.Kp = (c.hidden + kUnitK - 1) / kUnitK * kUnitK;
         op.n_rb = (c.vocab + kRowsPerBlock - 1) / kRowsPerBlock;
         op.upr = op.Kp / kUnitK;
         op.unit_bytes = unit_bytes_for_group(c.group);
         op.group = c.group;
         op.bytes = (size_t)op.n_rb * op.upr * op.unit_bytes;
         op.dims = OpDims{OP_O, 0, 0, 0, 0, c.vocab};  // natural row order, rows [0, vocab)
         for (int nt = 1; nt <= 2; ++nt) h->grid[nt] = gemv_grid(nt, h->num_sms);
         h->grid[0] = std::max(h->grid[1], h->grid[2]);
         if (((uint64_t)op.n_rb * op.upr + 1) * ((uint64_t)h->grid[0] * gemv_warps_per_cta()) >= (1ull << 32))
           return fail(SHARD_EUNSUPPORTED, "head_create: too many weight units for this GPU's warp count");
         HEAD_CUDA_TRY(cudaMalloc(&h->units, op.bytes));
         op.units = h->units;
         // upload the packed matrix and repack it into the unit stream
         const int G = (c.hidden + c.group - 1) / c.group;
         const size_t cb = (size_t)(c.hidden + 1) / 2 * c.vocab, sb = (size_t)G * 2 * c.vocab,
                      zb = (size_t)(G + 1) / 2 * c.vocab;
         uint8_t* src = nullptr;
         int* rowmap = nullptr;
         HEAD_CUDA_TRY(cudaMalloc(&src, cb + sb + zb + 3 * 256));
         const size_t so = (cb + 255) / 256 * 256, zo = so + (sb + 255) / 256 * 256;
         cudaError_t e = cudaMemcpy(src, w->lm_head.codes, cb, cudaMemcpyHostToDevice);
         if (e == cudaSuccess) e = cudaMemcpy(src + so, w->lm_head.scales, sb, cudaMemcpyHostToDevice);
         if (e == cudaSuccess) e = cudaMemcpy(src + zo, w->lm_head.zeros, zb, cudaMemcpyHostToDevice);
         std::vector<int> rm((size_t)op.n_rb * kRowsPerBlock, -1);
         for (int r = 0; r < c.vocab; ++r) rm[r] = r;
         if (e == cudaSuccess) e = cudaMalloc(&rowmap, sizeof(int) * rm.size());
         if (e == cudaSuccess) e = cudaMemcpy(rowmap, rm.data(), sizeof(int) * rm.size(), cudaMemcpyHostToDevice);
         if (e == cudaSuccess) {
           RepackSrc rs{};
           rs.codes[0] = src;
           rs.scales[0] = reinterpret_cast<const uint16_t*>(src + so);
           rs.zeros[0] = src + zo;
           rs.rows[0] = c.vocab;
           e = launch_repack(op, rowmap, rs, nullptr);
         }
         if (e == cudaSuccess) e = cudaDeviceSynchronize();
         cudaFree(src);
         cudaFree(rowmap);
         HEAD_CUDA_TRY(e);
         HEAD_CUDA_TRY(cudaMalloc(&h->norm, sizeof(uint16_t) * c.hidden));
         HEAD_CUDA_TRY(cudaMemcpy(h->norm, w->norm, sizeof(uint16_t) * c.hidden, cudaMemcpyHostToDevice));
         HEAD_CUDA_TRY(cudaMalloc(&h->act, sizeof(uint16_t) * kMaxTokens * op.Kp));
         HEAD_CUDA_TRY(cudaMemset(h->act, 0, sizeof(uint16_t) * kMaxTokens * op.Kp));
         h->ld = (c.vocab + 3) / 4 * 4;
         HEAD_CUDA_TRY(cudaMalloc(&h->logits, sizeof(float) * kMaxTokens * h->ld));
         const size_t acc_n = (size_t)kMaxTokens * op.n_rb * kRowsPerBlock;
         HEAD_CUDA_TRY(cudaMalloc(&h->acc, sizeof(long long) * acc_n));
         HEAD_CUDA_TRY(cudaMemset(h->acc, 0, sizeof(long long) * acc_n));
         HEAD_CUDA_TRY(cudaMalloc(&h->cnt, sizeof(int) * op.n_rb));
         HEAD_CUDA_TRY(cudaMemset(h->cnt, 0, sizeof(int) * op.n_rb));
         HEAD_CUDA_TRY(cudaMalloc(&h->status, sizeof(int)));
         HEAD_CUDA_TRY(cudaMemset(h->status, 0, sizeof(int)));
         h->max_chunks = (c.vocab + kTopChunkMin - 1) / kTopChunkMin + 1;
         HEAD_CUDA_TRY(cudaMalloc(&h->parts, sizeof(Top1Part) * kMaxTokens * h->max_chunks));
         HEAD_CUDA_TRY(cudaMalloc(&h->done, sizeof(int) * kMaxTokens));
         HEAD_CUDA_TRY(cudaMemset(h->done, 0, sizeof(int) * kMaxTokens));
         HEAD_CUDA_TRY(cudaMalloc(&h->hidden_dev, sizeof(uint16_t) * kMaxTokens * c.hidden));
         HEAD_CUDA_TRY(cudaMalloc(&h->token_dev, sizeof(int32_t) * kMaxTokens));
         HEAD_CUDA_TRY(cudaMalloc(&h->p_dev, sizeof(float) * kMaxTokens));
         return SHARD_OK;
       }()) != SHARD_OK)
    return bail(rc);
  *out = h;
  return SHARD_OK;
}

int head_destroy(head_t h) {
  if (!h) return fail(SHARD_EINVAL, "head_destroy: null head");
  destroy(h);
  return SHARD_OK;
}

int head_top1(head_t h, const uint16_t* hidden, int M, int32_t* token, float* p_max, void* cuda_stream) {
  if (!h || !hidden || !token) return fail(SHARD_EINVAL, "head_top1: null argument");
  if (M < 1 || M > SHARD_MAX_TOKENS) return fail(SHARD_EINVAL, "head_top1: M = %d outside [1, %d]", M, SHARD_MAX_TOKENS);
  HEAD_CUDA_TRY(cudaSetDevice(h->device));
  return run(h, hidden, M, token, p_max, h->logits, h->ld, static_cast<cudaStream_t>(cuda_stream));
}

int head_top1_host(head_t h, const uint16_t* hidden, int M, int32_t* token, float* p_max, void* cuda_stream) {
  if (!h || !hidden || !token) return fail(SHARD_EINVAL, "head_top1_host: null argument");
  if (M < 1 || M > SHARD_MAX_TOKENS)
    return fail(SHARD_EINVAL, "head_top1_host: M = %d outside [1, %d]", M, SHARD_MAX_TOKENS);
  HEAD_CUDA_TRY(cudaSetDevice(h->device));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  HEAD_CUDA_TRY(cudaMemcpyAsync(h->hidden_dev, hidden, sizeof(uint16_t) * M * h->cfg.hidden, cudaMemcpyHostToDevice, s));
  int rc = run(h, h->hidden_dev, M, h->token_dev, p_max ? h->p_dev : nullptr, h->logits, h->ld, s);
  if (rc) return rc;
  HEAD_CUDA_TRY(cudaMemcpyAsync(token, h->token_dev, sizeof(int32_t) * M, cudaMemcpyDeviceToHost, s));
  if (p_max) HEAD_CUDA_TRY(cudaMemcpyAsync(p_max, h->p_dev, sizeof(float) * M, cudaMemcpyDeviceToHost, s));
  HEAD_CUDA_TRY(cudaStreamSynchronize(s));
  for (int m = 0; m < M; ++m)
    if (token[m] < 0) {
      // a projection that gave up leaves partial sums and row-block counts
      // behind: clear them with the status so the next call starts clean
      cudaMemsetAsync(h->status, 0, sizeof(int), s);
      cudaMemsetAsync(h->acc, 0, sizeof(long long) * kMaxTokens * h->op.n_rb * kRowsPerBlock, s);
      cudaMemsetAsync(h->cnt, 0, sizeof(int) * h->op.n_rb, s);
      cudaStreamSynchronize(s);
      return fail(SHARD_ECUDA, "head_top1_host: a device wait of the projection timed out");
    }
  return SHARD_OK;
}

int head_debug_logits(head_t h, const uint16_t* hidden, int M, float* logits, int ld, void* cuda_stream) {
  if (!h || !hidden || !logits) return fail(SHARD_EINVAL, "head_debug_logits: null argument");
  if (M < 1 || M > SHARD_MAX_TOKENS) return fail(SHARD_EINVAL, "head_debug_logits: M = %d out of range", M);
  if (ld < h->cfg.vocab) return fail(SHARD_EINVAL, "head_debug_logits: ld %d < vocab %d", ld, h->cfg.vocab);
  HEAD_CUDA_TRY(cudaSetDevice(h->device));
  return run(h, hidden, M, nullptr, nullptr, logits, ld, static_cast<cudaStream_t>(cuda_stream));
}

}  // extern "C"
