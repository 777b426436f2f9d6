// The whole decode step of a shard as one persistent, cooperative kernel.
//
// One CTA per SM: kCtaWarps consumer warps and one producer warp that streams
// the weights into the consumers' rings (gemv_core.cuh).  The step runs as a
// sequence of phases separated by grid-wide barriers ('|'):
//   prologue (every CTA: its share of the beam-table gather, the new
//   entries' slots and the residual) ~ for each layer: RMSNorm + q|k|v
//   projection -> attention (chunk partials and merges, with RoPE and the K/V
//   append) | o projection (+residual) | RMSNorm + gate|up projection
//   (+SwiGLU) | down projection (+residual) | ... ; then hidden_out.
// '~' is a split barrier: CTAs arrive after their prologue share and wait only
// before the first attention, so the first norm and q|k|v projection overlap
// the prologue.  '->' is dataflow: q|k|v contributors count finished units
// per kv head (release) and an attention item waits (acquire, bounded) only
// for its kv head's count.
//
// The residual stream and the projections' sums are 64-bit fixed point
// (kernels.h): contributors add with integer atomics and nobody waits for a
// merge; results do not depend on the order of arrival.
// Each RMSNorm is computed by every CTA at the start of the projection that
// consumes it, from the whole residual (the same bits in every CTA).
//
// Every cross-CTA wait is bounded: a wait that runs out sets a status bit and
// proceeds (the step's results are then reported invalid) instead of hanging.
#include <type_traits>

#include <algorithm>

#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kWarps = kCtaWarps;           // consumer warps
constexpr int kThreads = kWarps * 32;       // consumer threads
constexpr int kBlockThreads = kThreads + (kSelfRefill ? 0 : 32);  // + the producer warp, if any
constexpr int kChunk = kAttnChunk;  // most cache entries per attention item (kChunk / 32 per lane)
constexpr bool kNormInSmem = true;   // normalised activations in shared memory when they fit
// Polls of a busy slot before the producer gives up: a slot may legitimately
// stay busy while its consumer works through a whole attention phase, so this
// bound is fixed and far above any step's length.
constexpr uint32_t kProducerLimit = 1u << 22;

// The attention area: one item's tiles at kChunk entries and head_dim 128
// (AttnSmem), rounded up to 1 KB; it also holds the normalised rows when they fit.
constexpr size_t kAttnArea =
    ((size_t)kChunk * (128 + 8) * 2 + (size_t)kChunk * 128 * 2 + 16 * 128 * 4 + 16 * kChunk * 4 + 2 * kChunk * 4 +
     (size_t)kMaxTokens * kChunk + 1023) / 1024 * 1024;

template <int GPU>
struct StepSmem {
  static constexpr int kSlots = Geom<GPU>::kStepSlots;
  static constexpr size_t kRing = (size_t)kWarps * kSlots * Geom<GPU>::kUnitBytes;
  static constexpr size_t kBars = (size_t)2 * kWarps * kSlots * sizeof(uint64_t);
  // attention item area (AttnSmem), also the normalised rows
  static constexpr size_t kQ = kAttnArea;
  static constexpr size_t kFixed = kRing + kBars + kQ;  // + the op table (4L entries)
  // gate|up partial sums of the shared-memory reduction (swiglu_cta_write)
  static constexpr size_t kPart = (size_t)kWarps * kGuCtaTokens * kRowsPerBlock * sizeof(float);
  __host__ __device__ static size_t ops_bytes(int n_layers) { return ((size_t)4 * n_layers * sizeof(OpDesc) + 15) / 16 * 16; }
  static size_t total(int n_layers) { return kFixed + ops_bytes(n_layers); }
  static size_t total_with_part(int n_layers) { return total(n_layers) + kPart; }
};

// Barrier among the consumer warps of a CTA (the producer warp runs on its own).
__device__ __forceinline__ void cbar() { named_bar_sync(1, kThreads); }

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ float2 h2f2(uint32_t u) {
  __half2 h;
  memcpy(&h, &u, sizeof(h));
  return __half22float2(h);
}

// two floats rounded to fp16 (to nearest even), lo in the low half
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  return (uint32_t)f2h(lo) | ((uint32_t)f2h(hi) << 16);
}

__device__ __forceinline__ void red_release_add(unsigned long long* p, unsigned long long v) {
  asm volatile("red.release.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Grid-wide barrier on a monotonically increasing counter, in two halves so
// that work may sit between arriving and waiting.  `target` is this CTA's
// running count of expected arrivals.  Called by the consumer warps; the
// caller has synchronised them (cbar) before grid_arrive.
struct GridBarrier {
  unsigned long long* ctr;
  unsigned long long target;
  int* status;
  unsigned long long* clock;
  int n_arrive, n_wait;
  int skip_arrival;  // test knob: CTA 1 leaves out this arrival (-1: none)
  uint32_t limit;

  __device__ __forceinline__ void arrive() {
    if (threadIdx.x == 0) {
      if (!(blockIdx.x == 1 && n_arrive == skip_arrival)) red_release_add(ctr, 1ULL);
    }
    ++n_arrive;
  }
  __device__ __forceinline__ void wait() {
    if (threadIdx.x == 0) {
      target += gridDim.x;
      // bounded: after `limit` polls, or once any CTA has given up, stop waiting
      uint32_t it = 0;
      while (ld_acquire_u64(ctr) < target) {
        if (++it > limit) {
          atomicOr(status, ST_WAIT_TIMEOUT);
          break;
        }
        if ((it & 1023) == 0 && (*reinterpret_cast<volatile int*>(status) & ST_WAIT_TIMEOUT)) break;
        __nanosleep(16);
      }
      if (blockIdx.x == 0) clock[n_wait + 1] = globaltimer();
    }
    ++n_wait;
    cbar();
  }
  __device__ __forceinline__ void sync() {
    cbar();
    arrive();
    wait();
  }
};

__device__ __forceinline__ bool wait_count(const int* p, int target, int* status, uint32_t limit) {
  uint32_t it = 0;
  while (ld_acquire_s32(p) < target) {
    if (++it > limit) {
      atomicOr(status, ST_WAIT_TIMEOUT);
      return false;
    }
    if ((it & 1023) == 0 && (*reinterpret_cast<volatile int*>(status) & ST_WAIT_TIMEOUT)) return false;
    __nanosleep(64);
  }
  return true;
}

// ---------------------------------------------------------------------------
// Prologue, part 1 (every CTA, all threads): the step's bookkeeping from its
// arguments -- Section 4's beam_idx gather (row b continues row beam_idx[b]'s
// entries; K/V stay where they are), the new entries' slots -- and the
// device-side argument checks.  Every CTA derives the same values.
// ---------------------------------------------------------------------------
__device__ __noinline__ void prologue_params(const PrologueArgs& a, StepParams* sp, const uint16_t** rowp) {
  __shared__ int s_err;
  const int tid = threadIdx.x;
  if (tid == 0) {
    // a step rejected earlier freezes the state until the host resets it
    s_err = __ldcg(a.status) != 0 ? ST_STICKY : 0;
    int t = 0;
    for (int b = 0; b < a.B; ++b) {
      sp->req_tok0[b] = t;
      for (int i = 0; i < a.n_new[b]; ++i, ++t) {
        sp->tok_req[t] = b;
        sp->tok_idx[t] = i;
      }
    }
    sp->req_tok0[a.B] = t;
    sp->M = a.M;
    sp->B = a.B;
  }
  __syncthreads();
  if (tid < a.B) {
    int src = a.beam_idx ? __ldcg(a.beam_idx + tid) : tid;
    if (src < 0 || src >= a.B) {
      atomicOr(&s_err, ST_BEAM_IDX);
      src = tid;
    }
    sp->req_src[tid] = src;
    const int P = __ldcg(a.lens + src);
    const int L = P + a.n_new[tid];
    if (L > a.cap || a.cursor[tid] + a.n_new[tid] > a.cap) atomicOr(&s_err, ST_CAPACITY);
    if (L > a.mask_stride) atomicOr(&s_err, ST_MASK_STRIDE);
    sp->req_P[tid] = P;
    sp->req_len[tid] = L;
  }
  __syncthreads();
  if (tid < a.M) {
    const int m = tid, b = sp->tok_req[m], i = sp->tok_idx[m], j = sp->req_P[b] + i;
    // a token must see its own entry (packed: in its own mask row, Section 8.6)
    const size_t mrow = a.packed ? (size_t)m : (size_t)b;
    if (j < a.mask_stride && __ldcg(a.mask + mrow * a.mask_stride + j) == 0) atomicOr(&s_err, ST_MASK_NEW);
    const int pos = __ldcg(a.position_ids + m);
    if (pos < 0 || pos >= a.max_position) atomicOr(&s_err, ST_POSITION);
    sp->tok_pos[m] = pos;
    sp->tok_slot[m] = b * a.cap + a.cursor[b] + i;
    if (a.token_ids) {
      const int tok = __ldcg(a.token_ids + m);
      if (tok < 0 || tok >= a.vocab) atomicOr(&s_err, ST_TOKEN);
      rowp[m] = a.embedding + (size_t)(tok < 0 || tok >= a.vocab ? 0 : tok) * a.H;
    } else {
      rowp[m] = a.hidden_in + (size_t)m * a.H;
    }
  }
  __syncthreads();
  if (tid == 0) sp->abort_step = s_err;
  __syncthreads();
}

// Prologue, part 2 (consumer threads of every CTA, a share each): the beam
// table's gather and appends, and the residual stream X = the fp16 inputs in
// fixed point (exact).
__device__ __noinline__ void prologue_work(const PrologueArgs& a, const StepParams* sp, const uint16_t* const* rowp,
                                           long long* X) {
  const int tid = threadIdx.x;
  const int gt = blockIdx.x * kThreads + tid, gs = gridDim.x * kThreads;
  if (a.beam_idx) {
    for (int b = 0; b < a.B; ++b) {
      const int* src = a.bt_src + (size_t)sp->req_src[b] * a.cap;
      int* dst = a.bt_dst + (size_t)b * a.cap;
      for (int j = gt; j < sp->req_P[b]; j += gs) dst[j] = __ldcg(src + j);
    }
  }
  if (blockIdx.x == 0 && tid < a.M) {
    const int b = sp->tok_req[tid], i = sp->tok_idx[tid];
    a.bt_dst[(size_t)b * a.cap + sp->req_P[b] + i] = sp->tok_slot[tid];
  }
  const int H4 = a.H / 4;
  for (int e = gt; e < a.M * H4; e += gs) {
    const int m = e / H4, k = 4 * (e % H4);
    const uint2 v = *reinterpret_cast<const uint2*>(rowp[m] + k);
    const float2 f01 = h2f2(v.x), f23 = h2f2(v.y);
    longlong2* dst = reinterpret_cast<longlong2*>(X + (size_t)m * a.H + k);
    dst[0] = make_longlong2(to_fixed(f01.x), to_fixed(f01.y));
    dst[1] = make_longlong2(to_fixed(f23.x), to_fixed(f23.y));
  }
}

// ---------------------------------------------------------------------------
// RMSNorm, run by every CTA at the start of the projection that consumes it:
// r[m] = 1 / sqrt(mean(x[m]^2) + eps), act = fp16(x * r * w).  x is the
// residual stream (fixed point) or, before the first layer, the step's fp16
// input rows (the same values).  Two passes: the sums of squares (added in a
// fixed order, so every CTA gets the same r), then the scaled rows; the first
// row's pieces stay in registers between the passes.  H is a multiple of 4.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float4 norm_load(bool from_x, const long long* X, const uint16_t* const* rowp, int H, int m,
                                            int k) {
  if (from_x) {
    const longlong2* p = reinterpret_cast<const longlong2*>(X + (size_t)m * H + k);
    const longlong2 a = __ldcg(p), b = __ldcg(p + 1);
    return make_float4(fixed_to_f32(a.x), fixed_to_f32(a.y), fixed_to_f32(b.x), fixed_to_f32(b.y));
  } else {
    const uint2 v = *reinterpret_cast<const uint2*>(rowp[m] + k);
    const float2 f01 = h2f2(v.x), f23 = h2f2(v.y);
    return make_float4(f01.x, f01.y, f23.x, f23.y);
  }
}

// kP pieces (float4) per row and thread are held in registers (the rest of a
// longer row is streamed).  Rows go kR at a time, every piece of the kR rows
// requested at once (one memory round trip per batch; the norm weights come
// with the first).  When all M rows fit in one batch they stay in registers
// for the second pass, so X is read once.
template <int kP, int kR>
__device__ __forceinline__ void rmsnorm_rows(bool from_x, const long long* X, const uint16_t* const* rowp, int H,
                                             const uint16_t* w, float eps, uint16_t* out, int out_ld, int M) {
  __shared__ float s_part[kWarps][kMaxTokens];
  __shared__ float s_r[kMaxTokens];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H4 = H / 4;
  uint2 wv[kP];
  float4 v[kR][kP];
#pragma unroll
  for (int i = 0; i < kP; ++i) {
    const int c = tid + i * kThreads;
    wv[i] = c < H4 ? *reinterpret_cast<const uint2*>(w + 4 * c) : make_uint2(0, 0);
  }
  auto load_batch = [&](int m0) {
#pragma unroll
    for (int h = 0; h < kR; ++h)
#pragma unroll
      for (int i = 0; i < kP; ++i) {
        const int c = tid + i * kThreads;
        v[h][i] = c < H4 && m0 + h < M ? norm_load(from_x, X, rowp, H, m0 + h, 4 * c) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
  };
  for (int m0 = 0; m0 < M; m0 += kR) {
    load_batch(m0);
    float t[kR];
#pragma unroll
    for (int h = 0; h < kR; ++h) {
      t[h] = 0.f;
#pragma unroll
      for (int i = 0; i < kP; ++i)
        t[h] += v[h][i].x * v[h][i].x + v[h][i].y * v[h][i].y + v[h][i].z * v[h][i].z + v[h][i].w * v[h][i].w;
      if (m0 + h < M)
        for (int c = tid + kP * kThreads; c < H4; c += kThreads) {
          const float4 u = norm_load(from_x, X, rowp, H, m0 + h, 4 * c);
          t[h] += u.x * u.x + u.y * u.y + u.z * u.z + u.w * u.w;
        }
    }
#pragma unroll
    for (int h = 0; h < kR; ++h) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) t[h] += __shfl_xor_sync(0xffffffffu, t[h], o);
      if (lane == 0 && m0 + h < M) s_part[warp][m0 + h] = t[h];
    }
  }
  cbar();
  if (tid < M) {
    float t = 0.f;
    for (int w8 = 0; w8 < kWarps; ++w8) t += s_part[w8][tid];
    s_r[tid] = rsqrtf(t / H + eps);
  }
  cbar();
  for (int m0 = 0; m0 < M; m0 += kR) {
    if (M > kR) load_batch(m0);  // else the one batch is still in registers
#pragma unroll
    for (int h = 0; h < kR; ++h) {
      const int m = m0 + h;
      if (m >= M) break;
      const float r = s_r[m];
      auto emit = [&](int c, float4 x, uint2 wq) {
        const float2 w01 = h2f2(wq.x), w23 = h2f2(wq.y);
        uint2 o;
        o.x = pack_h2(x.x * r * w01.x, x.y * r * w01.y);
        o.y = pack_h2(x.z * r * w23.x, x.w * r * w23.y);
        *reinterpret_cast<uint2*>(out + (size_t)m * out_ld + 4 * c) = o;
      };
#pragma unroll
      for (int i = 0; i < kP; ++i) {
        const int c = tid + i * kThreads;
        if (c < H4) emit(c, v[h][i], wv[i]);
      }
      for (int c = tid + kP * kThreads; c < H4; c += kThreads)
        emit(c, norm_load(from_x, X, rowp, H, m, 4 * c), *reinterpret_cast<const uint2*>(w + 4 * c));
    }
  }
  cbar();
}

// One row from the residual stream (M = 1, H <= 24 * kThreads) through
// shared memory: the row's H fixed-point values arrive with bulk copies
// (`stage`, 16-byte aligned, H * 8 bytes; completion on `bar`, whose phase
// the caller tracks), so the read runs at copy-engine bandwidth instead of
// being bounded by each thread's loads in flight; both passes then read
// shared memory.  The values and the arithmetic are those of rmsnorm_rows.
__device__ __forceinline__ void rmsnorm_staged(const long long* X, int H, const uint16_t* w, float eps, uint16_t* out,
                                               long long* stage, uint64_t* bar, uint32_t& phase, int* status) {
  constexpr int kP = 6;
  constexpr uint32_t kPiece = 8192;  // bytes per bulk copy
  __shared__ float s_part[kWarps];
  __shared__ float s_r;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H4 = H / 4;
  if (tid == 0) {
    // X was written through the generic proxy (made visible by the grid
    // barrier); the area was last used by generic accesses of this CTA
    asm volatile("fence.proxy.async;" ::: "memory");
    const uint32_t bytes = (uint32_t)H * 8u;
    mbar_arrive_expect_tx(bar, bytes);
    for (uint32_t off = 0; off < bytes; off += kPiece)
      bulk_g2s(reinterpret_cast<uint8_t*>(stage) + off, reinterpret_cast<const uint8_t*>(X) + off,
               bytes - off < kPiece ? bytes - off : kPiece, bar);
  }
  uint2 wv[kP];
#pragma unroll
  for (int i = 0; i < kP; ++i) {
    const int c = tid + i * kThreads;
    wv[i] = c < H4 ? *reinterpret_cast<const uint2*>(w + 4 * c) : make_uint2(0, 0);
  }
  if (!mbar_wait(bar, phase) && tid == 0) atomicOr(status, ST_WAIT_TIMEOUT);
  phase ^= 1u;
  float4 v[kP];
  float t = 0.f;
#pragma unroll
  for (int i = 0; i < kP; ++i) {
    const int c = tid + i * kThreads;
    v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c < H4) {
      const longlong2 a = reinterpret_cast<const longlong2*>(stage)[2 * c];
      const longlong2 b = reinterpret_cast<const longlong2*>(stage)[2 * c + 1];
      v[i] = make_float4(fixed_to_f32(a.x), fixed_to_f32(a.y), fixed_to_f32(b.x), fixed_to_f32(b.y));
    }
    t += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  if (lane == 0) s_part[warp] = t;
  cbar();
  if (tid == 0) {
    float u = 0.f;
    for (int w8 = 0; w8 < kWarps; ++w8) u += s_part[w8];
    s_r = rsqrtf(u / H + eps);
  }
  cbar();
  const float r = s_r;
#pragma unroll
  for (int i = 0; i < kP; ++i) {
    const int c = tid + i * kThreads;
    if (c < H4) {
      const float2 w01 = h2f2(wv[i].x), w23 = h2f2(wv[i].y);
      uint2 o;
      o.x = pack_h2(v[i].x * r * w01.x, v[i].y * r * w01.y);
      o.y = pack_h2(v[i].z * r * w23.x, v[i].w * r * w23.y);
      *reinterpret_cast<uint2*>(out + 4 * c) = o;
    }
  }
  cbar();
}

// Rows of up to 3 pieces per thread (H <= 4608) go three at a time; longer
// rows two at a time with 6 pieces in registers.  from_x: the residual
// stream, else the step's fp16 input rows (before the first layer).
__device__ __forceinline__ void rmsnorm_cta(bool from_x, const long long* X, const uint16_t* const* rowp, int H,
                                            const uint16_t* w, float eps, uint16_t* out, int out_ld, int M) {
  if (H / 4 <= 3 * kThreads)
    rmsnorm_rows<3, 3>(from_x, X, rowp, H, w, eps, out, out_ld, M);
  else
    rmsnorm_rows<6, 2>(from_x, X, rowp, H, w, eps, out, out_ld, M);
}

// ---------------------------------------------------------------------------
// Attention.  Item = (request b, kv head hk, chunk c of cs entries); one CTA
// per item, items dealt round-robin.  cs is the smallest of 32, 64, 128 that
// gives no more items than CTAs (short caches: more parallel items), else 128
// (long caches: fewer rounds and merges).  Each item writes (max, sum of exp,
// unnormalised output) per query (the request's new tokens x the kv head's
// query heads).  With several items per CTA, after its items the CTA that
// took the last chunk of (b, hk) waits for the chunk count and combines the
// chunks in order, so the merges are spread over CTAs and never delay
// anyone's items; with one item per CTA at most, the CTA that finishes the
// last chunk merges at once.
// ---------------------------------------------------------------------------
// A partial is (max, sum of exp, 2 unused, unnormalised output[d]): the
// output starts 16-byte aligned.
__host__ __device__ constexpr int part_stride(int d) { return d + 4; }

struct AttnView {
  const long long* acc;     // q|k|v sums [16][acc_ld] (fixed point), GPU row order
  int acc_ld;
  const float2* rope;       // [max_position][d/2]
  uint16_t* kpool;          // layer 0; layer l at + l * layer_stride
  uint16_t* vpool;
  size_t layer_stride;
  int cap, Hq, Hkv, d, n_chunks, qmax;
  float* part;
  int* cnt;                 // finished chunks per (request, kv head)
  const int* cnt_kv;        // q|k|v units finished per kv head
  int kv_units;             // units per kv head when its q|k|v rows are complete
  const int* bt;            // beam table (entry -> physical slot) of this step
  const uint8_t* mask;
  int mask_stride;
  int packed;               // a mask row per token of request 0 instead of one per request
  int cs;                   // entries per item this step: 32, 64 or 128 (kChunk)
  int last_merges;          // at most one item per CTA: the CTA finishing the last chunk merges at once
  uint32_t limit;
  uint16_t* out;
  int out_ld;
};

__device__ __forceinline__ int n_chunks_of(int L, int cs) { return (L + cs - 1) / cs; }

// Finds the item's (b, hk, c) from a flat index; false if past the end.
__device__ __forceinline__ bool decode_item(const StepParams* sp, int Hkv, int cs, int item, int& b, int& hk, int& c) {
  for (b = 0; b < sp->B; ++b) {
    const int per = Hkv * n_chunks_of(sp->req_len[b], cs);
    if (item < per) {
      hk = item / n_chunks_of(sp->req_len[b], cs);
      c = item % n_chunks_of(sp->req_len[b], cs);
      return true;
    }
    item -= per;
  }
  return false;
}

// q (fp32, shared) . K row (fp16, shared) over KP 8-element pieces; the
// two-row form scores rows k0 and k1 with one pass over q.
__device__ __forceinline__ float dot_q_k(const float* qq, const uint16_t* k0r, int KP) {
  float s0 = 0.f;
#pragma unroll 4
  for (int t = 0; t < KP; ++t) {
    const uint4 k0 = *reinterpret_cast<const uint4*>(k0r + t * 8);
    const float4 qa = *reinterpret_cast<const float4*>(qq + t * 8);
    const float4 qb = *reinterpret_cast<const float4*>(qq + t * 8 + 4);
    float2 f = h2f2(k0.x);
    s0 = fmaf(qa.x, f.x, s0);
    s0 = fmaf(qa.y, f.y, s0);
    f = h2f2(k0.y);
    s0 = fmaf(qa.z, f.x, s0);
    s0 = fmaf(qa.w, f.y, s0);
    f = h2f2(k0.z);
    s0 = fmaf(qb.x, f.x, s0);
    s0 = fmaf(qb.y, f.y, s0);
    f = h2f2(k0.w);
    s0 = fmaf(qb.z, f.x, s0);
    s0 = fmaf(qb.w, f.y, s0);
  }
  return s0;
}
__device__ __forceinline__ float dot_q_k2(const float* qq, const uint16_t* k0r, const uint16_t* k1r, float& s1,
                                          int KP) {
  float s0 = 0.f;
  s1 = 0.f;
#pragma unroll 4
  for (int t = 0; t < KP; ++t) {
    const uint4 k0 = *reinterpret_cast<const uint4*>(k0r + t * 8);
    const uint4 k1 = *reinterpret_cast<const uint4*>(k1r + t * 8);
    const float4 qa = *reinterpret_cast<const float4*>(qq + t * 8);
    const float4 qb = *reinterpret_cast<const float4*>(qq + t * 8 + 4);
    float2 f = h2f2(k0.x), g = h2f2(k1.x);
    s0 = fmaf(qa.x, f.x, s0);
    s0 = fmaf(qa.y, f.y, s0);
    s1 = fmaf(qa.x, g.x, s1);
    s1 = fmaf(qa.y, g.y, s1);
    f = h2f2(k0.y);
    g = h2f2(k1.y);
    s0 = fmaf(qa.z, f.x, s0);
    s0 = fmaf(qa.w, f.y, s0);
    s1 = fmaf(qa.z, g.x, s1);
    s1 = fmaf(qa.w, g.y, s1);
    f = h2f2(k0.z);
    g = h2f2(k1.z);
    s0 = fmaf(qb.x, f.x, s0);
    s0 = fmaf(qb.y, f.y, s0);
    s1 = fmaf(qb.x, g.x, s1);
    s1 = fmaf(qb.y, g.y, s1);
    f = h2f2(k0.w);
    g = h2f2(k1.w);
    s0 = fmaf(qb.z, f.x, s0);
    s0 = fmaf(qb.w, f.y, s0);
    s1 = fmaf(qb.z, g.x, s1);
    s1 = fmaf(qb.w, g.y, s1);
  }
  return s0;
}

// Shared-memory layout of one attention item.
template <int DPL>
struct AttnSmem {
  static constexpr int d = 32 * DPL;
  static constexpr int kKld = d + 8;  // padded K row (halves): consecutive rows start on different banks
  static constexpr int kQg = 16;      // queries per group
  static constexpr size_t kK = (size_t)kChunk * kKld * 2;
  static constexpr size_t kV = (size_t)kChunk * d * 2;
  static constexpr size_t kQ = (size_t)kQg * d * 4;
  static constexpr size_t kP = (size_t)kQg * kChunk * 4;
  static constexpr size_t kVisT = (size_t)kMaxTokens * kChunk;  // packed mode: [token][entry] mask bytes
  static constexpr size_t kBytes = kK + kV + kQ + kP + 2 * kChunk * sizeof(int) + kVisT;
};

// Row of the q|k|v projection holding dimension i (< d/2) of q head h, or of
// k head h when `first` is the first k row; dimension i + d/2 is 8 rows
// further (kernels.h: rotary pairs share a 16-row tile).
__device__ __forceinline__ int rot_row(int first, int h, int i, int d) {
  return first + 16 * (h * (d >> 4) + (i >> 3)) + (i & 7);
}

// Queries q0 .. q0 + qn of an item into shared memory: the fixed-point q sums
// of the query's head and token, rotated by the token's position (RoPE,
// pairs (i, i + d/2)), fp32.
template <int DPL>
__device__ __forceinline__ void attn_load_queries(const AttnView& a, const StepParams* sp, int hk, int tok0, int q0,
                                                  int qn, float* qsm) {
  constexpr int d = 32 * DPL, half = d / 2;
  const int G = a.Hq / a.Hkv;
  for (int e = threadIdx.x; e < qn * half; e += kThreads) {
    const int qi = e / half, i = e % half, q = q0 + qi;
    const int m = tok0 + q / G, h = hk * G + q % G;
    const long long* row = a.acc + (size_t)m * a.acc_ld;
    const int R = rot_row(0, h, i, d);
    const float lo = fixed_to_f32(__ldcg(row + R)), hi = fixed_to_f32(__ldcg(row + R + 8));
    const float2 cs = a.rope[(size_t)sp->tok_pos[m] * half + i];
    qsm[qi * d + i] = lo * cs.x - hi * cs.y;
    qsm[qi * d + half + i] = hi * cs.x + lo * cs.y;
  }
}

// Merge of one (request, kv head, query): chunks in order, kMergeBatch at a
// time with all their loads in flight; lane c of a batch holds chunk c's max
// and sum, each lane DPL output dims.  The running result is rescaled when a
// batch raises the maximum (online softmax).
template <int DPL>
__device__ __forceinline__ void attn_merge_warp(const AttnView* ap, const StepParams* sp, int b, int hk, int qi, int lane) {
  const AttnView& a = *ap;
  constexpr int d = 32 * DPL;
  constexpr int kMergeBatch = 16;
  using VecT = typename std::conditional<DPL == 4, float4, float2>::type;
  const int L = sp->req_len[b], tok0 = sp->req_tok0[b];
  const int G = a.Hq / a.Hkv;
  const int nc = n_chunks_of(L, a.cs);
  const size_t cstride = (size_t)a.qmax * part_stride(d);
  const float* base = a.part + (((size_t)b * a.Hkv + hk) * a.n_chunks) * cstride + (size_t)qi * part_stride(d);
  float M = -INFINITY, den = 0.f, num[DPL];
#pragma unroll
  for (int u = 0; u < DPL; ++u) num[u] = 0.f;
  for (int c0 = 0; c0 < nc; c0 += kMergeBatch) {
    float mc = -INFINITY, lc = 0.f;
    if (lane < kMergeBatch && c0 + lane < nc) {
      const float2 ml = __ldcg(reinterpret_cast<const float2*>(base + (size_t)(c0 + lane) * cstride));
      mc = ml.x;
      lc = ml.y;
    }
    VecT ov[kMergeBatch];
#pragma unroll
    for (int u = 0; u < kMergeBatch; ++u) {
      if (c0 + u < nc) {
        ov[u] = __ldcg(reinterpret_cast<const VecT*>(base + (size_t)(c0 + u) * cstride + 4) + lane);
      } else {
        ov[u] = VecT{};
      }
    }
    float bm = mc;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, o));
    const float Mn = fmaxf(M, bm);
    const float alpha = (M == -INFINITY) ? 0.f : expf(M - Mn);
    den *= alpha;
#pragma unroll
    for (int u = 0; u < DPL; ++u) num[u] *= alpha;
    const float wl = (mc == -INFINITY) ? 0.f : expf(mc - Mn);
    float dl = lc * wl;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dl += __shfl_xor_sync(0xffffffffu, dl, o);
    den += dl;
#pragma unroll
    for (int u = 0; u < kMergeBatch; ++u) {
      const float w = __shfl_sync(0xffffffffu, wl, u);
      const float* f = reinterpret_cast<const float*>(&ov[u]);
#pragma unroll
      for (int v = 0; v < DPL; ++v) num[v] = fmaf(f[v], w, num[v]);
    }
    M = Mn;
  }
  uint16_t* out = a.out + (size_t)(tok0 + qi / G) * a.out_ld + (hk * G + qi % G) * d + DPL * lane;
#pragma unroll
  for (int u = 0; u < DPL; ++u) out[u] = f2h(num[u] / den);
}

// One item, processed by the CTA's consumer warps:
//   1. the chunk's slots (beam table) and mask bits;
//   2. the K and V rows of earlier steps, in flight while the item waits
//      (bounded) for its kv head's q|k|v units;
//   3. the rows this step appends, from the fixed-point k and v sums (k
//      rotated by its token's position, both rounded to fp16) -- written to
//      the shared tile and, by the one item whose chunk holds them, to the
//      KV pool -- and the first query group;
//   4. scores: warp w takes queries w, w + kWarps, ...; lane = entry; the
//      softmax pieces (max, sum of exp) per query across the lanes;
//   5. values: thread = (query, pair of head dims), sum over the entries;
//   6. a release count of the finished chunk for its (request, kv head); when
//      every CTA has at most one item, the CTA that counts the last chunk
//      merges at once.
template <int DPL>
__device__ __forceinline__ void attn_item_cta(const AttnView* ap, int layer, const StepParams* sp, int b, int hk, int c,
                                           uint8_t* area, int* status) {
  const AttnView& a = *ap;
  uint16_t* kpool = a.kpool + (size_t)layer * a.layer_stride;
  uint16_t* vpool = a.vpool + (size_t)layer * a.layer_stride;
  using S = AttnSmem<DPL>;
  constexpr int d = S::d, KP = d / 8, half = d / 2;  // 16-byte pieces per row
  uint16_t* Ks = reinterpret_cast<uint16_t*>(area);
  uint16_t* Vs = reinterpret_cast<uint16_t*>(area + S::kK);
  float* qsm = reinterpret_cast<float*>(area + S::kK + S::kV);
  float* ps = reinterpret_cast<float*>(area + S::kK + S::kV + S::kQ);
  int* slot_s = reinterpret_cast<int*>(area + S::kK + S::kV + S::kQ + S::kP);
  int* vis_s = slot_s + kChunk;
  uint8_t* vis_t = reinterpret_cast<uint8_t*>(vis_s + kChunk);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int L = sp->req_len[b], P = sp->req_P[b];
  const int tok0 = sp->req_tok0[b], nb = sp->req_tok0[b + 1] - tok0;
  const int G = a.Hq / a.Hkv, Q = nb * G;
  const int j0 = c * a.cs, nj = min(a.cs, L - j0);
  const float scale = rsqrtf(static_cast<float>(d));
  float* part = a.part + ((((size_t)b * a.Hkv + hk) * a.n_chunks + c) * a.qmax) * part_stride(d);

  // 1. the chunk's slots and mask bits (independent of this step's projections);
  //    packed mode (Section 8.6): one mask row per token, each query reads its
  //    token's row and no implicit causal bound applies
  if (tid < kChunk) {
    int slot = 0, vis = 0;
    if (tid < nj) {
      slot = __ldcg(a.bt + (size_t)b * a.cap + j0 + tid);
      vis = a.packed ? 1 : __ldcg(a.mask + (size_t)b * a.mask_stride + j0 + tid) != 0;
    }
    slot_s[tid] = slot;
    vis_s[tid] = vis;
  }
  if (a.packed)
    for (int e = tid; e < nb * nj; e += kThreads)
      vis_t[(e / nj) * kChunk + e % nj] = __ldcg(a.mask + (size_t)(tok0 + e / nj) * a.mask_stride + j0 + e % nj) != 0;
  cbar();
  {
    constexpr int kRowPieces = kChunk * KP;
    constexpr int kPer = (2 * kRowPieces + kThreads - 1) / kThreads;
    uint4 v[kPer];
    auto row_of = [&](int r) {
      const int sl = slot_s[r];
      return (((size_t)(sl / a.cap) * a.Hkv + hk) * a.cap + sl % a.cap) * d;
    };
    // 2. K/V rows of entries from earlier steps: in flight during the wait
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int pi = tid + i * kThreads, r = (pi % kRowPieces) / KP;
      v[i] = make_uint4(0, 0, 0, 0);
      if (pi < 2 * kRowPieces && r < nj && j0 + r < P)
        v[i] = __ldcg(reinterpret_cast<const uint4*>((pi >= kRowPieces ? vpool : kpool) + row_of(r)) + pi % KP);
    }
    if (tid == 0) wait_count(a.cnt_kv + hk, a.kv_units, status, a.limit);
    cbar();
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int pi = tid + i * kThreads, r = (pi % kRowPieces) / KP;
      if (pi < 2 * kRowPieces && r < nj && j0 + r < P) {
        uint4* dst = pi >= kRowPieces ? reinterpret_cast<uint4*>(Vs + r * d) : reinterpret_cast<uint4*>(Ks + r * S::kKld);
        dst[pi % KP] = v[i];
      }
    }
  }
  // 3. the entries this step appends (they lie in the request's last chunks)
  {
    const int r0 = max(P - j0, 0), nnew = nj - r0;
    if (nnew > 0) {
      const int k_first = a.Hq * d, v_first = (a.Hq + a.Hkv) * d;
      for (int e = tid; e < nnew * half; e += kThreads) {
        const int r = r0 + e / half, i = e % half;
        const int m = tok0 + (j0 + r - P);
        const long long* row = a.acc + (size_t)m * a.acc_ld;
        const int R = rot_row(k_first, hk, i, d);
        const float lo = fixed_to_f32(__ldcg(row + R)), hi = fixed_to_f32(__ldcg(row + R + 8));
        const float2 cs = a.rope[(size_t)sp->tok_pos[m] * half + i];
        const uint16_t klo = f2h(lo * cs.x - hi * cs.y), khi = f2h(hi * cs.x + lo * cs.y);
        Ks[r * S::kKld + i] = klo;
        Ks[r * S::kKld + half + i] = khi;
        const int sl = sp->tok_slot[m];
        uint16_t* kp = kpool + (((size_t)(sl / a.cap) * a.Hkv + hk) * a.cap + sl % a.cap) * d;
        kp[i] = klo;
        kp[half + i] = khi;
      }
      for (int e = tid; e < nnew * d; e += kThreads) {
        const int r = r0 + e / d, i = e % d;
        const int m = tok0 + (j0 + r - P);
        const uint16_t vv = f2h(fixed_to_f32(__ldcg(a.acc + (size_t)m * a.acc_ld + v_first + hk * d + i)));
        Vs[r * d + i] = vv;
        const int sl = sp->tok_slot[m];
        vpool[(((size_t)(sl / a.cap) * a.Hkv + hk) * a.cap + sl % a.cap) * d + i] = vv;
      }
    }
    // rows past the chunk's end take part with weight zero: keep them finite
    for (int e = tid; e < (kChunk - nj) * KP; e += kThreads) {
      const int r = nj + e / KP;
      if (r < a.cs) {
        reinterpret_cast<uint4*>(Ks + r * S::kKld)[e % KP] = make_uint4(0, 0, 0, 0);
        reinterpret_cast<uint4*>(Vs + r * d)[e % KP] = make_uint4(0, 0, 0, 0);
      }
    }
  }
  for (int q0 = 0; q0 < Q; q0 += S::kQg) {
    const int qn = min(S::kQg, Q - q0);
    if (q0 > 0) cbar();
    attn_load_queries<DPL>(a, sp, hk, tok0, q0, qn, qsm);
    cbar();
    for (int qi = warp; qi < qn; qi += kWarps) {
      const float* qq = qsm + qi * d;
      // lane scores entries lane, lane + 32, ... (cs / 32 of them)
      float sc[kChunk / 32];
#pragma unroll
      for (int k = 0; k < kChunk / 32; ++k) sc[k] = 0.f;
      if (a.cs == 32) {
        sc[0] = dot_q_k(qq, Ks + lane * S::kKld, KP);
      } else {
#pragma unroll
        for (int k = 0; k < kChunk / 32; k += 2)
          if (32 * k < a.cs) sc[k] = dot_q_k2(qq, Ks + (lane + 32 * k) * S::kKld, Ks + (lane + 32 * k + 32) * S::kKld, sc[k + 1], KP);
      }
      const int q = q0 + qi;
      const int lim = P + q / G;  // causal limit of this query's token
      float mx = -INFINITY;
      bool vis[kChunk / 32];
#pragma unroll
      for (int k = 0; k < kChunk / 32; ++k) {
        const int e = lane + 32 * k;
        vis[k] = e < nj && vis_s[e] && (a.packed ? vis_t[(q / G) * kChunk + e] != 0 : j0 + e <= lim);
        sc[k] = vis[k] ? sc[k] * scale : -INFINITY;
        mx = fmaxf(mx, sc[k]);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float l = 0.f;
#pragma unroll
      for (int k = 0; k < kChunk / 32; ++k) {
        const float e = vis[k] ? expf(sc[k] - mx) : 0.f;
        l += e;
        if (32 * k < a.cs) ps[qi * kChunk + lane + 32 * k] = e;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
      if (lane == 0) {
        part[(size_t)q * part_stride(d)] = mx;
        part[(size_t)q * part_stride(d) + 1] = l;
      }
    }
    cbar();
    for (int w = tid; w < qn * (d / 2); w += kThreads) {
      const int qi = w / (d / 2), dp = w % (d / 2);
      const float* pq = ps + qi * kChunk;
      float o0 = 0.f, o1 = 0.f;
#pragma unroll 8
      for (int e = 0; e < a.cs; ++e) {  // rows past nj are zero with weight zero
        const float pe = pq[e];
        const float2 vf = h2f2(*reinterpret_cast<const uint32_t*>(Vs + e * d + 2 * dp));
        o0 = fmaf(pe, vf.x, o0);
        o1 = fmaf(pe, vf.y, o1);
      }
      *reinterpret_cast<float2*>(part + (size_t)(q0 + qi) * part_stride(d) + 4 + 2 * dp) = make_float2(o0, o1);
    }
  }
  // the item's partials are written (and the area is free for the next item);
  // the release orders them before the count the merging CTA acquires
  cbar();
  if (!a.last_merges) {
    if (tid == 0) red_release_add_s32(&a.cnt[b * a.Hkv + hk], 1);
    return;
  }
  __shared__ int s_last;
  if (tid == 0) s_last = atom_add_acq_rel(&a.cnt[b * a.Hkv + hk], 1) == n_chunks_of(L, a.cs) - 1;
  cbar();
  if (s_last) {
    for (int qi = warp; qi < Q; qi += kWarps) attn_merge_warp<DPL>(ap, sp, b, hk, qi, lane);
    cbar();
    if (tid == 0) a.cnt[b * a.Hkv + hk] = 0;
  }
}

// Merge of (request b, kv head hk) by its designated CTA, after that CTA's
// own items: wait until every chunk is counted (bounded), merge the queries
// (one warp each), reset the count.
template <int DPL>
__device__ __forceinline__ void attn_merge_cta(const AttnView* ap, const StepParams* sp, int b, int hk, int* status) {
  const AttnView& a = *ap;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int L = sp->req_len[b], nb = sp->req_tok0[b + 1] - sp->req_tok0[b];
  const int Q = nb * (a.Hq / a.Hkv);
  if (tid == 0) wait_count(&a.cnt[b * a.Hkv + hk], n_chunks_of(L, a.cs), status, a.limit);
  cbar();
  for (int qi = warp; qi < Q; qi += kWarps) attn_merge_warp<DPL>(ap, sp, b, hk, qi, lane);
  cbar();
  if (tid == 0) a.cnt[b * a.Hkv + hk] = 0;
}

template <int NT, int GPU, int DPL>
__global__ void __launch_bounds__(kBlockThreads, 1) step_kernel(const __grid_constant__ StepKernelArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ GemvPhase s_gp[4];            // per projection kind: q|k|v, o, gate|up, down
  constexpr int kSlots = Geom<GPU>::kStepSlots;
  __shared__ AttnView s_av;
  __shared__ uint64_t s_nbar;              // the staged RMSNorm's bulk copies
  __shared__ StepParams s_sp;
  __shared__ const uint16_t* s_rowp[kMaxTokens];  // the step's fp16 input rows
  using SS = StepSmem<GPU>;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* rings = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + SS::kRing);
  uint64_t* empty = full + kWarps * kSlots;
  uint8_t* att_area = smem + SS::kRing + SS::kBars;
  static_assert(AttnSmem<DPL>::kBytes <= SS::kQ, "attention area too small");
  OpDesc* s_ops = reinterpret_cast<OpDesc*>(smem + SS::kFixed);
  for (int i = threadIdx.x; i < 4 * a.L; i += kBlockThreads) s_ops[i] = a.ops[i];
  if (threadIdx.x == 0) {
    mbar_init(&s_nbar, 1);
    ring_init_barriers(full, empty, kWarps * kSlots);  // ends with the barrier-init fence
    if (blockIdx.x == 0) a.phase_clock[0] = globaltimer();
  }
  prologue_params(a.pro, &s_sp, s_rowp);  // ends with a block-wide barrier
  const int n_barriers = 4 * a.L + 1;
  if (s_sp.abort_step) {
    // every CTA sees the same inputs and rejects the step alike: count this
    // launch's barrier arrivals at once and write nothing
    if (threadIdx.x == 0) {
      red_release_add(a.barrier, (unsigned long long)n_barriers);
      if (blockIdx.x == 0) {
        atomicOr(a.pro.status, s_sp.abort_step & ~ST_STICKY);
        *reinterpret_cast<volatile int*>(a.status_out) = ld_acquire_s32(a.pro.status);
      }
    }
    return;
  }
  if (!kSelfRefill && warp == kWarps) {  // the producer warp
    ring_producer<GPU, kSlots>(s_ops, 4 * a.L, blockIdx.x, gridDim.x, kWarps, rings, full, empty, a.status,
                               kProducerLimit, lane);
    return;
  }
  // ---- consumer warps from here on: CTA barriers are cbar() ----
  const StepParams* sp = &s_sp;
  const int M = sp->M;
  GridBarrier gb{a.barrier, a.barrier_base, a.status, a.phase_clock, 0, 0, a.debug_skip_arrival, a.wait_limit};
  // this warp's ring (its state stays in registers for the whole step)
  WarpRing<GPU, kSlots> ring;
  ring.ring = rings + (size_t)warp * kSlots * Geom<GPU>::kUnitBytes;
  ring.full = full + warp * kSlots;
  ring.empty = empty + warp * kSlots;
  ring.n_used = 0;
  ring.timed_out = false;
  if (kSelfRefill) ring.start(s_ops, 4 * a.L, blockIdx.x * kWarps + warp, gridDim.x * kWarps, lane);
  // Each CTA normalises the whole hidden state for itself; when the M rows
  // fit, it keeps them in the attention area (idle during the q|k|v and
  // gate|up projections) and the projections read them from there.  Rows are
  // padded by 32 halves so that the two token rows a fragment load touches in
  // one phase fall on different banks.
  const int xn_ld = a.H + 32;
  const bool xn_smem = kNormInSmem && a.Kp_H == a.H && (size_t)M * xn_ld * 2 <= SS::kQ;
  uint16_t* xn = xn_smem ? reinterpret_cast<uint16_t*>(att_area) : a.act_h;
  const int xn_out_ld = xn_smem ? xn_ld : a.Kp_H;
  // one row from the residual stream: staged through shared memory behind
  // the normalised row (rmsnorm_staged)
  const size_t stage_off = ((size_t)M * xn_ld * 2 + 127) / 128 * 128;
  const bool norm_staged = M == 1 && xn_smem && a.H <= 24 * kThreads && stage_off + (size_t)a.H * 8 <= SS::kQ;
  long long* stage = reinterpret_cast<long long*>(att_area + stage_off);
  uint32_t nphase = 0;
  const int G = a.Hq / a.Hkv;
  if (threadIdx.x < 4) {
    const int k = threadIdx.x;
    GemvPhase gp{};
    gp.act = k == 0 || k == 2 ? a.act_h : k == 1 ? a.act_attn : a.act_f;
    gp.act_ld = k == 0 || k == 2 ? a.Kp_H : k == 1 ? a.Kp_dq : a.Kp_F;
    gp.M = M;
    gp.act_s = (k == 0 || k == 2) && xn_smem ? smem_addr(att_area) : 0u;
    gp.act_s_ld = xn_ld;
    gp.status = a.status;
    gp.ep.kind = k == 0 ? EPI_QKV : k == 2 ? EPI_SWIGLU : EPI_RESID;
    gp.ep.dims = OpDims{k, a.Hq, a.Hkv, a.d, a.F, a.H};
    gp.ep.acc = k == 0 ? a.acc_qkv : k == 2 ? a.acc_gu : a.X;
    gp.ep.acc_ld = k == 0 ? (a.Hq + 2 * a.Hkv) * a.d : k == 2 ? s_ops[2].n_rb * kRowsPerBlock : a.H;
    gp.ep.cnt = k == 0 ? a.cnt_kv : k == 2 ? a.cnt_gu : nullptr;
    gp.ep.h = a.act_f;
    gp.ep.h_ld = a.Kp_F;
    gp.kv_rb_q = G * a.d / kRowsPerBlock;
    gp.kv_rb_per_head = a.d / kRowsPerBlock;
    gp.kv_rb_k = a.Hq * a.d / kRowsPerBlock;
    gp.kv_rb_v = (a.Hq + a.Hkv) * a.d / kRowsPerBlock;
    gp.part = reinterpret_cast<float*>(smem + SS::kFixed + SS::ops_bytes(a.L));
    s_gp[k] = gp;
  }
  if (threadIdx.x == 32) {
    AttnView av{};
    av.acc = a.acc_qkv;
    av.acc_ld = (a.Hq + 2 * a.Hkv) * a.d;
    av.rope = a.rope;
    av.kpool = a.kpool;
    av.vpool = a.vpool;
    av.layer_stride = a.layer_stride;
    av.cap = a.cap;
    av.Hq = a.Hq;
    av.Hkv = a.Hkv;
    av.d = a.d;
    av.n_chunks = a.n_chunks;
    av.qmax = kMaxTokens * G;
    av.part = a.attn_part;
    av.cnt = a.attn_cnt;
    av.cnt_kv = a.cnt_kv;
    av.kv_units = (G + 2) * (a.d / kRowsPerBlock) * s_ops[0].upr;
    av.bt = a.pro.bt_dst;
    av.mask = a.mask;
    av.mask_stride = a.mask_stride;
    av.packed = a.packed;
    av.limit = a.wait_limit;
    int items = 0;
    for (int b = 0; b < sp->B; ++b) items += a.Hkv * n_chunks_of(sp->req_len[b], kAttnChunkMin);
    // the smallest item size that needs one round of CTAs, else the largest
    av.cs = kAttnChunkMin;
    while (av.cs < kChunk && items > (int)gridDim.x) {
      av.cs *= 2;
      items = 0;
      for (int b = 0; b < sp->B; ++b) items += a.Hkv * n_chunks_of(sp->req_len[b], av.cs);
    }
    av.last_merges = items <= (int)gridDim.x;
    av.out = a.act_attn;
    av.out_ld = a.Kp_dq;
    s_av = av;
  }
  cbar();
  prologue_work(a.pro, sp, s_rowp, a.X);
  cbar();
  gb.arrive();  // split barrier: waited for before the first attention

  const int g = blockIdx.x * kWarps + warp, nw = gridDim.x * kWarps;
  const int gt = blockIdx.x * kThreads + threadIdx.x, gs = gridDim.x * kThreads;
  const int qkv_rows = (a.Hq + 2 * a.Hkv) * a.d;

  // Phase k of layer l = ph / 4: q|k|v (k = 0), o, gate|up, down.  Every
  // phase body has one call site, so all of it is inlined into the kernel.
  for (int ph = 0; ph < 4 * a.L; ++ph) {
    const int l = ph >> 2, k = ph & 3;
    if (k == 0 || k == 2) {
      // RMSNorm of the attention (k = 0) or MLP block; before the first
      // layer from the step's input rows
      const uint16_t* nw_ = a.norms + (size_t)l * 2 * a.H + (k == 2 ? a.H : 0);
      if (norm_staged && ph != 0)
        rmsnorm_staged(a.X, a.H, nw_, a.eps, xn, stage, &s_nbar, nphase, a.status);
      else
        rmsnorm_cta(ph != 0, a.X, s_rowp, a.H, nw_, a.eps, xn, xn_out_ld, M);
    } else if (k == 1) {
      // the q|k|v sums and counts are consumed: clear them for the next layer
      for (int e = gt; e < M * qkv_rows; e += gs) __stcg(a.acc_qkv + e, 0LL);
      if (blockIdx.x == 0 && threadIdx.x < a.Hkv) __stcg(a.cnt_kv + threadIdx.x, 0);
    }
    gemv_run<NT, GPU, kSlots>(ring, &s_ops[ph], &s_gp[k], g, nw, lane);
    if (k == 0) {
      if (l == 0) gb.wait();        // the prologue's tables and residual are complete
      else if (xn_smem) cbar();     // the attention items reuse the normalised rows' space
      int total = 0;
      for (int b = 0; b < sp->B; ++b) total += a.Hkv * n_chunks_of(sp->req_len[b], s_av.cs);
      for (int item = blockIdx.x; item < total; item += gridDim.x) {
        int b, hk, c;
        if (decode_item(sp, a.Hkv, s_av.cs, item, b, hk, c)) attn_item_cta<DPL>(&s_av, l, sp, b, hk, c, att_area, a.status);
      }
      // merges, when CTAs take several items: (b, hk) goes to the CTA that
      // took its last chunk
      for (int b = 0, base = 0; !s_av.last_merges && b < sp->B; ++b) {
        const int nc = n_chunks_of(sp->req_len[b], s_av.cs);
        for (int hk = 0; hk < a.Hkv; ++hk)
          if ((base + hk * nc + nc - 1) % gridDim.x == blockIdx.x) attn_merge_cta<DPL>(&s_av, sp, b, hk, a.status);
        base += a.Hkv * nc;
      }
    }
    gb.sync();
  }
  // hidden_out = fp16(x): one rounding from the exact fixed-point value
  for (int e = gt; e < M * a.H; e += gs) {
    const double v = static_cast<double>(__ldcg(a.X + e)) * kFixInv;
    a.pro.hidden_out[e] = __half_as_ushort(__double2half(v));
  }
  if (blockIdx.x == 0 && threadIdx.x < sp->B) a.pro.lens[threadIdx.x] = sp->req_len[threadIdx.x];
  if (ring.timed_out && lane == 0) atomicOr(a.status, ST_WAIT_TIMEOUT);
  // The last CTA to finish hands a nonzero status to the host-mapped mirror,
  // so no copy-engine transfer has to follow the step on the stream.
  cbar();
  if (threadIdx.x == 0 && atom_add_acq_rel(a.exit_count, 1) == (int)gridDim.x - 1) {
    *a.exit_count = 0;
    const int st = ld_acquire_s32(a.status);
    if (st) *reinterpret_cast<volatile int*>(a.status_out) = st;
  }
}

template <int NT, int GPU, int DPL>
cudaError_t launch_t(const StepKernelArgs& a, int grid, cudaStream_t s) {
  auto kern = step_kernel<NT, GPU, DPL>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kBlockThreads);
  cfg.dynamicSmemBytes = a.gu_part ? StepSmem<GPU>::total_with_part(a.L) : StepSmem<GPU>::total(a.L);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int NT, int GPU, int DPL>
size_t dyn_limit_t() {
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return 0;
  cudaFuncAttributes fa;
  if (cudaFuncGetAttributes(&fa, step_kernel<NT, GPU, DPL>) != cudaSuccess) return 0;
  return (size_t)optin > fa.sharedSizeBytes ? (size_t)optin - fa.sharedSizeBytes : 0;
}

// The largest dynamic shared memory the kernel may take.
template <int NT, int GPU, int DPL>
cudaError_t setup_t() {
  return cudaFuncSetAttribute(step_kernel<NT, GPU, DPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)dyn_limit_t<NT, GPU, DPL>());
}

// Dynamic shared memory every kernel of a group size may take (0: unknown group).
template <int GPU>
size_t dyn_limit_group() {
  size_t m = dyn_limit_t<1, GPU, 4>();
  m = std::min(m, dyn_limit_t<2, GPU, 4>());
  m = std::min(m, dyn_limit_t<1, GPU, 2>());
  return std::min(m, dyn_limit_t<2, GPU, 2>());
}

template <int GPU>
bool part_fits(int L) {
  return StepSmem<GPU>::total_with_part(L) <= dyn_limit_group<GPU>();
}

}  // namespace

int step_barriers(int n_layers) { return 4 * n_layers + 1; }

int step_gu_cta_tokens() { return kGuCtaTokens; }

bool step_gu_part_fits(int group, int L) {
  if (group == 128) return part_fits<1>(L);
  if (group == 64) return part_fits<2>(L);
  if (group == 32) return part_fits<4>(L);
  return false;
}

int step_gu_split(int n_rb, int upr, int grid, int group, int L) {
  if (n_rb < 1 || upr < 1 || grid < 1 || !step_gu_part_fits(group, L)) return 0;
  const long long nw = (long long)grid * kWarps;
  const long long even = ((long long)n_rb * upr + nw - 1) / nw;  // most units per warp, grid-wide split
  int best = 0;
  for (int q = 1; q <= kWarps; ++q) {
    if (kWarps % q != 0 || (long long)n_rb * q > nw) continue;  // one round of CTAs
    const long long most = (upr + q - 1) / q;
    if (most <= even + std::max(1LL, even / 16)) best = q;  // about as balanced as the grid-wide split
  }
  return best;
}

size_t step_attention_part_floats(int B, int Hkv, int n_chunks, int G, int d) {
  return (size_t)B * Hkv * n_chunks * (kMaxTokens * G) * part_stride(d);
}

cudaError_t step_setup(int group, int head_dim) {
  cudaError_t e = cudaSuccess;
#define SETUP_PAIR(GPU, DPL)                                       \
  if ((e = setup_t<1, GPU, DPL>()) != cudaSuccess) return e;       \
  if ((e = setup_t<2, GPU, DPL>()) != cudaSuccess) return e;
  if (head_dim == 128) {
    if (group == 128) { SETUP_PAIR(1, 4) }
    else if (group == 64) { SETUP_PAIR(2, 4) }
    else if (group == 32) { SETUP_PAIR(4, 4) }
  } else if (head_dim == 64) {
    if (group == 128) { SETUP_PAIR(1, 2) }
    else if (group == 64) { SETUP_PAIR(2, 2) }
    else if (group == 32) { SETUP_PAIR(4, 2) }
  } else {
    return cudaErrorInvalidValue;
  }
#undef SETUP_PAIR
  return e;
}

cudaError_t launch_step(const StepKernelArgs& a, int nt, int group, int grid, cudaStream_t s) {
  const int dpl = a.d / 32;
#define LAUNCH(GPU, DPL) return nt == 1 ? launch_t<1, GPU, DPL>(a, grid, s) : launch_t<2, GPU, DPL>(a, grid, s);
  if (dpl == 4) {
    if (group == 128) LAUNCH(1, 4)
    if (group == 64) LAUNCH(2, 4)
    if (group == 32) LAUNCH(4, 4)
  } else if (dpl == 2) {
    if (group == 128) LAUNCH(1, 2)
    if (group == 64) LAUNCH(2, 2)
    if (group == 32) LAUNCH(4, 2)
  }
#undef LAUNCH
  return cudaErrorInvalidValue;
}

}  // namespace shard
