// The whole decode step of a shard as one persistent, cooperative kernel.
//
// One CTA per SM, kCtaWarps warps.  The step runs as a sequence of phases separated
// by grid-wide barriers ('|'):
//   prologue (CTA 0) | for each layer: RMSNorm + q|k|v projection (+RoPE,
//   K/V append) -> attention (chunk partials and merges) | o projection
//   (+residual) | RMSNorm + gate|up projection (+SwiGLU) | down projection
//   (+residual; the last layer writes hidden_out).
// '->' is dataflow instead of a barrier: each q|k|v row-block's finisher
// release-stores the launch's epoch of that projection into the row-block's
// flag, and an attention item waits (acquire loads, bounded) only for the
// row-blocks of its kv head.  Flags are never cleared: an epoch is unique per
// launch and op.
// Each RMSNorm is computed by every CTA at the start of the projection that
// consumes it, from per-row-block sums of squares left by the residual's
// producer, so it needs no barrier of its own.
// Every warp owns a ring of weight slots (gemv_core.cuh) that streams, in
// order, all the projection units the warp will process during the step.
// The ring refills as soon as a slot is consumed, independent of the
// barriers, so while a warp waits at a barrier or works on norms and
// attention, the next projection's weights are already arriving.
//
// Barrier waits are bounded: a wait that runs out sets a status bit and
// proceeds (the step's results are then reported invalid) instead of hanging.
#include <type_traits>

#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kWarps = kCtaWarps;
constexpr int kThreads = kWarps * 32;
constexpr int kChunk = kAttnChunk;  // most cache entries per attention item (four per lane)
constexpr bool kNormInSmem = true;   // normalised activations in shared memory when they fit
constexpr bool kNormPrefetch = true; // RMSNorm: first x loads issued with the sums-of-squares loads

template <int GPU>
struct StepSmem {
  static constexpr size_t kRing = (size_t)kWarps * kRingSlots * Geom<GPU>::kUnitBytes;
  static constexpr size_t kBars = (size_t)kWarps * kRingSlots * sizeof(uint64_t);
  // attention item area (AttnSmem)
  static constexpr size_t kQ = 96 * 1024;
  static constexpr size_t kFixed = kRing + kBars + kQ;  // + the op table (4L entries)
  static size_t total(int n_layers) { return kFixed + (size_t)4 * n_layers * sizeof(OpDesc); }
};

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Grid-wide barrier on a monotonically increasing counter.  `target` is this
// CTA's running count of expected arrivals.
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

__device__ __forceinline__ void red_release_add_s32(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_s32(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void red_release_add(unsigned long long* p, unsigned long long v) {
  asm volatile("red.release.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ void grid_sync(unsigned long long* ctr, unsigned long long& target, int* status,
                          unsigned long long* clock, int& nsync) {
  __syncthreads();
  if (threadIdx.x == 0) {
    target += gridDim.x;
    red_release_add(ctr, 1ULL);
    // bounded: after ~2^22 polls, or once any CTA has given up, stop waiting
    uint32_t it = 0;
    while (ld_acquire_u64(ctr) < target) {
      if (++it > (1u << 22)) {
        atomicOr(status, ST_WAIT_TIMEOUT);
        break;
      }
      if ((it & 1023) == 0 && (*reinterpret_cast<volatile int*>(status) & ST_WAIT_TIMEOUT)) break;
      __nanosleep(64);
    }
    if (blockIdx.x == 0) clock[nsync] = globaltimer();
  }
  ++nsync;
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Prologue (CTA 0): the beam_idx gather of the entry tables (Section 4: row b
// continues row beam_idx[b]'s entries; K/V stay where they are), the new
// entries' slots, device-side argument checks, and the residual stream.
// ---------------------------------------------------------------------------
__device__ __noinline__ void prologue_cta(const PrologueArgs& a) {
  __shared__ int s_src[kMaxRequests], s_P[kMaxRequests], s_len[kMaxRequests], s_tok0[kMaxRequests + 1];
  __shared__ int s_req[kMaxTokens], s_idx[kMaxTokens];
  __shared__ int s_err;
  const int tid = threadIdx.x, nth = blockDim.x;
  if (tid == 0) {
    // a step rejected earlier freezes the state until the host resets it
    s_err = __ldcg(a.status) != 0 ? ST_STICKY : 0;
    int t = 0;
    for (int b = 0; b < a.B; ++b) {
      s_tok0[b] = t;
      for (int i = 0; i < a.n_new[b]; ++i, ++t) {
        s_req[t] = b;
        s_idx[t] = i;
      }
    }
    s_tok0[a.B] = t;
  }
  __syncthreads();
  if (tid < a.B) {
    int src = a.beam_idx ? __ldcg(a.beam_idx + tid) : tid;
    if (src < 0 || src >= a.B) {
      atomicOr(&s_err, ST_BEAM_IDX);
      src = tid;
    }
    s_src[tid] = src;
    s_P[tid] = __ldcg(a.lens + src);
  }
  __syncthreads();
  if (tid < a.B) {
    const int L = s_P[tid] + a.n_new[tid];
    if (L > a.cap || a.cursor[tid] + a.n_new[tid] > a.cap) atomicOr(&s_err, ST_CAPACITY);
    if (L > a.mask_stride) atomicOr(&s_err, ST_MASK_STRIDE);
    s_len[tid] = L;
  }
  __syncthreads();
  for (int m = tid; m < a.M; m += nth) {
    const int b = s_req[m], j = s_P[b] + s_idx[m];
    if (j < a.mask_stride && __ldcg(a.mask + (size_t)b * a.mask_stride + j) == 0) atomicOr(&s_err, ST_MASK_NEW);
    const int pos = __ldcg(a.position_ids + m);
    if (pos < 0 || pos >= a.max_position) atomicOr(&s_err, ST_POSITION);
    if (a.token_ids) {
      const int tok = __ldcg(a.token_ids + m);
      if (tok < 0 || tok >= a.vocab) atomicOr(&s_err, ST_TOKEN);
    }
  }
  __syncthreads();
  if (s_err) {
    if (tid == 0) {
      atomicOr(a.status, s_err & ~ST_STICKY);
      a.sp->abort_step = 1;
    }
    return;
  }
  if (a.beam_idx) {
    for (int b = 0; b < a.B; ++b) {
      const int* src = a.bt_src + (size_t)s_src[b] * a.cap;
      int* dst = a.bt_dst + (size_t)b * a.cap;
      for (int j = tid; j < s_P[b]; j += nth) dst[j] = __ldcg(src + j);
    }
  }
  for (int m = tid; m < a.M; m += nth) {
    const int b = s_req[m], i = s_idx[m];
    a.bt_dst[(size_t)b * a.cap + s_P[b] + i] = b * a.cap + a.cursor[b] + i;
  }
  if (tid < a.B) a.lens[tid] = s_len[tid];
  // residual x: warp per (token, 64-row block), which also leaves the
  // block's sum of squares for the first RMSNorm
  {
    const int n_rb = (a.H + kRowsPerBlock - 1) / kRowsPerBlock;
    const int lane = tid & 31;
    for (int it = tid >> 5; it < a.M * n_rb; it += nth >> 5) {
      const int m = it / n_rb, rb = it % n_rb;
      const uint16_t* src = a.hidden_in ? a.hidden_in + (size_t)m * a.H
                                        : a.embedding + (size_t)__ldcg(a.token_ids + m) * a.H;
      float ss = 0.f;
#pragma unroll
      for (int r = 0; r < kRowsPerBlock; r += 32) {
        const int k = rb * kRowsPerBlock + r + lane;
        if (k < a.H) {
          const float v = h2f(a.hidden_in ? __ldcg(src + k) : src[k]);
          a.x[(size_t)m * a.H + k] = v;
          ss = fmaf(v, v, ss);
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
      if (lane == 0) a.ss[rb * kMaxTokens + m] = ss;
    }
  }
  if (tid == 0) {
    StepParams* sp = a.sp;
    sp->M = a.M;
    sp->B = a.B;
    sp->abort_step = 0;
    for (int m = 0; m < a.M; ++m) {
      const int b = s_req[m];
      sp->tok_req[m] = b;
      sp->tok_idx[m] = s_idx[m];
      sp->tok_pos[m] = __ldcg(a.position_ids + m);
      sp->tok_slot[m] = b * a.cap + a.cursor[b] + s_idx[m];
    }
    for (int b = 0; b <= a.B; ++b) sp->req_tok0[b] = s_tok0[b];
    for (int b = 0; b < a.B; ++b) {
      sp->req_P[b] = s_P[b];
      sp->req_len[b] = s_len[b];
    }
    sp->mask = a.mask;
    sp->mask_stride = a.mask_stride;
    sp->hidden_out = a.hidden_out;
    sp->bt = a.bt_dst;
  }
}

// ---------------------------------------------------------------------------
// RMSNorm, run by every CTA at the start of the projection that consumes it.
// r[m] = 1 / sqrt(mean(x[m]^2) + eps) from the per-row-block sums of squares
// that the residual's producer left (added in a fixed order, so every CTA
// gets the same r); then act = fp16(x * r * w).  Every CTA writes the whole
// act -- the same bits -- so its own warps can start as soon as it is done.
// H is a multiple of 4.
// ---------------------------------------------------------------------------
__device__ __noinline__ void rmsnorm_cta(const float* x, int H, const uint16_t* w, float eps, const float* ss,
                                         uint16_t* out, int out_ld, int M) {
  __shared__ float s_r[kMaxTokens];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_rb = (H + kRowsPerBlock - 1) / kRowsPerBlock;
  constexpr int kBatch = 4;  // float4 pieces per thread in flight
  const int H4 = H / 4, n4 = M * H4;
  float4 xv[kBatch];
  uint2 wv[kBatch];
  auto load = [&](int i0) {
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int i = i0 + j * kThreads;
      if (i < n4) {
        xv[j] = __ldcg(reinterpret_cast<const float4*>(x) + i);
        wv[j] = *reinterpret_cast<const uint2*>(w + 4 * (i % H4));
      }
    }
  };
  auto store = [&](int i0) {
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int i = i0 + j * kThreads;
      if (i < n4) {
        const int m = i / H4, k = 4 * (i % H4);
        const float r = s_r[m];
        const float2 w01 = h2f2(wv[j].x), w23 = h2f2(wv[j].y);
        uint2 o;
        o.x = pack_h2(xv[j].x * r * w01.x, xv[j].y * r * w01.y);
        o.y = pack_h2(xv[j].z * r * w23.x, xv[j].w * r * w23.y);
        *reinterpret_cast<uint2*>(out + (size_t)m * out_ld + k) = o;
      }
    }
  };
  // the first batch of x and weights is in flight with the sums of squares
  if (kNormPrefetch) load(tid);
  for (int m = warp; m < M; m += kWarps) {
    float t = 0.f;
    for (int rb = lane; rb < n_rb; rb += 32) t += __ldcg(ss + rb * kMaxTokens + m);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) s_r[m] = rsqrtf(t / H + eps);
  }
  __syncthreads();
  if (kNormPrefetch) store(tid);
  for (int i0 = tid + (kNormPrefetch ? kBatch * kThreads : 0); i0 < n4; i0 += kBatch * kThreads) {
    load(i0);
    store(i0);
  }
  __syncthreads();
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
  const float* q;
  const uint16_t* kpool;  // layer 0; layer l at + l * layer_stride
  const uint16_t* vpool;
  size_t layer_stride;
  int cap, Hq, Hkv, d, n_chunks, qmax;
  float* part;
  int* cnt;  // finished chunks per (request, kv head)
  const unsigned* rb_done;  // q|k|v row-block flags the items wait for
  int rb_k0, rb_v0;         // first k and v row-block of the q|k|v projection
  int cs;    // entries per item this step: 32, 64 or 128 (kChunk)
  int last_merges;  // at most one item per CTA: the CTA finishing the last chunk merges at once
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
  static constexpr size_t kBytes = kK + kV + kQ + kP + 2 * kChunk * sizeof(int);
};

// Merge of one (request, kv head, query): chunks in order, kMergeBatch at a
// time with all their loads in flight; lane c of a batch holds chunk c's max
// and sum, each lane DPL output dims.  The running result is rescaled when a
// batch raises the maximum (online softmax).
template <int DPL>
__device__ __noinline__ void attn_merge_warp(const AttnView* ap, const StepParams* sp, int b, int hk, int qi, int lane) {
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

// One item, processed by the whole CTA:
//   1. the chunk's slots (beam table) and mask bits;
//   2. its K and V rows -- those of earlier steps before waiting for this
//      step's q|k|v row-blocks, the appended ones after -- and the first query
//      group into shared memory, every load of a thread in flight at once;
//   3. scores: warp w takes queries w, w + kWarps, ...; lane = entry; the
//      softmax pieces (max, sum of exp) per query across the lanes;
//   4. values: thread = (query, pair of head dims), sum over the entries;
//   5. a release count of the finished chunk for its (request, kv head); when
//      every CTA has at most one item, the CTA that counts the last chunk
//      merges at once.
template <int DPL>
__device__ __noinline__ void attn_item_cta(const AttnView* ap, int layer, const StepParams* sp, int b, int hk, int c,
                                           uint8_t* area, unsigned qkv_epoch, int* status) {
  const AttnView& a = *ap;
  const uint16_t* kpool = a.kpool + (size_t)layer * a.layer_stride;
  const uint16_t* vpool = a.vpool + (size_t)layer * a.layer_stride;
  using S = AttnSmem<DPL>;
  constexpr int d = S::d, KP = d / 8;  // 16-byte pieces per row
  uint16_t* Ks = reinterpret_cast<uint16_t*>(area);
  uint16_t* Vs = reinterpret_cast<uint16_t*>(area + S::kK);
  float* qsm = reinterpret_cast<float*>(area + S::kK + S::kV);
  float* ps = reinterpret_cast<float*>(area + S::kK + S::kV + S::kQ);
  int* slot_s = reinterpret_cast<int*>(area + S::kK + S::kV + S::kQ + S::kP);
  int* vis_s = slot_s + kChunk;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int L = sp->req_len[b], P = sp->req_P[b];
  const int tok0 = sp->req_tok0[b], nb = sp->req_tok0[b + 1] - tok0;
  const int G = a.Hq / a.Hkv, Q = nb * G;
  const int j0 = c * a.cs, nj = min(a.cs, L - j0);
  const float scale = rsqrtf(static_cast<float>(d));
  float* part = a.part + ((((size_t)b * a.Hkv + hk) * a.n_chunks + c) * a.qmax) * part_stride(d);
  // query qi of the item is head hk * G + qi % G of token tok0 + qi / G
  auto q_src = [&](int qi) { return a.q + (size_t)(tok0 + qi / G) * a.Hq * d + (hk * G + qi % G) * d; };

  // 1. the chunk's slots and mask bits (independent of this step's projections)
  if (tid < kChunk) {
    int slot = 0, vis = 0;
    if (tid < nj) {
      slot = __ldcg(sp->bt + (size_t)b * a.cap + j0 + tid);
      vis = __ldcg(sp->mask + (size_t)b * sp->mask_stride + j0 + tid) != 0;
    }
    slot_s[tid] = slot;
    vis_s[tid] = vis;
  }
  __syncthreads();
  {
    constexpr int kRowPieces = kChunk * KP;
    constexpr int kPer = (2 * kRowPieces + kThreads - 1) / kThreads;
    constexpr int kQPieces = S::kQg * d / 4;
    constexpr int kQPer = (kQPieces + kThreads - 1) / kThreads;
    const int qn0 = min(S::kQg, Q);
    uint4 v[kPer];
    float4 qv[kQPer];
    auto load_row_piece = [&](int pi, int r) {
      const int sl = slot_s[r];
      const size_t row = (((size_t)(sl / a.cap) * a.Hkv + hk) * a.cap + sl % a.cap) * d;
      return __ldcg(reinterpret_cast<const uint4*>((pi >= kRowPieces ? vpool : kpool) + row) + pi % KP);
    };
    // 2. K/V rows of entries from earlier steps: in flight during the wait
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int pi = tid + i * kThreads, r = (pi % kRowPieces) / KP;
      v[i] = make_uint4(0, 0, 0, 0);
      if (pi < 2 * kRowPieces && r < nj && j0 + r < P) v[i] = load_row_piece(pi, r);
    }
    // 3. wait (bounded) for this kv head's q|k|v row-blocks: its G q heads,
    //    its k and its v
    {
      const int per_head = d / kRowsPerBlock > 0 ? d / kRowsPerBlock : 1;
      const int nq = G * d / kRowsPerBlock, n = nq + 2 * per_head;
      if (tid < n) {
        const int r = tid < nq ? hk * G * d / kRowsPerBlock + tid
                               : (tid < nq + per_head ? a.rb_k0 + hk * per_head + (tid - nq)
                                                      : a.rb_v0 + hk * per_head + (tid - nq - per_head));
        uint32_t it = 0;
        while (ld_acquire_u32(a.rb_done + r) != qkv_epoch) {
          if (++it > (1u << 22)) {
            atomicOr(status, ST_WAIT_TIMEOUT);
            break;
          }
          __nanosleep(64);
        }
      }
      __syncthreads();
    }
    // 4. the rows this step appended, and the queries
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int pi = tid + i * kThreads, r = (pi % kRowPieces) / KP;
      if (pi < 2 * kRowPieces && r < nj && j0 + r >= P) v[i] = load_row_piece(pi, r);
    }
#pragma unroll
    for (int i = 0; i < kQPer; ++i) {
      const int pi = tid + i * kThreads, qi = pi / (d / 4);
      qv[i] = (pi < kQPieces && qi < qn0) ? __ldcg(reinterpret_cast<const float4*>(q_src(qi)) + pi % (d / 4))
                                          : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int pi = tid + i * kThreads, r = (pi % kRowPieces) / KP;
      if (pi < 2 * kRowPieces) {
        uint4* dst = pi >= kRowPieces ? reinterpret_cast<uint4*>(Vs + r * d) : reinterpret_cast<uint4*>(Ks + r * S::kKld);
        dst[pi % KP] = v[i];
      }
    }
#pragma unroll
    for (int i = 0; i < kQPer; ++i) {
      const int pi = tid + i * kThreads;
      if (pi < kQPieces) reinterpret_cast<float4*>(qsm)[pi] = qv[i];
    }
  }
  for (int q0 = 0; q0 < Q; q0 += S::kQg) {
    const int qn = min(S::kQg, Q - q0);
    if (q0 > 0) {
      __syncthreads();
      for (int pi = tid; pi < qn * (d / 4); pi += kThreads)
        reinterpret_cast<float4*>(qsm)[pi] =
            __ldcg(reinterpret_cast<const float4*>(q_src(q0 + pi / (d / 4))) + pi % (d / 4));
    }
    __syncthreads();
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
        vis[k] = e < nj && vis_s[e] && j0 + e <= lim;
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
    __syncthreads();
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
  __syncthreads();
  if (!a.last_merges) {
    if (tid == 0) red_release_add_s32(&a.cnt[b * a.Hkv + hk], 1);
    return;
  }
  __shared__ int s_last;
  if (tid == 0) s_last = atom_add_acq_rel(&a.cnt[b * a.Hkv + hk], 1) == n_chunks_of(L, a.cs) - 1;
  __syncthreads();
  if (s_last) {
    for (int qi = warp; qi < Q; qi += kWarps) attn_merge_warp<DPL>(ap, sp, b, hk, qi, lane);
    __syncthreads();
    if (tid == 0) a.cnt[b * a.Hkv + hk] = 0;
  }
}

// Merge of (request b, kv head hk) by its designated CTA, after that CTA's
// own items: wait until every chunk is counted (bounded), merge the queries
// (one warp each), reset the count.
template <int DPL>
__device__ __noinline__ void attn_merge_cta(const AttnView* ap, const StepParams* sp, int b, int hk, int* status) {
  const AttnView& a = *ap;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int L = sp->req_len[b], nb = sp->req_tok0[b + 1] - sp->req_tok0[b];
  const int Q = nb * (a.Hq / a.Hkv);
  if (tid == 0) {
    uint32_t it = 0;
    while (ld_acquire_s32(&a.cnt[b * a.Hkv + hk]) < n_chunks_of(L, a.cs)) {
      if (++it > (1u << 22)) {
        atomicOr(status, ST_WAIT_TIMEOUT);
        break;
      }
      __nanosleep(64);
    }
  }
  __syncthreads();
  for (int qi = warp; qi < Q; qi += kWarps) attn_merge_warp<DPL>(ap, sp, b, hk, qi, lane);
  __syncthreads();
  if (tid == 0) a.cnt[b * a.Hkv + hk] = 0;
}

template <int NT, int GPU, int DPL>
__global__ void __launch_bounds__(kThreads, 1) step_kernel(const __grid_constant__ StepKernelArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ GemvPhase s_gp[4];            // per projection kind: q|k|v, o, gate|up, down
  __shared__ WarpStream<GPU> s_ws[kWarps];  // each warp's weight stream, between phases
  __shared__ AttnView s_av;
  using SS = StepSmem<GPU>;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* ring = smem + (size_t)warp * kRingSlots * Geom<GPU>::kUnitBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SS::kRing) + warp * kRingSlots;
  uint8_t* att_area = smem + SS::kRing + SS::kBars;
  static_assert(AttnSmem<DPL>::kBytes <= SS::kQ, "attention area too small");
  OpDesc* s_ops = reinterpret_cast<OpDesc*>(smem + SS::kFixed);
  for (int i = threadIdx.x; i < 4 * a.L; i += kThreads) s_ops[i] = a.ops[i];
  __syncthreads();
  unsigned long long target = a.barrier_base;
  int nsync = 1;
  if (threadIdx.x == 0 && blockIdx.x == 0) a.phase_clock[0] = globaltimer();
  {
    WarpStream<GPU> ws;
    ws.init(s_ops, 4 * a.L, blockIdx.x, gridDim.x, warp, kWarps, ring, bars, kRingSlots == 4 ? 2 : 1, lane);
    ws.fill(lane);
    if (lane == 0) s_ws[warp] = ws;
    __syncwarp();
  }

  if (blockIdx.x == 0) prologue_cta(a.pro);
  grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);

  const StepParams* sp = a.pro.sp;
  const bool skip = __ldcg(&sp->abort_step) != 0;
  const int M = a.pro.M;
  // Each CTA normalises the whole hidden state for itself; when the M rows
  // fit, it keeps them in the attention area (idle during the q|k|v and
  // gate|up projections) and the projections read them from there.  Rows are
  // padded by 32 halves so that the two token rows a fragment load touches in
  // one phase fall on different banks.
  const int xn_ld = a.H + 32;
  const bool xn_smem = kNormInSmem && a.Kp_H == a.H && (size_t)M * xn_ld * 2 <= SS::kQ;
  uint16_t* xn = xn_smem ? reinterpret_cast<uint16_t*>(att_area) : a.act_h;
  const int xn_out_ld = xn_smem ? xn_ld : a.Kp_H;
  if (threadIdx.x < 4) {
    const int k = threadIdx.x;
    GemvPhase gp{};
    gp.act = k == 0 || k == 2 ? a.act_h : k == 1 ? a.act_attn : a.act_f;
    gp.act_ld = k == 0 || k == 2 ? a.Kp_H : k == 1 ? a.Kp_dq : a.Kp_F;
    gp.M = M;
    gp.act_s = (k == 0 || k == 2) && xn_smem ? smem_addr(att_area) : 0u;
    gp.act_s_ld = xn_ld;
    gp.skip = skip;
    gp.partials = a.partials;
    gp.flags = a.flags;
    gp.status = a.status;
    gp.sp = sp;
    gp.ep.kind = k == 0 ? EPI_QKV : k == 2 ? EPI_SWIGLU : EPI_RESID;
    gp.ep.dims = OpDims{k, a.Hq, a.Hkv, a.d, a.F, a.H};
    gp.ep.q = a.q;
    gp.ep.kpool = a.kpool;
    gp.ep.vpool = a.vpool;
    gp.ep.layer_stride = a.layer_stride;
    gp.ep.cap = a.cap;
    gp.ep.rope = a.rope;
    gp.ep.x = a.x;
    gp.ep.ss = (k == 1 || k == 3) ? a.ss : nullptr;
    gp.ep.out_layer = k == 3 ? a.L - 1 : -1;
    gp.ep.h = a.act_f;
    gp.ep.h_ld = a.Kp_F;
    gp.done_flags = k == 0 ? a.rb_done : nullptr;
    s_gp[k] = gp;
  }
  if (threadIdx.x == 32) {
    AttnView av{};
    av.q = a.q;
    av.kpool = a.kpool;
    av.vpool = a.vpool;
    av.layer_stride = a.layer_stride;
    av.cap = a.cap;
    av.Hq = a.Hq;
    av.Hkv = a.Hkv;
    av.d = a.d;
    av.n_chunks = a.n_chunks;
    av.qmax = kMaxTokens * (a.Hq / a.Hkv);
    av.part = a.attn_part;
    av.cnt = a.attn_cnt;
    av.rb_done = a.rb_done;
    av.rb_k0 = a.Hq * a.d / kRowsPerBlock;
    av.rb_v0 = (a.Hq + a.Hkv) * a.d / kRowsPerBlock;
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
  __syncthreads();
  auto gemv = [&](int op, int l) { gemv_phase<NT, GPU>(&s_ws[warp], op, &s_gp[op & 3], l, a.epoch_base + op, lane); };

  for (int l = 0; l < a.L; ++l) {
    const uint16_t* nrm = a.norms + (size_t)l * 2 * a.H;
    // attention block
    if (!skip) rmsnorm_cta(a.x, a.H, nrm, a.eps, a.ss, xn, xn_out_ld, M);
    gemv(4 * l + 0, l);
    if (!skip) {
      if (xn_smem) __syncthreads();  // the attention items reuse the normalised rows' space
      int total = 0;
      for (int b = 0; b < sp->B; ++b) total += a.Hkv * n_chunks_of(sp->req_len[b], s_av.cs);
      for (int item = blockIdx.x; item < total; item += gridDim.x) {
        int b, hk, c;
        if (decode_item(sp, a.Hkv, s_av.cs, item, b, hk, c)) attn_item_cta<DPL>(&s_av, l, sp, b, hk, c, att_area, a.epoch_base + 4 * l, a.status);
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
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    gemv(4 * l + 1, l);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    // MLP block
    if (!skip) rmsnorm_cta(a.x, a.H, nrm + a.H, a.eps, a.ss, xn, xn_out_ld, M);
    gemv(4 * l + 2, l);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    gemv(4 * l + 3, l);
    if (l + 1 < a.L) grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
  }
  if (s_ws[warp].timed_out && lane == 0) atomicOr(a.status, ST_WAIT_TIMEOUT);
  // The last CTA to finish hands a nonzero status to the host-mapped mirror,
  // so no copy-engine transfer has to follow the step on the stream.
  __syncthreads();
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
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = StepSmem<GPU>::total(a.L);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int NT, int GPU, int DPL>
cudaError_t setup_t() {
  return cudaFuncSetAttribute(step_kernel<NT, GPU, DPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)StepSmem<GPU>::total(64));
}

}  // namespace

int step_barriers(int n_layers) { return 4 * n_layers; }

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
