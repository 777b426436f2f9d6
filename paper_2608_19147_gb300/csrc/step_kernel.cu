// The whole decode step of a shard as one persistent, cooperative kernel.
//
// One CTA per SM, kCtaWarps warps.  The step runs as a sequence of phases separated
// by grid-wide barriers:
//   prologue (CTA 0) | for each layer: RMSNorm | q|k|v projection (+RoPE,
//   K/V append) | attention partials | attention merge | o projection
//   (+residual) | RMSNorm | gate|up projection (+SwiGLU) | down projection
//   (+residual; the last layer writes hidden_out).
// Every warp owns a ring of weight slots (gemv_core.cuh) that streams, in
// order, all the projection units the warp will process during the step.
// The ring refills as soon as a slot is consumed, independent of the
// barriers, so while a warp waits at a barrier or works on norms and
// attention, the next projection's weights are already arriving.
//
// Barrier waits are bounded: a wait that runs out sets a status bit and
// proceeds (the step's results are then reported invalid) instead of hanging.
#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kWarps = kCtaWarps;
constexpr int kThreads = kWarps * 32;
constexpr int kQGroup = 8;        // queries staged per warp at a time
constexpr int kChunk = 32;        // cache entries per attention item (one per lane)

template <int GPU>
struct StepSmem {
  static constexpr size_t kRing = (size_t)kWarps * kRingSlots * Geom<GPU>::kUnitBytes;
  static constexpr size_t kBars = (size_t)kWarps * kRingSlots * sizeof(uint64_t);
  // attention query staging
  static constexpr size_t kQ = (size_t)kWarps * kQGroup * 128 * sizeof(float);  // d <= 128
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
  const size_t n = (size_t)a.M * a.H;
  for (size_t e = tid; e < n; e += nth) {
    const int m = static_cast<int>(e / a.H);
    const size_t k = e % a.H;
    const uint16_t h =
        a.hidden_in ? __ldcg(a.hidden_in + e) : a.embedding[(size_t)__ldcg(a.token_ids + m) * a.H + k];
    a.x[e] = h2f(h);
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
// RMSNorm: CTA m < M normalises token m (sum of squares in a fixed order).
// ---------------------------------------------------------------------------
__device__ __noinline__ void rmsnorm_cta(const float* x, int H, const uint16_t* w, float eps, uint16_t* out,
                                         int out_ld, int M) {
  __shared__ float s_part[kWarps];
  __shared__ float s_r;
  constexpr int kPer = 24;  // values per thread held in registers (H <= 24 * kThreads)
  for (int m = blockIdx.x; m < M; m += gridDim.x) {
    const float* xm = x + (size_t)m * H;
    float v[kPer];
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int k = threadIdx.x + i * kThreads;
      v[i] = k < H ? __ldcg(xm + k) : 0.f;
    }
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < kPer; ++i) ss = fmaf(v[i], v[i], ss);
    for (int k = threadIdx.x + kPer * kThreads; k < H; k += kThreads) {
      const float t = __ldcg(xm + k);
      ss = fmaf(t, t, ss);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x == 0) {
      float t = 0.f;
      for (int i = 0; i < kWarps; ++i) t += s_part[i];
      s_r = rsqrtf(t / H + eps);
    }
    __syncthreads();
    const float r = s_r;
    uint16_t* o = out + (size_t)m * out_ld;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int k = threadIdx.x + i * kThreads;
      if (k < H) o[k] = f2h(v[i] * r * h2f(w[k]));
    }
    for (int k = threadIdx.x + kPer * kThreads; k < H; k += kThreads) o[k] = f2h(__ldcg(xm + k) * r * h2f(w[k]));
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Attention.  Item = (request b, kv head hk, chunk c of kChunk entries); one
// warp per item.  Lane j scores entry j0 + j against every query of the item
// (the request's new tokens x the kv head's query heads), then lanes switch
// to owning head dims for the value sum.  Each item writes (max, sum of exp,
// unnormalised output) per query; the merge phase combines chunks in order.
// ---------------------------------------------------------------------------
struct AttnView {
  const float* q;
  const uint16_t* kpool;
  const uint16_t* vpool;
  int cap, Hq, Hkv, d, n_chunks, qmax;
  float* part;
  uint16_t* out;
  int out_ld;
};

__device__ __forceinline__ int n_chunks_of(int L) { return (L + kChunk - 1) / kChunk; }

// Finds the item's (b, hk, c) from a flat index; false if past the end.
__device__ __forceinline__ bool decode_item(const StepParams* sp, int Hkv, int item, int& b, int& hk, int& c) {
  for (b = 0; b < sp->B; ++b) {
    const int per = Hkv * n_chunks_of(sp->req_len[b]);
    if (item < per) {
      hk = item / n_chunks_of(sp->req_len[b]);
      c = item % n_chunks_of(sp->req_len[b]);
      return true;
    }
    item -= per;
  }
  return false;
}

template <int DPL>  // head dims per lane (d = 32 * DPL)
__device__ __noinline__ void attn_partial_warp(const AttnView& a, const StepParams* sp, int b, int hk, int c, float* qs,
                                               int lane) {
  constexpr int d = 32 * DPL;
  constexpr int KV8 = d / 8;  // 16-byte pieces per K row
  const int L = sp->req_len[b], P = sp->req_P[b];
  const int tok0 = sp->req_tok0[b], nb = sp->req_tok0[b + 1] - tok0;
  const int G = a.Hq / a.Hkv, Q = nb * G;
  const int j0 = c * kChunk, nj = min(kChunk, L - j0);
  const int jg = j0 + lane;
  const bool in_range = lane < nj;
  int slot = 0;
  bool visible_base = false;
  if (in_range) {
    slot = __ldcg(sp->bt + (size_t)b * a.cap + jg);
    visible_base = __ldcg(sp->mask + (size_t)b * sp->mask_stride + jg) != 0;
  }
  const size_t krow = (((size_t)(slot / a.cap) * a.Hkv + hk) * a.cap + slot % a.cap) * d;
  const float scale = rsqrtf(static_cast<float>(d));
  float* part = a.part + ((((size_t)b * a.Hkv + hk) * a.n_chunks + c) * a.qmax) * (d + 2);
  // this lane's K row, all pieces in flight at once
  uint4 kw[KV8];
  const uint4* kr = reinterpret_cast<const uint4*>(a.kpool + krow);
#pragma unroll
  for (int t = 0; t < KV8; ++t) kw[t] = in_range ? __ldcg(kr + t) : make_uint4(0, 0, 0, 0);
  for (int q0 = 0; q0 < Q; q0 += kQGroup) {
    const int qn = min(kQGroup, Q - q0);
    // stage this group's queries (fp32) in the warp's shared area
    __syncwarp();
    {
      float qv[kQGroup * DPL];
#pragma unroll
      for (int i = 0; i < kQGroup; ++i)
#pragma unroll
        for (int u = 0; u < DPL; ++u) {
          const int qi = q0 + i, t = u * 32 + lane;
          qv[i * DPL + u] = (i < qn) ? __ldcg(a.q + (size_t)(tok0 + qi / G) * a.Hq * d + (hk * G + qi % G) * d + t) : 0.f;
        }
#pragma unroll
      for (int i = 0; i < kQGroup; ++i)
#pragma unroll
        for (int u = 0; u < DPL; ++u) qs[i * d + u * 32 + lane] = qv[i * DPL + u];
    }
    __syncwarp();
    // scores: lane = entry
    float s[kQGroup];
#pragma unroll
    for (int i = 0; i < kQGroup; ++i) s[i] = 0.f;
#pragma unroll
    for (int t8 = 0; t8 < KV8; ++t8) {
      const uint32_t kk[4] = {kw[t8].x, kw[t8].y, kw[t8].z, kw[t8].w};
      float kf[8];
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        kf[2 * v] = h2f(static_cast<uint16_t>(kk[v] & 0xFFFFu));
        kf[2 * v + 1] = h2f(static_cast<uint16_t>(kk[v] >> 16));
      }
#pragma unroll
      for (int i = 0; i < kQGroup; ++i) {
        if (i < qn) {
          const float4 qa = *reinterpret_cast<const float4*>(qs + i * d + t8 * 8);
          const float4 qb = *reinterpret_cast<const float4*>(qs + i * d + t8 * 8 + 4);
          s[i] = fmaf(qa.x, kf[0], s[i]);
          s[i] = fmaf(qa.y, kf[1], s[i]);
          s[i] = fmaf(qa.z, kf[2], s[i]);
          s[i] = fmaf(qa.w, kf[3], s[i]);
          s[i] = fmaf(qb.x, kf[4], s[i]);
          s[i] = fmaf(qb.y, kf[5], s[i]);
          s[i] = fmaf(qb.z, kf[6], s[i]);
          s[i] = fmaf(qb.w, kf[7], s[i]);
        }
      }
    }
    // softmax pieces per query (entries across lanes)
    float p[kQGroup];
#pragma unroll
    for (int i = 0; i < kQGroup; ++i) {
      p[i] = 0.f;
      if (i >= qn) continue;
      const int qi = q0 + i;
      const bool vis = in_range && visible_base && jg <= P + qi / G;
      const float v = vis ? s[i] * scale : -INFINITY;
      float mx = v;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float e = vis ? expf(v - mx) : 0.f;
      float l = e;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
      p[i] = e;
      if (lane == 0) {
        part[(size_t)qi * (d + 2)] = mx;
        part[(size_t)qi * (d + 2) + 1] = l;
      }
    }
    // values: lane owns dims [DPL*lane, DPL*lane + DPL); rows in batches of 8,
    // the next batch in flight while one is summed
    float acc[kQGroup][DPL];
#pragma unroll
    for (int i = 0; i < kQGroup; ++i)
#pragma unroll
      for (int u = 0; u < DPL; ++u) acc[i][u] = 0.f;
    auto load_v = [&](int jb, uint32_t (&vw)[8][DPL / 2]) {
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int sj = __shfl_sync(0xffffffffu, slot, (jb + u) & 31);
        if (jb + u < nj) {
          const size_t vrow = (((size_t)(sj / a.cap) * a.Hkv + hk) * a.cap + sj % a.cap) * d;
          if constexpr (DPL == 4) {
            const uint2 t = __ldcg(reinterpret_cast<const uint2*>(a.vpool + vrow) + lane);
            vw[u][0] = t.x;
            vw[u][DPL / 2 - 1] = t.y;
          } else {
            vw[u][0] = __ldcg(reinterpret_cast<const uint32_t*>(a.vpool + vrow) + lane);
          }
        } else {
#pragma unroll
          for (int v = 0; v < DPL / 2; ++v) vw[u][v] = 0u;
        }
      }
    };
    uint32_t vbuf[2][8][DPL / 2];
    load_v(0, vbuf[0]);
#pragma unroll 1
    for (int jb = 0, cur = 0; jb < nj; jb += 8, cur ^= 1) {
      if (jb + 8 < nj) {
        if (cur == 0) load_v(jb + 8, vbuf[1]);
        else load_v(jb + 8, vbuf[0]);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        float vf[DPL];
#pragma unroll
        for (int v = 0; v < DPL / 2; ++v) {
          const uint32_t x = cur == 0 ? vbuf[0][u][v] : vbuf[1][u][v];
          vf[2 * v] = h2f(static_cast<uint16_t>(x & 0xFFFFu));
          vf[2 * v + 1] = h2f(static_cast<uint16_t>(x >> 16));
        }
#pragma unroll
        for (int i = 0; i < kQGroup; ++i) {
          const float pj = __shfl_sync(0xffffffffu, p[i], (jb + u) & 31);
#pragma unroll
          for (int v = 0; v < DPL; ++v) acc[i][v] = fmaf(pj, vf[v], acc[i][v]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < kQGroup; ++i) {
      if (i >= qn) continue;
      float* o = part + (size_t)(q0 + i) * (d + 2) + 2 + DPL * lane;
#pragma unroll
      for (int u = 0; u < DPL; ++u) o[u] = acc[i][u];
    }
  }
}

// Merge of one (request, kv head, query): chunks in order.  Lane c holds
// chunk c's max and sum; the outputs are summed with all loads in flight.
template <int DPL>
__device__ __noinline__ void attn_merge_warp(const AttnView& a, const StepParams* sp, int b, int hk, int qi, int lane) {
  constexpr int d = 32 * DPL;
  const int L = sp->req_len[b], tok0 = sp->req_tok0[b];
  const int G = a.Hq / a.Hkv;
  const int nc = n_chunks_of(L);
  const float* base = a.part + (((size_t)b * a.Hkv + hk) * a.n_chunks) * a.qmax * (d + 2) + (size_t)qi * (d + 2);
  const size_t cstride = (size_t)a.qmax * (d + 2);
  float M = -INFINITY;
  for (int c = lane; c < nc; c += 32) M = fmaxf(M, __ldcg(base + c * cstride));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float den = 0.f, num[DPL];
#pragma unroll
  for (int u = 0; u < DPL; ++u) num[u] = 0.f;
  for (int c0 = 0; c0 < nc; c0 += 32) {
    // lane c: weight of chunk c0 + c
    float wl = 0.f, ll = 0.f;
    if (c0 + lane < nc) {
      const float mc = __ldcg(base + (c0 + lane) * cstride);
      ll = __ldcg(base + (c0 + lane) * cstride + 1);
      wl = (mc == -INFINITY) ? 0.f : expf(mc - M);
    }
    float dl = ll * wl;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dl += __shfl_xor_sync(0xffffffffu, dl, o);
    den += dl;
    const int n = min(32, nc - c0);
    for (int cb = 0; cb < n; cb += 8) {
      float ov[8][DPL];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float* pc = base + (size_t)(c0 + cb + u) * cstride + 2 + DPL * lane;
#pragma unroll
        for (int v = 0; v < DPL; ++v) ov[u][v] = (cb + u < n) ? __ldcg(pc + v) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float w = __shfl_sync(0xffffffffu, wl, (cb + u) & 31);
#pragma unroll
        for (int v = 0; v < DPL; ++v) num[v] = fmaf(ov[u][v], w, num[v]);
      }
    }
  }
  uint16_t* out = a.out + (size_t)(tok0 + qi / G) * a.out_ld + (hk * G + qi % G) * d + DPL * lane;
#pragma unroll
  for (int u = 0; u < DPL; ++u) out[u] = f2h(num[u] / den);
}

template <int NT, int GPU, int DPL>
__global__ void __launch_bounds__(kThreads, 1) step_kernel(const StepKernelArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  using SS = StepSmem<GPU>;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kWarps + warp, NW = gridDim.x * kWarps;
  uint8_t* ring = smem + (size_t)warp * kRingSlots * Geom<GPU>::kUnitBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SS::kRing) + warp * kRingSlots;
  float* qs = reinterpret_cast<float*>(smem + SS::kRing + SS::kBars) + (size_t)warp * kQGroup * 128;
  OpDesc* s_ops = reinterpret_cast<OpDesc*>(smem + SS::kFixed);
  for (int i = threadIdx.x; i < 4 * a.L; i += kThreads) s_ops[i] = a.ops[i];
  __syncthreads();
  unsigned long long target = a.barrier_base;
  int nsync = 1;
  if (threadIdx.x == 0 && blockIdx.x == 0) a.phase_clock[0] = globaltimer();

  WarpStream<GPU> ws;
  ws.init(s_ops, 4 * a.L, blockIdx.x, gridDim.x, warp, ring, bars, lane);
  ws.fill(lane);

  if (blockIdx.x == 0) prologue_cta(a.pro);
  grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);

  const StepParams* sp = a.pro.sp;
  const bool skip = __ldcg(&sp->abort_step) != 0;
  const int M = a.pro.M;

  // Per-phase arguments are built where they are used (short live ranges).
  auto gemv = [&](int op, int epi, const uint16_t* act, int act_ld, int l) {
    GemvPhase gp{};
    gp.act = act;
    gp.act_ld = act_ld;
    gp.M = M;
    gp.skip = skip;
    gp.partials = a.partials;
    gp.counters = a.counters;
    gp.status = a.status;
    gp.sp = sp;
    gp.ep.kind = epi;
    gp.ep.dims = OpDims{op & 3, a.Hq, a.Hkv, a.d, a.F, a.H};
    gp.ep.q = a.q;
    gp.ep.kpool = a.kpool + (size_t)l * a.layer_stride;
    gp.ep.vpool = a.vpool + (size_t)l * a.layer_stride;
    gp.ep.cap = a.cap;
    gp.ep.rope = a.rope;
    gp.ep.x = a.x;
    gp.ep.write_out = (op == 4 * a.L - 1) ? 1 : 0;
    gp.ep.h = a.act_f;
    gp.ep.h_ld = a.Kp_F;
    gemv_phase<NT, GPU>(ws, op, gp, lane);
  };

  for (int l = 0; l < a.L; ++l) {
    const uint16_t* nrm = a.norms + (size_t)l * 2 * a.H;
    // attention block
    if (!skip) rmsnorm_cta(a.x, a.H, nrm, a.eps, a.act_h, a.Kp_H, M);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    gemv(4 * l + 0, EPI_QKV, a.act_h, a.Kp_H, l);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    if (!skip) {
      AttnView av{};
      av.q = a.q;
      av.kpool = a.kpool + (size_t)l * a.layer_stride;
      av.vpool = a.vpool + (size_t)l * a.layer_stride;
      av.cap = a.cap;
      av.Hq = a.Hq;
      av.Hkv = a.Hkv;
      av.d = a.d;
      av.n_chunks = a.n_chunks;
      av.qmax = kMaxTokens * (a.Hq / a.Hkv);
      av.part = a.attn_part;
      av.out = a.act_attn;
      av.out_ld = a.Kp_dq;
      int total = 0;
      for (int b = 0; b < sp->B; ++b) total += a.Hkv * n_chunks_of(sp->req_len[b]);
      for (int item = gw; item < total; item += NW) {
        int b, hk, c;
        if (decode_item(sp, a.Hkv, item, b, hk, c)) attn_partial_warp<DPL>(av, sp, b, hk, c, qs, lane);
      }
      grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
      // merge items: (b, hk, query)
      const int G = a.Hq / a.Hkv;
      total = 0;
      for (int b = 0; b < sp->B; ++b) total += a.Hkv * (sp->req_tok0[b + 1] - sp->req_tok0[b]) * G;
      for (int item = gw; item < total; item += NW) {
        int r = item, b = 0;
        for (; b < sp->B; ++b) {
          const int per = a.Hkv * (sp->req_tok0[b + 1] - sp->req_tok0[b]) * G;
          if (r < per) break;
          r -= per;
        }
        const int Qb = (sp->req_tok0[b + 1] - sp->req_tok0[b]) * G;
        attn_merge_warp<DPL>(av, sp, b, r / Qb, r % Qb, lane);
      }
    } else {
      grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    }
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    gemv(4 * l + 1, EPI_RESID, a.act_attn, a.Kp_dq, l);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    // MLP block
    if (!skip) rmsnorm_cta(a.x, a.H, nrm + a.H, a.eps, a.act_h, a.Kp_H, M);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    gemv(4 * l + 2, EPI_SWIGLU, a.act_h, a.Kp_H, l);
    grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
    gemv(4 * l + 3, EPI_RESID, a.act_f, a.Kp_F, l);
    if (l + 1 < a.L) grid_sync(a.barrier, target, a.status, a.phase_clock, nsync);
  }
  if (ws.timed_out && lane == 0) atomicOr(a.status, ST_WAIT_TIMEOUT);
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

int step_barriers(int n_layers) { return 8 * n_layers; }

size_t step_attention_part_floats(int B, int Hkv, int n_chunks, int G, int d) {
  return (size_t)B * Hkv * n_chunks * (kMaxTokens * G) * (d + 2);
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
