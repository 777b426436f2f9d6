// Split-KV (flash-decoding) attention over the stateful KV pool.
//
// Grid (chunk, kv head, request).  A CTA takes `chunk` consecutive cache
// entries of its request's row and every query that reads its kv head: the
// request's n_b new tokens times the Hq / Hkv query heads of the group (GQA),
// so each K/V entry is fetched once for all of them.  Entries are located
// through the row's entry table (the beam table): entry j of row b lives at
// physical slot bt[b][j], which the beam_idx gather rearranges without moving
// K/V (Section 4).  Visibility of entry j for new token i of request b:
// j < P_b + n_b, attention_mask[b][j] != 0 (Section 5.2), and j <= P_b + i.
//
// Each CTA writes its chunk's (max, sum of exp, unnormalised output) per
// query; the last CTA of a (request, kv head) to finish -- counted with an
// atomic -- merges the chunks in chunk order (deterministic) and writes the
// fp16 attention output.
#include "common.cuh"

namespace shard {
namespace {

constexpr int kAttnThreads = 256;

struct AttnSmem {
  static size_t bytes(int qmax, int chunk, int d) {
    return sizeof(float) * ((size_t)qmax * d + (size_t)d * chunk + (size_t)chunk * d + (size_t)qmax * chunk) +
           sizeof(int) * chunk;
  }
};

__global__ void __launch_bounds__(kAttnThreads) attention_kernel(const AttnArgs a, int qmax, float scale) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int s_last;
  pdl_launch_dependents();
  pdl_wait();
  const StepParams* sp = a.sp;
  if (sp->abort_step) return;
  const int c = blockIdx.x, hk = blockIdx.y, b = blockIdx.z;
  if (b >= sp->B) return;
  const int L = sp->req_len[b], P = sp->req_P[b];
  const int tok0 = sp->req_tok0[b], nb = sp->req_tok0[b + 1] - tok0;
  const int j0 = c * a.chunk;
  if (j0 >= L) return;
  const int nj = min(a.chunk, L - j0);
  const int G = a.Hq / a.Hkv, Q = nb * G, d = a.d, C = a.chunk;
  const int tid = threadIdx.x;

  float* qs = sm;                     // [qmax][d]
  float* kT = qs + (size_t)qmax * d;  // [d][C]
  float* vs = kT + (size_t)d * C;     // [C][d]
  float* S = vs + (size_t)C * d;      // [qmax][C]
  int* slots = reinterpret_cast<int*>(S + (size_t)qmax * C);

  for (int j = tid; j < nj; j += kAttnThreads) slots[j] = __ldcg(sp->bt + (size_t)b * a.cap + j0 + j);
  for (int e = tid; e < Q * d; e += kAttnThreads) {
    const int qi = e / d, t = e % d;
    const int tok = tok0 + qi / G, head = hk * G + qi % G;
    qs[e] = __ldcg(a.q + (size_t)tok * a.Hq * d + head * d + t);
  }
  __syncthreads();
  // K (transposed) and V of the chunk, 8 fp16 per load.
  const int vec = d / 8;
  for (int e = tid; e < nj * vec; e += kAttnThreads) {
    const int j = e / vec, t8 = (e % vec) * 8;
    const int slot = slots[j];
    const size_t off = (((size_t)(slot / a.cap) * a.Hkv + hk) * a.cap + slot % a.cap) * d + t8;
    const uint4 kw = __ldcg(reinterpret_cast<const uint4*>(a.kpool + off));
    const uint4 vw = __ldcg(reinterpret_cast<const uint4*>(a.vpool + off));
    const uint32_t kk[4] = {kw.x, kw.y, kw.z, kw.w}, vv[4] = {vw.x, vw.y, vw.z, vw.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      kT[(size_t)(t8 + 2 * u) * C + j] = h2f(static_cast<uint16_t>(kk[u] & 0xFFFFu));
      kT[(size_t)(t8 + 2 * u + 1) * C + j] = h2f(static_cast<uint16_t>(kk[u] >> 16));
      vs[(size_t)j * d + t8 + 2 * u] = h2f(static_cast<uint16_t>(vv[u] & 0xFFFFu));
      vs[(size_t)j * d + t8 + 2 * u + 1] = h2f(static_cast<uint16_t>(vv[u] >> 16));
    }
  }
  __syncthreads();
  // Scores with visibility.
  const uint8_t* mask = sp->mask + (size_t)b * sp->mask_stride;
  for (int e = tid; e < Q * C; e += kAttnThreads) {
    const int qi = e / C, j = e % C;
    const int jg = j0 + j;
    float s = -INFINITY;
    if (j < nj && jg <= P + qi / G && __ldcg(mask + jg) != 0) {
      const float* qv = qs + (size_t)qi * d;
      float acc = 0.f;
      for (int t = 0; t < d; ++t) acc = fmaf(qv[t], kT[(size_t)t * C + j], acc);
      s = acc * scale;
    }
    S[e] = s;
  }
  __syncthreads();
  // Per-query max and exp (one warp per query).
  const int warp = tid >> 5, lane = tid & 31;
  float* part = a.part + ((((size_t)b * a.Hkv + hk) * a.n_chunks + c) * qmax) * (d + 2);
  for (int qi = warp; qi < Q; qi += kAttnThreads / 32) {
    float mx = -INFINITY;
    for (int j = lane; j < C; j += 32) mx = fmaxf(mx, S[qi * C + j]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float l = 0.f;
    for (int j = lane; j < C; j += 32) {
      const float s = S[qi * C + j];
      const float p = (s == -INFINITY) ? 0.f : expf(s - mx);
      S[qi * C + j] = p;
      l += p;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    if (lane == 0) {
      part[(size_t)qi * (d + 2)] = mx;
      part[(size_t)qi * (d + 2) + 1] = l;
    }
  }
  __syncthreads();
  for (int e = tid; e < Q * d; e += kAttnThreads) {
    const int qi = e / d, t = e % d;
    const float* p = S + (size_t)qi * C;
    float acc = 0.f;
    for (int j = 0; j < nj; ++j) acc = fmaf(p[j], vs[(size_t)j * d + t], acc);
    part[(size_t)qi * (d + 2) + 2 + t] = acc;
  }
  // Merge across chunks: the last CTA of this (request, kv head) does it.
  __threadfence();
  __syncthreads();
  const int n_chunks_b = (L + C - 1) / C;
  if (tid == 0) {
    const int old = atomicAdd(&a.counters[b * a.Hkv + hk], 1);
    s_last = (old == n_chunks_b - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const float* base = a.part + (((size_t)b * a.Hkv + hk) * a.n_chunks) * qmax * (d + 2);
  for (int e = tid; e < Q * d; e += kAttnThreads) {
    const int qi = e / d, t = e % d;
    float M = -INFINITY;
    for (int cc = 0; cc < n_chunks_b; ++cc) M = fmaxf(M, __ldcg(base + ((size_t)cc * qmax + qi) * (d + 2)));
    float den = 0.f, num = 0.f;
    for (int cc = 0; cc < n_chunks_b; ++cc) {
      const float* pc = base + ((size_t)cc * qmax + qi) * (d + 2);
      const float mc = __ldcg(pc);
      if (mc == -INFINITY) continue;
      const float w = expf(mc - M);
      den = fmaf(__ldcg(pc + 1), w, den);
      num = fmaf(__ldcg(pc + 2 + t), w, num);
    }
    const int tok = tok0 + qi / G, head = hk * G + qi % G;
    a.out[(size_t)tok * a.out_ld + head * d + t] = f2h(num / den);
  }
  if (tid == 0) a.counters[b * a.Hkv + hk] = 0;
}

}  // namespace

size_t attention_smem_bytes(int G, int chunk, int d) { return AttnSmem::bytes(kMaxTokens * G, chunk, d); }

cudaError_t attention_setup(size_t max_smem) {
  return cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)max_smem);
}

size_t attention_part_floats(int B, int Hkv, int n_chunks, int G, int d) {
  return (size_t)B * Hkv * n_chunks * (kMaxTokens * G) * (d + 2);
}

cudaError_t launch_attention(const AttnArgs& a, int B, cudaStream_t s, bool pdl) {
  const int G = a.Hq / a.Hkv;
  const int qmax = kMaxTokens * G;
  const size_t smem = AttnSmem::bytes(qmax, a.chunk, a.d);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_chunks, a.Hkv, B);
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const float scale = 1.0f / sqrtf(static_cast<float>(a.d));
  return cudaLaunchKernelEx(&cfg, attention_kernel, a, qmax, scale);
}

}  // namespace shard
