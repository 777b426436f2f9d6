// Prefill: a prompt of S tokens through the stage in one call (Section 3.4:
// the stateful cache is filled by running the prompt through the shard).
// The arithmetic is the decode step's, for S new tokens of one request: the
// same rounding points (fp16 normalised activations, attention output,
// SwiGLU output, appended K/V and the output), causal attention among the new
// tokens and over the row's unmasked cache.  The projections are dense
// contractions here and run on the tensor cores (gemm_tc.cu); the rest are
// small per-token kernels, launched layer by layer on the caller's stream.
#include "common.cuh"

namespace shard {
namespace {

__device__ __forceinline__ float2 h2f2p(uint32_t u) {
  __half2 h;
  memcpy(&h, &u, sizeof(h));
  return __half22float2(h);
}

// Device-side argument checks (values that live on the device): token ids in
// [0, vocab), positions in [0, max_position), the mask open at every new
// entry.  A violation sets a status bit; the host then reports the call as
// rejected and the caller must reset the row.
__global__ void prefill_check_kernel(const int* token_ids, int vocab, const int* pos, int max_position,
                                     const uint8_t* mask, int P, int S, int* status) {
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < S; t += gridDim.x * blockDim.x) {
    int bits = 0;
    if (token_ids) {
      const int tok = token_ids[t];
      if (tok < 0 || tok >= vocab) bits |= ST_TOKEN;
    }
    const int p = pos[t];
    if (p < 0 || p >= max_position) bits |= ST_POSITION;
    if (mask[P + t] == 0) bits |= ST_MASK_NEW;
    if (bits) atomicOr(status, bits);
  }
}

__global__ void set_int_kernel(int* p, int v) { *p = v; }

// x[t][k] = fp32 of the step's fp16 input rows (hidden_in, or embedding rows).
__global__ void prefill_embed_kernel(const uint16_t* hidden_in, const int* token_ids, const uint16_t* embedding,
                                     int H, int S, int vocab, float* x) {
  const size_t n = (size_t)S * H;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const int t = (int)(e / H), k = (int)(e % H);
    int tok = 0;
    if (!hidden_in) {
      tok = __ldg(token_ids + t);
      tok = tok < 0 || tok >= vocab ? 0 : tok;  // out-of-range ids were flagged by the check; read a valid row
    }
    const uint16_t v = hidden_in ? hidden_in[e] : embedding[(size_t)tok * H + k];
    x[e] = h2f(v);
  }
}

// act[t][k] = fp16(x[t][k] * r[t] * w[k]), r = 1 / sqrt(mean(x[t]^2) + eps);
// one CTA per token.
__global__ void prefill_norm_kernel(const float* x, int H, const uint16_t* w, float eps, uint16_t* act, int act_ld) {
  __shared__ float s_part[32];
  const int t = blockIdx.x;
  const float* xr = x + (size_t)t * H;
  float ss = 0.f;
  for (int k = threadIdx.x; k < H; k += blockDim.x) ss = fmaf(xr[k], xr[k], ss);
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x == 0) {
    float tsum = 0.f;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) tsum += s_part[i];
    s_part[0] = rsqrtf(tsum / H + eps);
  }
  __syncthreads();
  const float r = s_part[0];
  for (int k = threadIdx.x; k < H; k += blockDim.x) act[(size_t)t * act_ld + k] = f2h(xr[k] * r * h2f(w[k]));
}

// RoPE (pairs (i, i + d/2), the token's position) on q (kept in fp32) and k;
// k and v rounded to fp16 and appended to the pool at the row's next slots.
__global__ void prefill_rope_append_kernel(const float* y, int y_ld, int S, int Hq, int Hkv, int d,
                                           const int* pos, int max_position, const float2* rope, float* q, uint16_t* kpool,
                                           uint16_t* vpool, int row, int cap, int slot0) {
  const int half = d / 2;
  const int per_tok = (Hq + Hkv) * half + Hkv * d;
  const size_t n = (size_t)S * per_tok;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const int t = (int)(e / per_tok), r = (int)(e % per_tok);
    const float* yr = y + (size_t)t * y_ld;
    const size_t kv = (((size_t)row * Hkv) * cap + (size_t)(slot0 + t)) * d;  // head 0's entry of this token
    if (r < (Hq + Hkv) * half) {
      const int h = r / half, i = r % half;
      const int p = __ldg(pos + t);
      const float2 cs = rope[(size_t)(p < 0 || p >= max_position ? 0 : p) * half + i];  // out-of-range positions were flagged
      const float lo = yr[h * d + i], hi = yr[h * d + half + i];
      const float olo = lo * cs.x - hi * cs.y, ohi = hi * cs.x + lo * cs.y;
      if (h < Hq) {
        q[(size_t)t * Hq * d + h * d + i] = olo;
        q[(size_t)t * Hq * d + h * d + half + i] = ohi;
      } else {
        uint16_t* kp = kpool + kv + (size_t)(h - Hq) * cap * d;
        kp[i] = f2h(olo);
        kp[half + i] = f2h(ohi);
      }
    } else {
      const int rv = r - (Hq + Hkv) * half, h = rv / d, i = rv % d;
      vpool[kv + (size_t)h * cap * d + i] = f2h(yr[(Hq + Hkv) * d + h * d + i]);
    }
  }
}

// Causal attention of the new tokens: CTA (token t, kv head hk), d threads
// (thread = head dimension).  Entries j <= P + t of the row with mask[j] != 0,
// read through the beam table; key tiles of 64 with an online softmax per
// query head.
constexpr int kPfTile = 64;
template <int D, int G>
__global__ void __launch_bounds__(D) prefill_attention_kernel(const float* q, int Hq, int Hkv, const uint16_t* kpool,
                                                              const uint16_t* vpool, const int* bt_row, int cap,
                                                              const uint8_t* mask, int P, uint16_t* out, int out_ld) {
  __shared__ float qs[G][D];
  __shared__ uint16_t Ks[kPfTile][D + 8];
  __shared__ uint16_t Vs[kPfTile][D];
  __shared__ float sc[G][kPfTile];
  __shared__ float s_m[G], s_l[G], s_alpha[G];
  const int t = blockIdx.x, hk = blockIdx.y, tid = threadIdx.x, warp = tid / 32, lane = tid % 32;
  const int n_warps = D / 32;
  for (int g = 0; g < G; ++g) qs[g][tid] = q[(size_t)t * Hq * D + (hk * G + g) * D + tid];
  if (tid < G) {
    s_m[tid] = -INFINITY;
    s_l[tid] = 0.f;
  }
  float acc[G];
#pragma unroll
  for (int g = 0; g < G; ++g) acc[g] = 0.f;
  const int last = P + t;  // causal limit
  const float scale = rsqrtf((float)D);
  for (int j0 = 0; j0 <= last; j0 += kPfTile) {
    const int nj = min(kPfTile, last + 1 - j0);
    __syncthreads();
    for (int e = tid; e < kPfTile * (D / 8); e += D) {
      const int r = e / (D / 8), c = e % (D / 8);
      uint4 kv4 = make_uint4(0, 0, 0, 0), vv4 = kv4;
      if (r < nj) {
        const int sl = __ldg(bt_row + j0 + r);
        const size_t off = (((size_t)(sl / cap) * Hkv + hk) * cap + sl % cap) * D;
        kv4 = *reinterpret_cast<const uint4*>(kpool + off + 8 * c);
        vv4 = *reinterpret_cast<const uint4*>(vpool + off + 8 * c);
      }
      *reinterpret_cast<uint4*>(&Ks[r][8 * c]) = kv4;
      *reinterpret_cast<uint4*>(&Vs[r][8 * c]) = vv4;
    }
    __syncthreads();
    for (int e = tid; e < G * kPfTile; e += D) {
      const int g = e / kPfTile, r = e % kPfTile;
      float s = -INFINITY;
      if (r < nj && mask[j0 + r]) {
        float dot = 0.f;
        for (int c = 0; c < D; c += 2) {
          const float2 kf = h2f2p(*reinterpret_cast<const uint32_t*>(&Ks[r][c]));
          dot = fmaf(qs[g][c], kf.x, dot);
          dot = fmaf(qs[g][c + 1], kf.y, dot);
        }
        s = dot * scale;
      }
      sc[g][r] = s;
    }
    __syncthreads();
    for (int g = warp; g < G; g += n_warps) {
      float mx = fmaxf(sc[g][lane], sc[g][lane + 32]);
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float m_new = fmaxf(s_m[g], mx);
      float p0 = 0.f, p1 = 0.f;
      if (m_new != -INFINITY) {
        p0 = sc[g][lane] == -INFINITY ? 0.f : expf(sc[g][lane] - m_new);
        p1 = sc[g][lane + 32] == -INFINITY ? 0.f : expf(sc[g][lane + 32] - m_new);
      }
      sc[g][lane] = p0;
      sc[g][lane + 32] = p1;
      float ps = p0 + p1;
      for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
      if (lane == 0) {
        const float alpha = s_m[g] == -INFINITY ? 0.f : expf(s_m[g] - m_new);
        s_alpha[g] = alpha;
        s_l[g] = s_l[g] * alpha + ps;
        s_m[g] = m_new;
      }
    }
    __syncthreads();
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float a = acc[g] * s_alpha[g];
      for (int r = 0; r < nj; ++r) a = fmaf(sc[g][r], h2f(Vs[r][tid]), a);
      acc[g] = a;
    }
  }
#pragma unroll
  for (int g = 0; g < G; ++g) out[(size_t)t * out_ld + (hk * G + g) * D + tid] = f2h(acc[g] / s_l[g]);
}

// h[t][j] = fp16(silu(gate) * up); y holds gate (0..F) then up (F..2F).
__global__ void prefill_swiglu_kernel(const float* y, int y_ld, int S, int F, uint16_t* h, int h_ld) {
  const size_t n = (size_t)S * F;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const int t = (int)(e / F), j = (int)(e % F);
    const float g = y[(size_t)t * y_ld + j], u = y[(size_t)t * y_ld + F + j];
    h[(size_t)t * h_ld + j] = f2h(g / (1.f + expf(-g)) * u);
  }
}

// x += y (the residual stream); on the last layer also hidden_out = fp16(x).
__global__ void prefill_residual_kernel(float* x, const float* y, int y_ld, int S, int H, uint16_t* out) {
  const size_t n = (size_t)S * H;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const int t = (int)(e / H), k = (int)(e % H);
    const float v = x[e] + y[(size_t)t * y_ld + k];
    x[e] = v;
    if (out) out[e] = f2h(v);
  }
}

template <int D, int G>
cudaError_t launch_attn_t(const PrefillLayerArgs& a, cudaStream_t s) {
  prefill_attention_kernel<D, G><<<dim3(a.S, a.Hkv), D, 0, s>>>(a.q, a.Hq, a.Hkv, a.kpool, a.vpool, a.bt_row, a.cap,
                                                                 a.mask, a.P, a.attn, a.attn_ld);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefill_check(const int* token_ids, int vocab, const int* pos, int max_position, const uint8_t* mask,
                                 int P, int S, int* status, cudaStream_t s) {
  prefill_check_kernel<<<(S + 255) / 256, 256, 0, s>>>(token_ids, vocab, pos, max_position, mask, P, S, status);
  return cudaGetLastError();
}

cudaError_t launch_set_int(int* p, int v, cudaStream_t s) {
  set_int_kernel<<<1, 1, 0, s>>>(p, v);
  return cudaGetLastError();
}

cudaError_t launch_prefill_embed(const uint16_t* hidden_in, const int* token_ids, const uint16_t* embedding, int H,
                                 int S, int vocab, float* x, cudaStream_t s) {
  prefill_embed_kernel<<<(int)std::min<size_t>(((size_t)S * H + 255) / 256, 4096), 256, 0, s>>>(hidden_in, token_ids,
                                                                                                embedding, H, S, vocab, x);
  return cudaGetLastError();
}

cudaError_t launch_prefill_norm(const float* x, int H, const uint16_t* w, float eps, uint16_t* act, int act_ld, int S,
                                cudaStream_t s) {
  prefill_norm_kernel<<<S, 256, 0, s>>>(x, H, w, eps, act, act_ld);
  return cudaGetLastError();
}

cudaError_t launch_prefill_rope_append(const PrefillLayerArgs& a, cudaStream_t s) {
  const size_t n = (size_t)a.S * ((a.Hq + a.Hkv) * (a.d / 2) + a.Hkv * a.d);
  prefill_rope_append_kernel<<<(int)std::min<size_t>((n + 255) / 256, 8192), 256, 0, s>>>(
      a.y, a.y_ld, a.S, a.Hq, a.Hkv, a.d, a.pos, a.max_position, a.rope, a.q, a.kpool, a.vpool, a.row, a.cap,
      a.slot0);
  return cudaGetLastError();
}

cudaError_t launch_prefill_attention(const PrefillLayerArgs& a, cudaStream_t s) {
  const int G = a.Hq / a.Hkv;
#define A(D)                                              \
  switch (G) {                                            \
    case 1: return launch_attn_t<D, 1>(a, s);             \
    case 2: return launch_attn_t<D, 2>(a, s);             \
    case 4: return launch_attn_t<D, 4>(a, s);             \
    case 8: return launch_attn_t<D, 8>(a, s);             \
    case 16: return launch_attn_t<D, 16>(a, s);           \
    default: return cudaErrorInvalidValue;                \
  }
  if (a.d == 128) { A(128) }
  if (a.d == 64) { A(64) }
#undef A
  return cudaErrorInvalidValue;
}

cudaError_t launch_prefill_swiglu(const float* y, int y_ld, int S, int F, uint16_t* h, int h_ld, cudaStream_t s) {
  prefill_swiglu_kernel<<<(int)std::min<size_t>(((size_t)S * F + 255) / 256, 8192), 256, 0, s>>>(y, y_ld, S, F, h,
                                                                                                 h_ld);
  return cudaGetLastError();
}

cudaError_t launch_prefill_residual(float* x, const float* y, int y_ld, int S, int H, uint16_t* out, cudaStream_t s) {
  prefill_residual_kernel<<<(int)std::min<size_t>(((size_t)S * H + 255) / 256, 4096), 256, 0, s>>>(x, y, y_ld, S, H,
                                                                                                   out);
  return cudaGetLastError();
}

}  // namespace shard
