// Prefill: a prompt of S tokens through the stage in one call (Section 3.4:
// the stateful cache is filled by running the prompt through the shard).
// The arithmetic is the decode step's, for S new tokens of one request: the
// same rounding points (fp16 normalised activations, attention output,
// SwiGLU output, appended K/V and the output), causal attention among the new
// tokens and over the row's unmasked cache.  The projections are dense
// contractions here and run on the tensor cores (gemm_tc.cu), the attention on
// mma.sync over blocks of tokens (prefill_flash_kernel); the rest are small
// per-token kernels, launched layer by layer on the caller's stream.
#include "common.cuh"

namespace shard {
namespace {


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

// Causal attention of the new tokens on the tensor cores (mma.sync m16n8k16),
// one CTA per (block of 64 / G tokens, kv head hk), 4 warps: query row r of
// the 64 is token t0 + r / G, query head hk G + r % G, and warp w owns rows
// 16 w .. + 15, so every K/V tile is read once for all the block's queries.
// Entry tiles of 64 come through the beam table into shared memory.  Scores
// S = Q K^T with Q split into fp16 hi + lo parts (together ~22 bits of q, so
// the scores match an fp32 q); online softmax per row in fp32; O += P V with
// P split the same way; fp32 accumulators.  Entry j is visible to token t iff
// j <= P + t and mask[j] != 0.
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4_trans(const void* p, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(smem_addr(p)));
}
// fp16x2 of (lo, hi) and the fp16x2 of what each rounding left out
__device__ __forceinline__ void split_h2(float lo, float hi, uint32_t& h, uint32_t& l) {
  const uint16_t a = f2h(lo), b = f2h(hi);
  h = (uint32_t)a | ((uint32_t)b << 16);
  l = (uint32_t)f2h(lo - h2f(a)) | ((uint32_t)f2h(hi - h2f(b)) << 16);
}

template <int D, int G>
__global__ void __launch_bounds__(128) prefill_flash_kernel(const float* q, int Hq, int Hkv, const uint16_t* kpool,
                                                           const uint16_t* vpool, const int* bt_row, int cap,
                                                           const uint8_t* mask, int P, int S, uint16_t* out,
                                                           int out_ld) {
  constexpr int TB = 64 / G;  // tokens per CTA
  constexpr int KS = D / 16;  // k16 steps over the head dimension
  constexpr int ND = D / 8;   // n8 tiles over the head dimension
  constexpr int LD = D + 8;   // shared row stride (halves): 16-byte rows, conflict-free fragment reads
  __shared__ __align__(16) uint16_t Ks[64][LD];
  __shared__ __align__(16) uint16_t Vs[64][LD];
  __shared__ uint8_t vis[64];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, gid = lane >> 2, tig = lane & 3;
  const int t0 = blockIdx.x * TB, hk = blockIdx.y;
  const float scale = rsqrtf((float)D);
  // Q rows as fp16 hi (in Ks) and lo (in Vs), then this warp's fragments
  for (int e = tid; e < 64 * D; e += 128) {
    const int r = e / D, c = e % D, t = t0 + r / G;
    const float v = t < S ? q[(size_t)t * Hq * D + (hk * G + r % G) * D + c] : 0.f;
    const uint16_t hi = f2h(v);
    Ks[r][c] = hi;
    Vs[r][c] = f2h(v - h2f(hi));
  }
  __syncthreads();
  const int ra = 16 * warp + gid, rb = ra + 8;  // this thread's two query rows
  uint32_t qh[KS][4], ql[KS][4];
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) {
    const int c = 16 * ks + 2 * tig;
    qh[ks][0] = *reinterpret_cast<const uint32_t*>(&Ks[ra][c]);
    qh[ks][1] = *reinterpret_cast<const uint32_t*>(&Ks[rb][c]);
    qh[ks][2] = *reinterpret_cast<const uint32_t*>(&Ks[ra][c + 8]);
    qh[ks][3] = *reinterpret_cast<const uint32_t*>(&Ks[rb][c + 8]);
    ql[ks][0] = *reinterpret_cast<const uint32_t*>(&Vs[ra][c]);
    ql[ks][1] = *reinterpret_cast<const uint32_t*>(&Vs[rb][c]);
    ql[ks][2] = *reinterpret_cast<const uint32_t*>(&Vs[ra][c + 8]);
    ql[ks][3] = *reinterpret_cast<const uint32_t*>(&Vs[rb][c + 8]);
  }
  const int tok_a = t0 + ra / G, tok_b = t0 + rb / G;
  const int lim_a = P + tok_a, lim_b = P + tok_b;  // causal limits
  float o[ND][4];
#pragma unroll
  for (int nd = 0; nd < ND; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
  float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;
  const int last = P + min(t0 + TB, S) - 1;  // the block's last token's limit
  for (int j0 = 0; j0 <= last; j0 += 64) {
    const int nj = min(64, last + 1 - j0);
    __syncthreads();  // the previous tile (or the Q staging) is read
    for (int e = tid; e < 64 * (D / 8); e += 128) {
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
    if (tid < 64) vis[tid] = tid < nj && mask[j0 + tid] ? 1 : 0;
    __syncthreads();
    float sc[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks)
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        const uint32_t b0 = *reinterpret_cast<const uint32_t*>(&Ks[8 * nt + gid][16 * ks + 2 * tig]);
        const uint32_t b1 = *reinterpret_cast<const uint32_t*>(&Ks[8 * nt + gid][16 * ks + 8 + 2 * tig]);
        mma16816(sc[nt], qh[ks], b0, b1);
        mma16816(sc[nt], ql[ks], b0, b1);
      }
    // mask and scale; row maxima over the quad that shares a row
    float mx_a = -INFINITY, mx_b = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int col = 8 * nt + 2 * tig + c, j = j0 + col;
        sc[nt][c] = vis[col] && j <= lim_a ? sc[nt][c] * scale : -INFINITY;
        sc[nt][2 + c] = vis[col] && j <= lim_b ? sc[nt][2 + c] * scale : -INFINITY;
        mx_a = fmaxf(mx_a, sc[nt][c]);
        mx_b = fmaxf(mx_b, sc[nt][2 + c]);
      }
#pragma unroll
    for (int o_ = 1; o_ <= 2; o_ <<= 1) {
      mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, o_));
      mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, o_));
    }
    const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
    const float al_a = m_a == -INFINITY ? 0.f : expf(m_a - mn_a), al_b = m_b == -INFINITY ? 0.f : expf(m_b - mn_b);
    float su_a = 0.f, su_b = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        sc[nt][c] = sc[nt][c] == -INFINITY ? 0.f : expf(sc[nt][c] - mn_a);
        sc[nt][2 + c] = sc[nt][2 + c] == -INFINITY ? 0.f : expf(sc[nt][2 + c] - mn_b);
        su_a += sc[nt][c];
        su_b += sc[nt][2 + c];
      }
#pragma unroll
    for (int o_ = 1; o_ <= 2; o_ <<= 1) {
      su_a += __shfl_xor_sync(0xffffffffu, su_a, o_);
      su_b += __shfl_xor_sync(0xffffffffu, su_b, o_);
    }
    l_a = l_a * al_a + su_a;
    l_b = l_b * al_b + su_b;
    m_a = mn_a;
    m_b = mn_b;
#pragma unroll
    for (int nd = 0; nd < ND; ++nd) {
      o[nd][0] *= al_a;
      o[nd][1] *= al_a;
      o[nd][2] *= al_b;
      o[nd][3] *= al_b;
    }
    // O += P V: the score accumulators of n-tiles 2 kk, 2 kk + 1 are the A
    // fragment of entries 16 kk .. + 15
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t ph[4], pl[4];
      split_h2(sc[2 * kk][0], sc[2 * kk][1], ph[0], pl[0]);
      split_h2(sc[2 * kk][2], sc[2 * kk][3], ph[1], pl[1]);
      split_h2(sc[2 * kk + 1][0], sc[2 * kk + 1][1], ph[2], pl[2]);
      split_h2(sc[2 * kk + 1][2], sc[2 * kk + 1][3], ph[3], pl[3]);
      const int mtx = lane >> 3, er = 16 * kk + 8 * (mtx & 1) + (lane & 7);
#pragma unroll
      for (int nd = 0; nd < ND; nd += 2) {
        uint32_t v0, v1, v2, v3;
        ldsm_x4_trans(&Vs[er][8 * (nd + (mtx >> 1))], v0, v1, v2, v3);
        mma16816(o[nd], ph, v0, v1);
        mma16816(o[nd], pl, v0, v1);
        mma16816(o[nd + 1], ph, v2, v3);
        mma16816(o[nd + 1], pl, v2, v3);
      }
    }
  }
  const float ia = l_a > 0.f ? 1.f / l_a : 0.f, ib = l_b > 0.f ? 1.f / l_b : 0.f;
#pragma unroll
  for (int nd = 0; nd < ND; ++nd)
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const int dcol = 8 * nd + 2 * tig + c;
      if (tok_a < S) out[(size_t)tok_a * out_ld + (hk * G + ra % G) * D + dcol] = f2h(o[nd][c] * ia);
      if (tok_b < S) out[(size_t)tok_b * out_ld + (hk * G + rb % G) * D + dcol] = f2h(o[nd][2 + c] * ib);
    }
}

template <int D, int G>
cudaError_t launch_attn_t(const PrefillLayerArgs& a, cudaStream_t s) {
  static_assert(64 % G == 0, "64 query rows per CTA");
  prefill_flash_kernel<D, G><<<dim3((a.S + 64 / G - 1) / (64 / G), a.Hkv), 128, 0, s>>>(
      a.q, a.Hq, a.Hkv, a.kpool, a.vpool, a.bt_row, a.cap, a.mask, a.P, a.S, a.attn, a.attn_ld);
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
