// W4A16 skinny GEMM / GEMV for M = 1..16 tokens over the unit stream
// described in kernels.h.
//
// Work split: the unit stream of a projection (n_rb row-blocks x upr units)
// is cut into gridDim.x contiguous ranges, one per CTA (stream-K), so every
// CTA streams the same number of bytes.  Within a CTA one producer lane
// issues bulk copies (TMA, non-tensor) of kW consecutive units per stage into
// an S-stage shared-memory ring guarded by mbarriers; consumer warp w
// processes slot w of every stage.  A warp dequantises its lane's 16 bytes of
// codes per 16-row tile and 64 inputs into m16n8k16 A fragments in registers
// ((q - z) exact in fp16, see dequant below), multiplies them against the
// activations (the B fragments) on the tensor cores with fp32 accumulation,
// and applies the group scale in fp32 once per group.
//
// A CTA's range may start or end inside a row-block.  Row-blocks wholly
// inside one CTA are finished there; the head/tail pieces of split row-blocks
// go to a scratch buffer and the last contributing CTA to arrive (counted by
// an atomic per row-block) sums the pieces in CTA order -- the order is fixed,
// so results are deterministic and independent of the token count M.
//
// Epilogues: plain store (tests), RoPE + K/V append (q/k/v), residual add
// (o, down; optionally writing the fp16 step output), SwiGLU (gate/up).
#include <cstdio>
#include <mutex>

#include "common.cuh"

namespace shard {
namespace {

constexpr int kW = 8;                  // consumer warps per CTA
constexpr int kThreads = (kW + 1) * 32;
constexpr int kStages = 2;             // ring depth (x kW units per stage)
constexpr int kCtasPerSm = 2;

template <int GPU>
struct Geom {
  static constexpr int kUnitBytes = kCodeBytes + GPU * kMetaBytesPerGroup;
  static constexpr int kBlocksPerGroup = 8 / GPU;
};

__device__ __forceinline__ uint32_t hsub2_u32(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t hfma2_u32(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// One unit (64 rows x 128 inputs) for one warp.
//
// Dequantisation of a code word: (w & 0x000F000F) | 0x64006400 is the fp16
// pair (1024 + q_lo, 1024 + q_hi) of the nibbles at bits 0 and 16, and
// subtracting (1024 + z) leaves q - z exactly.  The nibbles at bits 4 and 20
// give 1024 + 16 q; one fma with 1/16 and -(64 + z) leaves q - z exactly.
// Bits 8..15 / 24..31 are handled the same after a shift by 8.  q - z lies in
// [-15, 15], exact in fp16, and its products with fp16 activations are exact
// on the tensor core; the group scale multiplies the fp32 group sum.
template <int NT, int GPU>
__device__ __forceinline__ void mma_unit(const uint8_t* __restrict__ U, const uint4 (&act)[NT][2][2],
                                         float (&tot)[4][NT][4], int lane) {
  constexpr int BPG = Geom<GPU>::kBlocksPerGroup;
  const int gid = lane >> 2;
  uint32_t zsub[GPU][4], zfma[GPU][4];
  float slo[GPU][4], shi[GPU][4];
#pragma unroll
  for (int gi = 0; gi < GPU; ++gi) {
    const uint8_t* meta = U + kCodeBytes + gi * kMetaBytesPerGroup;
    const uint4 sc = *reinterpret_cast<const uint4*>(meta + gid * 16);
    const uint2 zz = *reinterpret_cast<const uint2*>(meta + 128 + gid * 8);
    const uint32_t scw[4] = {sc.x, sc.y, sc.z, sc.w};
#pragma unroll
    for (int rt = 0; rt < 4; ++rt) {
      slo[gi][rt] = h2f(static_cast<uint16_t>(scw[rt] & 0xFFFFu));
      shi[gi][rt] = h2f(static_cast<uint16_t>(scw[rt] >> 16));
      const uint32_t zw = rt < 2 ? zz.x : zz.y;
      const uint32_t zlo = (zw >> (16 * (rt & 1))) & 0xFFu;
      const uint32_t zhi = (zw >> (16 * (rt & 1) + 8)) & 0xFFu;
      zsub[gi][rt] = (0x6400u | zlo) * 0x00010001u;          // fp16x2 (1024 + z_lo)
      zfma[gi][rt] = (0xD400u + 16u * zhi) * 0x00010001u;    // fp16x2 -(64 + z_hi)
    }
  }
  constexpr uint32_t kSixteenth = 0x2C002C00u;  // fp16x2 1/16
  float accg[4][NT][4];
#pragma unroll
  for (int kc = 0; kc < 2; ++kc) {
    uint4 A[4];
#pragma unroll
    for (int rt = 0; rt < 4; ++rt) A[rt] = *reinterpret_cast<const uint4*>(U + (kc * 4 + rt) * 512 + lane * 16);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int blk = kc * 4 + j;
      const int gi = blk / BPG;
      if (blk % BPG == 0) {
#pragma unroll
        for (int rt = 0; rt < 4; ++rt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) accg[rt][nt][e] = 0.f;
      }
      uint32_t b0[NT], b1[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const uint4 v = act[nt][kc][j >> 1];
        b0[nt] = (j & 1) ? v.z : v.x;
        b1[nt] = (j & 1) ? v.w : v.y;
      }
#pragma unroll
      for (int rt = 0; rt < 4; ++rt) {
        const uint32_t w = (j == 0) ? A[rt].x : (j == 1) ? A[rt].y : (j == 2) ? A[rt].z : A[rt].w;
        const uint32_t w2 = w >> 8;
        const uint32_t a0 = hsub2_u32(lop3_and_or(w, 0x000F000Fu, 0x64006400u), zsub[gi][rt]);
        const uint32_t a1 = hfma2_u32(lop3_and_or(w, 0x00F000F0u, 0x64006400u), kSixteenth, zfma[gi][rt]);
        const uint32_t a2 = hsub2_u32(lop3_and_or(w2, 0x000F000Fu, 0x64006400u), zsub[gi][rt]);
        const uint32_t a3 = hfma2_u32(lop3_and_or(w2, 0x00F000F0u, 0x64006400u), kSixteenth, zfma[gi][rt]);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_16816(accg[rt][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
      }
      if (blk % BPG == BPG - 1) {
#pragma unroll
        for (int rt = 0; rt < 4; ++rt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            tot[rt][nt][0] = fmaf(slo[gi][rt], accg[rt][nt][0], tot[rt][nt][0]);
            tot[rt][nt][1] = fmaf(slo[gi][rt], accg[rt][nt][1], tot[rt][nt][1]);
            tot[rt][nt][2] = fmaf(shi[gi][rt], accg[rt][nt][2], tot[rt][nt][2]);
            tot[rt][nt][3] = fmaf(shi[gi][rt], accg[rt][nt][3], tot[rt][nt][3]);
          }
      }
    }
  }
}

__device__ __forceinline__ float silu(float v) { return v / (1.f + expf(-v)); }

// Epilogue over one finished row-block: res[row][m] for 64 rows and M tokens.
// Work items pair row r and row r + 8 of each 16-row tile (rotary pairs and
// gate/up pairs live there).
__device__ void epilogue(const EpiArgs& e, const StepParams* sp, const float* res, int nc, int rb, int M, int tid,
                         int nthreads) {
  const OpDims& o = e.dims;
  for (int it = tid; it < 32 * M; it += nthreads) {
    const int m = it % M, pr = it / M;
    const int lo = (pr >> 3) * 16 + (pr & 7), hi = lo + 8;
    const float vlo = res[lo * nc + m], vhi = res[hi * nc + m];
    const int Rlo = rb * kRowsPerBlock + lo, Rhi = rb * kRowsPerBlock + hi;
    switch (e.kind) {
      case EPI_STORE: {
        const int n1 = natural_row(o, Rlo), n2 = natural_row(o, Rhi);
        if (n1 >= 0) e.y[(size_t)m * e.y_ld + n1] = vlo;
        if (n2 >= 0) e.y[(size_t)m * e.y_ld + n2] = vhi;
        break;
      }
      case EPI_QKV: {
        const int tph = o.d >> 4, nq = o.Hq * tph, nk = o.Hkv * tph, half = o.d >> 1;
        const int T = Rlo >> 4;
        const int slot = sp->tok_slot[m];
        const int prow = slot / e.cap, ppos = slot % e.cap;
        if (T < nq + nk) {
          const int t = T < nq ? T : T - nq;
          const int head = t / tph, i = 8 * (t % tph) + (pr & 7);
          const float2 cs = e.rope[(size_t)sp->tok_pos[m] * half + i];
          const float olo = vlo * cs.x - vhi * cs.y;
          const float ohi = vhi * cs.x + vlo * cs.y;
          if (T < nq) {
            float* q = e.q + (size_t)m * o.Hq * o.d + head * o.d;
            q[i] = olo;
            q[half + i] = ohi;
          } else {
            uint16_t* k = e.kpool + (((size_t)prow * o.Hkv + head) * e.cap + ppos) * o.d;
            k[i] = f2h(olo);
            k[half + i] = f2h(ohi);
          }
        } else {
          const int base = (o.Hq + o.Hkv) * o.d;
          const int rv[2] = {Rlo - base, Rhi - base};
          const float vv[2] = {vlo, vhi};
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            if (rv[u] < o.Hkv * o.d) {
              const int head = rv[u] / o.d, dim = rv[u] % o.d;
              e.vpool[(((size_t)prow * o.Hkv + head) * e.cap + ppos) * o.d + dim] = f2h(vv[u]);
            }
          }
        }
        break;
      }
      case EPI_RESID: {
        const int rr[2] = {Rlo, Rhi};
        const float vv[2] = {vlo, vhi};
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          if (rr[u] < o.H) {
            float* xp = e.x + (size_t)m * o.H + rr[u];
            const float nx = __ldcg(xp) + vv[u];
            *xp = nx;
            if (e.write_out) sp->hidden_out[(size_t)m * o.H + rr[u]] = f2h(nx);
          }
        }
        break;
      }
      case EPI_SWIGLU: {
        const int j = 8 * (Rlo >> 4) + (pr & 7);
        if (j < o.F) e.h[(size_t)m * e.h_ld + j] = f2h(silu(vlo) * vhi);
        break;
      }
      default:
        break;
    }
  }
}

template <int NT, int GPU, int S>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) gemv_kernel(const GemvArgs a) {
  constexpr int UB = Geom<GPU>::kUnitBytes;
  constexpr int STAGE = kW * UB;
  constexpr int NC = 8 * NT;
  constexpr int NCONS = kW * 32;
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* stages = smem;
  float* red = reinterpret_cast<float*>(smem + S * STAGE);  // [kW][64][NC]
  float* res = red + kW * 64 * NC;                          // [64][NC]
  __shared__ __align__(8) uint64_t full_bar[S], empty_bar[S];
  __shared__ int s_last;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long T = (long long)a.n_rb * a.upr;
  const int G = gridDim.x, c = blockIdx.x;
  const long long u0 = T * c / G, u1 = T * (c + 1) / G;
  const int n_units = static_cast<int>(u1 - u0);
  const int n_stages = (n_units + kW - 1) / kW;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kW);
    }
    mbar_fence_init();
  }
  __syncthreads();
  pdl_launch_dependents();

  if (warp == kW) {
    // Producer: weights never depend on earlier kernels, so streaming starts
    // before the dependency wait.
    if (lane == 0) {
      for (int t = 0; t < n_stages; ++t) {
        const int s = t % S;
        if (t >= S && !mbar_wait(&empty_bar[s], ((t / S) & 1) ^ 1)) {
          atomicOr(a.status, ST_WAIT_TIMEOUT);
          break;
        }
        const int nu = min(kW, n_units - t * kW);
        const uint32_t bytes = static_cast<uint32_t>(nu * UB);
        mbar_arrive_expect_tx(&full_bar[s], bytes);
        bulk_g2s(stages + s * STAGE, a.units + (size_t)(u0 + (long long)t * kW) * UB, bytes, &full_bar[s]);
      }
    }
    return;
  }

  // Consumers.
  pdl_wait();
  const StepParams* sp = a.sp;
  const int M = sp ? sp->M : a.M;
  const bool skip = sp ? (sp->abort_step != 0) : false;
  const int gid = lane >> 2, tig = lane & 3;
  const int ctid = threadIdx.x;
  bool timed_out = false;

  auto start_of = [&](int cc) -> long long { return T * cc / G; };
  auto cta_of = [&](long long u) -> int { return static_cast<int>(((u + 1) * G + T - 1) / T - 1); };

  long long seg_begin = u0;
  while (seg_begin < u1) {
    const int rb = static_cast<int>(seg_begin / a.upr);
    const long long rb_begin = (long long)rb * a.upr, rb_end = rb_begin + a.upr;
    const long long seg_end = u1 < rb_end ? u1 : rb_end;
    float tot[4][NT][4];
#pragma unroll
    for (int rt = 0; rt < 4; ++rt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) tot[rt][nt][e] = 0.f;

    const int i_lo = static_cast<int>(seg_begin - u0), i_hi = static_cast<int>(seg_end - u0);
    for (int i = i_lo + ((warp - i_lo % kW) + kW) % kW; i < i_hi; i += kW) {
      const int t = i / kW, s = t % S;
      const int ku = static_cast<int>(u0 + i - rb_begin);
      uint4 act[NT][2][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int n = nt * 8 + gid;
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (n < M && !skip)
              act[nt][kc][h] = __ldcg(reinterpret_cast<const uint4*>(
                  a.act + (size_t)n * a.act_ld + ku * kUnitK + kc * 64 + h * 32 + tig * 8));
            else
              act[nt][kc][h] = make_uint4(0, 0, 0, 0);
          }
      }
      if (!timed_out && !mbar_wait(&full_bar[s], (t / S) & 1)) timed_out = true;
      if (!timed_out && !skip) mma_unit<NT, GPU>(stages + s * STAGE + warp * UB, act, tot, lane);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[s]);
    }

    if (skip) {
      seg_begin = seg_end;
      continue;
    }
    // Per-warp partial sums -> shared memory.
    float* rw = red + warp * 64 * NC;
#pragma unroll
    for (int rt = 0; rt < 4; ++rt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const int r0 = rt * 16 + gid, col = nt * 8 + 2 * tig;
        rw[r0 * NC + col] = tot[rt][nt][0];
        rw[r0 * NC + col + 1] = tot[rt][nt][1];
        rw[(r0 + 8) * NC + col] = tot[rt][nt][2];
        rw[(r0 + 8) * NC + col + 1] = tot[rt][nt][3];
      }
    named_bar_sync(1, NCONS);
    const bool whole = (seg_begin == rb_begin && seg_end == rb_end);
    const int slot = (u0 < rb_begin) ? 1 : 0;
    for (int e = ctid; e < 64 * M; e += NCONS) {
      const int row = e / M, m = e % M;
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < kW; ++w) v += red[w * 64 * NC + row * NC + m];
      if (whole)
        res[row * NC + m] = v;
      else
        a.partials[((size_t)c * 2 + slot) * 1024 + row * 16 + m] = v;
    }
    if (!whole) {
      __threadfence();
      named_bar_sync(1, NCONS);
      const int c_first = cta_of(rb_begin), c_last = cta_of(rb_end - 1);
      if (ctid == 0) {
        const int old = atomicAdd(&a.counters[rb], 1);
        s_last = (old == c_last - c_first);
      }
      named_bar_sync(1, NCONS);
      if (!s_last) {
        seg_begin = seg_end;
        continue;
      }
      __threadfence();
      for (int e = ctid; e < 64 * M; e += NCONS) {
        const int row = e / M, m = e % M;
        float v = 0.f;
        for (int cc = c_first; cc <= c_last; ++cc) {
          const int sl = (start_of(cc) < rb_begin) ? 1 : 0;
          v += __ldcg(&a.partials[((size_t)cc * 2 + sl) * 1024 + row * 16 + m]);
        }
        res[row * NC + m] = v;
      }
      if (ctid == 0) a.counters[rb] = 0;
    }
    named_bar_sync(1, NCONS);
    epilogue(a.ep, sp, res, NC, rb, M, ctid, NCONS);
    named_bar_sync(1, NCONS);
    seg_begin = seg_end;
  }
  if (timed_out) atomicOr(a.status, ST_WAIT_TIMEOUT);
}

template <int NT, int GPU, int S>
constexpr size_t smem_bytes() {
  return (size_t)S * kW * Geom<GPU>::kUnitBytes + (size_t)(kW + 1) * 64 * 8 * NT * sizeof(float);
}

template <int NT, int GPU, int S>
cudaError_t launch_t(const GemvArgs& a, int grid, cudaStream_t s, bool pdl) {
  constexpr size_t smem = smem_bytes<NT, GPU, S>();
  auto kern = gemv_kernel<NT, GPU, S>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int NT, int GPU, int S>
cudaError_t setup_t() {
  return cudaFuncSetAttribute(gemv_kernel<NT, GPU, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)smem_bytes<NT, GPU, S>());
}

}  // namespace

cudaError_t gemv_setup() {
  cudaError_t e;
  if ((e = setup_t<1, 1, kStages>()) != cudaSuccess) return e;
  if ((e = setup_t<1, 2, kStages>()) != cudaSuccess) return e;
  if ((e = setup_t<1, 4, kStages>()) != cudaSuccess) return e;
  if ((e = setup_t<2, 1, kStages>()) != cudaSuccess) return e;
  if ((e = setup_t<2, 2, kStages>()) != cudaSuccess) return e;
  return setup_t<2, 4, kStages>();
}

int gemv_grid(int nt, int num_sms) {
  (void)nt;
  return kCtasPerSm * num_sms;
}

size_t gemv_partials_floats(int grid) { return (size_t)grid * 2 * 1024; }

cudaError_t launch_gemv(const GemvArgs& a, int nt, int group, int grid, cudaStream_t s, bool pdl) {
  if (nt == 1) {
    if (group == 128) return launch_t<1, 1, kStages>(a, grid, s, pdl);
    if (group == 64) return launch_t<1, 2, kStages>(a, grid, s, pdl);
    if (group == 32) return launch_t<1, 4, kStages>(a, grid, s, pdl);
  } else if (nt == 2) {
    if (group == 128) return launch_t<2, 1, kStages>(a, grid, s, pdl);
    if (group == 64) return launch_t<2, 2, kStages>(a, grid, s, pdl);
    if (group == 32) return launch_t<2, 4, kStages>(a, grid, s, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace shard
