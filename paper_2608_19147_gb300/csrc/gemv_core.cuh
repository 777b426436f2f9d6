// The W4A16 projection as warp-level device code, shared by the whole-step
// kernel and the standalone projection kernel.
//
// Work split.  The unit stream of a projection (n_rb row-blocks x upr units,
// see kernels.h) is cut into gridDim.x contiguous ranges, one per CTA, so
// every CTA streams the same number of bytes; inside a CTA, warp w takes
// every kCtaWarps-th unit of the range starting at w.  Each warp owns a ring
// of kRingSlots shared-memory slots that its lane 0 fills with bulk copies
// (TMA, non-tensor), one unit per slot, completion tracked by one mbarrier
// per slot.  Because the weights never depend on earlier work, a warp's ring
// runs ahead through the *sequence* of projections it will process (the
// step's q|k|v, o, gate|up, down of every layer): while the warp waits for
// other work, its next projection's weights are already in flight.
//
// Per unit, a lane turns each 32-bit code word into the four registers of its
// m16n8k16 A fragment -- (q - z) exactly, in fp16 -- and multiplies them with
// the activations (the B fragment) on the tensor cores, accumulating in fp32;
// the fp16 group scale multiplies the fp32 group sum.
//
// Reduction.  A CTA's range covers a few row-block segments.  At the end of
// each segment every warp leaves its partial sums in shared memory; the last
// warp to arrive (shared-memory counter) adds the kCtaWarps pieces in warp
// order.  A row-block wholly inside the CTA's range is then finished at once;
// the pieces of a row-block split between CTAs go to a scratch buffer and the
// last CTA to arrive (global counter) adds them in CTA order.  Both orders
// are fixed, so results are deterministic and do not depend on the token
// count M.
#pragma once
#include "common.cuh"

namespace shard {

constexpr int kRingSlots = 3;  // units in flight per warp
constexpr int kCtaWarps = 12;  // warps per CTA that run projections

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
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Start of part i of n of a stream of T units (T * n < 2^63).
__device__ __forceinline__ int part_start(int T, int i, int n) { return static_cast<int>((long long)T * i / n); }

__device__ __forceinline__ int atom_add_acq_rel(int* p, int v) {
  int old;
  asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// ---------------------------------------------------------------------------
// Per-warp weight stream over a table of ops (in shared memory).
// ---------------------------------------------------------------------------
template <int GPU>
struct WarpStream {
  static constexpr int UB = Geom<GPU>::kUnitBytes;
  const OpDesc* ops;  // shared memory
  int n_ops, cta, n_cta, warp;
  uint8_t* ring;      // [kRingSlots][UB]
  uint64_t* bars;     // [kRingSlots]
  // fill cursor: op index, next unit, end of the CTA's range, op's units
  int f_op, f_u, f_end;
  const uint8_t* f_units;
  uint32_t n_filled, n_used;
  bool timed_out;

  __device__ __forceinline__ void cta_range(int op, int& cb, int& ce) const {
    const int T = ops[op].n_rb * ops[op].upr;
    cb = part_start(T, cta, n_cta);
    ce = part_start(T, cta + 1, n_cta);
  }
  __device__ __forceinline__ void open_op(int op) {
    int cb, ce;
    cta_range(op, cb, ce);
    f_u = cb + warp;
    f_end = ce;
    f_units = ops[op].units;
  }
  // lane 0 initialises the slot barriers; the warp is synced after.
  __device__ void init(const OpDesc* ops_, int n_ops_, int cta_, int n_cta_, int warp_, uint8_t* ring_, uint64_t* bars_,
                       int lane) {
    ops = ops_;
    n_ops = n_ops_;
    cta = cta_;
    n_cta = n_cta_;
    warp = warp_;
    ring = ring_;
    bars = bars_;
    n_filled = n_used = 0;
    timed_out = false;
    f_op = 0;
    f_u = f_end = 0;
    f_units = nullptr;
    if (n_ops > 0) open_op(0);
    if (lane == 0) {
      for (int s = 0; s < kRingSlots; ++s) mbar_init(&bars[s], 1);
      mbar_fence_init();
    }
    __syncwarp();
  }
  // Issues bulk copies until the ring is full or the stream ends.
  __device__ __forceinline__ void fill(int lane) {
    while (n_filled - n_used < (uint32_t)kRingSlots) {
      while (f_u >= f_end) {
        if (++f_op >= n_ops) return;
        open_op(f_op);
      }
      const uint8_t* src = f_units + (size_t)f_u * UB;
      f_u += kCtaWarps;
      if (lane == 0) {
        const int slot = n_filled % kRingSlots;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(&bars[slot], UB);
        bulk_g2s(ring + (size_t)slot * UB, src, UB, &bars[slot]);
      }
      ++n_filled;
    }
  }
  __device__ __forceinline__ const uint8_t* acquire() {
    const int slot = n_used % kRingSlots;
    if (!timed_out && !mbar_wait(&bars[slot], (n_used / kRingSlots) & 1)) timed_out = true;
    return ring + (size_t)slot * UB;
  }
  __device__ __forceinline__ void release(int lane) {
    __syncwarp();
    ++n_used;
    fill(lane);
  }
};

// ---------------------------------------------------------------------------
// One unit (64 rows x 128 inputs) of one warp.
//
// Dequantisation of a code word w: (w & 0x000F000F) | 0x64006400 is the fp16
// pair (1024 + q_lo, 1024 + q_hi) of the nibbles at bits 0 and 16; subtracting
// (1024 + z) leaves q - z exactly.  The nibbles at bits 4 and 20 give
// 1024 + 16 q; one fma with 1/16 and -(64 + z) leaves q - z exactly.  Bits
// 8..15 / 24..31 are handled the same way after a shift by 8.
// ---------------------------------------------------------------------------
template <int NT, int GPU>
__device__ __forceinline__ void mma_unit(const uint8_t* __restrict__ U, const uint4 (&act)[NT][2][2],
                                         float (&tot)[4][NT][4], int lane) {
  constexpr int BPG = Geom<GPU>::kBlocksPerGroup;
  constexpr uint32_t kSixteenth = 0x2C002C00u;  // fp16x2 1/16
  const int gid = lane >> 2;
  float accg[4][NT][4];
  uint32_t zsub[4], zfma[4];
#pragma unroll
  for (int kc = 0; kc < 2; ++kc) {
    uint4 A[4];
#pragma unroll
    for (int rt = 0; rt < 4; ++rt) A[rt] = *reinterpret_cast<const uint4*>(U + (kc * 4 + rt) * 512 + lane * 16);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int blk = kc * 4 + j;
      const int gi = blk / BPG;
      const uint8_t* meta = U + kCodeBytes + gi * kMetaBytesPerGroup;
      if (blk % BPG == 0) {
        // group start: clear the group sums; zero points as fp16x2
        // (1024 + z_lo) and -(64 + z_hi)
#pragma unroll
        for (int rt = 0; rt < 4; ++rt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) accg[rt][nt][e] = 0.f;
        const uint2 zz = *reinterpret_cast<const uint2*>(meta + 128 + gid * 8);
#pragma unroll
        for (int rt = 0; rt < 4; ++rt) {
          const uint32_t zw = rt < 2 ? zz.x : zz.y;
          const uint32_t zlo = (zw >> (16 * (rt & 1))) & 0xFFu;
          const uint32_t zhi = (zw >> (16 * (rt & 1) + 8)) & 0xFFu;
          zsub[rt] = (0x6400u | zlo) * 0x00010001u;
          zfma[rt] = (0xD400u + 16u * zhi) * 0x00010001u;
        }
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
        const uint32_t a0 = hsub2_u32(lop3_and_or(w, 0x000F000Fu, 0x64006400u), zsub[rt]);
        const uint32_t a1 = hfma2_u32(lop3_and_or(w, 0x00F000F0u, 0x64006400u), kSixteenth, zfma[rt]);
        const uint32_t a2 = hsub2_u32(lop3_and_or(w2, 0x000F000Fu, 0x64006400u), zsub[rt]);
        const uint32_t a3 = hfma2_u32(lop3_and_or(w2, 0x00F000F0u, 0x64006400u), kSixteenth, zfma[rt]);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_16816(accg[rt][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
      }
      if (blk % BPG == BPG - 1) {
        const uint4 sc = *reinterpret_cast<const uint4*>(meta + gid * 16);
        const uint32_t scw[4] = {sc.x, sc.y, sc.z, sc.w};
#pragma unroll
        for (int rt = 0; rt < 4; ++rt) {
          const float slo = h2f(static_cast<uint16_t>(scw[rt] & 0xFFFFu));
          const float shi = h2f(static_cast<uint16_t>(scw[rt] >> 16));
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            tot[rt][nt][0] = fmaf(slo, accg[rt][nt][0], tot[rt][nt][0]);
            tot[rt][nt][1] = fmaf(slo, accg[rt][nt][1], tot[rt][nt][1]);
            tot[rt][nt][2] = fmaf(shi, accg[rt][nt][2], tot[rt][nt][2]);
            tot[rt][nt][3] = fmaf(shi, accg[rt][nt][3], tot[rt][nt][3]);
          }
        }
      }
    }
  }
}

__device__ __forceinline__ float silu(float v) { return v / (1.f + expf(-v)); }

// Epilogue of one (row R_lo, row R_lo + 8, token m) pair of a finished
// row-block: rotary pairs and gate/up pairs sit on these two rows.
__device__ __forceinline__ void epilogue_pair(const EpiArgs& e, const StepParams* sp, int Rlo, int m, float vlo,
                                              float vhi) {
  const OpDims& o = e.dims;
  const int Rhi = Rlo + 8;
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
        const int head = t / tph, i = 8 * (t % tph) + (Rlo & 7);
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
      const int j = 8 * (Rlo >> 4) + (Rlo & 7);
      if (j < o.F) e.h[(size_t)m * e.h_ld + j] = f2h(silu(vlo) * vhi);
      break;
    }
    default:
      break;
  }
}

struct GemvPhase {
  const uint16_t* act;  // fp16 [M][act_ld]
  int act_ld, M;
  bool skip;            // consume the weights but compute nothing (aborted step)
  float* partials;      // [gridDim.x][2][64][16] pieces of split row-blocks
  int* counters;        // [n_rb], zero, self-resetting
  float* red;           // shared: [kCtaWarps][64][16] warp pieces of one segment
  int* red_cnt;         // shared: arrivals at the current segment (0 at phase start)
  int* red_seg;         // shared: segment number the buffer is open for (0 at phase start)
  int* status;
  const StepParams* sp;
  EpiArgs ep;
};

// Loads the B fragments of unit (ku) for tokens gid (and gid + 8).
template <int NT>
__device__ __forceinline__ void load_act(uint4 (&act)[NT][2][2], const uint16_t* actp, int act_ld, int M, bool skip,
                                         int ku, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int n = nt * 8 + gid;
#pragma unroll
    for (int kc = 0; kc < 2; ++kc)
#pragma unroll
      for (int h = 0; h < 2; ++h)
        act[nt][kc][h] = (n < M && !skip) ? __ldcg(reinterpret_cast<const uint4*>(
                                                actp + (size_t)n * act_ld + ku * kUnitK + kc * 64 + h * 32 + tig * 8))
                                          : make_uint4(0, 0, 0, 0);
  }
}

// End of one row-block segment of a CTA (the cold path): called by every
// warp of the CTA after leaving its partial sums in shared memory.  The last
// warp to arrive sums the pieces and finishes the row-block, or hands its
// piece to the last CTA to arrive at the row-block.  Work items of the
// reducing warp are (row pair, token): item i takes rows
// lo = (i % 32 / 8) * 16 + i % 8 and lo + 8 for token i / 32.  The items of a
// lane (at most kMaxTokens / 2 ... kMaxTokens) are processed together so
// that their global loads are in flight at the same time.
static __device__ __noinline__ void segment_end(const GemvPhase& p, int segno, int rb, bool whole, int slot, int cta,
                                                int n_cta, int T, int rb_begin, int rb_end, int lane) {
  __syncwarp();
  int last = 0;
  if (lane == 0) {
    __threadfence_block();
    last = (atomicAdd(p.red_cnt, 1) == kCtaWarps - 1);
  }
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) return;
  __threadfence_block();
  const int lo = (lane >> 3) * 16 + (lane & 7);
  const int M = p.M;
  float vlo[kMaxTokens], vhi[kMaxTokens];
#pragma unroll
  for (int m = 0; m < kMaxTokens; ++m) {
    vlo[m] = vhi[m] = 0.f;
    if (m < M) {
#pragma unroll
      for (int w = 0; w < kCtaWarps; ++w) {
        vlo[m] += p.red[(size_t)w * 1024 + lo * 16 + m];
        vhi[m] += p.red[(size_t)w * 1024 + (lo + 8) * 16 + m];
      }
    }
  }
  // reopen the buffer for the next segment
  __syncwarp();
  if (lane == 0) {
    *reinterpret_cast<volatile int*>(p.red_cnt) = 0;
    __threadfence_block();
    *reinterpret_cast<volatile int*>(p.red_seg) = segno + 1;
  }
  if (whole) {
#pragma unroll
    for (int m = 0; m < kMaxTokens; ++m)
      if (m < M) epilogue_pair(p.ep, p.sp, rb * kRowsPerBlock + lo, m, vlo[m], vhi[m]);
    return;
  }
  float* mine_g = p.partials + ((size_t)cta * 2 + slot) * 1024;
#pragma unroll
  for (int m = 0; m < kMaxTokens; ++m)
    if (m < M) {
      mine_g[lo * 16 + m] = vlo[m];
      mine_g[(lo + 8) * 16 + m] = vhi[m];
    }
  __syncwarp();
  auto cta_of = [&](int uu) { return static_cast<int>(((long long)(uu + 1) * n_cta + T - 1) / T - 1); };
  const int c_first = cta_of(rb_begin), c_last = cta_of(rb_end - 1);
  const int expected = (T >= n_cta) ? (c_last - c_first + 1) : (rb_end - rb_begin);
  int glast = 0;
  if (lane == 0) glast = (atom_add_acq_rel(&p.counters[rb], 1) == expected - 1);
  glast = __shfl_sync(0xffffffffu, glast, 0);
  if (!glast) return;
#pragma unroll
  for (int m = 0; m < kMaxTokens; ++m) vlo[m] = vhi[m] = 0.f;
  for (int cc = c_first; cc <= c_last; ++cc) {
    const int s0 = part_start(T, cc, n_cta), s1 = part_start(T, cc + 1, n_cta);
    if (s1 <= s0) continue;  // empty range
    const float* pc = p.partials + ((size_t)cc * 2 + ((s0 < rb_begin) ? 1 : 0)) * 1024;
    float a[kMaxTokens], b[kMaxTokens];
#pragma unroll
    for (int m = 0; m < kMaxTokens; ++m) {
      a[m] = (m < M) ? __ldcg(pc + lo * 16 + m) : 0.f;
      b[m] = (m < M) ? __ldcg(pc + (lo + 8) * 16 + m) : 0.f;
    }
#pragma unroll
    for (int m = 0; m < kMaxTokens; ++m) {
      vlo[m] += a[m];
      vhi[m] += b[m];
    }
  }
#pragma unroll
  for (int m = 0; m < kMaxTokens; ++m)
    if (m < M) epilogue_pair(p.ep, p.sp, rb * kRowsPerBlock + lo, m, vlo[m], vhi[m]);
  if (lane == 0) p.counters[rb] = 0;
}

// One projection for one warp of a CTA: consume the warp's units from the
// stream (which must be positioned at this op), then take part in the
// reduction of every row-block segment of the CTA's range.
template <int NT, int GPU>
__device__ __forceinline__ void gemv_phase(WarpStream<GPU>& ws, int op, const GemvPhase& p, int lane) {
  int cb, ce;
  ws.cta_range(op, cb, ce);
  if (cb >= ce) return;
  const int upr = ws.ops[op].upr;
  const int T = ws.ops[op].n_rb * upr;
  const int gid = lane >> 2, tig = lane & 3;
  const uint16_t* actp = p.act;
  const int act_ld = p.act_ld, M = p.M;
  const bool skip = p.skip;
  int u = cb + ws.warp;  // this warp's next unit
  int rb = cb / upr;
  int ku = u - rb * upr;  // input unit of u within its row-block (may pass upr)
  while (ku >= upr) ku -= upr;
  uint4 nxt[NT][2][2];
  if (u < ce) load_act<NT>(nxt, actp, act_ld, M, skip, ku, lane);
  int segno = 0;
  for (int seg = cb; seg < ce; ++segno, ++rb) {
    const int rb_begin = rb * upr, rb_end = rb_begin + upr;
    const int seg_end = ce < rb_end ? ce : rb_end;
    float tot[4][NT][4];
#pragma unroll
    for (int rt = 0; rt < 4; ++rt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int q = 0; q < 4; ++q) tot[rt][nt][q] = 0.f;
    for (; u < seg_end; u += kCtaWarps) {
      uint4 cur[NT][2][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
          for (int h = 0; h < 2; ++h) cur[nt][kc][h] = nxt[nt][kc][h];
      ku += kCtaWarps;
      while (ku >= upr) ku -= upr;
      if (u + kCtaWarps < ce) load_act<NT>(nxt, actp, act_ld, M, skip, ku, lane);
      const uint8_t* U = ws.acquire();
      if (!skip && !ws.timed_out) mma_unit<NT, GPU>(U, cur, tot, lane);
      ws.release(lane);
    }
    if (!skip) {
      if (lane == 0) {
        uint32_t it = 0;
        while (*reinterpret_cast<volatile int*>(p.red_seg) != segno) {
          if (++it > (1u << 22)) {
            atomicOr(p.status, ST_WAIT_TIMEOUT);
            break;
          }
          __nanosleep(32);
        }
      }
      __syncwarp();
      float* mine = p.red + (size_t)ws.warp * 1024;
#pragma unroll
      for (int rt = 0; rt < 4; ++rt)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const int m = nt * 8 + 2 * tig + c;
            if (m < M) {
              mine[(rt * 16 + gid) * 16 + m] = tot[rt][nt][c];
              mine[(rt * 16 + gid + 8) * 16 + m] = tot[rt][nt][2 + c];
            }
          }
      const bool whole = (seg == rb_begin && seg_end == rb_end);
      const int slot = (cb < rb_begin) ? 1 : 0;
      segment_end(p, segno, rb, whole, slot, ws.cta, ws.n_cta, T, rb_begin, rb_end, lane);
    }
    seg = seg_end;
  }
}

}  // namespace shard
