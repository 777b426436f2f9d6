// The W4A16 projection as warp-level device code, shared by the whole-step
// kernel and the standalone projection kernel.
//
// Work split.  The unit stream of a projection (n_rb row-blocks x upr units,
// see kernels.h) is cut into contiguous runs, one per warp of the grid
// (warp g = cta * warps per CTA + warp), so every warp streams the same number of
// bytes and keeps its sums in registers for as long as its run stays inside
// one row-block.  Each warp owns a ring of shared-memory slots (a power of two:
// kRingSlots in the step kernel, Geom::kGemvSlots in the standalone projection) that
// its lane 0 fills with bulk copies (TMA, non-tensor), one unit per slot,
// completion tracked by one mbarrier per slot.  Because the weights never
// depend on earlier work, a warp's ring runs ahead through the *sequence* of
// projections it will process (the step's q|k|v, o, gate|up, down of every
// layer): while the warp waits for other work, its next projection's weights
// are already in flight.
//
// Per unit, a lane turns each 32-bit code word into the four registers of its
// m16n8k16 A fragment -- (q - z) exactly, in fp16 -- and multiplies them with
// the activations (the B fragment) on the tensor cores, accumulating in fp32;
// the fp16 group scale multiplies the fp32 group sum.
//
// Reduction.  A row-block lying wholly inside one warp's run is finished by
// that warp.  A row-block split between warps gets one piece per warp; each
// contributor stores its piece and publishes it with a release-store of the
// launch's epoch into its flag, never waiting.  The warp that owns the
// row-block's last unit, after its own run, waits (acquire loads, all
// contributors polled at once, bounded) for the other flags, adds the pieces
// in warp order and runs the epilogue.  Waits only ever point to lower warp
// indices, so they cannot form a cycle; the fixed order makes results
// deterministic and independent of the token count M.
#pragma once
#include "common.cuh"

namespace shard {

constexpr int kRingSlots = 2;  // step kernel: units in flight per warp (measured: a third adds nothing)
static_assert(kRingSlots == 2 || kRingSlots == 4, "ring slots: a power of two the init call passes as a shift");
constexpr int kCtaWarps = 12;   // warps per CTA of the step kernel (all run projections)
constexpr int kGemvWarps = 12;  // warps per CTA of the standalone projection kernel

template <int GPU>
struct Geom {
  static constexpr int kUnitBytes = kCodeBytes + GPU * kMetaBytesPerGroup;
  static constexpr int kBlocksPerGroup = 8 / GPU;
  // the standalone projection (no attention area competes for shared
  // memory): four slots per warp where 12 warps' rings fit in 216 KB, else two
  static constexpr int kGemvSlots = kGemvWarps * 4 * kUnitBytes <= 216 * 1024 ? 4 : 2;
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
// bytes of (a, b) picked by the four selector nibbles of c (0..3: a, 4..7: b)
__device__ __forceinline__ uint32_t prmt_u32(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Start of part i of n of a stream of T units.  32-bit arithmetic: the host
// checks (T + 1) * n < 2^32 for every projection when a shard is created.
__device__ __forceinline__ int part_start(int T, int i, int n) {
  return static_cast<int>(static_cast<uint32_t>(T) * static_cast<uint32_t>(i) / static_cast<uint32_t>(n));
}
// The part owning unit x: the largest i with part_start(T, i, n) <= x.
__device__ __forceinline__ int part_of(int T, int x, int n) {
  return static_cast<int>((static_cast<uint32_t>(x + 1) * static_cast<uint32_t>(n) + static_cast<uint32_t>(T) - 1u) /
                          static_cast<uint32_t>(T)) - 1;
}

__device__ __forceinline__ int atom_add_acq_rel(int* p, int v) {
  int old;
  asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ void st_release_u32(unsigned* p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// ---------------------------------------------------------------------------
// Per-warp weight stream over a table of ops (in shared memory).
// ---------------------------------------------------------------------------
template <int GPU>
struct WarpStream {
  static constexpr int UB = Geom<GPU>::kUnitBytes;
  const OpDesc* ops;  // shared memory
  int n_ops, cta, n_cta, warp;
  int cta_warps;       // projection warps per CTA (the warp index space is cta * cta_warps + warp)
  uint8_t* ring;      // [slots][UB]
  uint64_t* bars;     // [slots]
  uint32_t slot_mask;  // slots - 1 (slots a power of two)
  int slot_shift;      // log2(slots)
  // fill cursor: op index, next unit, end of the CTA's range, op's units
  int f_op, f_u, f_end;
  const uint8_t* f_units;
  uint32_t n_filled, n_used;
  bool timed_out;

  // Run [wb, we) of this warp in op's unit stream.
  __device__ __forceinline__ void warp_range(int op, int& wb, int& we) const {
    const int T = ops[op].n_rb * ops[op].upr;
    const int g = cta * cta_warps + warp, nw = n_cta * cta_warps;
    wb = part_start(T, g, nw);
    we = part_start(T, g + 1, nw);
  }
  __device__ __forceinline__ void open_op(int op) {
    warp_range(op, f_u, f_end);
    f_units = ops[op].units;
  }
  // lane 0 initialises the slot barriers; the warp is synced after.
  __device__ void init(const OpDesc* ops_, int n_ops_, int cta_, int n_cta_, int warp_, int cta_warps_, uint8_t* ring_,
                       uint64_t* bars_, int slot_shift_, int lane) {
    ops = ops_;
    cta_warps = cta_warps_;
    slot_shift = slot_shift_;
    slot_mask = (1u << slot_shift_) - 1u;
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
      for (uint32_t s = 0; s <= slot_mask; ++s) mbar_init(&bars[s], 1);
      mbar_fence_init();
    }
    __syncwarp();
  }
  // Issues bulk copies until the ring is full or the stream ends.
  __device__ __forceinline__ void fill(int lane) {
    while (n_filled - n_used <= slot_mask) {
      while (f_u >= f_end) {
        if (++f_op >= n_ops) return;
        open_op(f_op);
      }
      const uint8_t* src = f_units + (size_t)f_u * UB;
      ++f_u;
      if (lane == 0) {
        const int slot = n_filled & slot_mask;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(&bars[slot], UB);
        // L2 evict-first: each weight byte is read once per step
        bulk_g2s_hint(ring + (size_t)slot * UB, src, UB, &bars[slot], l2_policy_evict_first());
      }
      ++n_filled;
    }
  }
  __device__ __forceinline__ const uint8_t* acquire() {
    const int slot = n_used & slot_mask;
    if (!timed_out && !mbar_wait(&bars[slot], (n_used >> slot_shift) & 1)) timed_out = true;
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
        // (1024 + z_lo) = bits 0x6400 | z and -(64 + z_hi) = bits 0xD400 | 16 z,
        // each one byte permute: the unit stores the upper rows' zero
        // points as 16 z
#pragma unroll
        for (int rt = 0; rt < 4; ++rt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) accg[rt][nt][e] = 0.f;
        const uint2 zz = *reinterpret_cast<const uint2*>(meta + 128 + gid * 8);
#pragma unroll
        for (int rt = 0; rt < 4; ++rt) {
          const uint32_t zw = rt < 2 ? zz.x : zz.y;  // bytes: z_lo, 16 z_hi of tiles 2i, then 2i + 1
          const uint32_t p = 2u * (rt & 1);
          zsub[rt] = prmt_u32(zw, 0x64646464u, 0x4040u + p * 0x0101u);
          zfma[rt] = prmt_u32(zw, 0xD4D4D4D4u, 0x4040u + (p + 1u) * 0x0101u);
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
// row-block: rotary pairs and gate/up pairs sit on these two rows.  Returns
// the sum of squares of the residual values written (EPI_RESID), else 0.
// xlo, xhi: the residual's current values at the two rows (EPI_RESID).
__device__ __forceinline__ float epilogue_pair(const EpiArgs& e, const StepParams* sp, int layer, int Rlo, int m,
                                               float vlo, float vhi, float xlo, float xhi) {
  float ss = 0.f;
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
          uint16_t* k = e.kpool + (size_t)layer * e.layer_stride + (((size_t)prow * o.Hkv + head) * e.cap + ppos) * o.d;
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
            e.vpool[(size_t)layer * e.layer_stride + (((size_t)prow * o.Hkv + head) * e.cap + ppos) * o.d + dim] =
                f2h(vv[u]);
          }
        }
      }
      break;
    }
    case EPI_RESID: {
      const int rr[2] = {Rlo, Rhi};
      const float vv[2] = {vlo, vhi}, xv[2] = {xlo, xhi};
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (rr[u] < o.H) {
          float* xp = e.x + (size_t)m * o.H + rr[u];
          const float nx = xv[u] + vv[u];
          *xp = nx;
          ss = fmaf(nx, nx, ss);
          if (e.out_layer == layer) sp->hidden_out[(size_t)m * o.H + rr[u]] = f2h(nx);
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
  return ss;
}

struct GemvPhase {
  const uint16_t* act;  // fp16 [M][act_ld]
  int act_ld, M;
  uint32_t act_s;       // 0, or the shared-memory address of this CTA's own copy of the activations,
  int act_s_ld;         // fp16 [M][act_s_ld], read instead of act
  bool skip;            // consume the weights but compute nothing (aborted step)
  float* partials;      // [n_cta * warps per CTA][2][kPieceFloats] pieces of split row-blocks
  unsigned* flags;      // [n_cta * warps per CTA][2] epoch of the piece last published in each slot
  int* status;
  const StepParams* sp;
  EpiArgs ep;
  unsigned* done_flags;  // nullptr, or row-block flags this projection publishes (release of the epoch
                         // after the row-block's epilogue)
};

// Floats of one stored piece: [token][64 rows] for up to kMaxTokens tokens.
constexpr int kPieceFloats = kMaxTokens * kRowsPerBlock;

// Loads the B fragments of input unit ku for tokens gid (and gid + 8).
template <int NT>
__device__ __forceinline__ void load_act(uint4 (&act)[NT][2][2], const uint16_t* actp, uint32_t acts, int act_ld,
                                         int M, bool skip, int ku, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int n = nt * 8 + gid;
#pragma unroll
    for (int kc = 0; kc < 2; ++kc)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int off = n * act_ld + ku * kUnitK + kc * 64 + h * 32 + tig * 8;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (n < M && !skip) {
          if (acts)
            asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                         : "r"(acts + 2u * (uint32_t)off));
          else
            v = __ldcg(reinterpret_cast<const uint4*>(actp + off));
        }
        act[nt][kc][h] = v;
      }
  }
}

// Finishes row-block rb from the stored pieces of warps g_first..g_last (the
// cold path), then runs the epilogue.  Lane L = rg + 8 * pg loads, as
// float4s, the four row pairs (R0 + i, R0 + 8 + i), R0 = 16 * (rg / 2) +
// 4 * (rg % 2), of the pieces g_first + pg, + pg + 4, ... and adds them in
// that order; two butterfly levels over pg then give every lane of the row
// group the same totals, and lane L finishes the pair R0 + pg (a rotary or
// gate/up pair).  The order is fixed, so the result is deterministic.
//
// Which slot holds a warp's piece: every contributor after the first started
// its run inside the row-block (slot 0); the first contributor used slot 1
// if its run started before the row-block.  When T < nw some runs are empty
// and each non-empty run is a single unit.
static __device__ __noinline__ void finish_rowblock(const GemvPhase* pp, int layer, int rb, int g_first, int g_last,
                                                    int T, int nw, int upr, int lane, unsigned epoch) {
  const GemvPhase& p = *pp;
  constexpr int kPerLane = 8;  // pieces per lane and batch (32 per batch over the 4 piece groups)
  const int rb_begin = rb * upr;
  const int rg = lane & 7, pg = lane >> 3;
  const int R0 = 16 * (rg >> 1) + 4 * (rg & 1);
  const int R = rb * kRowsPerBlock + R0 + pg;
  const bool dense = T >= nw;
  const size_t first_off = ((size_t)g_first * 2 + (part_start(T, g_first, nw) < rb_begin ? 1 : 0)) * kPieceFloats;
  for (int m = 0; m < p.M; ++m) {
    // the residual's current values, loaded with the pieces
    float xlo = 0.f, xhi = 0.f;
    if (p.ep.kind == EPI_RESID) {
      if (R < p.ep.dims.H) xlo = __ldcg(p.ep.x + (size_t)m * p.ep.dims.H + R);
      if (R + 8 < p.ep.dims.H) xhi = __ldcg(p.ep.x + (size_t)m * p.ep.dims.H + R + 8);
    }
    float4 slo = make_float4(0.f, 0.f, 0.f, 0.f), shi = slo;
    for (int g0 = g_first + pg; g0 <= g_last; g0 += 4 * kPerLane) {
      float4 a[kPerLane], b[kPerLane];
#pragma unroll
      for (int i = 0; i < kPerLane; ++i) {
        const int gg = g0 + 4 * i;
        a[i] = b[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        bool live = gg <= g_last;
        if (live && !dense) live = part_start(T, gg + 1, nw) > part_start(T, gg, nw);
        if (live) {
          const float* pc = p.partials + (gg == g_first ? first_off : (size_t)gg * 2 * kPieceFloats) + m * kRowsPerBlock;
          a[i] = __ldcg(reinterpret_cast<const float4*>(pc + R0));
          b[i] = __ldcg(reinterpret_cast<const float4*>(pc + R0 + 8));
        }
      }
#pragma unroll
      for (int i = 0; i < kPerLane; ++i) {
        slo.x += a[i].x; slo.y += a[i].y; slo.z += a[i].z; slo.w += a[i].w;
        shi.x += b[i].x; shi.y += b[i].y; shi.z += b[i].z; shi.w += b[i].w;
      }
    }
#pragma unroll
    for (int o = 8; o <= 16; o <<= 1) {
      slo.x += __shfl_xor_sync(0xffffffffu, slo.x, o);
      slo.y += __shfl_xor_sync(0xffffffffu, slo.y, o);
      slo.z += __shfl_xor_sync(0xffffffffu, slo.z, o);
      slo.w += __shfl_xor_sync(0xffffffffu, slo.w, o);
      shi.x += __shfl_xor_sync(0xffffffffu, shi.x, o);
      shi.y += __shfl_xor_sync(0xffffffffu, shi.y, o);
      shi.z += __shfl_xor_sync(0xffffffffu, shi.z, o);
      shi.w += __shfl_xor_sync(0xffffffffu, shi.w, o);
    }
    const float vlo = pg == 0 ? slo.x : pg == 1 ? slo.y : pg == 2 ? slo.z : slo.w;
    const float vhi = pg == 0 ? shi.x : pg == 1 ? shi.y : pg == 2 ? shi.z : shi.w;
    float ss = epilogue_pair(p.ep, p.sp, layer, R, m, vlo, vhi, xlo, xhi);
    if (p.ep.ss) {  // the row-block's sum of squares of the new residual, for the next RMSNorm
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
      if (lane == 0) p.ep.ss[rb * kMaxTokens + m] = ss;
    }
  }
  if (p.done_flags) {
    __syncwarp();
    if (lane == 0) st_release_u32(p.done_flags + rb, epoch);
  }
}

// Merge of split row-block rb by the warp owning its last unit: wait until
// every other contributor (g_first .. g_last - 1, non-empty runs) has
// published its piece for this epoch, then finish the row-block.
static __device__ __noinline__ void merge_rowblock(const GemvPhase* pp, int layer, int rb, int g_first, int g_last,
                                                   int T, int nw, int upr, unsigned epoch, int lane) {
  const GemvPhase& p = *pp;
  const int rb_begin = rb * upr;
  for (int g0 = g_first; g0 < g_last; g0 += 32) {
    const int gg = g0 + lane;
    if (gg < g_last) {
      const int s0 = part_start(T, gg, nw);
      if (part_start(T, gg + 1, nw) > s0) {  // non-empty run
        const unsigned* f = p.flags + (size_t)gg * 2 + (gg == g_first && s0 < rb_begin ? 1 : 0);
        uint32_t it = 0;
        while (ld_acquire_u32(f) != epoch) {
          if (++it > (1u << 22)) {
            atomicOr(p.status, ST_WAIT_TIMEOUT);
            break;
          }
          __nanosleep(32);
        }
      }
    }
  }
  __syncwarp();
  finish_rowblock(pp, layer, rb, g_first, g_last, T, nw, upr, lane, epoch);
}

// End of one row-block segment of a warp's run: store the piece (slot 0:
// the run's first segment, slot 1: a later one) and publish it.  A whole
// row-block is finished at once; a split one is merged by the owner of its
// last unit after that warp's run (gemv_phase) -- the owner itself (owner
// set) publishes nothing.
template <int NT>
__device__ __forceinline__ void piece_end(const GemvPhase* pp, int layer, const float (&tot)[4][NT][4], int rb, bool whole,
                                          bool owner, int slot, int g, int nw, int T, int upr, unsigned epoch,
                                          int lane) {
  const GemvPhase& p = *pp;
  const int gid = lane >> 2, tig = lane & 3;
  float* mine = p.partials + ((size_t)g * 2 + slot) * kPieceFloats;
#pragma unroll
  for (int rt = 0; rt < 4; ++rt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int m = nt * 8 + 2 * tig + c;
        if (m < p.M) {
          __stcg(mine + m * kRowsPerBlock + rt * 16 + gid, tot[rt][nt][c]);
          __stcg(mine + m * kRowsPerBlock + rt * 16 + gid + 8, tot[rt][nt][2 + c]);
        }
      }
  __syncwarp();
  if (whole) {
    finish_rowblock(pp, layer, rb, g, g, T, nw, upr, lane, epoch);
    return;
  }
  // The warp barrier above orders every lane's piece stores before lane 0's
  // release; the merging warp's acquire loads pair with it.
  if (!owner && lane == 0) st_release_u32(p.flags + (size_t)g * 2 + slot, epoch);
}

// One projection for one warp: consume the warp's run of units from the
// stream (which must be positioned at this op) and finish or hand on each
// row-block segment of it.
//
// Not inlined: the step's four projections run this one copy of the code, so
// it stays in the instruction cache.  The stream state and the phase
// arguments live in shared memory (ws_io, pp): nothing crosses the call
// through the stack, whose local memory would miss the small L1 left next to
// the weight rings.  The stream state is worked on in registers and written
// back at the end.
template <int NT, int GPU>
__device__ __noinline__ void gemv_phase(WarpStream<GPU>* ws_io, int op, const GemvPhase* pp, int layer, unsigned epoch,
                                        int lane) {
  WarpStream<GPU> ws = *ws_io;
  const GemvPhase& p = *pp;
  int wb, we;
  ws.warp_range(op, wb, we);
  if (wb >= we) return;
  const int upr = ws.ops[op].upr;
  const int T = ws.ops[op].n_rb * upr;
  const int g = ws.cta * ws.cta_warps + ws.warp, nw = ws.n_cta * ws.cta_warps;
  const uint16_t* actp = p.act;
  const uint32_t acts = p.act_s;
  const int act_ld = acts ? p.act_s_ld : p.act_ld, M = p.M;
  const bool skip = p.skip;
  int rb = wb / upr;
  int ku = wb - rb * upr;
  uint4 nxt[NT][2][2];
  load_act<NT>(nxt, actp, acts, act_ld, M, skip, ku, lane);
  for (int u = wb; u < we; ++rb) {
    const int seg_begin = u, rb_end = (rb + 1) * upr;
    const int seg_end = we < rb_end ? we : rb_end;
    float tot[4][NT][4];
#pragma unroll
    for (int rt = 0; rt < 4; ++rt)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int q = 0; q < 4; ++q) tot[rt][nt][q] = 0.f;
#pragma unroll 2  // alternating activation registers instead of copies (measured ~1 % faster)
    for (; u < seg_end; ++u) {
      uint4 cur[NT][2][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
          for (int h = 0; h < 2; ++h) cur[nt][kc][h] = nxt[nt][kc][h];
      if (++ku == upr) ku = 0;
      if (u + 1 < we) load_act<NT>(nxt, actp, acts, act_ld, M, skip, ku, lane);
      const uint8_t* U = ws.acquire();
      if (!skip && !ws.timed_out) mma_unit<NT, GPU>(U, cur, tot, lane);
      ws.release(lane);
    }
    if (!skip) {
      const bool whole = (seg_begin == rb * upr && seg_end == rb_end);
      piece_end<NT>(pp, layer, tot, rb, whole, seg_end == rb_end, seg_begin == wb ? 0 : 1, g, nw, T, upr, epoch,
                    lane);
    }
  }
  __syncwarp();
  if (lane == 0) *ws_io = ws;
  __syncwarp();
  if (!skip) {
    // merge the split row-blocks whose last unit is this warp's
    for (int r = wb / upr; r * upr + upr <= we; ++r) {
      if (r * upr >= wb) continue;  // whole inside the run: already finished
      merge_rowblock(pp, layer, r, part_of(T, r * upr, nw), g, T, nw, upr, epoch, lane);
    }
  }
}

}  // namespace shard
