// The W4A16 projection as warp-level device code, shared by the whole-step
// kernel and the standalone projection kernel.
//
// Work split.  The unit stream of a projection (n_rb row-blocks x upr units,
// see kernels.h) is cut into contiguous runs, one per consumer warp of the
// grid (warp g = cta * warps per CTA + warp), so every warp streams the same
// number of bytes and keeps its sums in registers for as long as its run
// stays inside one row-block.
//
// Weight streaming.  Every consumer warp owns a ring of shared-memory slots,
// filled with one bulk copy (TMA, non-tensor) per unit, completion signalled
// on the slot's "full" mbarrier.  The warp's stream is its run of every
// projection of the launch, in order; because the weights never depend on
// earlier work, the rings run ahead across projections: while consumers wait
// at a barrier or work on norms and attention, their next projection's first
// units are already arriving.  The slot a warp has consumed is refilled
// either by the warp's own lane 0 at once (kSelfRefill) or by a producer warp
// that watches the slots' "empty" mbarriers.
//
// Per unit, a lane turns each 32-bit code word into the four registers of its
// m16n8k16 A fragment with one AND per register (the codes as fp16
// subnormals) and multiplies them with the activations (the B fragment) on
// the tensor cores, accumulating in fp32; per group, the zero point is
// applied through the activations' group sum and the fp16 scale multiplies
// the result (mma_unit).
//
// Reduction.  At the end of each row-block segment of its run, a warp adds
// its fp32 sums, converted to 64-bit fixed point, to the projection's
// accumulator with integer atomics (kernels.h: EpiArgs).  Nothing waits:
// the residual projections add straight into the residual stream; q|k|v
// contributors count finished units per kv head for the attention items; for
// gate|up (and the standalone store) the contributor whose unit count
// completes a row-block finishes it.  Integer sums make every result
// independent of arrival order.
#pragma once
#include "common.cuh"

namespace shard {

// Weight streaming: with kSelfRefill, each consumer warp's lane 0 refills the
// slot the warp has just consumed with its next unit; otherwise a producer
// warp per CTA fills every consumer's ring.  Consumer warps per CTA: 12
// (3 per SM sub-partition), or 11 beside the producer (the sub-partition's
// register file caps 4 warps at 128 registers each).
constexpr bool kSelfRefill = true;
constexpr int kRingSlots = 2;  // step kernel: units in flight per consumer warp (a deeper ring takes the L1 that the norm and attention loads use)
constexpr int kCtaWarps = kSelfRefill ? 12 : 11;   // consumer warps per CTA of the step kernel
constexpr int kGemvWarps = kSelfRefill ? 12 : 11;  // consumer warps per CTA of the standalone projection kernel

template <int GPU>
struct Geom {
  static constexpr int kUnitBytes = kCodeBytes + GPU * kMetaBytesPerGroup;
  static constexpr int kBlocksPerGroup = 8 / GPU;
  // the step kernel's slots (group 32 units are larger: two)
  static constexpr int kStepSlots = GPU == 4 ? 2 : kRingSlots;
  // the standalone projection (no attention area competes for shared
  // memory): four slots per warp where the rings fit in 216 KB, else two
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

// Start of part i of n of a stream of T units.  32-bit arithmetic: the host
// checks (T + 1) * n < 2^32 for every projection when a shard is created.
__device__ __forceinline__ int part_start(int T, int i, int n) {
  return static_cast<int>(static_cast<uint32_t>(T) * static_cast<uint32_t>(i) / static_cast<uint32_t>(n));
}

__device__ __forceinline__ int atom_add_acq_rel(int* p, int v) {
  int old;
  asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ void red_release_add_s32(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_s32(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_add_s64(long long* p, long long v) {
  asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
// round(t) as a 64-bit integer, exact (ties to even) for |t| < 2^52, without
// the 64-bit conversion instructions (a slow path on this GPU).  Split
// t = h 2^31 + r with h = rint(t 2^-31), taken from the bits of a float sum
// with 1.5 2^23 (exact while |t 2^-31| < 2^22); r = t - h 2^31 is exact in
// fp32: for |t| < 2^30, h = 0 and r = t; otherwise t is a multiple of 2^7
// and |r| <= 2^30, so r has at most 23 significant bits.  One 32-bit
// conversion rounds r.
__device__ __forceinline__ long long f2fix(float t) {
  constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23
  const float y = __fadd_rn(t * 4.656612873077393e-10f, kMagic);  // rint(t 2^-31) + 1.5 2^23
  const int h = __float_as_int(y) - __float_as_int(kMagic);
  const float r = fmaf(__fsub_rn(y, kMagic), -2147483648.0f, t);
  return (static_cast<long long>(h) << 31) + static_cast<long long>(__float2int_rn(r));
}
__device__ __forceinline__ long long to_fixed(float v) { return f2fix(v * kFixOne); }
// value = v * 2^-32 with v = hi * 2^32 + lo (lo unsigned): hi + lo * 2^-32
// in fp32 from two 32-bit conversions (int64 conversions are a slow path).
// hi is exact (|hi| < 2^24); the result is within one fp32 ulp of the exact
// value and the same in every CTA.
__device__ __forceinline__ float fixed_to_f32(long long v) {
  const int hi = static_cast<int>(v >> 32);
  const unsigned lo = static_cast<unsigned>(v & 0xFFFFFFFFll);
  return fmaf(__uint2float_rn(lo), 2.3283064365386963e-10f, static_cast<float>(hi));
}

// ---------------------------------------------------------------------------
// Weight rings.
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Units [b, e) of warp g's run of op (OpDesc::q).  q > 0: row-block rb
// belongs to CTA rb / (kCtaWarps / q); its warps (rb % (kCtaWarps / q)) q + i,
// i < q, take K ranges i of ceil(upr / q) units.
__device__ __forceinline__ void run_range(const OpDesc& op, int g, int nw, int& b, int& e) {
  if (op.q == 0) {
    const int T = op.n_rb * op.upr;
    b = part_start(T, g, nw);
    e = part_start(T, g + 1, nw);
    return;
  }
  const int cta = g / kCtaWarps, w = g - cta * kCtaWarps;
  const int rb = cta * (kCtaWarps / op.q) + w / op.q, i = w % op.q;
  const int R = (op.upr + op.q - 1) / op.q;
  const int k0 = min(i * R, op.upr), k1 = min(k0 + R, op.upr);
  b = e = 0;
  if (rb < op.n_rb) {
    b = rb * op.upr + k0;
    e = rb * op.upr + k1;
  }
}

// One warp's view of the weight stream: the warp's run of every projection
// of the launch, in order (ops[0 .. n_ops)).
struct StreamCursor {
  const OpDesc* ops;
  int n_ops, g, nw;
  int op, u, end;
  const uint8_t* src;

  __device__ __forceinline__ void open(int o, int UB) {
    run_range(ops[o], g, nw, u, end);
    src = ops[o].units + (size_t)u * UB;
  }
  __device__ __forceinline__ void init(const OpDesc* ops_, int n_ops_, int g_, int nw_, int UB) {
    ops = ops_;
    n_ops = n_ops_;
    g = g_;
    nw = nw_;
    op = 0;
    u = end = 0;
    src = nullptr;
    if (n_ops > 0) open(0, UB);
  }
  // The next unit's address, or false at the end of the stream.
  __device__ __forceinline__ bool next(const uint8_t*& unit, int UB) {
    while (u >= end) {
      if (++op >= n_ops) return false;
      open(op, UB);
    }
    unit = src;
    src += UB;
    ++u;
    return true;
  }
};

// Consumer side of one warp's ring of S slots.
template <int GPU, int S>
struct WarpRing {
  static constexpr int UB = Geom<GPU>::kUnitBytes;
  uint8_t* ring;       // [S][UB]
  uint64_t* full;      // [S]
  uint64_t* empty;     // [S] (producer mode)
  uint32_t n_used;
  bool timed_out;
  StreamCursor cur;    // self-refill mode: lane 0's copy drives the refills
  uint64_t policy;

  __device__ __forceinline__ void issue(uint32_t slot, const uint8_t* src) {
    mbar_arrive_expect_tx(&full[slot], UB);
    // L2 evict-first: each weight byte is read once per launch
    bulk_g2s_hint(ring + (size_t)slot * UB, src, UB, &full[slot], policy);
  }
  // Self-refill mode: lane 0 fills the first S slots.
  __device__ __forceinline__ void start(const OpDesc* ops, int n_ops, int g, int nw, int lane) {
    cur.init(ops, n_ops, g, nw, UB);
    policy = l2_policy_evict_first();
    if (lane == 0)
      for (uint32_t s = 0; s < (uint32_t)S; ++s) {
        const uint8_t* src;
        if (!cur.next(src, UB)) break;
        issue(s, src);
      }
  }
  // Waits (bounded: 2^26 polls) for the next unit; returns its slot.  A
  // spinning test_wait measured slightly faster than the suspending try_wait.
  __device__ __forceinline__ const uint8_t* acquire() {
    const uint32_t slot = n_used % S;
    if (!timed_out) {
      uint32_t it = 0;
      while (!mbar_test_wait(&full[slot], (n_used / S) & 1))
        if (++it > (1u << 26)) {
          timed_out = true;
          break;
        }
    }
    return ring + (size_t)slot * UB;
  }
  // The unit's fragments are in registers: refill the slot with the warp's
  // next unit (self-refill), or hand it back to the producer.
  __device__ __forceinline__ void release(int lane) {
    __syncwarp();
    const uint32_t slot = n_used % S;
    if (lane == 0) {
      if (kSelfRefill) {
        const uint8_t* src;
        if (cur.next(src, UB)) {
          // the warp's generic-proxy reads of the slot come before the copy's writes
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          issue(slot, src);
        }
      } else {
        mbar_arrive(&empty[slot]);
      }
    }
    ++n_used;
  }
};

// Initialises the full/empty barriers of all rings of the CTA (one thread).
__device__ __forceinline__ void ring_init_barriers(uint64_t* full, uint64_t* empty, int n) {
  for (int i = 0; i < n; ++i) {
    mbar_init(&full[i], 1);
    mbar_init(&empty[i], 1);
  }
  mbar_fence_init();
}

// Producer mode: lane w < n_warps fills consumer warp w's ring of S slots
// with the warp's runs of ops[0 .. n_ops), in order; a slot is refilled once
// its previous unit was released.  Every lane runs the same loop (ready
// lanes issue, others wait for the next pass), so no lane's wait holds up
// another's copy.  Bounded: `limit` passes without any copy set
// ST_WAIT_TIMEOUT and end the producer (the consumers' own bounded waits
// then give up too).
template <int GPU, int S>
__device__ __noinline__ void ring_producer(const OpDesc* ops, int n_ops, int cta, int n_cta, int n_warps, uint8_t* rings,
                                           uint64_t* full, uint64_t* empty, int* status, uint32_t limit, int lane) {
  constexpr int UB = Geom<GPU>::kUnitBytes;
  const bool mine = lane < n_warps;
  uint8_t* ring = rings + (size_t)(mine ? lane : 0) * S * UB;
  uint64_t* f = full + (mine ? lane : 0) * S;
  uint64_t* e = empty + (mine ? lane : 0) * S;
  StreamCursor cur;
  cur.init(ops, mine ? n_ops : 0, cta * n_warps + lane, n_cta * n_warps, UB);
  const uint64_t policy = l2_policy_evict_first();
  bool active = mine;
  const uint8_t* src = nullptr;
  bool have = false;  // `src` holds the next unit, not yet issued
  uint32_t n = 0, idle = 0;
  while (true) {
    if (active && !have) {
      have = cur.next(src, UB);
      active = have;
    }
    bool issued = false;
    if (have) {
      const uint32_t slot = n % S;
      if (n < (uint32_t)S || mbar_test_wait(&e[slot], ((n / S) - 1) & 1)) {
        mbar_arrive_expect_tx(&f[slot], UB);
        bulk_g2s_hint(ring + (size_t)slot * UB, src, UB, &f[slot], policy);
        ++n;
        have = false;
        issued = true;
      }
    }
    if (!__any_sync(0xffffffffu, active)) break;
    if (__any_sync(0xffffffffu, issued)) {
      idle = 0;
    } else {
      if (++idle > limit) {
        if (lane == 0) atomicOr(status, ST_WAIT_TIMEOUT);
        break;
      }
      __nanosleep(20);
    }
  }
}

// ---------------------------------------------------------------------------
// One unit (64 rows x 128 inputs) of one warp.
//
// Codes enter the tensor cores as fp16 subnormals: the nibbles at bits 0..3
// (and 16..19) of a code word w are, read as fp16 bit patterns, exactly
// q * 2^-24, and the nibbles at bits 4..7 are 16 q * 2^-24, so each A
// register is one AND of w (or of w >> 8): a0 = w & 0x000F000F, a1 = w &
// 0x00F000F0 (rows gid + 8 of the tile, scaled by 16), a2 and a3 likewise
// from w >> 8.  The zero point is applied once per group instead of once per
// weight: sum_k (q - z) a = sum_k q a - z sum_k a, where sum_k a, the group
// sum of each token's activations, comes from one more MMA per k-block with
// an all-ones A.  The unit stores z (rows gid) and 16 z (rows gid + 8) as
// bytes, so one byte permute gives (-z * 2^-24, -16 z * 2^-24) as fp16
// subnormals in the same scale as the sums.  Per group and row:
//   tot += s * (acc + zs * sum_a)
// in units of 2^-24 (rows gid) and 2^-20 (rows gid + 8); segment_end applies
// the powers of two when it converts to fixed point.  Products are exact and
// accumulate in fp32.
// ---------------------------------------------------------------------------
constexpr float kTotScaleLo = 72057594037927936.0f;  // 2^56 = 2^32 (fixed point) * 2^24
constexpr float kTotScaleHi = 4503599627370496.0f;   // 2^52 = 2^32 * 2^20

template <int NT, int GPU>
__device__ __forceinline__ void mma_unit(const uint8_t* __restrict__ U, const uint4 (&act)[NT][2][2],
                                         float (&tot)[4][NT][4], int lane) {
  constexpr int BPG = Geom<GPU>::kBlocksPerGroup;
  constexpr uint32_t kOnes = 0x3C003C00u;  // fp16x2 (1, 1)
  const int gid = lane >> 2;
  float accg[4][NT][4];
  float sa[NT][4];  // group sums of the activations: tokens 2 tig, 2 tig + 1 (twice)
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
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
          for (int e = 0; e < 4; ++e) sa[nt][e] = 0.f;
#pragma unroll
          for (int rt = 0; rt < 4; ++rt)
#pragma unroll
            for (int e = 0; e < 4; ++e) accg[rt][nt][e] = 0.f;
        }
      }
      uint32_t b0[NT], b1[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const uint4 v = act[nt][kc][j >> 1];
        b0[nt] = (j & 1) ? v.z : v.x;
        b1[nt] = (j & 1) ? v.w : v.y;
        mma_16816(sa[nt], kOnes, kOnes, kOnes, kOnes, b0[nt], b1[nt]);
      }
#pragma unroll
      for (int rt = 0; rt < 4; ++rt) {
        const uint32_t w = (j == 0) ? A[rt].x : (j == 1) ? A[rt].y : (j == 2) ? A[rt].z : A[rt].w;
        const uint32_t w2 = w >> 8;
        const uint32_t a0 = w & 0x000F000Fu, a1 = w & 0x00F000F0u;
        const uint32_t a2 = w2 & 0x000F000Fu, a3 = w2 & 0x00F000F0u;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_16816(accg[rt][nt], a0, a1, a2, a3, b0[nt], b1[nt]);
      }
      if (blk % BPG == BPG - 1) {
        // group end: zero-point correction and scale
        const uint2 zz = *reinterpret_cast<const uint2*>(meta + 128 + gid * 8);
        const uint4 sc = *reinterpret_cast<const uint4*>(meta + gid * 16);
        const uint32_t scw[4] = {sc.x, sc.y, sc.z, sc.w};
#pragma unroll
        for (int rt = 0; rt < 4; ++rt) {
          const uint32_t zw = rt < 2 ? zz.x : zz.y;  // bytes: z_lo, 16 z_hi of tiles 2i, then 2i + 1
          const uint32_t p = 2u * (rt & 1);
          // fp16 bits 0x8000 | z and 0x8000 | 16 z: -z * 2^-24 and -16 z * 2^-24
          const uint32_t zp = prmt_u32(zw, 0x80u, p | (4u << 4) | ((p + 1u) << 8) | (4u << 12));
          const float zlo = h2f(static_cast<uint16_t>(zp & 0xFFFFu));
          const float zhi = h2f(static_cast<uint16_t>(zp >> 16));
          const float slo = h2f(static_cast<uint16_t>(scw[rt] & 0xFFFFu));
          const float shi = h2f(static_cast<uint16_t>(scw[rt] >> 16));
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            tot[rt][nt][0] = fmaf(slo, fmaf(zlo, sa[nt][0], accg[rt][nt][0]), tot[rt][nt][0]);
            tot[rt][nt][1] = fmaf(slo, fmaf(zlo, sa[nt][1], accg[rt][nt][1]), tot[rt][nt][1]);
            tot[rt][nt][2] = fmaf(shi, fmaf(zhi, sa[nt][0], accg[rt][nt][2]), tot[rt][nt][2]);
            tot[rt][nt][3] = fmaf(shi, fmaf(zhi, sa[nt][1], accg[rt][nt][3]), tot[rt][nt][3]);
          }
        }
      }
    }
  }
}

__device__ __forceinline__ float silu(float v) { return v / (1.f + expf(-v)); }

struct GemvPhase {
  const uint16_t* act;  // fp16 [M][act_ld]
  int act_ld, M;
  uint32_t act_s;       // 0, or the shared-memory address of this CTA's own copy of the activations,
  int act_s_ld;         // fp16 [M][act_s_ld], read instead of act
  int* status;
  EpiArgs ep;
  int kv_rb_q, kv_rb_k;  // EPI_QKV: row-blocks per q head group, first k and v row-block (see kv_head_of)
  int kv_rb_v, kv_rb_per_head;
  float* part;           // OpDesc::q > 0: the CTA's partial sums (shared memory), see swiglu_cta_write
};

// Loads the B fragments of input unit ku for tokens gid (and gid + 8).
template <int NT>
__device__ __forceinline__ void load_act(uint4 (&act)[NT][2][2], const uint16_t* actp, uint32_t acts, int act_ld,
                                         int M, int ku, int lane) {
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
        if (n < M) {
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

// kv head of q|k|v row-block rb (each row-block lies inside one head: d is a
// multiple of 64).
__device__ __forceinline__ int kv_head_of(const GemvPhase& p, int rb) {
  if (rb < p.kv_rb_k) return rb / p.kv_rb_q;
  if (rb < p.kv_rb_v) return (rb - p.kv_rb_k) / p.kv_rb_per_head;
  return (rb - p.kv_rb_v) / p.kv_rb_per_head;
}

// The contributor that completed row-block rb of a gate|up projection: lane
// = (tile t, row r) pair; gate is row 16 t + r, up row 16 t + r + 8, and h
// index j = 32 rb + 8 t + r.  Clears the sums and the count for the next use.
static __device__ __noinline__ void finish_swiglu(const GemvPhase* pp, int rb, int lane) {
  const GemvPhase& p = *pp;
  const int t = lane >> 3, r = lane & 7;
  const int Rg = rb * kRowsPerBlock + 16 * t + r, Ru = Rg + 8;
  const int j = 32 * rb + 8 * t + r;
  for (int m = 0; m < p.M; ++m) {
    long long* a = p.ep.acc + (size_t)m * p.ep.acc_ld;
    const float g = fixed_to_f32(__ldcg(a + Rg)), u = fixed_to_f32(__ldcg(a + Ru));
    if (j < p.ep.dims.F) p.ep.h[(size_t)m * p.ep.h_ld + j] = f2h(silu(g) * u);
    __stcg(a + Rg, 0LL);
    __stcg(a + Ru, 0LL);
  }
  if (lane == 0) __stcg(p.ep.cnt + rb, 0);
}

// The contributor that completed row-block rb of a stored projection: lane
// takes rows lane and lane + 32 of the row-block.
static __device__ __noinline__ void finish_store(const GemvPhase* pp, int rb, int lane) {
  const GemvPhase& p = *pp;
  for (int m = 0; m < p.M; ++m) {
    long long* a = p.ep.acc + (size_t)m * p.ep.acc_ld;
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int R = rb * kRowsPerBlock + lane + 32 * hh;
      const int nat = natural_row(p.ep.dims, R);
      if (nat >= 0) p.ep.y[(size_t)m * p.ep.y_ld + nat] = fixed_to_f32(__ldcg(a + R));
      __stcg(a + R, 0LL);
    }
  }
  if (lane == 0) __stcg(p.ep.cnt + rb, 0);
}

// ---------------------------------------------------------------------------
// Gate|up with OpDesc::q > 0: row-block rb is reduced inside its CTA.  Each
// of its q warps writes its sums, in natural scale, to its own slot of the
// CTA's partial area (fp32 [kCtaWarps][kGuCtaTokens][64]); after a named
// barrier of the q warps (id 2 + group) they add the q slots in a fixed order
// and write h = silu(gate) * up as fp16.  No global atomics; the result does
// not depend on arrival order.
// ---------------------------------------------------------------------------
constexpr int kGuCtaTokens = 5;  // tokens up to which the whole-step kernel reduces gate|up this way

template <int NT>
__device__ __forceinline__ void swiglu_cta_write(const GemvPhase& p, const float (&tot)[4][NT][4], int w, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
  float* slot = p.part + (size_t)w * kGuCtaTokens * kRowsPerBlock;
#pragma unroll
  for (int rt = 0; rt < 4; ++rt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int m = nt * 8 + 2 * tig + c;
        if (m < p.M) {
          slot[m * kRowsPerBlock + rt * 16 + gid] = tot[rt][nt][c] * 16777216.0f;        // 2^24
          slot[m * kRowsPerBlock + rt * 16 + gid + 8] = tot[rt][nt][2 + c] * 1048576.0f;  // 2^20
        }
      }
}

// After the group's barrier: gate row 16 t + r and up row 16 t + r + 8 of the
// row-block give h index 32 rb + 8 t + r (the unit row order of gate|up).
static __device__ __forceinline__ void swiglu_cta_finish(const GemvPhase* pp, int rb, int q, int w, int lane) {
  const GemvPhase& p = *pp;
  const int grp0 = w - w % q;
  const float* base = p.part + (size_t)grp0 * kGuCtaTokens * kRowsPerBlock;
  for (int it = (w - grp0) * 32 + lane; it < 32 * p.M; it += q * 32) {
    const int m = it >> 5, jl = it & 31;
    const int Rg = 16 * (jl >> 3) + (jl & 7);
    // each partial in fixed point as the atomic path adds it (exact integer
    // sums): the same bits for any token count
    long long gs = 0, us = 0;
    for (int i = 0; i < q; ++i) {
      const float* sl = base + (size_t)i * kGuCtaTokens * kRowsPerBlock + m * kRowsPerBlock;
      gs += f2fix(sl[Rg] * kFixOne);
      us += f2fix(sl[Rg + 8] * kFixOne);
    }
    const float gv = fixed_to_f32(gs), uv = fixed_to_f32(us);
    const int j = 32 * rb + jl;
    if (j < p.ep.dims.F) p.ep.h[(size_t)m * p.ep.h_ld + j] = f2h(silu(gv) * uv);
  }
}

// Whole end of a q > 0 run (called by every warp whose group owns a row-block,
// empty K range or not).
template <int NT>
__device__ __forceinline__ void swiglu_cta_end(const GemvPhase* pp, const OpDesc* op, const float (&tot)[4][NT][4],
                                               int g, int lane) {
  const int q = op->q;
  const int cta = g / kCtaWarps, w = g - cta * kCtaWarps;
  const int rb = cta * (kCtaWarps / q) + w / q;
  if (rb >= op->n_rb) return;  // the whole group has nothing (same test for each of its warps)
  swiglu_cta_write<NT>(*pp, tot, w, lane);
  named_bar_sync(2 + w / q, q * 32);
  swiglu_cta_finish(pp, rb, q, w, lane);
}

// End of one row-block segment (units of row-block rb) of a warp's run: add
// the sums to the accumulator, then count the units (see EpiArgs).
template <int NT>
__device__ __forceinline__ void segment_end(const GemvPhase* pp, const float (&tot)[4][NT][4], int rb, int units,
                                            int upr, int lane) {
  const GemvPhase& p = *pp;
  const int gid = lane >> 2, tig = lane & 3;
  const int kind = p.ep.kind;
  const int rows = kind == EPI_RESID ? p.ep.dims.H : 0x7FFFFFFF;
#pragma unroll
  for (int rt = 0; rt < 4; ++rt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int m = nt * 8 + 2 * tig + c;
        if (m < p.M) {
          long long* a = p.ep.acc + (size_t)m * p.ep.acc_ld + rb * kRowsPerBlock + rt * 16 + gid;
          if (rb * kRowsPerBlock + rt * 16 + gid < rows) red_add_s64(a, f2fix(tot[rt][nt][c] * kTotScaleLo));
          if (rb * kRowsPerBlock + rt * 16 + gid + 8 < rows)
            red_add_s64(a + 8, f2fix(tot[rt][nt][2 + c] * kTotScaleHi));
        }
      }
  if (kind == EPI_RESID) return;
  // The warp barrier orders every lane's additions before lane 0's release
  // (and lane 0's acquire before the finisher's loads).
  __syncwarp();
  if (kind == EPI_QKV) {
    if (lane == 0) red_release_add_s32(p.ep.cnt + kv_head_of(p, rb), units);
    return;
  }
  int last = 0;
  if (lane == 0) last = atom_add_acq_rel(p.ep.cnt + rb, units) + units == upr;
  last = __shfl_sync(0xffffffffu, last, 0);
  __syncwarp();
  if (!last) return;
  if (kind == EPI_SWIGLU)
    finish_swiglu(pp, rb, lane);
  else
    finish_store(pp, rb, lane);
}

// One projection for one warp: consume the warp's run of units from its ring
// (which is filled in the same order) and hand on each row-block segment of
// it.  Inlined at one call site (the whole-step kernel's layer loop, which
// keeps the ring in registers), so no call boundary spills the caller's
// registers.
template <int NT, int GPU, int S>
__device__ __forceinline__ void gemv_run(WarpRing<GPU, S>& ring, const OpDesc* op, const GemvPhase* pp, int g, int nw,
                                         int lane) {
  const GemvPhase& p = *pp;
  const int upr = op->upr;
  int wb, we;
  run_range(*op, g, nw, wb, we);
  if (wb >= we) {
    if (op->q > 0 && p.M <= kGuCtaTokens) {  // a group member without units still adds (zero) sums
      float zero[4][NT][4];
#pragma unroll
      for (int rt = 0; rt < 4; ++rt)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int e = 0; e < 4; ++e) zero[rt][nt][e] = 0.f;
      swiglu_cta_end<NT>(pp, op, zero, g, lane);
    }
    return;
  }
  const uint16_t* actp = p.act;
  const uint32_t acts = p.act_s;
  const int act_ld = acts ? p.act_s_ld : p.act_ld, M = p.M;
  int rb = wb / upr;
  int ku = wb - rb * upr;
  uint4 nxt[NT][2][2];
  load_act<NT>(nxt, actp, acts, act_ld, M, ku, lane);
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
#pragma unroll 2  // alternating activation registers instead of copies
    for (; u < seg_end; ++u) {
      uint4 cur[NT][2][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
          for (int h = 0; h < 2; ++h) cur[nt][kc][h] = nxt[nt][kc][h];
      if (++ku == upr) ku = 0;
      if (u + 1 < we) load_act<NT>(nxt, actp, acts, act_ld, M, ku, lane);
      const uint8_t* U = ring.acquire();
      if (!ring.timed_out) mma_unit<NT, GPU>(U, cur, tot, lane);
      ring.release(lane);
    }
    if (op->q > 0 && p.M <= kGuCtaTokens)
      swiglu_cta_end<NT>(pp, op, tot, g, lane);  // the run is one whole segment
    else
      segment_end<NT>(pp, tot, rb, seg_end - seg_begin, upr, lane);
  }
}

// gemv_run with the ring state in shared memory (the standalone kernel).
template <int NT, int GPU, int S>
__device__ __noinline__ void gemv_phase(WarpRing<GPU, S>* ring_io, const OpDesc* op, const GemvPhase* pp, int g, int nw,
                                        int lane) {
  WarpRing<GPU, S> ring = *ring_io;
  gemv_run<NT, GPU, S>(ring, op, pp, g, nw, lane);
  __syncwarp();
  if (lane == 0) *ring_io = ring;
  __syncwarp();
}

}  // namespace shard
