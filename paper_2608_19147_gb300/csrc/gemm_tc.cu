// W4A16 projection for many tokens on the 5th-generation tensor cores
// (tcgen05): Y[n][r] = sum_k W[r][k] x[n][k] for S tokens, W in the shard's
// unit stream (kernels.h).  Used where the token count makes the projection
// a dense contraction -- a prompt's prefill (Section 3.4: the stateful cache
// is filled by running the prompt through the stage) -- where the per-token
// GEMV of the decode step would stream every weight once per 16 tokens.
//
// One CTA computes a tile of 128 weight rows (two 64-row blocks) by N tokens,
// walking K one 128-input unit per step, with warp roles joined by mbarriers:
//   - warp 0 (producer): bulk-copies the step's two units (codes, scales,
//     zero points) and loads the token tile with two 2-D tensor copies (64
//     inputs x N tokens each, 128-byte swizzle); 3 stages ahead;
//   - warps 10..17 (dequantise): turn the codes into exact fp16 (q - z) in the
//     A tile; 2 stages;
//   - warp 1 (MMA): issues tcgen05.mma (kind::f16, M = 128, N tokens, K = 16
//     per instruction) into a TMEM accumulator per quantisation group and
//     commits to the stages' mbarriers; 2 accumulator stages;
//   - warps 2..9 (epilogue): read the step's accumulators (tcgen05.ld; warp w
//     owns TMEM lanes 32 (w % 4) .. + 31 = tile rows, half the token columns
//     each), multiply by the row's fp32 group scale and add into registers;
//     at the end they write their rows' outputs.
// Both operands sit in shared memory in the canonical K-major layout with the
// 128-byte swizzle: per 64-input half of the step, row r's 128 bytes at r *
// 128, its 16-byte chunk c at chunk c ^ (r % 8) -- what the tensor copy writes
// with that swizzle, whole 32-byte sectors from L2, and a layout in which the
// dequantise warps' 16-byte stores of 8 consecutive rows hit distinct banks.
// The
// arithmetic is the decode projection's: exact (q - z), fp32 sums per group,
// the fp16 scale applied in fp32.  Every wait is bounded; a wait that runs out
// sets the status word.  The TMEM columns are freed before the CTA exits.
#include <cuda.h>

#include <mutex>

#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kTcRows = 128;        // weight rows per CTA tile (two row-blocks)
constexpr int kTcWarps = 18;        // producer, MMA, 8 epilogue, 8 dequantise
constexpr int kDqWarps = 8;
constexpr int kTcThreads = kTcWarps * 32;
constexpr int kEpiWarp0 = 2, kDqWarp0 = 10;
constexpr int kUStages = 4, kBStages = 3, kAStages = 2, kDStages = 2;

template <int N, int GPU>
struct TcSmem {
  static constexpr size_t kUnit = Geom<GPU>::kUnitBytes;
  static constexpr size_t kUnits = 2 * kUnit;                          // the tile's two units
  static constexpr size_t kA = (size_t)kTcRows * 256;                  // 16 K chunks x 128 rows x 16 B
  static constexpr size_t kB = (size_t)N * 256;                        // 16 K chunks x N tokens x 16 B
  static constexpr size_t kAOff = 0;                                   // [kAStages][kA]
  static constexpr size_t kBOff = kAOff + kAStages * kA;               // [kBStages][kB]
  static constexpr size_t kUOff = kBOff + kBStages * kB;               // [kUStages][kUnits]
  static constexpr size_t kSc = (size_t)GPU * kTcRows * sizeof(float);  // a step's scales [group][row]
  static constexpr size_t kScOff = kUOff + kUStages * kUnits;          // [kAStages][kSc]
  static constexpr size_t kTotal = kScOff + kAStages * kSc + 1024;     // + alignment slack
};

// Shared-memory matrix descriptor, K-major with the 128-byte swizzle: 8-row
// groups 1024 bytes apart (the byte offset between K-adjacent core matrices is
// implied by the swizzle); the start address may move by 32 bytes per K = 16
// inside a 64-input half.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;            // leading byte offset: unused with this swizzle
  d |= (uint64_t)(1024 >> 4) << 32;  // stride byte offset
  d |= 1ull << 46;                   // descriptor version for this architecture
  d |= 2ull << 61;                   // layout: 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator, fp16 A and B, both
// K-major, M = 128, N tokens.
template <int N>
__device__ __forceinline__ uint32_t instr_desc() {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(kTcRows >> 4) << 24);
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, bool acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"((uint32_t)acc)
      : "memory");
}

// Arrive on `bar` once every tcgen05 operation this thread issued so far is done.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_addr(bar))
               : "memory");
}

// 16 consecutive fp32 columns of this thread's tensor-memory lane (into v[0..15]).
__device__ __forceinline__ void tc_ld16(uint32_t taddr, float (&v)[32]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, "
      "[%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// 2-D tensor copy of one box into shared memory, completion on `bar`.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

// Offset of element (row, k) of an operand tile of `rows` rows x 128 inputs,
// 128-byte swizzled K-major: [64-input half][row][128 B], chunk c at c ^ (row % 8).
__device__ __forceinline__ uint32_t op_off(int rows, int row, int k) {
  return (uint32_t)(k >> 6) * (uint32_t)(rows * 128) + (uint32_t)row * 128u +
         (uint32_t)((((k >> 3) & 7) ^ (row & 7)) << 4) + (uint32_t)(k & 7) * 2u;
}

// Kernel arguments: the projection and the tensor map of its activations
// (fp16 [S][act_ld], box 8 inputs x N tokens).
struct TcParams {
  GemmArgs a;
  CUtensorMap act_map;  // {K inputs, S tokens}, box 64 x N, 128-byte swizzle
};

template <int N, int GPU>
__global__ void __launch_bounds__(kTcThreads, 1) gemm_tc_kernel(const __grid_constant__ TcParams P) {
  const GemmArgs& a = P.a;
  using L = TcSmem<N, GPU>;
  constexpr int UB = Geom<GPU>::kUnitBytes;
  constexpr int G = GPU;                        // quantisation groups per unit
  constexpr int kMmaPerGroup = 8 / GPU;         // K = 16 per instruction
  constexpr int kHalf = N / 2;                  // token columns per epilogue thread
  constexpr uint32_t kHalfA = kTcRows * 128, kHalfB = N * 128;  // bytes per 64-input half
  constexpr uint32_t kColsNeed = (uint32_t)kDStages * G * N;
  constexpr uint32_t kCols = kColsNeed <= 32 ? 32u : kColsNeed <= 64 ? 64u : kColsNeed <= 128 ? 128u
                             : kColsNeed <= 256 ? 256u : 512u;
  static_assert(kColsNeed <= 512, "accumulators exceed tensor memory");
  static_assert(kHalf % 16 == 0, "columns per epilogue thread");
  static_assert(kAStages == kDStages, "the epilogue reads the scales of its accumulator stage");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t u_full[kUStages], u_empty[kUStages], b_full[kBStages], b_empty[kBStages];
  __shared__ uint64_t a_full[kAStages], a_empty[kAStages], d_full[kDStages], d_empty[kDStages];
  __shared__ uint32_t s_tmem;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb0 = 2 * blockIdx.x;   // the tile's first row-block
  const int n0 = blockIdx.y * N;    // the tile's first token
  const int steps = a.upr;
  auto A_of = [&](int s) { return smem + L::kAOff + (size_t)s * L::kA; };
  auto B_of = [&](int s) { return smem + L::kBOff + (size_t)s * L::kB; };
  auto U_of = [&](int s) { return smem + L::kUOff + (size_t)s * L::kUnits; };
  auto Sc_of = [&](int s) { return reinterpret_cast<float*>(smem + L::kScOff + (size_t)s * L::kSc); };
  if (tid == 0) {
    for (int i = 0; i < kUStages; ++i) {
      mbar_init(&u_full[i], 1);
      mbar_init(&u_empty[i], kDqWarps);
    }
    for (int i = 0; i < kBStages; ++i) {
      mbar_init(&b_full[i], 1);
      mbar_init(&b_empty[i], 1);
    }
    for (int i = 0; i < kAStages; ++i) {
      mbar_init(&a_full[i], kDqWarps);
      mbar_init(&a_empty[i], 1);
    }
    for (int i = 0; i < kDStages; ++i) {
      mbar_init(&d_full[i], 1);
      mbar_init(&d_empty[i], 8);
    }
    mbar_fence_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&s_tmem)),
                 "r"(kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  bool ok = true;  // false once a wait gave up: the role skips the rest of its waits
  auto wait = [&](uint64_t* bar, uint32_t parity) {
    if (ok && !mbar_wait(bar, parity)) ok = false;
  };

  if (warp == 0) {
    // ---- producer: units and token tiles, kUStages / kBStages steps ahead ----
    if (lane == 0) {
      for (int k = 0; k < steps; ++k) {
        const int su = k % kUStages, sb = k % kBStages;
        wait(&u_empty[su], ((k / kUStages) & 1) ^ 1);
        mbar_arrive_expect_tx(&u_full[su], 2 * UB);
        for (int u = 0; u < 2; ++u) {
          const int rb = rb0 + u < a.n_rb ? rb0 + u : rb0;  // a missing second block repeats the first (unused)
          bulk_g2s(U_of(su) + (size_t)u * UB, a.units + ((size_t)rb * a.upr + k) * UB, UB, &u_full[su]);
        }
        wait(&b_empty[sb], ((k / kBStages) & 1) ^ 1);
        mbar_arrive_expect_tx(&b_full[sb], N * 256);
        for (int h = 0; h < 2; ++h)  // tokens past S read as zero
          tma_load_2d(B_of(sb) + (size_t)h * kHalfB, &P.act_map, k * kUnitK + h * 64, n0, &b_full[sb]);
      }
    }
  } else if (warp == 1) {
    // ---- MMA issue: one thread ----
    if (lane == 0) {
      for (int k = 0; k < steps; ++k) {
        const int sa = k % kAStages, sb = k % kBStages, sd = k % kDStages;
        wait(&a_full[sa], (k / kAStages) & 1);
        wait(&b_full[sb], (k / kBStages) & 1);
        wait(&d_empty[sd], ((k / kDStages) & 1) ^ 1);
        tc_fence_after();
        if (ok) {
          const uint32_t aBase = smem_addr(A_of(sa)), bBase = smem_addr(B_of(sb));
#pragma unroll
          for (int gq = 0; gq < G; ++gq)
#pragma unroll
            for (int i = 0; i < kMmaPerGroup; ++i) {
              const int kk = gq * kMmaPerGroup + i;  // K = 16: inputs 16 kk .. + 15
              const uint32_t ko = (uint32_t)(kk & 3) * 32u;  // inside the 64-input half
              tc_mma(tmem + (uint32_t)((sd * G + gq) * N), smem_desc_sw128(aBase + (kk >> 2) * kHalfA + ko),
                     smem_desc_sw128(bBase + (kk >> 2) * kHalfB + ko), instr_desc<N>(), i > 0);
            }
        }
        tc_commit(&a_empty[sa]);
        tc_commit(&b_empty[sb]);
        tc_commit(&d_full[sd]);
      }
    }
  } else if (warp >= kDqWarp0) {
    // ---- dequantise: exact fp16 (q - z) into the A tile ----
    const int dt = (warp - kDqWarp0) * 32 + lane;
    const int gid = dt & 7, tig = (dt >> 3) & 3;  // 8 consecutive threads: rows gid 0..7 of one K chunk
    const int l = gid * 4 + tig;                  // the fragment lane whose words this thread takes
    for (int k = 0; k < steps; ++k) {
      const int su = k % kUStages, sa = k % kAStages;
      wait(&u_full[su], (k / kUStages) & 1);
      wait(&a_empty[sa], ((k / kAStages) & 1) ^ 1);
      wait(&d_empty[sa], ((k / kAStages) & 1) ^ 1);  // the epilogue is done with this stage's scales
      const uint8_t* Us = U_of(su);
      uint8_t* As = A_of(sa);
      // the step's fp32 scales [group][tile row], for the epilogue
      for (int e = dt; e < G * kTcRows; e += kDqWarps * 32) {
        const int gq = e / kTcRows, r = e % kTcRows, R = r & 63;
        const int sidx = (R & 7) * 8 + ((R >> 4) & 3) * 2 + ((R >> 3) & 1);
        Sc_of(sa)[e] = h2f(reinterpret_cast<const uint16_t*>(Us + (size_t)(r >> 6) * UB + kCodeBytes +
                                                            gq * kMetaBytesPerGroup)[sidx]);
      }
#pragma unroll
      for (int i = 0; i < 16 / kDqWarps; ++i) {
        const int uf = (warp - kDqWarp0) + kDqWarps * i;  // (unit, code tile) 0..15
        const int u = uf >> 3, ft = uf & 7, rt = ft & 3, kh = ft >> 2;
        const uint8_t* U = Us + (size_t)u * UB;
        const uint4 w4 = *reinterpret_cast<const uint4*>(U + ft * 512 + l * 16);
        const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
        const int row = 64 * u + 16 * rt + gid;
        uint32_t lo[2][4], hi[2][4];  // [K chunk: j / 2][4 fp16 pairs]
        uint32_t zsub[2], zfma[2];     // per K chunk (its 8 inputs lie in one group)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint8_t* meta = U + kCodeBytes + ((64 * kh + 32 * c + 8 * tig) / (kUnitK / G)) * kMetaBytesPerGroup;
          const uint16_t zz = *reinterpret_cast<const uint16_t*>(meta + 128 + gid * 8 + rt * 2);
          zsub[c] = (0x6400u | (zz & 0xFFu)) * 0x00010001u;  // fp16x2 (1024 + z)
          zfma[c] = (0xD400u | (zz >> 8)) * 0x00010001u;     // fp16x2 -(64 + z)
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          // word j: rows gid and gid + 8 at inputs 64 kh + 32 (j / 2) + 8 tig + 4 (j % 2) .. + 3
          const uint32_t w = wv[j], w2 = w >> 8;
          const uint32_t zs = zsub[j >> 1], zf = zfma[j >> 1];
          lo[j >> 1][2 * (j & 1)] = hsub2_u32(lop3_and_or(w, 0x000F000Fu, 0x64006400u), zs);
          lo[j >> 1][2 * (j & 1) + 1] = hsub2_u32(lop3_and_or(w2, 0x000F000Fu, 0x64006400u), zs);
          hi[j >> 1][2 * (j & 1)] = hfma2_u32(lop3_and_or(w, 0x00F000F0u, 0x64006400u), 0x2C002C00u, zf);
          hi[j >> 1][2 * (j & 1) + 1] = hfma2_u32(lop3_and_or(w2, 0x00F000F0u, 0x64006400u), 0x2C002C00u, zf);
        }
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const int kb = 64 * kh + 32 * c + 8 * tig;  // the 8-input chunk's first input
          *reinterpret_cast<uint4*>(As + op_off(kTcRows, row, kb)) = make_uint4(lo[c][0], lo[c][1], lo[c][2], lo[c][3]);
          *reinterpret_cast<uint4*>(As + op_off(kTcRows, row + 8, kb)) =
              make_uint4(hi[c][0], hi[c][1], hi[c][2], hi[c][3]);
        }
      }
      // the generic-proxy stores become visible to the tensor cores
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&a_full[sa]);
        mbar_arrive(&u_empty[su]);
      }
    }
  } else {
    // ---- epilogue: scale and add each step's group sums ----
    const int quad = warp & 3, half = (warp - kEpiWarp0) >> 2;
    const int row = 32 * quad + lane;  // tile row = TMEM lane
    const int c0 = half * kHalf;
    const int R = row & 63;
    float tot[kHalf];
#pragma unroll
    for (int c = 0; c < kHalf; ++c) tot[c] = 0.f;
    for (int k = 0; k < steps; ++k) {
      const int sd = k % kDStages;  // = the A stage: kAStages == kDStages
      wait(&d_full[sd], (k / kDStages) & 1);
      wait(&a_full[sd], (k / kAStages) & 1);  // the stage's scales (written before its A tile was released)
      tc_fence_after();
      const float* sc = Sc_of(sd);
#pragma unroll
      for (int gq = 0; gq < G; ++gq) {
        const float sv = sc[gq * kTcRows + row];
#pragma unroll
        for (int cc = 0; cc < kHalf; cc += 16) {
          float v[32];
          tc_ld16(tmem + ((uint32_t)(32 * quad) << 16) + (uint32_t)((sd * G + gq) * N + c0 + cc), v);
#pragma unroll
          for (int c = 0; c < 16; ++c) tot[cc + c] = fmaf(sv, v[c], tot[cc + c]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&d_empty[sd]);
    }
    // outputs: natural row order, [token][row]
    const int rbr = rb0 + (row >> 6);
    if (rbr < a.n_rb) {
      const int nat = natural_row(a.dims, rbr * kRowsPerBlock + R);
      if (nat >= 0)
#pragma unroll
        for (int c = 0; c < kHalf; ++c)
          if (n0 + c0 + c < a.S) a.y[(size_t)(n0 + c0 + c) * a.y_ld + nat] = tot[c];
    }
  }
  if (!ok) atomicOr(a.status, ST_WAIT_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kCols) : "memory");
}

// cuTensorMapEncodeTiled, from the driver through the runtime (no link
// against the driver library).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

template <int N, int GPU>
cudaError_t launch_tc(const GemmArgs& a, cudaStream_t s) {
  using L = TcSmem<N, GPU>;
  EncodeTiledFn enc = encode_tiled();
  if (!enc) return cudaErrorNotSupported;
  // the activations: fp16 [S][act_ld] (16-byte aligned rows); box = 8
  // inputs (16 bytes) x N tokens; tokens past S read as zero
  if ((reinterpret_cast<uintptr_t>(a.act) & 15) || a.act_ld % 8 || a.upr * kUnitK > a.act_ld || a.S < 1)
    return cudaErrorInvalidValue;
  TcParams p;
  p.a = a;
  const cuuint64_t dims[2] = {(cuuint64_t)a.upr * kUnitK, (cuuint64_t)a.S};
  const cuuint64_t strides[1] = {(cuuint64_t)a.act_ld * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)N};
  const cuuint32_t estr[2] = {1, 1};
  if (enc(&p.act_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<uint16_t*>(a.act), dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const dim3 grid((a.n_rb + 1) / 2, (a.S + N - 1) / N);
  gemm_tc_kernel<N, GPU><<<grid, kTcThreads, L::kTotal, s>>>(p);
  return cudaGetLastError();
}

template <int N, int GPU>
cudaError_t setup_tc() {
  return cudaFuncSetAttribute(gemm_tc_kernel<N, GPU>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)TcSmem<N, GPU>::kTotal);
}

}  // namespace

cudaError_t gemm_tc_setup() {
  cudaError_t e;
  if ((e = setup_tc<32, 1>()) != cudaSuccess) return e;
  if ((e = setup_tc<32, 2>()) != cudaSuccess) return e;
  if ((e = setup_tc<32, 4>()) != cudaSuccess) return e;
  if ((e = setup_tc<64, 1>()) != cudaSuccess) return e;
  if ((e = setup_tc<64, 2>()) != cudaSuccess) return e;
  if ((e = setup_tc<64, 4>()) != cudaSuccess) return e;
  if ((e = setup_tc<128, 1>()) != cudaSuccess) return e;
  if ((e = setup_tc<128, 2>()) != cudaSuccess) return e;
  return cudaSuccess;
}

// Token tile: 128 for long prompts, smaller for short ones; at group 32 (four
// accumulators per step) at most 64.
int gemm_tc_tile(int S) { return S > 64 ? 128 : S > 32 ? 64 : 32; }
int gemm_tc_tile(int S, int group) { return group == 32 ? (S > 32 ? 64 : 32) : gemm_tc_tile(S); }

cudaError_t launch_gemm_tc(const GemmArgs& a, int group, cudaStream_t s) {
  const int N = gemm_tc_tile(a.S, group);
  if (N == 32) {
    if (group == 128) return launch_tc<32, 1>(a, s);
    if (group == 64) return launch_tc<32, 2>(a, s);
    if (group == 32) return launch_tc<32, 4>(a, s);
  } else if (N == 64) {
    if (group == 128) return launch_tc<64, 1>(a, s);
    if (group == 64) return launch_tc<64, 2>(a, s);
    if (group == 32) return launch_tc<64, 4>(a, s);
  } else if (N == 128) {
    if (group == 128) return launch_tc<128, 1>(a, s);
    if (group == 64) return launch_tc<128, 2>(a, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace shard
