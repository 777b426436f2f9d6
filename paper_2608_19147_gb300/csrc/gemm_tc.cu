// W4A16 projection for many tokens on the 5th-generation tensor cores
// (tcgen05): Y[n][r] = sum_k W[r][k] x[n][k] for S tokens, W in the shard's
// unit stream (kernels.h).  Used where the token count makes the projection
// a dense contraction -- a prompt's prefill (Section 3.4: the stateful cache
// is filled by running the prompt through the stage) -- where the per-token
// GEMV of the decode step would stream every weight once per 16 tokens.
//
// One CTA (8 warps) computes a tile of 128 weight rows (two 64-row blocks)
// by N tokens, walking K one 128-input unit at a time, as a two-stage
// software pipeline (every buffer below exists twice, used by alternate
// steps):
//   - thread 0 bulk-copies the tile's two units (codes, scales, zero points)
//     into shared memory (TMA, non-tensor; mbarrier completion) two steps
//     ahead;
//   - the CTA stages the N x 128 token tile into shared memory in the
//     canonical K-major layout without swizzle (8-row x 16-byte core
//     matrices: element (row, k) at (row/8)*2048 + (k/8)*128 + (row%8)*16
//     + (k%8)*2 bytes) and dequantises the weights into the same layout as
//     exact fp16 (q - z) -- the per-group fp16 scale is applied later in
//     fp32, so no rounding is added to the W4A16 arithmetic;
//   - thread 0 issues tcgen05.mma (kind::f16, M = 128, N tokens, K = 16 per
//     instruction) from the two shared-memory operands into a tensor-memory
//     accumulator per quantisation group and commits them to an mbarrier;
//   - while those run, the CTA prepares the next step and reads back the
//     accumulators of the step before (tcgen05.ld; warp w holds rows
//     32 (w % 4) .. + 31, half of the token columns), multiplies them by the
//     row's group scale and adds them into fp32 registers.
// At the end each thread writes its row's outputs.  Waits are bounded; a wait
// that runs out sets the status word.  The tensor memory is freed before the
// CTA exits.
#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kTcRows = 128;       // weight rows per CTA tile (two row-blocks)
constexpr int kTcThreads = 256;    // 8 warps: warp w owns rows 32 (w % 4) .. + 31, columns half w / 4
constexpr uint32_t kCoreK = 128;   // bytes between core matrices adjacent in K
constexpr uint32_t kCoreMN = 2048; // bytes between 8-row groups (16 core matrices of K)

template <int N, int GPU>
struct TcSmem {
  static constexpr size_t kUnit = Geom<GPU>::kUnitBytes;
  static constexpr size_t kUnits = 2 * kUnit;          // the tile's two units
  static constexpr size_t kA = (size_t)kTcRows * 256;  // 128 rows x 128 fp16
  static constexpr size_t kB = (size_t)N * 256;        // N tokens x 128 fp16
  static constexpr size_t kSc = (size_t)GPU * kTcRows * 4;  // the step's scales, fp32 [group][row]
  static constexpr size_t kUnitsOff = 0;                            // [2][kUnits]
  static constexpr size_t kAOff = (2 * kUnits + 1023) / 1024 * 1024;  // [2][kA]
  static constexpr size_t kBOff = kAOff + 2 * kA;                   // [2][kB]
  static constexpr size_t kScOff = kBOff + 2 * kB;                  // [2][kSc]
  static constexpr size_t kTotal = kScOff + 2 * kSc;
};

// Shared-memory matrix descriptor: K-major, no swizzle; LBO = distance of
// core matrices adjacent in K, SBO = distance of 8-row groups.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)(kCoreK >> 4) << 16;
  d |= (uint64_t)(kCoreMN >> 4) << 32;
  d |= 1ull << 46;  // descriptor version for this architecture
  return d;         // base offset 0, layout type 0 (no swizzle)
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

__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_addr(bar))
               : "memory");
}

// 32 consecutive fp32 columns of this thread's tensor-memory lane.
__device__ __forceinline__ void tc_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 consecutive fp32 columns of this thread's tensor-memory lane.
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

__device__ __forceinline__ uint32_t a_off(int row, int k) {
  return (uint32_t)(row >> 3) * kCoreMN + (uint32_t)(k >> 3) * kCoreK + (uint32_t)(row & 7) * 16u + (uint32_t)(k & 7) * 2u;
}

template <int N, int GPU>
__global__ void __launch_bounds__(kTcThreads, 1) gemm_tc_kernel(const __grid_constant__ GemmArgs a) {
  using L = TcSmem<N, GPU>;
  constexpr int UB = Geom<GPU>::kUnitBytes;
  constexpr int G = GPU;                       // quantisation groups per unit
  constexpr int kMmaPerGroup = 8 / GPU;        // K = 16 per instruction
  constexpr int kHalf = N / 2;                 // token columns per thread
  constexpr int kBPer = (N * 16 + kTcThreads - 1) / kTcThreads;  // 16-byte token pieces per thread
  constexpr uint32_t kColsNeed = 2u * G * N;   // two steps' accumulators
  constexpr uint32_t kCols = kColsNeed <= 32 ? 32u : kColsNeed <= 64 ? 64u : kColsNeed <= 128 ? 128u
                             : kColsNeed <= 256 ? 256u : 512u;
  static_assert(kColsNeed <= 512, "accumulators exceed tensor memory");
  static_assert(kHalf % 32 == 0 || kHalf == 16, "columns per thread");
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ uint64_t s_ubar[2], s_mbar[2];
  __shared__ uint32_t s_tmem;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb0 = 2 * blockIdx.x;              // the tile's first row-block
  const int n0 = blockIdx.y * N;               // the tile's first token
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_ubar[i], 1);
      mbar_init(&s_mbar[i], 1);
    }
    mbar_fence_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&s_tmem)),
                 "r"(kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const int row = 32 * (warp & 3) + lane;      // this thread's row of the tile (its tensor-memory lane)
  const int c0 = kHalf * (warp >> 2);          // its first token column
  auto units_of = [&](int s) { return smem + L::kUnitsOff + (size_t)s * L::kUnits; };
  auto A_of = [&](int s) { return smem + L::kAOff + (size_t)s * L::kA; };
  auto B_of = [&](int s) { return smem + L::kBOff + (size_t)s * L::kB; };
  auto sc_of = [&](int s) { return reinterpret_cast<float*>(smem + L::kScOff + (size_t)s * L::kSc); };
  auto issue_units = [&](int ku, int s) {
    mbar_arrive_expect_tx(&s_ubar[s], 2 * UB);
    for (int u = 0; u < 2; ++u) {
      const int rb = rb0 + u < a.n_rb ? rb0 + u : rb0;  // a missing second block repeats the first (unused)
      bulk_g2s(units_of(s) + (size_t)u * UB, a.units + ((size_t)rb * a.upr + ku) * UB, UB, &s_ubar[s]);
    }
  };
  float tot[kHalf];
#pragma unroll
  for (int c = 0; c < kHalf; ++c) tot[c] = 0.f;
  bool ok = true;
  // scale and add the accumulators of step j (slot j & 1)
  auto epilogue = [&](int j) {
    const int s = j & 1;
    if (ok && !mbar_wait(&s_mbar[s], (j >> 1) & 1)) ok = false;
    tc_fence_after();
    const float* sc = sc_of(s);
#pragma unroll
    for (int gq = 0; gq < G; ++gq) {
      const float sv = sc[gq * kTcRows + row];
#pragma unroll
      for (int cc = 0; cc < kHalf; cc += 32) {
        float v[32];
        const uint32_t ta = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)((s * G + gq) * N + c0 + cc);
        if (kHalf >= 32)
          tc_ld32(ta, v);
        else
          tc_ld16(ta, v);  // 16 columns: only those of this thread's half
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (cc + c < kHalf) tot[cc + c] = fmaf(sv, v[c], tot[cc + c]);
      }
    }
  };
  if (tid == 0) {
    issue_units(0, 0);
    if (a.upr > 1) issue_units(1, 1);
  }
  for (int k = 0; k < a.upr; ++k) {
    const int s = k & 1;
    // the step's token tile, into registers (its latency overlaps the epilogue)
    uint4 bv[kBPer];
#pragma unroll
    for (int i = 0; i < kBPer; ++i) {
      const int e = tid + i * kTcThreads, n = e >> 4, kc = e & 15;
      bv[i] = make_uint4(0, 0, 0, 0);
      if (e < N * 16 && n0 + n < a.S)
        bv[i] = __ldcg(reinterpret_cast<const uint4*>(a.act + (size_t)(n0 + n) * a.act_ld + k * kUnitK + 8 * kc));
    }
    // step k - 2 used this slot: its MMAs are done once its accumulators are read
    if (k >= 2) epilogue(k - 2);
    tc_fence_before();
    __syncthreads();  // slot s (tiles, scales, accumulators) is free
    if (ok && !mbar_wait(&s_ubar[s], (k >> 1) & 1)) ok = false;
    uint8_t* Bs = B_of(s);
#pragma unroll
    for (int i = 0; i < kBPer; ++i) {
      const int e = tid + i * kTcThreads;
      if (e < N * 16) *reinterpret_cast<uint4*>(Bs + a_off(e >> 4, 8 * (e & 15))) = bv[i];
    }
    // dequantise: word (ft, l, j) of unit u holds rows 16 rt + gid (+8) at
    // inputs k0 .. k0 + 3 (kernels.h); q - z exactly, as fp16
    const uint8_t* Us = units_of(s);
    uint8_t* As = A_of(s);
    for (int e = tid; e < 2 * (kCodeBytes / 4); e += kTcThreads) {
      const int u = e / (kCodeBytes / 4), wi = e % (kCodeBytes / 4);
      const int ft = wi >> 7, l = (wi >> 2) & 31, j = wi & 3;
      const int kc = ft >> 2, rt = ft & 3, gid = l >> 2, tig = l & 3;
      const int k0 = 64 * kc + 32 * (j >> 1) + 8 * tig + 4 * (j & 1);
      const uint8_t* U = Us + (size_t)u * UB;
      const uint32_t w = reinterpret_cast<const uint32_t*>(U)[wi];
      const uint8_t* meta = U + kCodeBytes + (k0 / (kUnitK / G)) * kMetaBytesPerGroup;
      const int idx = gid * 8 + rt * 2;
      const uint32_t zlo = meta[128 + idx], z16hi = meta[128 + idx + 1];
      const uint32_t zsub = (0x6400u | zlo) * 0x00010001u;         // fp16x2 (1024 + z)
      const uint32_t zfma = (0xD400u | z16hi) * 0x00010001u;       // fp16x2 -(64 + z)
      const uint32_t w2 = w >> 8;
      const uint32_t q01 = hsub2_u32(lop3_and_or(w, 0x000F000Fu, 0x64006400u), zsub);
      const uint32_t q23 = hsub2_u32(lop3_and_or(w2, 0x000F000Fu, 0x64006400u), zsub);
      const uint32_t h01 = hfma2_u32(lop3_and_or(w, 0x00F000F0u, 0x64006400u), 0x2C002C00u, zfma);
      const uint32_t h23 = hfma2_u32(lop3_and_or(w2, 0x00F000F0u, 0x64006400u), 0x2C002C00u, zfma);
      const int r = 64 * u + 16 * rt + gid;
      *reinterpret_cast<uint2*>(As + a_off(r, k0)) = make_uint2(q01, q23);
      *reinterpret_cast<uint2*>(As + a_off(r + 8, k0)) = make_uint2(h01, h23);
    }
    // the step's scales, fp32 [group][row]
    float* sc = sc_of(s);
    for (int e = tid; e < G * kTcRows; e += kTcThreads) {
      const int gq = e / kTcRows, r = e % kTcRows, R = r & 63;
      const int sidx = (R & 7) * 8 + ((R >> 4) & 3) * 2 + ((R >> 3) & 1);
      sc[e] = h2f(reinterpret_cast<const uint16_t*>(Us + (size_t)(r >> 6) * UB + kCodeBytes +
                                                    gq * kMetaBytesPerGroup)[sidx]);
    }
    // generic-proxy writes of A and B become visible to the tensor cores
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
      if (k + 2 < a.upr) issue_units(k + 2, s);  // the slot's units were read above
      const uint32_t aBase = smem_addr(As), bBase = smem_addr(Bs);
#pragma unroll
      for (int gq = 0; gq < G; ++gq)
#pragma unroll
        for (int i = 0; i < kMmaPerGroup; ++i) {
          const int kk = gq * kMmaPerGroup + i;  // K = 16 per instruction: two core matrices
          tc_mma(tmem + (uint32_t)((s * G + gq) * N), smem_desc(aBase + kk * 2 * kCoreK),
                 smem_desc(bBase + kk * 2 * kCoreK), instr_desc<N>(), i > 0);
        }
      tc_commit(&s_mbar[s]);
    }
  }
  for (int j = a.upr >= 2 ? a.upr - 2 : 0; j < a.upr; ++j) epilogue(j);
  if (!ok && lane == 0) atomicOr(a.status, ST_WAIT_TIMEOUT);
  // outputs: natural row order, [token][row]
  const int rbr = rb0 + (row >> 6);
  if (rbr < a.n_rb) {
    const int nat = natural_row(a.dims, rbr * kRowsPerBlock + (row & 63));
    if (nat >= 0)
#pragma unroll
      for (int c = 0; c < kHalf; ++c)
        if (n0 + c0 + c < a.S) a.y[(size_t)(n0 + c0 + c) * a.y_ld + nat] = tot[c];
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kCols) : "memory");
}

template <int N, int GPU>
cudaError_t launch_tc(const GemmArgs& a, cudaStream_t s) {
  using L = TcSmem<N, GPU>;
  const dim3 grid((a.n_rb + 1) / 2, (a.S + N - 1) / N);
  gemm_tc_kernel<N, GPU><<<grid, kTcThreads, L::kTotal, s>>>(a);
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

// Token tile: 128 for long prompts, smaller for short ones.
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
