// W4A16 projection for many tokens on the 5th-generation tensor cores
// (tcgen05): Y[n][r] = sum_k W[r][k] x[n][k] for S tokens, W in the shard's
// unit stream (kernels.h).  Used where the token count makes the projection
// a dense contraction -- a prompt's prefill (Section 3.4: the stateful cache
// is filled by running the prompt through the stage) -- where the per-token
// GEMV of the decode step would stream every weight once per 16 tokens.
//
// One CTA (4 warps) computes a tile of 128 weight rows (two 64-row blocks)
// by N tokens, walking K one 128-input unit at a time:
//   1. thread 0 bulk-copies the tile's two units (codes, scales, zero points)
//      into shared memory (TMA, non-tensor; mbarrier completion);
//   2. the CTA stages the N x 128 token tile into shared memory in the
//      canonical K-major layout without swizzle (8-row x 16-byte core
//      matrices: element (row, k) at (row/8)*2048 + (k/8)*128 + (row%8)*16
//      + (k%8)*2 bytes), and dequantises the weights into the same layout as
//      exact fp16 (q - z) -- the per-group fp16 scale is applied later in
//      fp32, so no rounding is added to the W4A16 arithmetic;
//   3. thread 0 issues tcgen05.mma (kind::f16, M = 128, N tokens, K = 16 per
//      instruction) with A and B read from shared memory through matrix
//      descriptors and the accumulator in tensor memory, one accumulator per
//      quantisation group, and commits them to an mbarrier;
//   4. every warp reads its 32 rows of each group's accumulator back
//      (tcgen05.ld), multiplies by the row's group scale and adds into fp32
//      registers.
// At the end each thread (one row) writes its N outputs.  Waits are bounded;
// a wait that runs out sets the status word.  The tensor memory is freed
// before the CTA exits.
#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kTcRows = 128;       // weight rows per CTA tile (two row-blocks)
constexpr int kTcThreads = 128;    // 4 warps: warp w owns rows 32w .. 32w + 31 of the tile
constexpr uint32_t kCoreK = 128;   // bytes between core matrices adjacent in K
constexpr uint32_t kCoreMN = 2048; // bytes between 8-row groups (16 core matrices of K)

template <int N, int GPU>
struct TcSmem {
  static constexpr size_t kUnit = Geom<GPU>::kUnitBytes;
  static constexpr size_t kUnits = 2 * kUnit;          // the tile's two units
  static constexpr size_t kA = (size_t)kTcRows * 256;  // 128 rows x 128 fp16
  static constexpr size_t kB = (size_t)N * 256;        // N tokens x 128 fp16
  static constexpr size_t kUnitsOff = 0;
  static constexpr size_t kAOff = (kUnits + 1023) / 1024 * 1024;
  static constexpr size_t kBOff = kAOff + kA;
  static constexpr size_t kTotal = kBOff + kB;
};

__device__ __forceinline__ uint32_t tmem_cols_for(int n) {
  uint32_t c = 32;
  while (c < (uint32_t)n) c <<= 1;
  return c;
}

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

__device__ __forceinline__ uint32_t a_off(int row, int k) {
  return (uint32_t)(row >> 3) * kCoreMN + (uint32_t)(k >> 3) * kCoreK + (uint32_t)(row & 7) * 16u + (uint32_t)(k & 7) * 2u;
}

template <int N, int GPU>
__global__ void __launch_bounds__(kTcThreads, 1) gemm_tc_kernel(const __grid_constant__ GemmArgs a) {
  using L = TcSmem<N, GPU>;
  constexpr int UB = Geom<GPU>::kUnitBytes;
  constexpr int G = GPU;                       // quantisation groups per unit
  constexpr int kMmaPerGroup = 8 / GPU;        // K = 16 per instruction
  constexpr uint32_t kCols = (uint32_t)(G * N) <= 32 ? 32u : (uint32_t)(G * N) <= 64 ? 64u
                             : (uint32_t)(G * N) <= 128 ? 128u : (uint32_t)(G * N) <= 256 ? 256u : 512u;
  static_assert(G * N <= 512, "accumulators exceed tensor memory");
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ uint64_t s_bar_units, s_bar_mma;
  __shared__ uint32_t s_tmem;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb0 = 2 * blockIdx.x;              // the tile's first row-block
  const int n0 = blockIdx.y * N;               // the tile's first token
  uint8_t* units = smem + L::kUnitsOff;
  uint8_t* As = smem + L::kAOff;
  uint8_t* Bs = smem + L::kBOff;
  if (tid == 0) {
    mbar_init(&s_bar_units, 1);
    mbar_init(&s_bar_mma, 1);
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
  const int row = 32 * warp + lane;            // this thread's row of the tile (its tensor-memory lane)
  const int rbr = rb0 + (row >> 6);            // its row-block
  const int R = row & 63;                      // row within the row-block
  float tot[N];
#pragma unroll
  for (int c = 0; c < N; ++c) tot[c] = 0.f;
  bool ok = true;
  uint32_t phase = 0;
  for (int ku = 0; ku < a.upr; ++ku) {
    // 1. the tile's two units
    if (tid == 0) {
      mbar_arrive_expect_tx(&s_bar_units, 2 * UB);
      for (int u = 0; u < 2; ++u) {
        const int rb = rb0 + u < a.n_rb ? rb0 + u : rb0;  // a missing second block repeats the first (unused)
        bulk_g2s(units + (size_t)u * UB, a.units + ((size_t)rb * a.upr + ku) * UB, UB, &s_bar_units);
      }
    }
    // 2a. the token tile: N tokens x 128 inputs, 16-byte pieces
    for (int e = tid; e < N * 16; e += kTcThreads) {
      const int n = e >> 4, kc = e & 15;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (n0 + n < a.S) v = __ldcg(reinterpret_cast<const uint4*>(a.act + (size_t)(n0 + n) * a.act_ld + ku * kUnitK + 8 * kc));
      *reinterpret_cast<uint4*>(Bs + a_off(n, 8 * kc)) = v;
    }
    if (ok && !mbar_wait(&s_bar_units, phase)) ok = false;
    // 2b. dequantise: word (ft, l, j) of unit u holds rows 16 rt + gid (+8) at
    //     inputs k0 .. k0 + 3 (kernels.h); q - z exactly, as fp16
    for (int e = tid; e < 2 * (kCodeBytes / 4); e += kTcThreads) {
      const int u = e / (kCodeBytes / 4), wi = e % (kCodeBytes / 4);
      const int ft = wi >> 7, l = (wi >> 2) & 31, j = wi & 3;
      const int kc = ft >> 2, rt = ft & 3, gid = l >> 2, tig = l & 3;
      const int k0 = 64 * kc + 32 * (j >> 1) + 8 * tig + 4 * (j & 1);
      const uint8_t* U = units + (size_t)u * UB;
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
    // generic-proxy writes of A and B become visible to the tensor cores
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // 3. one accumulator per quantisation group
    if (tid == 0) {
      const uint32_t aBase = smem_addr(As), bBase = smem_addr(Bs);
#pragma unroll
      for (int gq = 0; gq < G; ++gq)
#pragma unroll
        for (int i = 0; i < kMmaPerGroup; ++i) {
          const int kk = gq * kMmaPerGroup + i;  // K = 16 per instruction: two core matrices
          tc_mma(tmem + (uint32_t)(gq * N), smem_desc(aBase + kk * 2 * kCoreK), smem_desc(bBase + kk * 2 * kCoreK),
                 instr_desc<N>(), i > 0);
        }
      tc_commit(&s_bar_mma);
    }
    if (ok && !mbar_wait(&s_bar_mma, phase)) ok = false;
    tc_fence_after();
    // 4. scale and add
    const uint8_t* Urow = units + (size_t)(row >> 6) * UB;
    const int sidx = (R & 7) * 8 + ((R >> 4) & 3) * 2 + ((R >> 3) & 1);
#pragma unroll
    for (int gq = 0; gq < G; ++gq) {
      const float s = h2f(reinterpret_cast<const uint16_t*>(Urow + kCodeBytes + gq * kMetaBytesPerGroup)[sidx]);
#pragma unroll
      for (int c0 = 0; c0 < N; c0 += 32) {
        float v[32];
        tc_ld32(tmem + ((uint32_t)(32 * warp) << 16) + (uint32_t)(gq * N + c0), v);
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (c0 + c < N) tot[c0 + c] = fmaf(s, v[c], tot[c0 + c]);
      }
    }
    tc_fence_before();
    __syncthreads();  // units, A, B and the accumulators are free for the next unit
    tc_fence_after();
    phase ^= 1;
  }
  if (!ok && lane == 0) atomicOr(a.status, ST_WAIT_TIMEOUT);
  // outputs: natural row order, [token][row]
  if (rbr < a.n_rb) {
    const int nat = natural_row(a.dims, rbr * kRowsPerBlock + R);
    if (nat >= 0)
#pragma unroll
      for (int c = 0; c < N; ++c)
        if (n0 + c < a.S) a.y[(size_t)(n0 + c) * a.y_ld + nat] = tot[c];
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
#define SETUP(N)                                               \
  if ((e = setup_tc<N, 1>()) != cudaSuccess) return e;         \
  if ((e = setup_tc<N, 2>()) != cudaSuccess) return e;         \
  if ((e = setup_tc<N, 4>()) != cudaSuccess) return e;
  SETUP(32)
  SETUP(64)
  SETUP(128)
#undef SETUP
  return cudaSuccess;
}

// Token tile: 128 for long prompts, smaller for short ones.
int gemm_tc_tile(int S) { return S > 64 ? 128 : S > 32 ? 64 : 32; }

cudaError_t launch_gemm_tc(const GemmArgs& a, int group, cudaStream_t s) {
  const int N = gemm_tc_tile(a.S);
#define L(NN)                                                  \
  if (N == NN) {                                               \
    if (group == 128) return launch_tc<NN, 1>(a, s);           \
    if (group == 64) return launch_tc<NN, 2>(a, s);            \
    if (group == 32) return launch_tc<NN, 4>(a, s);            \
  }
  L(32)
  L(64)
  L(128)
#undef L
  return cudaErrorInvalidValue;
}

}  // namespace shard
