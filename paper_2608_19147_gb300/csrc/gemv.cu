// Standalone launch of one W4A16 projection (the test export
// shard_debug_gemv, the allocation-free entry point and the LM head use it).
// The device code is the warp-level projection of gemv_core.cuh, the same
// code the whole-step kernel runs: kGemvWarps consumer warps and one producer
// warp per CTA, one CTA per SM.
#include "gemv_core.cuh"

namespace shard {
namespace {

constexpr int kW = kGemvWarps;  // consumer warps per CTA
constexpr int kBlock = (kW + (kSelfRefill ? 0 : 1)) * 32;
constexpr int kCtasPerSm = 1;

template <int GPU>
constexpr size_t smem_bytes() {
  return (size_t)kW * Geom<GPU>::kGemvSlots * Geom<GPU>::kUnitBytes +
         (size_t)2 * kW * Geom<GPU>::kGemvSlots * sizeof(uint64_t);
}

// 227 KB per CTA, less a margin for the kernel's static shared memory
static_assert(smem_bytes<1>() <= 225 * 1024 && smem_bytes<2>() <= 225 * 1024 && smem_bytes<4>() <= 225 * 1024,
              "standalone projection ring too large");

template <int NT, int GPU>
__global__ void __launch_bounds__(kBlock, 1) gemv_kernel(const __grid_constant__ GemvArgs a) {
  constexpr int kSlots = Geom<GPU>::kGemvSlots;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ OpDesc s_op[1];
  __shared__ GemvPhase s_gp;
  __shared__ WarpRing<GPU, kSlots> s_ring[kW];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t* rings = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)kW * kSlots * Geom<GPU>::kUnitBytes);
  uint64_t* empty = full + kW * kSlots;
  if (threadIdx.x == 0) {
    s_op[0] = OpDesc{a.units, a.n_rb, a.upr, 0};
    GemvPhase p{};
    p.act = a.act;
    p.act_ld = a.act_ld;
    p.M = a.M;
    p.status = a.status;
    p.ep = a.ep;
    s_gp = p;
    ring_init_barriers(full, empty, kW * kSlots);
  }
  __syncthreads();
  if (!kSelfRefill && warp == kW) {
    // the weights do not depend on the preceding kernel: start streaming them
    ring_producer<GPU, kSlots>(s_op, 1, blockIdx.x, gridDim.x, kW, rings, full, empty, a.status, 1u << 22, lane);
    return;
  }
  const int g = blockIdx.x * kW + warp, nw = gridDim.x * kW;
  {
    WarpRing<GPU, kSlots> r;
    r.ring = rings + (size_t)warp * kSlots * Geom<GPU>::kUnitBytes;
    r.full = full + warp * kSlots;
    r.empty = empty + warp * kSlots;
    r.n_used = 0;
    r.timed_out = false;
    if (kSelfRefill) r.start(s_op, 1, g, nw, lane);  // the weights do not depend on the preceding kernel
    if (lane == 0) s_ring[warp] = r;
    __syncwarp();
  }
  pdl_launch_dependents();
  pdl_wait();
  gemv_phase<NT, GPU, kSlots>(&s_ring[warp], &s_op[0], &s_gp, g, nw, lane);
  if (s_ring[warp].timed_out && lane == 0) atomicOr(a.status, ST_WAIT_TIMEOUT);
}

template <int NT, int GPU>
cudaError_t launch_t(const GemvArgs& a, int grid, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kBlock);
  cfg.dynamicSmemBytes = smem_bytes<GPU>();
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemv_kernel<NT, GPU>, a);
}

template <int NT, int GPU>
cudaError_t setup_t() {
  return cudaFuncSetAttribute(gemv_kernel<NT, GPU>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)smem_bytes<GPU>());
}

}  // namespace

cudaError_t gemv_setup() {
  cudaError_t e;
  if ((e = setup_t<1, 1>()) != cudaSuccess) return e;
  if ((e = setup_t<1, 2>()) != cudaSuccess) return e;
  if ((e = setup_t<1, 4>()) != cudaSuccess) return e;
  if ((e = setup_t<2, 1>()) != cudaSuccess) return e;
  if ((e = setup_t<2, 2>()) != cudaSuccess) return e;
  return setup_t<2, 4>();
}

int gemv_grid(int nt, int num_sms) {
  (void)nt;
  return kCtasPerSm * num_sms;
}

// the larger of the two kernels' consumer warp counts: index checks cover both
int gemv_warps_per_cta() { return kW > kCtaWarps ? kW : kCtaWarps; }

cudaError_t launch_gemv(const GemvArgs& a, int nt, int group, int grid, cudaStream_t s, bool pdl) {
  if (nt == 1) {
    if (group == 128) return launch_t<1, 1>(a, grid, s, pdl);
    if (group == 64) return launch_t<1, 2>(a, grid, s, pdl);
    if (group == 32) return launch_t<1, 4>(a, grid, s, pdl);
  } else if (nt == 2) {
    if (group == 128) return launch_t<2, 1>(a, grid, s, pdl);
    if (group == 64) return launch_t<2, 2>(a, grid, s, pdl);
    if (group == 32) return launch_t<2, 4>(a, grid, s, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace shard
