// shard_gemv_noalloc: the projection GEMV with its scratch in a fixed,
// file-scope device array instead of memory the library allocates.
//
// Who needs it: code that must not allocate device memory while it runs --
// for example a caller inside a memory pool that forbids outside
// cudaMalloc/cudaFree (a serving runtime that pre-reserves all of HBM), code
// running while another thread holds the allocator, or a latency-critical
// loop where an allocation's implicit device synchronisation is not
// allowed.  Such a caller still owns its inputs and outputs; only the
// kernel's scratch (the fixed-point row sums of split row-blocks, their
// arrival counts and a zero-padded copy of the activations) moves into the
// static array below, which every GPU that loads the library holds until
// exit.
#include <algorithm>
#include <cstdio>

#include "../../include/shard.h"
#include "../../include/shard_debug.h"
#include "common.cuh"

namespace shard {
namespace {

// 4 MiB: the arrival counts of the op's row-blocks, then the row sums
// (16 rows of up to 57344 int64 fit for M <= 8), then the padded
// activations.  Every part is cleared by the call before its kernel runs.
constexpr size_t kNoAllocScratchBytes = 4u << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
void* g_scratch_addr[kMaxDevices] = {};  // per-device address of g_noalloc_scratch

}  // namespace

// Shard fields the entry point needs, and the thread's last-error message
// (both defined in shard_api.cu).
struct NoAllocView {
  const PackedOp* op;
  int group, grid_nt1, grid_nt2, device, rows;
  int* status;  // the shard's device status word (shard_sync_status reports it)
};
int shard_noalloc_view(shard_t sh, int layer, int op, NoAllocView* v);
int shard_noalloc_fail(int code, const char* msg);

}  // namespace shard

using namespace shard;

namespace {
thread_local char g_msg[256];
size_t align256(size_t v) { return (v + 255) / 256 * 256; }
}

extern "C" {

// Declared in include/shard.h.
int shard_gemv_noalloc(shard_t sh, int layer, int op, const uint16_t* x, int M, float* y, int y_ld,
                       void* cuda_stream) {
  NoAllocView v{};
  int rc = shard_noalloc_view(sh, layer, op, &v);
  if (rc) return rc;
  if (!x || !y || M < 1 || M > SHARD_MAX_TOKENS) {
    snprintf(g_msg, sizeof(g_msg), "shard_gemv_noalloc: null pointer or M outside [1, %d]", SHARD_MAX_TOKENS);
    return shard_noalloc_fail(SHARD_EINVAL, g_msg);
  }
  const PackedOp& p = *v.op;
  const int nt = M <= 8 ? 1 : 2;
  // Scratch layout: [counts | sums | activations], 256-byte aligned parts.
  const size_t cnt_bytes = align256(sizeof(int) * (size_t)p.n_rb);
  const size_t acc_ld = (size_t)p.n_rb * kRowsPerBlock;
  const size_t acc_bytes = align256(sizeof(long long) * acc_ld * M);
  const size_t act_bytes = (size_t)M * p.Kp * sizeof(uint16_t);
  if (cnt_bytes + acc_bytes + act_bytes > kNoAllocScratchBytes) {
    snprintf(g_msg, sizeof(g_msg),
             "shard_gemv_noalloc: needs %zu bytes of scratch for M=%d, %d rows and K=%d; the fixed array has %zu",
             cnt_bytes + acc_bytes + act_bytes, M, v.rows, p.K, kNoAllocScratchBytes);
    return shard_noalloc_fail(SHARD_ECAPACITY, g_msg);
  }
  if (y_ld < v.rows) {
    snprintf(g_msg, sizeof(g_msg), "shard_gemv_noalloc: y_ld %d < the op's %d rows", y_ld, v.rows);
    return shard_noalloc_fail(SHARD_EINVAL, g_msg);
  }
  cudaError_t e = cudaSetDevice(v.device);
  if (e != cudaSuccess || v.device < 0 || v.device >= kMaxDevices) {
    snprintf(g_msg, sizeof(g_msg), "shard_gemv_noalloc: cannot select device %d", v.device);
    return shard_noalloc_fail(SHARD_ECUDA, g_msg);
  }
  // Set-up, once per device, with that device current: the host-side name of
  // the array is not a device address, so resolve it.
  if (!g_scratch_addr[v.device]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || !ptr) {
      snprintf(g_msg, sizeof(g_msg), "shard_gemv_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
      return shard_noalloc_fail(SHARD_ECUDA, g_msg);
    }
    g_scratch_addr[v.device] = ptr;
  }
  unsigned char* base = static_cast<unsigned char*>(g_scratch_addr[v.device]);
  int* cnt = reinterpret_cast<int*>(base);
  long long* acc = reinterpret_cast<long long*>(base + cnt_bytes);
  uint16_t* act = reinterpret_cast<uint16_t*>(base + cnt_bytes + acc_bytes);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  // The array keeps the previous call's contents: clear the counts, the sums
  // and the activation padding (a completed call leaves counts and sums zero,
  // one that gave up may not).
  e = cudaMemsetAsync(base, 0, cnt_bytes + acc_bytes + act_bytes, s);
  if (e == cudaSuccess)
    e = cudaMemcpy2DAsync(act, sizeof(uint16_t) * p.Kp, x, sizeof(uint16_t) * p.K, sizeof(uint16_t) * p.K, M,
                          cudaMemcpyDeviceToDevice, s);
  if (e != cudaSuccess) {
    snprintf(g_msg, sizeof(g_msg), "shard_gemv_noalloc: %s", cudaGetErrorString(e));
    return shard_noalloc_fail(SHARD_ECUDA, g_msg);
  }
  GemvArgs g{};
  g.units = p.units;
  g.n_rb = p.n_rb;
  g.upr = p.upr;
  g.act = act;
  g.act_ld = p.Kp;
  g.M = M;
  g.status = v.status;
  g.ep.kind = EPI_STORE;
  g.ep.dims = p.dims;
  g.ep.acc = acc;
  g.ep.acc_ld = static_cast<int>(acc_ld);
  g.ep.cnt = cnt;
  g.ep.y = y;
  g.ep.y_ld = y_ld;
  const int grid = std::min<long long>(nt == 1 ? v.grid_nt1 : v.grid_nt2, (long long)p.n_rb * p.upr);
  e = launch_gemv(g, nt, v.group, grid, s, false);
  if (e != cudaSuccess) {
    snprintf(g_msg, sizeof(g_msg), "shard_gemv_noalloc: launch failed: %s", cudaGetErrorString(e));
    return shard_noalloc_fail(SHARD_ECUDA, g_msg);
  }
  return SHARD_OK;
}

}  // extern "C"
