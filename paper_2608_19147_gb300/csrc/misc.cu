// Weight repacking and KV-pool utilities.
#include "common.cuh"

namespace shard {
namespace {

// ---------------------------------------------------------------------------
// Repacking into the unit stream (see kernels.h for the layout).
// ---------------------------------------------------------------------------
struct SrcView {
  RepackSrc s;
  int K, group, G;
  __device__ int code(int src, int row, int k) const {
    return (s.codes[src][(size_t)row * ((K + 1) / 2) + (k >> 1)] >> (4 * (k & 1))) & 15;
  }
  __device__ int zero(int src, int row, int gi) const {
    return (s.zeros[src][(size_t)row * ((G + 1) / 2) + (gi >> 1)] >> (4 * (gi & 1))) & 15;
  }
  __device__ uint16_t scale(int src, int row, int gi) const { return s.scales[src][(size_t)row * G + gi]; }
  // Code for GPU row entry `rm` (rowmap value) and input k, with padding.
  __device__ uint32_t nib(int rm, int k) const {
    if (rm < 0) return 0;
    const int src = rm >> 24, row = rm & 0xFFFFFF;
    if (k < K) return static_cast<uint32_t>(code(src, row, k));
    const int gi = k / group;
    return gi < G ? static_cast<uint32_t>(zero(src, row, gi)) : 0u;
  }
};

__global__ void repack_codes_kernel(PackedOp op, const int* __restrict__ rowmap, SrcView v) {
  const size_t n_words = (size_t)op.n_rb * op.upr * (kCodeBytes / 4);
  for (size_t wi = blockIdx.x * (size_t)blockDim.x + threadIdx.x; wi < n_words; wi += (size_t)gridDim.x * blockDim.x) {
    const size_t unit = wi / (kCodeBytes / 4);
    const int wu = static_cast<int>(wi % (kCodeBytes / 4));
    const int ft = wu / 128, lane = (wu % 128) / 4, j = wu % 4;
    const int kc = ft / 4, rt = ft % 4;
    const int rb = static_cast<int>(unit / op.upr), ku = static_cast<int>(unit % op.upr);
    const int gid = lane / 4, tig = lane % 4, h = j / 2, jj = j % 2;
    const int k0 = ku * kUnitK + kc * 64 + 32 * h + 8 * tig + 4 * jj;
    const int rlo = rb * kRowsPerBlock + rt * 16 + gid, rhi = rlo + 8;
    const int ml = rowmap[rlo], mh = rowmap[rhi];
    const uint32_t w = v.nib(ml, k0) | (v.nib(ml, k0 + 1) << 16) | (v.nib(mh, k0) << 4) | (v.nib(mh, k0 + 1) << 20) |
                       (v.nib(ml, k0 + 2) << 8) | (v.nib(ml, k0 + 3) << 24) | (v.nib(mh, k0 + 2) << 12) |
                       (v.nib(mh, k0 + 3) << 28);
    *reinterpret_cast<uint32_t*>(op.units + unit * op.unit_bytes + ft * 512 + lane * 16 + j * 4) = w;
  }
}

__global__ void repack_meta_kernel(PackedOp op, const int* __restrict__ rowmap, SrcView v) {
  const int gpu = kUnitK / op.group;
  const size_t n = (size_t)op.n_rb * op.upr * gpu * 64;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const size_t unit = e / (gpu * 64);
    const int gu = static_cast<int>((e / 64) % gpu), idx = static_cast<int>(e % 64);
    const int gid = idx / 8, rt = (idx % 8) / 2, hl = idx % 2;
    const int rb = static_cast<int>(unit / op.upr), ku = static_cast<int>(unit % op.upr);
    const int R = rb * kRowsPerBlock + rt * 16 + gid + 8 * hl;
    const int gi = ku * gpu + gu;
    const int rm = rowmap[R];
    uint16_t s = 0;
    uint8_t z = 0;
    if (rm >= 0 && gi < v.G) {
      s = v.scale(rm >> 24, rm & 0xFFFFFF, gi);
      z = static_cast<uint8_t>(v.zero(rm >> 24, rm & 0xFFFFFF, gi));
    }
    uint8_t* meta = op.units + unit * op.unit_bytes + kCodeBytes + gu * kMetaBytesPerGroup;
    reinterpret_cast<uint16_t*>(meta)[idx] = s;
    meta[128 + idx] = hl ? static_cast<uint8_t>(z << 4) : z;  // upper rows: 16 z (see kernels.h)
  }
}

// Reads the unit stream back into natural order: out[n][k] = (q - z) * s.
__global__ void unpack_kernel(PackedOp op, float* out, int ld) {
  const size_t rows = (size_t)op.n_rb * kRowsPerBlock;
  const size_t n = rows * op.K;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
    const int R = static_cast<int>(e / op.K), k = static_cast<int>(e % op.K);
    const int nat = natural_row(op.dims, R);
    if (nat < 0) continue;
    const int rb = R / kRowsPerBlock, rt = (R % kRowsPerBlock) / 16, r16 = R % 16, gid = r16 % 8, hl = r16 / 8;
    const int ku = k / kUnitK, kk = k % kUnitK;
    const int kc = kk / 64, h = (kk % 64) / 32, tig = (kk % 32) / 8, jj = (kk % 8) / 4, i = kk % 4;
    const int j = 2 * h + jj, lane = gid * 4 + tig;
    const uint8_t* unit = op.units + ((size_t)rb * op.upr + ku) * op.unit_bytes;
    const uint32_t w = *reinterpret_cast<const uint32_t*>(unit + (kc * 4 + rt) * 512 + lane * 16 + j * 4);
    const int p = (i < 2 ? 0 : 2) + hl;
    const int q = (w >> (4 * p + 16 * (i & 1))) & 15;
    const int gu = kk / op.group;
    const uint8_t* meta = unit + kCodeBytes + gu * kMetaBytesPerGroup;
    const int idx = gid * 8 + rt * 2 + hl;
    const float s = h2f(reinterpret_cast<const uint16_t*>(meta)[idx]);
    const int z = hl ? meta[128 + idx] >> 4 : meta[128 + idx];
    out[(size_t)nat * ld + k] = static_cast<float>(q - z) * s;
  }
}

// ---------------------------------------------------------------------------
// KV-pool utilities.  Pool layout per layer: [n_rows][Hkv][cap][d] fp16; a
// slot id is phys_row * cap + position.
// ---------------------------------------------------------------------------
__global__ void kv_gather_kernel(const uint16_t* pool, int n_layers, size_t layer_stride, int Hkv, int cap, int d,
                                 const int* slots, int n, uint16_t* out) {
  const size_t total = (size_t)n_layers * n * Hkv * d;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total; e += (size_t)gridDim.x * blockDim.x) {
    const int t = static_cast<int>(e % d);
    const int h = static_cast<int>((e / d) % Hkv);
    const int j = static_cast<int>((e / ((size_t)d * Hkv)) % n);
    const int l = static_cast<int>(e / ((size_t)d * Hkv * n));
    const int slot = slots[j];
    const int prow = slot / cap, pos = slot % cap;
    out[e] = pool[l * layer_stride + (((size_t)prow * Hkv + h) * cap + pos) * d + t];
  }
}

__global__ void kv_scatter_kernel(uint16_t* pool, int n_layers, size_t layer_stride, int Hkv, int cap, int d, int row,
                                  const uint16_t* in, int n) {
  const size_t total = (size_t)n_layers * n * Hkv * d;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total; e += (size_t)gridDim.x * blockDim.x) {
    const int t = static_cast<int>(e % d);
    const int h = static_cast<int>((e / d) % Hkv);
    const int j = static_cast<int>((e / ((size_t)d * Hkv)) % n);
    const int l = static_cast<int>(e / ((size_t)d * Hkv * n));
    pool[l * layer_stride + (((size_t)row * Hkv + h) * cap + j) * d + t] = in[e];
  }
}

__global__ void fill_identity_kernel(int* bt, int n_rows, int cap, int row) {
  const size_t total = (size_t)(row < 0 ? n_rows : 1) * cap;
  for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < total; e += (size_t)gridDim.x * blockDim.x) {
    const int r = row < 0 ? static_cast<int>(e / cap) : row;
    const int j = static_cast<int>(e % cap);
    bt[(size_t)r * cap + j] = r * cap + j;
  }
}

int grid_for(size_t n, int threads) {
  size_t g = (n + threads - 1) / threads;
  if (g > 65535 * 4) g = 65535 * 4;
  return g < 1 ? 1 : static_cast<int>(g);
}

}  // namespace

cudaError_t launch_repack(const PackedOp& op, const int* rowmap, const RepackSrc& src, cudaStream_t s) {
  SrcView v{src, op.K, op.group, (op.K + op.group - 1) / op.group};
  const size_t n_words = (size_t)op.n_rb * op.upr * (kCodeBytes / 4);
  repack_codes_kernel<<<grid_for(n_words, 256), 256, 0, s>>>(op, rowmap, v);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t n_meta = (size_t)op.n_rb * op.upr * (kUnitK / op.group) * 64;
  repack_meta_kernel<<<grid_for(n_meta, 256), 256, 0, s>>>(op, rowmap, v);
  return cudaGetLastError();
}

cudaError_t launch_unpack(const PackedOp& op, float* out, int ld, cudaStream_t s) {
  const size_t n = (size_t)op.n_rb * kRowsPerBlock * op.K;
  unpack_kernel<<<grid_for(n, 256), 256, 0, s>>>(op, out, ld);
  return cudaGetLastError();
}

cudaError_t launch_kv_gather(const uint16_t* pool, int n_layers, size_t layer_stride, int Hkv, int cap, int d,
                             const int* slots, int n, uint16_t* out, cudaStream_t s) {
  const size_t total = (size_t)n_layers * n * Hkv * d;
  if (total == 0) return cudaSuccess;
  kv_gather_kernel<<<grid_for(total, 256), 256, 0, s>>>(pool, n_layers, layer_stride, Hkv, cap, d, slots, n, out);
  return cudaGetLastError();
}

cudaError_t launch_kv_scatter(uint16_t* pool, int n_layers, size_t layer_stride, int Hkv, int cap, int d, int row,
                              const uint16_t* in, int n, cudaStream_t s) {
  const size_t total = (size_t)n_layers * n * Hkv * d;
  if (total == 0) return cudaSuccess;
  kv_scatter_kernel<<<grid_for(total, 256), 256, 0, s>>>(pool, n_layers, layer_stride, Hkv, cap, d, row, in, n);
  return cudaGetLastError();
}

cudaError_t launch_fill_identity(int* bt, int n_rows, int cap, int row, cudaStream_t s) {
  const size_t total = (size_t)(row < 0 ? n_rows : 1) * cap;
  fill_identity_kernel<<<grid_for(total, 256), 256, 0, s>>>(bt, n_rows, cap, row);
  return cudaGetLastError();
}

}  // namespace shard
