// Row compaction for the tensor-core log-prob path: the forward skips rows
// whose row_mask is 0 and the backward skips rows whose incoming gradient is
// 0 (observation and masked tokens), by running the GEMMs on a compacted,
// zero-padded copy of the active rows of H. The active count stays on the
// device; the persistent GEMM kernels read it at start-up.
#include <cuda_bf16.h>
#include <stdint.h>

#include "rows.cuh"
#include "sao_common.cuh"

namespace sao {
namespace {

constexpr int kScanThreads = 256;
constexpr int kRowsPerBlock = 4096;  // 16 rows per thread

__device__ __forceinline__ bool row_active(const uint8_t *mask, const float *g, int64_t t) {
  return mask ? (mask[t] != 0) : (g[t] != 0.f);
}

// Active rows per 4096-row block.
__global__ void __launch_bounds__(kScanThreads) compact_count_kernel(const uint8_t *mask, const float *g,
                                                                     int64_t N, int *block_count) {
  const int64_t r0 = int64_t(blockIdx.x) * kRowsPerBlock;
  int c = 0;
  for (int i = threadIdx.x; i < kRowsPerBlock; i += kScanThreads) {
    const int64_t t = r0 + i;
    if (t < N) c += row_active(mask, g, t);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  __shared__ int sh[kScanThreads / 32];
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int w = 0; w < kScanThreads / 32; ++w) s += sh[w];
    block_count[blockIdx.x] = s;
  }
}

// Exclusive scan of the block counts (one CTA) and the total.
__global__ void __launch_bounds__(1024) compact_scan_kernel(int *block_count, int nblocks, int *total) {
  __shared__ int sh[1024];
  const int per = (nblocks + 1023) / 1024;
  const int b0 = threadIdx.x * per;
  int s = 0;
  for (int i = 0; i < per; ++i)
    if (b0 + i < nblocks) s += block_count[b0 + i];
  sh[threadIdx.x] = s;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    const int v = threadIdx.x >= o ? sh[threadIdx.x - o] : 0;
    __syncthreads();
    sh[threadIdx.x] += v;
    __syncthreads();
  }
  int run = threadIdx.x ? sh[threadIdx.x - 1] : 0;
  for (int i = 0; i < per; ++i)
    if (b0 + i < nblocks) {
      const int c = block_count[b0 + i];
      block_count[b0 + i] = run;
      run += c;
    }
  if (threadIdx.x == 1023) *total = sh[1023];
}

// idx[compact] = row and pos[row] = compact (or -1), in row order.
__global__ void __launch_bounds__(kScanThreads) compact_scatter_kernel(const uint8_t *mask, const float *g,
                                                                       int64_t N, const int *block_offset,
                                                                       int *idx, int *pos) {
  const int64_t r0 = int64_t(blockIdx.x) * kRowsPerBlock;
  __shared__ int sh[kScanThreads / 32];
  __shared__ int base;
  if (threadIdx.x == 0) base = block_offset[blockIdx.x];
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i0 = 0; i0 < kRowsPerBlock; i0 += kScanThreads) {
    const int64_t t = r0 + i0 + threadIdx.x;
    const bool a = t < N && row_active(mask, g, t);
    const unsigned bal = __ballot_sync(0xffffffffu, a);
    if (lane == 0) sh[warp] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int w = 0; w < kScanThreads / 32; ++w) {
      before += (w < warp) ? sh[w] : 0;
      total += sh[w];
    }
    const int off = base + before + __popc(bal & ((1u << lane) - 1u));
    if (t < N) {
      pos[t] = a ? off : -1;
      if (a) idx[off] = int(t);
    }
    __syncthreads();
    if (threadIdx.x == 0) base += total;
    __syncthreads();
  }
}

// H_c[i] = H[idx[i]] for i < count; rows [count, round_up(count, 128)) = 0.
__global__ void gather_rows_kernel(const __nv_bfloat16 *H, int h, const int *idx, const int *count,
                                   __nv_bfloat16 *Hc, int64_t rows_cap) {
  const int n = *count;
  const int64_t pad = (int64_t(n) + 127) / 128 * 128;
  const int vec = h / 8;  // 16-byte vectors per row (h % 8 == 0)
  const int64_t total = (pad < rows_cap ? pad : rows_cap) * vec;
  for (int64_t e = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; e < total; e += int64_t(gridDim.x) * blockDim.x) {
    const int64_t i = e / vec;
    const int v = int(e - i * vec);
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (i < n) val = reinterpret_cast<const uint4 *>(H + int64_t(idx[i]) * h)[v];
    reinterpret_cast<uint4 *>(Hc + i * h)[v] = val;
  }
}

// dH[t] = bf16(acc[pos[t]]) for active rows; the others get 0.
__global__ void scatter_rows_f32_to_bf16_kernel(const float *acc, int h, const int *pos, int64_t N,
                                                __nv_bfloat16 *dH) {
  const int vec = h / 4;
  const int64_t total = N * vec;
  for (int64_t e = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; e < total; e += int64_t(gridDim.x) * blockDim.x) {
    const int64_t t = e / vec;
    const int v = int(e - t * vec);
    const int i = pos[t];
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i >= 0) x = reinterpret_cast<const float4 *>(acc + int64_t(i) * h)[v];
    const __nv_bfloat162 a = __floats2bfloat162_rn(x.x, x.y), b = __floats2bfloat162_rn(x.z, x.w);
    uint2 w;
    w.x = *reinterpret_cast<const uint32_t *>(&a);
    w.y = *reinterpret_cast<const uint32_t *>(&b);
    reinterpret_cast<uint2 *>(dH + t * h)[v] = w;
  }
}

// dH[idx[i]] = bf16(acc[i]) for the active rows i < count only.
__global__ void scatter_active_f32_to_bf16_kernel(const float *acc, int h, const int *idx, const int *count,
                                                  __nv_bfloat16 *dH) {
  const int vec = h / 4;
  const int64_t total = int64_t(*count) * vec;
  for (int64_t e = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; e < total; e += int64_t(gridDim.x) * blockDim.x) {
    const int64_t i = e / vec;
    const int v = int(e - i * vec);
    const float4 x = reinterpret_cast<const float4 *>(acc + i * h)[v];
    const __nv_bfloat162 a = __floats2bfloat162_rn(x.x, x.y), b = __floats2bfloat162_rn(x.z, x.w);
    uint2 w;
    w.x = *reinterpret_cast<const uint32_t *>(&a);
    w.y = *reinterpret_cast<const uint32_t *>(&b);
    reinterpret_cast<uint2 *>(dH + int64_t(idx[i]) * h)[v] = w;
  }
}

}  // namespace

size_t compact_ws_bytes(int64_t N, int32_t h) {
  const int64_t nblocks = (N + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t cap = (N + 127) / 128 * 128;
  return round256(sizeof(int) * (nblocks + 1)) + round256(sizeof(int) * 4) + round256(sizeof(int) * N) * 2 +
         round256(size_t(cap) * size_t(h) * 2);
}

sao_status compact_rows(const uint8_t *mask, const float *g, int64_t N, const __nv_bfloat16 *H, int32_t h,
                        CompactRows *out, Carver &c, cudaStream_t s) {
  const int64_t nblocks = (N + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t cap = (N + 127) / 128 * 128;
  int *block = c.take<int>(size_t(nblocks) + 1);
  int *count = c.take<int>(4);
  out->idx = c.take<int>(size_t(N));
  out->pos = c.take<int>(size_t(N));
  out->Hc = c.take<__nv_bfloat16>(size_t(cap) * size_t(h));
  out->count = count;
  out->cap = cap;
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for row compaction");
  int slot = launch_begin("compact_rows", s);
  compact_count_kernel<<<unsigned(nblocks), kScanThreads, 0, s>>>(mask, g, N, block);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("compact_rows", s);
  compact_scan_kernel<<<1, 1024, 0, s>>>(block, int(nblocks), count);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("compact_rows", s);
  compact_scatter_kernel<<<unsigned(nblocks), kScanThreads, 0, s>>>(mask, g, N, block, out->idx, out->pos);
  SAO_TRY(launch_end(slot, s));
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  slot = launch_begin("gather_rows", s);
  gather_rows_kernel<<<unsigned(di.sm_count * 8), 256, 0, s>>>(H, h, out->idx, count, out->Hc, cap);
  return launch_end(slot, s);
}

sao_status scatter_rows_to_bf16(const float *acc, int32_t h, const int *pos, const int *idx, const int *count,
                                int64_t N, __nv_bfloat16 *dH, bool all_rows, cudaStream_t s) {
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  int slot = launch_begin("scatter_dH", s);
  if (all_rows)
    scatter_rows_f32_to_bf16_kernel<<<unsigned(di.sm_count * 8), 256, 0, s>>>(acc, h, pos, N, dH);
  else
    scatter_active_f32_to_bf16_kernel<<<unsigned(di.sm_count * 8), 256, 0, s>>>(acc, h, idx, count, dH);
  return launch_end(slot, s);
}

}  // namespace sao
