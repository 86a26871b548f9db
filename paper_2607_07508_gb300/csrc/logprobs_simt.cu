// fp32 path of the LM-head log-probs (Eq. 1-2) and their gradient, on CUDA
// cores with fp32 FMA (no tensor cores, so fp32 inputs keep fp32 products).
// Same chunked structure as the tensor-core path:
//   forward : 64x64 logit tiles -> per-(row, vocab tile) (max, sum-exp) partials
//             and the gathered logit of the sampled token, merged by
//             lse_merge_kernel;
//   backward: per vocabulary chunk, dZ tiles written to a [N, Vc] fp32 buffer,
//             then dH (+)= dZ W_chunk and dW_chunk (+)= dZ^T H.
#include <math.h>
#include <stdint.h>

#include "logprobs_common.cuh"
#include "sao_common.cuh"
#include "sao_internal.h"

namespace sao {
namespace {

constexpr int TM = 64, TN = 64, TK = 16;

// 64x64 tile of Z = H W^T for rows [m0, m0+64) and vocab [n0, n0+64); each
// thread (ty, tx) holds rows 4*ty..4*ty+3 and columns tx + 16*j.
__device__ __forceinline__ void logit_tile(const float *__restrict__ H, const float *__restrict__ W,
                                           int64_t N, int h, int V, int64_t m0, int n0, float acc[4][4]) {
  __shared__ float sA[TK][TM + 4];
  __shared__ float sB[TK][TN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < h; k0 += TK) {
    for (int e = threadIdx.x; e < TM * TK; e += 256) {
      const int r = e / TK, k = e % TK;
      const int64_t row = m0 + r;
      sA[k][r] = (row < N && k0 + k < h) ? H[row * h + k0 + k] : 0.f;
      const int col = n0 + r;
      sB[k][r] = (col < V && k0 + k < h) ? W[int64_t(col) * h + k0 + k] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < TK; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = sA[k][4 * ty + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = sB[k][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
}

__global__ void __launch_bounds__(256) simt_fwd_kernel(const float *H, const float *W, const int32_t *y,
                                                       const uint8_t *row_mask, int64_t N, int h, int V,
                                                       float2 *part, float *zy, unsigned int *err) {
  const int64_t m0 = int64_t(blockIdx.y) * TM;
  const int n0 = blockIdx.x * TN;
  float acc[4][4];
  logit_tile(H, W, N, h, V, m0, n0, acc);
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t row = m0 + 4 * ty + i;
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (n0 + tx + 16 * j < V) m = fmaxf(m, acc[i][j]);
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (n0 + tx + 16 * j < V) s += expf(acc[i][j] - m);
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (row < N) {
      const bool active = row_mask == nullptr || row_mask[row] != 0;
      if (tx == 0) part[int64_t(blockIdx.x) * N + row] = make_float2(m, s);
      if (active) {
        const int yy = y[row];
        if (yy >= 0 && yy < V) {
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (n0 + tx + 16 * j == yy) zy[row] = acc[i][j];
        }
      }
    }
  }
}

// dZ tile of chunk [v0, v0+Vc): dz = G (1[v==y] - exp(z - lse)).
__global__ void __launch_bounds__(256) simt_dz_kernel(const float *H, const float *W, const int32_t *y,
                                                      const float *lse, const float *G, int64_t N, int h,
                                                      int V, int v0, int Vc, float *dZ) {
  const int64_t m0 = int64_t(blockIdx.y) * TM;
  const int n0 = v0 + blockIdx.x * TN;
  float acc[4][4];
  logit_tile(H, W, N, h, V, m0, n0, acc);
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t row = m0 + 4 * ty + i;
    if (row >= N) continue;
    const float g = G[row], l = lse[row];
    const int yy = y[row];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int col = n0 + tx + 16 * j;
      if (col >= V || col >= v0 + Vc) continue;
      float d = 0.f;
      if (g != 0.f) d = g * ((col == yy ? 1.f : 0.f) - expf(acc[i][j] - l));
      dZ[row * Vc + (col - v0)] = d;
    }
  }
}

// C[M, Nn] (+)= A[M, K] B[K, Nn] with element strides (A: sam, sak; B: sbk, sbn).
__global__ void __launch_bounds__(256) simt_gemm_kernel(const float *A, int64_t sam, int64_t sak,
                                                        const float *B, int64_t sbk, int64_t sbn, float *C,
                                                        int64_t ldc, int64_t M, int64_t Nn, int64_t K,
                                                        int accumulate) {
  __shared__ float sA[TK][TM + 4];
  __shared__ float sB[TK][TN + 4];
  const int64_t m0 = int64_t(blockIdx.y) * TM, n0 = int64_t(blockIdx.x) * TN;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int64_t k0 = 0; k0 < K; k0 += TK) {
    for (int e = threadIdx.x; e < TM * TK; e += 256) {
      const int r = e / TK, k = e % TK;
      sA[k][r] = (m0 + r < M && k0 + k < K) ? A[(m0 + r) * sam + (k0 + k) * sak] : 0.f;
      sB[k][r] = (n0 + r < Nn && k0 + k < K) ? B[(k0 + k) * sbk + (n0 + r) * sbn] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < TK; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = sA[k][4 * ty + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = sB[k][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t r = m0 + 4 * ty + i, c = n0 + tx + 16 * j;
      if (r < M && c < Nn) {
        float *p = C + r * ldc + c;
        *p = accumulate ? *p + acc[i][j] : acc[i][j];
      }
    }
}

int simt_chunk(int64_t N, int V) {
  // fp32 dZ chunk under the dZ budget, a multiple of the 64-wide tile
  int64_t vc = int64_t(dz_budget() / (size_t(N > 0 ? N : 1) * sizeof(float)));
  vc = (vc / TN) * TN;
  if (vc < TN) vc = TN;
  if (vc > V) vc = ((V + TN - 1) / TN) * TN;
  return int(vc);
}

}  // namespace

size_t simt_ws_bytes(int64_t N, int32_t h, int32_t V) {
  (void)h;
  const int64_t nvt = (V + TN - 1) / TN;
  const size_t fwd = round256(sizeof(float2) * size_t(nvt) * size_t(N)) + round256(sizeof(float) * size_t(N));
  const size_t bwd = round256(sizeof(float) * size_t(N) * size_t(simt_chunk(N, V)));
  return fwd > bwd ? fwd : bwd;
}

sao_status simt_fwd(const float *H, const float *W, const int32_t *y, const uint8_t *row_mask, int64_t N,
                    int32_t h, int32_t V, float *logp, float *lse, unsigned int *err, void *ws, size_t ws_bytes,
                    cudaStream_t s) {
  const int nvt = (V + TN - 1) / TN;
  Carver c(ws, ws_bytes);
  float2 *part = c.take<float2>(size_t(nvt) * size_t(N));
  float *zy = c.take<float>(size_t(N));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the fp32 log-prob forward");
  if ((N + TM - 1) / TM > 65535) return fail(SAO_ERR_SHAPE, "fp32 path supports at most %d tokens", 65535 * TM);
  dim3 grid(nvt, unsigned((N + TM - 1) / TM));
  int slot = launch_begin("simt_logits_fwd", s);
  simt_fwd_kernel<<<grid, 256, 0, s>>>(H, W, y, row_mask, N, h, V, part, zy, err);
  SAO_TRY(launch_end(slot, s));
  return lse_merge_launch(part, nvt, zy, y, row_mask, nullptr, N, V, logp, lse, err, s);
}

sao_status simt_bwd(const float *H, const float *W, const int32_t *y, const float *lse, const float *G,
                    int64_t N, int32_t h, int32_t V, float *dH, float *dW, int accumulate, void *ws,
                    size_t ws_bytes, cudaStream_t s) {
  const int Vc = simt_chunk(N, V);
  Carver c(ws, ws_bytes);
  float *dZ = c.take<float>(size_t(N) * size_t(Vc));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the fp32 log-prob backward");
  if ((N + TM - 1) / TM > 65535 || (int64_t(h) + TM - 1) / TM > 65535)
    return fail(SAO_ERR_SHAPE, "fp32 path size limit exceeded");
  for (int v0 = 0; v0 < V; v0 += Vc) {
    const int vc = (V - v0) < Vc ? (V - v0) : Vc;
    {
      dim3 grid((vc + TN - 1) / TN, unsigned((N + TM - 1) / TM));
      int slot = launch_begin("simt_dlogits", s);
      simt_dz_kernel<<<grid, 256, 0, s>>>(H, W, y, lse, G, N, h, V, v0, Vc, dZ);
      SAO_TRY(launch_end(slot, s));
    }
    {  // dH[N, h] (+)= dZ[N, vc] W[v0:v0+vc, h]
      dim3 grid((h + TN - 1) / TN, unsigned((N + TM - 1) / TM));
      int slot = launch_begin("simt_dH_gemm", s);
      simt_gemm_kernel<<<grid, 256, 0, s>>>(dZ, Vc, 1, W + int64_t(v0) * h, h, 1, dH, h, N, h, vc, v0 > 0);
      SAO_TRY(launch_end(slot, s));
    }
    {  // dW[v0:v0+vc, h] (+)= dZ^T[vc, N] H[N, h]
      dim3 grid((h + TN - 1) / TN, unsigned((vc + TM - 1) / TM));
      int slot = launch_begin("simt_dW_gemm", s);
      simt_gemm_kernel<<<grid, 256, 0, s>>>(dZ, 1, Vc, H, h, 1, dW + int64_t(v0) * h, h, vc, h, N, accumulate);
      SAO_TRY(launch_end(slot, s));
    }
  }
  return SAO_OK;
}

}  // namespace sao
