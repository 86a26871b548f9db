// Row compaction helpers of the tensor-core log-prob path (see rows.cu).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "sao_common.cuh"

namespace sao {

struct CompactRows {
  int *idx;            // [N] compact index -> original row
  int *pos;            // [N] original row -> compact index, or -1
  int *count;          // device scalar: number of active rows
  __nv_bfloat16 *Hc;   // [cap, h] active rows of H, zero-padded to a multiple of 128
  int64_t cap;         // rows allocated in Hc (N rounded up to 128)
};

size_t compact_ws_bytes(int64_t N, int32_t h);

// Active rows are those with mask[t] != 0 (mask given) or g[t] != 0.
sao_status compact_rows(const uint8_t *mask, const float *g, int64_t N, const __nv_bfloat16 *H, int32_t h,
                        CompactRows *out, Carver &c, cudaStream_t s);

// dH[t] = bf16(acc[pos[t]]) on the active rows; inactive rows get zeros when
// all_rows (a sweep over all N rows), else keep their contents (a sweep over
// the `*count` active rows idx[0..count) only).
sao_status scatter_rows_to_bf16(const float *acc, int32_t h, const int *pos, const int *idx, const int *count,
                                int64_t N, __nv_bfloat16 *dH, bool all_rows, cudaStream_t s);

}  // namespace sao
