// sao_advantages_noalloc: the advantage scan for callers that cannot allocate
// device memory (see include/sao.h). Its scratch is a fixed array that lives
// in this library's device image on every GPU that loads it.
#include <stdint.h>

#include <mutex>
#include <vector>

#include "sao_common.cuh"
#include "sao_internal.h"

namespace sao {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;  // 16 MiB

// Shared by every call on a device; held until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

struct DeviceScratch {
  int device;
  void *ptr;
};
std::mutex g_scratch_mu;
std::vector<DeviceScratch> g_scratch_ptrs;

// Device address of g_noalloc_scratch on the current device. Host code only
// sees a host-side stand-in for the array's name, so the address comes from
// cudaGetSymbolAddress with the device current. Outside stream capture it is
// looked up again on every call (a device reset or a new primary context
// reloads the module and can move the array) and remembered per device;
// under capture the remembered address is used, so the first call on a
// device must come before any capture.
sao_status scratch_address(cudaStream_t stream, void **out) {
  int dev = 0;
  SAO_CUDA_TRY(cudaGetDevice(&dev));
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  SAO_CUDA_TRY(cudaStreamIsCapturing(stream, &cs));
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  DeviceScratch *known = nullptr;
  for (auto &d : g_scratch_ptrs)
    if (d.device == dev) known = &d;
  if (cs != cudaStreamCaptureStatusNone) {
    if (!known)
      return fail(SAO_ERR_INVALID_ARG,
                  "sao_advantages_noalloc: the first call on device %d is under stream capture; make one call "
                  "before capturing",
                  dev);
    *out = known->ptr;
    return SAO_OK;
  }
  void *p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess || p == nullptr)
    return fail(SAO_ERR_CUDA, "cudaGetSymbolAddress of the static scratch failed: %s", cudaGetErrorString(e));
  if (known)
    known->ptr = p;
  else
    g_scratch_ptrs.push_back({dev, p});
  *out = p;
  return SAO_OK;
}

}  // namespace
}  // namespace sao

using namespace sao;

extern "C" sao_status sao_advantages_noalloc(const float *values, const float *rewards, const uint8_t *loss_mask,
                                             const int32_t *cu_seqlens, int32_t B, int64_t N, float gamma,
                                             float lambda_policy, float lambda_critic, float len_adaptive_alpha,
                                             float *adv, float *ret, sao_stream_t stream) {
  if (N < 0 || N >= (int64_t(1) << 31)) return fail(SAO_ERR_SHAPE, "N = %lld out of range", (long long)N);
  if (B < 0) return fail(SAO_ERR_SHAPE, "B = %d < 0", B);
  const size_t need = kWsHeader + gae_ws_bytes(N, B);
  if (need > kNoAllocScratchBytes)
    return fail(SAO_ERR_SHAPE,
                "sao_advantages_noalloc: %lld tokens in %d trajectories need %zu bytes of scratch, more than its "
                "fixed %zu bytes; use sao_advantages with a workspace",
                (long long)N, B, need, kNoAllocScratchBytes);
  if (N == 0) return sao_advantages(values, rewards, loss_mask, cu_seqlens, B, N, gamma, lambda_policy,
                                    lambda_critic, len_adaptive_alpha, adv, ret, nullptr, 0, stream);
  void *scratch = nullptr;
  SAO_TRY(scratch_address(reinterpret_cast<cudaStream_t>(stream), &scratch));
  return sao_advantages(values, rewards, loss_mask, cu_seqlens, B, N, gamma, lambda_policy, lambda_critic,
                        len_adaptive_alpha, adv, ret, scratch, kNoAllocScratchBytes, stream);
}
