// Shared host/device helpers of libsao: status handling, launch bookkeeping,
// the device error word and small device utilities.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/sao.h"

namespace sao {

// ----------------------------------------------------------------------------
// host side
// ----------------------------------------------------------------------------

// Records `msg` as the calling thread's last error and returns `st`.
sao_status fail(sao_status st, const char *fmt, ...);
const char *last_error();
void set_checked(int on);
void profile_enable(int on);
void profile_reset();
int profile_read(const char **names, int64_t *launches, double *total_ms, int cap);

// Wraps a CUDA runtime call: on failure records the error and returns SAO_ERR_CUDA.
#define SAO_CUDA_TRY(expr)                                                       \
  do {                                                                           \
    cudaError_t e_ = (expr);                                                     \
    if (e_ != cudaSuccess)                                                       \
      return ::sao::fail(SAO_ERR_CUDA, "%s: %s (%s:%d)", #expr,                  \
                         cudaGetErrorString(e_), __FILE__, __LINE__);            \
  } while (0)

#define SAO_TRY(expr)                                                            \
  do {                                                                           \
    sao_status s_ = (expr);                                                      \
    if (s_ != SAO_OK) return s_;                                                 \
  } while (0)

// Called after every kernel launch: picks up launch errors and, when kernel
// profiling is on, closes the event pair opened by launch_begin.
int launch_begin(const char *kind, cudaStream_t s);
sao_status launch_end(int slot, cudaStream_t s);

// Device properties of the current device (cached per device).
struct DeviceInfo {
  int device;
  int sm_count;
  int cc_major, cc_minor;
  size_t smem_optin;
};
sao_status device_info(DeviceInfo *out);

// Every workspace starts with a 256-byte header whose first word is the
// device error word of the calls that use it. begin_call clears it in checked
// mode; finish_call (checked mode) synchronises, reads and reports it.
constexpr size_t kWsHeader = 256;
sao_status begin_call(void *ws, cudaStream_t s);
sao_status finish_call(void *ws, cudaStream_t s);
bool checked_mode();

bool aligned16(const void *p);

// Workspace carving: hands out 256-byte aligned slices of the caller's buffer.
struct Carver {
  char *base;
  size_t cap;
  size_t off = 0;
  Carver(void *b, size_t c) : base(static_cast<char *>(b)), cap(c) {}
  template <class T>
  T *take(size_t count) {
    size_t bytes = (count * sizeof(T) + 255) & ~size_t(255);
    T *p = reinterpret_cast<T *>(base + off);
    off += bytes;
    return p;
  }
  bool ok() const { return off <= cap; }
};

inline size_t round256(size_t b) { return (b + 255) & ~size_t(255); }

// ----------------------------------------------------------------------------
// device side
// ----------------------------------------------------------------------------

// Kernels OR SAO_DEVERR_* bits into the workspace's error word.
__device__ __forceinline__ void raise_device_error(unsigned int *err, unsigned int bits) {
  atomicOr(err, bits);
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Every wait on another CTA or on an mbarrier gives up after this long (or
// after kSpinLimit polls), raises an error bit and lets the kernel finish.
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr uint32_t kSpinLimit = 1u << 28;

}  // namespace sao
