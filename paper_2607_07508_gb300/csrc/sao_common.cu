// Host-side helpers of libsao: error strings, launch bookkeeping, kernel
// profiling events, device queries and checked mode.
#include <stdarg.h>
#include <stdio.h>

#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "sao_common.cuh"

namespace sao {

static thread_local char t_last_error[512] = "no error";
static std::atomic<int> g_checked{0};

sao_status fail(sao_status st, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(t_last_error, sizeof(t_last_error), fmt, ap);
  va_end(ap);
  return st;
}

const char *last_error() { return t_last_error; }
void set_checked(int on) { g_checked.store(on ? 1 : 0); }
bool checked_mode() { return g_checked.load() != 0; }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ---------------------------------------------------------------------------
// kernel profiling: one event pair per launch, summed per kernel kind
// ---------------------------------------------------------------------------
struct ProfRecord {
  const char *kind;
  cudaEvent_t start, stop;
};
struct ProfKind {
  const char *kind;
  int64_t launches;
  double ms;
};
static std::mutex g_prof_mu;
static std::atomic<int> g_prof_on{0};
static std::vector<ProfRecord> g_prof_pending;
static std::vector<cudaEvent_t> g_prof_pool;
static std::vector<ProfKind> g_prof_kinds;

void profile_enable(int on) { g_prof_on.store(on ? 1 : 0); }

static cudaEvent_t pool_get() {
  if (!g_prof_pool.empty()) {
    cudaEvent_t e = g_prof_pool.back();
    g_prof_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

static void drain_locked() {
  for (auto &r : g_prof_pending) {
    float ms = 0.f;
    cudaEventSynchronize(r.stop);
    cudaEventElapsedTime(&ms, r.start, r.stop);
    bool found = false;
    for (auto &k : g_prof_kinds)
      if (k.kind == r.kind) {
        k.launches++;
        k.ms += ms;
        found = true;
        break;
      }
    if (!found) g_prof_kinds.push_back({r.kind, 1, ms});
    g_prof_pool.push_back(r.start);
    g_prof_pool.push_back(r.stop);
  }
  g_prof_pending.clear();
}

void profile_reset() {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  drain_locked();
  g_prof_kinds.clear();
}

int profile_read(const char **names, int64_t *launches, double *total_ms, int cap) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  drain_locked();
  int n = 0;
  for (auto &k : g_prof_kinds) {
    if (n >= cap) break;
    if (names) names[n] = k.kind;
    if (launches) launches[n] = k.launches;
    if (total_ms) total_ms[n] = k.ms;
    n++;
  }
  return n;
}

int launch_begin(const char *kind, cudaStream_t s) {
  if (!g_prof_on.load()) return -1;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  ProfRecord r{kind, pool_get(), pool_get()};
  cudaEventRecord(r.start, s);
  g_prof_pending.push_back(r);
  return int(g_prof_pending.size()) - 1;
}

sao_status launch_end(int slot, cudaStream_t s) {
  cudaError_t e = cudaGetLastError();
  if (slot >= 0) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (slot < int(g_prof_pending.size())) cudaEventRecord(g_prof_pending[slot].stop, s);
  }
  if (e != cudaSuccess) return fail(SAO_ERR_CUDA, "kernel launch failed: %s", cudaGetErrorString(e));
  return SAO_OK;
}

// ---------------------------------------------------------------------------
// device info
// ---------------------------------------------------------------------------
sao_status device_info(DeviceInfo *out) {
  static std::mutex mu;
  static std::vector<DeviceInfo> cache;
  int dev = 0;
  SAO_CUDA_TRY(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(mu);
  for (auto &d : cache)
    if (d.device == dev) {
      *out = d;
      return SAO_OK;
    }
  DeviceInfo d{};
  d.device = dev;
  SAO_CUDA_TRY(cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev));
  SAO_CUDA_TRY(cudaDeviceGetAttribute(&d.cc_major, cudaDevAttrComputeCapabilityMajor, dev));
  SAO_CUDA_TRY(cudaDeviceGetAttribute(&d.cc_minor, cudaDevAttrComputeCapabilityMinor, dev));
  int optin = 0;
  SAO_CUDA_TRY(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev));
  d.smem_optin = size_t(optin);
  cache.push_back(d);
  *out = d;
  return SAO_OK;
}

// ---------------------------------------------------------------------------
// checked mode
// ---------------------------------------------------------------------------
sao_status begin_call(void *ws, cudaStream_t s) {
  if (checked_mode()) SAO_CUDA_TRY(cudaMemsetAsync(ws, 0, sizeof(unsigned int), s));
  return SAO_OK;
}

sao_status finish_call(void *ws, cudaStream_t s) {
  if (!checked_mode()) return SAO_OK;
  unsigned int word = 0;
  SAO_CUDA_TRY(cudaMemcpyAsync(&word, ws, sizeof(word), cudaMemcpyDeviceToHost, s));
  SAO_CUDA_TRY(cudaStreamSynchronize(s));
  if (word != 0) {
    std::string what;
    if (word & SAO_DEVERR_TOKEN_ID) what += " token-id-out-of-range";
    if (word & SAO_DEVERR_CU_SEQLENS) what += " bad-cu_seqlens";
    if (word & SAO_DEVERR_SCAN_TIMEOUT) what += " scan-carry-timeout";
    if (word & SAO_DEVERR_PIPE_TIMEOUT) what += " pipeline-wait-timeout";
    if (word & SAO_DEVERR_CACHE_ROW) what += " cached-row-not-computed";
    return fail(SAO_ERR_DEVICE_CHECK, "device check failed (0x%x):%s", word, what.c_str());
  }
  return SAO_OK;
}

}  // namespace sao
