// slnr_sddmm_spmm_noalloc: the fused <SDDMM,SpMM> call for callers that
// cannot allocate device memory.
//
// Some callers may not call cudaMalloc at all: a real-time or signal-safe
// path that must not enter the allocator (which can block or take locks), or
// an embedding runtime that owns all device memory and hands out none to the
// libraries it hosts.  This entry point needs no caller workspace:
// its scratch is the file-scope array below, which the CUDA runtime creates
// with the module, so every GPU that loads this library holds
// kNoAllocScratchBytes of device memory until the process exits.
//
// The host code must not use the array's name as a device pointer (in host
// code it names a host-side stand-in), so the first call on each device looks
// up the array's device address with cudaGetSymbolAddress, with that device
// current, and caches it.  The cache outlives a device reset
// (cudaDeviceReset), after which the address is stale: a process that
// resets a device must not call this entry point on it again.  Every call shares the one array,
// which keeps the last call's contents: the call clears the part that must
// start at zero (the header of counters) itself, and calls whose work
// overlaps on the GPU (different streams, or different host threads on one
// device) race on the array and give wrong results.
#include <cstdio>
#include <cstring>
#include <mutex>

#include "launch.h"

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;  // 16 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mutex;
void* g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once
// per device).  Returns cudaSuccess and sets *ptr, or the lookup's error.
cudaError_t scratch_address(void** ptr) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (g_noalloc_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    if (p == nullptr) return cudaErrorInvalidSymbol;
    g_noalloc_ptr[dev] = p;
  }
  *ptr = g_noalloc_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" slnr_status slnr_sddmm_spmm_noalloc(const slnr_csr* B, const float* C, const float* D, int32_t L,
                                               const float* E, int32_t K, float* A, void* stream) {
  slnr_opts o;
  std::memset(&o, 0, sizeof(o));
  o.variant = SLNR_FUSED;
  o.stream = stream;
  size_t need = 0;
  slnr_status st = slnr_sddmm_spmm_workspace(B, L, K, &o, &need);
  if (st != SLNR_OK) return st;
  if (need > kNoAllocScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "slnr_sddmm_spmm_noalloc: these sizes need %zu bytes of scratch; the built-in scratch holds %zu "
             "bytes (use slnr_sddmm_spmm with a caller workspace)",
             need, kNoAllocScratchBytes);
    slnr::set_last_error(msg);
    return SLNR_ERR_UNSUPPORTED;
  }
  void* scratch = nullptr;
  const cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) {
    char msg[256];
    snprintf(msg, sizeof(msg), "slnr_sddmm_spmm_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
    slnr::set_last_error(msg);
    return SLNR_ERR_CUDA;
  }
  o.workspace = scratch;
  o.workspace_bytes = kNoAllocScratchBytes;
  return slnr_sddmm_spmm(B, C, D, L, E, K, A, &o);
}
