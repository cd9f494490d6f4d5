// ecokv_evict_noalloc: the whole eviction pass with its workspace taken from
// a fixed scratch area compiled into this translation unit, so that the call
// itself allocates nothing.
//
// Who needs it: a caller that may not allocate device memory where it evicts,
// e.g. a serving runtime that has handed all free HBM to its KV-cache pool
// before the first request and forbids allocation inside a step, or plain C
// code that has no allocator of its own and cannot afford cudaMalloc's
// implicit device synchronisation in the middle of a prefill.  Those callers
// still own K, V, Qwin and the outputs; only the scratch is provided here.
//
// The scratch is a file-scope __device__ array, so every device context that
// loads this module gets its own copy of ECOKV_NOALLOC_SCRATCH_BYTES, once,
// when the module is loaded (lazily, on the first use of this entry point).
// Its device address is looked up with cudaGetSymbolAddress once per device,
// with that device current, by the first call on that device.
//
// Zeroing: the status words at the start of the scratch must be zero when a
// call's kernels start.  A __device__ array starts at zero, and every call that
// launched anything copies its status out and clears the words again (in
// stream order) before it returns.  The per-call counters are cleared by the
// streaming passes themselves, as for ecokv_evict; nothing else needs to
// start at zero.
//
// Concurrency: every call on one device uses the same scratch.  Two calls whose
// executions overlap (different streams without an ordering between them, or
// different host threads) race on it and give undefined results; callers
// serialise them, e.g. by issuing them on one stream.

#include <mutex>

#include "ecokv_internal.cuh"

namespace ecokv {
namespace {

constexpr int kMaxDevices = 64;
static_assert(ECOKV_NOALLOC_SCRATCH_BYTES % 256 == 0, "scratch size a multiple of 256 bytes");

__device__ __align__(256) unsigned char g_noalloc_scratch[ECOKV_NOALLOC_SCRATCH_BYTES];

std::mutex g_setup_mu;
void* g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of this device's scratch; the first call per device looks it
// up (the device must be current).  nullptr on failure.
void* scratch_for_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return nullptr;
    if ((reinterpret_cast<uintptr_t>(p) & 255u) != 0) return nullptr;
    g_scratch_ptr[dev] = p;
  }
  return g_scratch_ptr[dev];
}

}  // namespace
}  // namespace ecokv

extern "C" ecokv_status ecokv_evict_noalloc(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                           const void* Qwin, int32_t* idx, void* K_out, void* V_out, float* S,
                                           float* lambda, uint32_t* dev_status, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (ecokv_workspace_size(p) > (size_t)ECOKV_NOALLOC_SCRATCH_BYTES) return ECOKV_ERR_WORKSPACE;
  if (dev_status != nullptr && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return ECOKV_ERR_INVALID_ARG;
  void* ws = ecokv::scratch_for_current_device();
  if (ws == nullptr) return ECOKV_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  st = ecokv_evict(p, dtype, K, V, Qwin, idx, K_out, V_out, S, lambda, ws, ECOKV_NOALLOC_SCRATCH_BYTES, stream);
  if (st != ECOKV_OK && st != ECOKV_ERR_CUDA) return st;  // rejected before anything was launched
  if (st == ECOKV_OK && dev_status != nullptr &&
      cudaMemcpyAsync(dev_status, ws, sizeof(uint32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    st = ECOKV_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, 256, s) != cudaSuccess) st = ECOKV_ERR_CUDA;
  return st;
}
