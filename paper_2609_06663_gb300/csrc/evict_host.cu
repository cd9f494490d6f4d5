// ecokv_evict_host: the eviction pass for a KV cache resident in host memory
// that the device addresses directly (pinned and mapped, unified addressing).
//
// Built on the public entry point: K and Qwin are copied once into the
// workspace (both streaming passes read K, so one copy beats two trips over
// the host link); ecokv_evict then runs on those copies with V, K_out, V_out
// and lambda left in host memory, so that the gather reads only the kept V
// rows over the link and writes the outputs there directly; the indices,
// made in the workspace, are copied back last.  With value-norm importance
// (ECOKV_FLAG_VNORM_IMP) the norm kernel reads every row of V where it lies,
// so then all of V crosses the link as well.
//
// Workspace layout: [ecokv_workspace_size bytes | K copy | Qwin copy | idx],
// each region 256-byte aligned.

#include <cuda_runtime.h>

#include "ecokv_internal.cuh"

namespace {

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t elem_bytes(ecokv_dtype dt) { return dt == ECOKV_F32 ? 4 : 2; }

struct HostLayout {
  size_t base, k_off, k_bytes, q_off, q_bytes, idx_off, idx_bytes, total;
};

HostLayout host_layout(const ecokv_params& p, ecokv_dtype dt) {
  HostLayout h{};
  h.base = align256(ecokv_workspace_size(&p));
  const size_t e = elem_bytes(dt);
  h.k_bytes = (size_t)p.n_layers * p.h_kv * p.n * p.d * e;
  h.q_bytes = (size_t)p.n_layers * p.h_q * p.window * p.d * e;
  h.idx_bytes = (size_t)p.n_layers * p.h_kv * (size_t)(p.budget < p.n ? p.budget : p.n) * sizeof(int32_t);
  h.k_off = h.base;
  h.q_off = h.k_off + align256(h.k_bytes);
  h.idx_off = h.q_off + align256(h.q_bytes);
  h.total = h.idx_off + align256(h.idx_bytes);
  return h;
}

// True when ptr is host memory the current device addresses at the same
// address (pinned or registered, mapped, unified addressing).
bool device_mapped_host(const void* ptr) {
  if (ptr == nullptr) return false;
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    cudaGetLastError();  // clear the error state the failed query leaves
    return false;
  }
  return a.type == cudaMemoryTypeHost && a.devicePointer == ptr;
}

}  // namespace

extern "C" size_t ecokv_workspace_size_host(const ecokv_params* p, ecokv_dtype dtype) {
  if (ecokv_check_params(p) != ECOKV_OK || (dtype != ECOKV_F32 && dtype != ECOKV_BF16)) return 0;
  return host_layout(*p, dtype).total;
}

extern "C" ecokv_status ecokv_evict_host(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                         const void* Qwin, int32_t* idx, void* K_out, void* V_out,
                                         float* lambda, void* ws, size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!device_mapped_host(K) || !device_mapped_host(V) || !device_mapped_host(Qwin) || !device_mapped_host(idx) ||
      !device_mapped_host(K_out) || !device_mapped_host(V_out) || (lambda && !device_mapped_host(lambda)))
    return ECOKV_ERR_INVALID_ARG;
  const HostLayout h = host_layout(*p, dtype);
  if (ws == nullptr || ((uintptr_t)ws & 15u) != 0 || ws_bytes < h.total) return ECOKV_ERR_WORKSPACE;
  char* w = static_cast<char*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void* K_dev = w + h.k_off;
  void* Q_dev = w + h.q_off;
  int32_t* idx_dev = reinterpret_cast<int32_t*>(w + h.idx_off);
  if (cudaMemcpyAsync(K_dev, K, h.k_bytes, cudaMemcpyHostToDevice, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  if (cudaMemcpyAsync(Q_dev, Qwin, h.q_bytes, cudaMemcpyHostToDevice, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  st = ecokv_evict(p, dtype, K_dev, V, Q_dev, idx_dev, K_out, V_out, nullptr, lambda, ws, h.base, stream);
  if (st != ECOKV_OK) return st;
  if (cudaMemcpyAsync(idx, idx_dev, h.idx_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  return ECOKV_OK;
}
