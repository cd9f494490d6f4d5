// Finalisation and selection kernels (one CTA per unit) and the compaction
// kernel (32 kept rows per CTA); the device code lives in finalize_select.cuh.

#include "finalize_select.cuh"

namespace ecokv {
namespace {

constexpr int kFinThreads = 1024;

// Scores of unit blockIdx.x and, with kSelect, its top-k.  kSmem keeps the
// unit's scores in shared memory.
template <bool kSmem, bool kSelect>
__global__ void __launch_bounds__(kFinThreads) finalize_kernel(FinalArgs f) {
  extern __shared__ float sS[];
  __shared__ float shf[64];
  __shared__ unsigned hist[256];
  __shared__ int shi[64];
  const int u = blockIdx.x;
  float* S = kSmem ? sS : (f.S ? f.S : f.S_scratch) + (size_t)u * f.Tv;
  finalize_unit<BlockSync>(f, u, S, shf, threadIdx.x, blockDim.x);
  if (kSelect) select_unit<BlockSync>(f, u, S, hist, shi, threadIdx.x, blockDim.x);
}

__global__ void __launch_bounds__(kFinThreads) select_kernel(FinalArgs f) {
  __shared__ unsigned hist[256];
  __shared__ int shi[64];
  const int u = blockIdx.x;
  select_unit<BlockSync>(f, u, f.S + (size_t)u * f.Tv, hist, shi, threadIdx.x, blockDim.x);
}

template <typename T>
__global__ void __launch_bounds__(256) compact_kernel(CompactArgs a) {
  // launched as a programmatic dependent: the indices come from the previous
  // grid (a no-op when launched plainly)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  constexpr int rows = 32;
  const int r0 = blockIdx.x * rows;
  gather_rows<T>(a, blockIdx.y, r0, r0 + rows, threadIdx.x, blockDim.x);
}

}  // namespace

// Scores of every unit and, with do_select, their top-k.
cudaError_t launch_finalize(const FinalArgs& f, int U, bool do_select, cudaStream_t s) {
  if (!do_select) {
    finalize_kernel<false, false><<<U, kFinThreads, 0, s>>>(f);
    return cudaGetLastError();
  }
  if (f.Tv > 0 && f.Tv <= kSmemScores) {
    const size_t smem = (size_t)f.Tv * sizeof(float);
    cudaError_t e =
        cudaFuncSetAttribute(finalize_kernel<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    finalize_kernel<true, true><<<U, kFinThreads, smem, s>>>(f);
  } else {
    finalize_kernel<false, true><<<U, kFinThreads, 0, s>>>(f);
  }
  return cudaGetLastError();
}

cudaError_t launch_select(const FinalArgs& f, int U, cudaStream_t s) {
  select_kernel<<<U, kFinThreads, 0, s>>>(f);
  return cudaGetLastError();
}

cudaError_t launch_compact(const CompactArgs& a, ecokv_dtype dt, int U, cudaStream_t s) {
  if (a.n_keep == 0 || U == 0) return cudaSuccess;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((a.n_keep + 31) / 32, U);
  cfg.blockDim = dim3(256, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (dt == ECOKV_F32) return cudaLaunchKernelEx(&cfg, compact_kernel<float>, a);
  return cudaLaunchKernelEx(&cfg, compact_kernel<__nv_bfloat16>, a);
}

}  // namespace ecokv
