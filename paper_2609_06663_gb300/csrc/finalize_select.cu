// Finalisation, selection and compaction kernels (one CTA per unit); the
// device code lives in finalize_select.cuh.

#include "finalize_select.cuh"

namespace ecokv {
namespace {

constexpr int kFinThreads = 1024;

// Scores of unit blockIdx.x; with kSelect the top-k, with kCompact the gather
// of the retained rows.  kSmem keeps the unit's scores in shared memory.
template <typename T, bool kSmem, bool kSelect, bool kCompact>
__global__ void __launch_bounds__(kFinThreads) finalize_kernel(FinalArgs f, CompactArgs c) {
  extern __shared__ float sS[];
  __shared__ float shf[64];
  __shared__ unsigned hist[256];
  __shared__ int shi[64];
  const int u = blockIdx.x;
  float* S = kSmem ? sS : (f.S ? f.S : f.S_scratch) + (size_t)u * f.Tv;
  finalize_unit<BlockSync>(f, u, S, shf, threadIdx.x, blockDim.x);
  if (kSelect) select_unit<BlockSync>(f, u, S, hist, shi, threadIdx.x, blockDim.x);
  if (kCompact) {
    __syncthreads();
    gather_rows<T>(c, u, 0, f.n_keep, threadIdx.x, blockDim.x);
  }
}

__global__ void __launch_bounds__(kFinThreads) select_kernel(FinalArgs f) {
  __shared__ unsigned hist[256];
  __shared__ int shi[64];
  const int u = blockIdx.x;
  select_unit<BlockSync>(f, u, f.S + (size_t)u * f.Tv, hist, shi, threadIdx.x, blockDim.x);
}

template <typename T>
__global__ void __launch_bounds__(256) compact_kernel(CompactArgs a) {
  constexpr int rows = 32;
  const int r0 = blockIdx.x * rows;
  gather_rows<T>(a, blockIdx.y, r0, r0 + rows, threadIdx.x, blockDim.x);
}

template <typename T>
cudaError_t launch_fc(const FinalArgs& f, const CompactArgs& c, int U, cudaStream_t s) {
  if (f.Tv > 0 && f.Tv <= kSmemScores) {
    const size_t smem = (size_t)f.Tv * sizeof(float);
    cudaError_t e =
        cudaFuncSetAttribute(finalize_kernel<T, true, true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    finalize_kernel<T, true, true, true><<<U, kFinThreads, smem, s>>>(f, c);
  } else {
    finalize_kernel<T, false, true, true><<<U, kFinThreads, 0, s>>>(f, c);
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_finalize(const FinalArgs& f, const CompactArgs* c, ecokv_dtype dt, int U, bool do_select,
                            cudaStream_t s) {
  if (!do_select || c == nullptr) {
    finalize_kernel<float, false, false, false><<<U, kFinThreads, 0, s>>>(f, CompactArgs{});
    return cudaGetLastError();
  }
  return dt == ECOKV_F32 ? launch_fc<float>(f, *c, U, s) : launch_fc<__nv_bfloat16>(f, *c, U, s);
}

cudaError_t launch_select(const FinalArgs& f, int U, cudaStream_t s) {
  select_kernel<<<U, kFinThreads, 0, s>>>(f);
  return cudaGetLastError();
}

cudaError_t launch_compact(const CompactArgs& a, ecokv_dtype dt, int U, cudaStream_t s) {
  if (a.n_keep == 0 || U == 0) return cudaSuccess;
  const dim3 grid((a.n_keep + 31) / 32, U);
  if (dt == ECOKV_F32)
    compact_kernel<float><<<grid, 256, 0, s>>>(a);
  else
    compact_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace ecokv
