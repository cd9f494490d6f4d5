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

// One CTA per (head, layer): the head's share of the layer's chosen positions
// (a contiguous run of the ascending list, found by binary search), written
// as positions in the head, then its window; the head's list starts at the
// number of chosen positions of lower heads plus their windows.
__global__ void __launch_bounds__(256) adaptive_split_kernel(AdaptArgs a) {
  const int h = blockIdx.x, l = blockIdx.y;
  __shared__ int s_lo, s_hi;
  const int32_t* ch = a.chosen + (size_t)l * a.k_layer;
  if (threadIdx.x == 0) {
    if (a.keep_all) {
      s_lo = h * a.Tv;
      s_hi = (h + 1) * a.Tv;
    } else {
      // first index with ch[i] >= key, for key = h Tv and (h + 1) Tv
      int lo = 0, hi = a.k_layer;
      while (lo < hi) {
        const int m = (lo + hi) >> 1;
        if (ch[m] < h * a.Tv) lo = m + 1; else hi = m;
      }
      s_lo = lo;
      hi = a.k_layer;
      while (lo < hi) {
        const int m = (lo + hi) >> 1;
        if (ch[m] < (h + 1) * a.Tv) lo = m + 1; else hi = m;
      }
      s_hi = lo;
    }
  }
  __syncthreads();
  const int lo = s_lo, cnt = s_hi - s_lo, off = lo + h * a.W;
  const size_t base = (size_t)l * a.h_kv * a.n_keep + off;
  for (int r = threadIdx.x; r < cnt + a.W; r += blockDim.x) {
    const int pos = r < cnt ? (a.keep_all ? r : ch[lo + r] - h * a.Tv) : a.Tv + (r - cnt);
    a.idx[base + r] = pos;
    a.src[base + r] = h * a.N + pos;
  }
  if (threadIdx.x == 0) {
    int32_t* o = a.head_off + (size_t)l * (a.h_kv + 1);
    o[h] = off;
    if (h == a.h_kv - 1) o[a.h_kv] = a.h_kv * a.n_keep;
  }
}

// ||v_i|| for the candidate rows: 16-byte vectors, the lanes of a row summing
// their squares in fp32 and combining by shuffles (a streaming read of V).
template <typename T>
__global__ void __launch_bounds__(256) value_norm_kernel(const T* V, float* vn, int N, int Tv) {
  constexpr int kVpr = kD * sizeof(T) / 16;  // 16-byte vectors per row: 16 (bf16) or 32 (fp32)
  constexpr int kRows = 32 / kVpr;           // rows a warp takes per step
  const int u = blockIdx.y, lane = threadIdx.x & 31;
  const int r_lane = lane / kVpr, v = lane % kVpr;
  const uint4* Vu = reinterpret_cast<const uint4*>(V) + (size_t)u * N * kVpr;
  const int warps = gridDim.x * (blockDim.x >> 5), w = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int step = warps * kRows;
  for (int r0 = w * kRows; r0 < Tv; r0 += 4 * step) {
    uint4 q[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int r = r0 + j * step + r_lane;
      q[j] = r < Tv ? __ldcs(Vu + (size_t)r * kVpr + v) : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int r = r0 + j * step + r_lane;
      float acc = 0.f;
      if constexpr (sizeof(T) == 2) {
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&q[j]);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(h[e]);
          acc = fmaf(f.x, f.x, acc);
          acc = fmaf(f.y, f.y, acc);
        }
      } else {
        const float* f = reinterpret_cast<const float*>(&q[j]);
#pragma unroll
        for (int e = 0; e < 4; ++e) acc = fmaf(f[e], f[e], acc);
      }
#pragma unroll
      for (int o = kVpr / 2; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (v == 0 && r < Tv) vn[(size_t)u * Tv + r] = sqrtf(acc);
    }
  }
}

}  // namespace

cudaError_t launch_value_norms(const void* V, ecokv_dtype dt, int U, int N, int Tv, float* vn, cudaStream_t s) {
  if (U <= 0 || Tv <= 0) return cudaSuccess;
  const dim3 grid((unsigned)((Tv + 255) / 256 < 64 ? (Tv + 255) / 256 : 64), U);
  if (dt == ECOKV_F32)
    value_norm_kernel<float><<<grid, 256, 0, s>>>(static_cast<const float*>(V), vn, N, Tv);
  else
    value_norm_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(V), vn, N, Tv);
  return cudaGetLastError();
}

cudaError_t launch_adaptive_split(const AdaptArgs& a, int n_layers, cudaStream_t s) {
  adaptive_split_kernel<<<dim3(a.h_kv, n_layers), 256, 0, s>>>(a);
  return cudaGetLastError();
}

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
