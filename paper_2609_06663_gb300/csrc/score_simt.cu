// Streaming score passes on the CUDA cores (any dtype, any window size).
//
// Pass 1 (one CTA per 128-key chunk of one (layer, KV head) unit):
//   window logits l = q . k / sqrt(d) for the g*W window rows of the group
//   (Sec. 3 softmax(QK^T/sqrt(d_k)), SnapKV observation window, Appendix A),
//   per-row chunk maximum and exp-sum (online-softmax partials), the key norms
//   ||k_i||, and the chunk sums of k_i and k_i/||k_i|| for the centroid kbar
//   (Eq. 1) and the mean normalised key mu (MixKV, Appendix A).  The last CTA
//   of a unit to finish folds the partials into the unit statistics: kbar, mu
//   and the log-sum-exp of every window row.
// Pass 2 (same grid) recomputes the logits and turns them into the
//   importance vote sum_{rows} p(row, i) for the candidates i < N - W, the
//   distance d_E(i) = ||k_i - kbar|| (Eq. 1) and the cosine khat_i . mu; it
//   also emits per-chunk sums of d_E over all N keys for D_E (Eq. 4).
//
// Logits are accumulated in 8-term partial sums (fp32) which keeps the fp32
// path well inside a 1e-5 relative tolerance on the final score.

#include <math.h>

#include "ecokv_internal.cuh"

namespace ecokv {
namespace {

constexpr int kThreads = kChunk;  // one key per thread
constexpr int kWarps = kThreads / 32;

template <typename T> struct Tile;
template <> struct Tile<float> { static constexpr int stride = kD + 4; };          // 528 B rows
template <> struct Tile<__nv_bfloat16> { static constexpr int stride = kD + 8; };  // 272 B rows

__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 a = *reinterpret_cast<const uint4*>(p);
  v[0] = bf_lo(a.x); v[1] = bf_hi(a.x); v[2] = bf_lo(a.y); v[3] = bf_hi(a.y);
  v[4] = bf_lo(a.z); v[5] = bf_hi(a.z); v[6] = bf_lo(a.w); v[7] = bf_hi(a.w);
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// Stage the chunk's keys (rows i0 .. i0+kChunk-1 of one unit) into shared
// memory with a 16-byte row skew; rows past N are zero.
template <typename T>
__device__ void load_tile(T* ks, const T* Ku, int i0, int N) {
  constexpr int per_vec = 16 / sizeof(T);
  constexpr int vpr = kD / per_vec;
  for (int e = threadIdx.x; e < kChunk * vpr; e += blockDim.x) {
    const int row = e / vpr, v = e % vpr;
    const int key = i0 + row;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (key < N) val = __ldg(reinterpret_cast<const uint4*>(Ku + (size_t)key * kD) + v);
    *reinterpret_cast<uint4*>(ks + row * Tile<T>::stride + v * per_vec) = val;
  }
}

// acc[r] = k . q_r for RB query rows held in shared memory as fp32, with
// 8-term partial sums; optionally also the squared norm of k.
template <typename T, int RB>
__device__ __forceinline__ void dot_rows(const T* krow, const float* qblk, float (&acc)[RB], float* nrm2) {
#pragma unroll
  for (int r = 0; r < RB; ++r) acc[r] = 0.f;
  float n2 = 0.f;
#pragma unroll 2
  for (int c = 0; c < kD / 8; ++c) {
    float kv[8];
    load8(krow + c * 8, kv);
    if (nrm2) {
      float pn = kv[0] * kv[0];
#pragma unroll
      for (int e = 1; e < 8; ++e) pn = fmaf(kv[e], kv[e], pn);
      n2 += pn;
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const float4 q0 = *reinterpret_cast<const float4*>(qblk + r * kD + c * 8);
      const float4 q1 = *reinterpret_cast<const float4*>(qblk + r * kD + c * 8 + 4);
      float pp = kv[0] * q0.x;
      pp = fmaf(kv[1], q0.y, pp);
      pp = fmaf(kv[2], q0.z, pp);
      pp = fmaf(kv[3], q0.w, pp);
      pp = fmaf(kv[4], q1.x, pp);
      pp = fmaf(kv[5], q1.y, pp);
      pp = fmaf(kv[6], q1.z, pp);
      pp = fmaf(kv[7], q1.w, pp);
      acc[r] += pp;
    }
  }
  if (nrm2) *nrm2 = n2;
}

// Chunked squared distance to kbar and dot with mu (both fp32 in smem).
template <typename T>
__device__ __forceinline__ void dist_and_dot(const T* krow, const float* kbar, const float* mu, float* d2, float* dmu) {
  float s2 = 0.f, sm = 0.f;
#pragma unroll 2
  for (int c = 0; c < kD / 8; ++c) {
    float kv[8];
    load8(krow + c * 8, kv);
    float pd, pm;
    {
      const float t0 = kv[0] - kbar[c * 8];
      pd = t0 * t0;
      pm = kv[0] * mu[c * 8];
    }
#pragma unroll
    for (int e = 1; e < 8; ++e) {
      const float te = kv[e] - kbar[c * 8 + e];
      pd = fmaf(te, te, pd);
      pm = fmaf(kv[e], mu[c * 8 + e], pm);
    }
    s2 += pd;
    sm += pm;
  }
  *d2 = s2;
  *dmu = sm;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Per-row block maximum and exp2-sum relative to it, over the CTA's keys.
template <int RB>
__device__ void rows_max_expsum(float (&x)[RB], float* red, float* mrow, float* out_m, float* out_z, int nvalid) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int r = 0; r < RB; ++r) {
    const float m = warp_max(x[r]);
    if (lane == 0) red[warp * RB + r] = m;
  }
  __syncthreads();
  if (threadIdx.x < RB) {
    float m = red[threadIdx.x];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) m = fmaxf(m, red[w * RB + threadIdx.x]);
    mrow[threadIdx.x] = m;
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < RB; ++r) {
    const float m = mrow[r];
    const float e = (m == -INFINITY) ? 0.f : exp2f(x[r] - m);
    const float z = warp_sum(e);
    if (lane == 0) red[warp * RB + r] = z;
  }
  __syncthreads();
  if (threadIdx.x < nvalid) {
    float z = red[threadIdx.x];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) z += red[w * RB + threadIdx.x];
    out_m[threadIdx.x] = mrow[threadIdx.x];
    out_z[threadIdx.x] = z;
  }
  __syncthreads();
}

__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float block_min128(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_min(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = red[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) s = fminf(s, red[w]);
  __syncthreads();
  return s;
}

__device__ __forceinline__ float block_max128(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_max(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = red[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) s = fmaxf(s, red[w]);
  __syncthreads();
  return s;
}

__device__ __forceinline__ float block_sum128(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = red[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) s += red[w];
  __syncthreads();
  return s;
}

template <typename T>
__device__ void stage_queries(float* qs, const ScoreArgs& a, int u, int Rpad) {
  const int layer = u / a.h_kv, head = u % a.h_kv;
  const T* Qu = static_cast<const T*>(a.Q) + ((size_t)layer * a.h_q + (size_t)head * a.g) * a.W * kD;
  for (int e = threadIdx.x; e < Rpad * kD; e += blockDim.x)
    qs[e] = (e < a.R * kD) ? to_f32(Qu[e]) : 0.f;
}

template <typename T, int RB>
__global__ void __launch_bounds__(kThreads) pass1_kernel(ScoreArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int u = blockIdx.y, chunk = blockIdx.x, t = threadIdx.x;
  const int Rpad = (a.R + RB - 1) / RB * RB;
  float* qs = reinterpret_cast<float*>(smem);                       // [Rpad][kD]
  T* ks = reinterpret_cast<T*>(qs + Rpad * kD);                      // [kChunk][stride]
  float* invn = reinterpret_cast<float*>(ks + kChunk * Tile<T>::stride);
  float* red = invn + kChunk;                                        // [kWarps * RB]
  float* mrow = red + kWarps * 32;                                   // [RB]
  __shared__ int s_last;

  stage_queries<T>(qs, a, u, Rpad);
  const int i0 = chunk * kChunk;
  load_tile<T>(ks, static_cast<const T*>(a.K) + (size_t)u * a.N * kD, i0, a.N);
  __syncthreads();

  const int i = i0 + t;
  const bool valid = i < a.N;
  const T* krow = ks + t * Tile<T>::stride;
  float* part = a.p1part + ((size_t)u * a.nchunks + chunk) * a.p1_stride;
  float nrm2 = 0.f;
  for (int rb = 0; rb < Rpad; rb += RB) {
    float acc[RB];
    dot_rows<T, RB>(krow, qs + rb * kD, acc, rb == 0 ? &nrm2 : nullptr);
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int row = rb + r;
      const int j = row % a.W;
      const bool vis = valid && row < a.R && i <= a.N - a.W + j;
      acc[r] = vis ? acc[r] * a.scale_log2 : -INFINITY;
    }
    const int nvalid = min(RB, a.R - rb);
    rows_max_expsum<RB>(acc, red, mrow, part + rb, part + a.R + rb, nvalid);
  }

  invn[t] = valid ? 1.f / fmaxf(sqrtf(nrm2), 1e-12f) : 0.f;
  __syncthreads();
  {
    // thread t owns dimension t: chunk sums of k and k/||k||
    float sk = 0.f, skh = 0.f;
    for (int r = 0; r < kChunk; ++r) {
      const float v = to_f32(ks[r * Tile<T>::stride + t]);
      if (i0 + r < a.kbar_n) sk += v;  // the centroid's keys (all, or the candidates only)
      skh = fmaf(v, invn[r], skh);
    }
    part[2 * a.R + t] = sk;
    part[2 * a.R + kD + t] = skh;
  }

  // The last CTA of this unit folds the partials into the unit statistics.
  __threadfence();
  __syncthreads();
  if (t == 0) s_last = (atomicAdd(&a.cnt[u], 1u) == gridDim.x - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  const float* base = a.p1part + (size_t)u * a.nchunks * a.p1_stride;
  float* us = a.ustat + (size_t)u * a.ustat_stride;
  float sk = 0.f, skh = 0.f;
  for (int c = 0; c < a.nchunks; ++c) {
    sk += __ldcg(base + (size_t)c * a.p1_stride + 2 * a.R + t);
    skh += __ldcg(base + (size_t)c * a.p1_stride + 2 * a.R + kD + t);
  }
  const float inv_n = 1.f / (float)a.N;
  const float kb = sk * (1.f / (float)a.kbar_n), mu = skh * inv_n;
  us[ustat_kbar() + t] = kb;
  us[ustat_mu() + t] = mu;
  for (int row = t; row < a.R; row += kThreads) {
    float M = -INFINITY;
    for (int c = 0; c < a.nchunks; ++c) M = fmaxf(M, __ldcg(base + (size_t)c * a.p1_stride + row));
    float Z = 0.f;
    for (int c = 0; c < a.nchunks; ++c) {
      const float m = __ldcg(base + (size_t)c * a.p1_stride + row);
      if (m != -INFINITY) Z += __ldcg(base + (size_t)c * a.p1_stride + a.R + row) * exp2f(m - M);
    }
    us[ustat_lse() + row] = M + log2f(Z);
  }
  const float ksq = block_sum128(kb * kb, red);
  const float msq = block_sum128(mu * mu, red);
  if (t == 0) {
    us[ustat_ksq()] = ksq;
    us[ustat_musq()] = msq;
  }
}

template <typename T, int RB>
__global__ void __launch_bounds__(kThreads) pass2_kernel(ScoreArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int u = blockIdx.y, chunk = blockIdx.x, t = threadIdx.x;
  const int Rpad = (a.R + RB - 1) / RB * RB;
  float* qs = reinterpret_cast<float*>(smem);                        // [Rpad][kD]
  T* ks = reinterpret_cast<T*>(qs + Rpad * kD);                       // [kChunk][stride]
  float* kbar = reinterpret_cast<float*>(ks + kChunk * Tile<T>::stride);
  float* mu = kbar + kD;
  float* lse = mu + kD;                                               // [Rpad]
  float* red = lse + Rpad;                                            // [kWarps]

  const float* us = a.ustat + (size_t)u * a.ustat_stride;
  stage_queries<T>(qs, a, u, Rpad);
  kbar[t] = __ldcg(us + ustat_kbar() + t);
  mu[t] = __ldcg(us + ustat_mu() + t);
  for (int r = t; r < Rpad; r += kThreads) lse[r] = r < a.R ? __ldcg(us + ustat_lse() + r) : 0.f;
  const int i0 = chunk * kChunk;
  load_tile<T>(ks, static_cast<const T*>(a.K) + (size_t)u * a.N * kD, i0, a.N);
  __syncthreads();

  const int i = i0 + t;
  const bool valid = i < a.N;
  const T* krow = ks + t * Tile<T>::stride;
  float nrm2 = 0.f, vote = 0.f;
  for (int rb = 0; rb < Rpad; rb += RB) {
    float acc[RB];
    dot_rows<T, RB>(krow, qs + rb * kD, acc, rb == 0 ? &nrm2 : nullptr);
#pragma unroll
    for (int r = 0; r < RB; ++r)
      if (rb + r < a.R) vote += exp2f(acc[r] * a.scale_log2 - lse[rb + r]);
  }
  float d2, dmu;
  dist_and_dot<T>(krow, kbar, mu, &d2, &dmu);
  const float dE = sqrtf(d2);
  const float cosv = dmu * (1.f / fmaxf(sqrtf(nrm2), 1e-12f));
  const bool cand = i < a.Tv;
  if (cand) {
    const size_t o = (size_t)u * a.Tv + i;
    a.simp[o] = vote;
    a.dE[o] = dE;
    a.cosv[o] = cosv;
  }
  const float s_all = block_sum128(valid ? dE : 0.f, red);
  const float mn = block_min128(cand ? dE : INFINITY, red);
  const float mx = block_max128(cand ? dE : -INFINITY, red);
  const float s_de = block_sum128(cand ? dE : 0.f, red);
  const float s_c = block_sum128(cand ? cosv : 0.f, red);
  const float s_raw = block_sum128(cand ? vote : 0.f, red);
  if (t == 0) {
    float* p = a.p2part + ((size_t)u * a.nchunks + chunk) * kP2Stride;
    p[P2_SUM_DE_ALL] = s_all;
    p[P2_MIN_DE] = mn;
    p[P2_MAX_DE] = mx;
    p[P2_SUM_DE] = s_de;
    p[P2_SUM_COS] = s_c;
    p[P2_SUM_RAW] = s_raw;
  }
}

template <typename T, int RB>
size_t smem_pass1(int R) {
  const int Rpad = (R + RB - 1) / RB * RB;
  return (size_t)Rpad * kD * 4 + (size_t)kChunk * Tile<T>::stride * sizeof(T) + kChunk * 4 +
         (kWarps * 32 + RB) * 4;
}
template <typename T, int RB>
size_t smem_pass2(int R) {
  const int Rpad = (R + RB - 1) / RB * RB;
  return (size_t)Rpad * kD * 4 + (size_t)kChunk * Tile<T>::stride * sizeof(T) + 2 * kD * 4 + Rpad * 4 +
         kWarps * 4 * 4;
}

template <typename T, int RB>
cudaError_t launch_rb(const ScoreArgs& a, int U, cudaStream_t s) {
  const dim3 grid(a.nchunks, U);
  const size_t s1 = smem_pass1<T, RB>(a.R), s2 = smem_pass2<T, RB>(a.R);
  cudaError_t e = cudaFuncSetAttribute(pass1_kernel<T, RB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)s1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(pass2_kernel<T, RB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)s2);
  if (e != cudaSuccess) return e;
  pass1_kernel<T, RB><<<grid, kThreads, s1, s>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  pass2_kernel<T, RB><<<grid, kThreads, s2, s>>>(a);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const ScoreArgs& a, int U, cudaStream_t s) {
  if (a.R <= 8) return launch_rb<T, 8>(a, U, s);
  if (a.R <= 16) return launch_rb<T, 16>(a, U, s);
  return launch_rb<T, 32>(a, U, s);
}

}  // namespace

cudaError_t launch_score_simt(const ScoreArgs& a, ecokv_dtype dt, int U, cudaStream_t s) {
  return dt == ECOKV_F32 ? launch_t<float>(a, U, s) : launch_t<__nv_bfloat16>(a, U, s);
}

}  // namespace ecokv
