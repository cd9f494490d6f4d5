// Per-head finalisation, top-k selection and gather-compaction.
//
// finalize (one CTA per (layer, KV head) unit):
//   D_E = mean of d_E over all N keys (Eq. 4), r_E = 2 - 2 sigma(D_E / tau)
//   (Eq. 5), r_C = (N ||mu||^2 - 1) / (N - 1) (MixKV, Appendix A), lambda =
//   beta r_E + (1 - beta) r_C (Eq. 6); pooled importance S_imp (SnapKV average
//   pooling, centred, zero padding counted); s_E = min-max of d_E (Eq. 2),
//   s_C = (1 - khat.mu)/2, S_div = alpha s_E + (1 - alpha) s_C (Eq. 3); the
//   rescale Sbar = minmax(S_div), Stilde = Sbar mean(S_imp) / mean(Sbar)
//   (Sec. 5.2); S = lambda Stilde + (1 - lambda) S_imp (Eq. 7).
// select: the top (B - W) candidates by (S descending, position ascending)
//   (Sec. 3), found by an MSB-first radix select on the order-preserving
//   32-bit image of S; emitted in ascending position, followed by the window.
// compact: K_out[r] = K[idx[r]], V_out[r] = V[idx[r]] with 16-byte copies.

#include <math.h>

#include "ecokv_internal.cuh"

namespace ecokv {
namespace {

constexpr int kFinThreads = 1024;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Deterministic block reductions (fixed lane/warp order); sh holds >= 33 floats.
enum class Op { Sum, Min, Max };
template <Op op>
__device__ __forceinline__ float wred(float v) {
  return op == Op::Sum ? warp_sum(v) : op == Op::Min ? warp_min(v) : warp_max(v);
}
template <Op op>
__device__ float block_reduce(float v, float* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  v = wred<op>(v);
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  if (warp == 0) {
    const float ident = op == Op::Sum ? 0.f : op == Op::Min ? INFINITY : -INFINITY;
    float x = lane < nw ? sh[lane] : ident;
    x = wred<op>(x);
    if (lane == 0) sh[32] = x;
  }
  __syncthreads();
  const float r = sh[32];
  __syncthreads();
  return r;
}

// Exclusive prefix sum over the block; *total receives the block total.
__device__ int block_exclusive_scan(int v, int* sh, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sh[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  const int before = (warp > 0 ? sh[warp - 1] : 0) + x - v;
  *total = sh[nw - 1];
  __syncthreads();
  return before;
}

// Composite diversity (Eq. 2 and Eq. 3; s_C = (1 - c)/2, or -c for the MixKV
// variant).  Explicit round-to-nearest intrinsics keep every pass that
// recomputes it bit-identical.
__device__ __forceinline__ float sdiv_of(float dE, float c, float mnE, float denE, float alpha, bool mix) {
  const float sE = __fdiv_rn(__fsub_rn(dE, mnE), denE);
  const float sC = mix ? -c : __fmul_rn(__fsub_rn(1.f, c), 0.5f);
  return __fadd_rn(__fmul_rn(alpha, sE), __fmul_rn(__fsub_rn(1.f, alpha), sC));
}

// Centred average pooling, zero padding counted in the divisor.
__device__ __forceinline__ float pooled(const float* raw, int i, int Tv, int pool) {
  const int half = pool >> 1;
  float s = 0.f;
  for (int o = -half; o <= half; ++o) {
    const int j = i + o;
    if (j >= 0 && j < Tv) s = __fadd_rn(s, raw[j]);
  }
  return __fdiv_rn(s, (float)pool);
}

__device__ void finalize_unit(const FinalArgs& a, int u, float* shf) {
  const int t = threadIdx.x, nt = blockDim.x;
  const int Tv = a.Tv;
  const float* us = a.ustat + (size_t)u * a.ustat_stride;
  const float* raw = a.simp + (size_t)u * Tv;
  const float* dE = a.dE + (size_t)u * Tv;
  const float* cv = a.cosv + (size_t)u * Tv;
  float* S = a.S + (size_t)u * Tv;
  float* dbg = a.dbg ? a.dbg + (size_t)u * 5 * Tv : nullptr;
  const bool mix = (a.flags & ECOKV_FLAG_SC_MIXKV_SIGN) != 0;

  // Per-head redundancy and lambda (a few scalar ops, in double).
  float part = 0.f;
  for (int c = t; c < a.nchunks; c += nt) part += __ldcg(a.p2part + (size_t)u * a.nchunks + c);
  const float sum_dE = block_reduce<Op::Sum>(part, shf);
  const double N = (double)a.N;
  const double D_E = (double)sum_dE / N;
  const double tau = a.tau > 0.f ? (double)a.tau : sqrt((double)kD);
  const double r_E = 2.0 - 2.0 / (1.0 + exp(-D_E / tau));
  const double mu_sq = (double)__ldcg(us + ustat_musq());
  const double r_C = a.N == 1 ? 1.0 : (N * mu_sq - 1.0) / (N - 1.0);
  double lam = (double)a.beta * r_E + (1.0 - (double)a.beta) * r_C;
  if (a.flags & ECOKV_FLAG_LAMBDA_OVERRIDE) lam = (double)a.lambda_override;
  const float lamf = (float)lam;
  if (a.lambda != nullptr && t == 0) a.lambda[u] = lamf;
  if (Tv == 0) return;

  // Pass A: pooled importance (kept in S for now), its sum, extrema of d_E.
  float s_sum = 0.f, mnE = INFINITY, mxE = -INFINITY;
  for (int i = t; i < Tv; i += nt) {
    const float sp = pooled(raw, i, Tv, a.pool);
    S[i] = sp;
    s_sum += sp;
    const float e = dE[i];
    mnE = fminf(mnE, e);
    mxE = fmaxf(mxE, e);
  }
  const float sum_imp = block_reduce<Op::Sum>(s_sum, shf);
  mnE = block_reduce<Op::Min>(mnE, shf);
  mxE = block_reduce<Op::Max>(mxE, shf);
  const float denE = __fadd_rn(__fsub_rn(mxE, mnE), a.eps);

  // Pass B: extrema of the composite diversity.
  float mnD = INFINITY, mxD = -INFINITY;
  for (int i = t; i < Tv; i += nt) {
    const float sd = sdiv_of(dE[i], cv[i], mnE, denE, a.alpha, mix);
    mnD = fminf(mnD, sd);
    mxD = fmaxf(mxD, sd);
  }
  mnD = block_reduce<Op::Min>(mnD, shf);
  mxD = block_reduce<Op::Max>(mxD, shf);
  const float denD = __fadd_rn(__fsub_rn(mxD, mnD), a.eps);

  // Pass C: mean of the min-max normalised diversity.
  float sb_sum = 0.f;
  for (int i = t; i < Tv; i += nt) {
    const float sd = sdiv_of(dE[i], cv[i], mnE, denE, a.alpha, mix);
    sb_sum += __fdiv_rn(__fsub_rn(sd, mnD), denD);
  }
  const float sum_sbar = block_reduce<Op::Sum>(sb_sum, shf);
  // Stilde = Sbar * mean(S_imp) / mean(Sbar); zero when Sbar vanishes.
  const float scale = sum_sbar > 0.f ? __fdiv_rn(sum_imp, sum_sbar) : 0.f;

  // Pass D: final score (Eq. 7).
  const float one_m_lam = __fsub_rn(1.f, lamf);
  for (int i = t; i < Tv; i += nt) {
    const float sd = sdiv_of(dE[i], cv[i], mnE, denE, a.alpha, mix);
    const float sbar = __fdiv_rn(__fsub_rn(sd, mnD), denD);
    const float sp = S[i];
    S[i] = __fadd_rn(__fmul_rn(lamf, __fmul_rn(sbar, scale)), __fmul_rn(one_m_lam, sp));
    if (dbg) {
      dbg[i] = raw[i];
      dbg[Tv + i] = sp;
      dbg[2 * Tv + i] = dE[i];
      dbg[3 * Tv + i] = cv[i];
      dbg[4 * Tv + i] = sd;
    }
  }
  __syncthreads();
}

// Order-preserving image of a float: larger float -> larger unsigned.
__device__ __forceinline__ unsigned ordered_key(float f) {
  unsigned b = __float_as_uint(f);
  if (b == 0x80000000u) b = 0u;  // -0 ranks with +0
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Top-k of S[0..Tv) by (value desc, position asc), written in ascending
// position to out[0..k).  hist: 256 ints of shared memory, shi: >= 34 ints.
__device__ void topk_ascending(const float* S, int Tv, int k, int32_t* out, unsigned* hist, int* shi) {
  const int t = threadIdx.x, nt = blockDim.x;
  if (k <= 0) return;
  unsigned prefix = 0u, mask = 0u;
  int rem = k;  // how many still to take from the current bucket
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = t; b < 256; b += nt) hist[b] = 0u;
    __syncthreads();
    for (int i = t; i < Tv; i += nt) {
      const unsigned key = ordered_key(S[i]);
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (t == 0) {
      int above = 0, sel = 0;
      for (int b = 255; b >= 0; --b) {
        const int h = (int)hist[b];
        if (above + h >= rem) { sel = b; break; }
        above += h;
      }
      shi[32] = sel;
      shi[33] = rem - above;
    }
    __syncthreads();
    prefix |= (unsigned)shi[32] << shift;
    mask |= 255u << shift;
    rem = shi[33];
    __syncthreads();
  }
  // prefix is now the k-th largest key; take every key above it and the first
  // `rem` keys equal to it (lowest positions first).
  const unsigned thr = prefix;
  const int seg = (Tv + nt - 1) / nt;
  const int lo = min(Tv, t * seg), hi = min(Tv, lo + seg);
  int n_gt = 0, n_eq = 0;
  for (int i = lo; i < hi; ++i) {
    const unsigned key = ordered_key(S[i]);
    n_gt += key > thr;
    n_eq += key == thr;
  }
  int tot;
  const int eq_before = block_exclusive_scan(n_eq, shi, &tot);
  const int take_eq = max(0, min(n_eq, rem - eq_before));
  const int pos0 = block_exclusive_scan(n_gt + take_eq, shi, &tot);
  int pos = pos0, eq_seen = 0;
  for (int i = lo; i < hi; ++i) {
    const unsigned key = ordered_key(S[i]);
    bool keep = key > thr;
    if (key == thr) {
      keep = eq_seen < take_eq;
      ++eq_seen;
    }
    if (keep && pos < k) out[pos++] = i;
  }
  __syncthreads();
}

__device__ void select_unit(const FinalArgs& a, int u, unsigned* hist, int* shi) {
  int32_t* out = a.idx + (size_t)u * a.n_keep;
  if (a.budget >= a.N) {
    for (int r = threadIdx.x; r < a.N; r += blockDim.x) out[r] = r;
    return;
  }
  const int k = a.budget - a.W;
  topk_ascending(a.S + (size_t)u * a.Tv, a.Tv, k, out, hist, shi);
  for (int j = threadIdx.x; j < a.W; j += blockDim.x) out[k + j] = a.Tv + j;
}

template <bool kScore, bool kSelect>
__global__ void __launch_bounds__(kFinThreads) finalize_kernel(FinalArgs a) {
  __shared__ float shf[64];
  __shared__ unsigned hist[256];
  __shared__ int shi[64];
  const int u = blockIdx.x;
  if (kScore) finalize_unit(a, u, shf);
  if (kSelect) select_unit(a, u, hist, shi);
}

template <typename T>
__global__ void __launch_bounds__(256) compact_kernel(CompactArgs a) {
  constexpr int vpr = kD * sizeof(T) / 16;  // 16-byte vectors per row
  constexpr int rows = 32;
  const int u = blockIdx.y;
  const int r0 = blockIdx.x * rows;
  const uint4* K = reinterpret_cast<const uint4*>(a.K) + (size_t)u * a.N * vpr;
  const uint4* V = reinterpret_cast<const uint4*>(a.V) + (size_t)u * a.N * vpr;
  uint4* Ko = reinterpret_cast<uint4*>(a.K_out) + (size_t)u * a.n_keep * vpr;
  uint4* Vo = reinterpret_cast<uint4*>(a.V_out) + (size_t)u * a.n_keep * vpr;
  const int32_t* idx = a.idx + (size_t)u * a.n_keep;
  for (int e = threadIdx.x; e < rows * vpr; e += blockDim.x) {
    const int r = r0 + e / vpr, v = e % vpr;
    if (r >= a.n_keep) break;
    const int src = __ldg(idx + r);
    uint4 kv = make_uint4(0u, 0u, 0u, 0u), vv = kv;
    if (src >= 0 && src < a.N) {
      kv = __ldg(K + (size_t)src * vpr + v);
      vv = __ldg(V + (size_t)src * vpr + v);
    } else if (a.status != nullptr) {
      atomicCAS(a.status, 0u, (unsigned)ECOKV_ERR_DEVICE_INDEX);
      a.status[1] = (unsigned)u;
    }
    Ko[(size_t)r * vpr + v] = kv;
    Vo[(size_t)r * vpr + v] = vv;
  }
}

}  // namespace

cudaError_t launch_finalize(const FinalArgs& a, int U, bool do_score, bool do_select, cudaStream_t s) {
  if (do_score && do_select)
    finalize_kernel<true, true><<<U, kFinThreads, 0, s>>>(a);
  else if (do_score)
    finalize_kernel<true, false><<<U, kFinThreads, 0, s>>>(a);
  else
    finalize_kernel<false, true><<<U, kFinThreads, 0, s>>>(a);
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
