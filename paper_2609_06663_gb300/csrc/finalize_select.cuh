// Per-head finalisation, top-k selection and row gather as device functions
// run by a group of `nt` threads (tid in [0, nt), nt a multiple of 32) that
// synchronise through the policy `Sync`.
//
// finalize_unit (one (layer, KV head) unit), from the per-chunk partials of
// pass 2 and the per-candidate arrays (raw vote, d_E, cosine):
//   D_E = mean of d_E over all N keys (Eq. 4), r_E = 2 - 2 sigma(D_E / tau)
//   (Eq. 5), r_C = (N ||mu||^2 - 1) / (N - 1) (MixKV, Appendix A), lambda =
//   beta r_E + (1 - beta) r_C (Eq. 6); S_imp = centred average pooling of the
//   vote (SnapKV, zero padding counted); s_E = min-max of d_E (Eq. 2), s_C =
//   (1 - khat.mu)/2, S_div = alpha s_E + (1 - alpha) s_C (Eq. 3); Sbar =
//   minmax(S_div), Stilde = Sbar mean(S_imp) / mean(Sbar) (Sec. 5.2);
//   S = lambda Stilde + (1 - lambda) S_imp (Eq. 7).
//   The extrema of d_E and the sums behind every mean come from the pass-2
//   partials; mean(S_imp) and mean(Sbar) follow from them exactly in real
//   arithmetic (pooling and min-max are linear), so only two sweeps over the
//   candidates remain: one for the extrema of S_div, one for S.
// select_unit: the top (B - W) candidates by (S descending, position
//   ascending) (Sec. 3), by an MSB-first radix select on the order-preserving
//   32-bit image of S, emitted in ascending position (warp ballots over
//   contiguous ranges) and followed by the window.
// gather_rows: K_out[r] = K[idx[r]], V_out[r] = V[idx[r]], 16-byte copies.
#pragma once

#include <math.h>

#include "ecokv_internal.cuh"

namespace ecokv {

struct BlockSync {
  __device__ __forceinline__ static void sync() { __syncthreads(); }
};

__device__ __forceinline__ float fs_warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float fs_warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float fs_warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

enum class Op { Sum, Min, Max };
template <Op op>
__device__ __forceinline__ float fs_wred(float v) {
  return op == Op::Sum ? fs_warp_sum(v) : op == Op::Min ? fs_warp_min(v) : fs_warp_max(v);
}

// Deterministic group reduction (fixed lane/warp order); sh holds >= 33 floats.
template <Op op, class Sync>
__device__ float group_reduce(float v, float* sh, int tid, int nt) {
  const int lane = tid & 31, warp = tid >> 5, nw = nt >> 5;
  v = fs_wred<op>(v);
  if (lane == 0) sh[warp] = v;
  Sync::sync();
  if (warp == 0) {
    const float ident = op == Op::Sum ? 0.f : op == Op::Min ? INFINITY : -INFINITY;
    float x = lane < nw ? sh[lane] : ident;
    x = fs_wred<op>(x);
    if (lane == 0) sh[32] = x;
  }
  Sync::sync();
  const float r = sh[32];
  Sync::sync();
  return r;
}

// Composite diversity (Eq. 2 and Eq. 3; s_C = (1 - c)/2, or -c for the MixKV
// variant).  Explicit round-to-nearest intrinsics keep every sweep that
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
    if (j >= 0 && j < Tv) s = __fadd_rn(s, __ldg(raw + j));
  }
  return __fdiv_rn(s, (float)pool);
}

// Scores of one unit into Sbuf[0..Tv) (shared or global memory); also to
// a.S (global) when Sbuf is not a.S and a.S is set.
template <class Sync>
__device__ void finalize_unit(const FinalArgs& a, int u, float* Sbuf, float* shf, int tid, int nt) {
  const int Tv = a.Tv;
  const float* us = a.ustat + (size_t)u * a.ustat_stride;
  const float* raw = a.simp + (size_t)u * Tv;
  const float* dE = a.dE + (size_t)u * Tv;
  const float* cv = a.cosv + (size_t)u * Tv;
  float* Sg = (a.S != nullptr && a.S + (size_t)u * Tv != Sbuf) ? a.S + (size_t)u * Tv : nullptr;
  float* dbg = a.dbg ? a.dbg + (size_t)u * 5 * Tv : nullptr;
  const bool mix = (a.flags & ECOKV_FLAG_SC_MIXKV_SIGN) != 0;

  // unit scalars from the pass-2 chunk partials
  float s_all = 0.f, mnE = INFINITY, mxE = -INFINITY, s_de = 0.f, s_c = 0.f, s_raw = 0.f;
  for (int c = tid; c < a.nchunks; c += nt) {
    const float* p = a.p2part + ((size_t)u * a.nchunks + c) * kP2Stride;
    s_all += __ldg(p + P2_SUM_DE_ALL);
    mnE = fminf(mnE, __ldg(p + P2_MIN_DE));
    mxE = fmaxf(mxE, __ldg(p + P2_MAX_DE));
    s_de += __ldg(p + P2_SUM_DE);
    s_c += __ldg(p + P2_SUM_COS);
    s_raw += __ldg(p + P2_SUM_RAW);
  }
  s_all = group_reduce<Op::Sum, Sync>(s_all, shf, tid, nt);
  mnE = group_reduce<Op::Min, Sync>(mnE, shf, tid, nt);
  mxE = group_reduce<Op::Max, Sync>(mxE, shf, tid, nt);
  s_de = group_reduce<Op::Sum, Sync>(s_de, shf, tid, nt);
  s_c = group_reduce<Op::Sum, Sync>(s_c, shf, tid, nt);
  s_raw = group_reduce<Op::Sum, Sync>(s_raw, shf, tid, nt);

  // per-head redundancy and lambda (a few scalar ops, in double)
  const double N = (double)a.N;
  const double D_E = (double)s_all / N;
  const double tau = a.tau > 0.f ? (double)a.tau : sqrt((double)kD);
  const double r_E = 2.0 - 2.0 / (1.0 + exp(-D_E / tau));
  const double mu_sq = (double)__ldg(us + ustat_musq());
  const double r_C = a.N == 1 ? 1.0 : (N * mu_sq - 1.0) / (N - 1.0);
  double lam = (double)a.beta * r_E + (1.0 - (double)a.beta) * r_C;
  if (a.flags & ECOKV_FLAG_LAMBDA_OVERRIDE) lam = (double)a.lambda_override;
  const float lamf = (float)lam;
  if (a.lambda != nullptr && tid == 0) a.lambda[u] = lamf;
  if (Tv == 0) return;
  const float denE = __fadd_rn(__fsub_rn(mxE, mnE), a.eps);

  // sweep 1: extrema of S_div, pooled importance into Sbuf (four candidates
  // per thread in flight)
  float mnD = INFINITY, mxD = -INFINITY;
  for (int i0 = tid; i0 < Tv; i0 += 4 * nt) {
    float e4[4], c4[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + q * nt;
      e4[q] = i < Tv ? __ldg(dE + i) : 0.f;
      c4[q] = i < Tv ? __ldg(cv + i) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + q * nt;
      if (i < Tv) {
        const float sd = sdiv_of(e4[q], c4[q], mnE, denE, a.alpha, mix);
        mnD = fminf(mnD, sd);
        mxD = fmaxf(mxD, sd);
        Sbuf[i] = pooled(raw, i, Tv, a.pool);
      }
    }
  }
  mnD = group_reduce<Op::Min, Sync>(mnD, shf, tid, nt);
  mxD = group_reduce<Op::Max, Sync>(mxD, shf, tid, nt);
  const float denD = __fadd_rn(__fsub_rn(mxD, mnD), a.eps);

  // means: sum_i S_imp(i) = (1/kp) sum_j raw(j) cnt(j), where cnt(j) = kp
  // except within kp/2 of either end; mean(Sbar) is affine in the means of
  // d_E and of the cosine.
  if (tid == 0) {
    const int h = a.pool >> 1;
    double edge = 0.0;
    for (int j = 0; j < Tv && j < h; ++j) edge += (double)__ldg(raw + j) * (double)(h - j);
    for (int j = (Tv - h > 0 ? Tv - h : 0); j < Tv; ++j) edge += (double)__ldg(raw + j) * (double)(h - (Tv - 1 - j));
    const double sum_imp = ((double)a.pool * (double)s_raw - edge) / (double)a.pool;
    const double mean_imp = sum_imp / Tv;
    const double mean_sE = ((double)s_de / Tv - (double)mnE) / (double)denE;
    const double mean_c = (double)s_c / Tv;
    const double mean_sC = mix ? -mean_c : (1.0 - mean_c) * 0.5;
    const double mean_div = (double)a.alpha * mean_sE + (1.0 - (double)a.alpha) * mean_sC;
    const double mean_sbar = (mean_div - (double)mnD) / (double)denD;
    shf[40] = mean_sbar > 0.0 ? (float)(mean_imp / mean_sbar) : 0.f;
  }
  Sync::sync();
  const float scale = shf[40];
  const float one_m_lam = __fsub_rn(1.f, lamf);

  // sweep 2: final score (Eq. 7)
  for (int i0 = tid; i0 < Tv; i0 += 4 * nt) {
    float e4[4], c4[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + q * nt;
      e4[q] = i < Tv ? __ldg(dE + i) : 0.f;
      c4[q] = i < Tv ? __ldg(cv + i) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + q * nt;
      if (i < Tv) {
        const float sd = sdiv_of(e4[q], c4[q], mnE, denE, a.alpha, mix);
        const float sbar = __fdiv_rn(__fsub_rn(sd, mnD), denD);
        const float sp = Sbuf[i];
        const float S = __fadd_rn(__fmul_rn(lamf, __fmul_rn(sbar, scale)), __fmul_rn(one_m_lam, sp));
        Sbuf[i] = S;
        if (Sg) Sg[i] = S;
        if (dbg) {
          dbg[i] = __ldg(raw + i);
          dbg[Tv + i] = sp;
          dbg[2 * Tv + i] = e4[q];
          dbg[3 * Tv + i] = c4[q];
          dbg[4 * Tv + i] = sd;
        }
      }
    }
  }
  Sync::sync();
}

// Order-preserving image of a float: larger float -> larger unsigned.
__device__ __forceinline__ unsigned ordered_key(float f) {
  unsigned b = __float_as_uint(f);
  if (b == 0x80000000u) b = 0u;  // -0 ranks with +0
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// The float an order-preserving key stands for (the inverse of ordered_key).
__device__ __forceinline__ float key_float(unsigned k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Top-k of S[0..Tv) by (value desc, position asc), written in ascending
// position to out[0..k).  hist: 256 unsigned, shi: >= 64 ints (shared).
template <class Sync>
__device__ void topk_ascending(const float* S, int Tv, int k, int32_t* out, unsigned* hist, int* shi, int tid,
                               int nt) {
  if (k <= 0) return;
  const int lane = tid & 31, warp = tid >> 5, nw = nt >> 5;
  unsigned prefix = 0u, mask = 0u;
  int rem = k;  // how many still to take from the current bucket
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = tid; b < 256; b += nt) hist[b] = 0u;
    Sync::sync();
    for (int i0 = tid - lane; i0 < Tv; i0 += nt) {
      const int i = i0 + lane;
      unsigned bin = 0xffffffffu;
      if (i < Tv) {
        const unsigned key = ordered_key(S[i]);
        if ((key & mask) == prefix) bin = (key >> shift) & 255u;
      }
      // warp-aggregated increment: scores of one head share few exponents
      const unsigned peers = __match_any_sync(0xffffffffu, bin);
      if (bin != 0xffffffffu && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], (unsigned)__popc(peers));
    }
    Sync::sync();
    if (tid == 0) {
      int above = 0, sel = 0;
      for (int b = 255; b >= 0; --b) {
        const int h = (int)hist[b];
        if (above + h >= rem) {
          sel = b;
          break;
        }
        above += h;
      }
      shi[0] = sel;
      shi[1] = rem - above;
    }
    Sync::sync();
    prefix |= (unsigned)shi[0] << shift;
    mask |= 255u << shift;
    rem = shi[1];
    Sync::sync();
  }
  // prefix is now the k-th largest key: keep every key above it and the first
  // `rem` keys equal to it.  Each warp owns one contiguous range of positions.
  const unsigned thr = prefix;
  const int span = (((Tv + nw - 1) / nw) + 31) & ~31;
  const int lo = min(Tv, warp * span), hi = min(Tv, lo + span);
  const unsigned lt = (1u << lane) - 1u;
  int n_gt = 0, n_eq = 0;
  for (int b = lo; b < hi; b += 32) {
    const int i = b + lane;
    const unsigned key = i < hi ? ordered_key(S[i]) : 0u;
    n_gt += __popc(__ballot_sync(0xffffffffu, i < hi && key > thr));
    n_eq += __popc(__ballot_sync(0xffffffffu, i < hi && key == thr));
  }
  if (lane == 0) shi[warp] = n_eq;
  Sync::sync();
  int eq_before = 0;
  for (int w = 0; w < warp; ++w) eq_before += shi[w];
  const int take_eq = max(0, min(n_eq, rem - eq_before));
  Sync::sync();
  if (lane == 0) shi[warp] = n_gt + take_eq;
  Sync::sync();
  int pos = 0;
  for (int w = 0; w < warp; ++w) pos += shi[w];
  int eq_seen = 0;
  for (int b = lo; b < hi; b += 32) {
    const int i = b + lane;
    const unsigned key = i < hi ? ordered_key(S[i]) : 0u;
    const bool gt = i < hi && key > thr;
    const bool eq = i < hi && key == thr;
    const unsigned eqm = __ballot_sync(0xffffffffu, eq);
    const bool take = gt || (eq && eq_seen + __popc(eqm & lt) < take_eq);
    const unsigned sel = __ballot_sync(0xffffffffu, take);
    if (take) {
      const int p = pos + __popc(sel & lt);
      if (p < k) out[p] = i;
    }
    pos += __popc(sel);
    eq_seen += __popc(eqm);
  }
  Sync::sync();
}

// idx[u] = top-k candidates then the window (or 0..N-1 when B >= N).
template <class Sync>
__device__ void select_unit(const FinalArgs& a, int u, const float* S, unsigned* hist, int* shi, int tid, int nt) {
  int32_t* out = a.idx + (size_t)u * a.n_keep;
  const int budget = unit_budget(a, u);
  // slots past this unit's budget (per-layer budgets) hold -1
  for (int r = (budget < a.N ? budget : a.N) + tid; r < a.n_keep; r += nt) out[r] = -1;
  if (budget >= a.N) {
    for (int r = tid; r < a.N; r += nt) out[r] = r;
    return;
  }
  const int k = budget - a.W;
  topk_ascending<Sync>(S, a.Tv, k, out, hist, shi, tid, nt);
  for (int j = tid; j < a.W; j += nt) out[k + j] = a.Tv + j;
}

// Copy rows [r0, r1) of unit u: K_out[r] = K[idx[r]] and V_out[r] = V[idx[r]],
// four 16-byte vectors of each in flight per thread.
template <typename T>
__device__ void gather_rows(const CompactArgs& a, int u, int r0, int r1, int tid, int nt) {
  constexpr int vpr = kD * sizeof(T) / 16;  // 16-byte vectors per row
  const uint4* K = reinterpret_cast<const uint4*>(a.K) + (size_t)u * a.N * vpr;
  const uint4* V = reinterpret_cast<const uint4*>(a.V) + (size_t)u * a.N * vpr;
  uint4* Ko = reinterpret_cast<uint4*>(a.K_out) + (size_t)u * a.n_keep * vpr;
  uint4* Vo = reinterpret_cast<uint4*>(a.V_out) + (size_t)u * a.n_keep * vpr;
  const int32_t* idx = a.idx + (size_t)u * a.n_keep;
  r1 = min(r1, a.n_lb ? a.keep[u / a.h_kv] : a.n_keep);
  const int total = (r1 - r0) * vpr;
  for (int e0 = tid; e0 < total; e0 += 4 * nt) {
    uint4 kv[4], vv[4];
    int dst[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = e0 + j * nt;
      dst[j] = -1;
      kv[j] = make_uint4(0u, 0u, 0u, 0u);
      vv[j] = kv[j];
      if (e < total) {
        const int r = r0 + e / vpr, v = e % vpr;
        const int src = __ldcg(idx + r);
        dst[j] = r * vpr + v;
        if (src >= 0 && src < a.N) {
          kv[j] = __ldcs(K + (size_t)src * vpr + v);  // each row is read once
          vv[j] = __ldcs(V + (size_t)src * vpr + v);
        } else if (a.status != nullptr) {
          atomicCAS(a.status, 0u, (unsigned)ECOKV_ERR_DEVICE_INDEX);
          a.status[1] = (unsigned)u;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (dst[j] >= 0) {
        __stcs(Ko + dst[j], kv[j]);
        __stcs(Vo + dst[j], vv[j]);
      }
  }
}

}  // namespace ecokv
