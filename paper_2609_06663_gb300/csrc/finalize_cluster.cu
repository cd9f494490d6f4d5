// Finalisation and selection of one (layer, KV head) unit by a thread-block
// cluster of C CTAs: the arithmetic of finalize_unit / select_unit
// (finalize_select.cuh), spread over the cluster so that every SM takes part,
// with the cluster-wide reductions done through distributed shared memory.
//
// Two shapes: 16 candidates a thread and up to 8 CTAs (units up to 32768
// candidates, used up to 16384), or 32 candidates a thread and up to 4 CTAs
// (units of 16385 to 32768): at four CTAs per SM the GPU holds about 74
// clusters of 8 but 148 of 4, so the long units of a prefill (e.g. 28 layers
// x 4 KV heads of 32k tokens) run in one wave instead of one and a half.
//
// CTA rank r of the cluster owns candidates [r * cap, (r + 1) * cap) of the
// unit (cap = 256 threads x kJ); thread t of it owns the kJ consecutive
// candidates from r * cap + kJ * t and keeps their pooled importance, then
// the keys of their scores, in registers.  The raw votes of the CTA (with the
// pooling halo) are staged in shared memory with one pad word after every 32,
// so that the 32 lanes of a warp, kJ positions apart, read distinct banks.
// Steps:
//   1. unit scalars from the pass-2 partials (every CTA, same inputs, same
//      result), lambda (Eq. 4-6);
//   2. S_div (Eq. 2, 3) and pooled S_imp of the owned candidates; extrema of
//      S_div over the cluster;
//   3. S (Eq. 7) as finalize_unit computes it, divisions by the min-max
//      ranges and the pooling kernel taken as reciprocal products;
//   4. MSB-first radix select over the order-preserving image of S, one
//      256-bin histogram per CTA, summed over the cluster for each 8-bit digit;
//   5. counts of keys above / equal to the threshold, scanned over the
//      threads and exchanged between the CTAs, so that each thread knows how
//      many kept candidates precede its own (ties to the lower position);
//      then its kept positions in ascending order (the last CTA adds the
//      window).  The gather of the kept rows is its own launch.
// Cluster barriers are reached by every CTA on every path (no early exit).
// Every exchange between CTAs is a store into the peers' shared memory
// (each CTA keeps every rank's contribution) followed by a cluster barrier,
// so no CTA waits on a remote load.

#include <atomic>

#include <cooperative_groups.h>

#include "finalize_select.cuh"

namespace cg = cooperative_groups;

namespace ecokv {
namespace {

constexpr int kCThreads = 256;
constexpr int kCWarps = kCThreads / 32;
constexpr int kHalo = 16;  // pooling halo kept in shared memory (kernel <= 33)

// Shapes (kSh): 0 = 16 candidates a thread, up to 8 CTAs; 1 = 32 a thread,
// up to 4 CTAs; 2 = 32 a thread, up to 16 CTAs (clusters past the portable 8,
// for units of 32769 to 131072 candidates; their larger exchange buffers
// would cost the 4-CTA shape occupancy).
template <int kSh>
struct Shape {
  static constexpr int kJ = kSh == 0 ? 16 : 32;                            // candidates a thread owns
  static constexpr int kCap = kCThreads * kJ;                              // candidates a CTA owns
  static constexpr int kMaxCluster = kSh == 0 ? 8 : (kSh == 1 ? 4 : 16);  // CTAs a unit may take
  static constexpr int kQ = kCap + 2 * kHalo;                              // staged raw votes
};

// Padded shared-memory index of staged position q.
__device__ __forceinline__ int pad_idx(int q) { return q + (q >> 5); }

template <int kSh>
struct ClusterSmem {
  // raw vote of candidate lo - kHalo + q at raw[pad_idx(q)]
  float raw[Shape<kSh>::kQ + Shape<kSh>::kQ / 32 + 1];
  unsigned whist[kCWarps][256];  // per radix pass, each warp's own histogram
  // Written by the peers (distributed shared memory stores): per radix pass
  // the histogram of every rank (double-buffered across passes), the S_div
  // extrema and the counts above / equal to the threshold of every rank.
  unsigned hall[2][Shape<kSh>::kMaxCluster][256];
  float ext_all[Shape<kSh>::kMaxCluster][2];
  double simp_all[Shape<kSh>::kMaxCluster];  // value-norm importance: every rank's sum of S_imp
  double wsum_all[Shape<kSh>::kMaxCluster];  // winsorised min-max / MAD scaling: every rank's sum of s_E terms
  int cnt_all[Shape<kSh>::kMaxCluster][2];
  float red[kCWarps][8];  // per-warp partials
  float edge[32];         // pooling edge values
  float sc[8];            // broadcast scalars
  double dsc[2];          // sums behind the means of S_imp and of S_div
  double dred[kCWarps];   // per-warp sums of S_imp (value-norm importance)
  double dredw[kCWarps];  // per-warp sums of the clipped d_E (winsorised min-max) or of s_E (MAD scaling)
  float wmax;             // winsorised min-max: the upper clip bound
  float mmed, minv;       // MAD scaling: the median of d_E and 1 / (MAD + eps)
  unsigned wsum[kCWarps];
  int wscan[kCWarps][2];  // per-warp counts above / equal to the threshold
  int shi[4];
};

// Composite diversity (Eq. 2 and Eq. 3) with the min-max divisor applied as a
// reciprocal (one rounding more than a division; every score of a call uses
// the same formula, and ecokv_score and ecokv_evict share this kernel).
__device__ __forceinline__ float sdiv_rcp(float dE, float c, float mnE, float invE, float alpha, bool mix) {
  const float sE = __fmul_rn(__fsub_rn(dE, mnE), invE);
  const float sC = mix ? -c : __fmul_rn(__fsub_rn(1.f, c), 0.5f);
  return __fadd_rn(__fmul_rn(alpha, sE), __fmul_rn(__fsub_rn(1.f, alpha), sC));
}

// MAD scaling of a distance (the robust form of Eq. 2): the logistic
// function of (d_E - median) / (MAD + eps), the divisor as a reciprocal.
__device__ __forceinline__ float mad_logistic(float dE, float med, float inv) {
  return 1.f / (1.f + expf(-__fmul_rn(__fsub_rn(dE, med), inv)));
}

// Store v into the same object of every CTA of the cluster (its own included).
template <int kMaxC, typename T>
__device__ __forceinline__ void push_all(cg::cluster_group& cl, T* obj, T v, int C) {
#pragma unroll
  for (int r = 0; r < kMaxC; ++r)
    if (r < C) *cl.map_shared_rank(obj, r) = v;
}

// kMode: 0 = scores, 1 = scores and top-k, 2 = top-k of given scores (f.S).
// kVar: the value-norm importance, winsorised min-max and MAD scaling
// variants are compiled in (their code is left out of the default kernel, whose register budget it
// would cost).
template <int kMode, int kSh, bool kVar>
__global__ void __launch_bounds__(kCThreads, 4) finalize_cluster_kernel(FinalArgs f) {
  constexpr bool kSelect = kMode != 0;
  constexpr int kJ = Shape<kSh>::kJ, kCap = Shape<kSh>::kCap, kMaxC = Shape<kSh>::kMaxCluster;
  extern __shared__ __align__(16) uint8_t fc_smem[];
  ClusterSmem<kSh>& sm = *reinterpret_cast<ClusterSmem<kSh>*>(fc_smem);
  cg::cluster_group cl = cg::this_cluster();
  // The peers must have started before the first store into their shared
  // memory: this arrival is waited for just before it.
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  // Launched as a programmatic dependent of the streaming pass: let the gather
  // be scheduled behind this grid, and wait for the previous grid's results
  // (a no-op when launched plainly).
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int C = (int)cl.num_blocks();
  const int rank = (int)cl.block_rank();
  const int u = blockIdx.x / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int Tv = f.Tv;
  const int lo = rank * kCap;       // first candidate of this CTA
  const int c0 = lo + kJ * tid;     // first candidate of this thread
  const int q0 = kJ * tid + kHalo;  // staged position of candidate c0
  const int nv = max(0, min(kJ, Tv - c0));  // of this thread's candidates, those below Tv
  const int budget = unit_budget(f, u);
  const bool keep_all = budget >= f.N;
  const int k = keep_all ? 0 : budget - f.W;
  const bool mix = (f.flags & ECOKV_FLAG_SC_MIXKV_SIGN) != 0;
  const int hpool = f.pool >> 1;
  const bool pool_smem = hpool <= kHalo;
  const float* us = f.ustat + (size_t)u * f.ustat_stride;
  const float* raw = f.simp + (size_t)u * Tv;
  // the per-candidate arrays of this unit start 16-byte aligned: sweeps in
  // groups of four
  const bool vec4 = ((u * Tv) & 3) == 0;

  // pooled importance (as float bits), then the order-preserving keys of S
  unsigned key[kJ];

  if (kMode == 2) {
    // scores given (absent when nothing is to be chosen): staged in
    // coalesced order, then each thread's keys
    if (k > 0) {
      const float* Su = f.S + (size_t)u * Tv;
#pragma unroll 8
      for (int j = 0; j < kJ; ++j) {
        const int i = lo + kCThreads * j + tid;
        if (i < Tv) sm.raw[pad_idx(i - lo + kHalo)] = __ldg(Su + i);
      }
      __syncthreads();
#pragma unroll
      for (int c = 0; c < kJ; ++c) key[c] = ordered_key(sm.raw[pad_idx(q0 + c)]);
    }
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
  } else {
    // 1. the six pass-2 partials (sum over all N of d_E, min / max / sum of
    //    d_E, sums of cosines and of raw votes over the candidates); meanwhile
    //    the CTA's raw votes with the pooling halo and the edge values
    float v6[6] = {0.f, INFINITY, -INFINITY, 0.f, 0.f, 0.f};
    for (int ch = tid; ch < f.nchunks; ch += kCThreads) {
      const float* p = f.p2part + ((size_t)u * f.nchunks + ch) * kP2Stride;
      v6[0] += __ldg(p + P2_SUM_DE_ALL);
      v6[1] = fminf(v6[1], __ldg(p + P2_MIN_DE));
      v6[2] = fmaxf(v6[2], __ldg(p + P2_MAX_DE));
      v6[3] += __ldg(p + P2_SUM_DE);
      v6[4] += __ldg(p + P2_SUM_COS);
      v6[5] += __ldg(p + P2_SUM_RAW);
    }
    if (pool_smem) {
      if (vec4) {
        // the whole halo of kHalo each side in 16-byte loads (kHalo and lo are
        // multiples of four, so each group of four lies inside [0, Tv) or
        // outside it entirely except at the ragged end)
        for (int q = 4 * tid; q < kCap + 2 * kHalo; q += 4 * kCThreads) {
          const int j = lo - kHalo + q;
          float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
          if (j >= 0 && j + 3 < Tv) {
            v = __ldg(reinterpret_cast<const float4*>(raw + j));
          } else if (j >= 0 && j < Tv) {
            v.x = __ldg(raw + j);
            if (j + 1 < Tv) v.y = __ldg(raw + j + 1);
            if (j + 2 < Tv) v.z = __ldg(raw + j + 2);
          }
          sm.raw[pad_idx(q)] = v.x;
          sm.raw[pad_idx(q + 1)] = v.y;
          sm.raw[pad_idx(q + 2)] = v.z;
          sm.raw[pad_idx(q + 3)] = v.w;
        }
      } else {
        for (int q = kHalo - hpool + tid; q < kHalo + kCap + hpool; q += kCThreads) {
          const int j = lo - kHalo + q;
          sm.raw[pad_idx(q)] = (j >= 0 && j < Tv) ? __ldg(raw + j) : 0.f;
        }
      }
    }
    if (warp == 1 && lane < 2 * hpool && pool_smem) {
      const int j = lane < hpool ? lane : Tv - 2 * hpool + lane;
      sm.edge[lane] = (j >= 0 && j < Tv) ? __ldg(raw + j) : 0.f;
    }
  #pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      v6[0] += __shfl_xor_sync(0xffffffffu, v6[0], o);
      v6[1] = fminf(v6[1], __shfl_xor_sync(0xffffffffu, v6[1], o));
      v6[2] = fmaxf(v6[2], __shfl_xor_sync(0xffffffffu, v6[2], o));
      v6[3] += __shfl_xor_sync(0xffffffffu, v6[3], o);
      v6[4] += __shfl_xor_sync(0xffffffffu, v6[4], o);
      v6[5] += __shfl_xor_sync(0xffffffffu, v6[5], o);
    }
    if (lane == 0)
  #pragma unroll
      for (int q = 0; q < 6; ++q) sm.red[warp][q] = v6[q];
    __syncthreads();

    // pooled importance of the owned candidates (needs no unit scalar): the
    // same sum, in the same order, as pooled(); halo entries outside [0, Tv)
    // hold +0 and leave it unchanged
    {
      const float inv_pool = __frcp_rn((float)f.pool);
      if (pool_smem && hpool == 2) {
        // the default kernel of 5: each staged vote read once
        float x[kJ + 4];
#pragma unroll
        for (int s = 0; s < kJ + 4; ++s) x[s] = sm.raw[pad_idx(q0 - 2 + s)];
#pragma unroll
        for (int c = 0; c < kJ; ++c) {
          const float acc = __fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(0.f, x[c]), x[c + 1]), x[c + 2]),
                                                x[c + 3]), x[c + 4]);
          key[c] = __float_as_uint(c < nv ? __fmul_rn(acc, inv_pool) : 0.f);
        }
      } else {
#pragma unroll
        for (int c = 0; c < kJ; ++c) {
          float acc = 0.f;
          if (c < nv) {
            if (pool_smem) {
              for (int o = -hpool; o <= hpool; ++o) acc = __fadd_rn(acc, sm.raw[pad_idx(q0 + c + o)]);
            } else {
              const int i = c0 + c;
              for (int o = -hpool; o <= hpool; ++o)
                if (i + o >= 0 && i + o < Tv) acc = __fadd_rn(acc, __ldg(raw + i + o));
            }
          }
          key[c] = __float_as_uint(__fmul_rn(acc, inv_pool));
        }
      }
    }
    if (tid == 0) {
      float s_all = sm.red[0][0], mnE = sm.red[0][1], mxE = sm.red[0][2];
      float s_de = sm.red[0][3], s_c = sm.red[0][4], s_raw = sm.red[0][5];
      for (int w = 1; w < kCWarps; ++w) {
        s_all += sm.red[w][0];
        mnE = fminf(mnE, sm.red[w][1]);
        mxE = fmaxf(mxE, sm.red[w][2]);
        s_de += sm.red[w][3];
        s_c += sm.red[w][4];
        s_raw += sm.red[w][5];
      }
      if (kVar && f.wlo != nullptr) {  // winsorised min-max: the order statistics replace the extrema
        mnE = key_float(f.wlo[4 * u]);
        mxE = key_float(f.whi[4 * u]);
      }
      sm.wmax = mxE;
      sm.sc[0] = s_all;
      sm.sc[1] = mnE;
      sm.sc[2] = __fadd_rn(__fsub_rn(mxE, mnE), f.eps);
      if (kVar && f.mad != nullptr) {
        // MAD scaling: the sweep maps d_E to s_E itself, so the affine map
        // that follows it is the identity
        const int nu = f.n_units;
        const float lo2 = key_float(f.mad[4 * u]), hi2 = key_float(f.mad[4 * (nu + u)]);
        const float dlo = key_float(f.mad[4 * (2 * nu + u)]), dhi = key_float(f.mad[4 * (3 * nu + u)]);
        sm.mmed = __fmul_rn(0.5f, __fadd_rn(lo2, hi2));
        sm.minv = 1.f / __fadd_rn(__fmul_rn(0.5f, __fadd_rn(dlo, dhi)), f.eps);
        sm.sc[1] = 0.f;
        sm.sc[2] = 1.f;
      }
      sm.sc[3] = s_de;
      sm.sc[4] = s_c;
      sm.sc[5] = s_raw;
    }
    // (this barrier also ends every thread's reads of the staged raw votes)
    __syncthreads();
    const float mnE = sm.sc[1], denE = sm.sc[2];
    const float invE = __frcp_rn(denE);
    if (kVar && f.vnorm != nullptr) {
      // value-norm importance: S_imp = pooled vote * ||v||, the norms staged
      // in coalesced order where the raw votes were; the sum of S_imp (its
      // mean is no longer a function of the raw-vote sums) goes round the
      // cluster with the S_div extrema
      const float* vnu = f.vnorm + (size_t)u * Tv;
  #pragma unroll 8
      for (int j = 0; j < kJ; ++j) {
        const int i = lo + kCThreads * j + tid;
        if (i < Tv) sm.raw[pad_idx(i - lo + kHalo)] = __ldg(vnu + i);
      }
      __syncthreads();
      float psf = 0.f;  // a thread's at most 32 terms in single precision, the reductions in double
  #pragma unroll
      for (int c = 0; c < kJ; ++c)
        if (c < nv) {
          const float si = __fmul_rn(__uint_as_float(key[c]), sm.raw[pad_idx(q0 + c)]);
          key[c] = __float_as_uint(si);
          psf = __fadd_rn(psf, si);
        }
      double ps = (double)psf;
  #pragma unroll
      for (int o = 16; o > 0; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
      if (lane == 0) sm.dred[warp] = ps;
      __syncthreads();  // also: every norm read before the S_div sweep reuses the buffer
    }

    if (tid == 32) {
      // off the critical path, while the other threads compute S_div:
      // per-head redundancy and lambda (Eq. 4-6) in single precision (lambda
      // weighs two terms of order one: its rounding stays at the level of the
      // scores' own), and the parts of the means that need no cluster extremum
      const float D_E = __fdiv_rn(sm.sc[0], (float)f.N);
      const float tau = f.tau > 0.f ? f.tau : sqrtf((float)kD);
      const float r_E = 2.f - 2.f / (1.f + expf(-D_E / tau));
      const float mu_sq = __ldg(us + ustat_musq());
      const float r_C = f.N == 1 ? 1.f : ((float)f.N * mu_sq - 1.f) / (float)(f.N - 1);
      float lam = f.beta * r_E + (1.f - f.beta) * r_C;
      if (f.flags & ECOKV_FLAG_LAMBDA_OVERRIDE) lam = f.lambda_override;
      if (f.lambda != nullptr && rank == 0) f.lambda[u] = lam;
      sm.sc[0] = lam;
      // means, in double and scaled by Tv: sum_i S_imp(i) = (1/kp) sum_j
      // raw(j) cnt(j), where cnt(j) = kp except within kp/2 of either end;
      // mean(Sbar) is affine in the means of d_E and of the cosine (as
      // finalize_unit)
      const int h = hpool;
      double edge = 0.0;
      if (pool_smem) {
        // sm.edge[l] = raw[l] for l < h, raw[Tv - 2h + l] for h <= l < 2h
        for (int j = 0; j < Tv && j < h; ++j) edge += (double)sm.edge[j] * (double)(h - j);
        for (int j = (Tv - h > 0 ? Tv - h : 0); j < Tv; ++j)
          edge += (double)sm.edge[j - Tv + 2 * h] * (double)(h - (Tv - 1 - j));
      } else {
        for (int j = 0; j < Tv && j < h; ++j) edge += (double)__ldg(raw + j) * (double)(h - j);
        for (int j = (Tv - h > 0 ? Tv - h : 0); j < Tv; ++j) edge += (double)__ldg(raw + j) * (double)(h - (Tv - 1 - j));
      }
      const double T = (double)Tv;
      const double sum_sE = ((double)sm.sc[3] - (double)mnE * T) / (double)denE;
      const double sum_cs = (double)sm.sc[4];
      const double sum_sC = mix ? -sum_cs : (T - sum_cs) * 0.5;
      sm.dsc[0] = (double)f.pool * (double)sm.sc[5] - edge;                      // kp * Tv * mean(S_imp)
      sm.dsc[1] = (double)f.alpha * sum_sE + (1.0 - (double)f.alpha) * sum_sC;  // Tv * mean(S_div)
    }

    // 2. S_div (Eq. 2, 3) of the CTA's candidates, read in coalesced order
    //    and staged where the raw votes were, and its extrema over the
    //    cluster
    float mnD = INFINITY, mxD = -INFINITY;
    const bool wins = kVar && f.wlo != nullptr;
    const bool madv = kVar && f.mad != nullptr;
    const float wmax = sm.wmax, mmed = sm.mmed, minv = sm.minv;
    // this thread's sum of the clipped d_E (winsorised min-max) or of s_E (MAD
    // scaling): at most 32 terms in single precision, the reductions in double
    float wsumf = 0.f;
    {
      const float* dEu = f.dE + (size_t)u * Tv;
      const float* cvu = f.cosv + (size_t)u * Tv;
      if (vec4) {
  #pragma unroll 4
        for (int j = 0; j < kJ / 4; ++j) {
          const int i = lo + 4 * (kCThreads * j + tid);
          if (i < Tv) {
            float e[4] = {0.f, 0.f, 0.f, 0.f}, cs[4] = {0.f, 0.f, 0.f, 0.f};
            if (i + 3 < Tv) {
              const float4 a4 = __ldg(reinterpret_cast<const float4*>(dEu + i));
              const float4 b4 = __ldg(reinterpret_cast<const float4*>(cvu + i));
              e[0] = a4.x; e[1] = a4.y; e[2] = a4.z; e[3] = a4.w;
              cs[0] = b4.x; cs[1] = b4.y; cs[2] = b4.z; cs[3] = b4.w;
            } else {
              for (int r = 0; r < 4 && i + r < Tv; ++r) {
                e[r] = __ldg(dEu + i + r);
                cs[r] = __ldg(cvu + i + r);
              }
            }
  #pragma unroll
            for (int r = 0; r < 4; ++r)
              if (i + r < Tv) {
                if (wins) {
                  e[r] = fminf(fmaxf(e[r], mnE), wmax);
                  wsumf = __fadd_rn(wsumf, e[r]);
                } else if (madv) {
                  e[r] = mad_logistic(e[r], mmed, minv);
                  wsumf = __fadd_rn(wsumf, e[r]);
                }
                const float sd = sdiv_rcp(e[r], cs[r], mnE, invE, f.alpha, mix);
                sm.raw[pad_idx(i + r - lo + kHalo)] = sd;
                mnD = fminf(mnD, sd);
                mxD = fmaxf(mxD, sd);
              }
          }
        }
      } else {
  #pragma unroll 8
        for (int j = 0; j < kJ; ++j) {
          const int i = lo + kCThreads * j + tid;
          if (i < Tv) {
            float e = __ldg(dEu + i);
            if (wins) {
              e = fminf(fmaxf(e, mnE), wmax);
              wsumf = __fadd_rn(wsumf, e);
            } else if (madv) {
              e = mad_logistic(e, mmed, minv);
              wsumf = __fadd_rn(wsumf, e);
            }
            const float sd = sdiv_rcp(e, __ldg(cvu + i), mnE, invE, f.alpha, mix);
            sm.raw[pad_idx(i - lo + kHalo)] = sd;
            mnD = fminf(mnD, sd);
            mxD = fmaxf(mxD, sd);
          }
        }
      }
    }
    if (wins || madv) {
      double wsum = (double)wsumf;
  #pragma unroll
      for (int o = 16; o > 0; o >>= 1) wsum += __shfl_xor_sync(0xffffffffu, wsum, o);
      if (lane == 0) sm.dredw[warp] = wsum;
    }
  #pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      mnD = fminf(mnD, __shfl_xor_sync(0xffffffffu, mnD, o));
      mxD = fmaxf(mxD, __shfl_xor_sync(0xffffffffu, mxD, o));
    }
    if (lane == 0) {
      sm.red[warp][6] = mnD;
      sm.red[warp][7] = mxD;
    }
    __syncthreads();
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    if (tid == 0) {
      float a0 = sm.red[0][6], a1 = sm.red[0][7];
      for (int w = 1; w < kCWarps; ++w) {
        a0 = fminf(a0, sm.red[w][6]);
        a1 = fmaxf(a1, sm.red[w][7]);
      }
      push_all<kMaxC>(cl, &sm.ext_all[rank][0], a0, C);
      push_all<kMaxC>(cl, &sm.ext_all[rank][1], a1, C);
      if (kVar && f.vnorm != nullptr) {
        double cs = 0.0;
        for (int w = 0; w < kCWarps; ++w) cs += sm.dred[w];
        push_all<kMaxC>(cl, &sm.simp_all[rank], cs, C);
      }
      if (wins || madv) {
        double cs = 0.0;
        for (int w = 0; w < kCWarps; ++w) cs += sm.dredw[w];
        push_all<kMaxC>(cl, &sm.wsum_all[rank], cs, C);
      }
    }
    cl.sync();
    if (tid == 0) {
      float a0 = INFINITY, a1 = -INFINITY;
      for (int r = 0; r < C; ++r) {
        a0 = fminf(a0, sm.ext_all[r][0]);
        a1 = fmaxf(a1, sm.ext_all[r][1]);
      }
      const float denD = __fadd_rn(__fsub_rn(a1, a0), f.eps);
      // mean(S_imp) / mean(Sbar) with Sbar = (S_div - a0) / denD
      double dsc1 = sm.dsc[1];  // Tv * mean(S_div)
      if (wins || madv) {  // s_E from the clipped distances (or s_E itself): that sum replaces the sum of d_E
        double sum_clip = 0.0;
        for (int r = 0; r < C; ++r) sum_clip += sm.wsum_all[r];
        const double T = (double)Tv, s_c = (double)sm.sc[4];
        const double sum_sE = (sum_clip - (double)mnE * T) / (double)denE;
        const double sum_sC = mix ? -s_c : (T - s_c) * 0.5;
        dsc1 = (double)f.alpha * sum_sE + (1.0 - (double)f.alpha) * sum_sC;
      }
      const double num = dsc1 - (double)a0 * (double)Tv;  // Tv * denD * mean(Sbar)
      sm.sc[6] = a0;
      sm.sc[7] = denD;
      double dsc0 = sm.dsc[0];  // kp * Tv * mean(S_imp)
      if (kVar && f.vnorm != nullptr) {
        double sum_imp = 0.0;
        for (int r = 0; r < C; ++r) sum_imp += sm.simp_all[r];
        dsc0 = (double)f.pool * sum_imp;
      }
      sm.sc[5] = (Tv > 0 && num > 0.0) ? (float)(dsc0 * (double)denD / ((double)f.pool * num)) : 0.f;
    }
    __syncthreads();
    const float lamf = sm.sc[0], mnD2 = sm.sc[6], denD = sm.sc[7], scale = sm.sc[5];
    const float invD = __frcp_rn(denD);
    const float one_m_lam = __fsub_rn(1.f, lamf);

    // 3. final scores (Eq. 7); the keys replace the pooled importance, and
    //    the scores go out through the staging buffer in coalesced order
  #pragma unroll
    for (int c = 0; c < kJ; ++c) {
      const float sd = sm.raw[pad_idx(q0 + c)];
      const float sbar = __fmul_rn(__fsub_rn(sd, mnD2), invD);
      const float S = __fadd_rn(__fmul_rn(lamf, __fmul_rn(sbar, scale)), __fmul_rn(one_m_lam, __uint_as_float(key[c])));
      key[c] = ordered_key(S);
      sm.raw[pad_idx(q0 + c)] = S;
    }
    if (f.dbg != nullptr) {
      // per-candidate terms for inspection: raw vote, pooled importance, d_E,
      // cosine, S_div, recomputed by the same operations (kept out of the
      // loop above, whose code size sets its speed)
      float* dbg = f.dbg + (size_t)u * 5 * Tv;
      const float* dEu = f.dE + (size_t)u * Tv;
      const float* cvu = f.cosv + (size_t)u * Tv;
      const float inv_pool = __frcp_rn((float)f.pool);
  #pragma unroll 1
      for (int c = 0; c < nv; ++c) {
        const int i = c0 + c;
        float acc = 0.f;
        for (int o = -hpool; o <= hpool; ++o)
          if (i + o >= 0 && i + o < Tv) acc = __fadd_rn(acc, __ldg(raw + i + o));
        const float e = __ldg(dEu + i), cs = __ldg(cvu + i);
        dbg[i] = __ldg(raw + i);
        dbg[Tv + i] = __fmul_rn(acc, inv_pool);
        dbg[2 * Tv + i] = e;
        dbg[3 * Tv + i] = cs;
        const float ev = wins ? fminf(fmaxf(e, mnE), wmax) : madv ? mad_logistic(e, mmed, minv) : e;
        dbg[4 * Tv + i] = sdiv_rcp(ev, cs, mnE, invE, f.alpha, mix);
      }
    }
    if (f.S != nullptr) {
      __syncthreads();
      float* Sg = f.S + (size_t)u * Tv;
      if (vec4) {
  #pragma unroll 4
        for (int j = 0; j < kJ / 4; ++j) {
          const int i = lo + 4 * (kCThreads * j + tid);
          const int q = i - lo + kHalo;
          if (i + 3 < Tv) {
            *reinterpret_cast<float4*>(Sg + i) =
                make_float4(sm.raw[pad_idx(q)], sm.raw[pad_idx(q + 1)], sm.raw[pad_idx(q + 2)], sm.raw[pad_idx(q + 3)]);
          } else {
            for (int r = 0; r < 4 && i + r < Tv; ++r) Sg[i + r] = sm.raw[pad_idx(q + r)];
          }
        }
      } else {
  #pragma unroll 8
        for (int j = 0; j < kJ; ++j) {
          const int i = lo + kCThreads * j + tid;
          if (i < Tv) Sg[i] = sm.raw[pad_idx(i - lo + kHalo)];
        }
      }
    }
  }

  if (kSelect) {
    // 4. radix select of the k-th largest key over the cluster
    unsigned prefix = 0u, mask = 0u;
    int rem = k;
    if (k > 0) {
      int pass = 0;
      for (int shift = 24; shift >= 0; shift -= 8, ++pass) {
        // each warp counts into its own histogram, a thread adding runs of
        // equal bins among its consecutive candidates (neighbouring scores
        // share their leading bits), then the CTA's histogram is the sum of
        // its warps'
        unsigned* wh = sm.whist[warp];
#pragma unroll
        for (int b = lane; b < 256; b += 32) wh[b] = 0u;
        __syncwarp();
        unsigned cur = 0u, run = 0u;
#pragma unroll
        for (int c = 0; c < kJ; ++c) {
          if (c < nv && (key[c] & mask) == prefix) {
            const unsigned bin = (key[c] >> shift) & 255u;
            if (bin != cur) {
              if (run) atomicAdd(&wh[cur], run);
              cur = bin;
              run = 0u;
            }
            ++run;
          }
        }
        if (run) atomicAdd(&wh[cur], run);
        __syncthreads();
        {
          unsigned cnt = 0u;  // kCThreads == 256 bins: thread tid sums bin tid
#pragma unroll
          for (int w = 0; w < kCWarps; ++w) cnt += sm.whist[w][tid];
          push_all<kMaxC>(cl, &sm.hall[pass & 1][rank][tid], cnt, C);
        }
        cl.sync();
        // the cluster's histogram (rank order: deterministic), bin tid; suffix
        // sums from the top bin find the bin holding the rem-th largest key
        unsigned tot = 0u;
#pragma unroll
        for (int r = 0; r < kMaxC; ++r)
          if (r < C) tot += sm.hall[pass & 1][r][tid];
        unsigned suf = tot;  // sum of bins tid .. 32 * warp + 31
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned y = __shfl_down_sync(0xffffffffu, suf, o);
          if (lane + o < 32) suf += y;
        }
        if (lane == 0) sm.wsum[warp] = suf;
        __syncthreads();
        for (int w = warp + 1; w < kCWarps; ++w) suf += sm.wsum[w];
        // suf = keys in bins >= tid; the wanted bin has suf >= rem > suf - tot
        if (suf >= (unsigned)rem && suf - tot < (unsigned)rem) {
          sm.shi[1] = tid;
          sm.shi[2] = rem - (int)(suf - tot);
        }
        __syncthreads();
        prefix |= (unsigned)sm.shi[1] << shift;
        mask |= 255u << shift;
        rem = sm.shi[2];
        // (the next write of shi follows the next pass's first barrier, which
        // every thread reaches only after reading this one)
      }
    }
    const unsigned thr = prefix;

    // 5. kept candidates: above the threshold, or equal to it among the first
    //    `rem` equal ones by position, emitted in ascending position
    int n_gt = 0, n_eq = 0;
    if (k > 0) {
#pragma unroll
      for (int c = 0; c < kJ; ++c)
        if (c < nv) {
          n_gt += key[c] > thr;
          n_eq += key[c] == thr;
        }
    }
    // exclusive prefix over the threads of the CTA (position order)
    int gi = n_gt, ei = n_eq;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int yg = __shfl_up_sync(0xffffffffu, gi, o), ye = __shfl_up_sync(0xffffffffu, ei, o);
      if (lane >= o) {
        gi += yg;
        ei += ye;
      }
    }
    if (lane == 31) {
      sm.wscan[warp][0] = gi;
      sm.wscan[warp][1] = ei;
    }
    __syncthreads();
    int gt_excl = gi - n_gt, eq_excl = ei - n_eq;
    for (int w = 0; w < warp; ++w) {
      gt_excl += sm.wscan[w][0];
      eq_excl += sm.wscan[w][1];
    }
    if (tid == 0) {
      int g = 0, q = 0;
      for (int w = 0; w < kCWarps; ++w) {
        g += sm.wscan[w][0];
        q += sm.wscan[w][1];
      }
      push_all<kMaxC>(cl, &sm.cnt_all[rank][0], g, C);
      push_all<kMaxC>(cl, &sm.cnt_all[rank][1], q, C);
    }
    cl.sync();
    // candidates kept by lower ranks, and the ties they took
    int pos = 0, eq_before = 0;
    for (int r = 0; r < rank; ++r) {
      const int g = sm.cnt_all[r][0], q = sm.cnt_all[r][1];
      pos += g + max(0, min(q, rem - eq_before));
      eq_before += q;
    }
    // ties still to take from this CTA on, in position order
    const int ties = max(0, rem - eq_before);
    int p = pos + gt_excl + min(ties, eq_excl);
    int take_eq = max(0, min(n_eq, ties - eq_excl));
    int32_t* out = f.idx + (size_t)u * f.n_keep;
    if (k > 0) {
#pragma unroll
      for (int c = 0; c < kJ; ++c)
        if (c < nv) {
          bool take = key[c] > thr;
          if (!take && key[c] == thr && take_eq > 0) {
            take = true;
            --take_eq;
          }
          if (take) {
            if (p < k) out[p] = c0 + c;
            ++p;
          }
        }
    }
    if (keep_all) {
      // B >= N: every row in order; rank r writes its candidates, the last rank the window
      const int hi = min(Tv, lo + kCap);
      for (int i = lo + tid; i < hi; i += kCThreads) out[i] = i;
      if (rank == C - 1)
        for (int j = tid; j < f.W; j += kCThreads) out[Tv + j] = Tv + j;
    } else if (rank == C - 1) {
      for (int j = tid; j < f.W; j += kCThreads) out[k + j] = Tv + j;
    }
    if (rank == C - 1)  // slots past this unit's budget (per-layer budgets) hold -1
      for (int r = (keep_all ? f.N : budget) + tid; r < f.n_keep; r += kCThreads) out[r] = -1;
  }
  // No CTA touches a peer's shared memory after the last cluster barrier it
  // passed (every exchange is a store made before that barrier), so the
  // CTAs may leave independently.
}

template <int kSh>
cudaError_t set_attrs() {
  const int bytes = (int)sizeof(ClusterSmem<kSh>);
  const void* kernels[5] = {(const void*)finalize_cluster_kernel<0, kSh, false>,
                            (const void*)finalize_cluster_kernel<1, kSh, false>,
                            (const void*)finalize_cluster_kernel<0, kSh, true>,
                            (const void*)finalize_cluster_kernel<1, kSh, true>,
                            (const void*)finalize_cluster_kernel<2, kSh, false>};
  for (const void* k : kernels) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && Shape<kSh>::kMaxCluster > 8)
      e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

template <int kSh>
cudaError_t launch_shape(const FinalArgs& f, int U, int C, bool select_only, cudaStream_t s) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(U * C), 1, 1);
  cfg.blockDim = dim3(kCThreads, 1, 1);
  cfg.dynamicSmemBytes = sizeof(ClusterSmem<kSh>);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const bool var = f.vnorm != nullptr || f.wlo != nullptr || f.mad != nullptr;
  if (select_only) return cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<2, kSh, false>, f);
  if (f.idx == nullptr)
    return var ? cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<0, kSh, true>, f)
               : cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<0, kSh, false>, f);
  return var ? cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<1, kSh, true>, f)
             : cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<1, kSh, false>, f);
}

// Per device: the attributes set, and whether clusters of 16 CTAs of the
// long shape can be resident (cudaOccupancyMaxActiveClusters > 0).
std::atomic<int> g_setup[64];  // 0 = not yet, 1 = set, clusters of 16 unavailable, 2 = set and available

int device_setup() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  int st = g_setup[dev].load();
  if (st != 0) return st;
  if (set_attrs<0>() != cudaSuccess || set_attrs<1>() != cudaSuccess) return -1;
  st = 1;
  if (set_attrs<2>() == cudaSuccess) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(16u * 16u, 1, 1);
    cfg.blockDim = dim3(kCThreads, 1, 1);
    cfg.dynamicSmemBytes = sizeof(ClusterSmem<2>);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 16;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, (const void*)finalize_cluster_kernel<1, 2, false>, &cfg) == cudaSuccess &&
        n > 0)
      st = 2;
  }
  cudaGetLastError();  // an unavailable configuration leaves no error behind
  g_setup[dev].store(st);
  return st;
}

// Shape and cluster size for units of Tv candidates; shape -1 when no cluster
// shape takes them.
void pick_shape(int Tv, int long_ok, int& sh, int& C) {
  const int t = Tv > 0 ? Tv : 1;
  const int C16 = (t + Shape<0>::kCap - 1) / Shape<0>::kCap;
  const int C32 = (t + Shape<1>::kCap - 1) / Shape<1>::kCap;
  if (C16 <= 4) {
    sh = 0;
    C = C16;
  } else if (C32 <= Shape<1>::kMaxCluster) {
    sh = 1;
    C = C32;
  } else if (C32 <= (long_ok ? Shape<2>::kMaxCluster : 8)) {
    sh = 2;
    C = C32;
  } else {
    sh = -1;
    C = 0;
  }
}

}  // namespace

bool cluster_finalize_fits(int Tv) {
  const int st = device_setup();
  if (st < 0) return false;
  int sh, C;
  pick_shape(Tv, st == 2, sh, C);
  return sh >= 0;
}

cudaError_t launch_finalize_cluster(const FinalArgs& f, int U, bool select_only, cudaStream_t s) {
  const int st = device_setup();
  if (st < 0) return cudaErrorUnknown;
  int sh, C;
  pick_shape(f.Tv, st == 2, sh, C);
  switch (sh) {
    case 0: return launch_shape<0>(f, U, C, select_only, s);
    case 1: return launch_shape<1>(f, U, C, select_only, s);
    case 2: return launch_shape<2>(f, U, C, select_only, s);
  }
  return cudaErrorNotSupported;
}

}  // namespace ecokv
