// Finalisation and selection of one (layer, KV head) unit by a thread-block
// cluster of C CTAs (C <= 8): the arithmetic of finalize_unit / select_unit
// (finalize_select.cuh), spread over the cluster so that every SM takes part,
// with the cluster-wide reductions done through distributed shared memory.
//
// CTA rank r of the cluster owns candidates [r * cap, (r + 1) * cap) of the
// unit (cap = 8 warps x 32 lanes x kJ); warp w of it owns a contiguous span of
// 32 * kJ of those, lane l position span0 + 32 j + l for j < kJ, kept in
// registers from the first load to the emitted index.  Steps:
//   1. unit scalars from the pass-2 partials (every CTA, same inputs, same
//      result), lambda (Eq. 4-6);
//   2. S_div (Eq. 2, 3) and pooled S_imp of the owned candidates; extrema of
//      S_div over the cluster;
//   3. S (Eq. 7) as finalize_unit computes it, divisions by the min-max
//      ranges and the pooling kernel taken as reciprocal products;
//   4. MSB-first radix select over the order-preserving image of S, one
//      256-bin histogram per CTA, summed over the cluster for each 8-bit digit;
//   5. counts of keys above / equal to the threshold, exchanged so that each
//      CTA knows how many kept candidates precede it (ties to the lower
//      position), then its kept positions in ascending order (the last CTA
//      adds the window).  The gather of the kept rows is its own launch.
// Cluster barriers are reached by every CTA on every path (no early exit).

#include <cooperative_groups.h>

#include "finalize_select.cuh"

namespace cg = cooperative_groups;

namespace ecokv {
namespace {

constexpr int kCThreads = 256;
constexpr int kCWarps = kCThreads / 32;
constexpr int kJ = 16;                          // candidates a thread owns
constexpr int kCap = kCThreads * kJ;            // candidates a CTA owns
constexpr int kMaxCluster = 8;
constexpr int kHalo = 16;                       // pooling halo kept in shared memory (kernel <= 33)

struct ClusterSmem {
  float rawS[kCap + 2 * kHalo];  // the CTA's raw votes with the pooling halo
  unsigned buf[kCap];            // pooled importance, then the order-preserving keys of S
  unsigned hist[2][256];         // per radix pass, the CTA's sum (double-buffered across passes)
  unsigned whist[kCWarps][256];  // per radix pass, each warp's own histogram
  float red[kCWarps][8];         // per-warp partials
  float edge[32];                // pooling edge values
  float sc[8];                   // broadcast scalars
  float ext[2];                  // this CTA's min / max of S_div
  int cnt[2];                    // this CTA's keys above / equal to the threshold
  unsigned wsum[kCWarps];
  int shi[32];
};

// Composite diversity (Eq. 2 and Eq. 3) with the min-max divisor applied as a
// reciprocal (one rounding more than a division; every score of a call uses
// the same formula, and ecokv_score and ecokv_evict share this kernel).
__device__ __forceinline__ float sdiv_rcp(float dE, float c, float mnE, float invE, float alpha, bool mix) {
  const float sE = __fmul_rn(__fsub_rn(dE, mnE), invE);
  const float sC = mix ? -c : __fmul_rn(__fsub_rn(1.f, c), 0.5f);
  return __fadd_rn(__fmul_rn(alpha, sE), __fmul_rn(__fsub_rn(1.f, alpha), sC));
}

// kMode: 0 = scores, 1 = scores and top-k, 2 = top-k of given scores (f.S).
template <int kMode>
__global__ void __launch_bounds__(kCThreads, 4) finalize_cluster_kernel(FinalArgs f) {
  constexpr bool kSelect = kMode != 0;
  extern __shared__ __align__(16) uint8_t fc_smem[];
  ClusterSmem& sm = *reinterpret_cast<ClusterSmem*>(fc_smem);
  cg::cluster_group cl = cg::this_cluster();
  const int C = (int)cl.num_blocks();
  const int rank = (int)cl.block_rank();
  const int u = blockIdx.x / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int Tv = f.Tv;
  const int lo = rank * kCap;                      // first candidate of this CTA
  const int span0 = lo + warp * 32 * kJ;           // first candidate of this warp
  const bool keep_all = f.budget >= f.N;
  const int k = keep_all ? 0 : f.budget - f.W;
  const bool mix = (f.flags & ECOKV_FLAG_SC_MIXKV_SIGN) != 0;
  const int hpool = f.pool >> 1;
  const bool pool_smem = hpool <= kHalo;
  const float* us = f.ustat + (size_t)u * f.ustat_stride;
  const float* raw = f.simp + (size_t)u * Tv;
  const float* dEp = f.dE + (size_t)u * Tv;
  const float* cvp = f.cosv + (size_t)u * Tv;

  if (kMode == 2) {
    // scores given (absent when nothing is to be chosen): their
    // order-preserving keys
    if (k > 0)
      for (int j = 0; j < kJ; ++j) {
        const int i = span0 + 32 * j + lane;
        if (i < Tv) sm.buf[i - lo] = ordered_key(__ldg(f.S + (size_t)u * Tv + i));
      }
  } else {
    // 1. the six pass-2 partials (sum over all N of d_E, min / max / sum of
    //    d_E, sums of cosines and of raw votes over the candidates); meanwhile
    //    the CTA's raw votes with the pooling halo and the edge values
    // this thread's d_E and cosines, in flight through the scalar phase
    float e_[kJ], c_[kJ];
#pragma unroll
    for (int j = 0; j < kJ; ++j) {
      const int i = span0 + 32 * j + lane;
      e_[j] = i < Tv ? __ldg(dEp + i) : 0.f;
      c_[j] = i < Tv ? __ldg(cvp + i) : 0.f;
    }
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
    if (pool_smem)
      for (int q = tid; q < kCap + 2 * hpool; q += kCThreads) {
        const int j = lo - hpool + q;
        sm.rawS[q] = (j >= 0 && j < Tv) ? __ldg(raw + j) : 0.f;
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
    // pooled importance of the owned candidates (needs no unit scalar)
    const float inv_pool = __frcp_rn((float)f.pool);
  #pragma unroll 4
    for (int j = 0; j < kJ; ++j) {
      const int i = span0 + 32 * j + lane;
      if (i < Tv) {
        float sp;
        if (pool_smem) {
          // the same sum, in the same order, as pooled(); halo entries outside
          // [0, Tv) hold +0 and leave it unchanged
          const float* r0 = sm.rawS + (i - lo);
          float acc = 0.f;
          if (hpool == 2) {  // the default kernel of 5, loads in parallel
            const float x0 = r0[0], x1 = r0[1], x2 = r0[2], x3 = r0[3], x4 = r0[4];
            acc = __fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(__fadd_rn(acc, x0), x1), x2), x3), x4);
          } else {
            for (int o = 0; o <= 2 * hpool; ++o) acc = __fadd_rn(acc, r0[o]);
          }
          sp = __fmul_rn(acc, inv_pool);
        } else {
          float acc = 0.f;
          for (int o = -hpool; o <= hpool; ++o)
            if (i + o >= 0 && i + o < Tv) acc = __fadd_rn(acc, __ldg(raw + i + o));
          sp = __fmul_rn(acc, inv_pool);
        }
        sm.buf[i - lo] = __float_as_uint(sp);
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
      // per-head redundancy and lambda (Eq. 4-6), a few scalar ops in double
      const double N = (double)f.N;
      const double D_E = (double)s_all / N;
      const double tau = f.tau > 0.f ? (double)f.tau : sqrt((double)kD);
      const double r_E = 2.0 - 2.0 / (1.0 + exp(-D_E / tau));
      const double mu_sq = (double)__ldg(us + ustat_musq());
      const double r_C = f.N == 1 ? 1.0 : (N * mu_sq - 1.0) / (N - 1.0);
      double lam = (double)f.beta * r_E + (1.0 - (double)f.beta) * r_C;
      if (f.flags & ECOKV_FLAG_LAMBDA_OVERRIDE) lam = (double)f.lambda_override;
      sm.sc[0] = (float)lam;
      sm.sc[1] = mnE;
      sm.sc[2] = __fadd_rn(__fsub_rn(mxE, mnE), f.eps);
      sm.sc[3] = s_de;
      sm.sc[4] = s_c;
      sm.sc[5] = s_raw;
      if (f.lambda != nullptr && rank == 0) f.lambda[u] = (float)lam;
    }
    __syncthreads();
    const float lamf = sm.sc[0], mnE = sm.sc[1], denE = sm.sc[2];
    const float invE = __frcp_rn(denE);

    // 2. S_div (Eq. 2, 3) of the owned candidates and its extrema
    float mnD = INFINITY, mxD = -INFINITY;
  #pragma unroll
    for (int j = 0; j < kJ; ++j) {
      const int i = span0 + 32 * j + lane;
      if (i < Tv) {
        const float sd = sdiv_rcp(e_[j], c_[j], mnE, invE, f.alpha, mix);
        mnD = fminf(mnD, sd);
        mxD = fmaxf(mxD, sd);
      }
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
    if (tid == 0) {
      float a0 = sm.red[0][6], a1 = sm.red[0][7];
      for (int w = 1; w < kCWarps; ++w) {
        a0 = fminf(a0, sm.red[w][6]);
        a1 = fmaxf(a1, sm.red[w][7]);
      }
      sm.ext[0] = a0;
      sm.ext[1] = a1;
    }
    cl.sync();
    if (tid == 0) {
      float a0 = INFINITY, a1 = -INFINITY;
      for (int r = 0; r < C; ++r) {
        const float* pe = cl.map_shared_rank(sm.ext, r);
        a0 = fminf(a0, pe[0]);
        a1 = fmaxf(a1, pe[1]);
      }
      const float denD = __fadd_rn(__fsub_rn(a1, a0), f.eps);
      // means: sum_i S_imp(i) = (1/kp) sum_j raw(j) cnt(j), where cnt(j) = kp
      // except within kp/2 of either end; mean(Sbar) is affine in the means of
      // d_E and of the cosine (as finalize_unit)
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
      const double sum_imp = ((double)f.pool * (double)sm.sc[5] - edge) / (double)f.pool;
      const double mean_imp = Tv > 0 ? sum_imp / Tv : 0.0;
      const double mean_sE = Tv > 0 ? ((double)sm.sc[3] / Tv - (double)mnE) / (double)denE : 0.0;
      const double mean_cs = Tv > 0 ? (double)sm.sc[4] / Tv : 0.0;
      const double mean_sC = mix ? -mean_cs : (1.0 - mean_cs) * 0.5;
      const double mean_div = (double)f.alpha * mean_sE + (1.0 - (double)f.alpha) * mean_sC;
      const double mean_sbar = (mean_div - (double)a0) / (double)denD;
      sm.sc[6] = a0;
      sm.sc[7] = denD;
      sm.sc[5] = mean_sbar > 0.0 ? (float)(mean_imp / mean_sbar) : 0.f;
    }
    __syncthreads();
    const float mnD2 = sm.sc[6], denD = sm.sc[7], scale = sm.sc[5];
    const float invD = __frcp_rn(denD);
    const float one_m_lam = __fsub_rn(1.f, lamf);

    // 3. final scores (Eq. 7); the order-preserving keys replace the pooled
    //    importance in buf
    float* Sg = f.S ? f.S + (size_t)u * Tv : nullptr;
    float* dbg = f.dbg ? f.dbg + (size_t)u * 5 * Tv : nullptr;
  #pragma unroll
    for (int j = 0; j < kJ; ++j) {
      const int i = span0 + 32 * j + lane;
      if (i < Tv) {
        const float e = e_[j], c = c_[j];
        const float sd = sdiv_rcp(e, c, mnE, invE, f.alpha, mix);
        const float sbar = __fmul_rn(__fsub_rn(sd, mnD2), invD);
        const float sp = __uint_as_float(sm.buf[i - lo]);
        const float S = __fadd_rn(__fmul_rn(lamf, __fmul_rn(sbar, scale)), __fmul_rn(one_m_lam, sp));
        sm.buf[i - lo] = ordered_key(S);
        if (Sg) Sg[i] = S;
        if (dbg) {
          dbg[i] = __ldg(raw + i);
          dbg[Tv + i] = sp;
          dbg[2 * Tv + i] = e;
          dbg[3 * Tv + i] = c;
          dbg[4 * Tv + i] = sd;
        }
      }
    }
  }

  if (kSelect) {
    // 4. radix select of the k-th largest key over the cluster (each thread
    //    reads back only the keys it wrote)
    unsigned prefix = 0u, mask = 0u;
    int rem = k;
    if (k > 0) {
      int pass = 0;
      for (int shift = 24; shift >= 0; shift -= 8, ++pass) {
        // each warp counts into its own histogram (no two warps contend for
        // one address: the keys of a head crowd into few bins), then the
        // CTA's histogram is their sum
        unsigned* wh = sm.whist[warp];
#pragma unroll
        for (int b = lane; b < 256; b += 32) wh[b] = 0u;
        __syncwarp();
#pragma unroll 4
        for (int j = 0; j < kJ; ++j) {
          const int i = span0 + 32 * j + lane;
          unsigned bin = 0xffffffffu;
          if (i < Tv) {
            const unsigned key = sm.buf[i - lo];
            if ((key & mask) == prefix) bin = (key >> shift) & 255u;
          }
          const unsigned peers = __match_any_sync(0xffffffffu, bin);
          if (bin != 0xffffffffu && lane == __ffs(peers) - 1) atomicAdd(&wh[bin], (unsigned)__popc(peers));
        }
        __syncthreads();
        unsigned* hist = sm.hist[pass & 1];
        {
          unsigned cnt = 0u;  // kCThreads == 256 bins: thread tid sums bin tid
#pragma unroll
          for (int w = 0; w < kCWarps; ++w) cnt += sm.whist[w][tid];
          hist[tid] = cnt;
        }
        cl.sync();
        // the cluster's histogram (rank order: deterministic), bin tid; suffix
        // sums from the top bin find the bin holding the rem-th largest key
        unsigned tot = 0u;
        for (int r = 0; r < C; ++r) tot += cl.map_shared_rank(hist, r)[tid];
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
        __syncthreads();
      }
    }
    const unsigned thr = prefix;

    // 5. kept candidates: above the threshold, or equal to it among the first
    //    `rem` equal ones by position, emitted in ascending position
    const unsigned lt = (1u << lane) - 1u;
    int n_gt = 0, n_eq = 0;
    if (k > 0) {
#pragma unroll 4
      for (int j = 0; j < kJ; ++j) {
        const int i = span0 + 32 * j + lane;
        const unsigned key = i < Tv ? sm.buf[i - lo] : 0u;
        n_gt += __popc(__ballot_sync(0xffffffffu, i < Tv && key > thr));
        n_eq += __popc(__ballot_sync(0xffffffffu, i < Tv && key == thr));
      }
    }
    if (lane == 0) {
      sm.shi[8 + warp] = n_gt;
      sm.shi[16 + warp] = n_eq;
    }
    __syncthreads();
    if (tid == 0) {
      int g = 0, q = 0;
      for (int w = 0; w < kCWarps; ++w) {
        g += sm.shi[8 + w];
        q += sm.shi[16 + w];
      }
      sm.cnt[0] = g;
      sm.cnt[1] = q;
    }
    cl.sync();
    // candidates kept by lower ranks, and the ties they took
    int pos = 0, eq_before = 0;
    for (int r = 0; r < rank; ++r) {
      const int* pc = cl.map_shared_rank(sm.cnt, r);
      const int g = pc[0], q = pc[1];
      const int tq = max(0, min(q, rem - eq_before));
      pos += g + tq;
      eq_before += q;
    }
    // within the CTA: warps in order
    int w_eq_before = eq_before, w_pos = pos;
    for (int w = 0; w < warp; ++w) {
      const int q = sm.shi[16 + w];
      const int tq = max(0, min(q, rem - w_eq_before));
      w_pos += sm.shi[8 + w] + tq;
      w_eq_before += q;
    }
    const int take_eq = max(0, min(n_eq, rem - w_eq_before));
    int32_t* out = f.idx + (size_t)u * f.n_keep;
    int eq_seen = 0;
    if (k > 0) {
#pragma unroll 4
      for (int j = 0; j < kJ; ++j) {
        const int i = span0 + 32 * j + lane;
        const unsigned key = i < Tv ? sm.buf[i - lo] : 0u;
        const bool gt = i < Tv && key > thr;
        const bool eq = i < Tv && key == thr;
        const unsigned eqm = __ballot_sync(0xffffffffu, eq);
        const bool take = gt || (eq && eq_seen + __popc(eqm & lt) < take_eq);
        const unsigned sel = __ballot_sync(0xffffffffu, take);
        if (take) {
          const int p = w_pos + __popc(sel & lt);
          if (p < k) out[p] = i;
        }
        w_pos += __popc(sel);
        eq_seen += __popc(eqm);
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
  }
  cl.sync();  // no CTA leaves while a peer may still read its shared memory
}

}  // namespace

// Scores (and with f.idx the top-k) of every unit, or with select_only the
// top-k of the scores in f.S; one cluster per unit; cudaErrorNotSupported
// when Tv exceeds what eight CTAs hold.
cudaError_t launch_finalize_cluster(const FinalArgs& f, int U, bool select_only, cudaStream_t s) {
  const int C = f.Tv <= 0 ? 1 : (f.Tv + kCap - 1) / kCap;
  if (C > kMaxCluster) return cudaErrorNotSupported;
  static bool attr_set[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!attr_set[dev]) {
    const int bytes = (int)sizeof(ClusterSmem);
    if ((e = cudaFuncSetAttribute(finalize_cluster_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  bytes)) != cudaSuccess ||
        (e = cudaFuncSetAttribute(finalize_cluster_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  bytes)) != cudaSuccess ||
        (e = cudaFuncSetAttribute(finalize_cluster_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  bytes)) != cudaSuccess)
      return e;
    attr_set[dev] = true;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(U * C), 1, 1);
  cfg.blockDim = dim3(kCThreads, 1, 1);
  cfg.dynamicSmemBytes = sizeof(ClusterSmem);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (select_only) return cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<2>, f);
  if (f.idx == nullptr) return cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<0>, f);
  return cudaLaunchKernelEx(&cfg, finalize_cluster_kernel<1>, f);
}

}  // namespace ecokv
