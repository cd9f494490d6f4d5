// Order statistics of d_E per unit for the robust forms of Eq. 2 (the
// normalisation ablation of Appendix B): the winsorised min-max's clip bounds,
// and for MAD scaling the median of d_E and the median of |d_E - median|.
//
// One CTA per unit: its Tv <= 32768 distances are read in coalesced order
// into shared memory as order-preserving keys, 64 thread-contiguous keys per
// thread (padded so that a quarter-warp's 16-byte reads fall in distinct
// banks), and an MSB-first radix select on the keys finds two ranks at once
// (longer rows are read from L2 until the keys left under the ranks'
// prefixes fit those slots, see os_select2_long):
// - the row's smallest and largest keys give the prefix every key shares;
// - one digit of up to 12 bits just below it, counted by direct atomics into
//   a block-wide histogram (the keys spread over its bins), and a suffix
//   scan give both ranks' bins;
// - each thread moves its keys under either rank's new prefix (a few per
//   row) to the front of its own keys, and the remaining digits run over
//   those short lists.
// Every loop is a short rolled loop over shared memory (a body unrolled over
// register-held keys overflows the instruction cache, every warp running it
// once), and nothing leaves the CTA between digits, so one launch finds both
// ranks (MAD: all four, the second pair over |d_E - median|) where a
// grid-wide select needs a launch per digit.

#include <atomic>

#include "ecokv_internal.cuh"
#include "finalize_select.cuh"

namespace ecokv {
namespace {

constexpr int kOsThreads = 512;
constexpr int kOsWarps = kOsThreads / 32;
constexpr int kOsPer = 64;  // keys a thread holds: kOsThreads * kOsPer = 32768
constexpr int kOsPad = 4;   // stage: thread t's keys at t (kOsPer + kOsPad)
constexpr int kOsSeg = kOsPer + kOsPad;
constexpr int kOsDigit = 12;  // widest digit
constexpr int kOsBins = 1 << kOsDigit;

struct OsSmem {
  unsigned hist[2][kOsBins];  // per selection, the counts of the current digit
  unsigned wt[2][8];          // per selection, the suffix totals of the scanning warps
  unsigned pfx[2], mask[2], rem[2];
  unsigned red[2][kOsWarps];  // per-warp smallest / largest key
  alignas(16) unsigned stage[kOsThreads * kOsSeg];
};

// Stage index of row position q (thread q / kOsPer's key q % kOsPer).
__device__ __forceinline__ int os_pad(int q) { return q + (q / kOsPer) * kOsPad; }

// The key of a value: of v, or with kDev of |v - m|.
template <bool kDev>
__device__ __forceinline__ unsigned os_key(float v, float m) {
  return ordered_key(kDev ? fabsf(__fsub_rn(v, m)) : v);
}

// The row's T values at xr into the stage as keys, coalesced; a thread
// issues all of its loads before its first store.
template <bool kDev>
__device__ __forceinline__ void os_stage(const float* xr, int T, float m, OsSmem& sm, int tid) {
  constexpr int kV = kOsPer / 4;  // 16-byte loads per thread
  if ((reinterpret_cast<uintptr_t>(xr) & 15u) == 0) {
    const int n4 = T >> 2;
    float4 v[kV];
#pragma unroll
    for (int r = 0; r < kV; ++r) {
      const int j = tid + r * kOsThreads;
      if (j < n4) v[r] = __ldg(reinterpret_cast<const float4*>(xr) + j);
    }
#pragma unroll
    for (int r = 0; r < kV; ++r) {
      const int j = tid + r * kOsThreads;  // 4 j .. 4 j + 3 stay in one thread's keys
      if (j < n4)
        *reinterpret_cast<uint4*>(&sm.stage[os_pad(4 * j)]) = make_uint4(
            os_key<kDev>(v[r].x, m), os_key<kDev>(v[r].y, m), os_key<kDev>(v[r].z, m), os_key<kDev>(v[r].w, m));
    }
    for (int q = 4 * n4 + tid; q < T; q += kOsThreads) sm.stage[os_pad(q)] = os_key<kDev>(__ldg(xr + q), m);
  } else {
#pragma unroll 1
    for (int q0 = 0; q0 < T; q0 += kV * kOsThreads) {
      float v[kV];
#pragma unroll
      for (int r = 0; r < kV; ++r) {
        const int q = q0 + tid + r * kOsThreads;
        if (q < T) v[r] = __ldg(xr + q);
      }
#pragma unroll
      for (int r = 0; r < kV; ++r) {
        const int q = q0 + tid + r * kOsThreads;
        if (q < T) sm.stage[os_pad(q)] = os_key<kDev>(v[r], m);
      }
    }
  }
}

// The digit of width w at `shift` of both selections from the counts: a
// suffix scan over the 2^w bins per selection (threads 0-255: selection 0,
// 256-511: 1; thread t owns bins t per .. t per + per - 1, visited from bin
// (t mod per) on, so that a warp's reads and clears fall in distinct banks
// but for pairs).  While the two
// prefixes agree both read the first histogram.  The state is read before
// the first barrier and written after the second; the histograms are
// cleared between the third and the fourth; so no thread sees a half-updated
// state, a cleared count or a stale one.
__device__ __forceinline__ void os_scan(OsSmem& sm, int shift, int w, int tid) {
  const int lane = tid & 31;
  const int s = tid >> 8, t = tid & 255, gw = (tid >> 5) & 7;
  const int nb = 1 << w, per = nb > 256 ? nb >> 8 : 1;
  const bool own = t * per < nb;
  const bool same = sm.pfx[0] == sm.pfx[1] && sm.mask[0] == sm.mask[1];
  const unsigned rem = sm.rem[s];
  const unsigned* h = sm.hist[same ? 0 : s] + t * per;
  __syncthreads();
  unsigned cnt = 0u;
  if (own)
    for (int q = 0; q < per; ++q) cnt += h[(q + t) & (per - 1)];
  unsigned suf = cnt;  // the keys in bins >= t per under the prefix
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned y = __shfl_down_sync(0xffffffffu, suf, o);
    if (lane + o < 32) suf += y;
  }
  if (lane == 0) sm.wt[s][gw] = suf;
  __syncthreads();
  for (int w2 = gw + 1; w2 < 8; ++w2) suf += sm.wt[s][w2];
  if (own && suf >= rem && suf - cnt < rem) {  // a bin of this thread holds the rem-th largest
    unsigned above = suf - cnt;
    for (int q = per - 1; q >= 0; --q) {
      const unsigned c = h[q];
      if (above + c >= rem) {
        sm.pfx[s] |= (unsigned)(t * per + q) << shift;
        sm.mask[s] |= (unsigned)(nb - 1) << shift;
        sm.rem[s] = rem - above;
        break;
      }
      above += c;
    }
  }
  __syncthreads();
  if (own) {
    unsigned* hc = sm.hist[s] + t * per;
    for (int q = 0; q < per; ++q) hc[(q + t) & (per - 1)] = 0u;  // ready for the next digit
  }
  __syncthreads();
}

__device__ __forceinline__ void os_tail(unsigned* seg, int n, OsSmem& sm, int left, int tid);

// The ka-th and kb-th largest of the staged keys, into sm.pfx[0] and
// sm.pfx[1]; the thread's keys at seg (nv of them) are reordered.  Enters
// after a barrier that ends the staging.
__device__ __forceinline__ void os_select2(unsigned* seg, int nv, OsSmem& sm, int ka, int kb, int tid) {
  const int lane = tid & 31, warp = tid >> 5;
  // the shared prefix: from the smallest and the largest key
  unsigned lo = 0xffffffffu, hi = 0u;
  const uint4* seg4 = reinterpret_cast<const uint4*>(seg);
#pragma unroll 2
  for (int c4 = 0; c4 < (nv >> 2); ++c4) {
    const uint4 k = seg4[c4];
    lo = min(min(lo, k.x), min(k.y, min(k.z, k.w)));
    hi = max(max(hi, k.x), max(k.y, max(k.z, k.w)));
  }
  for (int c = nv & ~3; c < nv; ++c) {
    lo = min(lo, seg[c]);
    hi = max(hi, seg[c]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  if (lane == 0) {
    sm.red[0][warp] = lo;
    sm.red[1][warp] = hi;
  }
  __syncthreads();
  lo = sm.red[0][0];
  hi = sm.red[1][0];
  for (int w = 1; w < kOsWarps; ++w) {
    lo = min(lo, sm.red[0][w]);
    hi = max(hi, sm.red[1][w]);
  }
  const int common = __clz(lo ^ hi);  // 32 when every key is equal
  const unsigned cmask = common == 32 ? 0xffffffffu : ~(0xffffffffu >> common);
  if (tid < 2) {
    sm.pfx[tid] = lo & cmask;
    sm.mask[tid] = cmask;
    sm.rem[tid] = (unsigned)(tid == 0 ? ka : kb);
  }
  __syncthreads();  // the state is set before any thread reads it
  int left = 32 - common;  // bits still to decide, the same in every thread
  if (left == 0) return;
  // first digit: every key (all share the prefix) into one histogram
  {
    const int w = min(kOsDigit, left), shift = left - w;
    const unsigned dm = (1u << w) - 1u;
#pragma unroll 2
    for (int c4 = 0; c4 < (nv >> 2); ++c4) {
      const uint4 k = seg4[c4];
      atomicAdd(&sm.hist[0][(k.x >> shift) & dm], 1u);
      atomicAdd(&sm.hist[0][(k.y >> shift) & dm], 1u);
      atomicAdd(&sm.hist[0][(k.z >> shift) & dm], 1u);
      atomicAdd(&sm.hist[0][(k.w >> shift) & dm], 1u);
    }
    for (int c = nv & ~3; c < nv; ++c) atomicAdd(&sm.hist[0][(seg[c] >> shift) & dm], 1u);
    os_scan(sm, shift, w, tid);
    left = shift;
  }
  if (left == 0) return;
  // the keys under either new prefix to the front of the thread's keys
  const unsigned p0 = sm.pfx[0], m0 = sm.mask[0], p1 = sm.pfx[1], m1 = sm.mask[1];
  int n = 0;
  for (int c4 = 0; c4 < ((nv + 3) >> 2); ++c4) {  // (writes never pass the keys read)
    const uint4 k4 = seg4[c4];
    const unsigned kk[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
    for (int r = 0; r < 4; ++r)
      if (4 * c4 + r < nv && ((kk[r] & m0) == p0 || (kk[r] & m1) == p1)) seg[n++] = kk[r];
  }
  os_tail(seg, n, sm, left, tid);
}

// The remaining digits (left bits below both prefixes) over the thread's
// short list of n keys at seg, the keys under either prefix.
__device__ __forceinline__ void os_tail(unsigned* seg, int n, OsSmem& sm, int left, int tid) {
  while (left > 0) {
    const int w = min(kOsDigit, left), shift = left - w;
    const unsigned dm = (1u << w) - 1u;
    const unsigned q0 = sm.pfx[0], n0 = sm.mask[0], q1 = sm.pfx[1], n1 = sm.mask[1];
    const bool same = q0 == q1 && n0 == n1;
    for (int c = 0; c < n; ++c) {
      const unsigned k = seg[c];
      if ((k & n0) == q0) atomicAdd(&sm.hist[0][(k >> shift) & dm], 1u);
      if (!same && (k & n1) == q1) atomicAdd(&sm.hist[1][(k >> shift) & dm], 1u);
    }
    os_scan(sm, shift, w, tid);
    left = shift;
  }
}

// The ka-th and kb-th largest keys of a row too long for the stage (T >
// kOsThreads * kOsPer), into sm.pfx[0] and sm.pfx[1]: the row is read from
// global memory (L2) for the shared prefix and then for whole radix digits,
// until every thread's keys under either prefix (of its positions tid, tid +
// kOsThreads, ...) fit its kOsPer stage slots; those keys are then copied to
// the slots at seg and the remaining digits run over them as for a short row.
template <bool kDev>
__device__ void os_select2_long(const float* xr, int T, float m, unsigned* seg, OsSmem& sm, int ka, int kb, int tid) {
  const int lane = tid & 31, warp = tid >> 5;
  unsigned lo = 0xffffffffu, hi = 0u;
  for (int q = tid; q < T; q += kOsThreads) {
    const unsigned k = os_key<kDev>(__ldg(xr + q), m);
    lo = min(lo, k);
    hi = max(hi, k);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  if (lane == 0) {
    sm.red[0][warp] = lo;
    sm.red[1][warp] = hi;
  }
  __syncthreads();
  lo = sm.red[0][0];
  hi = sm.red[1][0];
  for (int w = 1; w < kOsWarps; ++w) {
    lo = min(lo, sm.red[0][w]);
    hi = max(hi, sm.red[1][w]);
  }
  const int common = __clz(lo ^ hi);  // 32 when every key is equal
  const unsigned cmask = common == 32 ? 0xffffffffu : ~(0xffffffffu >> common);
  if (tid < 2) {
    sm.pfx[tid] = lo & cmask;
    sm.mask[tid] = cmask;
    sm.rem[tid] = (unsigned)(tid == 0 ? ka : kb);
  }
  __syncthreads();  // the state is set (and sm.red read) before any thread goes on
  int left = 32 - common;
  while (left > 0) {
    const unsigned p0 = sm.pfx[0], m0 = sm.mask[0], p1 = sm.pfx[1], m1 = sm.mask[1];
    unsigned cnt = 0u;
    for (int q = tid; q < T; q += kOsThreads) {
      const unsigned k = os_key<kDev>(__ldg(xr + q), m);
      cnt += ((k & m0) == p0 || (k & m1) == p1) ? 1u : 0u;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cnt = max(cnt, __shfl_xor_sync(0xffffffffu, cnt, o));
    if (lane == 0) sm.red[0][warp] = cnt;
    __syncthreads();
    unsigned mx = 0u;
    for (int w = 0; w < kOsWarps; ++w) mx = max(mx, sm.red[0][w]);
    if (mx <= (unsigned)kOsPer) break;  // the same decision in every thread
    // one digit over the whole row (os_scan's barriers order the next
    // iteration's writes to sm.red after these reads)
    const int w = min(kOsDigit, left), shift = left - w;
    const unsigned dm = (1u << w) - 1u;
    const bool same = p0 == p1 && m0 == m1;
    for (int q = tid; q < T; q += kOsThreads) {
      const unsigned k = os_key<kDev>(__ldg(xr + q), m);
      if ((k & m0) == p0) atomicAdd(&sm.hist[0][(k >> shift) & dm], 1u);
      if (!same && (k & m1) == p1) atomicAdd(&sm.hist[1][(k >> shift) & dm], 1u);
    }
    os_scan(sm, shift, w, tid);
    left = shift;
  }
  if (left == 0) return;
  const unsigned p0 = sm.pfx[0], m0 = sm.mask[0], p1 = sm.pfx[1], m1 = sm.mask[1];
  int n = 0;
  for (int q = tid; q < T; q += kOsThreads) {
    const unsigned k = os_key<kDev>(__ldg(xr + q), m);
    if ((k & m0) == p0 || (k & m1) == p1) seg[n++] = k;
  }
  os_tail(seg, n, sm, left, tid);
}

// Row u of x (T values): the ka-th and kb-th largest, their keys to
// out[4 u] and out[4 (rows + u)]; with kMad also those of |x - m|, m the
// mean of the first two, to out[4 (2 rows + u)] and out[4 (3 rows + u)].
template <bool kMad>
__global__ void __launch_bounds__(kOsThreads, 1) order_stats_kernel(const float* x, int rows, int T, int ka, int kb,
                                                                   unsigned* out) {
  extern __shared__ __align__(16) unsigned char os_smem_raw[];
  OsSmem& sm = *reinterpret_cast<OsSmem*>(os_smem_raw);
  const int u = blockIdx.x, tid = threadIdx.x;
  for (int i = tid; i < 2 * kOsBins; i += kOsThreads) (&sm.hist[0][0])[i] = 0u;
  asm volatile("griddepcontrol.wait;" ::: "memory");  // x comes from the launch before
  // the finalize after this launch may be scheduled now (it waits for this
  // grid's completion before reading)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const float* xr = x + (size_t)u * T;
  const int nv = max(0, min(kOsPer, T - tid * kOsPer));
  unsigned* seg = &sm.stage[tid * kOsSeg];
  const bool long_row = T > kOsThreads * kOsPer;
  if (long_row) {
    os_select2_long<false>(xr, T, 0.f, seg, sm, ka, kb, tid);
  } else {
    os_stage<false>(xr, T, 0.f, sm, tid);
    __syncthreads();
    os_select2(seg, nv, sm, ka, kb, tid);
  }
  const unsigned a = sm.pfx[0], b = sm.pfx[1];
  if (tid == 0) {
    out[4 * u] = a;
    out[4 * (rows + u)] = b;
  }
  if (!kMad) return;
  // the second pair over |d_E - median|, the row read again (the first
  // select reordered the stage)
  const float m = __fmul_rn(0.5f, __fadd_rn(key_float(a), key_float(b)));
  __syncthreads();  // every thread has read the first pair and its last list
  if (long_row) {
    os_select2_long<true>(xr, T, m, seg, sm, ka, kb, tid);
  } else {
    os_stage<true>(xr, T, m, sm, tid);
    __syncthreads();
    os_select2(seg, nv, sm, ka, kb, tid);
  }
  if (tid == 0) {
    out[4 * (2 * rows + u)] = sm.pfx[0];
    out[4 * (3 * rows + u)] = sm.pfx[1];
  }
}

}  // namespace

cudaError_t launch_order_stats(const float* x, int rows, int T, int ka, int kb, bool mad, unsigned* out,
                               cudaStream_t s) {
  if (rows <= 0 || T <= 0 || T > kMaxN || ka < 1 || ka > T || kb < 1 || kb > T)
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)rows);
  cfg.blockDim = dim3(kOsThreads);
  cfg.dynamicSmemBytes = sizeof(OsSmem);
  cfg.stream = s;
  static std::atomic<bool> attr_set[64];  // a racing thread repeats the idempotent setup
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!attr_set[dev].load()) {
    if ((e = cudaFuncSetAttribute(order_stats_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)sizeof(OsSmem))) != cudaSuccess ||
        (e = cudaFuncSetAttribute(order_stats_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)sizeof(OsSmem))) != cudaSuccess)
      return e;
    attr_set[dev].store(true);
  }
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return mad ? cudaLaunchKernelEx(&cfg, order_stats_kernel<true>, x, rows, T, ka, kb, out)
             : cudaLaunchKernelEx(&cfg, order_stats_kernel<false>, x, rows, T, ka, kb, out);
}

}  // namespace ecokv
