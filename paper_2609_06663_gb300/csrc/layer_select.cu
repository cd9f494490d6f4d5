// Top-k of a layer's concatenated scores for the layer-wide budget (AdaKV,
// Appendix A): the k largest of T = h_kv * T_v scores per layer, ties to the
// lower concatenated position, emitted in ascending position.
//
// An MSB-first radix select on the order-preserving integer image of S, as in
// the per-head select, spread over many CTAs per layer without any CTA waiting
// on another: three digits of 11, 11 and 10 bits, each one launch that
// histograms blocks of 4096 scores into a per-layer global histogram (a
// shared-memory histogram per block, one atomic add per non-empty bin) and one
// launch in which a CTA per layer finds the digit by a suffix scan and clears
// the histogram for the next digit.  Then one launch counts each block's
// scores above / equal to the threshold, and one emits: each block adds up the
// counts of the blocks before it (ties taken in position order) and writes its
// kept positions in order.  Each launch is a programmatic dependent of the one
// before it (prepared while that one runs; it waits for its results first).

#include "ecokv_internal.cuh"
#include "finalize_select.cuh"

namespace ecokv {
namespace {

constexpr int kLsThreads = 256;
constexpr int kLsWarps = kLsThreads / 32;
constexpr int kLsPer = 16;                       // scores a thread handles
constexpr int kLsSpan = kLsThreads * kLsPer;     // scores a block handles
constexpr int kLsWarpSpan = kLsSpan / kLsWarps;  // contiguous scores a warp emits

struct LsArgs {
  const float* S;     // [L][T]
  int T, k, nblk;
  unsigned* ghist;    // [L][kLsMaxBins], zero before the first digit
  unsigned* state;    // [L][4]: prefix, mask, remaining count at the threshold (zero before the first digit)
  int* cnt;           // [L][nblk][2]: a block's scores above / equal to the threshold
  int32_t* chosen;    // [L][k]
};

constexpr int kLsMaxBins = 2048;

__device__ __forceinline__ void ls_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Digit of `bits` bits at `shift` of the scores under the layer's prefix.
template <int kBits>
__global__ void __launch_bounds__(kLsThreads) ls_hist(LsArgs a, int shift) {
  constexpr int kBins = 1 << kBits;
  const int l = blockIdx.y, lo = blockIdx.x * kLsSpan;
  const int tid = threadIdx.x, lane = tid & 31;
  __shared__ unsigned hist[kBins];
  for (int b = tid; b < kBins; b += kLsThreads) hist[b] = 0u;
  ls_wait();
  __syncthreads();
  const float* S = a.S + (size_t)l * a.T;
  const unsigned* st = a.state + 4 * l;
  const unsigned prefix = st[0], mask = st[1];
#pragma unroll 4
  for (int j = 0; j < kLsPer; ++j) {
    const int i = lo + j * kLsThreads + tid;
    unsigned bin = 0xffffffffu;
    if (i < a.T) {
      const unsigned key = ordered_key(__ldg(S + i));
      if ((key & mask) == prefix) bin = (key >> shift) & (kBins - 1);
    }
    // lanes with equal bins counted once (the scores of a layer crowd into
    // few bins of the first digit)
    const unsigned peers = __match_any_sync(0xffffffffu, bin);
    if (bin != 0xffffffffu && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], (unsigned)__popc(peers));
  }
  __syncthreads();
  for (int b = tid; b < kBins; b += kLsThreads)
    if (hist[b]) atomicAdd(a.ghist + (size_t)l * kLsMaxBins + b, hist[b]);
}

template <int kBits>
__global__ void __launch_bounds__(256) ls_digit(LsArgs a, int shift, int first) {
  constexpr int kBins = 1 << kBits, kPer = kBins / 256;  // bins a thread owns, highest last
  const int l = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ unsigned wsum[8];
  ls_wait();
  unsigned* st = a.state + 4 * l;
  unsigned* gh = a.ghist + (size_t)l * kLsMaxBins + tid * kPer;
  const unsigned rem = first ? (unsigned)a.k : st[2];
  unsigned h[kPer], tot = 0u;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    h[q] = gh[q];
    tot += h[q];
  }
  unsigned suf = tot;  // scores in the bins of threads tid .. 32 warp + 31
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned y = __shfl_down_sync(0xffffffffu, suf, o);
    if (lane + o < 32) suf += y;
  }
  if (lane == 0) wsum[warp] = suf;
  __syncthreads();
  for (int w = warp + 1; w < 8; ++w) suf += wsum[w];
#pragma unroll
  for (int q = 0; q < kPer; ++q) gh[q] = 0u;  // ready for the next digit
  // suf = scores in bins >= tid kPer; the wanted bin is this thread's when
  // suf >= rem > suf - tot; then the highest of its bins that reaches rem
  if (suf >= rem && suf - tot < rem) {
    unsigned above = suf - tot;
#pragma unroll
    for (int q = kPer - 1; q >= 0; --q) {
      if (above + h[q] >= rem) {
        st[0] |= (unsigned)(tid * kPer + q) << shift;
        st[1] |= (unsigned)(kBins - 1) << shift;
        st[2] = rem - above;
        break;
      }
      above += h[q];
    }
  }
}

__global__ void __launch_bounds__(kLsThreads) ls_count(LsArgs a) {
  const int l = blockIdx.y, lo = blockIdx.x * kLsSpan, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ int red[kLsWarps][2];
  ls_wait();
  const float* S = a.S + (size_t)l * a.T;
  const unsigned thr = a.state[4 * l];
  int gt = 0, eq = 0;
#pragma unroll 4
  for (int j = 0; j < kLsPer; ++j) {
    const int i = lo + j * kLsThreads + tid;
    if (i < a.T) {
      const unsigned key = ordered_key(__ldg(S + i));
      gt += key > thr;
      eq += key == thr;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    gt += __shfl_xor_sync(0xffffffffu, gt, o);
    eq += __shfl_xor_sync(0xffffffffu, eq, o);
  }
  if (lane == 0) {
    red[warp][0] = gt;
    red[warp][1] = eq;
  }
  __syncthreads();
  if (tid == 0) {
    int g = 0, q = 0;
    for (int w = 0; w < kLsWarps; ++w) {
      g += red[w][0];
      q += red[w][1];
    }
    int* c = a.cnt + ((size_t)l * a.nblk + blockIdx.x) * 2;
    c[0] = g;
    c[1] = q;
  }
}

__global__ void __launch_bounds__(kLsThreads) ls_emit(LsArgs a) {
  const int l = blockIdx.y, b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ int wcnt[kLsWarps][2];
  __shared__ int base[2];
  ls_wait();
  const float* S = a.S + (size_t)l * a.T;
  const unsigned thr = a.state[4 * l];
  const int rem = (int)a.state[4 * l + 2];
  if (tid == 0) {
    // kept scores before this block, and the ties they took
    int pos = 0, eq_before = 0;
    const int* c = a.cnt + (size_t)l * a.nblk * 2;
    for (int j = 0; j < b; ++j) {
      pos += c[2 * j] + max(0, min(c[2 * j + 1], rem - eq_before));
      eq_before += c[2 * j + 1];
    }
    base[0] = pos;
    base[1] = eq_before;
  }
  // each warp's contiguous span, in 32-score steps
  const int w0 = b * kLsSpan + warp * kLsWarpSpan;
  int gt = 0, eq = 0;
  for (int s = 0; s < kLsWarpSpan; s += 32) {
    const int i = w0 + s + lane;
    const unsigned key = i < a.T ? ordered_key(__ldg(S + i)) : 0u;
    gt += __popc(__ballot_sync(0xffffffffu, i < a.T && key > thr));
    eq += __popc(__ballot_sync(0xffffffffu, i < a.T && key == thr));
  }
  if (lane == 0) {
    wcnt[warp][0] = gt;
    wcnt[warp][1] = eq;
  }
  __syncthreads();
  int pos = base[0], eq_before = base[1];
  for (int w = 0; w < warp; ++w) {
    pos += wcnt[w][0] + max(0, min(wcnt[w][1], rem - eq_before));
    eq_before += wcnt[w][1];
  }
  const int take_eq = max(0, min(eq, rem - eq_before));
  const unsigned lt = (1u << lane) - 1u;
  int32_t* out = a.chosen + (size_t)l * a.k;
  int eq_seen = 0;
  for (int s = 0; s < kLsWarpSpan; s += 32) {
    const int i = w0 + s + lane;
    const unsigned key = i < a.T ? ordered_key(__ldg(S + i)) : 0u;
    const bool g = i < a.T && key > thr;
    const bool e = i < a.T && key == thr;
    const unsigned em = __ballot_sync(0xffffffffu, e);
    const bool take = g || (e && eq_seen + __popc(em & lt) < take_eq);
    const unsigned sel = __ballot_sync(0xffffffffu, take);
    if (take) {
      const int p = pos + __popc(sel & lt);
      if (p < a.k) out[p] = i;
    }
    pos += __popc(sel);
    eq_seen += __popc(em);
  }
}

}  // namespace

template <typename... P, typename... A>
cudaError_t launch_dependent(void (*kernel)(P...), dim3 grid, dim3 block, cudaStream_t s, A... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

size_t layer_select_scratch_bytes(int n_layers, int T) {
  const int nblk = (T + kLsSpan - 1) / kLsSpan;
  return (size_t)n_layers * (kLsMaxBins + 4 + 2 * (size_t)nblk) * 4;
}

// k largest of each layer's T scores S[l][0..T), positions ascending, into
// chosen[l][0..k); scratch: layer_select_scratch_bytes, any contents.
cudaError_t launch_layer_select(const float* S, int n_layers, int T, int k, int32_t* chosen, void* scratch,
                                cudaStream_t s) {
  if (k <= 0 || n_layers <= 0) return cudaSuccess;
  LsArgs a{};
  a.S = S;
  a.T = T;
  a.k = k;
  a.nblk = (T + kLsSpan - 1) / kLsSpan;
  a.ghist = static_cast<unsigned*>(scratch);
  a.state = a.ghist + (size_t)n_layers * kLsMaxBins;
  a.cnt = reinterpret_cast<int*>(a.state + (size_t)n_layers * 4);
  a.chosen = chosen;
  cudaError_t e = cudaMemsetAsync(scratch, 0, (size_t)n_layers * (kLsMaxBins + 4) * 4, s);
  if (e != cudaSuccess) return e;
  const dim3 grid(a.nblk, n_layers), blk(kLsThreads);
  if ((e = launch_dependent(ls_hist<11>, grid, blk, s, a, 21)) != cudaSuccess ||
      (e = launch_dependent(ls_digit<11>, dim3(n_layers), dim3(256), s, a, 21, 1)) != cudaSuccess ||
      (e = launch_dependent(ls_hist<11>, grid, blk, s, a, 10)) != cudaSuccess ||
      (e = launch_dependent(ls_digit<11>, dim3(n_layers), dim3(256), s, a, 10, 0)) != cudaSuccess ||
      (e = launch_dependent(ls_hist<10>, grid, blk, s, a, 0)) != cudaSuccess ||
      (e = launch_dependent(ls_digit<10>, dim3(n_layers), dim3(256), s, a, 0, 0)) != cudaSuccess ||
      (e = launch_dependent(ls_count, grid, blk, s, a)) != cudaSuccess ||
      (e = launch_dependent(ls_emit, grid, blk, s, a)) != cudaSuccess)
    return e;
  return cudaSuccess;
}

}  // namespace ecokv
