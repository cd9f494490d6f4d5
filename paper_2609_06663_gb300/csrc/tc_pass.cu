// Persistent tensor-core kernel for bf16 inputs: both streaming passes of the
// eviction pass in one launch on sm_103a.
//
// Work items (u = unit = (layer, KV head); a chunk is a run of consecutive
// tiles of 128 keys of one unit, the part of a CTA's slice inside the unit):
//   P1(u, c)  pass 1 over chunk c: window logits (tcgen05 MMA, keys as M,
//             window rows as N), per-row online-softmax partials, key norms,
//             and the chunk sums of k and k/||k|| (a second tcgen05 MMA with the
//             key tile as an MN-major operand against [1, w_hi, w_mid, w_lo]
//             weight rows, w = 1/||k|| split into three bf16 terms).
//   P2(u, c)  pass 2: logits again plus five extra MMA columns holding k . kbar
//             (kbar split into three bf16 terms) and k . mu (two terms), giving
//             the importance vote, the cosine khat . mu, and d_E (Eq. 1) by the
//             expansion of Sec. 4 from ||k||^2 (recomputed from the tile in
//             shared memory).  Where that expansion cancels (d_E^2 below 2^-6
//             of ||k||^2 + ||kbar||^2, keys close to their centroid) the key is
//             recomputed directly from its row in global memory.
//
// Schedule (static, one CTA per SM, cooperative launch).  The units form
// waves of `uw` units in unit order; the tiles of a wave are cut into
// n = min(P, L) contiguous slices of near-equal length (L = the wave's
// tiles), and CTA c takes slice c of every wave, one item per unit the slice
// touches (pass 2 walks a slice backwards, units and tiles, so that it starts
// with the keys pass 1 read last, the likeliest still to be in L2).  Step s of CTA c holds: the P1 items of its slice of wave s; the
// fold items of the units of wave s - 1 it owns (unit u belongs to CTA
// u mod P); the P2 items of its slice of wave s - lag.  With one wave (the
// default) all of pass 1 precedes pass 2 and K is read twice; with small
// waves and lag 1..2 a unit's keys are still in L2 at its pass 2 (pass-1
// reads carry an evict-last policy then), at the cost of more items.  Every
// CTA is resident, so waits on other CTAs' items end.
//
// Unit statistics (kbar, mu, ||kbar||^2, ||mu||^2, per-row log2-sum-exp):
// every P1 item writes a record to its slot (its slice's index among the
// slices the unit meets) and then adds one to the unit's arrival counter with
// release semantics.  The fold item of unit u waits until all of the unit's
// slices have arrived, folds the records in a fixed order with the 256
// epilogue threads, publishes the statistics record and raises the unit's
// ready flag (release).  The stats warp readies each P2 item about one item
// ahead of the epilogue: it waits for the flag, copies the record and writes
// the statistics rows of the MMA operand.  Nothing but the MMA and the
// epilogue of a P2 item waits for it: the producer keeps loading key tiles
// meanwhile.  The fold order and every partial's arithmetic depend only on
// the schedule's parameters, so results are reproducible for a given
// (uw, lag, P).
//
// Warp roles (512 threads, one CTA per SM): warp 0 walks the CTA's schedule
// and issues TMA loads of the window queries and of 32 KB key tiles into a
// 4- or 5-stage ring; warp 1 issues the logits MMAs into up to four TMEM
// accumulators; warp 3 issues the sum MMAs of pass-1 tiles (two more
// accumulators) as soon as a tile's logits are done and its weights written,
// and frees the stage; warp 2 (stats warp) readies the unit statistics of P2
// items; warps 12-15 (key warps, one key per thread) compute the key norms of
// every tile as it lands (the sum weights in pass 1, a hand-off to the
// epilogue in pass 2) and read the chunk sums; warps 4-11 are the epilogue
// (one key per TMEM lane; in pass 1 the window rows split in two halves, in
// pass 2 the tiles: half h takes every row of the item's tiles t with
// t % 2 == h), which also runs the fold items.  setmaxnreg gives the two epilogue warpgroups 176
// registers a thread and the others 80.
// Every mbarrier wait and spin is bounded (a limit in nanoseconds of the
// global timer): on timeout the kernel records ECOKV_ERR_TIMEOUT, raises a
// gpu-wide abort flag, drains its own copies (key tiles and window queries)
// and MMAs, frees TMEM and exits.

#include <cuda.h>

#include <atomic>
#include <stddef.h>

#include "finalize_select.cuh"
#include "ptx.cuh"
#include "tc_pass.cuh"

namespace ecokv {
namespace {

using namespace ptx;

constexpr int kIQ = 2;
constexpr int kPrefetchTiles = 8;  // pass-1 tiles of an item prefetched into L2 when the item starts
constexpr int kTile = 128;
constexpr int kThreads = 512;
constexpr int kEpi = 256;
constexpr int kEpiWarp0 = 4;          // first epilogue warp (warps 4..11)
constexpr int kKeyWarp0 = 12;         // first key warp (warps 12..15, one key per thread)
constexpr int kKeyWarps = 4;
constexpr uint32_t kRegsEpi = 176;    // registers a thread after the split: epilogue warpgroups
constexpr uint32_t kRegsOther = 80;   // producer / MMA / key warpgroups
static_assert(2 * 128 * kRegsEpi + 2 * 128 * kRegsOther == 65536, "register split must fit the launch's 512 x 128");
static_assert(kRegsEpi % 8 == 0 && kRegsOther % 8 == 0 && kRegsOther >= 24 && kRegsEpi <= 256, "setmaxnreg range");
constexpr int kNPMax = 128;
constexpr uint32_t kTileBytes = kTile * kD * 2;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSigmaCol = 256;
constexpr uint32_t kEpiBar = 1;

enum : int { kP1 = 0, kP2 = 1, kFold = 2, kExit = 3 };

constexpr int kNB = 4;                // pass-2 norm hand-off slots
constexpr int kUstatMax = 2 * kD + 4 + kNPMax;  // floats of a unit statistics record (lse padded to NP rows)

struct __align__(16) ItemDesc {
  int type, u, rec, i0, ntiles;  // rec: the item's record slot (its slice's index among the unit's slices)
  int pad[3];
  float ust[kUstatMax];  // pass 2: copy of the unit statistics record (kbar, mu, norms, log2-LSE)
};

// Shared memory of the kernel instance with RH window rows per half: the
// query buffers take just 2 * RH rows, which leaves room for a fifth key-tile
// stage unless RH = 64.
template <int RH>
struct __align__(1024) Smem {
  static constexpr int kS = RH >= 64 ? 4 : 5;  // key-tile stages
  static constexpr int kQB = 2 * RH * 256;      // bytes of one query buffer (2 boxes of 2*RH rows)
  uint8_t ktile[kS][kTileBytes];                // 2 boxes [128 keys x 64 d], 128-byte swizzle
  uint8_t qbuf[kIQ][kQB < 1024 ? 1024 : kQB];   // B operand, 2 boxes [NP rows x 64 d]
  uint8_t wbuf[kS][4096];                       // sum weights: 2 boxes [16 rows x 64 keys]; rows 1, w_hi, w_mid, w_lo
  ItemDesc desc[kIQ];
  float red[8][RH][2];                          // [epilogue warp][row][max, sum]
  float red6[8][8];                             // [epilogue warp][pass-2 partial]
  uint64_t full[kS], empty[kS], wready[kS];
  uint64_t item_full[kIQ], item_empty[kIQ], qfull[kIQ];
  uint64_t tmem_full[4], tmem_empty[4];
  uint64_t sigma_full[2], sigma_empty[2], drain, drain2;
  uint64_t lgdone[kS];  // pass-1 tile: its logits MMA is complete (for the sum-MMA issuer)
  float nbuf[kNB][kTile];                        // pass-2 squared key norms, key warps -> epilogue
  uint64_t nfull[kNB], nempty[kNB];
  uint64_t kpub[kIQ];    // key warps have written this pass-1 item's chunk sums
  uint64_t sready[kIQ];  // pass 2: unit statistics in desc.ust and statistics rows in qbuf (stats warp ->
                         // MMA and epilogue)
  float fold[512];       // epilogue scratch: combining the fold's thread groups
  uint32_t tmem_base;
  int epi_abort;         // an epilogue warp gave up a wait (read after a named barrier)
};

static_assert(sizeof(Smem<8>) + 1024 <= 232448 && sizeof(Smem<16>) + 1024 <= 232448 &&
                  sizeof(Smem<32>) + 1024 <= 232448 && sizeof(Smem<64>) + 1024 <= 232448,
              "shared-memory plan exceeds the 227 KB per-CTA limit");
static_assert(sizeof(ItemDesc) % 16 == 0 && offsetof(ItemDesc, ust) % 16 == 0, "bulk-copy target alignment");

__device__ __forceinline__ unsigned* abort_flag(const TcArgs& a) { return a.sync + 1; }
__device__ __forceinline__ unsigned* arrivals(const TcArgs& a, int u) { return a.sync + 4 + u; }
__device__ __forceinline__ unsigned* stats_ready(const TcArgs& a, int u) { return a.sync + 4 + a.U + u; }

__device__ __forceinline__ unsigned long long now_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

__device__ void raise_abort(const TcArgs& a, unsigned code, unsigned detail) {
  if (atomicCAS(a.status, 0u, code) == 0u) a.status[1] = detail;
  atomicExch(abort_flag(a), 1u);
}

__device__ __forceinline__ bool aborted(const TcArgs& a) {
  return *reinterpret_cast<volatile unsigned*>(abort_flag(a)) != 0u;
}

// Bounded wait on an mbarrier phase; false on timeout or abort.
__device__ bool wait_bar(uint64_t* bar, uint32_t parity, const TcArgs& a, unsigned where) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = now_ns();
  for (unsigned spins = 1;; ++spins) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((spins & 63u) == 0u) {
      if (aborted(a)) return false;
      if (now_ns() - t0 > a.timeout_ns) {
        raise_abort(a, ECOKV_ERR_TIMEOUT, where);
        return false;
      }
    }
  }
}

// Wait for an mbarrier phase without regard to the abort flag, bounded: the
// drain of copies in flight before a CTA leaves.
__device__ void drain_bar(uint64_t* bar, uint32_t parity, const TcArgs& a) {
  const unsigned long long t0 = now_ns();
  while (!mbar_try_wait(bar, parity) && now_ns() - t0 < a.timeout_ns) {
  }
}

// Static schedule.  Wave w holds units [w uw, (w + 1) uw) (fewer in the last
// wave), L = their tiles in unit order; it is cut into n = min(P, L)
// contiguous slices, slice c covering wave tiles [floor(c L / n),
// floor((c + 1) L / n)).  CTA c takes slice c of every wave.
__device__ __forceinline__ int wave_tiles(const TcArgs& a, int w) { return min(a.uw, a.U - w * a.uw) * a.T; }
__device__ __forceinline__ int slice_start(int c, int L, int n) { return (int)((long long)c * L / n); }
// The slice holding wave tile o: the largest c with slice_start(c) <= o.
__device__ __forceinline__ int slice_at(int o, int L, int n) {
  return (int)(((long long)(o + 1) * n + L - 1) / L) - 1;
}
// The slices unit u meets: the first one, and how many (= its pass-1 records).
__device__ __forceinline__ void unit_slices(const TcArgs& a, int u, int& c0, int& nrec) {
  const int w = u / a.uw, L = wave_tiles(a, w), n = min(a.P, L);
  const int o = (u - w * a.uw) * a.T;
  c0 = slice_at(o, L, n);
  nrec = slice_at(o + a.T - 1, L, n) - c0 + 1;
}

// Bounded spin until a gpu-scope counter written by other CTAs reaches
// `target` (acquire); false on timeout or abort.
__device__ bool wait_count(const unsigned* f, unsigned target, const TcArgs& a, unsigned where) {
  const unsigned long long t0 = now_ns();
  while (ld_acquire(f) < target) {
    if (aborted(a)) return false;
    if (now_ns() - t0 > a.timeout_ns) {
      raise_abort(a, ECOKV_ERR_TIMEOUT, where);
      return false;
    }
    __nanosleep(64);
  }
  return true;
}

__device__ __forceinline__ uint32_t sw128(int row, int chunk16) {
  return (uint32_t)(row * 128 + ((chunk16 ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Pass-2 rows of the B operand (128-byte-swizzled, K-major): rows NP-8..NP-6
// hold kbar split into three bf16 terms (hi, mid, lo), rows NP-5, NP-4 hold
// mu_hi and mu_lo, all from the unit statistics copy (the last eight columns
// of the accumulator belong to the second row half); the window queries in
// rows 0..R-1 arrive by TMA.  Task e (0 <= e < 80) writes one 16-byte
// vector: term row e / 16, dimensions 8 (e % 16) .. 8 (e % 16) + 7.
__device__ void build_stat_rows(uint8_t* qb, const TcArgs& a, const float* ust, int e) {
  const int which = e >> 4, j = e & 15;
  const float* src = ust + (which < 3 ? ustat_kbar() : ustat_mu()) + j * 8;
  const int term = which < 3 ? which : which - 3;  // 0 = hi, 1 = mid / lo, 2 = lo
  float o[8];
#pragma unroll
  for (int t = 0; t < 8; ++t) {
    const float x = src[t];
    const float hi = __bfloat162float(__float2bfloat16_rn(x));
    const float r1 = x - hi;
    const float mid = __bfloat162float(__float2bfloat16_rn(r1));
    o[t] = term == 0 ? hi : (which < 3 ? (term == 1 ? mid : r1 - mid) : r1);
  }
  const uint4 val = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]), pack_bf16x2(o[4], o[5]),
                               pack_bf16x2(o[6], o[7]));
  *reinterpret_cast<uint4*>(qb + (j >> 3) * (a.NP * 128) + sw128(a.NP - 8 + which, j & 7)) = val;
}

// Joint (max, sum) of partial softmax sums: (m1, z1) + (m2, z2) with z
// relative to 2^m; an empty pair has m = -inf, z = 0.
__device__ __forceinline__ void combine_maxsum(float& m, float& z, float m2, float z2) {
  const float M = fmaxf(m, m2);
  const float Ms = M == -INFINITY ? 0.f : M;
  z = z * ex2(m - Ms) + z2 * ex2(m2 - Ms);
  m = M;
}

// Fold the nch pass-1 records of unit u into its statistics record, by the
// 256 epilogue threads (tid), with all loads of a thread issued together
// (one round trip for up to 48 records).  Record: [sum k (d)] [sum k/||k||
// (d)] [row max (R4)] [row sum (R4)].  Sums: thread (q, c) = (tid >> 7, tid &
// 127) adds floats 2c, 2c + 1 of the records q, q + 2, ... in order; the two
// groups are added in order.  Rows: thread (g, r) = (tid / R, tid % R), g <
// G = min(8, 256 / R), combines the (max, sum) pairs of row r in the records
// g, g + G, ... in order, then the G groups in order.  The record goes to the
// unit's place in global memory.  Uses s_fold (512 floats) and named barrier
// kEpiBar among the 256 threads.
__device__ void fold_unit_stats(const TcArgs& a, int u, int nch, int tid, float* s_fold) {
  const float* base = a.p1part + (size_t)u * a.rmax * a.p1_stride;
  float* gus = a.ustat + (size_t)u * a.ustat_stride;
  const int q = tid >> 7, c = tid & 127;
  const int R = a.R, G = min(8, kEpi / R);
  const bool lrow = tid < G * R;
  const int g = lrow ? tid / R : 0, r = lrow ? tid - g * R : 0;
  float sx = 0.f, sy = 0.f, M = -INFINITY, Z = 0.f;
  constexpr int kS = 24, kL = 12;
  for (int b = 0;; ++b) {
    const int r0 = q + 2 * kS * b, l0 = g + G * kL * b;
    if (r0 >= nch && (!lrow || l0 >= nch)) break;
    float2 v[kS];
    float mv[kL], zv[kL];
#pragma unroll
    for (int j = 0; j < kS; ++j)
      v[j] = __ldcg(reinterpret_cast<const float2*>(base + (size_t)min(r0 + 2 * j, nch - 1) * a.p1_stride) + c);
#pragma unroll
    for (int j = 0; j < kL; ++j) {
      const float* p = base + (size_t)min(l0 + G * j, nch - 1) * a.p1_stride + 2 * kD;
      mv[j] = __ldcg(p + r);
      zv[j] = __ldcg(p + a.R4 + r);
    }
#pragma unroll
    for (int j = 0; j < kS; ++j)
      if (r0 + 2 * j < nch) {
        sx += v[j].x;
        sy += v[j].y;
      }
#pragma unroll
    for (int j = 0; j < kL; ++j)
      if (lrow && l0 + G * j < nch && zv[j] > 0.f) combine_maxsum(M, Z, mv[j], zv[j]);
  }
  if (q == 1) {
    s_fold[2 * c] = sx;
    s_fold[2 * c + 1] = sy;
  }
  named_bar_sync(kEpiBar, kEpi);
  if (q == 0) {
    sx += s_fold[2 * c];
    sy += s_fold[2 * c + 1];
    // columns 2c, 2c + 1: sum of k for c < 64, sum of k/||k|| for c >= 64
    const float sc = c < 64 ? 1.f / (float)a.kbar_n : 1.f / (float)a.N;
    const float x = sx * sc, y = sy * sc;
    __stcg(reinterpret_cast<float2*>(gus) + c, make_float2(x, y));
    // ||kbar||^2 (warps 0, 1 of the group) and ||mu||^2 (warps 2, 3)
    float sq = fmaf(x, x, y * y);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if ((c & 31) == 0) s_fold[256 + (c >> 5)] = sq;
  }
  named_bar_sync(kEpiBar, kEpi);
  if (tid == 0) {
    gus[ustat_ksq()] = s_fold[256] + s_fold[257];
    gus[ustat_musq()] = s_fold[258] + s_fold[259];
  }
  named_bar_sync(kEpiBar, kEpi);
  if (lrow) {
    s_fold[2 * tid] = M;
    s_fold[2 * tid + 1] = Z;
  }
  named_bar_sync(kEpiBar, kEpi);
  if (tid < R) {
    float Mx = -INFINITY, Zx = 0.f;
    for (int gg = 0; gg < G; ++gg) {
      const float m2 = s_fold[2 * (gg * R + tid)], z2 = s_fold[2 * (gg * R + tid) + 1];
      if (z2 > 0.f) combine_maxsum(Mx, Zx, m2, z2);
    }
    gus[ustat_lse() + a.row0 + tid] = Mx + log2f(Zx);
  }
}

template <int RH>
__device__ __forceinline__ void warp_reduce_scatter_maxsum(float (&m)[RH], float (&z)[RH], int lane) {
  int n = RH;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    if (n > 1 && (RH > 32 || n > 1)) {
      const bool up = (lane & o) != 0;
      const int hf = n / 2;
#pragma unroll
      for (int j = 0; j < RH / 2; ++j) {
        if (j < hf) {
          const float km = up ? m[j + hf] : m[j], kz = up ? z[j + hf] : z[j];
          const float sm = up ? m[j] : m[j + hf], sz = up ? z[j] : z[j + hf];
          const float rm = __shfl_xor_sync(0xffffffffu, sm, o), rz = __shfl_xor_sync(0xffffffffu, sz, o);
          m[j] = km;
          z[j] = kz;
          combine_maxsum(m[j], z[j], rm, rz);
        }
      }
      n = hf;
    } else {
      const float rm = __shfl_xor_sync(0xffffffffu, m[0], o), rz = __shfl_xor_sync(0xffffffffu, z[0], o);
      combine_maxsum(m[0], z[0], rm, rz);
    }
  }
}

template <int RH>
__global__ void __launch_bounds__(kThreads, 1)
    tc_evict_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  using SM = Smem<RH>;
  constexpr int kStages = SM::kS;
  SM& s = *reinterpret_cast<SM*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nbuf_log = a.NP <= 64 ? 2 : 1;  // 4 or 2 TMEM accumulators of NP columns (<= 256 columns)

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], kKeyWarps + 1);  // key warps + MMA commit
      mbar_init(&s.wready[i], kKeyWarps);
    }
    for (int i = 0; i < kIQ; ++i) {
      mbar_init(&s.item_full[i], 1);
      mbar_init(&s.item_empty[i], 1 + 8 + kKeyWarps + 2);  // MMA commit + epilogue + key warps + stats + sum warps
      mbar_init(&s.qfull[i], 1);
      mbar_init(&s.sready[i], 1);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(&s.tmem_full[i], 1);
      mbar_init(&s.tmem_empty[i], 8);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.sigma_full[i], 1);
      mbar_init(&s.sigma_empty[i], 4);
    }
    for (int i = 0; i < kIQ; ++i) mbar_init(&s.kpub[i], kKeyWarps);
    for (int i = 0; i < kNB; ++i) {
      mbar_init(&s.nfull[i], kKeyWarps);
      mbar_init(&s.nempty[i], 4);  // the 4 epilogue warps of the half that takes the tile
    }
    s.epi_abort = 0;
    mbar_init(&s.drain, 1);
    mbar_init(&s.drain2, 1);
    for (int i = 0; i < kStages; ++i) mbar_init(&s.lgdone[i], 1);
    fence_mbar_init();
  }
  // constant rows of the sum-weight operand: row 0 = 1, rows 4..15 = 0
  for (int e = threadIdx.x; e < kStages * 2 * 16 * 8; e += blockDim.x) {
    const int st = e / 256, rem = e % 256, box = rem / 128, r = (rem % 128) / 8, j = rem % 8;
    const uint32_t one2 = 0x3F803F80u;  // bf16 1.0 pair
    const uint4 v = r == 0 ? make_uint4(one2, one2, one2, one2) : make_uint4(0u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(s.wbuf[st] + box * 2048 + sw128(r, j)) = v;
  }
  if (warp == 1) {
    tmem_alloc(&s.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmQ);
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  bool ok = true;

  if (warp >= kEpiWarp0 && warp < kKeyWarp0) {
    // register split: the two epilogue warpgroups take the registers the
    // other two give back
    reg_alloc<kRegsEpi>();
    // ------------------------------------------------ epilogue (warps 4..11)
    // Named barriers among the eight warps sit only at item boundaries and are
    // reached by every warp; a warp that gives up a wait marks epi_abort and
    // all of them leave together after the next barrier.
    const int e = warp - kEpiWarp0, q = warp & 3, h = e >> 2;
    const int kk = 32 * q + lane;  // key row within a tile = TMEM lane
    const int tid = threadIdx.x - 32 * kEpiWarp0;
    const uint32_t tl = tmem + ((uint32_t)(32 * q) << 16);
    const uint32_t bmask = (1u << nbuf_log) - 1u;
    uint32_t tcount = 0, pcount = 0;
    uint32_t spar = 0u;  // per slot: parity of the next sready phase (completed by P2 items only)
    auto epi_sync = [&]() -> bool {
      if (!ok) s.epi_abort = 1;
      named_bar_sync(kEpiBar, kEpi);
      return s.epi_abort == 0;
    };
    for (int seq = 0;; ++seq) {
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      ok = __all_sync(0xffffffffu, wait_bar(&s.item_full[slot], qphase, a, 10u));
      if (!epi_sync()) {
        ok = false;
        break;
      }
      const ItemDesc& d = s.desc[slot];
      const int type = d.type;
      if (type == kExit) break;
      const int u = d.u, rec = d.rec, i0 = d.i0, ntiles = d.ntiles;

      if (type == kFold) {
        // unit statistics: once every P1 item of unit u has arrived, fold
        // their partials with all 256 threads and publish the record
        int c0, nrec;
        unit_slices(a, u, c0, nrec);
        const unsigned need = (unsigned)nrec + (u == a.stall_unit ? 1u : 0u);
        if (tid == 0) ok = wait_count(arrivals(a, u), need, a, 30u);
        if (!epi_sync()) {
          ok = false;
          break;
        }
        fold_unit_stats(a, u, nrec, tid, s.fold);
        named_bar_sync(kEpiBar, kEpi);
        if (tid == 0) {
          __threadfence();
          st_release(stats_ready(a, u), 1u);
        }
      } else if (type == kP1) {
        float m[RH], z[RH];
#pragma unroll
        for (int c = 0; c < RH; ++c) {
          m[c] = 0.f;
          z[c] = 0.f;
        }
        for (int t = 0; t < ntiles && ok; ++t) {
          const int it0 = i0 + t * kTile;
          const int i = it0 + kk;
          const bool valid = i < a.N;
          const uint32_t b = tcount & bmask, tph = (tcount >> nbuf_log) & 1u;
          if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.tmem_full[b], tph, a, 12u)))) break;
          tc_fence_after();
          uint32_t rc[RH];
          tmem_ld<RH>(tl + b * (uint32_t)a.NP + (uint32_t)(h * RH), rc);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.tmem_empty[b]);
          ++tcount;
          // online softmax partials against a per-row reference m (the
          // lane's first visible logit, 0 while there is none): z += 2^(x - m)
          // with x - m kept at most 2^6 by re-basing the rare rows that jump
          // above it.  Rows past R (padding, statistics) run unmasked; their
          // partials are not kept.  x - m is computed in place in rc.
          const bool full_vis = it0 + kTile - 1 <= a.N - a.W;  // every window row sees every key
          const int vis_from = i - (a.N - a.W);                 // else row j sees key i iff j >= vis_from
          if (t == 0) {
            int j = (a.row0 + h * RH) % a.W;  // the window position of the half's first row
#pragma unroll
            for (int c = 0; c < RH; ++c) {
              const bool vis = full_vis || (valid && j >= vis_from);
              if (++j == a.W) j = 0;
              m[c] = vis ? __uint_as_float(rc[c]) * a.scale_log2 : 0.f;
              z[c] = vis ? 1.f : 0.f;
            }
          } else {
            float mx = -INFINITY;
            if (full_vis) {
#pragma unroll
              for (int c = 0; c < RH; ++c) {
                const float dl = fmaf(__uint_as_float(rc[c]), a.scale_log2, -m[c]);
                rc[c] = __float_as_uint(dl);
                mx = fmaxf(mx, dl);
              }
            } else {
              int j = (a.row0 + h * RH) % a.W;  // the window position of the half's first row
#pragma unroll
              for (int c = 0; c < RH; ++c) {
                const bool vis = valid && j >= vis_from;
                if (++j == a.W) j = 0;
                const float dl = vis ? fmaf(__uint_as_float(rc[c]), a.scale_log2, -m[c]) : -INFINITY;
                rc[c] = __float_as_uint(dl);
                mx = fmaxf(mx, dl);
              }
            }
            if (mx > 64.f) {
#pragma unroll
              for (int c = 0; c < RH; ++c) {
                const float dl = __uint_as_float(rc[c]);
                if (dl > 20.f) {
                  z[c] *= ex2(-dl);
                  m[c] += dl;
                  rc[c] = 0u;
                }
              }
            }
#pragma unroll
            for (int c = 0; c < RH; ++c) z[c] += ex2(__uint_as_float(rc[c]));
          }
        }
        // item end: per-row (max, sum) over the 32 keys of the warp by a
        // reduce-scatter (31 shuffle pairs instead of 5 per row)
#pragma unroll
        for (int c = 0; c < RH; ++c) m[c] = z[c] > 0.f ? m[c] : -INFINITY;  // lanes without a visible key do not count
        warp_reduce_scatter_maxsum<RH>(m, z, lane);
        constexpr int kShift = RH >= 32 ? 0 : (RH == 16 ? 1 : 2);  // lanes sharing a row after the scatter
        constexpr int kPer = RH > 32 ? RH / 32 : 1;                  // rows a lane holds
        if ((lane & ((1 << kShift) - 1)) == 0) {
#pragma unroll
          for (int j = 0; j < kPer; ++j) {
            const int row = (lane >> kShift) * kPer + j;
            s.red[e][row][0] = m[j];
            s.red[e][row][1] = z[j];
          }
        }
        if (!epi_sync()) {
          ok = false;
          break;
        }
        float* part = a.p1part + ((size_t)u * a.rmax + rec) * a.p1_stride;
        if (tid < a.R) {
          const int hh = tid / RH, c = tid % RH;
          float Mx = -INFINITY;
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) Mx = fmaxf(Mx, s.red[4 * hh + w4][c][0]);
          float Z = 0.f;
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) {
            const float mm = s.red[4 * hh + w4][c][0];
            if (mm != -INFINITY) Z += s.red[4 * hh + w4][c][1] * ex2(mm - Mx);
          }
          part[2 * kD + tid] = Mx;
          part[2 * kD + a.R4 + tid] = Z;
        }
        // once the key warps' chunk sums are written too, one gpu-scope
        // release publishes the item (every partial write is ordered before
        // it by the barrier and the kpub wait)
        named_bar_sync(kEpiBar, kEpi);
        if (tid == 0) {
          ok = wait_bar(&s.kpub[slot], qphase, a, 19u);
          if (ok) red_add_release(arrivals(a, u), 1u);
          else s.epi_abort = 1;
        }
      } else {  // kP2
        // Pass 2 splits the tiles, not the rows: the warps of row half h take
        // the tiles t of the item with t % 2 == h and every row of them, so
        // no warp waits for another within a tile and the two halves work on
        // consecutive tiles at once.  Within an item a TMEM buffer (tcount
        // mod 4 or 2) and a norm slot (tile mod kNB) always serve the same
        // half; at item boundaries every epilogue warp meets at the item's
        // first barrier, so a half never waits on a phase whose previous
        // use the other half has not consumed.  The stats warp has copied
        // the unit statistics and built the statistics rows.
        ok = __all_sync(0xffffffffu, wait_bar(&s.sready[slot], (spar >> slot) & 1u, a, 18u));
        spar ^= 1u << slot;
        const float* kbv = d.ust + ustat_kbar();
        const float ksq = d.ust[ustat_ksq()];
        // log2-sum-exp of every row (+inf past R: those vote terms, padding
        // and statistics columns, are exactly zero), in registers unless the
        // rows are too many; the tile's accumulator columns are read in
        // chunks of kCW
        constexpr int kCW = RH <= 32 ? 2 * RH : RH;
        constexpr bool kLseReg = RH <= 32;
        float lse_r[kLseReg ? 2 * RH : 1];
#pragma unroll
        for (int c = 0; c < (kLseReg ? 2 * RH : 1); ++c) lse_r[c] = d.ust[ustat_lse() + c];
        const float* lse_s = d.ust + ustat_lse();
        float s_all = 0.f, mn = INFINITY, mx = -INFINITY, s_de = 0.f, s_c = 0.f, s_raw = 0.f;
        for (int t = 0; t < ntiles && ok; ++t) {
          const uint32_t b = tcount & bmask, tph = (tcount >> nbuf_log) & 1u;
          const uint32_t ps = pcount % kNB, pph = (pcount / kNB) & 1u;
          ++tcount;
          ++pcount;
          if ((t & 1) != h) continue;
          const int i = i0 + (ntiles - 1 - t) * kTile + kk;  // pass 2 walks the item backwards
          const bool valid = i < a.N;
          if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.tmem_full[b], tph, a, 14u)))) break;
          tc_fence_after();
          // the vote of every row, chunk by chunk; the statistics columns
          // are the last eight of the accumulator: k . kbar in three terms,
          // k . mu in two
          float vp[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
          float kkb = 0.f, kmu = 0.f;
#pragma unroll
          for (int c0 = 0; c0 < 2 * RH; c0 += kCW) {
            uint32_t rc[kCW];
            tmem_ld<kCW>(tl + b * (uint32_t)a.NP + (uint32_t)c0, rc);
            tmem_wait_ld();
            if (c0 + kCW == 2 * RH) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive_cnt(&s.tmem_empty[b], 2u);  // this half's four warps stand for all eight
              kkb = (__uint_as_float(rc[kCW - 8]) + __uint_as_float(rc[kCW - 7])) + __uint_as_float(rc[kCW - 6]);
              kmu = __uint_as_float(rc[kCW - 5]) + __uint_as_float(rc[kCW - 4]);
            }
#pragma unroll
            for (int c = 0; c < kCW; ++c)
              vp[c & 7] += ex2(fmaf(__uint_as_float(rc[c]), a.scale_log2, -(kLseReg ? lse_r[c0 + c] : lse_s[c0 + c])));
          }
          const float v = ((vp[0] + vp[1]) + (vp[2] + vp[3])) + ((vp[4] + vp[5]) + (vp[6] + vp[7]));
          // the key's squared norm from the key warps
          if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.nfull[ps], pph, a, 15u)))) break;
          const float n2 = s.nbuf[ps][kk];
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.nempty[ps]);
          float d2 = fmaf(-2.f, kkb, n2) + ksq;
          if (valid && d2 < 0.015625f * (n2 + ksq)) {
            // cancellation regime: recompute |k - kbar|^2 from the key row
            const uint4* row = reinterpret_cast<const uint4*>(a.K) + ((size_t)u * a.N + i) * 16;
            float dp[4] = {0.f, 0.f, 0.f, 0.f};
            for (int c = 0; c < 16; ++c) {
              const uint4 kv = __ldg(row + c);
              const uint32_t w4[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
              for (int t2 = 0; t2 < 4; ++t2) {
                const float dl = __uint_as_float(w4[t2] << 16) - kbv[c * 8 + 2 * t2];
                const float dh = __uint_as_float(w4[t2] & 0xffff0000u) - kbv[c * 8 + 2 * t2 + 1];
                dp[t2] = fmaf(dl, dl, dp[t2]);
                dp[t2] = fmaf(dh, dh, dp[t2]);
              }
            }
            d2 = (dp[0] + dp[1]) + (dp[2] + dp[3]);
          }
          const float dEv = sqrtf(fmaxf(d2, 0.f));
          const float cs = kmu * rsqrtf(fmaxf(n2, 1e-24f));
          if (valid) {
            s_all += dEv;
            if (i < a.Tv) {
              mn = fminf(mn, dEv);
              mx = fmaxf(mx, dEv);
              s_de += dEv;
              s_c += cs;
              s_raw += v;
              const size_t o = (size_t)u * a.Tv + i;
              a.simp[o] = a.row0 == 0 ? v : __ldcg(a.simp + o) + v;
              a.dE[o] = dEv;
              a.cosv[o] = cs;
            }
          }
        }
        // the chunk's six partials: warp butterflies, then one thread per
        // partial combines the eight warps in a fixed order
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          s_all += __shfl_xor_sync(0xffffffffu, s_all, o);
          mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
          s_de += __shfl_xor_sync(0xffffffffu, s_de, o);
          s_c += __shfl_xor_sync(0xffffffffu, s_c, o);
          s_raw += __shfl_xor_sync(0xffffffffu, s_raw, o);
        }
        if (lane == 0) {
          s.red6[e][0] = s_all;
          s.red6[e][1] = mn;
          s.red6[e][2] = mx;
          s.red6[e][3] = s_de;
          s.red6[e][4] = s_c;
          s.red6[e][5] = s_raw;
        }
        if (!epi_sync()) {
          ok = false;
          break;
        }
        if (tid < 6) {
          float acc = s.red6[0][tid];
#pragma unroll
          for (int w8 = 1; w8 < 8; ++w8) {
            const float x = s.red6[w8][tid];
            acc = tid == 1 ? fminf(acc, x) : tid == 2 ? fmaxf(acc, x) : acc + x;
          }
          // the item's record slot; the unit's first record also fills every
          // slot past the unit's records with the identity of its reduction
          float* p = a.p2part + (size_t)u * a.rmax * kP2Stride;
          // P2_SUM_DE_ALL, P2_MIN_DE, P2_MAX_DE, P2_SUM_DE, P2_SUM_COS, P2_SUM_RAW; a later row group
          // adds its vote sum, the distance and cosine partials are the same in every group
          if (tid == P2_SUM_RAW && a.row0 > 0) acc += __ldcg(p + rec * kP2Stride + tid);
          p[rec * kP2Stride + tid] = acc;
          if (rec == 0) {
            int c0, nrec;
            unit_slices(a, u, c0, nrec);
            const float idn = tid == P2_MIN_DE ? INFINITY : tid == P2_MAX_DE ? -INFINITY : 0.f;
            for (int q = nrec; q < a.rmax; ++q) p[q * kP2Stride + tid] = idn;
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_empty[slot]);
    }
  } else {
    reg_dealloc<kRegsOther>();
  if (warp == 0) {
    // ------------------------------------------------ scheduler + TMA producer
    int stage = 0;
    uint32_t sphase = 0;
    uint32_t used_bits = 0u, par_bits = 0u;    // per key stage: loaded at least once / parity of loads
    uint32_t qused_bits = 0u, qpar_bits = 0u;  // the same per window-query slot
    // the first read of a key is kept in L2 for its second read when pass 2
    // follows pass 1 by a few blocks; the second read is the last
    const uint64_t pol_p1 = a.lag < a.nw ? l2_policy_evict_last() : l2_policy_evict_first();
    const uint64_t pol_p2 = l2_policy_evict_first();
    int seq = 0;
    // One item: publish its descriptor (and start its window-query copy),
    // then load its key tiles into the ring.
    auto emit = [&](int type, int u, int t_lo, int ntiles, int rec) -> bool {
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      const int i0 = t_lo * kTile;
      const uint64_t pol = type == kP1 ? pol_p1 : pol_p2;
      if (type == kP1) {
        // the item's first pass-1 tiles go to L2 now, ahead of the
        // shared-memory ring (a few only: more floods the memory queues)
        for (int e = lane; e < 2 * min(ntiles, kPrefetchTiles); e += 32)
          tma_prefetch_3d(&tmK, (e & 1) * 64, i0 + (e >> 1) * kTile, u, pol_p1);
      }
      bool good = true;
      if (lane == 0) good = wait_bar(&s.item_empty[slot], qphase ^ 1u, a, 1u);
      if (__shfl_sync(0xffffffffu, good, 0) == 0) return false;
      ItemDesc& d = s.desc[slot];
      if (lane == 0) {
        d.type = type;
        d.u = u;
        d.rec = rec;
        d.i0 = i0;
        d.ntiles = ntiles;
        if (type == kP1 || type == kP2) {
          // window queries by TMA (swizzled in flight); the MMA (pass 1) or
          // the stats warp (pass 2) waits for them, not this warp
          const int layer = u / a.h_kv, head = u % a.h_kv;
          const int qrow = (layer * a.h_q + head * a.g) * a.W + a.row0;
          mbar_expect_tx(&s.qfull[slot], (uint32_t)a.NP * 256u);
          tma_load_2d(s.qbuf[slot], &tmQ, &s.qfull[slot], 0, qrow);
          tma_load_2d(s.qbuf[slot] + a.NP * 128, &tmQ, &s.qfull[slot], 64, qrow);
          qused_bits |= 1u << slot;
          qpar_bits ^= 1u << slot;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_full[slot]);
      ++seq;
      for (int t = 0; t < ntiles; ++t) {
        if (lane == 0) {
          good = wait_bar(&s.empty[stage], sphase ^ 1u, a, 4u);
          if (good) {
            mbar_expect_tx(&s.full[stage], kTileBytes);
            const int y = i0 + (type == kP2 ? ntiles - 1 - t : t) * kTile;
            tma_load_3d_hint(s.ktile[stage], &tmK, &s.full[stage], 0, y, u, pol);
            tma_load_3d_hint(s.ktile[stage] + kTileBytes / 2, &tmK, &s.full[stage], 64, y, u, pol);
            used_bits |= 1u << stage;
            par_bits ^= 1u << stage;
          }
        }
        if (__shfl_sync(0xffffffffu, good, 0) == 0) return false;
        if (++stage == kStages) {
          stage = 0;
          sphase ^= 1u;
        }
      }
      return true;
    };
    // Step s: pass 1 of this CTA's slice of wave s; the folds of the units of
    // wave s - 1 it owns (unit u belongs to CTA u mod P, so that no CTA folds
    // in every wave); pass 2 of its slice of wave s - lag.  A fold holds its
    // CTA's epilogue until the unit's last pass-1 item has arrived; a step
    // later every CTA has long finished wave s - 1, and pass 2 of those units
    // (lag >= 2) comes a step later still.
    const int c = blockIdx.x;
    for (int st = 0; st < a.nw + a.lag && ok; ++st) {
      for (int ph = 0; ph < 3 && ok; ++ph) {  // 0: pass 1, 1: folds, 2: pass 2
        const int w = ph == 0 ? st : (ph == 1 ? st - 1 : st - a.lag);
        if (w < 0 || w >= a.nw) continue;
        if (ph == 1) {
          const int u1 = min((w + 1) * a.uw, a.U);
          for (int u = w * a.uw + ((c - w * a.uw) % a.P + a.P) % a.P; u < u1 && ok; u += a.P)
            ok = emit(kFold, u, 0, 0, 0);
          continue;
        }
        const int L = wave_tiles(a, w), n = min(a.P, L);
        if (c >= n) continue;
        const int g0 = w * a.uw * a.T;  // the wave's first tile, counted over all units
        const int lo = g0 + slice_start(c, L, n), hi = g0 + slice_start(c + 1, L, n);
        // pass 2 walks the slice backwards (units and tiles): the keys pass 1
        // read last are the likeliest still to be in L2
        const int u_first = lo / a.T, u_last = (hi - 1) / a.T;
        for (int k = 0; u_first + k <= u_last && ok; ++k) {
          const int u = ph == 0 ? u_first + k : u_last - k;
          const int t_lo = max(lo, u * a.T) - u * a.T, t_hi = min(hi, (u + 1) * a.T) - u * a.T;
          int c0, nrec;
          unit_slices(a, u, c0, nrec);
          ok = emit(ph == 0 ? kP1 : kP2, u, t_lo, t_hi - t_lo, c - c0);
        }
      }
    }
    if (ok) {
      // no work left for this CTA: the next launch (finalisation) may be
      // scheduled on SMs as they drain; it waits for this grid's completion
      // before reading anything
      ok = emit(kExit, 0, 0, 0, 0);
      asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    }
    if (!ok && lane == 0) {
      // let this CTA's copies in flight land before its shared memory goes
      // away: the last key tile of every stage and the last window-query copy
      // of every slot (a slot or stage is reloaded only after its previous
      // copy was consumed, so only the last one can be pending)
      for (int st = 0; st < kStages; ++st)
        if (used_bits & (1u << st)) drain_bar(&s.full[st], ((par_bits >> st) & 1u) ^ 1u, a);
      for (int sl = 0; sl < kIQ; ++sl)
        if (qused_bits & (1u << sl)) drain_bar(&s.qfull[sl], ((qpar_bits >> sl) & 1u) ^ 1u, a);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t sphase = 0, tcount = 0;
      uint32_t spar = 0u;  // per slot: parity of the next sready phase (completed by P2 items only)
      uint32_t qpar = 0u;  // per slot: parity of the next qfull phase (completed by P1 and P2 items)
      const uint32_t idesc_l = idesc_bf16(128, a.NP, false, false);
      for (int seq = 0; ok; ++seq) {
        const int slot = seq % kIQ;
        const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
        if (!(ok = wait_bar(&s.item_full[slot], qphase, a, 5u))) break;
        const ItemDesc& d = s.desc[slot];
        const int type = d.type, ntiles = d.ntiles;
        if (type == kExit) break;
        if (type == kP1 || type == kP2) qpar ^= 1u << slot;
        if (type == kP1) {
          // the window queries landed
          if (!(ok = wait_bar(&s.qfull[slot], ((qpar >> slot) & 1u) ^ 1u, a, 17u))) break;
        } else if (type == kP2) {
          // the stats warp has the unit statistics and wrote the statistics rows
          if (!(ok = wait_bar(&s.sready[slot], (spar >> slot) & 1u, a, 17u))) break;
          spar ^= 1u << slot;
        }
        tc_fence_after();
        const uint32_t qb = smem_u32(s.qbuf[slot]);
        for (int t = 0; t < ntiles; ++t) {
          const uint32_t b = tcount & ((1u << nbuf_log) - 1u), tph = (tcount >> nbuf_log) & 1u;
          if (!(ok = wait_bar(&s.full[stage], sphase, a, 6u))) break;
          if (!(ok = wait_bar(&s.tmem_empty[b], tph ^ 1u, a, 7u))) break;
          tc_fence_after();
          const uint32_t kt = smem_u32(s.ktile[stage]);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t ad = smem_desc(kt + (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32, 16, 1024, 2);
            const uint64_t bd = smem_desc(qb + (kk >> 2) * (a.NP * 128) + (kk & 3) * 32, 16, 1024, 2);
            mma_bf16(tmem + b * (uint32_t)a.NP, ad, bd, idesc_l, kk > 0 ? 1u : 0u);
          }
          mma_commit(&s.tmem_full[b]);
          // pass 1: the sum MMA (warp 3) still reads the stage; pass 2: free it
          mma_commit(type == kP1 ? &s.lgdone[stage] : &s.empty[stage]);
          ++tcount;
          if (++stage == kStages) {
            stage = 0;
            sphase ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(&s.item_empty[slot]);
      }
      if (!ok) {
        mma_commit(&s.drain);
        drain_bar(&s.drain, 0u, a);
      }
    }
  } else if (warp == 3) {
    // ------------------------------------------------ sum-MMA issuer
    // For each pass-1 tile, once its logits MMA is complete and the key warps
    // have written the weights: the MMA of the key tile (MN-major view)
    // against [1, w_hi, w_mid, w_lo] that accumulates the chunk's sums of k
    // and k/||k||, then the release of the stage.  A thread of its own, so
    // that neither the logits issuer waits for the key warps nor a stage
    // waits for the next tile.
    if (lane == 0) {
      int stage = 0;
      uint32_t sigcount = 0, wpar = 0u, lpar = 0u;  // per stage: parity of the next wready / lgdone phase
      const uint32_t idesc_s = idesc_bf16(128, 16, true, false);
      for (int seq = 0; ok; ++seq) {
        const int slot = seq % kIQ;
        const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
        if (!(ok = wait_bar(&s.item_full[slot], qphase, a, 28u))) break;
        const ItemDesc& d = s.desc[slot];
        const int type = d.type, ntiles = d.ntiles;
        if (type == kExit) break;
        mbar_arrive(&s.item_empty[slot]);  // the descriptor is read
        for (int t = 0; t < ntiles; ++t) {
          if (type == kP1) {
            if (!(ok = wait_bar(&s.lgdone[stage], (lpar >> stage) & 1u, a, 29u))) break;
            lpar ^= 1u << stage;
            if (!(ok = wait_bar(&s.wready[stage], (wpar >> stage) & 1u, a, 8u))) break;
            wpar ^= 1u << stage;
            const uint32_t sb = sigcount & 1u, sph = (sigcount >> 1) & 1u;
            if (t == 0 && !(ok = wait_bar(&s.sigma_empty[sb], sph ^ 1u, a, 9u))) break;
            tc_fence_after();
            const uint32_t kt = smem_u32(s.ktile[stage]);
            const uint32_t wb = smem_u32(s.wbuf[stage]);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              // A = key tile viewed MN-major (d contiguous): 16 keys per step
              const uint64_t ad = smem_desc(kt + kk * 2048, kTileBytes / 2, 1024, 2);
              const uint64_t bd = smem_desc(wb + (kk >> 2) * 2048 + (kk & 3) * 32, 16, 1024, 2);
              mma_bf16(tmem + kSigmaCol + 16u * sb, ad, bd, idesc_s, (t > 0 || kk > 0) ? 1u : 0u);
            }
            mma_commit(&s.empty[stage]);
            if (t == ntiles - 1) {
              mma_commit(&s.sigma_full[sb]);
              ++sigcount;
            }
          }
          if (++stage == kStages) stage = 0;
        }
      }
      if (!ok) {
        mma_commit(&s.drain2);
        drain_bar(&s.drain2, 0u, a);
      }
    }
  } else if (warp == 2) {
    // ------------------------------------------------ stats warp
    // Readies the unit statistics of every P2 item, about one item ahead of
    // the epilogue: waits for the unit's ready flag (raised by the fold
    // item), copies the record into the item descriptor, gives the rows past
    // R an infinite log-sum-exp (their vote terms are then exactly zero) and,
    // once the window queries have landed, writes the statistics rows of the
    // MMA operand over them.
    uint32_t qpar = 0u;  // per slot: parity of the next qfull phase (completed by P1 and P2 items)
    for (int seq = 0; ok; ++seq) {
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.item_full[slot], qphase, a, 26u)))) break;
      const ItemDesc& d = s.desc[slot];
      const int type = d.type, u = d.u;
      if (type == kExit) break;
      if (type == kP1 || type == kP2) qpar ^= 1u << slot;
      if (type == kP2) {
        float* ust = s.desc[slot].ust;
        if (lane == 0) ok = wait_count(stats_ready(a, u), 1u, a, 31u);
        ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
        if (!ok) break;
        __syncwarp();  // lane 0's acquire orders the record's loads below
        const float4* g = reinterpret_cast<const float4*>(a.ustat + (size_t)u * a.ustat_stride);
        for (int e4 = lane; e4 < ustat_lse() / 4; e4 += 32) reinterpret_cast<float4*>(ust)[e4] = __ldcg(g + e4);
        // this row group's log2-sum-exp rows; +inf past them
        const float* gl = a.ustat + (size_t)u * a.ustat_stride + ustat_lse() + a.row0;
        for (int r = lane; r < a.NP; r += 32) ust[ustat_lse() + r] = r < a.R ? __ldcg(gl + r) : INFINITY;
        if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.qfull[slot], ((qpar >> slot) & 1u) ^ 1u, a, 27u)))) break;
        for (int e = lane; e < 5 * 16; e += 32) build_stat_rows(s.qbuf[slot], a, ust, e);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.sready[slot]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_empty[slot]);
    }
  } else if (warp >= kKeyWarp0) {
    // ------------------------------------------------ key warps (12..15)
    const int kk = threadIdx.x - 32 * kKeyWarp0;  // 0..127: this thread's key row of each tile
    int stage = 0;
    uint32_t sphase = 0, p2count = 0, sigcount = 0;
    for (int seq = 0; ok; ++seq) {
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.item_full[slot], qphase, a, 20u)))) break;
      const ItemDesc& d = s.desc[slot];
      const int type = d.type, ntiles = d.ntiles, i0 = d.i0, u = d.u;
      if (type == kExit) break;
      for (int t = 0; t < ntiles && ok; ++t) {
        if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.full[stage], sphase, a, 22u)))) break;
        const int i = i0 + (type == kP2 ? ntiles - 1 - t : t) * kTile + kk;
        const bool valid = i < a.N;
        // squared norm of this thread's key (packed fp32 pairs), the same
        // arithmetic in both passes
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int hb = 0; hb < 2; ++hb) {
          const uint8_t* row = s.ktile[stage] + hb * (kTileBytes / 2) + kk * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 v = *reinterpret_cast<const uint4*>(row + ((c ^ (kk & 7)) << 4));
            sq_acc_bf16x2(v.x, acc[0], acc[1]);
            sq_acc_bf16x2(v.y, acc[2], acc[3]);
            sq_acc_bf16x2(v.z, acc[4], acc[5]);
            sq_acc_bf16x2(v.w, acc[6], acc[7]);
          }
        }
        const float n2 = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.empty[stage]);  // done with the key tile
        if (type == kP1) {
          // the sum weights w = 1/||k|| in three bf16 terms
          const float w = valid ? rsqrtf(fmaxf(n2, 1e-24f)) : 0.f;
          const __nv_bfloat16 whi = __float2bfloat16_rn(w);
          const float r1 = w - __bfloat162float(whi);
          const __nv_bfloat16 wmid = __float2bfloat16_rn(r1);
          const __nv_bfloat16 wlo = __float2bfloat16_rn(r1 - __bfloat162float(wmid));
          uint8_t* base = s.wbuf[stage] + (kk >> 6) * 2048 + (kk & 7) * 2;
          const int j = (kk & 63) >> 3;
          if (a.kbar_n < a.N)  // non-window centroid: the window keys leave the sum of k
            *reinterpret_cast<__nv_bfloat16*>(base + sw128(0, j)) = __float2bfloat16_rn(i < a.kbar_n ? 1.f : 0.f);
          *reinterpret_cast<__nv_bfloat16*>(base + sw128(1, j)) = whi;
          *reinterpret_cast<__nv_bfloat16*>(base + sw128(2, j)) = wmid;
          *reinterpret_cast<__nv_bfloat16*>(base + sw128(3, j)) = wlo;
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.wready[stage]);
        } else {
          // pass 2: the norm goes to the epilogue through shared memory
          const uint32_t nb = p2count % kNB, nph = (p2count / kNB) & 1u;
          ++p2count;
          if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.nempty[nb], nph ^ 1u, a, 23u)))) break;
          s.nbuf[nb][kk] = valid ? n2 : 0.f;
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.nfull[nb]);
        }
        if (++stage == kStages) {
          stage = 0;
          sphase ^= 1u;
        }
      }
      if (!ok) break;
      if (type == kP1) {
        // chunk sums of k and k/||k|| from the sum MMA (TMEM lane = dimension kk)
        const uint32_t sb = sigcount & 1u, sph = (sigcount >> 1) & 1u;
        ++sigcount;
        if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.sigma_full[sb], sph, a, 13u)))) break;
        tc_fence_after();
        uint32_t v[4];
        tmem_ld_x4(tmem + ((uint32_t)(32 * (warp & 3)) << 16) + kSigmaCol + 16u * sb, v);
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.sigma_empty[sb]);
        float* part = a.p1part + ((size_t)u * a.rmax + d.rec) * a.p1_stride;
        part[kk] = __uint_as_float(v[0]);
        part[kD + kk] = (__uint_as_float(v[1]) + __uint_as_float(v[2])) + __uint_as_float(v[3]);
      }
      // the item's chunk sums are written: the epilogue's gpu-scope arrival
      // (after it has waited for kpub) publishes them
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&s.kpub[slot]);
        mbar_arrive(&s.item_empty[slot]);
      }
    }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// per-device host state; a racing thread repeats the idempotent setup
std::atomic<int> g_num_sms[64];
std::atomic<bool> g_attr_set[64][4];

template <int RH>
cudaError_t launch_rh(const CUtensorMap& tm, const CUtensorMap& tq, const TcArgs& a, int dev, cudaStream_t st) {
  const size_t smem = sizeof(Smem<RH>) + 1024;
  const int rh_i = RH == 8 ? 0 : RH == 16 ? 1 : RH == 32 ? 2 : 3;
  if (!g_attr_set[dev][rh_i].load()) {
    // the warpgroups' register split needs the launch to give every thread
    // 65536 / kThreads registers; refuse to launch otherwise
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, tc_evict_kernel<RH>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs * kThreads < 2 * 128 * (int)(kRegsEpi + kRegsOther)) return cudaErrorInvalidConfiguration;
    e = cudaFuncSetAttribute(tc_evict_kernel<RH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    g_attr_set[dev][rh_i].store(true);
  }
  // a cooperative launch: every CTA of the grid is resident at once (the
  // static schedule has CTAs wait for other CTAs' pass-1 items), or the
  // launch fails
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)a.P);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, tc_evict_kernel<RH>, tm, tq, a);
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::atomic<EncodeTiledFn> fn{nullptr};  // a racing thread repeats the lookup
  EncodeTiledFn f = fn.load();
  if (f == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess) {
      f = reinterpret_cast<EncodeTiledFn>(p);
      fn.store(f);
    }
  }
  return f;
}

}  // namespace

size_t tc_smem_bytes() { return sizeof(Smem<32>) + 1024; }

int tc_record_slots(int T, int Lmin) {
  // slices of a wave of L >= Lmin tiles cut in n = min(P, L) pieces, P <=
  // kTcMaxSms, hold at least s = max(1, floor(Lmin / kTcMaxSms)) tiles; a
  // unit's T consecutive tiles meet at most ceil((T - 1) / s) + 1 of them
  const int s = Lmin / kTcMaxSms > 1 ? Lmin / kTcMaxSms : 1;
  return (T - 1 + s - 1) / s + 1;
}

int tc_rows_half(int R) {
  const int r4 = (R + 3) & ~3;
  int np = 16;
  while (np < r4 + 8) np <<= 1;  // window rows, then the statistics rows in the last eight
  return np > kNPMax ? 0 : np / 2;
}

cudaError_t launch_tc(const void* K, const TcArgs& args, cudaStream_t st) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (g_num_sms[dev].load() == 0) {
    int n = 0;
    e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    g_num_sms[dev].store(n);
  }
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return cudaErrorNotSupported;
  CUtensorMap tm;
  const cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)args.N, (cuuint64_t)args.U};
  const cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)args.N * kD * 2};
  const cuuint32_t box[3] = {64, (cuuint32_t)kTile, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(K), dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  // window queries as a 2-D [L * h_q * W rows, 128] bf16 tensor, boxes of
  // [NP rows x 64 columns] with the same 128-byte swizzle as the key tiles
  CUtensorMap tq;
  const cuuint64_t qdims[2] = {(cuuint64_t)kD, (cuuint64_t)args.q_rows};
  const cuuint64_t qstrides[1] = {(cuuint64_t)kD * 2};
  const cuuint32_t qbox[2] = {64, (cuuint32_t)args.NP};
  if (enc(&tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(args.Q), qdims, qstrides, qbox, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  switch (args.NP / 2) {
    case 8: return launch_rh<8>(tm, tq, args, dev, st);
    case 16: return launch_rh<16>(tm, tq, args, dev, st);
    case 32: return launch_rh<32>(tm, tq, args, dev, st);
    case 64: return launch_rh<64>(tm, tq, args, dev, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace ecokv
