// Persistent tensor-core kernel for bf16 inputs: the whole eviction pass in
// one launch on sm_103a.
//
// Work is a global, ticket-ordered list of items:
//   P1(u, c)  pass 1 over chunk c (up to 32 tiles of 128 keys) of unit u
//             (u = (layer, KV head)): window logits (tcgen05 MMA, keys as M,
//             window rows as N), per-row online-softmax partials, key norms,
//             and the chunk sums of k and k/||k|| (a second tcgen05 MMA with the
//             key tile as an MN-major operand against [1, w_hi, w_mid, w_lo]
//             weight rows, w = 1/||k|| split into three bf16 terms).  The last P1 item of a unit folds the partials into the unit
//             statistics (kbar, mu, per-row log2-sum-exp).
//   P2(u, c)  pass 2: logits again plus five extra MMA columns holding k . kbar
//             (kbar split into three bf16 terms) and k . mu (two terms), giving
//             the importance vote, the cosine khat . mu, and d_E (Eq. 1) by the
//             expansion of Sec. 4 from ||k||^2 (stored by pass 1).  Where that
//             expansion cancels (d_E^2 below 2^-6 of ||k||^2 + ||kbar||^2, keys
//             close to their centroid) the key is recomputed directly from its
//             row in global memory.
// Work is a global, ticket-ordered list of items.  Within a schedule step s
// the list holds P1(s, *) then P2(s - lag_p2, *): pass 2 of a unit runs lag_p2
// units after its pass 1 (a short lag re-reads the keys from L2, a long one
// never waits for unit statistics; the host picks), and every item depends
// only on items with smaller tickets: dispatch is deadlock-free without
// co-residency.  Pass 2 leaves per-candidate arrays and per-chunk partial
// sums; finalisation, selection and the gather of the kept rows run in the
// next launches (finalize_select.cu).
//
// Warp roles (512 threads, one CTA per SM): warp 0 takes tickets, resolves
// dependencies (bounded spins on gpu-scope flags), loads the window queries
// (TMA) and the unit statistics (bulk copy) and issues TMA loads of 32 KB key
// tiles into a 5-stage ring; warp 1 issues the logits MMAs into up to four
// TMEM accumulators; warp 3 issues the sum MMAs of pass-1 tiles (two more
// accumulators) as soon as a tile's logits are done and its weights written,
// and frees the stage; warp 2 counts finished pass-1 items and folds completed
// units; warps 12-15 (key warps, one key per thread) compute the key norms
// and the sum weights of each pass-1 tile as soon as it lands, store the norms
// for pass 2, read the chunk sums, and hand the norms to the epilogue in pass
// 2; warps 4-11 are the epilogue (one key per TMEM lane, window rows split in
// two halves).  A stage is held only as long as its own tile needs it: the
// number of key bytes in flight per SM, not the arithmetic, sets the pace.
// setmaxnreg gives the two epilogue warpgroups 176 registers a thread and the
// others 80.  Every mbarrier wait and spin is bounded: on timeout the kernel
// records ECOKV_ERR_TIMEOUT, raises a gpu-wide abort flag, drains its own
// copies and MMAs, frees TMEM and exits.

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

enum : int { kP1 = 0, kP2 = 1, kExit = 3 };

constexpr int kNB = 4;                // pass-2 norm hand-off slots
constexpr int kUstatMax = 2 * kD + 4 + kNPMax;  // floats of a unit statistics record (lse padded to NP rows)

struct __align__(16) ItemDesc {
  int type, u, chunk, part, i0, ntiles;
  int pad[2];
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
  float xch[kNB][kTile];                        // pass-2 vote of the first row half, per key
  float red[8][RH][2];                          // [epilogue warp][row][max, sum]
  float red6[4][8];                             // [second-half warp][pass-2 partial]
  uint64_t full[kS], empty[kS], wready[kS];
  uint64_t item_full[kIQ], item_empty[kIQ], qfull[kIQ];
  uint64_t tmem_full[4], tmem_empty[4];
  uint64_t sigma_full[2], sigma_empty[2], drain, drain2;
  uint64_t lgdone[kS];  // pass-1 tile: its logits MMA is complete (for the sum-MMA issuer)
  float nbuf[kNB][kTile];                        // pass-2 squared key norms, key warps -> epilogue
  uint64_t nfull[kNB], nempty[kNB];
  uint64_t xfull[kNB], xempty[kNB];             // first row half -> second row half, per pass-2 tile
  uint64_t kpub[kIQ];    // key warps have published this item's key norms (gpu scope)
  uint64_t p1done[kIQ];  // the epilogue has written this pass-1 item's partials
  uint32_t tmem_base;
  int epi_abort;         // an epilogue warp gave up a wait (read after a named barrier)
};

static_assert(sizeof(Smem<8>) + 1024 <= 232448 && sizeof(Smem<16>) + 1024 <= 232448 &&
                  sizeof(Smem<32>) + 1024 <= 232448 && sizeof(Smem<64>) + 1024 <= 232448,
              "shared-memory plan exceeds the 227 KB per-CTA limit");
static_assert(sizeof(ItemDesc) % 16 == 0 && offsetof(ItemDesc, ust) % 16 == 0, "bulk-copy target alignment");

__device__ __forceinline__ unsigned* abort_flag(const TcArgs& a) { return a.sync + 1; }

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
  const long long t0 = clock64();
  for (unsigned spins = 1;; ++spins) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((spins & 63u) == 0u) {
      if (aborted(a)) return false;
      if (clock64() - t0 > a.timeout_cycles) {
        raise_abort(a, ECOKV_ERR_TIMEOUT, where);
        return false;
      }
    }
  }
}

// Tiles of a chunk, and of part p (1..nparts) of it (its first tile in *t0);
// part 0 is the whole chunk.
__device__ __forceinline__ int chunk_tiles(const TcArgs& a, int chunk) {
  return min(a.tiles_per_chunk, (a.N - chunk * a.tiles_per_chunk * kTile + kTile - 1) / kTile);
}
__device__ __forceinline__ int part_tiles(const TcArgs& a, int chunk, int part, int* t0) {
  const int nt = chunk_tiles(a, chunk);
  if (part == 0) {
    if (t0) *t0 = 0;
    return nt;
  }
  const int per = (nt + a.nparts - 1) / a.nparts, first = (part - 1) * per;
  if (t0) *t0 = first;
  return min(per, nt - first);
}

struct Item {
  int type, u, chunk, part;
  bool valid;
};

// Item of a ticket.  Schedule step s holds the P1 items of unit s and then
// the P2 items of unit s - lag_p2; steps are numbered so that no ticket falls
// outside [0, U): the first lag_p2 steps hold P1 items only, the last lag_p2
// steps P2 items only, 2 * U * nchunks tickets in all.  lag_p2 = U runs all of
// pass 1 before any of pass 2.
__device__ Item decode(int ticket, const TcArgs& a) {
  Item it{kExit, 0, 0, 0, true};
  if (ticket >= a.total_tickets) return it;
  int part = 0;
  if (ticket >= a.split_from) {
    // the last pass-2 items, each split in nparts consecutive parts
    const int rel = ticket - a.split_from;
    part = 1 + rel % a.nparts;
    ticket = a.split_from + rel / a.nparts;
  }
  it.part = part;
  const int nc = a.nchunks, L = a.lag_p2;
  const int head = L * nc, body = (a.U - L) * 2 * nc;
  if (ticket < head) {
    it.type = kP1;
    it.u = ticket / nc;
    it.chunk = ticket - it.u * nc;
  } else if (ticket < head + body) {
    const int rel = ticket - head, st = rel / (2 * nc), slot = rel - st * 2 * nc;
    if (slot < nc) {
      it.type = kP1;
      it.u = L + st;
      it.chunk = slot;
    } else {
      it.type = kP2;
      it.u = st;
      it.chunk = slot - nc;
    }
  } else {
    const int rel = ticket - head - body, v = rel / nc;
    it.type = kP2;
    it.u = a.U - L + v;
    it.chunk = rel - v * nc;
  }
  it.valid = it.u >= 0 && it.u < a.U;
  if (part > 0 && part_tiles(a, it.chunk, part, nullptr) <= 0) it.valid = false;  // a part past the chunk's end
  return it;
}

// Bounded spin on a gpu-scope flag written by another CTA.
__device__ bool wait_flag(const unsigned* f, const TcArgs& a, unsigned where) {
  const long long t0 = clock64();
  while (ld_acquire(f) == 0u) {
    if (aborted(a)) return false;
    if (clock64() - t0 > a.timeout_cycles) {
      raise_abort(a, ECOKV_ERR_TIMEOUT, where);
      return false;
    }
    __nanosleep(128);
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
// rows 0..R-1 arrive by TMA.  Run by the 32 lanes of warp 0.
__device__ void build_stat_rows(uint8_t* qb, const TcArgs& a, float* ust, int lane) {
  // rows past the window rows (padding and the statistics rows) get an
  // infinite log-sum-exp, so that their vote terms are exactly zero
  for (int r = a.R + lane; r < a.NP; r += 32) ust[ustat_lse() + r] = INFINITY;
  for (int e = lane; e < 5 * 16; e += 32) {
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
}

// Fold every chunk's pass-1 partials of unit u into its statistics record,
// one warp: lane l sums key dimensions 4l..4l+3 (16-byte loads) and combines
// the (max, sum) pairs of window rows l, l + 32, ... online.  Loads go out in
// batches so that the L2 latency is paid a few times per unit.  Chunk record:
// [sum k (d)] [sum k/||k|| (d)] [row max (R4)] [row sum (R4)].
__device__ void unit_reduce_warp(const TcArgs& a, int u, int lane) {
  const int nch = a.nchunks;
  const float* base = a.p1part + (size_t)u * nch * a.p1_stride;
  float* us = a.ustat + (size_t)u * a.ustat_stride;
  constexpr int kB = 8;
  float4 sk = make_float4(0.f, 0.f, 0.f, 0.f), sh = sk;
  for (int c0 = 0; c0 < nch; c0 += kB) {
    float4 kv[kB], hv[kB];
#pragma unroll
    for (int j = 0; j < kB; ++j) {
      const float4* p = reinterpret_cast<const float4*>(base + (size_t)min(c0 + j, nch - 1) * a.p1_stride);
      kv[j] = __ldcg(p + lane);
      hv[j] = __ldcg(p + kD / 4 + lane);
    }
#pragma unroll
    for (int j = 0; j < kB; ++j)
      if (c0 + j < nch) {
        sk.x += kv[j].x; sk.y += kv[j].y; sk.z += kv[j].z; sk.w += kv[j].w;
        sh.x += hv[j].x; sh.y += hv[j].y; sh.z += hv[j].z; sh.w += hv[j].w;
      }
  }
  const float inv_n = 1.f / (float)a.N, inv_k = 1.f / (float)a.kbar_n;
  const float4 kb = make_float4(sk.x * inv_k, sk.y * inv_k, sk.z * inv_k, sk.w * inv_k);
  const float4 mu = make_float4(sh.x * inv_n, sh.y * inv_n, sh.z * inv_n, sh.w * inv_n);
  reinterpret_cast<float4*>(us + ustat_kbar())[lane] = kb;
  reinterpret_cast<float4*>(us + ustat_mu())[lane] = mu;
  float ksq = (kb.x * kb.x + kb.y * kb.y) + (kb.z * kb.z + kb.w * kb.w);
  float msq = (mu.x * mu.x + mu.y * mu.y) + (mu.z * mu.z + mu.w * mu.w);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ksq += __shfl_xor_sync(0xffffffffu, ksq, o);
    msq += __shfl_xor_sync(0xffffffffu, msq, o);
  }
  if (lane == 0) {
    us[ustat_ksq()] = ksq;
    us[ustat_musq()] = msq;
  }
  for (int r = lane; r < a.R; r += 32) {
    float M = -INFINITY, Z = 0.f;
    constexpr int kR = 16;
    for (int c0 = 0; c0 < nch; c0 += kR) {
      float mv[kR], zv[kR];
#pragma unroll
      for (int j = 0; j < kR; ++j) {
        const float* p = base + (size_t)min(c0 + j, nch - 1) * a.p1_stride + 2 * kD;
        mv[j] = __ldcg(p + r);
        zv[j] = c0 + j < nch ? __ldcg(p + a.R4 + r) : 0.f;
      }
#pragma unroll
      for (int j = 0; j < kR; ++j)
        if (zv[j] > 0.f) {
          const float Mn = fmaxf(M, mv[j]);
          Z = Z * ex2(M - Mn) + zv[j] * ex2(mv[j] - Mn);
          M = Mn;
        }
    }
    us[ustat_lse() + r] = M + log2f(Z);
  }
}

// Joint (max, sum) of partial softmax sums: (m1, z1) + (m2, z2) with z
// relative to 2^m; an empty pair has m = -inf, z = 0.
__device__ __forceinline__ void combine_maxsum(float& m, float& z, float m2, float z2) {
  const float M = fmaxf(m, m2);
  const float Ms = M == -INFINITY ? 0.f : M;
  z = z * ex2(m - Ms) + z2 * ex2(m2 - Ms);
  m = M;
}

// Reduce-scatter of RH (max, sum) rows over the 32 lanes of a warp: each
// step exchanges half of the remaining rows with the partner lane, so lane l
// ends with row (l >> shift) * per + j in m[j], z[j] (shift = 0, 1, 2 for
// RH = 32 (or more), 16, 8; per = RH / 32 rows when RH > 32); lanes that share
// a row hold the same value.
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
      mbar_init(&s.p1done[i], 8);
      mbar_init(&s.qfull[i], 1);
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
      mbar_init(&s.nempty[i], 4);  // the 4 epilogue warps of the second row half
      mbar_init(&s.xfull[i], 4);   // first row half
      mbar_init(&s.xempty[i], 4);  // second row half
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
      const int u = d.u, chunk = d.chunk, i0 = d.i0, ntiles = d.ntiles;

      if (type == kP1) {
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
            int j = (h * RH) % a.W;
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
              int j = (h * RH) % a.W;
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
        float* part = a.p1part + ((size_t)u * a.nchunks + chunk) * a.p1_stride;
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
        // the stats warp counts the item once all eight warps have written
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.p1done[slot]);
      } else {  // kP2
        ok = __all_sync(0xffffffffu, wait_bar(&s.qfull[slot], qphase, a, 18u));  // statistics copy landed
        const float* lse = d.ust + ustat_lse();
        const float* kbv = d.ust + ustat_kbar();
        const float ksq = d.ust[ustat_ksq()];
        float s_all = 0.f, mn = INFINITY, mx = -INFINITY, s_de = 0.f, s_c = 0.f, s_raw = 0.f;
        for (int t = 0; t < ntiles && ok; ++t) {
          const int i = i0 + t * kTile + kk;
          const bool valid = i < a.N;
          const uint32_t b = tcount & bmask, tph = (tcount >> nbuf_log) & 1u;
          if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.tmem_full[b], tph, a, 14u)))) break;
          tc_fence_after();
          uint32_t rc[RH];
          tmem_ld<RH>(tl + b * (uint32_t)a.NP + (uint32_t)(h * RH), rc);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.tmem_empty[b]);
          ++tcount;
          const uint32_t ps = pcount % kNB, pph = (pcount / kNB) & 1u;
          ++pcount;
          // vote of this half's rows; the lse of rows past R is +inf, so
          // padding and statistics columns add exactly zero
          float vp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int c = 0; c < RH; ++c) vp[c & 3] += ex2(fmaf(__uint_as_float(rc[c]), a.scale_log2, -lse[h * RH + c]));
          const float vh = (vp[0] + vp[1]) + (vp[2] + vp[3]);
          if (h == 0) {
            // hand the first half's vote to the second half
            if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.xempty[ps], pph ^ 1u, a, 24u)))) break;
            s.xch[ps][kk] = vh;
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.xfull[ps]);
          } else {
            // the statistics columns (the last eight of the accumulator):
            // k . kbar in three terms, k . mu in two
            const float kkb =
                (__uint_as_float(rc[RH - 8]) + __uint_as_float(rc[RH - 7])) + __uint_as_float(rc[RH - 6]);
            const float kmu = __uint_as_float(rc[RH - 5]) + __uint_as_float(rc[RH - 4]);
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
            if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.xfull[ps], pph, a, 25u)))) break;
            const float v = vh + s.xch[ps][kk];
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.xempty[ps]);
            if (valid) {
              s_all += dEv;
              if (i < a.Tv) {
                mn = fminf(mn, dEv);
                mx = fmaxf(mx, dEv);
                s_de += dEv;
                s_c += cs;
                s_raw += v;
                const size_t o = (size_t)u * a.Tv + i;
                a.simp[o] = v;
                a.dE[o] = dEv;
                a.cosv[o] = cs;
              }
            }
          }
        }
        // the chunk's six partials: warp butterflies in the second half, then
        // its first warp combines the four warps in a fixed order
        if (h == 1) {
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
            s.red6[e - 4][0] = s_all;
            s.red6[e - 4][1] = mn;
            s.red6[e - 4][2] = mx;
            s.red6[e - 4][3] = s_de;
            s.red6[e - 4][4] = s_c;
            s.red6[e - 4][5] = s_raw;
          }
        }
        if (!epi_sync()) {
          ok = false;
          break;
        }
        if (tid < 6) {
          float acc = s.red6[0][tid];
#pragma unroll
          for (int w4 = 1; w4 < 4; ++w4) {
            const float x = s.red6[w4][tid];
            acc = tid == 1 ? fminf(acc, x) : tid == 2 ? fmaxf(acc, x) : acc + x;
          }
          // the chunk's slot of this part; the first part also fills every
          // slot no part writes with the identity of its reduction
          float* p = a.p2part + ((size_t)u * a.nchunks + chunk) * kTcP2Parts * kP2Stride;
          const int part = d.part;
          p[(part > 0 ? part - 1 : 0) * kP2Stride + tid] = acc;  // P2_SUM_DE_ALL, P2_MIN_DE, P2_MAX_DE, P2_SUM_DE, P2_SUM_COS, P2_SUM_RAW
          if (part <= 1) {
            const float idn = tid == P2_MIN_DE ? INFINITY : tid == P2_MAX_DE ? -INFINITY : 0.f;
            for (int q = 1; q < kTcP2Parts; ++q)
              if (part == 0 || q >= a.nparts || part_tiles(a, chunk, q + 1, nullptr) <= 0) p[q * kP2Stride + tid] = idn;
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
    uint32_t used_bits = 0u, par_bits = 0u;  // per stage: loaded at least once / parity of loads
    const uint64_t pol_keep = l2_policy_evict_last(), pol_drop = l2_policy_evict_first();
    for (int seq = 0; ok;) {
      int ticket = 0;
      if (lane == 0) ticket = (int)atomicAdd(a.sync, 1u);
      ticket = __shfl_sync(0xffffffffu, ticket, 0);
      const Item it = decode(ticket, a);
      if (!it.valid) continue;
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      if (lane == 0) {
        ok = wait_bar(&s.item_empty[slot], qphase ^ 1u, a, 1u);
        if (ok && it.type == kP2) {
          ok = wait_flag(a.sync + 4 + a.U + it.u, a, 2u);
          fence_proxy_async_global();  // the statistics are read next by a bulk copy (async proxy)
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
      if (!ok) break;
      ItemDesc& d = s.desc[slot];
      int t0 = 0;
      const int ntiles = it.type == kExit ? 0 : part_tiles(a, it.chunk, it.part, &t0);
      const int i0 = (it.chunk * a.tiles_per_chunk + t0) * kTile;
      if (lane == 0) {
        d.type = it.type;
        d.u = it.u;
        d.chunk = it.chunk;
        d.part = it.part;
        d.i0 = i0;
        d.ntiles = ntiles;
      }
      if (it.type == kP1 || it.type == kP2) {
        // window queries by TMA (swizzled in flight); pass 2 also copies the
        // unit statistics record
        const uint32_t ust_bytes = (uint32_t)a.ustat_stride * 4u;
        if (lane == 0) {
          const int layer = it.u / a.h_kv, head = it.u % a.h_kv;
          const int qrow = (layer * a.h_q + head * a.g) * a.W;
          mbar_expect_tx(&s.qfull[slot], (uint32_t)a.NP * 256u + (it.type == kP2 ? ust_bytes : 0u));
          tma_load_2d(s.qbuf[slot], &tmQ, &s.qfull[slot], 0, qrow);
          tma_load_2d(s.qbuf[slot] + a.NP * 128, &tmQ, &s.qfull[slot], 64, qrow);
          if (it.type == kP2) bulk_load(d.ust, a.ustat + (size_t)it.u * a.ustat_stride, ust_bytes, &s.qfull[slot]);
          ok = wait_bar(&s.qfull[slot], qphase, a, 16u);
        }
        ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
        if (!ok) break;
        if (it.type == kP2) build_stat_rows(s.qbuf[slot], a, d.ust, lane);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_full[slot]);
      ++seq;
      if (it.type == kExit) {
        // no work left for this CTA: the next launch (finalisation) may be
        // scheduled on SMs as they drain; it waits for this grid's completion
        // before reading anything
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        break;
      }
      for (int t = 0; t < ntiles && ok; ++t) {
        if (lane == 0) {
          ok = wait_bar(&s.empty[stage], sphase ^ 1u, a, 4u);
          if (ok) {
            mbar_expect_tx(&s.full[stage], kTileBytes);
            const int y = i0 + t * kTile;
            // with pass 2 close behind pass 1 (a short lag), pass 1 keeps its
            // keys in L2 for it; with all of pass 1 first no key survives in L2
            // until its pass 2, and keeping them only crowds out the data the
            // finalisation reads next, so every load is evict-first
            const uint64_t pol = (it.type == kP1 && a.lag_p2 < a.U) ? pol_keep : pol_drop;
            tma_load_3d_hint(s.ktile[stage], &tmK, &s.full[stage], 0, y, it.u, pol);
            tma_load_3d_hint(s.ktile[stage] + kTileBytes / 2, &tmK, &s.full[stage], 64, y, it.u, pol);
            used_bits |= 1u << stage;
            par_bits ^= 1u << stage;
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
        if (++stage == kStages) {
          stage = 0;
          sphase ^= 1u;
        }
      }
    }
    if (!ok && lane == 0) {
      // let this CTA's copies in flight land before its shared memory goes away
      for (int st = 0; st < kStages; ++st)
        if (used_bits & (1u << st)) {
          const uint32_t last = ((par_bits >> st) & 1u) ^ 1u;  // parity of the last load's phase
          const long long t0 = clock64();
          while (!mbar_try_wait(&s.full[st], last) && clock64() - t0 < a.timeout_cycles) {
          }
        }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t sphase = 0, tcount = 0;
      const uint32_t idesc_l = idesc_bf16(128, a.NP, false, false);
      for (int seq = 0; ok; ++seq) {
        const int slot = seq % kIQ;
        const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
        if (!(ok = wait_bar(&s.item_full[slot], qphase, a, 5u))) break;
        const ItemDesc& d = s.desc[slot];
        const int type = d.type, ntiles = d.ntiles;
        if (type == kExit) break;
        if (!(ok = wait_bar(&s.qfull[slot], qphase, a, 17u))) break;  // queries landed (already observed by warp 0)
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
        const long long t0 = clock64();
        while (!mbar_try_wait(&s.drain, 0u) && clock64() - t0 < a.timeout_cycles) {
        }
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
        const long long t0 = clock64();
        while (!mbar_try_wait(&s.drain2, 0u) && clock64() - t0 < a.timeout_cycles) {
        }
      }
    }
  } else if (warp == 2) {
    // ------------------------------------------------ stats warp
    // Counts finished pass-1 items per unit (gpu-scope atomic); the item that
    // completes a unit folds its chunk partials into the unit statistics and
    // releases pass 2 of the unit.  Runs beside the epilogue so that neither
    // the count's round trip nor the fold holds up the tiles.
    uint32_t p1par = 0u;  // per slot: parity of the next p1done phase
    for (int seq = 0; ok; ++seq) {
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.item_full[slot], qphase, a, 26u)))) break;
      const ItemDesc& d = s.desc[slot];
      const int type = d.type, u = d.u;
      if (type == kExit) break;
      if (type == kP1) {
        // the epilogue's partials and the key warps' norms of the item are written
        if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.p1done[slot], (p1par >> slot) & 1u, a, 27u)))) break;
        p1par ^= 1u << slot;
        if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.kpub[slot], qphase, a, 19u)))) break;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_empty[slot]);  // free the slot before the long part
      if (type == kP1) {
        // the arrival is a gpu-scope release of everything this CTA wrote for
        // the item (the mbarrier waits above ordered it before this thread)
        unsigned old = 0u;
        if (lane == 0) old = atom_add_acq_rel(a.sync + 4 + u, 1u);
        old = __shfl_sync(0xffffffffu, old, 0);
        if (old == (unsigned)(a.nchunks - 1)) {
          unit_reduce_warp(a, u, lane);
          __syncwarp();
          if (lane == 0) st_release(a.sync + 4 + a.U + u, 1u);
        }
      }
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
        const int i = i0 + t * kTile + kk;
        const bool valid = i < a.N;
        if (type == kP1) {
          // squared norm of this thread's key (packed fp32 pairs), kept for
          // pass 2, and the sum weights w = 1/||k|| in three bf16 terms
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
          if (valid) __stcs(a.norm2 + (size_t)u * a.N + i, n2);  // read once, by pass 2
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
          // pass 2: the keys are only needed by the MMA; the norms pass 1
          // stored go to the epilogue through shared memory
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.empty[stage]);
          const uint32_t nb = p2count % kNB, nph = (p2count / kNB) & 1u;
          ++p2count;
          const float n2 = valid ? __ldcs(a.norm2 + (size_t)u * a.N + i) : 0.f;
          if (!(ok = __all_sync(0xffffffffu, wait_bar(&s.nempty[nb], nph ^ 1u, a, 23u)))) break;
          s.nbuf[nb][kk] = n2;
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
        float* part = a.p1part + ((size_t)u * a.nchunks + d.chunk) * a.p1_stride;
        part[kk] = __uint_as_float(v[0]);
        part[kD + kk] = (__uint_as_float(v[1]) + __uint_as_float(v[2])) + __uint_as_float(v[3]);
      }
      // the item's key norms and sums are written: the stats warp's gpu-scope
      // arrival (after it has waited for kpub) publishes them
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
  tc_evict_kernel<RH><<<g_num_sms[dev].load(), kThreads, smem, st>>>(tm, tq, a);
  return cudaGetLastError();
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
