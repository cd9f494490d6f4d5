// Persistent tensor-core kernel for bf16 inputs: the whole eviction pass in
// one launch on sm_103a.
//
// Work is a global, ticket-ordered list of items:
//   P1(u, c)  pass 1 over chunk c (up to 8 tiles of 128 keys) of unit u
//             (u = (layer, KV head)): window logits (tcgen05 MMA, keys as M,
//             window rows as N), per-row online-softmax partials, key norms,
//             and the chunk sums of k and k/||k|| (a second tcgen05 MMA with the
//             key tile as an MN-major operand against [1, w_hi, w_mid, w_lo]
//             weight rows, w = 1/||k|| split into three bf16 terms).  The last P1 item of a unit folds the partials into the unit
//             statistics (kbar, mu, per-row log2-sum-exp).
//   P2(u, c)  pass 2: logits again plus two extra MMA columns holding k . mu
//             (bf16 hi + lo split of mu), giving the importance vote and the
//             cosine khat . mu; d_E = ||k - kbar|| (Eq. 1) is taken directly
//             from the staged key tile in fp32 (the expansion of Sec. 4 cancels
//             badly when keys sit close to their centroid).
// Within a schedule step s the list holds P1(s, *) then P2(s - lag_p2, *), so
// pass 2 of a unit re-reads its keys a few units after pass 1 (from L2, not
// HBM), and every item depends only on items with smaller tickets: dispatch is
// deadlock-free without co-residency.  Pass 2 leaves per-candidate arrays and
// per-chunk partial sums; finalisation, selection and the gather of the kept
// rows run in the next launch (finalize_select.cu).
//
// Warp roles (320 threads, one CTA per SM): warp 0 takes tickets, resolves
// dependencies (bounded spins on gpu-scope flags), builds the MMA B operand
// (window queries, plus the kbar / mu rows for pass 2) and issues TMA loads of
// 32 KB key tiles into a 4-stage ring; warp 1 issues tcgen05 MMAs into a
// double-buffered TMEM accumulator; warps 2-9 are the epilogue (one key per
// TMEM lane, window rows split in two halves).  Every mbarrier wait and spin
// is bounded: on timeout the kernel records ECOKV_ERR_TIMEOUT, raises a
// gpu-wide abort flag, drains its own copies and MMAs, frees TMEM and exits.

#include <cuda.h>

#include "finalize_select.cuh"
#include "ptx.cuh"
#include "tc_pass.cuh"

namespace ecokv {
namespace {

using namespace ptx;

constexpr int kStages = 4;
constexpr int kIQ = 2;
constexpr int kTile = 128;
constexpr int kThreads = 320;
constexpr int kEpi = 256;
constexpr int kNPMax = 128;
constexpr uint32_t kTileBytes = kTile * kD * 2;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSigmaCol = 256;
constexpr uint32_t kEpiBar = 1;

enum : int { kP1 = 0, kP2 = 1, kExit = 3 };

struct ItemDesc {
  int type, u, chunk, part, i0, ntiles;
  float lse[kNPMax];
  float kbar[kD];
};

struct __align__(1024) Smem {
  uint8_t ktile[kStages][kTileBytes];   // 2 boxes [128 keys x 64 d], 128-byte swizzle
  uint8_t qbuf[kIQ][kNPMax * 256];      // B operand, 2 boxes [NP rows x 64 d]
  uint8_t wbuf[kStages][4096];          // sum weights: 2 boxes [16 rows x 64 keys]; rows 1, w_hi, w_mid, w_lo
  ItemDesc desc[kIQ];
  float xch[2][2][kTile];               // [tile parity][row half][key]
  float xd2[2][2][kTile];               // squared distance to kbar, per half
  float xn2[2][2][kTile];               // squared key norm, per half
  float red[8][64][2];                  // [epilogue warp][row][max, sum]
  float shf[64];
  uint64_t full[kStages], empty[kStages], wready[kStages];
  uint64_t item_full[kIQ], item_empty[kIQ];
  uint64_t tmem_full[2], tmem_empty[2];
  uint64_t sigma_full, sigma_empty, drain;
  uint32_t tmem_base;
  int flag_last;
};

static_assert(sizeof(Smem) + 1024 <= 232448, "shared-memory plan exceeds the 227 KB per-CTA limit");

struct EpiSync {
  __device__ __forceinline__ static void sync() { named_bar_sync(kEpiBar, kEpi); }
};

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

// Bounded spin on a gpu-scope flag written by another CTA.
__device__ bool wait_flag(const unsigned* f, const TcArgs& a, unsigned where) {
  const long long t0 = clock64();
  while (ld_acquire(f) == 0u) {
    if (aborted(a)) return false;
    if (clock64() - t0 > a.timeout_cycles) {
      raise_abort(a, ECOKV_ERR_TIMEOUT, where);
      return false;
    }
    __nanosleep(256);
  }
  return true;
}

struct Item {
  int type, u, chunk, part;
  bool valid;
};

__device__ Item decode(int ticket, const TcArgs& a) {
  Item it{kExit, 0, 0, 0, true};
  if (ticket >= a.total_tickets) return it;
  const int s = ticket / a.step_items, slot = ticket % a.step_items;
  if (slot < a.nchunks) {
    it.type = kP1;
    it.u = s;
    it.chunk = slot;
  } else {
    it.type = kP2;
    it.u = s - a.lag_p2;
    it.chunk = slot - a.nchunks;
  }
  it.valid = it.u >= 0 && it.u < a.U;
  return it;
}

__device__ __forceinline__ uint32_t sw128(int row, int chunk16) {
  return (uint32_t)(row * 128 + ((chunk16 ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// B operand of one item in the 128-byte-swizzled K-major layout: rows 0..R-1
// are the group's window queries; for pass 2, rows R4 and R4+1 hold mu_hi and
// mu_lo; every other row is zero.  Run by the 32 lanes of warp 0.
__device__ void build_qbuf(uint8_t* qb, const TcArgs& a, const Item& it, int lane) {
  const int layer = it.u / a.h_kv, head = it.u % a.h_kv;
  const uint4* Qu = reinterpret_cast<const uint4*>(a.Q) + ((size_t)layer * a.h_q + (size_t)head * a.g) * a.W * 16;
  const float* us = a.ustat + (size_t)it.u * a.ustat_stride;
  for (int e = lane; e < a.NP * 16; e += 32) {
    const int r = e >> 4, j = e & 15;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (r < a.R) {
      val = __ldg(Qu + (size_t)r * 16 + j);
    } else if (it.type == kP2 && r >= a.R4 && r < a.R4 + 2) {
      const int which = r - a.R4;
      const float* src = us + ustat_mu() + j * 8;
      float x[8], o[8];
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        x[t] = __ldcg(src + t);
        const float hi = __bfloat162float(__float2bfloat16_rn(x[t]));
        o[t] = (which & 1) ? (x[t] - hi) : hi;
      }
      val = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]), pack_bf16x2(o[4], o[5]),
                       pack_bf16x2(o[6], o[7]));
    }
    *reinterpret_cast<uint4*>(qb + (j >> 3) * (a.NP * 128) + sw128(r, j & 7)) = val;
  }
}

__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Fold every chunk's pass-1 partials of unit u into its statistics record.
__device__ void unit_reduce(const TcArgs& a, int u, Smem& s, int tid) {
  __threadfence();
  const float* base = a.p1part + (size_t)u * a.nchunks * a.p1_stride;
  float* us = a.ustat + (size_t)u * a.ustat_stride;
  float kb = 0.f, mu = 0.f;
  if (tid < kD) {
    float sk = 0.f, skh = 0.f;
    for (int c = 0; c < a.nchunks; ++c) {
      sk += __ldcg(base + (size_t)c * a.p1_stride + 2 * a.R + tid);
      skh += __ldcg(base + (size_t)c * a.p1_stride + 2 * a.R + kD + tid);
    }
    const float inv_n = 1.f / (float)a.N;
    kb = sk * inv_n;
    mu = skh * inv_n;
    us[ustat_kbar() + tid] = kb;
    us[ustat_mu() + tid] = mu;
  }
  for (int row = tid; row < a.R; row += kEpi) {
    float M = -INFINITY;
    for (int c = 0; c < a.nchunks; ++c) M = fmaxf(M, __ldcg(base + (size_t)c * a.p1_stride + row));
    float Z = 0.f;
    for (int c = 0; c < a.nchunks; ++c) {
      const float m = __ldcg(base + (size_t)c * a.p1_stride + row);
      if (m != -INFINITY) Z += __ldcg(base + (size_t)c * a.p1_stride + a.R + row) * exp2f(m - M);
    }
    us[ustat_lse() + row] = M + log2f(Z);
  }
  const float ksq = group_reduce<Op::Sum, EpiSync>(kb * kb, s.shf, tid, kEpi);
  const float msq = group_reduce<Op::Sum, EpiSync>(mu * mu, s.shf, tid, kEpi);
  if (tid == 0) {
    us[ustat_ksq()] = ksq;
    us[ustat_musq()] = msq;
  }
}

template <int RH>
__global__ void __launch_bounds__(kThreads, 1) tc_evict_kernel(const __grid_constant__ CUtensorMap tmK, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  Smem& s = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 9);
      mbar_init(&s.wready[i], 8);
    }
    for (int i = 0; i < kIQ; ++i) {
      mbar_init(&s.item_full[i], 1);
      mbar_init(&s.item_empty[i], 2);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.tmem_full[i], 1);
      mbar_init(&s.tmem_empty[i], 8);
    }
    mbar_init(&s.sigma_full, 1);
    mbar_init(&s.sigma_empty, 4);
    mbar_init(&s.drain, 1);
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
  if (warp == 0 && lane == 0) tma_prefetch_desc(&tmK);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  bool ok = true;

  if (warp == 0) {
    // ------------------------------------------------ scheduler + TMA producer
    int stage = 0;
    uint32_t sphase = 0;
    uint32_t used_bits = 0u, par_bits = 0u;  // per stage: loaded at least once / parity of loads
    for (int seq = 0; ok;) {
      int ticket = 0;
      if (lane == 0) ticket = atomicAdd(a.sync, 1u);
      ticket = __shfl_sync(0xffffffffu, ticket, 0);
      const Item it = decode(ticket, a);
      if (!it.valid) continue;
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      if (lane == 0) {
        ok = wait_bar(&s.item_empty[slot], qphase ^ 1u, a, 1u);
        if (ok && it.type == kP2) ok = wait_flag(a.sync + 4 + a.U + it.u, a, 2u);
      }
      ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
      if (!ok) break;
      ItemDesc& d = s.desc[slot];
      const int i0 = it.chunk * a.tiles_per_chunk * kTile;
      const int ntiles = it.type == kExit ? 0 : min(a.tiles_per_chunk, (a.N - i0 + kTile - 1) / kTile);
      if (lane == 0) {
        d.type = it.type;
        d.u = it.u;
        d.chunk = it.chunk;
        d.part = it.part;
        d.i0 = i0;
        d.ntiles = ntiles;
      }
      if (it.type == kP1 || it.type == kP2) {
        build_qbuf(s.qbuf[slot], a, it, lane);
        if (it.type == kP2) {
          const float* us = a.ustat + (size_t)it.u * a.ustat_stride;
          for (int r = lane; r < a.R; r += 32) d.lse[r] = __ldcg(us + ustat_lse() + r);
          for (int c = lane; c < kD; c += 32) d.kbar[c] = __ldcg(us + ustat_kbar() + c);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_full[slot]);
      ++seq;
      if (it.type == kExit) break;
      for (int t = 0; t < ntiles && ok; ++t) {
        if (lane == 0) {
          ok = wait_bar(&s.empty[stage], sphase ^ 1u, a, 4u);
          if (ok) {
            mbar_expect_tx(&s.full[stage], kTileBytes);
            const int y = i0 + t * kTile;
            tma_load_3d(s.ktile[stage], &tmK, &s.full[stage], 0, y, it.u);
            tma_load_3d(s.ktile[stage] + kTileBytes / 2, &tmK, &s.full[stage], 64, y, it.u);
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
      uint32_t sphase = 0, tcount = 0, sigcount = 0;
      uint32_t wpar = 0u;  // per stage: parity of the next wready phase (pass-1 tiles only)
      const uint32_t idesc_l = idesc_bf16(128, a.NP, false, false);
      const uint32_t idesc_s = idesc_bf16(128, 16, true, false);
      for (int seq = 0; ok; ++seq) {
        const int slot = seq % kIQ;
        const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
        if (!(ok = wait_bar(&s.item_full[slot], qphase, a, 5u))) break;
        const ItemDesc& d = s.desc[slot];
        const int type = d.type, ntiles = d.ntiles;
        if (type == kExit) break;
        const uint32_t qb = smem_u32(s.qbuf[slot]);
        for (int t = 0; t < ntiles; ++t) {
          const uint32_t b = tcount & 1u, tph = (tcount >> 1) & 1u;
          if (!(ok = wait_bar(&s.full[stage], sphase, a, 6u))) break;
          if (!(ok = wait_bar(&s.tmem_empty[b], tph ^ 1u, a, 7u))) break;
          tc_fence_after();
          const uint32_t kt = smem_u32(s.ktile[stage]);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t ad = smem_desc(kt + (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32, 16, 1024, 2);
            const uint64_t bd = smem_desc(qb + (kk >> 2) * (a.NP * 128) + (kk & 3) * 32, 16, 1024, 2);
            mma_bf16(tmem + b * 128u, ad, bd, idesc_l, kk > 0 ? 1u : 0u);
          }
          mma_commit(&s.tmem_full[b]);
          if (type == kP1) {
            if (!(ok = wait_bar(&s.wready[stage], (wpar >> stage) & 1u, a, 8u))) break;
            wpar ^= 1u << stage;
            if (t == 0 && !(ok = wait_bar(&s.sigma_empty, (sigcount & 1u) ^ 1u, a, 9u))) break;
            tc_fence_after();
            const uint32_t wb = smem_u32(s.wbuf[stage]);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              // A = key tile viewed MN-major (d contiguous): 16 keys per step
              const uint64_t ad = smem_desc(kt + kk * 2048, kTileBytes / 2, 1024, 2);
              const uint64_t bd = smem_desc(wb + (kk >> 2) * 2048 + (kk & 3) * 32, 16, 1024, 2);
              mma_bf16(tmem + kSigmaCol, ad, bd, idesc_s, (t > 0 || kk > 0) ? 1u : 0u);
            }
          }
          mma_commit(&s.empty[stage]);
          if (type == kP1 && t == ntiles - 1) {
            mma_commit(&s.sigma_full);
            ++sigcount;
          }
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
  } else {
    // ------------------------------------------------ epilogue (warps 2..9)
    const int e = warp - 2, q = warp & 3, h = e >> 2;
    const int kk = 32 * q + lane;  // key row within a tile = TMEM lane
    const int tid = threadIdx.x - 64;
    const uint32_t tl = tmem + ((uint32_t)(32 * q) << 16);
    int stage = 0;
    uint32_t sphase = 0, tcount = 0, sigcount = 0;
    for (int seq = 0; ok; ++seq) {
      const int slot = seq % kIQ;
      const uint32_t qphase = (uint32_t)(seq / kIQ) & 1u;
      if (!(ok = wait_bar(&s.item_full[slot], qphase, a, 10u))) break;
      const ItemDesc& d = s.desc[slot];
      const int type = d.type;
      if (type == kExit) break;
      const int u = d.u, chunk = d.chunk, i0 = d.i0, ntiles = d.ntiles;

      if (type == kP1) {
        float m[RH], z[RH];
#pragma unroll
        for (int c = 0; c < RH; ++c) {
          m[c] = -INFINITY;
          z[c] = 0.f;
        }
        for (int t = 0; t < ntiles && ok; ++t) {
          const int it0 = i0 + t * kTile;
          const int i = it0 + kk;
          const bool valid = i < a.N;
          // key norm: this half of the row, exchanged with the other half
          if (!(ok = wait_bar(&s.full[stage], sphase, a, 11u))) break;
          const uint8_t* row = s.ktile[stage] + h * (kTileBytes / 2) + kk * 128;
          float n2h = 0.f;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 v = *reinterpret_cast<const uint4*>(row + ((c ^ (kk & 7)) << 4));
            const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
            float p = 0.f;
#pragma unroll
            for (int t2 = 0; t2 < 4; ++t2) {
              const float lo = __uint_as_float(w4[t2] << 16), hi = __uint_as_float(w4[t2] & 0xffff0000u);
              p = fmaf(lo, lo, p);
              p = fmaf(hi, hi, p);
            }
            n2h += p;
          }
          s.xch[t & 1][h][kk] = n2h;
          named_bar_sync(kEpiBar, kEpi);
          const float n2 = s.xch[t & 1][0][kk] + s.xch[t & 1][1][kk];
          const float w = valid ? 1.f / fmaxf(sqrtf(n2), 1e-12f) : 0.f;
          {
            // w = w_hi + w_mid + w_lo in bf16 (about 24 significant bits)
            const __nv_bfloat16 whi = __float2bfloat16_rn(w);
            const float r1 = w - __bfloat162float(whi);
            const __nv_bfloat16 wmid = __float2bfloat16_rn(r1);
            const __nv_bfloat16 wlo = __float2bfloat16_rn(r1 - __bfloat162float(wmid));
            uint8_t* base = s.wbuf[stage] + (kk >> 6) * 2048 + (kk & 7) * 2;
            const int j = (kk & 63) >> 3;
            if (h == 0) {
              *reinterpret_cast<__nv_bfloat16*>(base + sw128(1, j)) = whi;
            } else {
              *reinterpret_cast<__nv_bfloat16*>(base + sw128(2, j)) = wmid;
              *reinterpret_cast<__nv_bfloat16*>(base + sw128(3, j)) = wlo;
            }
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&s.wready[stage]);
            mbar_arrive(&s.empty[stage]);  // done reading the key tile
          }

          // window logits of this key
          const uint32_t b = tcount & 1u, tph = (tcount >> 1) & 1u;
          if (!(ok = wait_bar(&s.tmem_full[b], tph, a, 12u))) break;
          tc_fence_after();
          uint32_t r[RH];
          tmem_ld<RH>(tl + b * 128u + (uint32_t)(h * RH), r);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.tmem_empty[b]);
          const bool all_vis = it0 + kTile - 1 <= a.N - a.W;
#pragma unroll
          for (int c = 0; c < RH; ++c) {
            const int rowi = h * RH + c;
            if (rowi < a.R) {
              const bool vis = all_vis || (valid && i <= a.N - a.W + (rowi % a.W));
              if (vis) {
                const float x = __uint_as_float(r[c]) * a.scale_log2;
                const float dlt = x - m[c];
                if (dlt > 20.f) {
                  z[c] = fmaf(z[c], exp2f(-dlt), 1.f);
                  m[c] = x;
                } else {
                  z[c] += exp2f(dlt);
                }
              }
            }
          }
          ++tcount;
          if (++stage == kStages) {
            stage = 0;
            sphase ^= 1u;
          }
        }
        if (!ok) break;
        // item end: per-row (max, sum) over the 32 keys of the warp
#pragma unroll
        for (int c = 0; c < RH; ++c) {
          const float M = warp_max_f(m[c]);
          const float zz = (m[c] == -INFINITY) ? 0.f : z[c] * exp2f(m[c] - M);
          const float Z = warp_sum_f(zz);
          if (lane == 0) {
            s.red[e][c][0] = M;
            s.red[e][c][1] = Z;
          }
        }
        named_bar_sync(kEpiBar, kEpi);
        float* part = a.p1part + ((size_t)u * a.nchunks + chunk) * a.p1_stride;
        if (tid < a.R) {
          const int hh = tid / RH, c = tid % RH;
          float M = -INFINITY;
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) M = fmaxf(M, s.red[4 * hh + w4][c][0]);
          float Z = 0.f;
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) {
            const float mm = s.red[4 * hh + w4][c][0];
            if (mm != -INFINITY) Z += s.red[4 * hh + w4][c][1] * exp2f(mm - M);
          }
          part[tid] = M;
          part[a.R + tid] = Z;
        }
        // chunk sums of k and k/||k|| from the weight MMA (TMEM lane = dimension)
        if (h == 0) {
          if (!(ok = wait_bar(&s.sigma_full, sigcount & 1u, a, 13u))) break;
          tc_fence_after();
          uint32_t v[4];
          tmem_ld_x4(tl + kSigmaCol, v);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.sigma_empty);
          part[2 * a.R + kk] = __uint_as_float(v[0]);
          part[2 * a.R + kD + kk] = (__uint_as_float(v[1]) + __uint_as_float(v[2])) + __uint_as_float(v[3]);
        }
        ++sigcount;
        __threadfence();  // this thread's partials and key norms before the arrival count
        named_bar_sync(kEpiBar, kEpi);
        if (tid == 0) {
          __threadfence();
          const unsigned old = atom_add_acq_rel(a.sync + 4 + u, 1u);
          s.flag_last = old == (unsigned)(a.nchunks - 1);
        }
        named_bar_sync(kEpiBar, kEpi);
        if (s.flag_last) {
          unit_reduce(a, u, s, tid);
          __threadfence();
          named_bar_sync(kEpiBar, kEpi);
          if (tid == 0) {
            __threadfence();
            st_release(a.sync + 4 + a.U + u, 1u);
          }
        }
      } else if (type == kP2) {
        float s_all = 0.f, mn = INFINITY, mx = -INFINITY, s_de = 0.f, s_c = 0.f, s_raw = 0.f;
        const float* kb = d.kbar + h * 64;
        for (int t = 0; t < ntiles && ok; ++t) {
          const int i = i0 + t * kTile + kk;
          const bool valid = i < a.N;
          // distance to the centroid and squared norm over this half's 64 dims
          if (!(ok = wait_bar(&s.full[stage], sphase, a, 15u))) break;
          const uint8_t* row = s.ktile[stage] + h * (kTileBytes / 2) + kk * 128;
          float d2h = 0.f, n2h = 0.f;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 v = *reinterpret_cast<const uint4*>(row + ((c ^ (kk & 7)) << 4));
            const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int t2 = 0; t2 < 4; ++t2) {
              const float lo = __uint_as_float(w4[t2] << 16), hi = __uint_as_float(w4[t2] & 0xffff0000u);
              const float dl = lo - kb[c * 8 + 2 * t2], dh = hi - kb[c * 8 + 2 * t2 + 1];
              d2h = fmaf(dl, dl, d2h);
              d2h = fmaf(dh, dh, d2h);
              n2h = fmaf(lo, lo, n2h);
              n2h = fmaf(hi, hi, n2h);
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.empty[stage]);  // done reading the key tile
          const uint32_t b = tcount & 1u, tph = (tcount >> 1) & 1u;
          if (!(ok = wait_bar(&s.tmem_full[b], tph, a, 14u))) break;
          tc_fence_after();
          uint32_t r[RH], st4[4];
          tmem_ld<RH>(tl + b * 128u + (uint32_t)(h * RH), r);
          if (h == 0) tmem_ld_x4(tl + b * 128u + (uint32_t)a.R4, st4);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.tmem_empty[b]);
          float vote = 0.f;
#pragma unroll
          for (int c = 0; c < RH; ++c) {
            const int rowi = h * RH + c;
            if (rowi < a.R) vote += exp2f(fmaf(__uint_as_float(r[c]), a.scale_log2, -d.lse[rowi]));
          }
          s.xch[t & 1][h][kk] = vote;
          s.xd2[t & 1][h][kk] = d2h;
          s.xn2[t & 1][h][kk] = n2h;
          named_bar_sync(kEpiBar, kEpi);
          if (h == 0 && valid) {
            const float v = s.xch[t & 1][0][kk] + s.xch[t & 1][1][kk];
            const float d2 = s.xd2[t & 1][0][kk] + s.xd2[t & 1][1][kk];
            const float n2 = s.xn2[t & 1][0][kk] + s.xn2[t & 1][1][kk];
            const float kmu = __uint_as_float(st4[0]) + __uint_as_float(st4[1]);
            const float dEv = sqrtf(d2);
            const float cs = kmu * (1.f / fmaxf(sqrtf(n2), 1e-12f));
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
          ++tcount;
          if (++stage == kStages) {
            stage = 0;
            sphase ^= 1u;
          }
        }
        if (!ok) break;
        s_all = group_reduce<Op::Sum, EpiSync>(s_all, s.shf, tid, kEpi);
        mn = group_reduce<Op::Min, EpiSync>(mn, s.shf, tid, kEpi);
        mx = group_reduce<Op::Max, EpiSync>(mx, s.shf, tid, kEpi);
        s_de = group_reduce<Op::Sum, EpiSync>(s_de, s.shf, tid, kEpi);
        s_c = group_reduce<Op::Sum, EpiSync>(s_c, s.shf, tid, kEpi);
        s_raw = group_reduce<Op::Sum, EpiSync>(s_raw, s.shf, tid, kEpi);
        if (tid == 0) {
          float* p = a.p2part + ((size_t)u * a.nchunks + chunk) * kP2Stride;
          p[P2_SUM_DE_ALL] = s_all;
          p[P2_MIN_DE] = mn;
          p[P2_MAX_DE] = mx;
          p[P2_SUM_DE] = s_de;
          p[P2_SUM_COS] = s_c;
          p[P2_SUM_RAW] = s_raw;
        }
      }
      named_bar_sync(kEpiBar, kEpi);
      if (tid == 0) mbar_arrive(&s.item_empty[slot]);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

int g_num_sms[64] = {0};
bool g_attr_set[64][4] = {};

template <int RH>
cudaError_t launch_rh(const CUtensorMap& tm, const TcArgs& a, int dev, cudaStream_t st) {
  const size_t smem = sizeof(Smem) + 1024;
  const int rh_i = RH == 8 ? 0 : RH == 16 ? 1 : RH == 32 ? 2 : 3;
  if (!g_attr_set[dev][rh_i]) {
    cudaError_t e = cudaFuncSetAttribute(tc_evict_kernel<RH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    g_attr_set[dev][rh_i] = true;
  }
  tc_evict_kernel<RH><<<g_num_sms[dev], kThreads, smem, st>>>(tm, a);
  return cudaGetLastError();
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

}  // namespace

size_t tc_smem_bytes() { return sizeof(Smem) + 1024; }

int tc_rows_half(int R) {
  const int r4 = (R + 3) & ~3;
  int np = 16;
  while (np < r4 + 4) np <<= 1;
  return np > kNPMax ? 0 : np / 2;
}

cudaError_t launch_tc(const void* K, const TcArgs& args, cudaStream_t st) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (g_num_sms[dev] == 0) {
    e = cudaDeviceGetAttribute(&g_num_sms[dev], cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
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
  switch (args.NP / 2) {
    case 8: return launch_rh<8>(tm, args, dev, st);
    case 16: return launch_rh<16>(tm, args, dev, st);
    case 32: return launch_rh<32>(tm, args, dev, st);
    case 64: return launch_rh<64>(tm, args, dev, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace ecokv
