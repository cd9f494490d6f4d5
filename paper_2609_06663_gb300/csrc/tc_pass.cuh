// Launch interface of the persistent tensor-core kernel (tc_pass.cu).
#pragma once

#include "ecokv_internal.cuh"

namespace ecokv {

constexpr int kTcMaxTiles = 64;                // largest item: 64 tiles of 128 keys
constexpr int kTcMinTiles = 2;                 // smallest item the workspace is sized for
constexpr int kTcChunk = 128 * kTcMinTiles;
constexpr int kTcP2Parts = 4;                  // parts a tail pass-2 item is split into (its partial slots)

struct TcArgs {
  int U, N, W, R, R4, NP, g, h_kv, h_q, Tv;
  int kbar_n;                       // keys 0 .. kbar_n - 1 form the centroid (N, or Tv for the non-window centroid)
  int q_rows;                       // rows of the window-query tensor: n_layers * h_q * W
  int tiles_per_chunk, nchunks;     // chunks of kTcChunk keys per unit
  int lag_p2;                       // schedule lag (in units) of pass 2 behind pass 1 (<= U)
  int split_from;                   // tickets from here on: pass-2 items split in nparts parts
  int nparts;                       // 1 .. kTcP2Parts
  int total_tickets;                // split_from + nparts * (2 * U * nchunks - split_from)
  int p1_stride, ustat_stride;
  float scale_log2;
  long long timeout_cycles;
  const void* Q;
  const void* K;                    // keys, for the direct distance fallback
  float* norm2;                     // [U][N] squared key norms written by pass 1
  float* p1part;
  float* ustat;
  float* p2part;                    // [U][nchunks][kTcP2Parts][kP2Stride]
  float* simp;
  float* dE;
  float* cosv;
  unsigned* sync;                   // [0] ticket, [1] abort, [4+u] pass-1 arrivals, [4+U+u] stats ready
  unsigned* status;
};

// Half the MMA N extent (window rows, padded to a multiple of four, plus the
// mu rows, rounded up to a power of two) for R window rows; 0 when R is too
// large for this kernel.
int tc_rows_half(int R);
size_t tc_smem_bytes();
cudaError_t launch_tc(const void* K, const TcArgs& args, cudaStream_t st);

}  // namespace ecokv
