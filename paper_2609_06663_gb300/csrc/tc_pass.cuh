// Launch interface of the persistent tensor-core kernel (tc_pass.cu).
#pragma once

#include "ecokv_internal.cuh"

namespace ecokv {

constexpr int kTcMaxSms = 256;                 // largest grid the record slots are sized for

struct TcArgs {
  int U, N, W, R, R4, NP, g, h_kv, h_q, Tv;  // R, R4: rows of this launch's row group
  int row0;                         // the group's first window row among the unit's (h_q / h_kv) * W
  int kbar_n;                       // keys 0 .. kbar_n - 1 form the centroid (N, or Tv for the non-window centroid)
  int q_rows;                       // rows of the window-query tensor: n_layers * h_q * W
  int T;                            // tiles of 128 keys per unit: ceil(N / 128)
  int uw, nw;                       // units per wave, waves: ceil(U / uw)
  int lag;                          // waves between a wave's pass 1 and its pass 2 (1 .. nw)
  int P;                            // CTAs of the grid: slices per wave (fewer when a wave has fewer tiles)
  int rmax;                         // record slots per unit (at least the slices any unit meets)
  int p1_stride, ustat_stride;
  int stall_unit;                   // fault injection: this unit's statistics never complete (-1: none)
  float scale_log2;
  unsigned long long timeout_ns;    // limit of every bounded wait (global timer)
  const void* Q;
  const void* K;                    // keys, for the direct distance fallback
  float* p1part;                    // [U][rmax][p1_stride]
  float* ustat;                     // [U][ustat_stride]
  float* p2part;                    // [U][rmax][kP2Stride]
  float* simp;
  float* dE;
  float* cosv;
  unsigned* sync;                   // [0] unused, [1] abort, [4+u] pass-1 arrivals, [4+U+u] statistics ready
  unsigned* status;
};

// Half the MMA N extent (window rows, padded to a multiple of four, plus the
// mu rows, rounded up to a power of two) for R window rows; 0 when R is too
// large for this kernel.
int tc_rows_half(int R);
// Record slots per unit for T tiles per unit and waves of at least Lmin tiles:
// the most slices (of at least floor(Lmin / P) tiles each, P <= kTcMaxSms) a
// unit can meet.
int tc_record_slots(int T, int Lmin);
size_t tc_smem_bytes();
cudaError_t launch_tc(const void* K, const TcArgs& args, cudaStream_t st);

}  // namespace ecokv
