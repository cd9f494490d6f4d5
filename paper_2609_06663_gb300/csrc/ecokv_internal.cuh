// Internal declarations shared by the libecokv translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "ecokv.h"

namespace ecokv {

constexpr int kD = 128;          // supported head dimension
constexpr int kMaxRows = 256;    // max (h_q / h_kv) * window
constexpr int kChunk = 128;      // keys per chunk of the streaming passes
constexpr int kMaxN = 1 << 24;

// Device status word (first bytes of the workspace).
struct DevStatus {
  unsigned code;     // ecokv_status of the first device-side error (0 = none)
  unsigned detail;   // unit or item that raised it
};

// Byte offsets of the workspace regions for one parameter block.
struct Layout {
  int U;             // units = n_layers * h_kv
  int R;             // window rows per unit = (h_q / h_kv) * window
  int N, W, Tv;      // tokens, window, candidates
  int nchunks;       // ceil(N / kChunk)
  int p1_stride;     // floats per (unit, chunk) pass-1 partial: 2R + 2D
  int ustat_stride;  // floats per unit statistics record
  size_t status, cnt, p1part, ustat, p2part, simp, dE, cosv, sbuf, total;
};

Layout make_layout(const ecokv_params& p);

// unit statistics record (floats):  [0,D) kbar | [D,2D) mu | [2D] ||kbar||^2 |
//                                    [2D+1] ||mu||^2 | [2D+2, 2D+2+R) log2-LSE of the window rows
__host__ __device__ inline int ustat_kbar() { return 0; }
__host__ __device__ inline int ustat_mu() { return kD; }
__host__ __device__ inline int ustat_ksq() { return 2 * kD; }
__host__ __device__ inline int ustat_musq() { return 2 * kD + 1; }
__host__ __device__ inline int ustat_lse() { return 2 * kD + 2; }

struct ScoreArgs {
  const void* K;
  const void* Q;
  int N, W, g, R, h_kv, h_q, Tv, nchunks, p1_stride, ustat_stride;
  float scale_log2;  // log2(e) / sqrt(d): logits are kept in log2 units
  float* p1part;
  float* ustat;
  unsigned* cnt;
  float* p2part;
  float* simp;
  float* dE;
  float* cosv;
};

struct FinalArgs {
  int N, W, Tv, nchunks, budget, pool, ustat_stride;
  float alpha, beta, tau, eps, lambda_override;
  unsigned flags;
  int n_keep;
  const float* p2part;
  const float* ustat;
  const float* simp;
  const float* dE;
  const float* cosv;
  float* S;          // [U][Tv] scores (output of finalize, input of select)
  float* lambda;     // [U] or null
  float* dbg;        // [U][5][Tv] or null
  int32_t* idx;      // [U][n_keep] or null
};

struct CompactArgs {
  const void* K;
  const void* V;
  const int32_t* idx;
  void* K_out;
  void* V_out;
  int N, n_keep;
  unsigned* status;  // may be null
};

// launchers (return cudaGetLastError() after the launch)
cudaError_t launch_score_simt(const ScoreArgs& a, ecokv_dtype dt, int U, cudaStream_t s);
cudaError_t launch_finalize(const FinalArgs& a, int U, bool do_score, bool do_select, cudaStream_t s);
cudaError_t launch_compact(const CompactArgs& a, ecokv_dtype dt, int U, cudaStream_t s);

}  // namespace ecokv
