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
constexpr int kP2Stride = 8;     // floats per (unit, chunk) pass-2 partial, see P2_* below
constexpr int kSmemScores = 48 * 1024;  // candidates whose scores the finaliser keeps in shared memory

// pass-2 partial record of one (unit, chunk)
enum : int {
  P2_SUM_DE_ALL = 0,  // sum of d_E over the chunk's keys i < N (Eq. 4 uses all T keys)
  P2_MIN_DE = 1,      // min of d_E over candidates i < N - W (+inf if none)
  P2_MAX_DE = 2,      // max of d_E over candidates (-inf if none)
  P2_SUM_DE = 3,      // sum of d_E over candidates
  P2_SUM_COS = 4,     // sum of khat . mu over candidates
  P2_SUM_RAW = 5      // sum of the raw importance vote over candidates
};
static_assert(P2_SUM_DE_ALL == 0 && P2_MIN_DE == 1 && P2_MAX_DE == 2 && P2_SUM_DE == 3 && P2_SUM_COS == 4 &&
                  P2_SUM_RAW == 5,
              "the pass-2 reductions write the record in this order");

// Device status word (first bytes of the workspace).
struct DevStatus {
  unsigned code;     // ecokv_status of the first device-side error (0 = none)
  unsigned detail;   // unit or item that raised it
};

// Byte offsets of the workspace regions for one parameter block and a number
// of partial-record slots per unit (chunks of kChunk keys on the CUDA-core
// path, the slices a unit meets on the tensor-core path).
struct Layout {
  int U;             // units = n_layers * h_kv
  int R;             // window rows per unit = (h_q / h_kv) * window
  int N, W, Tv;      // tokens, window, candidates
  int nchunks;       // record slots per unit: streaming chunks (CUDA-core passes) or slices met
                     // (tensor-core passes)
  int p1_stride;     // floats per (unit, chunk) pass-1 partial: 2R + 2D
  int ustat_stride;  // floats per unit statistics record
  size_t status, sync, p1part, ustat, p2part, simp, dE, cosv, sbuf, norm2;
  size_t chosen, src;  // layer-wide budget: chosen positions, gathered rows (U * min(B, N) int32 each)
  size_t lsel;         // layer-wide budget: the layer select's histograms, state and block counts
  size_t vnorm;        // value-norm importance: ||v_i|| of the candidates, U * Tv floats
  size_t wins;         // winsorised min-max: the order statistics' selection state and histograms
  size_t total;
  size_t sync_bytes; // bytes of the per-call counters cleared before each call
};

Layout make_layout(const ecokv_params& p, int nrec);

// unit statistics record (floats):  [0,D) kbar | [D,2D) mu | [2D] ||kbar||^2 |
//                                    [2D+1] ||mu||^2 | [2D+2, 2D+2+R) log2-LSE of the window rows
__host__ __device__ inline int ustat_kbar() { return 0; }
__host__ __device__ inline int ustat_mu() { return kD; }
__host__ __device__ inline int ustat_ksq() { return 2 * kD; }
__host__ __device__ inline int ustat_musq() { return 2 * kD + 1; }
__host__ __device__ inline int ustat_lse() { return 2 * kD + 4; }  // 16-byte aligned

struct ScoreArgs {
  const void* K;
  const void* Q;
  int N, W, g, R, h_kv, h_q, Tv, nchunks, p1_stride, ustat_stride;
  int kbar_n;        // keys 0 .. kbar_n - 1 form the centroid (N, or Tv for the non-window centroid)
  float scale_log2;  // log2(e) / sqrt(d): logits are kept in log2 units
  float* p1part;
  float* ustat;
  unsigned* cnt;     // per-unit pass-1 arrival counters
  float* p2part;
  float* simp;
  float* dE;
  float* cosv;
};

constexpr int kMaxLayerBudgets = 256;  // layers a per-layer budget schedule may have

struct FinalArgs {
  int N, W, Tv, nchunks, budget, pool, ustat_stride;
  float alpha, beta, tau, eps, lambda_override;
  unsigned flags;
  int n_keep;
  const float* p2part;  // [U][nchunks][kP2Stride]: nchunks counts every pass-2 partial slot
  const float* ustat;
  const float* simp;
  const float* dE;
  const float* cosv;
  float* S;          // [U][Tv] scores out, or null
  float* S_scratch;  // [U][Tv] workspace scores, used when S is null and Tv > kSmemScores
  float* lambda;     // [U] or null
  float* dbg;        // [U][5][Tv] or null
  int32_t* idx;      // [U][n_keep] or null
  const float* vnorm;  // [U][Tv] ||v_i|| multiplying the pooled vote (value-norm importance), or null
  // winsorised min-max: per unit the order-preserving keys of the clip
  // bounds of d_E, at wlo[4 u] and whi[4 u]; null for the plain min-max
  const unsigned* wlo;
  const unsigned* whi;
  // MAD scaling: the order-preserving keys of the two middle order
  // statistics of d_E at mad[4 u] and mad[4 (n_units + u)] (their mean is
  // the median), and of |d_E - median| at mad[4 (2 n_units + u)] and
  // mad[4 (3 n_units + u)] (their mean is the MAD); null otherwise
  const unsigned* mad;
  int n_units;
  // per-layer budgets (PyramidKV schedule): with n_lb > 0 the heads of layer
  // l keep lb[l] rows (window included) in slots of stride n_keep
  int h_kv, n_lb;
  int lb[kMaxLayerBudgets];
};

// The budget of unit u (layer u / h_kv).
__host__ __device__ inline int unit_budget(const FinalArgs& f, int u) { return f.n_lb ? f.lb[u / f.h_kv] : f.budget; }

struct CompactArgs {
  const void* K;
  const void* V;
  const int32_t* idx;
  void* K_out;
  void* V_out;
  int N, n_keep;
  unsigned* status;  // may be null
  // per-layer budgets: unit u copies keep[u / h_kv] rows (of stride n_keep)
  int h_kv, n_lb;
  int keep[kMaxLayerBudgets];
};

// Layer-wide budget (AdaKV): the split of each layer's chosen positions into
// per-head lists (kept candidates ascending, then the window), their offsets,
// and the rows of the layer's [h_kv * N] block the gather reads.
struct AdaptArgs {
  const int32_t* chosen;  // [L][k_layer] ascending positions in the layer's concatenated scores
  int32_t* idx;           // [L][h_kv * n_keep]
  int32_t* head_off;      // [L][h_kv + 1]
  int32_t* src;           // [L][h_kv * n_keep]
  int h_kv, N, W, Tv, n_keep, k_layer;
  int keep_all;           // B >= N: every row of every head
};

// launchers (return cudaGetLastError() after the launch)
cudaError_t launch_score_simt(const ScoreArgs& a, ecokv_dtype dt, int U, cudaStream_t s);
// finalize (scores), then optionally select and gather, one CTA per unit
cudaError_t launch_finalize(const FinalArgs& f, int U, bool do_select, cudaStream_t s);
// select only, on caller scores f.S
cudaError_t launch_select(const FinalArgs& f, int U, cudaStream_t s);
cudaError_t launch_compact(const CompactArgs& a, ecokv_dtype dt, int U, cudaStream_t s);
cudaError_t launch_adaptive_split(const AdaptArgs& a, int n_layers, cudaStream_t s);
// ||v_i|| of the Tv candidate rows of every unit: vn[u][i]
cudaError_t launch_value_norms(const void* V, ecokv_dtype dt, int U, int N, int Tv, float* vn, cudaStream_t s);
// Whether the cluster finalize takes units of Tv candidates (else one CTA per unit).
bool cluster_finalize_fits(int Tv);
// k largest of each layer's T scores, ascending positions (layer_select.cu)
size_t layer_select_scratch_bytes(int n_layers, int T);
// the order-preserving keys of the ka-th and kb-th largest of each row's
// T <= 32768 values at out[4 row] and out[4 (rows + row)]; with mad also
// those of |x - m| (m the mean of the first two) at out[4 (2 rows + row)]
// and out[4 (3 rows + row)] (order_stats.cu)
cudaError_t launch_order_stats(const float* x, int rows, int T, int ka, int kb, bool mad, unsigned* out,
                               cudaStream_t s);
cudaError_t launch_layer_select(const float* S, int n_layers, int T, int k, int32_t* chosen, void* scratch,
                                cudaStream_t s);
// One thread-block cluster per unit: scores, and the top-k when f.idx is set
// (select_only: the top-k of the given scores f.S); cudaErrorNotSupported
// when the unit is too long for one cluster.
cudaError_t launch_finalize_cluster(const FinalArgs& f, int U, bool select_only, cudaStream_t s);

}  // namespace ecokv
