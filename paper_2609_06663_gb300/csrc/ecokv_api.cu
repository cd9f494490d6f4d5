// C ABI of libecokv.so: argument checks, workspace layout, path choice and
// launches.  Every entry point validates on the host and returns before
// launching anything when an argument is wrong.
//
// Paths.  bf16 inputs with n >= 128 stream K through the persistent
// tensor-core kernel (tc_pass.cu, one launch for both passes, or one launch
// per group of at most 120 window rows when (h_q/h_kv)*W exceeds 120);
// fp32 inputs, other shapes and calls with ECOKV_FLAG_FORCE_SIMT use the
// CUDA-core passes (score_simt.cu, two launches).  Either way one more launch
// (finalize_select.cu) turns the pass-2 outputs into scores, selects and
// gathers the kept rows.

#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>

#include "ecokv_internal.cuh"
#include "tc_pass.cuh"

namespace ecokv {

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

Layout make_layout(const ecokv_params& p, int nrec) {
  Layout L{};
  L.U = p.n_layers * p.h_kv;
  L.R = (p.h_q / p.h_kv) * p.window;
  L.N = p.n;
  L.W = p.window;
  L.Tv = p.n - p.window;
  L.nchunks = nrec;
  L.p1_stride = 2 * ((L.R + 3) & ~3) + 2 * kD;
  L.ustat_stride = (ustat_lse() + L.R + 3) & ~3;
  const size_t U = (size_t)L.U;
  size_t off = 0;
  L.status = off;  off += 256;
  L.sync = off;    L.sync_bytes = (4 + 2 * U) * 4;  off += align256(L.sync_bytes);
  L.p1part = off;  off += align256(U * L.nchunks * L.p1_stride * 4);
  L.ustat = off;   off += align256(U * L.ustat_stride * 4);
  L.p2part = off;  off += align256(U * L.nchunks * kP2Stride * 4);
  L.simp = off;    off += align256(U * L.Tv * 4);
  L.dE = off;      off += align256(U * L.Tv * 4);
  L.cosv = off;    off += align256(U * L.Tv * 4);
  L.sbuf = off;    off += align256(U * L.Tv * 4);
  const size_t n_keep = (size_t)(p.budget < p.n ? p.budget : p.n);
  L.chosen = off;  off += align256(U * n_keep * 4);
  L.src = off;     off += align256(U * n_keep * 4);
  L.lsel = off;    off += align256(layer_select_scratch_bytes(p.n_layers, p.h_kv * L.Tv));
  L.vnorm = off;   off += align256(U * (size_t)L.Tv * 4);
  L.wins = off;    off += align256(U * 4 * 4 * 4);
  L.total = off;
  return L;
}

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

static int simt_records(const ecokv_params& p) { return (p.n + kChunk - 1) / kChunk; }
static int tc_records(const ecokv_params& p);

static size_t workspace_bytes(const ecokv_params& p) {
  const size_t a = make_layout(p, simt_records(p)).total, b = make_layout(p, tc_records(p)).total;
  return a > b ? a : b;
}

static ecokv_status check_ws(const ecokv_params* p, void* ws, size_t ws_bytes) {
  if (ws == nullptr || !aligned16(ws)) return ECOKV_ERR_WORKSPACE;
  if (ws_bytes < workspace_bytes(*p)) return ECOKV_ERR_WORKSPACE;
  return ECOKV_OK;
}

// Window rows per launch of the tensor-core kernel: all R of a unit when
// R <= 120 (the MMA's N holds the rows padded to four plus eight statistics
// columns, at most 128), else R split into ceil(R / 120) near-equal groups.
static int tc_groups(int R) { return (R + 119) / 120; }
static int tc_group_rows(int R) { return (R + tc_groups(R) - 1) / tc_groups(R); }

static bool use_tensor_path(const ecokv_params& p, ecokv_dtype dt) {
  if (dt != ECOKV_BF16 || (p.flags & ECOKV_FLAG_FORCE_SIMT)) return false;
  if (p.n < 128) return false;
  return tc_rows_half(tc_group_rows((p.h_q / p.h_kv) * p.window)) > 0;
}

// Stage events of this host thread (ecokv_set_stage_events), recorded on the
// call's stream between its launches when set.
thread_local cudaEvent_t g_stage_ev[4] = {nullptr, nullptr, nullptr, nullptr};

static void stage_event(int i, cudaStream_t s) {
  if (g_stage_ev[i] != nullptr) cudaEventRecord(g_stage_ev[i], s);
}

// Static schedule of the tensor-core kernel.  Units (heads) form waves
// (ecokv_params.sched_wave heads each; 0 = one wave of every unit), each wave
// cut into one slice per SM; every CTA streams pass 1 of its slice of wave s,
// then pass 2 of its slice of wave s - lag (ecokv_params.sched_lag, 0 = 1).
// Waves of a few heads make a key's second read an L2 hit; one wave (the
// default) runs all of pass 1 first, which measured fastest so far: the
// per-tile cost of the pipeline, not DRAM, bounds the small-wave schedules.
static int tc_wave_units(const ecokv_params& p) {
  const long long U = (long long)p.n_layers * p.h_kv;
  const long long uw = p.sched_wave > 0 ? p.sched_wave : U;
  return (int)(uw < U ? uw : U);
}

// Record slots per unit of the tensor-core passes (a bound over grids of up
// to kTcMaxSms CTAs, so that it does not depend on the device).
static int tc_records(const ecokv_params& p) {
  const long long U = (long long)p.n_layers * p.h_kv;
  const int T = (p.n + 127) / 128, uw = tc_wave_units(p);
  const long long nw = (U + uw - 1) / uw, last = U - (nw - 1) * uw;
  return tc_record_slots(T, (int)((uw < last ? uw : last) * T));
}

// SMs of the current device (cached per device).
static int num_sms() {
  static std::atomic<int> cached[64];  // a racing thread repeats the query
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  if (cached[dev].load() == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
    cached[dev].store(n);
  }
  return cached[dev].load();
}

// Keys forming the centroid of Eq. 1: all N, or with the non-window centroid
// the Tv candidates (all N when there are none).
static int kbar_count(const ecokv_params& p, const Layout& L) {
  return (p.flags & ECOKV_FLAG_CENTROID_NONWIN) && L.Tv > 0 ? L.Tv : L.N;
}

static ScoreArgs score_args(const ecokv_params& p, const Layout& L, const void* K, const void* Q, char* ws) {
  ScoreArgs a{};
  a.K = K;
  a.Q = Q;
  a.N = p.n;
  a.W = p.window;
  a.g = p.h_q / p.h_kv;
  a.R = L.R;
  a.h_kv = p.h_kv;
  a.h_q = p.h_q;
  a.Tv = L.Tv;
  a.kbar_n = kbar_count(p, L);
  a.nchunks = L.nchunks;
  a.p1_stride = L.p1_stride;
  a.ustat_stride = L.ustat_stride;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)p.d));
  a.p1part = reinterpret_cast<float*>(ws + L.p1part);
  a.ustat = reinterpret_cast<float*>(ws + L.ustat);
  a.cnt = reinterpret_cast<unsigned*>(ws + L.sync) + 4;
  a.p2part = reinterpret_cast<float*>(ws + L.p2part);
  a.simp = reinterpret_cast<float*>(ws + L.simp);
  a.dE = reinterpret_cast<float*>(ws + L.dE);
  a.cosv = reinterpret_cast<float*>(ws + L.cosv);
  return a;
}

static FinalArgs final_args(const ecokv_params& p, const Layout& L, char* ws) {
  FinalArgs f{};
  f.N = p.n;
  f.W = p.window;
  f.Tv = L.Tv;
  f.nchunks = L.nchunks;
  f.budget = p.budget;
  f.pool = p.pool_kernel;
  f.ustat_stride = L.ustat_stride;
  f.alpha = p.alpha;
  f.beta = p.beta;
  f.tau = p.tau;
  f.eps = p.eps;
  f.lambda_override = p.lambda_override;
  f.flags = p.flags;
  f.n_keep = p.budget < p.n ? p.budget : p.n;
  f.h_kv = p.h_kv;
  f.n_units = L.U;
  if (ws != nullptr) {
    f.p2part = reinterpret_cast<const float*>(ws + L.p2part);
    f.ustat = reinterpret_cast<const float*>(ws + L.ustat);
    f.simp = reinterpret_cast<const float*>(ws + L.simp);
    f.dE = reinterpret_cast<const float*>(ws + L.dE);
    f.cosv = reinterpret_cast<const float*>(ws + L.cosv);
  }
  return f;
}

static CompactArgs compact_args(const ecokv_params& p, const void* K, const void* V, const int32_t* idx, void* Ko,
                                void* Vo, unsigned* status) {
  CompactArgs c{};
  c.K = K;
  c.V = V;
  c.idx = idx;
  c.K_out = Ko;
  c.V_out = Vo;
  c.N = p.n;
  c.n_keep = p.budget < p.n ? p.budget : p.n;
  c.status = status;
  c.h_kv = p.h_kv;
  return c;
}

// Device-side wait limit of a call: ecokv_params.timeout_us, 0 = 2 s.
static unsigned long long wait_limit_ns(const ecokv_params& p) {
  return (p.timeout_us ? (unsigned long long)p.timeout_us : 2000000ull) * 1000ull;
}

// Both streaming passes on the tensor cores in one launch (after clearing
// the per-call counters), or one launch per window-row group: pass 1 of a
// group gives its rows' log-sum-exp (the centroid sums are the same in every
// group), pass 2 adds the group's vote to the vote of the groups before it.
// Every group reads K twice.
static ecokv_status run_tc_group(const ecokv_params& p, const Layout& L, const void* K, const void* Q, char* ws,
                                 int row0, int rows, int rows_max, cudaStream_t s);

static ecokv_status run_tc_passes(const ecokv_params& p, const void* K, const void* Q, char* ws, cudaStream_t s) {
  const Layout L = make_layout(p, tc_records(p));
  const int Rg = tc_group_rows(L.R);
  for (int row0 = 0; row0 < L.R; row0 += Rg) {
    const int rows = L.R - row0 < Rg ? L.R - row0 : Rg;
    const ecokv_status st = run_tc_group(p, L, K, Q, ws, row0, rows, Rg, s);
    if (st != ECOKV_OK) return st;
  }
  return ECOKV_OK;
}

static ecokv_status run_tc_group(const ecokv_params& p, const Layout& L, const void* K, const void* Q, char* ws,
                                 int row0, int rows, int rows_max, cudaStream_t s) {
  if (cudaMemsetAsync(ws + L.sync, 0, L.sync_bytes, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  TcArgs a{};
  a.U = L.U;
  a.N = p.n;
  a.W = p.window;
  a.R = rows;
  a.R4 = (rows + 3) & ~3;
  a.row0 = row0;
  a.NP = 2 * tc_rows_half(rows_max);
  a.g = p.h_q / p.h_kv;
  a.h_kv = p.h_kv;
  a.h_q = p.h_q;
  a.Tv = L.Tv;
  a.kbar_n = kbar_count(p, L);
  a.q_rows = p.n_layers * p.h_q * p.window;
  a.T = (p.n + 127) / 128;
  a.uw = tc_wave_units(p);
  a.nw = (L.U + a.uw - 1) / a.uw;
  a.lag = p.sched_lag > 0 ? p.sched_lag : 1;
  if (a.lag > a.nw) a.lag = a.nw;
  const int sms = num_sms();
  a.P = sms < kTcMaxSms ? sms : kTcMaxSms;
  a.rmax = L.nchunks;
  a.p1_stride = L.p1_stride;
  a.ustat_stride = L.ustat_stride;
  a.stall_unit = (p.flags & ECOKV_FLAG_TEST_STALL) ? 0 : -1;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)p.d));
  a.timeout_ns = wait_limit_ns(p);
  a.Q = Q;
  a.K = K;
  a.p1part = reinterpret_cast<float*>(ws + L.p1part);
  a.ustat = reinterpret_cast<float*>(ws + L.ustat);
  a.p2part = reinterpret_cast<float*>(ws + L.p2part);
  a.simp = reinterpret_cast<float*>(ws + L.simp);
  a.dE = reinterpret_cast<float*>(ws + L.dE);
  a.cosv = reinterpret_cast<float*>(ws + L.cosv);
  a.sync = reinterpret_cast<unsigned*>(ws + L.sync);
  a.status = reinterpret_cast<unsigned*>(ws + L.status);
  if (launch_tc(K, a, s) != cudaSuccess) return ECOKV_ERR_CUDA;  // a grid of a.P CTAs
  return ECOKV_OK;
}

// CUDA-core streaming passes: fill the per-token arrays and unit statistics.
static ecokv_status run_simt_passes(const ecokv_params& p, ecokv_dtype dt, const void* K, const void* Q, char* ws,
                                    cudaStream_t s) {
  if (p.flags & ECOKV_FLAG_TEST_STALL) return ECOKV_ERR_UNSUPPORTED;  // the stall exists on the tensor-core path
  const Layout L = make_layout(p, simt_records(p));
  if (cudaMemsetAsync(ws + L.sync, 0, L.sync_bytes, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  const ScoreArgs a = score_args(p, L, K, Q, ws);
  if (launch_score_simt(a, dt, L.U, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  return ECOKV_OK;
}

// Scores (and the top-k) of every unit: one cluster per unit when the unit
// fits a cluster (up to sixteen CTAs of 8192 candidates), one CTA per unit
// otherwise.
// Value-norm importance: reject heads the cluster finalize does not take
// (before anything is launched), else the norms' launch and their place.
static ecokv_status vnorm_check(const ecokv_params& p, const Layout& L) {
  if (!(p.flags & ECOKV_FLAG_VNORM_IMP)) return ECOKV_OK;
  return cluster_finalize_fits(L.Tv) ? ECOKV_OK : ECOKV_ERR_UNSUPPORTED;
}
static ecokv_status vnorm_launch(const ecokv_params& p, ecokv_dtype dt, const Layout& L, const void* V, char* ws,
                                 FinalArgs& f, cudaStream_t s) {
  if (!(p.flags & ECOKV_FLAG_VNORM_IMP)) return ECOKV_OK;
  float* vn = reinterpret_cast<float*>(ws + L.vnorm);
  f.vnorm = vn;
  return launch_value_norms(V, dt, L.U, p.n, L.Tv, vn, s) == cudaSuccess ? ECOKV_OK : ECOKV_ERR_CUDA;
}

// Order statistics of d_E for the robust forms of Eq. 2, found as
// (Tv - rank)-th largest values by one radix-select launch (a CTA per unit)
// over the pass-2 distances:
// - winsorised min-max: the clip bounds, ranks floor(p (Tv - 1)) and
//   ceil((1 - p)(Tv - 1)) (0-based ascending);
// - MAD scaling: the two middle ranks floor((Tv - 1) / 2) and floor(Tv / 2)
//   of d_E (their mean is the median), then the same ranks of |d_E - median|.
static bool winsor(const ecokv_params& p) { return (p.flags & (ECOKV_FLAG_WINSOR_1 | ECOKV_FLAG_WINSOR_5)) != 0; }
static bool robust(const ecokv_params& p) { return winsor(p) || (p.flags & ECOKV_FLAG_MAD) != 0; }
static ecokv_status robust_check(const ecokv_params& p, const Layout& L) {
  if (!robust(p)) return ECOKV_OK;
  return cluster_finalize_fits(L.Tv) && L.Tv > 0 ? ECOKV_OK : ECOKV_ERR_UNSUPPORTED;
}
static ecokv_status robust_launch(const ecokv_params& p, const Layout& L, char* ws, FinalArgs& f, cudaStream_t s) {
  if (!robust(p)) return ECOKV_OK;
  unsigned* st = reinterpret_cast<unsigned*>(ws + L.wins);  // [4][U][4]
  const float* dE = reinterpret_cast<const float*>(ws + L.dE);
  const int T = L.Tv;
  if (winsor(p)) {
    const double q = (p.flags & ECOKV_FLAG_WINSOR_1) ? 0.01 : 0.05;
    const int r_lo = (int)floor(q * (double)(T - 1)), r_hi = (int)ceil((1.0 - q) * (double)(T - 1));
    if (launch_order_stats(dE, L.U, T, T - r_lo, T - r_hi, false, st, s) != cudaSuccess) return ECOKV_ERR_CUDA;
    f.wlo = st;
    f.whi = st + (size_t)L.U * 4;
    return ECOKV_OK;
  }
  const int m_lo = (T - 1) / 2, m_hi = T / 2;
  if (launch_order_stats(dE, L.U, T, T - m_lo, T - m_hi, true, st, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  f.mad = st;
  return ECOKV_OK;
}

static ecokv_status run_finalize(FinalArgs f, int U, bool do_select, cudaStream_t s) {
  if (!do_select) f.idx = nullptr;
  const cudaError_t e = launch_finalize_cluster(f, U, false, s);
  if (e == cudaSuccess) return ECOKV_OK;
  if (e != cudaErrorNotSupported) return ECOKV_ERR_CUDA;
  return launch_finalize(f, U, do_select, s) == cudaSuccess ? ECOKV_OK : ECOKV_ERR_CUDA;
}

}  // namespace ecokv

using namespace ecokv;

extern "C" {

void ecokv_params_default(ecokv_params* p) {
  if (p == nullptr) return;
  memset(p, 0, sizeof(*p));
  p->window = 4;
  p->pool_kernel = 5;
  p->alpha = 0.8f;
  p->beta = 0.6f;
  p->tau = 0.f;
  p->eps = 1e-6f;
  p->flags = 0u;
  p->lambda_override = 0.f;
}

ecokv_status ecokv_check_params(const ecokv_params* p) {
  if (p == nullptr) return ECOKV_ERR_INVALID_ARG;
  if (p->n_layers < 1 || p->h_kv < 1 || p->h_q < 1 || p->n < 1 || p->d < 1) return ECOKV_ERR_INVALID_ARG;
  if (p->h_q % p->h_kv != 0) return ECOKV_ERR_INVALID_ARG;
  if (p->window < 1 || p->window > p->n || p->budget < p->window) return ECOKV_ERR_INVALID_ARG;
  if (p->pool_kernel < 1 || (p->pool_kernel & 1) == 0) return ECOKV_ERR_INVALID_ARG;
  if (!(p->alpha >= 0.f && p->alpha <= 1.f) || !(p->beta >= 0.f && p->beta <= 1.f)) return ECOKV_ERR_INVALID_ARG;
  if (!(p->eps > 0.f) || !isfinite(p->eps) || !isfinite(p->tau)) return ECOKV_ERR_INVALID_ARG;
  const uint32_t known =
      ECOKV_FLAG_SC_MIXKV_SIGN | ECOKV_FLAG_LAMBDA_OVERRIDE | ECOKV_FLAG_VNORM_IMP | ECOKV_FLAG_CENTROID_NONWIN |
      ECOKV_FLAG_WINSOR_1 | ECOKV_FLAG_WINSOR_5 | ECOKV_FLAG_MAD | ECOKV_FLAG_FORCE_SIMT | ECOKV_FLAG_TEST_STALL;
  if ((p->flags & ~known) != 0u) return ECOKV_ERR_INVALID_ARG;
  if ((p->flags & ECOKV_FLAG_WINSOR_1) && (p->flags & ECOKV_FLAG_WINSOR_5)) return ECOKV_ERR_INVALID_ARG;
  if ((p->flags & ECOKV_FLAG_MAD) && (p->flags & (ECOKV_FLAG_WINSOR_1 | ECOKV_FLAG_WINSOR_5)))
    return ECOKV_ERR_INVALID_ARG;
  if ((p->flags & ECOKV_FLAG_LAMBDA_OVERRIDE) && !isfinite(p->lambda_override)) return ECOKV_ERR_INVALID_ARG;
  if (p->sched_wave < 0 || p->sched_lag < 0) return ECOKV_ERR_INVALID_ARG;
  if (p->d != kD) return ECOKV_ERR_UNSUPPORTED;
  if (p->n > kMaxN) return ECOKV_ERR_UNSUPPORTED;
  if ((long long)(p->h_q / p->h_kv) * p->window > kMaxRows) return ECOKV_ERR_UNSUPPORTED;
  if ((long long)p->n_layers * p->h_kv > (1 << 20)) return ECOKV_ERR_UNSUPPORTED;
  if ((long long)p->n_layers * p->h_kv * p->n > (1LL << 31) / kD) return ECOKV_ERR_UNSUPPORTED;
  return ECOKV_OK;
}

size_t ecokv_workspace_size(const ecokv_params* p) {
  if (ecokv_check_params(p) != ECOKV_OK) return 0;
  return workspace_bytes(*p);
}

ecokv_status ecokv_score(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* Qwin, float* S,
                         float* lambda, float* dbg, void* ws, size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (p->flags & ECOKV_FLAG_VNORM_IMP) return ECOKV_ERR_UNSUPPORTED;  // needs V: use ecokv_evict
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!K || !Qwin || !aligned16(K) || !aligned16(Qwin)) return ECOKV_ERR_INVALID_ARG;
  if (p->n > p->window && (!S || !aligned16(S))) return ECOKV_ERR_INVALID_ARG;
  if ((lambda && ((uintptr_t)lambda & 3u)) || (dbg && !aligned16(dbg))) return ECOKV_ERR_INVALID_ARG;
  if ((st = check_ws(p, ws, ws_bytes)) != ECOKV_OK) return st;
  char* w = static_cast<char*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool tc = use_tensor_path(*p, dtype);
  const Layout L = make_layout(*p, tc ? tc_records(*p) : simt_records(*p));
  FinalArgs f = final_args(*p, L, w);
  f.S = S;
  f.lambda = lambda;
  f.dbg = dbg;
  if ((st = robust_check(*p, L)) != ECOKV_OK) return st;
  stage_event(0, s);
  st = tc ? run_tc_passes(*p, K, Qwin, w, s) : run_simt_passes(*p, dtype, K, Qwin, w, s);
  if (st != ECOKV_OK) return st;
  stage_event(1, s);
  if ((st = robust_launch(*p, L, w, f, s)) != ECOKV_OK) return st;
  if (run_finalize(f, L.U, false, s) != ECOKV_OK) return ECOKV_ERR_CUDA;
  stage_event(2, s);
  return ECOKV_OK;
}

ecokv_status ecokv_select(const ecokv_params* p, const float* S, int32_t* idx, void* ws, size_t ws_bytes,
                          void* stream) {
  (void)ws;
  (void)ws_bytes;
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (!idx || !aligned16(idx)) return ECOKV_ERR_INVALID_ARG;
  if (p->budget < p->n && p->n > p->window && (!S || !aligned16(S))) return ECOKV_ERR_INVALID_ARG;
  const Layout L = make_layout(*p, simt_records(*p));
  FinalArgs f = final_args(*p, L, nullptr);
  f.S = const_cast<float*>(S);
  f.idx = idx;
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  const cudaError_t e = launch_finalize_cluster(f, L.U, true, s);
  if (e == cudaSuccess) return ECOKV_OK;
  if (e != cudaErrorNotSupported) return ECOKV_ERR_CUDA;
  if (launch_select(f, L.U, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  return ECOKV_OK;
}

ecokv_status ecokv_compact(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                           const int32_t* idx, void* K_out, void* V_out, void* ws, size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!K || !V || !idx || !K_out || !V_out) return ECOKV_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(V) || !aligned16(K_out) || !aligned16(V_out) || ((uintptr_t)idx & 3u))
    return ECOKV_ERR_INVALID_ARG;
  if (ws != nullptr && (!aligned16(ws) || ws_bytes < 256)) return ECOKV_ERR_WORKSPACE;
  const Layout L = make_layout(*p, simt_records(*p));
  unsigned* status = ws ? reinterpret_cast<unsigned*>(static_cast<char*>(ws) + L.status) : nullptr;
  const CompactArgs c = compact_args(*p, K, V, idx, K_out, V_out, status);
  if (launch_compact(c, dtype, L.U, static_cast<cudaStream_t>(stream)) != cudaSuccess) return ECOKV_ERR_CUDA;
  return ECOKV_OK;
}

ecokv_status ecokv_evict_adaptive(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                  const void* Qwin, int32_t* idx, int32_t* head_off, void* K_out, void* V_out,
                                  float* lambda, void* ws, size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!K || !V || !Qwin || !idx || !head_off || !K_out || !V_out) return ECOKV_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(V) || !aligned16(Qwin) || !aligned16(idx) || !aligned16(K_out) ||
      !aligned16(V_out) || ((uintptr_t)head_off & 3u) || (lambda && ((uintptr_t)lambda & 3u)))
    return ECOKV_ERR_INVALID_ARG;
  if ((st = check_ws(p, ws, ws_bytes)) != ECOKV_OK) return st;
  char* w = static_cast<char*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool tc = use_tensor_path(*p, dtype);
  const Layout L = make_layout(*p, tc ? tc_records(*p) : simt_records(*p));
  const int n_keep = p->budget < p->n ? p->budget : p->n;
  const bool keep_all = p->budget >= p->n;
  // 1. every head's scores, into the workspace
  FinalArgs f = final_args(*p, L, w);
  f.S = reinterpret_cast<float*>(w + L.sbuf);
  f.lambda = lambda;
  if ((st = vnorm_check(*p, L)) != ECOKV_OK || (st = robust_check(*p, L)) != ECOKV_OK) return st;
  stage_event(0, s);
  st = tc ? run_tc_passes(*p, K, Qwin, w, s) : run_simt_passes(*p, dtype, K, Qwin, w, s);
  if (st != ECOKV_OK) return st;
  if ((st = vnorm_launch(*p, dtype, L, V, w, f, s)) != ECOKV_OK) return st;
  if ((st = robust_launch(*p, L, w, f, s)) != ECOKV_OK) return st;
  stage_event(1, s);
  if (run_finalize(f, L.U, false, s) != ECOKV_OK) return ECOKV_ERR_CUDA;
  // 2. one top-h_kv (B - W) per layer over its heads' concatenated scores
  //    ([h_kv][Tv] per layer is contiguous), ties to the lower (head, position)
  AdaptArgs a{};
  a.chosen = reinterpret_cast<const int32_t*>(w + L.chosen);
  a.idx = idx;
  a.head_off = head_off;
  a.src = reinterpret_cast<int32_t*>(w + L.src);
  a.h_kv = p->h_kv;
  a.N = p->n;
  a.W = p->window;
  a.Tv = L.Tv;
  a.n_keep = n_keep;
  a.k_layer = keep_all ? 0 : p->h_kv * (p->budget - p->window);
  a.keep_all = keep_all ? 1 : 0;
  if (!keep_all && a.k_layer > 0 &&
      launch_layer_select(f.S, p->n_layers, p->h_kv * L.Tv, a.k_layer, reinterpret_cast<int32_t*>(w + L.chosen),
                          w + L.lsel, s) != cudaSuccess)
    return ECOKV_ERR_CUDA;
  // 3. per-head lists and offsets, then the gather over each layer's
  //    [h_kv * N] rows
  if (launch_adaptive_split(a, p->n_layers, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  stage_event(2, s);
  ecokv_params pl = *p;
  pl.n = p->h_kv * p->n;
  pl.budget = p->h_kv * n_keep;
  CompactArgs c = compact_args(pl, K, V, reinterpret_cast<const int32_t*>(w + L.src), K_out, V_out,
                               reinterpret_cast<unsigned*>(w + L.status));
  if (launch_compact(c, dtype, p->n_layers, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  stage_event(3, s);
  return ECOKV_OK;
}

static ecokv_status evict_impl(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                               const void* Qwin, int32_t* idx, void* K_out, void* V_out, float* S, float* lambda,
                               void* ws, size_t ws_bytes, void* stream, const int32_t* layer_budget) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!K || !V || !Qwin || !idx || !K_out || !V_out) return ECOKV_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(V) || !aligned16(Qwin) || !aligned16(idx) || !aligned16(K_out) ||
      !aligned16(V_out))
    return ECOKV_ERR_INVALID_ARG;
  if ((S && !aligned16(S)) || (lambda && ((uintptr_t)lambda & 3u))) return ECOKV_ERR_INVALID_ARG;
  if ((st = check_ws(p, ws, ws_bytes)) != ECOKV_OK) return st;
  char* w = static_cast<char*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool tc = use_tensor_path(*p, dtype);
  const Layout L = make_layout(*p, tc ? tc_records(*p) : simt_records(*p));
  FinalArgs f = final_args(*p, L, w);
  f.S = S;
  f.S_scratch = reinterpret_cast<float*>(w + L.sbuf);
  f.lambda = lambda;
  f.idx = idx;
  CompactArgs c = compact_args(*p, K, V, idx, K_out, V_out, reinterpret_cast<unsigned*>(w + L.status));
  if (layer_budget != nullptr) {
    f.n_lb = c.n_lb = p->n_layers;
    for (int l = 0; l < p->n_layers; ++l) {
      f.lb[l] = layer_budget[l];
      c.keep[l] = layer_budget[l] < p->n ? layer_budget[l] : p->n;
    }
  }
  if ((st = vnorm_check(*p, L)) != ECOKV_OK || (st = robust_check(*p, L)) != ECOKV_OK) return st;
  stage_event(0, s);
  st = tc ? run_tc_passes(*p, K, Qwin, w, s) : run_simt_passes(*p, dtype, K, Qwin, w, s);
  if (st != ECOKV_OK) return st;
  if ((st = vnorm_launch(*p, dtype, L, V, w, f, s)) != ECOKV_OK) return st;
  if ((st = robust_launch(*p, L, w, f, s)) != ECOKV_OK) return st;
  stage_event(1, s);
  if (run_finalize(f, L.U, true, s) != ECOKV_OK) return ECOKV_ERR_CUDA;
  stage_event(2, s);
  if (launch_compact(c, dtype, L.U, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  stage_event(3, s);
  return ECOKV_OK;
}

ecokv_status ecokv_evict(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V, const void* Qwin,
                         int32_t* idx, void* K_out, void* V_out, float* S, float* lambda, void* ws,
                         size_t ws_bytes, void* stream) {
  return evict_impl(p, dtype, K, V, Qwin, idx, K_out, V_out, S, lambda, ws, ws_bytes, stream, nullptr);
}

ecokv_status ecokv_evict_layered(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                 const void* Qwin, const int32_t* layer_budget, int32_t* idx, void* K_out,
                                 void* V_out, float* S, float* lambda, void* ws, size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (layer_budget == nullptr) return ECOKV_ERR_INVALID_ARG;
  if (p->n_layers > kMaxLayerBudgets) return ECOKV_ERR_UNSUPPORTED;
  for (int l = 0; l < p->n_layers; ++l)
    if (layer_budget[l] < p->window || layer_budget[l] > p->budget) return ECOKV_ERR_INVALID_ARG;
  return evict_impl(p, dtype, K, V, Qwin, idx, K_out, V_out, S, lambda, ws, ws_bytes, stream, layer_budget);
}

ecokv_status ecokv_pyramid_budgets(int32_t n_layers, int32_t budget, int32_t window, float beta, int32_t* out) {
  if (n_layers < 1 || budget < window || window < 1 || !(beta > 0.f) || !isfinite(beta) || out == nullptr)
    return ECOKV_ERR_INVALID_ARG;
  // PyramidKV (Appendix A): b^{m-1} = b_total / (beta m), b^0 = 2 b_total / m
  // - b^{m-1}, linear between; b_total = m B; rounded half up, at least W
  const double m = (double)n_layers, total = m * (double)budget, b = (double)beta;
  if (n_layers == 1) {
    out[0] = budget;
    return ECOKV_OK;
  }
  const double b_last = total / (b * m);
  const double b_first = 2.0 * total / m - b_last;
  for (int l = 0; l < n_layers; ++l) {
    const double x = b_first - (b_first - b_last) / (m - 1.0) * (double)l;
    const double r = floor(x + 0.5);
    out[l] = r < (double)window ? window : (r > 2147483647.0 ? 2147483647 : (int32_t)r);
  }
  return ECOKV_OK;
}

ecokv_status ecokv_device_status(void* ws, void* stream) {
  if (ws == nullptr || !aligned16(ws)) return ECOKV_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return ECOKV_ERR_CUDA;
  DevStatus h{};
  if (cudaMemcpy(&h, ws, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return ECOKV_ERR_CUDA;
  if (h.code != 0u) {
    const DevStatus z{};
    if (cudaMemcpy(ws, &z, sizeof(z), cudaMemcpyHostToDevice) != cudaSuccess) return ECOKV_ERR_CUDA;
  }
  return static_cast<ecokv_status>(h.code);
}

ecokv_status ecokv_set_stage_events(void* const* events, int n) {
  if (events == nullptr) {
    for (int i = 0; i < 4; ++i) g_stage_ev[i] = nullptr;
    return ECOKV_OK;
  }
  if (n != 4) return ECOKV_ERR_INVALID_ARG;
  for (int i = 0; i < 4; ++i) g_stage_ev[i] = static_cast<cudaEvent_t>(events[i]);
  return ECOKV_OK;
}

const char* ecokv_status_string(ecokv_status s) {
  switch (s) {
    case ECOKV_OK: return "ok";
    case ECOKV_ERR_INVALID_ARG: return "invalid argument";
    case ECOKV_ERR_UNSUPPORTED: return "unsupported configuration";
    case ECOKV_ERR_WORKSPACE: return "workspace missing or too small";
    case ECOKV_ERR_CUDA: return "CUDA runtime error";
    case ECOKV_ERR_TIMEOUT: return "device-side wait timed out";
    case ECOKV_ERR_DEVICE_INDEX: return "index outside [0, n) seen on the device";
  }
  return "unknown status";
}

}  // extern "C"
