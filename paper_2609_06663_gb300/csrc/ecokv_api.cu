// C ABI of libecokv.so: argument checks, workspace layout and launches.
// Every entry point validates on the host and returns before launching
// anything when an argument is wrong.

#include <math.h>
#include <string.h>

#include "ecokv_internal.cuh"

namespace ecokv {

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

Layout make_layout(const ecokv_params& p) {
  Layout L{};
  L.U = p.n_layers * p.h_kv;
  L.R = (p.h_q / p.h_kv) * p.window;
  L.N = p.n;
  L.W = p.window;
  L.Tv = p.n - p.window;
  L.nchunks = (p.n + kChunk - 1) / kChunk;
  L.p1_stride = 2 * L.R + 2 * kD;
  L.ustat_stride = (2 * kD + 2 + L.R + 3) & ~3;
  const size_t U = (size_t)L.U;
  size_t off = 0;
  L.status = off;  off += 256;
  L.cnt = off;     off += align256(U * 4);
  L.p1part = off;  off += align256(U * L.nchunks * L.p1_stride * 4);
  L.ustat = off;   off += align256(U * L.ustat_stride * 4);
  L.p2part = off;  off += align256(U * L.nchunks * 4);
  L.simp = off;    off += align256(U * L.Tv * 4);
  L.dE = off;      off += align256(U * L.Tv * 4);
  L.cosv = off;    off += align256(U * L.Tv * 4);
  L.sbuf = off;    off += align256(U * L.Tv * 4);
  L.total = off;
  return L;
}

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

static ecokv_status check_ws(const ecokv_params* p, void* ws, size_t ws_bytes) {
  if (ws == nullptr || !aligned16(ws)) return ECOKV_ERR_WORKSPACE;
  if (ws_bytes < make_layout(*p).total) return ECOKV_ERR_WORKSPACE;
  return ECOKV_OK;
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
  a.nchunks = L.nchunks;
  a.p1_stride = L.p1_stride;
  a.ustat_stride = L.ustat_stride;
  a.scale_log2 = (float)(1.4426950408889634 / sqrt((double)p.d));
  a.p1part = reinterpret_cast<float*>(ws + L.p1part);
  a.ustat = reinterpret_cast<float*>(ws + L.ustat);
  a.cnt = reinterpret_cast<unsigned*>(ws + L.cnt);
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
  if (ws != nullptr) {
    f.p2part = reinterpret_cast<const float*>(ws + L.p2part);
    f.ustat = reinterpret_cast<const float*>(ws + L.ustat);
    f.simp = reinterpret_cast<const float*>(ws + L.simp);
    f.dE = reinterpret_cast<const float*>(ws + L.dE);
    f.cosv = reinterpret_cast<const float*>(ws + L.cosv);
  }
  return f;
}

// Run both streaming passes: fills the per-token arrays and unit statistics.
static ecokv_status run_passes(const ecokv_params& p, const Layout& L, ecokv_dtype dt, const void* K,
                               const void* Q, char* ws, cudaStream_t s) {
  if (cudaMemsetAsync(ws + L.cnt, 0, (size_t)L.U * 4, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  const ScoreArgs a = score_args(p, L, K, Q, ws);
  if (launch_score_simt(a, dt, L.U, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  return ECOKV_OK;
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
  if ((p->flags & ~(ECOKV_FLAG_SC_MIXKV_SIGN | ECOKV_FLAG_LAMBDA_OVERRIDE)) != 0u) return ECOKV_ERR_INVALID_ARG;
  if ((p->flags & ECOKV_FLAG_LAMBDA_OVERRIDE) && !isfinite(p->lambda_override)) return ECOKV_ERR_INVALID_ARG;
  if (p->d != kD) return ECOKV_ERR_UNSUPPORTED;
  if (p->n > kMaxN) return ECOKV_ERR_UNSUPPORTED;
  if ((long long)(p->h_q / p->h_kv) * p->window > kMaxRows) return ECOKV_ERR_UNSUPPORTED;
  if ((long long)p->n_layers * p->h_kv > (1 << 20)) return ECOKV_ERR_UNSUPPORTED;
  return ECOKV_OK;
}

size_t ecokv_workspace_size(const ecokv_params* p) {
  if (ecokv_check_params(p) != ECOKV_OK) return 0;
  return make_layout(*p).total;
}

ecokv_status ecokv_score(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* Qwin, float* S,
                         float* lambda, float* dbg, void* ws, size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!K || !Qwin || !aligned16(K) || !aligned16(Qwin)) return ECOKV_ERR_INVALID_ARG;
  if (p->n > p->window && (!S || !aligned16(S))) return ECOKV_ERR_INVALID_ARG;
  if ((lambda && ((uintptr_t)lambda & 3u)) || (dbg && !aligned16(dbg))) return ECOKV_ERR_INVALID_ARG;
  if ((st = check_ws(p, ws, ws_bytes)) != ECOKV_OK) return st;
  const Layout L = make_layout(*p);
  char* w = static_cast<char*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = run_passes(*p, L, dtype, K, Qwin, w, s)) != ECOKV_OK) return st;
  FinalArgs f = final_args(*p, L, w);
  f.S = S;
  f.lambda = lambda;
  f.dbg = dbg;
  if (launch_finalize(f, L.U, true, false, s) != cudaSuccess) return ECOKV_ERR_CUDA;
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
  const Layout L = make_layout(*p);
  FinalArgs f = final_args(*p, L, nullptr);
  f.S = const_cast<float*>(S);
  f.idx = idx;
  if (launch_finalize(f, L.U, false, true, static_cast<cudaStream_t>(stream)) != cudaSuccess) return ECOKV_ERR_CUDA;
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
  const Layout L = make_layout(*p);
  CompactArgs c{};
  c.K = K;
  c.V = V;
  c.idx = idx;
  c.K_out = K_out;
  c.V_out = V_out;
  c.N = p->n;
  c.n_keep = p->budget < p->n ? p->budget : p->n;
  c.status = ws ? reinterpret_cast<unsigned*>(static_cast<char*>(ws) + L.status) : nullptr;
  if (launch_compact(c, dtype, L.U, static_cast<cudaStream_t>(stream)) != cudaSuccess) return ECOKV_ERR_CUDA;
  return ECOKV_OK;
}

ecokv_status ecokv_evict(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V, const void* Qwin,
                         int32_t* idx, void* K_out, void* V_out, float* S, float* lambda, void* ws,
                         size_t ws_bytes, void* stream) {
  ecokv_status st = ecokv_check_params(p);
  if (st != ECOKV_OK) return st;
  if (dtype != ECOKV_F32 && dtype != ECOKV_BF16) return ECOKV_ERR_INVALID_ARG;
  if (!K || !V || !Qwin || !idx || !K_out || !V_out) return ECOKV_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(V) || !aligned16(Qwin) || !aligned16(idx) || !aligned16(K_out) ||
      !aligned16(V_out))
    return ECOKV_ERR_INVALID_ARG;
  if ((S && !aligned16(S)) || (lambda && ((uintptr_t)lambda & 3u))) return ECOKV_ERR_INVALID_ARG;
  if ((st = check_ws(p, ws, ws_bytes)) != ECOKV_OK) return st;
  const Layout L = make_layout(*p);
  char* w = static_cast<char*>(ws);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = run_passes(*p, L, dtype, K, Qwin, w, s)) != ECOKV_OK) return st;
  FinalArgs f = final_args(*p, L, w);
  f.S = S ? S : reinterpret_cast<float*>(w + L.sbuf);
  f.lambda = lambda;
  f.idx = idx;
  if (launch_finalize(f, L.U, true, true, s) != cudaSuccess) return ECOKV_ERR_CUDA;
  CompactArgs c{};
  c.K = K;
  c.V = V;
  c.idx = idx;
  c.K_out = K_out;
  c.V_out = V_out;
  c.N = p->n;
  c.n_keep = f.n_keep;
  c.status = reinterpret_cast<unsigned*>(w + L.status);
  if (launch_compact(c, dtype, L.U, s) != cudaSuccess) return ECOKV_ERR_CUDA;
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
