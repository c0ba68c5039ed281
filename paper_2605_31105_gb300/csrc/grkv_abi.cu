// C ABI of the GRKV compression path: host-side validation, workspace plan
// and the launch sequence of each entry point declared in grkv.h.
#include <algorithm>
#include <atomic>
#include <cmath>

#include "grkv_internal.cuh"

using namespace grkv;

namespace {

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int check_ws(const WsLayout& L, const void* ws, size_t ws_bytes) {
  if (!ws) return GRKV_ERR_INVALID_ARG;
  if (!aligned16(ws)) return GRKV_ERR_MISALIGNED;
  if (ws_bytes < L.total) return GRKV_ERR_WORKSPACE_TOO_SMALL;
  return GRKV_OK;
}

// Non-null (unless the array is empty) and 16-byte aligned.
int check_ptr(const void* p, size_t elems) {
  if (elems == 0) return GRKV_OK;
  if (!p) return GRKV_ERR_INVALID_ARG;
  return aligned16(p) ? GRKV_OK : GRKV_ERR_MISALIGNED;
}

int cuda_rc(cudaError_t e) { return e == cudaSuccess ? GRKV_OK : GRKV_ERR_CUDA; }

#define GRKV_TRY(expr)            \
  do {                            \
    const int rc_ = (expr);       \
    if (rc_ != GRKV_OK) return rc_; \
  } while (0)

int check_inputs(const Shape& s, const void* q, const void* k, const void* v) {
  GRKV_TRY(check_ptr(q, (size_t)s.U * s.m));
  GRKV_TRY(check_ptr(k, (size_t)s.U * s.n));
  GRKV_TRY(check_ptr(v, (size_t)s.U * s.n));
  return GRKV_OK;
}

}  // namespace

namespace grkv {

// The value step (and gather) on the tensor cores or the portable kernels.
cudaError_t launch_merge_any(const Shape& s, const void* q, const void* k, const void* v,
                             const float* scores, const float* y, const float* row_stats,
                             const int32_t* idx, void* k_out, void* v_out, char* ws,
                             const WsLayout& L, cudaStream_t st) {
  if (s.tc_merge)
    return launch_merge_tc(s, q, k, v, scores, y, row_stats, idx, k_out, v_out, ws, L, st);
  return launch_merge_simt(s, q, k, v, scores, y, idx, k_out, v_out, ws, L, st);
}

// Window scoring: the two-launch tensor-core kernel (default), the one-read
// kernel, or the portable kernels.
cudaError_t launch_score_any(const Shape& s, const void* q, const void* k, const void* v,
                             float* scores, float* y, float* row_stats, char* ws,
                             const WsLayout& L, cudaStream_t st) {
  if (s.tc && s.one_read && !s.deterministic)
    return launch_score_pipe(s, q, k, v, scores, y, row_stats, ws, L, st);
  if (s.tc) return launch_score_tc(s, q, k, v, scores, y, row_stats, ws, L, 0, st);
  return launch_score_simt(s, q, k, v, scores, y, row_stats, ws, L, st);
}

int make_shape(const grkv_params* p, Shape* s) {
  if (!p) return GRKV_ERR_INVALID_ARG;
  if (p->units < 0 || p->group < 1 || p->window < 1 || p->n < p->window) return GRKV_ERR_INVALID_ARG;
  if (p->budget < p->window || p->budget > p->n) return GRKV_ERR_INVALID_ARG;
  if (p->pool_kernel < 1 || (p->pool_kernel & 1) == 0) return GRKV_ERR_INVALID_ARG;
  if (p->pool_type != GRKV_POOL_MAX && p->pool_type != GRKV_POOL_AVG) return GRKV_ERR_INVALID_ARG;
  if (p->n_sink < 0) return GRKV_ERR_INVALID_ARG;
  if (!(p->beta >= 0.f && p->beta < 1.f)) return GRKV_ERR_INVALID_ARG;
  if (!(p->lambda_v >= 0.f)) return GRKV_ERR_INVALID_ARG;          // rejects NaN
  if (!(p->scale >= 0.f) || std::isinf(p->scale)) return GRKV_ERR_INVALID_ARG;
  if (p->causal != 0 && p->causal != 1) return GRKV_ERR_INVALID_ARG;
  if (p->dtype != GRKV_F32 && p->dtype != GRKV_BF16) return GRKV_ERR_INVALID_ARG;
  if (p->flags & ~(GRKV_UPDATE_K | GRKV_FORCE_SIMT | GRKV_ONE_READ_SCORE | GRKV_DETERMINISTIC |
                   GRKV_CHECKS | GRKV_TEST_TIMEOUT)) return GRKV_ERR_INVALID_ARG;
  if (p->d < 1) return GRKV_ERR_INVALID_ARG;
  if (p->flags & GRKV_UPDATE_K) {
    if (!(p->lambda_k >= 0.f) || std::isinf(p->lambda_k)) return GRKV_ERR_INVALID_ARG;
    if (p->cg_iters < 0 || p->cg_iters > kMaxCgIters) return GRKV_ERR_INVALID_ARG;
    if (!(p->cg_tol >= 0.f) || std::isinf(p->cg_tol)) return GRKV_ERR_INVALID_ARG;
  }
  if (p->steps < 1 || p->steps > kMaxSteps) return GRKV_ERR_INVALID_ARG;
  if (p->steps > 1 && !(p->flags & GRKV_UPDATE_K)) return GRKV_ERR_INVALID_ARG;
  if (!(p->step_tol >= 0.f) || std::isinf(p->step_tol)) return GRKV_ERR_INVALID_ARG;
  if (p->d != kD) return GRKV_ERR_UNSUPPORTED;
  if ((int64_t)p->group * p->window > kMaxM) return GRKV_ERR_UNSUPPORTED;
  if ((int64_t)p->n * kD > (int64_t)1 << 31) return GRKV_ERR_UNSUPPORTED;
  s->U = p->units;
  s->g = p->group;
  s->n = p->n;
  s->d = p->d;
  s->w = p->window;
  s->B = p->budget;
  s->m = p->group * p->window;
  s->P = p->n - p->window;
  s->kk = p->budget - p->window;
  s->pool_k = p->pool_kernel;
  s->pool_type = p->pool_type;
  s->n_sink = p->n_sink;
  s->n_fix = (int)std::floor((double)p->beta * (double)p->budget);
  s->causal = p->causal;
  s->dtype = p->dtype;
  s->lambda = p->lambda_v;
  s->lambda_inf = std::isinf(p->lambda_v) ? 1 : 0;
  s->scale = p->scale != 0.f ? p->scale : (float)(1.0 / std::sqrt((double)p->d));
  s->tc = (p->flags & GRKV_FORCE_SIMT) ? 0 : (score_tc_supported(*s) ? 1 : 0);
  s->tc_merge = (s->tc && merge_tc_supported(*s)) ? 1 : 0;
  s->one_read = (p->flags & GRKV_ONE_READ_SCORE) ? 1 : 0;
  s->deterministic = (p->flags & GRKV_DETERMINISTIC) ? 1 : 0;
  s->test_timeout = (p->flags & GRKV_TEST_TIMEOUT) ? 1 : 0;
  s->checks = (p->flags & GRKV_CHECKS) ? 1 : 0;
  s->update_k = (p->flags & GRKV_UPDATE_K) ? 1 : 0;
  s->cg_iters = p->cg_iters;
  s->cg_tol = p->cg_tol;
  s->steps = p->steps;
  s->step_tol = p->step_tol;
  s->lambda_k = p->lambda_k;
  return GRKV_OK;
}

static std::atomic<uint64_t> g_launches{0};

void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

WsLayout plan_workspace(const Shape& s) {
  WsLayout L{};
  const size_t U = (size_t)s.U, m = (size_t)s.m, d = (size_t)kD;
  // portable scoring: chunks of a multiple of 64 keys, enough of them that
  // U x chunks fills the GPU a few times over (608 CTAs) without splitting a
  // unit into chunks of fewer than 64 keys
  {
    const int per_unit = std::max(1, std::min((608 + std::max(s.U, 1) - 1) / std::max(s.U, 1),
                                              (s.n + 63) / 64));
    L.chunk = std::max(64, ((s.n + per_unit - 1) / per_unit + 63) / 64 * 64);
  }
  L.nchunk = (s.n + L.chunk - 1) / L.chunk;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + bytes);
    return at;
  };
  L.status = take(256);
  if (s.tc) {
    int maxc, gu, rounds;
    L.pstats_tc = take(std::max(score_tc_pstats_bytes(s, &maxc, &gu, &rounds, kMaxScoreCtas),
                                score_pipe_slot_bytes(s)));
    L.flags_tc = take(U * sizeof(int));
    L.lam_tc = take(U * 128 * sizeof(float));
    if (s.deterministic) L.ypart_tc = take(U * (size_t)maxc * m * d * sizeof(float));
  } else {
    L.pstats = take(U * L.nchunk * m * 8);
    L.ypart = take(U * L.nchunk * m * d * 4);
  }
  L.pooled = take(U * (size_t)s.P * 4);
  if (s.tc_merge) {
    L.merge_tc = take(merge_tc_ws_bytes(s));
  } else {
    L.xbuf = take(U * m * (size_t)s.B * 4);
    L.flags = take(U * (size_t)s.B);
    L.gram = take(U * m * m * 8);
    L.rz = take(U * m * d * 8);
  }
  L.scores = take(U * (size_t)s.P * 4);
  L.y = take(U * m * d * 4);
  L.rstats = take(U * m * 8);
  if (s.update_k) L.key = take(key_ws_bytes(s));
  L.total = off;
  return L;
}

}  // namespace grkv

extern "C" {

void grkv_params_init(grkv_params* p, int32_t units, int32_t group, int32_t n, int32_t window,
                      int32_t budget) {
  if (!p) return;
  p->units = units;
  p->group = group;
  p->n = n;
  p->d = kD;
  p->window = window;
  p->budget = budget;
  p->pool_kernel = 7;
  p->pool_type = GRKV_POOL_MAX;
  p->n_sink = 4;
  p->beta = 0.10f;
  p->lambda_v = 1e-2f;
  p->lambda_k = 1e-2f;
  p->scale = 0.f;
  p->causal = 1;
  p->dtype = GRKV_BF16;
  p->flags = 0;
  p->cg_iters = 512;
  p->cg_tol = 1e-4f;
  p->steps = 1;
  p->step_tol = 1e-9f;
}

int grkv_workspace_size(const grkv_params* p, size_t* bytes) {
  Shape s;
  GRKV_TRY(make_shape(p, &s));
  if (!bytes) return GRKV_ERR_INVALID_ARG;
  *bytes = plan_workspace(s).total;
  return GRKV_OK;
}

int grkv_score(const grkv_params* p, const void* q, const void* k, const void* v, float* scores,
               float* y, float* row_stats, void* ws, size_t ws_bytes, void* stream) {
  Shape s;
  GRKV_TRY(make_shape(p, &s));
  const WsLayout L = plan_workspace(s);
  GRKV_TRY(check_ws(L, ws, ws_bytes));
  GRKV_TRY(check_inputs(s, q, k, v));
  GRKV_TRY(check_ptr(scores, (size_t)s.U * s.P));
  GRKV_TRY(check_ptr(y, (size_t)s.U * s.m));
  GRKV_TRY(check_ptr(row_stats, (size_t)s.U * s.m));
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  GRKV_TRY(cuda_rc(cudaMemsetAsync(w + L.status, 0, 4, st)));
  if (s.U == 0) return GRKV_OK;
  return cuda_rc(launch_score_any(s, q, k, v, scores, y, row_stats, w, L, st));
}

int grkv_select(const grkv_params* p, const float* scores, int32_t* idx, void* ws,
                size_t ws_bytes, void* stream) {
  Shape s;
  GRKV_TRY(make_shape(p, &s));
  const WsLayout L = plan_workspace(s);
  GRKV_TRY(check_ws(L, ws, ws_bytes));
  GRKV_TRY(check_ptr(scores, (size_t)s.U * s.P));
  GRKV_TRY(check_ptr(idx, (size_t)s.U * s.B));
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  GRKV_TRY(cuda_rc(cudaMemsetAsync(w + L.status, 0, 4, st)));
  if (s.U == 0) return GRKV_OK;
  return cuda_rc(launch_select(s, scores, idx, w, L, st));
}

int grkv_merge(const grkv_params* p, const void* q, const void* k, const void* v,
               const float* scores, const float* y, const float* row_stats, const int32_t* idx,
               void* k_out, void* v_out, void* ws, size_t ws_bytes, void* stream) {
  Shape s;
  GRKV_TRY(make_shape(p, &s));
  const WsLayout L = plan_workspace(s);
  GRKV_TRY(check_ws(L, ws, ws_bytes));
  GRKV_TRY(check_inputs(s, q, k, v));
  GRKV_TRY(check_ptr(scores, (size_t)s.U * s.P));
  GRKV_TRY(check_ptr(y, (size_t)s.U * s.m));
  if (row_stats) GRKV_TRY(check_ptr(row_stats, (size_t)s.U * s.m));
  GRKV_TRY(check_ptr(idx, (size_t)s.U * s.B));
  GRKV_TRY(check_ptr(k_out, (size_t)s.U * s.B));
  GRKV_TRY(check_ptr(v_out, (size_t)s.U * s.B));
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  GRKV_TRY(cuda_rc(cudaMemsetAsync(w + L.status, 0, 4, st)));
  if (s.U == 0) return GRKV_OK;
  if (s.checks) {
    GRKV_TRY(cuda_rc(launch_check_inputs(s, q, k, v, (int*)(w + L.status), st)));
    GRKV_TRY(cuda_rc(launch_check_idx(s, idx, (int*)(w + L.status), st)));
  }
  GRKV_TRY(cuda_rc(launch_merge_any(s, q, k, v, scores, y, row_stats, idx, k_out, v_out, w, L, st)));
  if (!s.update_k) return GRKV_OK;
  return cuda_rc(launch_key_step(s, q, k, v, y, scores, idx, v_out, k_out, w, L, st));
}

int grkv_compress(const grkv_params* p, const void* q, const void* k, const void* v, void* k_out,
                  void* v_out, int32_t* idx, void* ws, size_t ws_bytes, void* stream) {
  Shape s;
  GRKV_TRY(make_shape(p, &s));
  const WsLayout L = plan_workspace(s);
  GRKV_TRY(check_ws(L, ws, ws_bytes));
  GRKV_TRY(check_inputs(s, q, k, v));
  GRKV_TRY(check_ptr(idx, (size_t)s.U * s.B));
  GRKV_TRY(check_ptr(k_out, (size_t)s.U * s.B));
  GRKV_TRY(check_ptr(v_out, (size_t)s.U * s.B));
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  GRKV_TRY(cuda_rc(cudaMemsetAsync(w + L.status, 0, 4, st)));
  if (s.U == 0) return GRKV_OK;
  float* scores = (float*)(w + L.scores);
  float* y = (float*)(w + L.y);
  float* rstats = (float*)(w + L.rstats);
  if (s.checks) GRKV_TRY(cuda_rc(launch_check_inputs(s, q, k, v, (int*)(w + L.status), st)));
  GRKV_TRY(cuda_rc(launch_score_any(s, q, k, v, scores, y, rstats, w, L, st)));
  GRKV_TRY(cuda_rc(launch_select(s, scores, idx, w, L, st)));
  GRKV_TRY(cuda_rc(launch_merge_any(s, q, k, v, scores, y, rstats, idx, k_out, v_out, w, L, st)));
  if (!s.update_k) return GRKV_OK;
  return cuda_rc(launch_key_step(s, q, k, v, y, scores, idx, v_out, k_out, w, L, st));
}

int grkv_status(const void* ws, int* device_status, void* stream) {
  if (!ws || !device_status) return GRKV_ERR_INVALID_ARG;
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return GRKV_ERR_CUDA;
  int h = 0;
  if (cudaMemcpy(&h, ws, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return GRKV_ERR_CUDA;
  *device_status = h;
  return GRKV_OK;
}

uint64_t grkv_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char* grkv_strerror(int code) {
  switch (code) {
    case GRKV_OK: return "ok";
    case GRKV_ERR_INVALID_ARG: return "invalid argument";
    case GRKV_ERR_UNSUPPORTED: return "unsupported configuration";
    case GRKV_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case GRKV_ERR_MISALIGNED: return "device pointer not 16-byte aligned";
    case GRKV_ERR_CUDA: return "CUDA error";
    case GRKV_ERR_NUMERIC: return "non-positive Cholesky pivot";
    case GRKV_ERR_TIMEOUT: return "bounded device wait expired";
    case GRKV_ERR_BOUNDS: return "idx breaks its contract (GRKV_CHECKS)";
    default: return "unknown error";
  }
}

}  // extern "C"
