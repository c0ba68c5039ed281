// Per-unit budgets: grkv_compress with a budget B_u for every unit, as the
// paper pairs GRKV with layer-wise (PyramidKV) and head-wise (Ada-KV) budget
// allocations (Sec. 4.2).  The scoring step does not depend on the budget and
// runs once over all units; selection and the value (and key) step run once
// per run of consecutive units that share a budget, on that run's slice of
// the inputs, each with the same kernels as grkv_compress.  Outputs are
// packed: unit u's B_u rows start at row off_u = B_0 + ... + B_{u-1}.
#include <algorithm>
#include <vector>

#include "grkv_internal.cuh"

namespace grkv {
namespace {

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Copies a run's device status into the call's status word unless that
// already holds an error (the first error wins, as in every call).
__global__ void k_status_merge(int* status, const int* run_status) {
  const int s = *run_status;
  if (s != 0) atomicCAS(status, 0, s);
}

struct RaggedPlan {
  Shape all;                  // every unit, the largest budget (scoring only)
  std::vector<int> begin;     // first unit of each run
  std::vector<int> budget;    // its budget
  std::vector<size_t> off;    // packed row offset of each unit (U + 1 entries)
  size_t main_total;          // the scoring workspace (status word first)
  size_t run_ws;              // offset of the per-run workspace
  size_t run_total;           // its size (the largest run's)
  size_t idx_scratch;         // 16-byte aligned idx of the current run
  size_t total;
};

int plan_ragged(const grkv_params* p, const int32_t* budgets, RaggedPlan* r) {
  if (!p || (p->units > 0 && !budgets)) return GRKV_ERR_INVALID_ARG;
  grkv_params q = *p;
  int bmax = p->window;
  for (int u = 0; u < p->units; ++u) {
    if (budgets[u] < p->window || budgets[u] > p->n) return GRKV_ERR_INVALID_ARG;
    bmax = std::max(bmax, (int)budgets[u]);
  }
  q.budget = bmax;
  int rc = make_shape(&q, &r->all);
  if (rc != GRKV_OK) return rc;
  r->begin.clear();
  r->budget.clear();
  r->off.assign(1, 0);
  size_t run_total = 0, idx_max = 0;
  for (int u = 0; u < p->units; ++u) {
    r->off.push_back(r->off.back() + (size_t)budgets[u]);
    if (u == 0 || budgets[u] != budgets[u - 1]) {
      r->begin.push_back(u);
      r->budget.push_back(budgets[u]);
    }
  }
  for (size_t i = 0; i < r->begin.size(); ++i) {
    const int u1 = i + 1 < r->begin.size() ? r->begin[i + 1] : p->units;
    grkv_params rp = *p;
    rp.units = u1 - r->begin[i];
    rp.budget = r->budget[i];
    Shape s;
    if ((rc = make_shape(&rp, &s)) != GRKV_OK) return rc;
    run_total = std::max(run_total, plan_workspace(s).total);
    idx_max = std::max(idx_max, (size_t)s.U * s.B);
  }
  r->main_total = plan_workspace(r->all).total;
  r->run_ws = align256(r->main_total);
  r->run_total = run_total;
  r->idx_scratch = align256(r->run_ws + run_total);
  r->total = align256(r->idx_scratch + idx_max * sizeof(int32_t));
  return GRKV_OK;
}

}  // namespace
}  // namespace grkv

using namespace grkv;

extern "C" int grkv_compress_ragged_workspace_size(const grkv_params* p, const int32_t* budgets,
                                                   size_t* bytes) {
  RaggedPlan r;
  const int rc = plan_ragged(p, budgets, &r);
  if (rc != GRKV_OK) return rc;
  if (!bytes) return GRKV_ERR_INVALID_ARG;
  *bytes = r.total;
  return GRKV_OK;
}

extern "C" int grkv_compress_ragged(const grkv_params* p, const int32_t* budgets, const void* q,
                                    const void* k, const void* v, void* k_out, void* v_out,
                                    int32_t* idx, void* ws, size_t ws_bytes, void* stream) {
  RaggedPlan r;
  int rc = plan_ragged(p, budgets, &r);
  if (rc != GRKV_OK) return rc;
  const Shape& s = r.all;
  if (!ws) return GRKV_ERR_INVALID_ARG;
  if ((uintptr_t)ws & 15u) return GRKV_ERR_MISALIGNED;
  if (ws_bytes < r.total) return GRKV_ERR_WORKSPACE_TOO_SMALL;
  const size_t rows = r.off.back();
  auto bad = [](const void* ptr, size_t n) {
    if (n == 0) return GRKV_OK;
    if (!ptr) return GRKV_ERR_INVALID_ARG;
    return ((uintptr_t)ptr & 15u) ? GRKV_ERR_MISALIGNED : GRKV_OK;
  };
  if ((rc = bad(q, (size_t)s.U * s.m)) || (rc = bad(k, (size_t)s.U * s.n)) ||
      (rc = bad(v, (size_t)s.U * s.n)) || (rc = bad(k_out, rows)) || (rc = bad(v_out, rows)) ||
      (rc = bad(idx, rows)))
    return rc;
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  const WsLayout L = plan_workspace(s);
  if (cudaMemsetAsync(w + L.status, 0, 4, st) != cudaSuccess) return GRKV_ERR_CUDA;
  if (s.U == 0) return GRKV_OK;
  float* scores = (float*)(w + L.scores);
  float* y = (float*)(w + L.y);
  float* rstats = (float*)(w + L.rstats);
  if (launch_score_any(s, q, k, v, scores, y, rstats, w, L, st) != cudaSuccess) return GRKV_ERR_CUDA;
  const size_t es = s.dtype == GRKV_BF16 ? 2 : 4, row_bytes = (size_t)kD * es;
  char* rw = w + r.run_ws;
  int32_t* idx_run = (int32_t*)(w + r.idx_scratch);
  for (size_t i = 0; i < r.begin.size(); ++i) {
    const int u0 = r.begin[i];
    const int u1 = i + 1 < r.begin.size() ? r.begin[i + 1] : s.U;
    grkv_params rp = *p;
    rp.units = u1 - u0;
    rp.budget = r.budget[i];
    Shape rs;
    if ((rc = make_shape(&rp, &rs)) != GRKV_OK) return rc;
    const WsLayout RL = plan_workspace(rs);
    if (cudaMemsetAsync(rw + RL.status, 0, 4, st) != cudaSuccess) return GRKV_ERR_CUDA;
    const char* qb = (const char*)q + (size_t)u0 * s.m * row_bytes;
    const char* kb = (const char*)k + (size_t)u0 * s.n * row_bytes;
    const char* vb = (const char*)v + (size_t)u0 * s.n * row_bytes;
    const float* sb = scores + (size_t)u0 * s.P;
    const float* yb = y + (size_t)u0 * s.m * kD;
    const float* rb = rstats + (size_t)u0 * s.m * 2;
    char* ko = (char*)k_out + r.off[u0] * row_bytes;
    char* vo = (char*)v_out + r.off[u0] * row_bytes;
    cudaError_t e = launch_select(rs, sb, idx_run, rw, RL, st);
    if (e == cudaSuccess) e = launch_merge_any(rs, qb, kb, vb, sb, yb, rb, idx_run, ko, vo, rw, RL, st);
    if (e == cudaSuccess && rs.update_k)
      e = launch_key_step(rs, qb, kb, vb, yb, sb, idx_run, vo, ko, rw, RL, st);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(idx + r.off[u0], idx_run, (size_t)rs.U * rs.B * sizeof(int32_t),
                          cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return GRKV_ERR_CUDA;
    k_status_merge<<<1, 1, 0, st>>>((int*)(w + L.status), (const int*)(rw + RL.status));
    count_launches(1);
    if (cudaGetLastError() != cudaSuccess) return GRKV_ERR_CUDA;
  }
  return GRKV_OK;
}
