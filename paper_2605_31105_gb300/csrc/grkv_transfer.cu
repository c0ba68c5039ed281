// Decode-side transfer check (App. G of the paper: the normalised discrepancy
// of the loss-performance diagnostic and the held-out-query stress test).
//
// For every unit it compares two retained caches against the full cache: the
// eviction-only cache (K0, V0) = (K[idx], V[idx]) and the compressed cache
// (k_out, v_out).  With Y = A V the attention output of a set of queries,
//   e_win(c)  = ||Y_win_full  - Y_win(c)||_F^2   surrogate window queries,
//                                                the window rule on slots
//   e_held(c) = ||Y_held_full - Y_held(c)||_F^2  held-out decoding queries,
//                                                every slot visible
// and a unit fails when the compressed cache lowers the window error but
// raises the held-out error.  Every attention output is computed by the
// scoring path (grkv_score's kernels) on a cache of n or B slots; a gather
// kernel forms K0, V0 and a reduction kernel writes the per-unit report.
#include <algorithm>

#include "grkv_internal.cuh"

namespace grkv {
namespace {

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// K0 = K[idx], V0 = V[idx]: one row (128 elements of `es` bytes) per warp
// step, 16-byte chunks per lane.  An idx entry outside [0, n) reads row 0
// (grkv_merge reports such entries; this check only reads).
__global__ void k_gather_rows(const uint8_t* __restrict__ k, const uint8_t* __restrict__ v,
                              const int32_t* __restrict__ idx, int U, int n, int B, int es,
                              uint8_t* __restrict__ k0, uint8_t* __restrict__ v0) {
  const size_t row_bytes = (size_t)kD * es;
  const int chunks = (int)(row_bytes / 16);
  const size_t rows = (size_t)U * B;
  const int lane = threadIdx.x & 31;
  for (size_t r = (size_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32; r < rows;
       r += (size_t)gridDim.x * (blockDim.x / 32)) {
    const size_t u = r / B;
    int j = __ldg(idx + r);
    j = (unsigned)j < (unsigned)n ? j : 0;
    const uint4* ks = (const uint4*)(k + (u * n + j) * row_bytes);
    const uint4* vs = (const uint4*)(v + (u * n + j) * row_bytes);
    uint4* kd = (uint4*)(k0 + r * row_bytes);
    uint4* vd = (uint4*)(v0 + r * row_bytes);
    for (int c = lane; c < chunks; c += 32) {
      kd[c] = __ldg(ks + c);
      vd[c] = __ldg(vs + c);
    }
  }
}

// Per-unit report: [e_win_base, e_win_comp, e_held_base, e_held_comp,
// ||Y_win_full||^2, ||Y_held_full||^2, cos(mean window output, mean
// held-out output), fail].  Sums in fp64, one CTA of 256 threads per unit.
__global__ void __launch_bounds__(256) k_transfer_report(
    const float* __restrict__ yw_full, const float* __restrict__ yw_base,
    const float* __restrict__ yw_comp, const float* __restrict__ yh_full,
    const float* __restrict__ yh_base, const float* __restrict__ yh_comp, int mw, int mh,
    float* __restrict__ report) {
  __shared__ double red[8][8];
  __shared__ double sw[kD], sh[kD];
  const int u = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  double acc[6] = {0, 0, 0, 0, 0, 0};
  const size_t ow = (size_t)u * mw * kD, oh = (size_t)u * mh * kD;
  for (int i = tid; i < mw * kD; i += blockDim.x) {
    const double f = yw_full[ow + i], b = yw_base[ow + i], c = yw_comp[ow + i];
    acc[0] += (f - b) * (f - b);
    acc[1] += (f - c) * (f - c);
    acc[4] += f * f;
  }
  for (int i = tid; i < mh * kD; i += blockDim.x) {
    const double f = yh_full[oh + i], b = yh_base[oh + i], c = yh_comp[oh + i];
    acc[2] += (f - b) * (f - b);
    acc[3] += (f - c) * (f - c);
    acc[5] += f * f;
  }
  // mean output rows over the full cache
  if (tid < kD) {
    double a = 0, b = 0;
    for (int r = 0; r < mw; ++r) a += yw_full[ow + (size_t)r * kD + tid];
    for (int r = 0; r < mh; ++r) b += yh_full[oh + (size_t)r * kD + tid];
    sw[tid] = a / mw;
    sh[tid] = b / mh;
  }
  __syncthreads();
  double dots[3] = {0, 0, 0};
  if (tid < kD) {
    dots[0] = sw[tid] * sh[tid];
    dots[1] = sw[tid] * sw[tid];
    dots[2] = sh[tid] * sh[tid];
  }
  double vals[8] = {acc[0], acc[1], acc[2], acc[3], acc[4], acc[5], 0, 0};
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    double x = q < 6 ? vals[q] : 0.0;
    if (q == 6) x = dots[0];
    if (q == 7) x = dots[1];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if (lane == 0) red[q][warp] = x;
  }
  double d2 = dots[2];
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) d2 += __shfl_xor_sync(0xffffffffu, d2, o);
  __shared__ double red2[8];
  if (lane == 0) red2[warp] = d2;
  __syncthreads();
  if (tid == 0) {
    double t[8] = {0, 0, 0, 0, 0, 0, 0, 0}, n2 = 0;
    for (int w8 = 0; w8 < 8; ++w8) {
      for (int q = 0; q < 8; ++q) t[q] += red[q][w8];
      n2 += red2[w8];
    }
    float* out = report + (size_t)u * 8;
    for (int q = 0; q < 6; ++q) out[q] = (float)t[q];
    const double den = sqrt(t[7]) * sqrt(n2);
    out[6] = (float)(den > 0 ? t[6] / den : 0.0);
    out[7] = (t[1] < t[0] && t[3] > t[2]) ? 1.f : 0.f;
  }
}

// The four score shapes: window or held-out queries over the full cache or
// over a B-slot cache.  Returns GRKV_OK or the validation error.
struct TransferShapes {
  Shape win_full, held_full, win_cache, held_cache;
};

int transfer_shapes(const grkv_params* p, int32_t held, TransferShapes* t) {
  if (!p || held < 1) return GRKV_ERR_INVALID_ARG;
  grkv_params q = *p;
  q.flags &= ~GRKV_UPDATE_K;
  int rc = make_shape(&q, &t->win_full);
  if (rc != GRKV_OK) return rc;
  if (held > p->budget) return GRKV_ERR_INVALID_ARG;
  grkv_params h = q;
  h.window = held;
  h.budget = held;
  h.causal = 0;
  if ((rc = make_shape(&h, &t->held_full)) != GRKV_OK) return rc;
  grkv_params c = q;
  c.n = p->budget;
  if ((rc = make_shape(&c, &t->win_cache)) != GRKV_OK) return rc;
  grkv_params hc = h;
  hc.n = p->budget;
  if ((rc = make_shape(&hc, &t->held_cache)) != GRKV_OK) return rc;
  return GRKV_OK;
}

struct TransferLayout {
  size_t score_ws;          // the scoring workspace (its status word first)
  size_t scores, rstats;    // scratch outputs of the scoring calls
  size_t yw[3], yh[3];      // full, eviction-only, compressed
  size_t k0, v0;
  size_t total;
};

TransferLayout plan_transfer(const TransferShapes& t) {
  TransferLayout L{};
  const Shape* all[4] = {&t.win_full, &t.held_full, &t.win_cache, &t.held_cache};
  size_t score_ws = 0, pmax = 0, mmax = 0;
  for (const Shape* s : all) {
    score_ws = std::max(score_ws, plan_workspace(*s).total);
    pmax = std::max(pmax, (size_t)s->P);
    mmax = std::max(mmax, (size_t)s->m);
  }
  const Shape& s = t.win_full;
  const size_t U = (size_t)s.U, es = s.dtype == GRKV_BF16 ? 2 : 4;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + bytes);
    return at;
  };
  L.score_ws = take(score_ws);
  L.scores = take(U * pmax * 4);
  L.rstats = take(U * mmax * 8);
  for (int i = 0; i < 3; ++i) L.yw[i] = take(U * (size_t)t.win_full.m * kD * 4);
  for (int i = 0; i < 3; ++i) L.yh[i] = take(U * (size_t)t.held_full.m * kD * 4);
  L.k0 = take(U * (size_t)s.B * kD * es);
  L.v0 = take(U * (size_t)s.B * kD * es);
  L.total = off;
  return L;
}

bool aligned16(const void* ptr) { return ((uintptr_t)ptr & 15u) == 0; }

int check_ptr(const void* ptr, size_t elems) {
  if (elems == 0) return GRKV_OK;
  if (!ptr) return GRKV_ERR_INVALID_ARG;
  return aligned16(ptr) ? GRKV_OK : GRKV_ERR_MISALIGNED;
}

// Scoring of one shape into y (prefix scores and row statistics go to
// scratch), with the scoring workspace at ws.
cudaError_t score_into(const Shape& s, const void* q, const void* k, const void* v, float* y,
                       char* ws, const TransferLayout& T, cudaStream_t st) {
  const WsLayout L = plan_workspace(s);
  float* scores = (float*)(ws - T.score_ws + T.scores);
  float* rstats = (float*)(ws - T.score_ws + T.rstats);
  if (s.tc) return launch_score_tc(s, q, k, v, scores, y, rstats, ws, L, 0, st);
  return launch_score_simt(s, q, k, v, scores, y, rstats, ws, L, st);
}

}  // namespace
}  // namespace grkv

using namespace grkv;

extern "C" int grkv_transfer_workspace_size(const grkv_params* p, int32_t held, size_t* bytes) {
  TransferShapes t;
  const int rc = transfer_shapes(p, held, &t);
  if (rc != GRKV_OK) return rc;
  if (!bytes) return GRKV_ERR_INVALID_ARG;
  *bytes = plan_transfer(t).total;
  return GRKV_OK;
}

extern "C" int grkv_transfer_check(const grkv_params* p, int32_t held, const void* q_win,
                                   const void* q_held, const void* k, const void* v,
                                   const int32_t* idx, const void* k_out, const void* v_out,
                                   float* report, void* ws, size_t ws_bytes, void* stream) {
  TransferShapes t;
  int rc = transfer_shapes(p, held, &t);
  if (rc != GRKV_OK) return rc;
  const Shape& s = t.win_full;
  const TransferLayout T = plan_transfer(t);
  if (!ws) return GRKV_ERR_INVALID_ARG;
  if (!aligned16(ws)) return GRKV_ERR_MISALIGNED;
  if (ws_bytes < T.total) return GRKV_ERR_WORKSPACE_TOO_SMALL;
  const size_t U = (size_t)s.U;
  if ((rc = check_ptr(q_win, U * s.m)) != GRKV_OK || (rc = check_ptr(q_held, U * t.held_full.m)) ||
      (rc = check_ptr(k, U * s.n)) || (rc = check_ptr(v, U * s.n)) ||
      (rc = check_ptr(idx, U * s.B)) || (rc = check_ptr(k_out, U * s.B)) ||
      (rc = check_ptr(v_out, U * s.B)) || (rc = check_ptr(report, U)))
    return rc;
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  char* sw = w + T.score_ws;   // the scoring workspace; its status word is ws's first word
  if (cudaMemsetAsync(sw, 0, 4, st) != cudaSuccess) return GRKV_ERR_CUDA;
  if (s.U == 0) return GRKV_OK;
  const int es = s.dtype == GRKV_BF16 ? 2 : 4;
  float* yw[3];
  float* yh[3];
  for (int i = 0; i < 3; ++i) {
    yw[i] = (float*)(w + T.yw[i]);
    yh[i] = (float*)(w + T.yh[i]);
  }
  void* k0 = w + T.k0;
  void* v0 = w + T.v0;
  const int blocks = (int)std::min<size_t>((U * s.B + 7) / 8, 4096);
  k_gather_rows<<<blocks, 256, 0, st>>>((const uint8_t*)k, (const uint8_t*)v, idx, s.U, s.n, s.B,
                                        es, (uint8_t*)k0, (uint8_t*)v0);
  count_launches(1);
  cudaError_t e = cudaGetLastError();
  const void* kc[3] = {k, k0, k_out};
  const void* vc[3] = {v, v0, v_out};
  for (int i = 0; i < 3 && e == cudaSuccess; ++i) {
    const Shape& shw = i == 0 ? t.win_full : t.win_cache;
    const Shape& shh = i == 0 ? t.held_full : t.held_cache;
    e = score_into(shw, q_win, kc[i], vc[i], yw[i], sw, T, st);
    if (e == cudaSuccess) e = score_into(shh, q_held, kc[i], vc[i], yh[i], sw, T, st);
  }
  if (e != cudaSuccess) return GRKV_ERR_CUDA;
  k_transfer_report<<<s.U, 256, 0, st>>>(yw[0], yw[1], yw[2], yh[0], yh[1], yh[2], s.m,
                                        t.held_full.m, report);
  count_launches(1);
  return cudaGetLastError() == cudaSuccess ? GRKV_OK : GRKV_ERR_CUDA;
}
