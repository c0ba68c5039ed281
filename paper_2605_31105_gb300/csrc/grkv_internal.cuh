// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

#include "grkv.h"

namespace grkv {

constexpr int kD = 128;          // supported head dimension
constexpr int kMaxM = 256;       // stacked window rows g*w supported
constexpr int kMaxScoreCtas = 256;  // persistent score grid bound used to size slots
constexpr int kMaxCgIters = 4096;   // bound on the key step's conjugate-gradient iterations
constexpr int kMaxSteps = 64;       // bound on the alternating steps S

// Validated problem sizes, derived once on the host.
struct Shape {
  int U, g, n, d, w, B, m;
  int P;          // prefix length n - w (scored, pooled, selectable)
  int kk;         // prefix tokens kept: B - w
  int pool_k, pool_type, n_sink, n_fix, causal, dtype;
  float lambda, scale;
  int lambda_inf; // lambda_v == +inf: values stay V0
  int tc;         // bf16, m <= 256, not forced portable: tensor-core scoring
  int tc_merge;   // ... and B <= 32768: tensor-core value merge
  int one_read;   // tensor-core scoring in one launch that reads K from HBM once
  int deterministic;  // Y summed in a fixed order (GRKV_DETERMINISTIC)
  int test_timeout;   // GRKV_TEST_TIMEOUT (tests of the bounded-wait exit)
  int checks;         // GRKV_CHECKS: device-side argument checks
  int update_k;   // key step after the value step (GRKV_UPDATE_K)
  int cg_iters;   // most conjugate-gradient iterations of the key step
  float cg_tol;   // ... until ||r|| <= cg_tol ||e||
  float lambda_k; // ridge weight of the key step
  int steps;      // S alternating value / key steps (Algorithm 1)
  float step_tol; // stop once max |K^(t+1) - K^(t)|, max |V^(t+1) - V^(t)| <= step_tol
};

// Byte offsets of the workspace regions (each 256-B aligned).
struct WsLayout {
  size_t status;  // int32 device status word
  // score path (portable kernels)
  size_t pstats;  // float2 [U][nchunk][m]      per-chunk (max, sum)
  size_t ypart;   // float  [U][nchunk][m][d]   per-chunk target partials
  int chunk, nchunk;
  // score path (tensor cores)
  size_t pstats_tc;  // float2 [U][maxc][128] pass-A statistics slots
  size_t flags_tc;   // int [U] pass-A slots written per unit
  size_t lam_tc;     // float [U][128] combined log2 row normalisers (one-read scoring)
  size_t ypart_tc;   // float [U][maxc][m][128] segment Y partials (deterministic mode)
  // select
  size_t pooled;  // float [U][P]
  // merge
  size_t xbuf;    // float [U][m][B]   retained logits, then X
  size_t flags;   // uint8 [U][B]      fixed-token flags
  size_t gram;    // acc   [U][m][m]   X_G X_G^T + lambda I, then its Cholesky factor
  size_t rz;      // acc   [U][m][d]   residual R, then Z
  size_t merge_tc;  // tensor-core merge: R/Z, Gram [U][128][128] fp32, normalisers, positions, fixed flags
  // compress intermediates
  size_t scores;  // float [U][P]
  size_t y;       // float [U][m][d]
  size_t rstats;  // float2 [U][m]
  size_t key;     // key step: CG vectors [U][C][5][m][d], X, T, T2 [U][m][B], dK [U][B][d], fixed [U][B]
  size_t total;
};

WsLayout plan_workspace(const Shape& s);

// Order-preserving map of an fp32 value to an unsigned key.
__host__ __device__ inline uint32_t order_key(float f) {
#ifdef __CUDA_ARCH__
  uint32_t b = __float_as_uint(f);
#else
  uint32_t b;
  memcpy(&b, &f, 4);
#endif
  return b ^ ((b >> 31) ? 0xFFFFFFFFu : 0x80000000u);
}

__device__ inline void set_status(int* status, int code) { atomicCAS(status, 0, code); }

// Adds n to the process-wide count of kernels this library enqueued.
void count_launches(int n);

// Launchers (all asynchronous on `st`).
cudaError_t launch_score_simt(const Shape& s, const void* q, const void* k, const void* v,
                              float* scores, float* y, float* row_stats, char* ws,
                              const WsLayout& L, cudaStream_t st);
cudaError_t launch_select(const Shape& s, const float* scores, int32_t* idx, char* ws,
                          const WsLayout& L, cudaStream_t st);
// Tensor-core window scoring (bf16, m <= 256 in blocks of 128 rows).  The
// default, launch_score_tc, runs two launches per row block that each read
// K; launch_score_pipe (GRKV_ONE_READ_SCORE) reads K once.
bool score_tc_supported(const Shape& s);
struct PipePlan {
  int ng, gs;   // CTA groups, CTAs per group
};
PipePlan score_pipe_plan(const Shape& s, int sms);
size_t score_pipe_slot_bytes(const Shape& s);
cudaError_t launch_score_pipe(const Shape& s, const void* q, const void* k, const void* v,
                              float* scores, float* y, float* row_stats, char* ws,
                              const WsLayout& L, cudaStream_t st);
size_t score_tc_pstats_bytes(const Shape& s, int* maxc, int* gu, int* rounds, int sms);
int sm_count();
cudaError_t launch_score_tc(const Shape& s, const void* q, const void* k, const void* v,
                            float* scores, float* y, float* row_stats, char* ws,
                            const WsLayout& L, int mode, cudaStream_t st);

// Tensor-core value merge (bf16, m <= 256 in 128-row blocks, B <= 32768).
bool merge_tc_supported(const Shape& s);
// The regression solve for m <= 256 (grkv_merge_tc.cu): gram [U][ld][ld]
// (N with lambda when sym = 0; raw Gram blocks, symmetrised with lambda added,
// when sym = 1), rz [U][ld][128] (R in, Z out).
cudaError_t launch_solve_dense(int U, int m, int ld, int sym, float lambda, int lambda_inf,
                               const float* gram, float* rz, int* status, cudaStream_t st);
size_t merge_tc_ws_bytes(const Shape& s);
// row_stats (nullable): the full-cache row statistics; with them the Gram
// needs one pass over the retained keys.
size_t key_ws_bytes(const Shape& s);
// The key step (GRKV_UPDATE_K) and, for S > 1, the remaining alternating
// steps; k, v are the full caches (K0 and V0 of steps t >= 1).
cudaError_t launch_key_step(const Shape& s, const void* q, const void* k, const void* v,
                            const float* y, const float* scores, const int32_t* idx,
                            void* v_out, void* k_out, char* ws, const WsLayout& L,
                            cudaStream_t st);
cudaError_t launch_merge_tc(const Shape& s, const void* q, const void* k, const void* v,
                            const float* scores, const float* y, const float* row_stats,
                            const int32_t* idx, void* k_out, void* v_out, char* ws,
                            const WsLayout& L, cudaStream_t st);

// Selection with the pooled-score scratch [U][n-w] given directly; the
// scratch is touched only when select_uses_pooled_buffer(s) holds (prefixes
// longer than the shared-memory selection takes).
bool select_uses_pooled_buffer(const Shape& s);
cudaError_t launch_select_pooled(const Shape& s, const float* scores, int32_t* idx,
                                 float* pooled, cudaStream_t st);
// Dispatch of the scoring step and of the value step to the kernels the
// shape selects (as every entry point runs them).
cudaError_t launch_score_any(const Shape& s, const void* q, const void* k, const void* v,
                             float* scores, float* y, float* row_stats, char* ws,
                             const WsLayout& L, cudaStream_t st);
cudaError_t launch_merge_any(const Shape& s, const void* q, const void* k, const void* v,
                             const float* scores, const float* y, const float* row_stats,
                             const int32_t* idx, void* k_out, void* v_out, char* ws,
                             const WsLayout& L, cudaStream_t st);
// GRKV_CHECKS: finite inputs (GRKV_ERR_INVALID_ARG) and the idx contract
// (GRKV_ERR_BOUNDS), written to the status word.
cudaError_t launch_check_inputs(const Shape& s, const void* q, const void* k, const void* v,
                                int* status, cudaStream_t st);
cudaError_t launch_check_idx(const Shape& s, const int32_t* idx, int* status, cudaStream_t st);
// Host-side parameter validation shared by the entry points.
int make_shape(const grkv_params* p, Shape* s);
cudaError_t launch_merge_simt(const Shape& s, const void* q, const void* k, const void* v,
                              const float* scores, const float* y, const int32_t* idx,
                              void* k_out, void* v_out, char* ws, const WsLayout& L,
                              cudaStream_t st);

}  // namespace grkv
