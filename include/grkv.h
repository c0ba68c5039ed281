/*
 * grkv.h — C ABI of the GRKV prefill-time KV-cache compression path.
 *
 * GRKV (arXiv 2605.31105) compresses each layer's KV cache right after its
 * prefill.  For every *unit* (one layer x KV head of one sequence) the path:
 *   1. scores every cached key with the window queries (the last w prompt
 *      queries, Sec. 3.2, Eq. 4): softmax(Q_win K^T / sqrt(d));
 *   2. keeps the B - w keys with the best span-pooled score plus the window
 *      (SnapKV-style span retention, Sec. 1-2);
 *   3. forms the full-cache target Y = A_win^full V_full (Algorithm 1);
 *   4. runs GRKV's value step: the ridge regression of Eq. 6 solved in dual
 *      (Woodbury) form, Sec. 3.4 and App. D.1, over the free retained tokens
 *      (fixed tokens, Sec. 3.4 and App. D.3, stay as they are).
 *
 * Units are independent.  Query heads are grouped onto their KV head (GQA):
 * the g query heads that read one KV head stack their w window rows into
 * m = g*w rows r = h*w + a; window slot a sits at position n - w + a.
 *
 * Layouts (row-major, contiguous, `dtype` elements unless stated):
 *   q        [U][g][w][d]      window queries
 *   k, v     [U][n][d]         full key / value caches
 *   scores   [U][n-w]  fp32    per-key prefix score c_j = sum_r A_rj
 *   y        [U][m][d] fp32    target Y
 *   row_stats[U][m][2] fp32    (M_r, L_r): row max of the logits and
 *                              sum_j exp(l_rj - M_r)
 *   idx      [U][B]    int32   retained positions, ascending; the last w are
 *                              the window n-w..n-1.  grkv_merge reports an
 *                              entry outside [0, n) as GRKV_ERR_INVALID_ARG in
 *                              the device status (and reads position 0 there)
 *   k_out, v_out [U][B][d]     compressed cache
 *
 * Ownership and ordering: every pointer except `params` and the output
 * `bytes` / `device_status` is DEVICE memory owned by the caller.  The
 * library allocates nothing, keeps no pointer after a call returns, and
 * enqueues all work asynchronously on `stream` (a cudaStream_t passed as
 * void*, NULL = legacy default stream).  Device pointers must be 16-byte
 * aligned.  Nothing is written if host-side validation fails.
 *
 * Errors: calls return GRKV_OK (0) or a negative code.  Host-detected errors
 * are returned directly.  Errors found on the device (a non-positive Cholesky
 * pivot, an expired bounded wait) are written to a status word at the start
 * of the workspace; every call clears that word first, so it reports the
 * most recent call; read it with grkv_status().
 */
#ifndef GRKV_H
#define GRKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GRKV_OK                       0
#define GRKV_ERR_INVALID_ARG         -1  /* a parameter is out of range         */
#define GRKV_ERR_UNSUPPORTED         -2  /* valid but not implemented (d != 128) */
#define GRKV_ERR_WORKSPACE_TOO_SMALL -3
#define GRKV_ERR_MISALIGNED          -4  /* a device pointer is not 16-B aligned */
#define GRKV_ERR_CUDA                -5  /* a CUDA call or launch failed          */
#define GRKV_ERR_NUMERIC             -6  /* device: Cholesky pivot <= 0 (lambda ~ 0) */
#define GRKV_ERR_TIMEOUT             -7  /* device: a bounded wait expired        */
#define GRKV_ERR_BOUNDS              -8  /* device, GRKV_CHECKS: idx breaks its contract */

#define GRKV_F32  0
#define GRKV_BF16 1

#define GRKV_POOL_MAX 0
#define GRKV_POOL_AVG 1

#define GRKV_UPDATE_K      0x1u  /* grkv_merge / grkv_compress also run the key step of
                                    Algorithm 1 at t = 0 (Sec. 3.4 "Key step", App. D.2):
                                    with the merged values V* fixed, alpha = (J_G J_G^T +
                                    lambda_k I)^-1 vec(Y - X V*) by conjugate gradients
                                    from alpha = 0 (at most cg_iters iterations, until the
                                    residual is cg_tol of ||e||; matrix-free JVP / VJP,
                                    fp32 on CUDA cores), K_out = K0 + J_G^T alpha on
                                    the free slots, K0 on the fixed ones.  V* is v_out as
                                    written (rounded to dtype).  Without it K_out = K0 */
#define GRKV_FORCE_SIMT    0x2u  /* use the portable CUDA-core kernels even for bf16 */
#define GRKV_ONE_READ_SCORE 0x4u /* tensor-core scoring in one launch per 128 window rows
                                    that reads K from HBM once: groups of CTAs interleave
                                    the statistics pass of one unit with the probability
                                    pass of the previous one, which re-reads its keys from
                                    L2.  Default: two launches per 128 rows (statistics,
                                    then probabilities), each reading K from HBM, which
                                    measures faster on GB300 */

#define GRKV_DETERMINISTIC  0x8u /* bitwise run-to-run reproducible outputs: the target Y
                                    is summed from per-CTA partials in a fixed order
                                    instead of with float atomics (costs a workspace of
                                    U x slots x m x d floats and one more kernel; selects
                                    the two-launch scoring even with GRKV_ONE_READ_SCORE).
                                    Every other step is reproducible in either mode */

#define GRKV_CHECKS        0x10u /* device-side argument checks, written to the status word:
                                    a non-finite q, k or v element -> GRKV_ERR_INVALID_ARG;
                                    an idx given to grkv_merge outside [0, n), not ascending
                                    or without the window n-w..n-1 in its last w slots ->
                                    GRKV_ERR_BOUNDS.  The kernels still run (reading in-range
                                    rows only); outputs are then unspecified.  Costs one
                                    read of q, k and v */
#define GRKV_TEST_TIMEOUT 0x80000000u /* tests only: exercises the exit of the bounded device
                                    waits.  In the tensor-core scoring kernels (either path)
                                    the first CTA withholds one arrive and the waits' budget
                                    is cut to ~2 ms: the kernel gives up, frees its tensor
                                    memory, returns, and grkv_status reports
                                    GRKV_ERR_TIMEOUT; outputs are unspecified.  Ignored by
                                    the other kernels */

typedef struct {
  int32_t units;        /* U >= 0: independent (batch x layer x KV head) problems   */
  int32_t group;        /* g >= 1: query heads per KV head                          */
  int32_t n;            /* context length, window included, n >= window             */
  int32_t d;            /* head dimension; 128 only                                 */
  int32_t window;       /* w >= 1: positions n-w..n-1, always retained              */
  int32_t budget;       /* B: window <= B <= n, window included                     */
  int32_t pool_kernel;  /* odd >= 1 (7)                                             */
  int32_t pool_type;    /* GRKV_POOL_MAX (default) or GRKV_POOL_AVG                 */
  int32_t n_sink;       /* >= 0: retained tokens j < n_sink stay fixed (4)          */
  float   beta;         /* [0, 1): floor(beta*B) best-scored retained prefix
                           tokens stay fixed (0.10)                                 */
  float   lambda_v;     /* >= 0 (may be +inf: values unchanged): ridge weight of
                           the value step, Eq. 6                                    */
  float   lambda_k;     /* >= 0, finite: ridge weight of the key step (1e-2); read
                           only under GRKV_UPDATE_K                                 */
  float   scale;        /* logit scale; 0 -> fp32(1/sqrt(d))                        */
  int32_t causal;       /* 1: window slot a sees keys j <= n-w+a; 0: all n keys      */
  int32_t dtype;        /* GRKV_BF16 or GRKV_F32 for q, k, v, k_out, v_out          */
  uint32_t flags;       /* GRKV_UPDATE_K, GRKV_FORCE_SIMT, GRKV_ONE_READ_SCORE,
                           GRKV_DETERMINISTIC, GRKV_CHECKS, GRKV_TEST_TIMEOUT */
  int32_t cg_iters;     /* 0..4096: most conjugate-gradient iterations of the key
                           step (512); read only under GRKV_UPDATE_K                */
  float   cg_tol;       /* >= 0, finite: the key step's CG stops once ||r|| <=
                           cg_tol ||e|| (1e-4); read only under GRKV_UPDATE_K       */
  int32_t steps;        /* 1..64: S, the alternating value / key steps of Algorithm 1
                           (1, the paper's setting); S > 1 needs GRKV_UPDATE_K.  Step
                           t >= 1 re-runs the value step from V0 with the retained
                           attention at the current keys K^(t), then the key step
                           linearised at K^(t) (its right-hand side gains J_G (K^(t) -
                           K0)); a unit stops early once max |K^(t+1) - K^(t)| and
                           max |V^(t+1) - V^(t)| are both <= step_tol                 */
  float   step_tol;     /* >= 0, finite: the alternation's stop test (1e-9)         */
} grkv_params;

/* Fills `p` with the defaults above for the given sizes (bf16, lambda 1e-2, CG 512 / 1e-4,
 * max pool 7, 4 sinks, beta 0.10, causal). */
void grkv_params_init(grkv_params* p, int32_t units, int32_t group, int32_t n,
                      int32_t window, int32_t budget);

/* Workspace bytes that every call below needs for `p` (the largest of them).
 * Returns GRKV_ERR_INVALID_ARG / UNSUPPORTED like the calls would. */
int grkv_workspace_size(const grkv_params* p, size_t* bytes);

/* Steps 1 and 3: window attention statistics, prefix scores and target.
 *   row_stats = (max_j l_rj, sum_j exp(l_rj - M_r)),  l_rj = scale * q_r.k_j
 *   scores[j] = sum_r exp(l_rj - M_r) / L_r  for j < n - w  (Eq. 4, summed
 *               over the window rows: SnapKV's aggregated window attention)
 *   y         = A_win^full V_full                     (Algorithm 1, target Y) */
int grkv_score(const grkv_params* p, const void* q, const void* k, const void* v,
               float* scores, float* y, float* row_stats,
               void* ws, size_t ws_bytes, void* stream);

/* Step 2: pool the prefix scores with kernel `pool_kernel` (max over the
 * in-range neighbours, or the zero-padded mean), keep the B - w largest
 * (ties to the smaller position), sort them ascending and append the window. */
int grkv_select(const grkv_params* p, const float* scores, int32_t* idx,
                void* ws, size_t ws_bytes, void* stream);

/* Step 4 given the retained set: gather K0 = K[idx], V0 = V[idx]; fixed set F
 * = retained sinks + window + the floor(beta*B) retained prefix non-sink
 * tokens with the largest scores[j] (ties to the smaller position); retained
 * attention X = softmax(Q_win K0^T * scale) over the B retained keys;
 *   R = Y - X V0,  Z = (X_G X_G^T + lambda_v I_m)^-1 R,
 *   V_out[G] = V0[G] + X_G^T Z,  V_out[F] = V0[F],  K_out = K0
 * (Algorithm 1 value step; App. D.1 dual form; App. D.3 fixed tokens).
 * Outputs are rounded to `dtype` (round to nearest even).
 * row_stats may be NULL; given (as grkv_score writes it), the tensor-core
 * path accumulates the retained softmax against the full-cache row maximum
 * in one pass over K0 instead of two (same results up to rounding; units
 * whose retained maximum lies more than 2^64 below it are recomputed with
 * two passes). */
int grkv_merge(const grkv_params* p, const void* q, const void* k, const void* v,
               const float* scores, const float* y, const float* row_stats, const int32_t* idx,
               void* k_out, void* v_out, void* ws, size_t ws_bytes, void* stream);

/* The whole path: grkv_score, grkv_select and grkv_merge with every
 * intermediate in the workspace.  Writes idx, k_out and v_out. */
int grkv_compress(const grkv_params* p, const void* q, const void* k, const void* v,
                  void* k_out, void* v_out, int32_t* idx,
                  void* ws, size_t ws_bytes, void* stream);

/* grkv_compress with a budget per unit (the paper pairs GRKV with layer-wise
 * (PyramidKV) and head-wise (Ada-KV) budget allocations, Sec. 4.2).
 * budgets: HOST array [U], window <= budgets[u] <= n; p->budget is ignored.
 * Outputs are packed: unit u's budgets[u] entries of idx and rows of k_out /
 * v_out start at row off_u = budgets[0] + ... + budgets[u-1] (idx [sum B_u]
 * int32, k_out / v_out [sum B_u][d]); each unit's results are those of
 * grkv_compress with B = budgets[u].  The scoring step runs once over all
 * units; selection and the value (and key) step run once per run of
 * consecutive units with equal budgets.  ws must hold
 * grkv_compress_ragged_workspace_size bytes; device errors of any run go to
 * its status word (grkv_status). */
int grkv_compress_ragged_workspace_size(const grkv_params* p, const int32_t* budgets,
                                        size_t* bytes);
int grkv_compress_ragged(const grkv_params* p, const int32_t* budgets, const void* q,
                         const void* k, const void* v, void* k_out, void* v_out, int32_t* idx,
                         void* ws, size_t ws_bytes, void* stream);

/* Decode-side transfer check (the paper's App. G: the normalised discrepancy
 * L_common of its loss-performance diagnostic and its held-out-query stress
 * test).  For every unit it compares the eviction-only cache (K0, V0) =
 * (K[idx], V[idx]) and the compressed cache (k_out, v_out) with the full
 * cache, through the attention outputs Y = A V of two query sets:
 *   q_win  [U][g][w][d]     the surrogate window (the same rule as grkv_score:
 *                           over a B-slot cache, window row a sees slots
 *                           j <= B - w + a when causal)
 *   q_held [U][g][held][d]  held-out decoding queries, which see every slot
 * and writes report [U][8] fp32:
 *   [0] e_win(K0,V0)  = ||Y_win_full - Y_win(K0,V0)||_F^2
 *   [1] e_win(out)    = ||Y_win_full - Y_win(k_out,v_out)||_F^2
 *   [2] e_held(K0,V0) and [3] e_held(out), the same for the held-out queries
 *   [4] ||Y_win_full||_F^2, [5] ||Y_held_full||_F^2
 *   [6] cosine between the mean window output and the mean held-out output
 *       over the full cache (the surrogate-actual similarity)
 *   [7] 1 if the compressed cache lowers the window error but raises the
 *       held-out error (the paper's failure case), else 0.
 * L_common over a set of units is sum([3]) / sum([5]).  idx, k_out and v_out
 * are laid out as grkv_compress writes them; held must satisfy 1 <= held <=
 * budget and group * held <= 256.  Uses the default scoring kernels
 * (GRKV_FORCE_SIMT and GRKV_DETERMINISTIC apply, the other flags are
 * ignored); sums in fp64; a tie of the two caches' errors is not a failure.  ws must hold
 * grkv_transfer_workspace_size bytes; device errors go to its status word,
 * read with grkv_status. */
int grkv_transfer_workspace_size(const grkv_params* p, int32_t held, size_t* bytes);
int grkv_transfer_check(const grkv_params* p, int32_t held, const void* q_win,
                        const void* q_held, const void* k, const void* v, const int32_t* idx,
                        const void* k_out, const void* v_out, float* report,
                        void* ws, size_t ws_bytes, void* stream);

/* grkv_select without a workspace.  The paper has no counterpart: this entry
 * point exists for callers that cannot give the library scratch device
 * memory, such as a plugin inside an inference engine that owns all device
 * memory through its own pool and passes plugins no workspace, or a serving
 * loop that must not call cudaMalloc on the request path (it synchronises the
 * device and fails once a pool has taken the free memory).  It allocates
 * nothing: the pooled scores go to a 16 MiB array in the library's device
 * image, which every GPU that loads the library holds until the process exits.
 * Prefixes of n - window <= 32768 positions are selected in shared memory and
 * use no scratch, at any unit count.  Longer prefixes use the array, limited
 * to units * (n - window) <= 4,194,304 floats; larger sizes return
 * GRKV_ERR_WORKSPACE_TOO_SMALL.  The first call on a device looks up the
 * array's device address (cudaGetSymbolAddress) with that device current;
 * make that first call before any stream capture.  All calls share the array
 * and it keeps the last call's contents; every element a call reads is first
 * written by the same call, so nothing needs clearing.  Calls that overlap on
 * the GPU (two streams, or two host threads) race on the array: serialise
 * them.  scores and idx are device pointers laid out as for grkv_select. */
int grkv_select_noalloc(const grkv_params* p, const float* scores, int32_t* idx, void* stream);

/* Synchronises `stream`, then stores in *device_status the device-side
 * status of the most recent call that used `ws` (GRKV_OK, GRKV_ERR_NUMERIC or
 * GRKV_ERR_TIMEOUT).  Returns GRKV_ERR_CUDA if the stream reports an error. */
int grkv_status(const void* ws, int* device_status, void* stream);

/* Static description of an error code. */
const char* grkv_strerror(int code);

/* Diagnostic with no counterpart in the paper: the number of CUDA kernels
 * this library has enqueued in the calling process so far (all calls, all
 * streams).  Lets a caller count the library's launches in a timed region. */
uint64_t grkv_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* GRKV_H */
