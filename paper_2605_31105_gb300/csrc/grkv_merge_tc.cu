// GRKV value step on the tensor cores (bf16, d = 128, m <= 256, B <= 32768).
//
// Algorithm 1's value step in dual form (Sec. 3.4, App. D.1) with the fixed
// tokens of App. D.3, one unit per CTA:
//   k_merge_fixed   the fixed set (retained sinks, the window, and the n_fix
//                   retained prefix tokens with the largest scores), a flag per
//                   slot, and a stable partition of the B retained slots into
//                   "positions": the n_G non-fixed slots first, then the fixed
//                   ones, each in slot order.  The window stays last in both
//                   orders, so slot or position p is visible to window row r
//                   exactly when p <= B - w + r % w.
//   k_merge_gram    pass 1 over the slots: row max / sum of l = s Q K0^T (K0
//                   gathered with TMA gather4); pass 2 over the positions:
//                   X = softmax, R~ += Xh V0 and the Gram G += Xh XGh^T +
//                   (2 Xl) XGh^T on tcgen05 (Xh, Xl the bf16 high / low parts
//                   of X; XGh is Xh with the fixed columns zeroed, which removes
//                   them from both terms; N = (G + G^T) / 2 restores the cross
//                   terms).  Writes R = Y - R~, G and the row normalisers to the
//                   workspace.  With the full-cache row statistics only pass 2
//                   runs.
//   k_merge_solve   fp32 in shared memory: N = sym(G) + lambda I, blocked
//                   Cholesky, Z = N^-1 R by blocked triangular solves.
//   k_merge_update  over the slots: S^T = K0 Q^T (one TMEM lane per token),
//                   X_G^T (zero for fixed slots) as bf16 high / low parts back
//                   into TMEM, dV = XGh^T Zh + XGh^T Zl + XGl^T Zh with X_G^T
//                   as the TMEM A operand, V_out = V0 + dV in the gathered V0
//                   tile, and K_out = K0, V_out by TMA tile stores.
//
// The kernels rely on the idx contract of grkv.h: ascending, with the window
// n-w..n-1 in the last w slots.
#include <cmath>

#include "block_select.cuh"
#include "grkv_internal.cuh"
#include "sm100.cuh"
#include "tmap.cuh"

namespace grkv {
namespace {

using namespace sm100;

constexpr int kTile = 128;
constexpr int kRows = 128;
constexpr int kThreads = 384;    // k_merge_gram
constexpr int kThreadsU = 736;   // k_merge_update
constexpr uint32_t kTileBytes = kTile * kD * 2;   // 32 KB
constexpr int kMaxB = 32768;
constexpr long long kBudget = 1ll << 32;
constexpr int kLD = 129;   // fp32 row stride of N and R/Z in k_merge_solve

// Shared memory (offsets from a 1024-byte aligned base).  k_merge_gram: Q, a
// ring of four gathered tiles, two XGh tiles.  k_merge_update: Q, two K0
// tiles, two V0 / V_out tiles, Zh, Zl.  Both continue with the barriers.
constexpr int kRingG = 4;
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffRing = kTileBytes;
constexpr uint32_t kOffXG = kOffRing + kRingG * kTileBytes;   // gram: 2 tiles
constexpr uint32_t kOffBar = 7 * kTileBytes;
static_assert(kOffXG + 2 * kTileBytes == kOffBar, "shared-memory layout");
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;
// k_merge_solve: packed N (tri(128) + 4 floats), R/Z [128][129] fp32, 1 / L_jj, the failure flag
constexpr uint32_t kSolveSmem = ((128 * 129) / 2 + 4 + kRows * kLD + kRows + 32) * 4;

// TMEM columns.  gram: S[2] 0..255, R~ 256..383, Gram 384..511.
// update: S^T[2] (then X_G^T) 0..255, D[2] 256..511.
constexpr uint32_t kColS = 0;
constexpr uint32_t kColR = 256;
constexpr uint32_t kColG = 384;
constexpr uint32_t kColD = 256;

struct MArgs {
  int U, n, w, m, P, B, causal, n_sink, n_fix;
  float sl2, lambda;
  int lambda_inf;
  const int32_t* idx;        // [U][B]
  const float* scores;       // [U][P]
  const float* y;            // [U][m][128]
  const __nv_bfloat16* k;    // [U][n][128]
  const __nv_bfloat16* v;
  __nv_bfloat16* k_out;      // [U][B][128]
  __nv_bfloat16* v_out;
  const float* rstats;       // [U][m][2] full-cache row max / sum (natural units) or null
  float* rz;                 // [U][128][128]  R (gram) -> Z (solve)
  float* gram;               // [U][128][128]  raw Gram
  float* lam;                // [U][128]       log2 normaliser of each window row
  int32_t* src;              // [U][B]         K / V row of each position
  int32_t* ng;               // [U]            number of non-fixed slots
  int32_t* redo;             // [U]            single-pass result unusable: run two passes
  uint8_t* fixed;            // [U][B]         1 for a fixed slot
  int gram_mode;             // 0 two passes; 1 one pass against rstats; 2 two passes for redo units
  // Row blocks (m > 128): a launch takes the 128 window rows row0 .. row0+127
  // of block rb (of nrb); the per-unit arrays hold ldr rows (128 or 256):
  // rz [U][ldr][128], gram [U][ldr][ldr], lam [U][ldr], redo [U][nrb].
  int row0, rb, nrb, ldr;
  int upd_mode;              // update: 0 V_out = V0 + dV; 1 vpart = V0 + dV; 2 V_out = vpart + dV
  float* vpart;              // [U][B][128] fp32, between the update's two row blocks
  int* status;
};

struct MBars {
  uint64_t ring_full[4], ring_empty[4];
  uint64_t q_full;
  uint64_t s_full[2], s_done[2];
  uint64_t xg_full[2], xg_empty[2];
  uint64_t acc_done;
  uint64_t d_full[2], d_empty[2];
  uint64_t drain;
  uint32_t tmem;
  int abort;
  int bad;
};
static_assert(sizeof(MBars) <= 256, "barrier block");

__device__ __forceinline__ float lo_half(uint32_t h) { return __uint_as_float(h << 16); }
__device__ __forceinline__ float hi_half(uint32_t h) { return __uint_as_float(h & 0xFFFF0000u); }

// TMEM column, within a 128-column buffer, of the packed high (lo = 0) or low
// (lo = 1) parts of K rows 16kk .. 16kk+15 of an A operand written back in
// place over 32-column chunks (chunk c: high parts in 32c .. 32c+15, low parts
// in 32c+16 .. 32c+31).
__device__ __forceinline__ uint32_t xt_col(int kk, int lo) {
  return (kk >> 1) * 32 + lo * 16 + (kk & 1) * 8;
}

// mbar_wait for all lanes of a warp with one answer, so that warp-collective
// instructions after a wait are reached by all lanes or by none.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort, kBudget));
}

// Four rows (64 columns each) of a 2-D tensor map into consecutive 128-byte rows.
__device__ __forceinline__ void tma_gather4(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int r0, int r1, int r2, int r3) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6, %7}], [%2];" ::"r"(smem_u32(dst)),
      "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(r0), "r"(r1), "r"(r2), "r"(r3)
      : "memory");
}

// Producer side of a ring of R gathered tiles, run by W warps: warp pw
// (0 <= pw < W) gathers its share of the tile's 32 four-row groups (the rows
// rows_u[t*128 + row], clamped to B-1; a row outside [0, n) reads row 0) with
// TMA gather4 into the 128-byte-swizzled tile and arrives on the slot's full
// barrier (initialised with W arrivals) with its share of the transaction
// bytes, so a slot is full once every share has landed.  The issue cost of
// gather4 is paid by the issuing warp, so more warps fill a tile faster.  The
// row indices are fetched by rows() one tile ahead of load(), so their
// latency overlaps the wait for a free slot, and one fetch can serve the K and
// V tiles of the same rows.
template <int R, int W>
struct Gatherer {
  // warp pw takes the four-row groups g0(pw) .. g0(pw + 1) - 1 of the 32 in a tile
  static constexpr int g0(int pw) { return pw * (kTile / 4) / W; }
  static_assert(kTile / 4 / W <= 32 && W >= 1, "gather split");
  uint8_t* ring;
  uint64_t* full;
  uint64_t* empty;
  uint32_t use = 0;
  // lanes < the warp's group count: the four rows of group g0(pw) + lane of tile t, as map rows
  __device__ __forceinline__ void rows(const int32_t* rows_u, int B, int n, int row0, int t,
                                       int pw, int lane, int* j) const {
    if (lane < g0(pw + 1) - g0(pw)) {
      const int r = 4 * (g0(pw) + lane);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int jj = __ldg(rows_u + min(t * kTile + r + e, B - 1));
        j[e] = row0 + ((unsigned)jj < (unsigned)n ? jj : 0);
      }
    }
  }
  __device__ __forceinline__ bool load(const CUtensorMap* map, const int* j, int pw, int lane,
                                       volatile int* abort_flag) {
    const uint32_t slot = use % R;
    bool ok = true;
    if (use >= R) ok = mbar_wait(&empty[slot], (use / R - 1) & 1, abort_flag, kBudget);
    ok = __all_sync(0xffffffffu, ok);
    if (!ok) return false;
    uint8_t* dst = ring + slot * kTileBytes;
    uint64_t* bar = &full[slot];
    const int ng = g0(pw + 1) - g0(pw);
    if (lane == 0) mbar_expect_tx(bar, ng * 4 * kD * 2);
    __syncwarp();
    if (lane < ng) {
      const int r = 4 * (g0(pw) + lane);
      tma_gather4(dst + r * 128, map, bar, 0, j[0], j[1], j[2], j[3]);
      tma_gather4(dst + kTileBytes / 2 + r * 128, map, bar, 64, j[0], j[1], j[2], j[3]);
    }
    ++use;
    return true;
  }
  // every issued gather lands before the CTA can exit
  __device__ __forceinline__ void drain(volatile int* abort_flag) {
    for (uint32_t i = use > R ? use - R : 0; i < use; ++i)
      mbar_wait(&full[i % R], (i / R) & 1, abort_flag, kBudget);
  }
};

// ring_empty_count: arrivals that release a ring slot; group_count: threads
// of the compute warps that arrive on s_done, xg_full and d_empty.
__device__ __forceinline__ void init_common(MBars* bars, int warp, uint32_t ring_empty_count,
                                            uint32_t group_count, uint32_t epi_count) {
  if (threadIdx.x == 0) {
    for (int i = 0; i < 4; ++i) {
      mbar_init(&bars->ring_full[i], 3);   // one expect_tx arrival per gathering warp
      mbar_init(&bars->ring_empty[i], ring_empty_count);
    }
    mbar_init(&bars->q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_done[i], group_count);
      mbar_init(&bars->xg_full[i], group_count);
      mbar_init(&bars->xg_empty[i], 1);
      mbar_init(&bars->d_full[i], 1);
      mbar_init(&bars->d_empty[i], epi_count);
    }
    mbar_init(&bars->acc_done, 1);
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    bars->bad = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem, 512);
    tmem_relinquish();
  }
}

// S = Q K0^T for one gathered tile into TMEM columns s_col (issued by one thread).
__device__ __forceinline__ void issue_s(uint32_t s_tmem, uint32_t qa, uint32_t ka) {
  const uint32_t id_s = idesc_bf16(kRows, kTile, 0, 0);
#pragma unroll
  for (int kk = 0; kk < kD / 16; ++kk) {
    const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
    mma_bf16(s_tmem, sw128_desc(qa + off, 16, 1024), sw128_desc(ka + off, 16, 1024), id_s, kk > 0);
  }
}

__device__ __forceinline__ void store_row_chunk(uint8_t* tile, int row, int C, const uint32_t* w) {
  // row `row`, tokens 32C..32C+31 of a SW128 tile of 128-byte rows: token
  // block C/2, 16-byte chunks (C&1)*4 .. +3
#pragma unroll
  for (int qq = 0; qq < 4; ++qq)
    *(uint4*)(tile + (C >> 1) * (kTileBytes / 2) + sw128_offset(row, (C & 1) * 4 + qq)) =
        make_uint4(w[4 * qq], w[4 * qq + 1], w[4 * qq + 2], w[4 * qq + 3]);
}

// One 32-position chunk of a gram tile whose positions are all non-fixed (and
// so visible): Xh to TMEM (the A operand of R~ and of the Gram's first term),
// XGh = Xh to shared memory (the Gram's B operand) and 2 (X - Xh) returned (it
// goes to TMEM once the S columns it overwrites are read).
template <int C>
__device__ __forceinline__ void gram_chunk_fast(const float* v, float sl2, float lam,
                                                uint32_t sbase, uint8_t* xg, int row,
                                                uint32_t* lo, float& vmax, float& xsum) {
  uint32_t hi[16];
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    const float x0 = fast_exp2(fmaf(v[e], sl2, -lam)), x1 = fast_exp2(fmaf(v[e + 1], sl2, -lam));
    vmax = fmaxf(vmax, fmaxf(v[e], v[e + 1]));
    xsum += x0 + x1;
    const uint32_t h = pack_bf16(x0, x1);
    hi[e / 2] = h;
    lo[e / 2] = pack_bf16(2.f * (x0 - lo_half(h)), 2.f * (x1 - hi_half(h)));
  }
  tmem_st16(sbase + C * 16, hi);
  store_row_chunk(xg, row, C, hi);
}
// The same for a tile with fixed or invisible positions: X = 0 past vlim,
// XGh = 0 from position ng on; XGh is written only when the tile has
// non-fixed positions (want_g).
template <int C>
__device__ __forceinline__ void gram_chunk_masked(const float* v, int p0, int vlim, int ng,
                                                  float sl2, float lam, uint32_t sbase,
                                                  uint8_t* xg, int row, uint32_t* lo,
                                                  bool want_g, float& vmax, float& xsum) {
  uint32_t hi[16], ghi[16];
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    const int p = p0 + C * 32 + e;
    const float x0 = p <= vlim ? fast_exp2(fmaf(v[e], sl2, -lam)) : 0.f;
    const float x1 = p + 1 <= vlim ? fast_exp2(fmaf(v[e + 1], sl2, -lam)) : 0.f;
    vmax = fmaxf(vmax, fmaxf(p <= vlim ? v[e] : -INFINITY, p + 1 <= vlim ? v[e + 1] : -INFINITY));
    xsum += x0 + x1;
    const uint32_t h = pack_bf16(x0, x1);
    hi[e / 2] = h;
    lo[e / 2] = pack_bf16(2.f * (x0 - lo_half(h)), 2.f * (x1 - hi_half(h)));
    ghi[e / 2] = (p < ng ? (h & 0xFFFFu) : 0u) | (p + 1 < ng ? (h & 0xFFFF0000u) : 0u);
  }
  tmem_st16(sbase + C * 16, hi);
  if (want_g) store_row_chunk(xg, row, C, ghi);
}

// Online max / sum of exp2 over one 32-column chunk (log2 units); positions
// past vlim are skipped when kMasked.
template <bool kMasked>
__device__ __forceinline__ void stats32(float* v, int p0, int vlim, float sl2, float& M, float& L) {
  if (kMasked) {
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (p0 + e > vlim) v[e] = -INFINITY;
  }
  float m16[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) m16[e] = fmaxf(v[e], v[e + 16]);
#pragma unroll
  for (int h = 8; h >= 1; h >>= 1)
#pragma unroll
    for (int e = 0; e < h; ++e) m16[e] = fmaxf(m16[e], m16[e + h]);
  if (kMasked && m16[0] == -INFINITY) return;
  const float cm = m16[0] * sl2;
  if (cm > M) {
    L *= fast_exp2(M - cm);
    M = cm;
  }
  float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < 32; ++e) s[e & 3] += fast_exp2(fmaf(v[e], sl2, -M));
  L += (s[0] + s[1]) + (s[2] + s[3]);
}

// ======================================================== k_merge_fixed
// One CTA (256 threads) per unit; shared memory holds one key per slot.
__global__ void __launch_bounds__(256) k_merge_fixed(MArgs a) {
  extern __shared__ uint32_t fkey[];   // [B] candidate keys, 0 = not a candidate
  __shared__ int hist[256], sh[64];
  const int tid = threadIdx.x, nt = blockDim.x;
  const int u = blockIdx.x, B = a.B;
  const int32_t* idx_u = a.idx + (size_t)u * B;
  const float* sc_u = a.scores + (size_t)u * a.P;
  // Candidates for the score-ranked part: retained prefix tokens past the sinks.
  // Their scores are non-negative, so every key is above 0.
  // An idx entry outside [0, n) is reported and read as position 0.
  auto pos = [&](int i) {
    const int j = __ldg(idx_u + i);
    return (unsigned)j < (unsigned)a.n ? j : 0;
  };
  int nc = 0;
  for (int i = tid; i < B; i += nt) {
    if ((unsigned)__ldg(idx_u + i) >= (unsigned)a.n) set_status(a.status, GRKV_ERR_INVALID_ARG);
    const int j = pos(i);
    const bool cand = j >= a.n_sink && j < a.P;
    fkey[i] = cand ? max(order_key(__ldg(sc_u + j)), 1u) : 0u;
    nc += cand;
  }
  __syncthreads();
  int ncand;
  (void)block_exclusive_scan(nc, sh + 8, &ncand);
  const int nf = min(a.n_fix, ncand);
  uint32_t tau = 0xFFFFFFFFu;
  int need_eq = 0;
  if (nf > 0) {
    auto get = [&](int i, uint32_t* key) {
      *key = fkey[i];
      return *key != 0u;
    };
    block_kth_largest(get, B, nf, hist, sh, &tau, &need_eq);
  }
  // fixed: not a candidate, above tau, or among the first need_eq ties
  const int seg = (B + nt - 1) / nt;
  const int lo = min(B, tid * seg), hi = min(B, lo + seg);
  int eq = 0;
  for (int i = lo; i < hi; ++i) eq += (fkey[i] == tau);
  int tot;
  int er = block_exclusive_scan(eq, sh + 8, &tot);
  int keep = 0;
  for (int i = lo; i < hi; ++i) {
    const uint32_t kx = fkey[i];
    bool fixed = kx == 0u || kx > tau;
    if (kx == tau) fixed = er++ < need_eq;
    fkey[i] = fixed ? 1u : 0u;   // each thread rewrites only its own segment
    a.fixed[(size_t)u * B + i] = fixed ? 1 : 0;
    keep += !fixed;
  }
  int ng;
  const int gpos = block_exclusive_scan(keep, sh + 8, &ng);
  int g = gpos;
  for (int i = lo; i < hi; ++i) {
    const int at = fkey[i] ? ng + (i - g) : g;
    g += !fkey[i];
    a.src[(size_t)u * B + at] = pos(i);
  }
  if (tid == 0) a.ng[u] = ng;
}

// ======================================================== k_merge_gram
// Roles (384 threads): warp 0 the Q load; warp 1 MMA issue; warps 0, 2, 3 the gathers;
// warps 4-7 and 8-11 two compute groups (one thread per window row / TMEM
// lane) taking alternate jobs.  Job k < T: statistics of slot tile k;
// T <= k < 2T: R~ and Gram of position tile k - T.  Ring loads: K of each
// pass-1 job, then K and V of each pass-2 job.
//
// gram_mode 1 (the full-cache row statistics are known) runs only the second
// pass, with X accumulated against the full row maximum M_r instead of the
// retained one: X' = exp2(l - M_r) = X L'_r with L'_r = sum of X' over the
// visible retained keys, so R = Y - R~'/L'_r and G_ij = G'_ij/(L'_i L'_j).  The
// retained maximum is at most M_r; if it is more than 64 (log2 units) below
// it for some row, or L' underflows, the unit is flagged and gram_mode 2
// recomputes it with both passes.
__global__ void __launch_bounds__(kThreads, 1)
    k_merge_gram(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, MArgs a) {
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  MBars* bars = (MBars*)(sm + kOffBar);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x, B = a.B, T = (B + kTile - 1) / kTile;
  if (a.gram_mode == 2 && __ldg(a.redo + u * a.nrb + a.rb) == 0) return;   // the single pass was valid
  const bool single = a.gram_mode == 1;
  const int k0 = single ? T : 0;   // first job
  const int ng = __ldg(a.ng + u);
  init_common(bars, warp, 1, 128, 128);   // ring slots are released by the MMA
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem;
  volatile int* abort_flag = &bars->abort;

  if (warp == 0 || warp == 2 || warp == 3) {
    if (warp == 0 && lane == 0) {
      prefetch_tensormap(&tmQ);
      mbar_expect_tx(&bars->q_full, kTileBytes);
      const uint64_t pol = l2_evict_last();
      tma_load_3d(sm + kOffQ, &tmQ, &bars->q_full, 0, a.row0, u, pol);
      tma_load_3d(sm + kOffQ + kTileBytes / 2, &tmQ, &bars->q_full, 64, a.row0, u, pol);
    }
    __syncwarp();
    // the gathers: warps 0, 2 and 3 (three SM sub-partitions)
    const int32_t* idx_u = a.idx + (size_t)u * B;
    const int32_t* src_u = a.src + (size_t)u * B;
    const int row0 = u * a.n;   // first row of this unit in the 2-D K / V maps
    const int pw = warp == 0 ? 0 : warp - 1;
    Gatherer<kRingG, 3> gt{sm + kOffRing, bars->ring_full, bars->ring_empty};
    // job k < T reads K at the slots' rows, job k >= T K and V at the positions' rows
    auto rows_of = [&](int k, int* j) {
      gt.rows(k < T ? idx_u : src_u, B, a.n, row0, k < T ? k : k - T, pw, lane, j);
    };
    int jn[4];
    if (k0 < 2 * T) rows_of(k0, jn);
    bool ok = true;
    for (int k = k0; k < 2 * T && ok; ++k) {
      const int j[4] = {jn[0], jn[1], jn[2], jn[3]};
      if (k + 1 < 2 * T) rows_of(k + 1, jn);
      ok = gt.load(&tmK, j, pw, lane, abort_flag);
      if (ok && k >= T) ok = gt.load(&tmV, j, pw, lane, abort_flag);
    }
    gt.drain(abort_flag);
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_r = idesc_bf16(kRows, kD, 0, 1);     // R~ += Xh V0 (V0 MN-major)
      const uint32_t id_g = idesc_bf16(kRows, kRows, 0, 0);  // G += A XGh^T
      bool ok = mbar_wait(&bars->q_full, 0, abort_flag, kBudget);
      const uint32_t qa = smem_u32(sm + kOffQ);
      uint32_t use = 0;
      int pend = -1;
      uint32_t pend_v = 0;
      bool g_started = false;
      auto issue_rg = [&](int kp, uint32_t vuse) -> bool {
        const int t = kp - T, b = (kp - k0) & 1, xb = t & 1;
        bool w = mbar_wait(&bars->s_done[b], ((kp - k0) >> 1) & 1, abort_flag, kBudget);
        if (w) w = mbar_wait(&bars->xg_full[xb], (t >> 1) & 1, abort_flag, kBudget);
        if (w)
          w = mbar_wait(&bars->ring_full[vuse % kRingG], (vuse / kRingG) & 1, abort_flag, kBudget);
        if (!w) return false;
        tc_fence_after();
        const uint32_t va = smem_u32(sm + kOffRing + (vuse % kRingG) * kTileBytes);
        const uint32_t xa = smem_u32(sm + kOffXG + xb * kTileBytes);
        const uint32_t hi = tmem + kColS + b * kTile, lo2 = hi + 64;
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk)
          mma_bf16_ts(tmem + kColR, hi + kk * 8,
                      sw128_desc(va + kk * 2048, kTileBytes / 2, 1024), id_r, (t > 0 || kk > 0));
        if (t * kTile < ng) {   // the tile has non-fixed positions
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
            mma_bf16_ts(tmem + kColG, hi + kk * 8, sw128_desc(xa + off, 16, 1024), id_g,
                        (g_started || kk > 0));
          }
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
            mma_bf16_ts(tmem + kColG, lo2 + kk * 8, sw128_desc(xa + off, 16, 1024), id_g, 1);
          }
          g_started = true;
        }
        mma_commit(&bars->ring_empty[vuse % kRingG]);
        mma_commit(&bars->xg_empty[xb]);
        return true;
      };
      for (int k = k0; k < 2 * T && ok; ++k) {
        const int jk = k - k0, b = jk & 1;
        const uint32_t kuse = use++;
        ok = mbar_wait(&bars->ring_full[kuse % kRingG], (kuse / kRingG) & 1, abort_flag, kBudget);
        if (ok && jk >= 2) ok = mbar_wait(&bars->s_done[b], ((jk >> 1) - 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
        issue_s(tmem + kColS + b * kTile, qa,
                smem_u32(sm + kOffRing + (kuse % kRingG) * kTileBytes));
        mma_commit(&bars->ring_empty[kuse % kRingG]);
        mma_commit(&bars->s_full[b]);
        uint32_t vuse = 0;
        if (k >= T) vuse = use++;
        if (pend >= 0) {
          ok = issue_rg(pend, pend_v);
          pend = -1;
        }
        if (k >= T) {
          pend = k;
          pend_v = vuse;
        }
      }
      if (ok && pend >= 0) ok = issue_rg(pend, pend_v);
      mma_commit(&bars->acc_done);
      mma_commit(&bars->drain);
      mbar_wait(&bars->drain, 0, abort_flag, kBudget);
    }
  } else if (warp >= 4) {
    const int wg = (warp - 4) >> 2, q = warp & 3, row = q * 32 + lane;
    const int grow = a.row0 + row;   // window row of the stacked m
    const bool row_ok = grow < a.m;
    // slots / positions past vlim are invisible to this row (and so are those >= B)
    const int vlim = !row_ok ? -1 : (a.causal ? B - a.w + grow % a.w : B - 1);
    const int open = B - a.w;   // below this everything is visible to every window row
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    float M = -INFINITY, L = 0.f, lam = INFINITY;
    float vmax = -INFINITY, xsum = 0.f;   // visible retained logits (raw) and sum of X
    if (single && row_ok) lam = __ldg(a.rstats + ((size_t)u * a.m + grow) * 2) * 1.4426950408889634f;
    bool ok = true;
    for (int k = k0; k < 2 * T; ++k) {
      if (k == T && !single) {
        // both groups combine their statistics (reached even after an abort);
        // the XGh tiles are not in use yet
        float2* comb = (float2*)(sm + kOffXG);
        comb[wg * kRows + row] = make_float2(M, L);
        named_bar(4, 256);
        const float2 o = comb[(wg ^ 1) * kRows + row];
        named_bar(4, 256);
        if (o.x != -INFINITY) {
          if (o.x > M) {
            L = L * fast_exp2(M - o.x) + o.y;
            M = o.x;
          } else {
            L += o.y * fast_exp2(o.x - M);
          }
        }
        lam = (row_ok && L > 0.f) ? M + __log2f(L) : INFINITY;
        if (wg == 0) a.lam[(size_t)u * a.ldr + grow] = lam;
      }
      if (!ok) {
        if (k < T) continue;
        break;
      }
      if (((k - k0) & 1) != wg) continue;
      const int b = (k - k0) & 1, t = k < T ? k : k - T, p0 = t * kTile;
      ok = mbar_wait(&bars->s_full[b], ((k - k0) >> 1) & 1, abort_flag, kBudget);
      if (!ok) continue;
      tc_fence_after();
      const uint32_t sbase = lane_addr + kColS + b * kTile;
      float va[32], vb[32];
      if (k < T) {
        // warp-uniform: the TMEM loads below are .sync.aligned
        const bool masked = __any_sync(0xffffffffu, !row_ok) || p0 + kTile > open + 1;
        tmem_ld32f(sbase, va);
        tmem_wait32(va);
        tmem_ld32f(sbase + 32, vb);
        if (masked) {
          stats32<true>(va, p0, vlim, a.sl2, M, L);
          tmem_wait32(vb);
          tmem_ld32f(sbase + 64, va);
          stats32<true>(vb, p0 + 32, vlim, a.sl2, M, L);
          tmem_wait32(va);
          tmem_ld32f(sbase + 96, vb);
          stats32<true>(va, p0 + 64, vlim, a.sl2, M, L);
          tmem_wait32(vb);
          tc_fence_before();
          mbar_arrive(&bars->s_done[b]);
          stats32<true>(vb, p0 + 96, vlim, a.sl2, M, L);
        } else {
          stats32<false>(va, p0, vlim, a.sl2, M, L);
          tmem_wait32(vb);
          tmem_ld32f(sbase + 64, va);
          stats32<false>(vb, p0 + 32, vlim, a.sl2, M, L);
          tmem_wait32(va);
          tmem_ld32f(sbase + 96, vb);
          stats32<false>(va, p0 + 64, vlim, a.sl2, M, L);
          tmem_wait32(vb);
          tc_fence_before();
          mbar_arrive(&bars->s_done[b]);
          stats32<false>(vb, p0 + 96, vlim, a.sl2, M, L);
        }
      } else {
        const int xb = t & 1;
        if (t >= 2) ok = mbar_wait(&bars->xg_empty[xb], ((t >> 1) - 1) & 1, abort_flag, kBudget);
        if (!ok) continue;
        uint8_t* xg = sm + kOffXG + xb * kTileBytes;
        // 2 (X - Xh) goes to TMEM columns 64..127, which hold S chunks 2 and 3:
        // chunks 0 and 1 are written once chunk 2 is read, 2 and 3 once chunk 3 is
        uint32_t lo0[16], lo1[16], lo2[16], lo3[16];
        tmem_ld32f(sbase, va);
        tmem_wait32(va);
        tmem_ld32f(sbase + 32, vb);
        if (__all_sync(0xffffffffu, row_ok) && p0 + kTile <= ng) {
          gram_chunk_fast<0>(va, a.sl2, lam, sbase, xg, row, lo0, vmax, xsum);
          tmem_wait32(vb);
          tmem_ld32f(sbase + 64, va);
          gram_chunk_fast<1>(vb, a.sl2, lam, sbase, xg, row, lo1, vmax, xsum);
          tmem_wait32(va);
          tmem_st16(sbase + 64, lo0);
          tmem_st16(sbase + 80, lo1);
          tmem_ld32f(sbase + 96, vb);
          gram_chunk_fast<2>(va, a.sl2, lam, sbase, xg, row, lo2, vmax, xsum);
          tmem_wait32(vb);
          tmem_st16(sbase + 96, lo2);
          gram_chunk_fast<3>(vb, a.sl2, lam, sbase, xg, row, lo3, vmax, xsum);
        } else {
          const bool want_g = p0 < ng;
          gram_chunk_masked<0>(va, p0, vlim, ng, a.sl2, lam, sbase, xg, row, lo0, want_g, vmax, xsum);
          tmem_wait32(vb);
          tmem_ld32f(sbase + 64, va);
          gram_chunk_masked<1>(vb, p0, vlim, ng, a.sl2, lam, sbase, xg, row, lo1, want_g, vmax, xsum);
          tmem_wait32(va);
          tmem_st16(sbase + 64, lo0);
          tmem_st16(sbase + 80, lo1);
          tmem_ld32f(sbase + 96, vb);
          gram_chunk_masked<2>(va, p0, vlim, ng, a.sl2, lam, sbase, xg, row, lo2, want_g, vmax, xsum);
          tmem_wait32(vb);
          tmem_st16(sbase + 96, lo2);
          gram_chunk_masked<3>(vb, p0, vlim, ng, a.sl2, lam, sbase, xg, row, lo3, want_g, vmax, xsum);
        }
        tmem_st16(sbase + 112, lo3);
        tmem_st_wait();
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&bars->s_done[b]);
        mbar_arrive(&bars->xg_full[xb]);
      }
    }
    // R = Y - R~ and the raw Gram rows to the workspace, half the columns per group
    if (ok) ok = mbar_wait(&bars->acc_done, 0, abort_flag, kBudget);
    tc_fence_after();
    float ci = 1.f;   // 1 / L'_row in the single pass
    float* cs = (float*)(sm + kOffXG) + 2 * 2 * kRows;   // [128] after the float2 pairs
    if (single) {
      // combine the groups' sums and maxima (the XGh tiles are free now)
      float2* comb = (float2*)(sm + kOffXG);
      comb[wg * kRows + row] = make_float2(vmax, xsum);
      named_bar(4, 256);
      const float2 o = comb[(wg ^ 1) * kRows + row];
      const float lsum = xsum + o.y, vm = fmaxf(vmax, o.x);
      const bool bad = row_ok && !(lsum > 0.f && lam - vm * a.sl2 <= 64.f);
      if (bad) bars->bad = 1;
      ci = (row_ok && lsum > 0.f) ? 1.f / lsum : 0.f;
      if (wg == 0) {
        cs[row] = ci;
        a.lam[(size_t)u * a.ldr + grow] = (row_ok && lsum > 0.f) ? lam + __log2f(lsum) : INFINITY;
      }
      named_bar(4, 256);
      if (tid == 128) a.redo[u * a.nrb + a.rb] = bars->bad;
      if (bars->bad) ok = false;   // gram_mode 2 redoes this unit; not a failure
    }
    if (ok) {
      float* R = a.rz + ((size_t)u * a.ldr + grow) * kD;
      float* G = a.gram + ((size_t)u * a.ldr + grow) * a.ldr + a.row0;   // the diagonal block
      const float* yr = a.y + ((size_t)u * a.m + (row_ok ? grow : 0)) * kD;
#pragma unroll 1
      for (int c = 2 * wg; c < 2 * wg + 2; ++c) {
        float v[32];
        tmem_ld32f(lane_addr + kColR + c * 32, v);
        tmem_wait32(v);
#pragma unroll
        for (int e = 0; e < 32; e += 4) {
          const float4 yv = row_ok ? __ldg((const float4*)(yr + c * 32 + e))
                                   : make_float4(0.f, 0.f, 0.f, 0.f);
          *(float4*)(R + c * 32 + e) =
              row_ok ? make_float4(yv.x - ci * v[e], yv.y - ci * v[e + 1], yv.z - ci * v[e + 2],
                                   yv.w - ci * v[e + 3])
                     : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        tmem_ld32f(lane_addr + kColG + c * 32, v);
        tmem_wait32(v);
        if (ng == 0) {   // no Gram MMA ran
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = 0.f;
        }
        if (single) {
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] *= ci * cs[c * 32 + e];
        }
#pragma unroll
        for (int e = 0; e < 32; e += 4)
          *(float4*)(G + c * 32 + e) = make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]);
      }
    }
    if (!ok && row == 0 && !bars->bad) set_status(a.status, GRKV_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// ======================================================== k_merge_solve
// N lives in shared memory as a packed lower triangle (row i at tri(i)), so
// two CTAs fit on an SM.  The register-resident pieces of the blocked
// Cholesky and of the triangular solves are separate (non-inlined) functions
// so that their 32-element arrays stay in registers.
__host__ __device__ constexpr int tri(int i) { return (i * (i + 1)) >> 1; }
constexpr int kTri = tri(kRows) + 4;   // packed N, padded to 16 bytes
constexpr int kSolveThreads = 256;

// Factors the 32 x 32 diagonal block at k0 (right-looking; lane l holds row
// k0 + l) and stores 1 / L_jj.  Returns true on a non-positive pivot.
__device__ __noinline__ bool chol_diag(float* N, float* dinv, int k0, int lane) {
  const int rb = tri(k0 + lane) + k0;
  float x[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) x[j] = j <= lane ? N[rb + j] : 0.f;
  bool bad = false;
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    const float dkk = __shfl_sync(0xffffffffu, x[k], k);
    bad |= !(dkk > 0.f);
    const float inv = dkk > 0.f ? rsqrtf(dkk) : 0.f;   // 1 / L_kk
    const float piv = dkk * inv;                         // L_kk
    x[k] = lane == k ? piv : (lane > k ? x[k] * inv : x[k]);
    const float lk = x[k];
#pragma unroll
    for (int j = k + 1; j < 32; ++j) {
      const float ljk = __shfl_sync(0xffffffffu, x[k], j);
      x[j] = lane >= j ? x[j] - lk * ljk : x[j];
    }
    if (lane == 0) dinv[k0 + k] = inv;
  }
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (j <= lane) N[rb + j] = x[j];
  return bad;
}

// Row i of the panel below the diagonal block at k0: L_i,k0.. = A_i,k0.. L_kk^-T.
__device__ __noinline__ void chol_panel_row(float* N, const float* dinv, int k0, int i) {
  const int rb = tri(i) + k0;
  float x[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) x[j] = N[rb + j];
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float* lj = N + tri(k0 + j) + k0;
    float s0 = x[j], s1 = 0.f;
#pragma unroll
    for (int p = 0; p < j; ++p) {
      if (p & 1) s1 += x[p] * lj[p];
      else s0 -= x[p] * lj[p];
    }
    x[j] = (s0 - s1) * dinv[k0 + j];
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) N[rb + j] = x[j];
}

// Inverts the lower-triangular 32 x 32 diagonal block at k0 in place: lane l
// computes column l of L_bb^-1 by forward substitution (its entries above the
// diagonal come out zero) and writes it once every lane has read the block.
__device__ __noinline__ void tri_inv_diag(float* N, const float* dinv, int k0, int lane) {
  float x[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const float* li = N + tri(k0 + i) + k0;
    float s0 = i == lane ? 1.f : 0.f, s1 = 0.f;
#pragma unroll
    for (int k = 0; k < i; ++k) {
      if (k & 1) s1 += li[k] * x[k];
      else s0 -= li[k] * x[k];
    }
    x[i] = (s0 - s1) * dinv[k0 + i];
  }
  __syncwarp();
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (i >= lane) N[tri(k0 + i) + k0 + lane] = x[i];
}

// N = (G + G^T) / 2 + lambda I on the window rows (identity on padding rows),
// Cholesky N = L L^T in 32-row blocks, then Z = L^-T L^-1 R by block
// substitution with the inverted diagonal blocks; fp32 in shared memory.  A non-positive pivot reports GRKV_ERR_NUMERIC and leaves Z = 0
// (values stay V0); lambda = +inf also gives Z = 0.
__global__ void __launch_bounds__(kSolveThreads, 2) k_merge_solve(MArgs a) {
  extern __shared__ __align__(16) float ssm[];
  float* N = ssm;                   // packed lower triangle
  float* R = N + kTri;              // [128][kLD]: G first, then R, then Z
  float* dinv = R + kRows * kLD;    // [128]
  int* fail = (int*)(dinv + kRows);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nt = blockDim.x;
  const int u = blockIdx.x, m = a.m;
  float* RZ = a.rz + (size_t)u * kRows * kD;
  if (a.lambda_inf) {
    for (int p = tid; p < kRows * kD / 4; p += nt) ((float4*)RZ)[p] = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  if (tid == 0) *fail = 0;
  // G into the R buffer with every load of a half in flight at once (one
  // element per lane and step: conflict-free stores into the padded rows)
  const float* Gs = a.gram + (size_t)u * kRows * kRows;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    float g[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) g[k] = __ldg(Gs + tid + kSolveThreads * (32 * h + k));
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const int p = tid + kSolveThreads * (32 * h + k);
      R[(p >> 7) * kLD + (p & 127)] = g[k];
    }
  }
  // R's loads are issued before the symmetric part is formed and stored after
  float rr[64];
#pragma unroll
  for (int k = 0; k < 64; ++k) rr[k] = __ldg(RZ + tid + kSolveThreads * k);
  __syncthreads();
  for (int i = warp; i < kRows; i += kSolveThreads / 32)
    for (int j = lane; j <= i; j += 32) {
      float val;
      if (i >= m || j >= m) val = (i == j) ? 1.f : 0.f;
      else if (i == j) val = R[i * kLD + i] + a.lambda;
      else val = 0.5f * (R[i * kLD + j] + R[j * kLD + i]);
      N[tri(i) + j] = val;
    }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < 64; ++k) {
    const int p = tid + kSolveThreads * k;
    R[(p >> 7) * kLD + (p & 127)] = rr[k];
  }
  for (int kb = 0; kb < kRows / 32; ++kb) {
    const int k0 = kb * 32;
    if (warp == 0 && chol_diag(N, dinv, k0, lane) && lane == 0) *fail = 1;
    __syncthreads();
    for (int i = k0 + 32 + tid; i < kRows; i += nt) chol_panel_row(N, dinv, k0, i);
    __syncthreads();
    // trailing update of the lower triangle in 4x4 register blocks
    const int k1 = k0 + 32, t4 = (kRows - k1) / 4, nb = t4 * (t4 + 1) / 2;
    for (int t = tid; t < nb; t += nt) {
      int bi = (int)((sqrtf(8.f * t + 1.f) - 1.f) * 0.5f);
      while ((bi + 1) * (bi + 2) / 2 <= t) ++bi;
      while (bi * (bi + 1) / 2 > t) --bi;
      const int i = k1 + 4 * bi, j = k1 + 4 * (t - bi * (bi + 1) / 2);
      float acc[4][4] = {};
      const float* li[4];
      const float* lj[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        li[r] = N + tri(i + r) + k0;
        lj[r] = N + tri(j + r) + k0;
      }
#pragma unroll 4
      for (int pp = 0; pp < 32; ++pp) {
        float vi[4], vj[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          vi[r] = li[r][pp];
          vj[r] = lj[r][pp];
        }
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += vi[r] * vj[c];
      }
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (j + c <= i + r) N[tri(i + r) + j + c] -= acc[r][c];
    }
    __syncthreads();
  }
  if (*fail) {
    if (tid == 0) set_status(a.status, GRKV_ERR_NUMERIC);
    for (int p = tid; p < kRows * kD / 4; p += nt) ((float4*)RZ)[p] = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  // the diagonal blocks of L are replaced by their inverses (one warp each)
  if (warp < kRows / 32) tri_inv_diag(N, dinv, warp * 32, lane);
  __syncthreads();
  // forward: L W = R in 32-row blocks, W_b = L_bb^-1 (R_b - L_b,<b W_<b);
  // thread: rows 4 rg .. 4 rg + 3 of the block, columns e + 32 c
  const int rg = warp, e = lane;
  for (int ib = 0; ib < kRows / 32; ++ib) {
    const int i0 = ib * 32;
    {
      float acc[4][4] = {};
      const float* lr[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) lr[r] = N + tri(i0 + 4 * rg + r) + i0;
#pragma unroll 4
      for (int kx = 0; kx < 4 * rg + 4; ++kx) {
        float l[4], z[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) l[r] = kx <= 4 * rg + r ? lr[r][kx] : 0.f;
#pragma unroll
        for (int c = 0; c < 4; ++c) z[c] = R[(i0 + kx) * kLD + e + 32 * c];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += l[r] * z[c];
      }
      __syncthreads();
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) R[(i0 + 4 * rg + r) * kLD + e + 32 * c] = acc[r][c];
    }
    __syncthreads();
    // rows below: 4 rows x 4 columns (stride 32) per thread
    const int i1 = i0 + 32, nb = (kRows - i1) / 4 * 32;
    for (int t = tid; t < nb; t += nt) {
      const int i = i1 + 4 * (t >> 5), e = t & 31;
      float acc[4][4] = {};
      const float* li[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) li[r] = N + tri(i + r) + i0;
#pragma unroll 4
      for (int kx = 0; kx < 32; ++kx) {
        float l[4], z[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) l[r] = li[r][kx];
#pragma unroll
        for (int c = 0; c < 4; ++c) z[c] = R[(i0 + kx) * kLD + e + 32 * c];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += l[r] * z[c];
      }
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) R[(i + r) * kLD + e + 32 * c] -= acc[r][c];
    }
    __syncthreads();
  }
  // backward: L^T Z = W, Z_b = L_bb^-T (W_b - L_>b,b^T Z_>b)
  for (int ib = kRows / 32 - 1; ib >= 0; --ib) {
    const int i0 = ib * 32;
    {
      float acc[4][4] = {};
#pragma unroll 4
      for (int kx = 4 * rg; kx < 32; ++kx) {
        const float* lk = N + tri(i0 + kx) + i0 + 4 * rg;
        float l[4], z[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) l[r] = 4 * rg + r <= kx ? lk[r] : 0.f;
#pragma unroll
        for (int c = 0; c < 4; ++c) z[c] = R[(i0 + kx) * kLD + e + 32 * c];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += l[r] * z[c];
      }
      __syncthreads();
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) R[(i0 + 4 * rg + r) * kLD + e + 32 * c] = acc[r][c];
    }
    __syncthreads();
    // rows above: 4 rows x 4 columns (stride 32) per thread
    const int nb = i0 / 4 * 32;
    for (int t = tid; t < nb; t += nt) {
      const int i = 4 * (t >> 5), e = t & 31;
      float acc[4][4] = {};
#pragma unroll 4
      for (int kx = 0; kx < 32; ++kx) {
        const float* lk = N + tri(i0 + kx) + i;
        float l[4], z[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) l[r] = lk[r];
#pragma unroll
        for (int c = 0; c < 4; ++c) z[c] = R[(i0 + kx) * kLD + e + 32 * c];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += l[r] * z[c];
      }
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) R[(i + r) * kLD + e + 32 * c] -= acc[r][c];
    }
    __syncthreads();
  }
  for (int p = tid; p < kRows * kD / 4; p += nt) {
    const float* rr = R + (p >> 5) * kLD + (p & 31) * 4;
    ((float4*)RZ)[p] = make_float4(rr[0], rr[1], rr[2], rr[3]);
  }
}

// ======================================================== k_merge_cross
// The off-diagonal Gram block of a unit with two row blocks (128 < m <= 256):
// G01 = X_G0 X_G1^T over the non-fixed positions, as the split products
// Xh0 Xh1^T + Xl0 Xh1^T + Xh0 Xl1^T (the low-low term dropped, as in the
// diagonal blocks).  X uses the final row normalisers of both blocks (from
// the diagonal launches), so nothing is rescaled afterwards.  G01 goes to
// gram[u][r0][128 + r1] and, transposed, to gram[u][128 + r1][r0].  Roles
// (384 threads): warp 0 the Q loads; warps 0, 2, 3 the K0 gathers; warp 1 MMA
// issue; warps 4-7 the rows of block 0 (X_0 high / low parts written back
// over S_0 in TMEM, the A operands); warps 8-11 the rows of block 1 (XGh_1,
// XGl_1 in shared memory, the B operands).  One tile in flight: the S MMAs of
// a tile are issued after the Gram MMAs of the previous one, so s_full also
// tells both groups that their buffers are free.
struct CBars {
  uint64_t ring_full[2], ring_empty[2];
  uint64_t q_full, s_full, x0_full, x1_full, acc_done, drain;
  uint32_t tmem;
  int abort;
};
static_assert(sizeof(CBars) <= 256, "barrier block");
constexpr uint32_t kOffQ1C = kTileBytes, kOffRingC = 2 * kTileBytes, kOffXhC = 4 * kTileBytes,
                   kOffXlC = 5 * kTileBytes, kOffBarC = 6 * kTileBytes;
constexpr uint32_t kSmemBytesC = kOffBarC + 256 + 1024;

__global__ void __launch_bounds__(kThreads, 1)
    k_merge_cross(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  MArgs a) {
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  CBars* bars = (CBars*)(sm + kOffBarC);
  uint8_t* xgh = sm + kOffXhC;
  uint8_t* xgl = sm + kOffXlC;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x, B = a.B;
  const int ng = __ldg(a.ng + u), TG = (ng + kTile - 1) / kTile;
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->ring_full[i], 3);   // one expect_tx arrival per gathering warp
      mbar_init(&bars->ring_empty[i], 1);
    }
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->s_full, 1);
    mbar_init(&bars->x0_full, 128);
    mbar_init(&bars->x1_full, 128);
    mbar_init(&bars->acc_done, 1);
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem, 512);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem;
  volatile int* abort_flag = &bars->abort;
  constexpr uint32_t kColS0 = 0, kColS1 = 128, kColGC = 256;

  if (warp == 0 || warp == 2 || warp == 3) {
    if (warp == 0 && lane == 0) {
      prefetch_tensormap(&tmQ);
      mbar_expect_tx(&bars->q_full, 2 * kTileBytes);
      const uint64_t pol = l2_evict_last();
      for (int h = 0; h < 2; ++h) {
        tma_load_3d(sm + h * kTileBytes, &tmQ, &bars->q_full, 0, h * kRows, u, pol);
        tma_load_3d(sm + h * kTileBytes + kTileBytes / 2, &tmQ, &bars->q_full, 64, h * kRows, u, pol);
      }
    }
    __syncwarp();
    const int32_t* src_u = a.src + (size_t)u * B;
    const int pw = warp == 0 ? 0 : warp - 1;
    Gatherer<2, 3> gt{sm + kOffRingC, bars->ring_full, bars->ring_empty};
    int jn[4];
    if (TG > 0) gt.rows(src_u, B, a.n, u * a.n, 0, pw, lane, jn);
    bool ok = true;
    for (int t = 0; t < TG && ok; ++t) {
      const int j[4] = {jn[0], jn[1], jn[2], jn[3]};
      if (t + 1 < TG) gt.rows(src_u, B, a.n, u * a.n, t + 1, pw, lane, jn);
      ok = gt.load(&tmK, j, pw, lane, abort_flag);
    }
    gt.drain(abort_flag);
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_g = idesc_bf16(kRows, kRows, 0, 0);   // G01 += A XG1^T
      bool ok = mbar_wait(&bars->q_full, 0, abort_flag, kBudget);
      const uint32_t qa0 = smem_u32(sm), qa1 = smem_u32(sm + kOffQ1C);
      const uint32_t ha = smem_u32(xgh), la = smem_u32(xgl);
      for (int t = 0; t < TG && ok; ++t) {
        ok = mbar_wait(&bars->ring_full[t & 1], (t >> 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t ka = smem_u32(sm + kOffRingC + (t & 1) * kTileBytes);
        issue_s(tmem + kColS0, qa0, ka);
        issue_s(tmem + kColS1, qa1, ka);
        mma_commit(&bars->ring_empty[t & 1]);
        mma_commit(&bars->s_full);
        ok = mbar_wait(&bars->x0_full, t & 1, abort_flag, kBudget);
        if (ok) ok = mbar_wait(&bars->x1_full, t & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_bf16_ts(tmem + kColGC, tmem + kColS0 + xt_col(kk, 0), sw128_desc(ha + off, 16, 1024),
                      id_g, (t > 0 || kk > 0));
        }
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_bf16_ts(tmem + kColGC, tmem + kColS0 + xt_col(kk, 1), sw128_desc(ha + off, 16, 1024),
                      id_g, 1);
        }
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_bf16_ts(tmem + kColGC, tmem + kColS0 + xt_col(kk, 0), sw128_desc(la + off, 16, 1024),
                      id_g, 1);
        }
      }
      mma_commit(&bars->acc_done);
      mma_commit(&bars->drain);
      mbar_wait(&bars->drain, 0, abort_flag, kBudget);
    }
  } else {
    const int grp = (warp - 4) >> 2, q = warp & 3, row = q * 32 + lane;
    const int grow = grp * kRows + row;
    const float lam = grow < a.m ? a.lam[(size_t)u * a.ldr + grow] : INFINITY;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    const uint32_t sbase = lane_addr + (grp ? kColS1 : kColS0);
    bool ok = true;
    for (int t = 0; t < TG && ok; ++t) {
      ok = mbar_wait_warp(&bars->s_full, t & 1, abort_flag);
      if (!ok) break;
      tc_fence_after();
      float v[32];
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        tmem_ld32f(sbase + 32 * c, v);
        tmem_wait32(v);
        uint32_t hi[16], lo[16];
        const int p0 = t * kTile + 32 * c;
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          const float x0 = p0 + e < ng ? fast_exp2(fmaf(v[e], a.sl2, -lam)) : 0.f;
          const float x1 = p0 + e + 1 < ng ? fast_exp2(fmaf(v[e + 1], a.sl2, -lam)) : 0.f;
          const uint32_t h = pack_bf16(x0, x1);
          hi[e / 2] = h;
          lo[e / 2] = pack_bf16(x0 - lo_half(h), x1 - hi_half(h));
        }
        if (grp == 0) {
          tmem_st16(sbase + 32 * c, hi);
          tmem_st16(sbase + 32 * c + 16, lo);
        } else {
          store_row_chunk(xgh, row, c, hi);
          store_row_chunk(xgl, row, c, lo);
        }
      }
      if (grp == 0) {
        tmem_st_wait();
      } else {
        fence_proxy_async_smem();
      }
      tc_fence_before();
      mbar_arrive(grp == 0 ? &bars->x0_full : &bars->x1_full);
    }
    if (grp == 0) {
      if (ok) ok = mbar_wait_warp(&bars->acc_done, 0, abort_flag);
      tc_fence_after();
      if (ok) {
        float* up = a.gram + ((size_t)u * a.ldr + row) * a.ldr + kRows;   // row r0, columns 128 + r1
        float* lo = a.gram + ((size_t)u * a.ldr + kRows) * a.ldr + row;    // rows 128 + r1, column r0
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float g[32];
          tmem_ld32f(lane_addr + kColGC + 32 * c, g);
          tmem_wait32(g);
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float x = TG > 0 ? g[e] : 0.f;
            up[32 * c + e] = x;
            lo[(size_t)(32 * c + e) * a.ldr] = x;
          }
        }
      }
    }
    if (!ok && row == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// ======================================================== k_solve_dense
// The regression solve for m <= 256: N and R ([m][128]) from the workspace,
// Z = N^-1 R written over R.  With sym = 0, gram holds N = X_G X_G^T +
// lambda I (the portable merge); with sym = 1 it holds the raw Gram blocks of
// the tensor-core merge and N = (G + G^T) / 2 + lambda I.  Each unit's arrays
// hold ld rows.  The same blocked fp32 algorithm as k_merge_solve, for up to
// 256 rows: N as a packed lower triangle in shared memory (rows past m are
// identity), Cholesky in 32-row blocks, the diagonal blocks inverted in place,
// then block substitution over R in two passes of 64 columns.  lambda = +inf
// gives Z = 0.  One 512-thread CTA per unit.
constexpr int kDenseM = 256, kDenseNT = 512, kDenseC = 64, kDenseLD = kDenseC + 1;
constexpr int kDenseTri = tri(kDenseM) + 4;
constexpr uint32_t kDenseSmem = (kDenseTri + kDenseM * kDenseLD + kDenseM + 32) * 4;

__global__ void __launch_bounds__(kDenseNT, 1)
    k_solve_dense(const float* __restrict__ gram, float* __restrict__ rz, int m, int ld, int sym,
                  float lambda, int lambda_inf, int* status) {
  extern __shared__ __align__(16) float dsm[];
  float* N = dsm;                       // packed lower triangle
  float* R = N + kDenseTri;             // [256][kDenseLD]: one column pass of R, then of Z
  float* dinv = R + kDenseM * kDenseLD; // [256]
  int* fail = (int*)(dinv + kDenseM);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x;
  const float* Gu = gram + (size_t)u * ld * ld;
  float* RZ = rz + (size_t)u * ld * kD;
  if (lambda_inf) {
    for (int p = tid; p < m * kD; p += kDenseNT) RZ[p] = 0.f;
    return;
  }
  if (tid == 0) *fail = 0;
  // the lower triangle row by row (with sym: halved off the diagonal, lambda
  // added on it), then with sym the upper triangle's halves added, also read
  // row by row: both passes load whole rows
  for (int i = warp; i < kDenseM; i += kDenseNT / 32)
    for (int j = lane; j <= i; j += 32) {
      float val = i == j ? 1.f : 0.f;
      if (i < m && j < m) {
        val = __ldg(Gu + (size_t)i * ld + j);
        if (sym) val = i == j ? val + lambda : 0.5f * val;
      }
      N[tri(i) + j] = val;
    }
  if (sym) {
    __syncthreads();
    for (int r = warp; r < m; r += kDenseNT / 32)
      for (int c = r + 1 + lane; c < m; c += 32) N[tri(c) + r] += 0.5f * __ldg(Gu + (size_t)r * ld + c);
  }
  __syncthreads();
  for (int kb = 0; kb < kDenseM / 32; ++kb) {
    const int k0 = kb * 32;
    if (warp == 0 && chol_diag(N, dinv, k0, lane) && lane == 0) *fail = 1;
    __syncthreads();
    for (int i = k0 + 32 + tid; i < kDenseM; i += kDenseNT) chol_panel_row(N, dinv, k0, i);
    __syncthreads();
    // trailing update of the lower triangle in 4x4 register blocks
    const int k1 = k0 + 32, t4 = (kDenseM - k1) / 4, nb = t4 * (t4 + 1) / 2;
    for (int t = tid; t < nb; t += kDenseNT) {
      int bi = (int)((sqrtf(8.f * t + 1.f) - 1.f) * 0.5f);
      while ((bi + 1) * (bi + 2) / 2 <= t) ++bi;
      while (bi * (bi + 1) / 2 > t) --bi;
      const int i = k1 + 4 * bi, j = k1 + 4 * (t - bi * (bi + 1) / 2);
      float acc[4][4] = {};
#pragma unroll 4
      for (int pp = 0; pp < 32; ++pp) {
        float vi[4], vj[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          vi[r] = N[tri(i + r) + k0 + pp];
          vj[r] = N[tri(j + r) + k0 + pp];
        }
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] += vi[r] * vj[c];
      }
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (j + c <= i + r) N[tri(i + r) + j + c] -= acc[r][c];
    }
    __syncthreads();
  }
  if (*fail) {
    if (tid == 0) set_status(status, GRKV_ERR_NUMERIC);
    for (int p = tid; p < m * kD; p += kDenseNT) RZ[p] = 0.f;
    return;
  }
  if (warp < kDenseM / 32) tri_inv_diag(N, dinv, warp * 32, lane);
  __syncthreads();
  // block steps: thread = rows 4 rg .. 4 rg + 3 of a 32-row block, column cc
  const int rg = warp & 7, cc = (tid >> 8) * 32 + lane;
  for (int c0 = 0; c0 < kD; c0 += kDenseC) {
    for (int p = tid; p < kDenseM * kDenseC; p += kDenseNT) {
      const int r = p / kDenseC, c = p % kDenseC;
      R[r * kDenseLD + c] = r < m ? RZ[(size_t)r * kD + c0 + c] : 0.f;
    }
    __syncthreads();
    // forward: W_b = L_bb^-1 (R_b - L_b,<b W_<b)
    for (int ib = 0; ib < kDenseM / 32; ++ib) {
      const int i0 = ib * 32;
      float acc[4] = {};
      for (int kx = 0; kx < 4 * rg + 4; ++kx) {
        const float z = R[(i0 + kx) * kDenseLD + cc];
#pragma unroll
        for (int r = 0; r < 4; ++r)
          acc[r] += (kx <= 4 * rg + r ? N[tri(i0 + 4 * rg + r) + i0 + kx] : 0.f) * z;
      }
      __syncthreads();
#pragma unroll
      for (int r = 0; r < 4; ++r) R[(i0 + 4 * rg + r) * kDenseLD + cc] = acc[r];
      __syncthreads();
      // rows below: 4 rows x 1 column per task
      const int i1 = i0 + 32, ntask = (kDenseM - i1) / 4 * kDenseC;
      for (int t = tid; t < ntask; t += kDenseNT) {
        const int i = i1 + 4 * (t / kDenseC), c = t % kDenseC;
        float a4[4] = {};
#pragma unroll 8
        for (int kx = 0; kx < 32; ++kx) {
          const float z = R[(i0 + kx) * kDenseLD + c];
#pragma unroll
          for (int r = 0; r < 4; ++r) a4[r] += N[tri(i + r) + i0 + kx] * z;
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) R[(i + r) * kDenseLD + c] -= a4[r];
      }
      __syncthreads();
    }
    // backward: Z_b = L_bb^-T (W_b - L_>b,b^T Z_>b)
    for (int ib = kDenseM / 32 - 1; ib >= 0; --ib) {
      const int i0 = ib * 32;
      float acc[4] = {};
      for (int kx = 4 * rg; kx < 32; ++kx) {
        const float z = R[(i0 + kx) * kDenseLD + cc];
#pragma unroll
        for (int r = 0; r < 4; ++r)
          acc[r] += (4 * rg + r <= kx ? N[tri(i0 + kx) + i0 + 4 * rg + r] : 0.f) * z;
      }
      __syncthreads();
#pragma unroll
      for (int r = 0; r < 4; ++r) R[(i0 + 4 * rg + r) * kDenseLD + cc] = acc[r];
      __syncthreads();
      // rows above: 4 rows x 1 column per task
      const int ntask = i0 / 4 * kDenseC;
      for (int t = tid; t < ntask; t += kDenseNT) {
        const int i = 4 * (t / kDenseC), c = t % kDenseC;
        float a4[4] = {};
#pragma unroll 8
        for (int kx = 0; kx < 32; ++kx) {
          const float z = R[(i0 + kx) * kDenseLD + c];
#pragma unroll
          for (int r = 0; r < 4; ++r) a4[r] += N[tri(i0 + kx) + i + r] * z;
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) R[(i + r) * kDenseLD + c] -= a4[r];
      }
      __syncthreads();
    }
    for (int p = tid; p < m * kDenseC; p += kDenseNT) {
      const int r = p / kDenseC, c = p % kDenseC;
      RZ[(size_t)r * kD + c0 + c] = R[r * kDenseLD + c];
    }
    __syncthreads();
  }
}

// ======================================================== k_merge_update
// Slot order, one unit per CTA, 736 threads.  Roles: warp 0 the Q load and
// the K_out tile stores, warp 22 the V_out tile stores; warp 1 MMA issue;
// warps 2, 3, 16, 17 the K0 gathers and 18-21 the V0 gathers (two-slot rings
// each, on all four SM sub-partitions); warps 4-7 and 8-11
// two compute groups taking alternate tiles (one thread per token = TMEM lane
// of S^T): X_G^T from S^T, zero for fixed slots, written back over S^T as
// packed bf16 (rows 32c .. 32c+31 of chunk c: high parts to columns 32c ..
// 32c+15, low parts to 32c+16 .. 32c+31, each chunk read before it is
// overwritten); warps 12-15 the epilogue (thread = token): V_out = V0 + dV in
// the V0 tile, which warp 0 then stores.  A fixed slot has X = 0 and so
// dV = 0: its row is left as V0.
struct UBars {
  uint64_t k_full[2], k_empty[2], v_full[2], v_empty[2];
  uint64_t q_full;
  uint64_t s_full[2], x_full[2], d_full[2], d_empty[2], vo_full[2];
  uint64_t drain;
  uint32_t tmem;
  int abort;
};
static_assert(sizeof(UBars) <= 256, "barrier block");
constexpr uint32_t kOffKU = kTileBytes;                    // K0 ring, 2 tiles
constexpr uint32_t kOffVU = kOffKU + 2 * kTileBytes;       // V0 / V_out ring, 2 tiles
constexpr uint32_t kOffZU = kOffVU + 2 * kTileBytes;       // Zh, Zl
constexpr uint32_t kOffLamU = kOffBar + 256;               // [128] row normalisers
static_assert(kOffZU + 2 * kTileBytes == kOffBar, "update shared-memory layout");
constexpr uint32_t kSmemBytesU = kOffLamU + kRows * 4 + 1024;

__global__ void __launch_bounds__(kThreadsU, 1)
    k_merge_update(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmKo,
                   const __grid_constant__ CUtensorMap tmVo, MArgs a) {
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  UBars* bars = (UBars*)(sm + kOffBar);
  float* lam_s = (float*)(sm + kOffLamU);
  uint8_t* zh = sm + kOffZU;
  uint8_t* zl = zh + kTileBytes;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x, B = a.B, T = (B + kTile - 1) / kTile;
  const int32_t* idx_u = a.idx + (size_t)u * B;
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->k_full[i], 4);    // one expect_tx arrival per gathering warp
      mbar_init(&bars->v_full[i], 4);
      mbar_init(&bars->k_empty[i], 2);   // the S^T MMA and the K_out store
      mbar_init(&bars->v_empty[i], 1);   // the V_out store
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->x_full[i], 128);
      mbar_init(&bars->d_full[i], 1);
      mbar_init(&bars->d_empty[i], 128);
      mbar_init(&bars->vo_full[i], 128);
    }
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem, 512);
    tmem_relinquish();
  }
  // rows past m have lam = +inf and give X = 0
  if (tid < kRows) lam_s[tid] = a.lam[(size_t)u * a.ldr + a.row0 + tid];
  // Z (fp32 [row][d]) to the bf16 B operands Zh, Zl: MN-major tiles of
  // 128-byte rows (d contiguous), two blocks of 64 columns
  {
    const float* Z = a.rz + ((size_t)u * a.ldr + a.row0) * kD;
    for (int i = tid; i < kRows * (kD / 8); i += kThreadsU) {
      const int r = i >> 4, d8 = i & 15;
      const float4 z0 = __ldg((const float4*)(Z + r * kD + d8 * 8));
      const float4 z1 = __ldg((const float4*)(Z + r * kD + d8 * 8 + 4));
      const float zz[8] = {z0.x, z0.y, z0.z, z0.w, z1.x, z1.y, z1.z, z1.w};
      uint32_t h[4], l[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        h[j] = pack_bf16(zz[2 * j], zz[2 * j + 1]);
        l[j] = pack_bf16(zz[2 * j] - lo_half(h[j]), zz[2 * j + 1] - hi_half(h[j]));
      }
      const uint32_t off = (d8 >> 3) * (kTileBytes / 2) + sw128_offset(r, d8 & 7);
      *(uint4*)(zh + off) = make_uint4(h[0], h[1], h[2], h[3]);
      *(uint4*)(zl + off) = make_uint4(l[0], l[1], l[2], l[3]);
    }
    fence_proxy_async_smem();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem;
  volatile int* abort_flag = &bars->abort;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&tmQ);
      prefetch_tensormap(&tmKo);
      mbar_expect_tx(&bars->q_full, kTileBytes);
      const uint64_t pol = l2_evict_last();
      tma_load_3d(sm + kOffQ, &tmQ, &bars->q_full, 0, a.row0, u, pol);
      tma_load_3d(sm + kOffQ + kTileBytes / 2, &tmQ, &bars->q_full, 64, a.row0, u, pol);
      // K_out = K0 tile by tile (the map clips the rows past B)
      bool ok = true;
      for (int t = 0; t < T && ok; ++t) {
        const int sl = t & 1;
        ok = mbar_wait(&bars->k_full[sl], (t >> 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        if (a.upd_mode != 2) {   // the second row block's K_out is the first's
          const uint8_t* kt = sm + kOffKU + sl * kTileBytes;
          tma_store_3d(&tmKo, kt, 0, t * kTile, u);
          tma_store_3d(&tmKo, kt + kTileBytes / 2, 64, t * kTile, u);
          bulk_commit();
          bulk_wait_read<0>();
        }
        mbar_arrive(&bars->k_empty[sl]);
      }
      bulk_wait_all();
      if (!ok) set_status(a.status, GRKV_ERR_TIMEOUT);
    }
  } else if (warp == 22) {
    if (lane == 0) {
      prefetch_tensormap(&tmVo);
      // V_out tile by tile, once the epilogue has written it
      bool ok = true;
      for (int t = 0; t < T && ok; ++t) {
        const int sl = t & 1;
        ok = mbar_wait(&bars->vo_full[sl], (t >> 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        if (a.upd_mode != 1) {   // mode 1 leaves its result in vpart
          const uint8_t* vt = sm + kOffVU + sl * kTileBytes;
          tma_store_3d(&tmVo, vt, 0, t * kTile, u);
          tma_store_3d(&tmVo, vt + kTileBytes / 2, 64, t * kTile, u);
          bulk_commit();
          bulk_wait_read<0>();
        }
        mbar_arrive(&bars->v_empty[sl]);
      }
      bulk_wait_all();
      if (!ok) set_status(a.status, GRKV_ERR_TIMEOUT);
    }
  } else if (warp == 2 || warp == 3 || (warp >= 16 && warp < 22)) {
    // K0 gathers: warps 2, 3, 16, 17; V0 gathers: warps 18 - 21 (own rings, so
    // that a K tile never waits for a V slot)
    const bool is_v = warp >= 18;
    const int pw = warp < 4 ? warp - 2 : (is_v ? warp - 18 : warp - 14), row0 = u * a.n;
    // mode 2 builds V_out from vpart: no V0 tiles
    const int TG = is_v && a.upd_mode == 2 ? 0 : T;
    Gatherer<2, 4> g{sm + (is_v ? kOffVU : kOffKU), is_v ? bars->v_full : bars->k_full,
                     is_v ? bars->v_empty : bars->k_empty};
    const CUtensorMap* map = is_v ? &tmV : &tmK;
    int jn[4];
    if (TG > 0) g.rows(idx_u, B, a.n, row0, 0, pw, lane, jn);
    bool ok = true;
    for (int t = 0; t < TG && ok; ++t) {
      const int j[4] = {jn[0], jn[1], jn[2], jn[3]};
      if (t + 1 < TG) g.rows(idx_u, B, a.n, row0, t + 1, pw, lane, jn);
      ok = g.load(map, j, pw, lane, abort_flag);
    }
    g.drain(abort_flag);
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(kTile, kRows, 0, 0);   // S^T = K0 Q^T
      const uint32_t id_d = idesc_bf16(kTile, kD, 0, 1);      // dV = X_G^T Z (Z MN-major)
      const uint32_t qa = smem_u32(sm + kOffQ);
      const uint32_t bh = smem_u32(zh), bl = smem_u32(zl);
      bool ok = mbar_wait(&bars->q_full, 0, abort_flag, kBudget);
      auto issue_d = [&](int t) -> bool {
        const uint32_t d = tmem + kColD + (t & 1) * kD, x = tmem + kColS + (t & 1) * kTile;
        bool w = mbar_wait(&bars->x_full[t & 1], (t >> 1) & 1, abort_flag, kBudget);
        if (w && t >= 2) w = mbar_wait(&bars->d_empty[t & 1], ((t >> 1) - 1) & 1, abort_flag, kBudget);
        if (!w) return false;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kRows / 16; ++kk)
          mma_bf16_ts(d, x + xt_col(kk, 0), sw128_desc(bh + kk * 2048, kTileBytes / 2, 1024), id_d,
                      kk > 0);
#pragma unroll
        for (int kk = 0; kk < kRows / 16; ++kk)
          mma_bf16_ts(d, x + xt_col(kk, 0), sw128_desc(bl + kk * 2048, kTileBytes / 2, 1024), id_d, 1);
#pragma unroll
        for (int kk = 0; kk < kRows / 16; ++kk)
          mma_bf16_ts(d, x + xt_col(kk, 1), sw128_desc(bh + kk * 2048, kTileBytes / 2, 1024), id_d, 1);
        mma_commit(&bars->d_full[t & 1]);
        return true;
      };
      for (int t = 0; t < T && ok; ++t) {
        const int sl = t & 1;
        ok = mbar_wait(&bars->k_full[sl], (t >> 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
        // S^T into buffer sl: its previous contents (X_G^T of tile t - 2) were
        // read by the dV MMAs issued before this one
        const uint32_t ka = smem_u32(sm + kOffKU + sl * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_bf16(tmem + kColS + sl * kTile, sw128_desc(ka + off, 16, 1024),
                   sw128_desc(qa + off, 16, 1024), id_s, kk > 0);
        }
        mma_commit(&bars->k_empty[sl]);
        mma_commit(&bars->s_full[sl]);
        if (t >= 1) ok = issue_d(t - 1);
      }
      if (ok && T > 0) ok = issue_d(T - 1);
      mma_commit(&bars->drain);
      mbar_wait(&bars->drain, 0, abort_flag, kBudget);
    }
  } else if (warp >= 4 && warp < 12) {
    // compute groups: group cg takes the tiles t with t % 2 == cg
    const int cg = (warp - 4) >> 2, q = warp & 3, tok = q * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    bool ok = true;
    for (int t = cg; t < T && ok; t += 2) {
      const int sl = t & 1, slot = t * kTile + tok;
      const bool zero = slot >= B || __ldg(a.fixed + (size_t)u * B + min(slot, B - 1)) != 0;
      ok = mbar_wait_warp(&bars->s_full[sl], (t >> 1) & 1, abort_flag);
      if (!ok) break;
      tc_fence_after();
      const uint32_t sbase = lane_addr + kColS + sl * kTile;
      float v[32];
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        tmem_ld32f(sbase + 32 * c, v);
        tmem_wait32(v);
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          const float4 l4 = *(const float4*)(lam_s + 32 * c + (e & ~3));
          const float la = (e & 2) ? l4.z : l4.x, lb = (e & 2) ? l4.w : l4.y;
          float x0 = fast_exp2(fmaf(v[e], a.sl2, -la)), x1 = fast_exp2(fmaf(v[e + 1], a.sl2, -lb));
          if (zero) x0 = x1 = 0.f;
          const uint32_t h = pack_bf16(x0, x1);
          hi[e / 2] = h;
          lo[e / 2] = pack_bf16(x0 - lo_half(h), x1 - hi_half(h));
        }
        tmem_st16(sbase + 32 * c, hi);
        tmem_st16(sbase + 32 * c + 16, lo);
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&bars->x_full[sl]);
    }
    if (!ok && tok == 0 && cg == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  } else if (warp >= 12 && warp < 16) {
    // epilogue: thread = token (TMEM lane of D).  Mode 0: V_out = V0 + dV in
    // the V tile; mode 1: vpart = V0 + dV (fp32, every retained slot); mode 2:
    // V_out = vpart + dV into the V tile slot (no V0 there)
    const int q = warp & 3, tok = q * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    const int mode = a.upd_mode;
    bool ok = true;
    for (int t = 0; t < T && ok; ++t) {
      const int sl = t & 1, slot = t * kTile + tok;
      const bool in = slot < B;
      const bool live = in && (mode != 0 || __ldg(a.fixed + (size_t)u * B + min(slot, B - 1)) == 0);
      ok = mbar_wait_warp(&bars->d_full[sl], (t >> 1) & 1, abort_flag);
      if (ok && mode != 2) ok = mbar_wait_warp(&bars->v_full[sl], (t >> 1) & 1, abort_flag);
      if (ok && mode == 2 && t >= 2)
        ok = mbar_wait_warp(&bars->v_empty[sl], ((t >> 1) - 1) & 1, abort_flag);
      if (!ok) break;
      tc_fence_after();
      uint8_t* vt = sm + kOffVU + sl * kTileBytes;
      const uint32_t dcol = lane_addr + kColD + sl * kD;
      float* vp = mode != 0 ? a.vpart + ((size_t)u * B + min(slot, B - 1)) * kD : nullptr;
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        float dv[32];
        tmem_ld32f(dcol + c * 32, dv);
        tmem_wait32(dv);
        if (c == 3) {
          tc_fence_before();
          mbar_arrive(&bars->d_empty[sl]);
        }
        if (live) {
          // columns 32c .. 32c+31: half c/2, 16-byte chunks (c%2)*4 .. +3
          uint8_t* row = vt + (c >> 1) * (kTileBytes / 2);
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            uint4* p = (uint4*)(row + sw128_offset(tok, (c & 1) * 4 + h));
            float x[8];
            if (mode == 2) {
              const float4 p0 = *(const float4*)(vp + 32 * c + 8 * h);
              const float4 p1 = *(const float4*)(vp + 32 * c + 8 * h + 4);
              x[0] = p0.x; x[1] = p0.y; x[2] = p0.z; x[3] = p0.w;
              x[4] = p1.x; x[5] = p1.y; x[6] = p1.z; x[7] = p1.w;
            } else {
              const uint4 v0 = *p;
              const uint32_t w[4] = {v0.x, v0.y, v0.z, v0.w};
#pragma unroll
              for (int z = 0; z < 4; ++z) {
                x[2 * z] = lo_half(w[z]);
                x[2 * z + 1] = hi_half(w[z]);
              }
            }
#pragma unroll
            for (int z = 0; z < 8; ++z) x[z] += dv[8 * h + z];
            if (mode == 1) {
              *(float4*)(vp + 32 * c + 8 * h) = make_float4(x[0], x[1], x[2], x[3]);
              *(float4*)(vp + 32 * c + 8 * h + 4) = make_float4(x[4], x[5], x[6], x[7]);
            } else {
              *p = make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]),
                              pack_bf16(x[6], x[7]));
            }
          }
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(&bars->vo_full[sl]);
    }
    if (!ok && tok == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

}  // namespace

bool merge_tc_supported(const Shape& s) {
  return s.dtype == GRKV_BF16 && s.m <= 2 * kRows && s.B <= kMaxB && s.B >= 1;
}

// Workspace of the tensor-core merge: rz [U][ldr][128], gram [U][ldr][ldr],
// lam [U][ldr] (fp32), src [U][B], ng [U], redo [U][nrb] (int32), fixed [U][B]
// (bytes), and for two row blocks vpart [U][B][128] (fp32).
struct MergeWs {
  int ldr, nrb;
  size_t rz, gram, lam, src, ng, redo, fixed, vpart, total;
};
MergeWs merge_ws(const Shape& s) {
  MergeWs w;
  const size_t U = (size_t)s.U, B = (size_t)s.B;
  w.nrb = s.m > kRows ? 2 : 1;
  w.ldr = w.nrb * kRows;
  const size_t ldr = (size_t)w.ldr;
  w.rz = 0;
  w.gram = w.rz + U * ldr * kD * 4;
  w.lam = w.gram + U * ldr * ldr * 4;
  w.src = w.lam + U * ldr * 4;
  w.ng = w.src + U * B * 4;
  w.redo = w.ng + U * 4;
  w.fixed = w.redo + U * w.nrb * 4;
  w.vpart = (w.fixed + U * B + 15) & ~(size_t)15;
  w.total = w.vpart + (w.nrb > 1 ? U * B * kD * 4 : 0);
  return w;
}

size_t merge_tc_ws_bytes(const Shape& s) { return merge_ws(s).total; }

cudaError_t launch_solve_dense(int U, int m, int ld, int sym, float lambda, int lambda_inf,
                               const float* gram, float* rz, int* status, cudaStream_t st) {
  if (m > kDenseM || ld < m) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(k_solve_dense, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kDenseSmem);
  if (e != cudaSuccess) return e;
  k_solve_dense<<<U, kDenseNT, kDenseSmem, st>>>(gram, rz, m, ld, sym, lambda, lambda_inf, status);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_merge_tc(const Shape& s, const void* q, const void* k, const void* v,
                            const float* scores, const float* y, const float* row_stats,
                            const int32_t* idx, void* k_out, void* v_out, char* ws,
                            const WsLayout& L, cudaStream_t st) {
  CUtensorMap mq, mk, mv, mko, mvo;
  if (!encode_bf16_3d(&mq, q, kD, s.m, s.U, 64, kRows) ||
      !encode_bf16_2d_rows(&mk, k, kD, (uint64_t)s.U * s.n) ||
      !encode_bf16_2d_rows(&mv, v, kD, (uint64_t)s.U * s.n) ||
      !encode_bf16_3d(&mko, k_out, kD, s.B, s.U, 64, kTile) ||
      !encode_bf16_3d(&mvo, v_out, kD, s.B, s.U, 64, kTile))
    return cudaErrorInvalidValue;
  MArgs a{};
  a.U = s.U;
  a.n = s.n;
  a.w = s.w;
  a.m = s.m;
  a.P = s.P;
  a.B = s.B;
  a.causal = s.causal;
  a.n_sink = s.n_sink;
  a.n_fix = s.n_fix;
  a.sl2 = (float)((double)s.scale * 1.4426950408889634);
  a.lambda = s.lambda;
  a.lambda_inf = s.lambda_inf;
  a.idx = idx;
  a.scores = scores;
  a.y = y;
  a.k = (const __nv_bfloat16*)k;
  a.v = (const __nv_bfloat16*)v;
  a.k_out = (__nv_bfloat16*)k_out;
  a.v_out = (__nv_bfloat16*)v_out;
  a.rstats = row_stats;
  const MergeWs W = merge_ws(s);
  char* mw = ws + L.merge_tc;
  a.rz = (float*)(mw + W.rz);
  a.gram = (float*)(mw + W.gram);
  a.lam = (float*)(mw + W.lam);
  a.src = (int32_t*)(mw + W.src);
  a.ng = (int32_t*)(mw + W.ng);
  a.redo = (int32_t*)(mw + W.redo);
  a.fixed = (uint8_t*)(mw + W.fixed);
  a.vpart = W.nrb > 1 ? (float*)(mw + W.vpart) : nullptr;
  a.ldr = W.ldr;
  a.nrb = W.nrb;
  a.status = (int*)(ws + L.status);
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(k_merge_gram, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kSmemBytes)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(k_merge_update, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kSmemBytesU)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(k_merge_solve, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kSolveSmem)) != cudaSuccess ||
      (e = cudaFuncSetAttribute(k_merge_fixed, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                s.B * 4)) != cudaSuccess)
    return e;
  if (W.nrb > 1 && (e = cudaFuncSetAttribute(k_merge_cross, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmemBytesC)) != cudaSuccess)
    return e;
  k_merge_fixed<<<s.U, 256, s.B * 4, st>>>(a);
  int launches = 1;
  // the retained statistics, R and the diagonal Gram block of every row block
  for (int rb = 0; rb < W.nrb; ++rb) {
    a.rb = rb;
    a.row0 = rb * kRows;
    if (row_stats) {
      a.gram_mode = 1;
      k_merge_gram<<<s.U, kThreads, kSmemBytes, st>>>(mq, mk, mv, a);
      a.gram_mode = 2;
      k_merge_gram<<<s.U, kThreads, kSmemBytes, st>>>(mq, mk, mv, a);
      launches += 2;
    } else {
      a.gram_mode = 0;
      k_merge_gram<<<s.U, kThreads, kSmemBytes, st>>>(mq, mk, mv, a);
      launches += 1;
    }
  }
  if (W.nrb == 1) {
    a.rb = 0;
    a.row0 = 0;
    a.upd_mode = 0;
    k_merge_solve<<<s.U, kSolveThreads, kSolveSmem, st>>>(a);
    k_merge_update<<<s.U, kThreadsU, kSmemBytesU, st>>>(mq, mk, mv, mko, mvo, a);
    launches += 2;
  } else {
    // two row blocks: the cross Gram block, the 256-row solve, and the value
    // update of each row block (the first leaves V0 + dV_0 in vpart)
    k_merge_cross<<<s.U, kThreads, kSmemBytesC, st>>>(mq, mk, a);
    launches += 1;
    count_launches(launches);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = launch_solve_dense(s.U, s.m, W.ldr, 1, s.lambda, s.lambda_inf, a.gram, a.rz,
                                a.status, st)) != cudaSuccess)
      return e;
    launches = 0;
    for (int rb = 0; rb < 2; ++rb) {
      a.rb = rb;
      a.row0 = rb * kRows;
      a.upd_mode = rb == 0 ? 1 : 2;
      k_merge_update<<<s.U, kThreadsU, kSmemBytesU, st>>>(mq, mk, mv, mko, mvo, a);
      launches += 1;
    }
  }
  count_launches(launches);
  return cudaGetLastError();
}

}  // namespace grkv
