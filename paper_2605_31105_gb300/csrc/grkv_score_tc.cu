// Window scoring on the 5th-generation tensor cores in two launches per 128
// window rows (bf16, d = 128, m <= 256), the default scoring path.  The
// one-read path of GRKV_ONE_READ_SCORE is in grkv_score_pipe.cu.
//
// For every unit the path needs, over all n keys, the row statistics of the
// window logits (pass A: M_r, L_r) and then, with those, the probabilities,
// the per-key prefix scores c_j = sum_r P_rj and the target Y = P V (pass B);
// Eq. 4 and Algorithm 1 of the paper.  The row normaliser depends on every
// key, so this path reads the keys twice: pass A (mode 0) and pass B (mode 1)
// are two persistent launches over all units (one CTA per SM), each CTA on a
// contiguous range of the units' tiles.
//
// Roles (512 threads): warp 0 issues TMA loads (the unit's Q, then K and V
// tiles of 128 tokens through the ring; each V one job after its K, as
// it stays in the ring through the tile's compute), warp 1 issues tcgen05
// MMAs (S = Q K^T into TMEM; Y += P V with P read from TMEM), warps 4-7 and
// 8-11 are two compute groups that share every tile, tokens 0..63 and
// 64..127.  A compute thread owns one window row (one TMEM lane): pass A
// keeps its running max / sum in registers, pass B writes exp2(l - Lambda_r)
// back into TMEM as bf16 (the A operand of the Y MMA) and sums probabilities
// over rows with a warp transpose-reduction plus a 4-way shared-memory sum.
// Warp 2 merges the two groups' statistics of each pass-A segment into the
// segment's global slot and counts it; warp 3, ahead of each pass-B segment,
// waits (bounded) until all of the unit's slots are counted and combines
// them; warps 12-15 add each segment's Y partial to the unit's Y with float4
// atomics.
#include <algorithm>
#include <cmath>

#include "grkv_internal.cuh"
#include "sm100.cuh"
#include "tmap.cuh"

namespace grkv {
namespace {

using namespace sm100;

constexpr int kTile = 128;            // tokens per tile
constexpr int kRows = 128;            // window rows (m padded to 128)
constexpr int kThreads = 512;
constexpr uint32_t kTileBytes = kTile * kD * 2;   // 32 KB
constexpr long long kWaitBudget = 1ll << 32;      // cycles (~2 s) before a wait gives up
constexpr long long kTestWaitBudget = 1ll << 22;  // ~2 ms: the budget of GRKV_TEST_TIMEOUT

// Shared-memory layout (offsets from a 1024-byte aligned base) for kRing K/V
// ring slots and kQBuf Q tiles: 5 + 1 (a CTA switches units two or three
// times per launch).
template <int kRing, int kQBuf>
struct Layout {
  static constexpr uint32_t kOffQ = 0;                                 // kQBuf x 32 KB
  static constexpr uint32_t kOffRing = kOffQ + kQBuf * kTileBytes;     // kRing x 32 KB
  static constexpr uint32_t kOffRed = kOffRing + kRing * kTileBytes;   // [2 wg][2 buf][4][128] fp32
  static constexpr uint32_t kOffAstat = kOffRed + 2 * 2 * 4 * kTile * 4;   // [2 buf][2 wg][128] float2
  static constexpr uint32_t kOffLam = kOffAstat + 2 * 2 * kRows * 8;       // [2 buf][128] float
  static constexpr uint32_t kOffBar = kOffLam + 2 * kRows * 4;
  static constexpr uint32_t kSmemBytes = kOffBar + 512 + 1024;         // + alignment slack
};
constexpr int kRingTwo = 5, kQBufTwo = 1;

// TMEM columns: two S buffers, two Y accumulators.
constexpr uint32_t kColS = 0, kColY = 256;

struct Args {
  int U, n, w, m, P, causal;
  int row0, mr;   // stacked rows row0 .. row0 + mr - 1 (mr <= 128) in this launch
  int acc;        // a later row block: its prefix scores go to scores2 (added by k_add_scores)
  int tpu;        // tiles per unit
  int mode;       // 0: pass A, 1: pass B
  int gu;         // units per round (all of them)
  int rounds;     // 1
  int maxc;       // stats slots per unit
  float sl2;      // scale * log2(e)
  float* scores;   // [U][P]
  float* scores2;  // [U][P] prefix scores of the second row block (m > 128)
  float* y;       // [U][m][128], zeroed by the host
  float* row_stats;  // [U][m][2]
  float2* pstats;    // [U][maxc][128]  (max in log2 units, sum)
  int* unit_cnt;     // [U] pass-A slots written, zeroed by the host
  int* status;
  float* ypart;      // [U][maxc][m][128] segment Y partials (deterministic mode) or null
  long long wait_budget;   // cycles before a bounded wait gives up
  int test_withhold;       // GRKV_TEST_TIMEOUT: CTA 0 withholds one arrive
};

// ------------------------------------------------------------ job schedule
struct Job {
  int kind;       // 0 = pass A, 1 = pass B
  int u, r;       // unit, round
  int j0, len;    // first token, tokens in the tile
  int seg_first, seg_last;
};

// One block of jobs per launch: pass A (mode 0) or pass B (mode 1) over all
// units, in one round.
struct Sched {
  int U, tpu, G, cta, mode, gu, rounds;
  __device__ int nblocks() const { return 1; }
  __device__ void block(int, int* kind, int* r) const {
    *kind = mode;
    *r = 0;
  }
  __device__ int round_units(int r) const { return min(gu, U - r * gu); }
  __device__ long long tiles(int r) const { return (long long)round_units(r) * tpu; }
  __device__ long long start(int r, int c) const { return tiles(r) * c / G; }
  // CTA whose range holds round-local tile t.
  __device__ int owner(int r, long long t) const {
    const long long T = tiles(r);
    return (int)(((t + 1) * G + T - 1) / T) - 1;
  }
  __device__ int first_cta(int u) const {
    const int r = u / gu;
    return owner(r, (long long)(u - r * gu) * tpu);
  }
  // True if CTA c holds no tile of round r (only when the round has fewer
  // tiles than there are CTAs).
  __device__ bool empty(int r, int c) const {
    return tiles(r) < G && start(r, c) == start(r, c + 1);
  }
  // Pass-A statistics slots written for unit u (one per CTA that holds its tiles).
  __device__ int writers(int u) const {
    const int r = u / gu, ns = nslots(u);
    if (tiles(r) >= G) return ns;
    const int c0 = first_cta(u);
    int w = 0;
    for (int k = 0; k < ns; ++k) w += empty(r, c0 + k) ? 0 : 1;
    return w;
  }
  __device__ int nslots(int u) const {
    const int r = u / gu;
    const long long t0 = (long long)(u - r * gu) * tpu;
    return owner(r, t0 + tpu - 1) - owner(r, t0) + 1;
  }
};

struct JobIter {
  const Sched* sc;
  int n;
  int p, kind, r;
  long long t, t_end, t_begin;
  __device__ void init(const Sched* s, int n_) {
    sc = s;
    n = n_;
    p = -1;
    t = t_end = 0;
  }
  // Advances to the next block; returns false when none are left.
  __device__ bool next_block() {
    if (++p >= sc->nblocks()) return false;
    sc->block(p, &kind, &r);
    t_begin = t = sc->start(r, sc->cta);
    t_end = sc->start(r, sc->cta + 1);
    return true;
  }
  __device__ bool has_job() const { return t < t_end; }
  __device__ Job job() const {
    Job j;
    j.kind = kind;
    j.r = r;
    // round-local tile indices stay below U * tiles per unit, well inside int
    const int lu = (int)t / sc->tpu, ti = (int)t - lu * sc->tpu;
    j.u = r * sc->gu + lu;
    j.j0 = ti * kTile;
    j.len = min(kTile, n - j.j0);
    j.seg_first = (t == t_begin) || ti == 0;
    j.seg_last = (t + 1 == t_end) || ti == sc->tpu - 1;
    return j;
  }
  __device__ void advance() { ++t; }
};

// Three-operand maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float fmax3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ float max32(const float* v) {
  float m[11];
#pragma unroll
  for (int e = 0; e < 10; ++e) m[e] = fmax3f(v[3 * e], v[3 * e + 1], v[3 * e + 2]);
  m[10] = fmaxf(v[30], v[31]);
  const float x0 = fmax3f(m[0], m[1], m[2]), x1 = fmax3f(m[3], m[4], m[5]),
              x2 = fmax3f(m[6], m[7], m[8]), x3 = fmaxf(m[9], m[10]);
  return fmaxf(fmax3f(x0, x1, x2), x3);
}

// Pass A on 32 logits: online row max / sum of exp2 in log2 units.
__device__ __forceinline__ void stats_chunk(float* v, bool full, int j0, int lim, int n,
                                            bool row_ok, float sl2, float& M, float& L) {
  if (!full) {
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (j0 + e > lim || j0 + e >= n || !row_ok) v[e] = -INFINITY;
  }
  const float vmax = max32(v);
  if (vmax == -INFINITY) return;
  const float cm = vmax * sl2;
  if (cm > M) {
    L *= fast_exp2(M - cm);
    M = cm;
  }
  float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < 32; ++e) s[e & 3] += fast_exp2(fmaf(v[e], sl2, -M));
  L += (s[0] + s[1]) + (s[2] + s[3]);
}

// mbar_wait for all lanes of a warp with one answer, so that warp-collective
// instructions after a wait are reached by all lanes or by none.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort,
                                               long long budget) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort, budget));
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// TMEM column of the packed bf16 P for tokens 16kk..16kk+15 of a tile: the
// compute group that owns tokens 0..63 packs them into S columns 0..31, the
// one that owns 64..127 into S columns 64..95 (each inside the S columns it
// has already read).
__device__ __forceinline__ uint32_t p_col(int kk) { return kk < 4 ? kk * 8 : 64 + (kk - 4) * 8; }

template <int kRing, int kQBuf>
struct Bars {
  uint64_t ring_full[kRing], ring_empty[kRing];
  uint64_t q_full[kQBuf], q_empty[kQBuf];
  uint64_t s_full[2], s_done[2];
  uint64_t y_full[2], y_empty[2];
  uint64_t astat_full[2], astat_empty[2];   // compute groups -> statistics publisher
  uint64_t lam_full[2], lam_empty[2];       // statistics fetcher -> compute groups
  uint64_t grp[2][2];                       // per compute group, alternating per pass-B tile
  uint64_t drain;
  uint32_t tmem;
  int abort;
};
static_assert(sizeof(Bars<kRingTwo, kQBufTwo>) <= 512, "barrier block");

// Merges two (max, sum) row statistics in log2 units.
__device__ __forceinline__ float2 stat_merge(float2 x, float2 y) {
  if (x.x == -INFINITY) return y;
  if (y.x == -INFINITY) return x;
  const float M = fmaxf(x.x, y.x);
  return make_float2(M, x.y * fast_exp2(x.x - M) + y.y * fast_exp2(y.x - M));
}

template <int kRing, int kQBuf>
__global__ void __launch_bounds__(kThreads, 1)
    k_score_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, Args a) {
  using Lay = Layout<kRing, kQBuf>;
  constexpr uint32_t kOffQ = Lay::kOffQ, kOffRing = Lay::kOffRing, kOffRed = Lay::kOffRed,
                     kOffAstat = Lay::kOffAstat, kOffLam = Lay::kOffLam, kOffBar = Lay::kOffBar;
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  Bars<kRing, kQBuf>* bars = (Bars<kRing, kQBuf>*)(sm + kOffBar);
  float* red = (float*)(sm + kOffRed);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  Sched sc{a.U, a.tpu, (int)gridDim.x, (int)blockIdx.x, a.mode, a.gu, a.rounds};

  if (tid == 0) {
    for (int i = 0; i < kQBuf; ++i) {
      mbar_init(&bars->q_full[i], 1);
      mbar_init(&bars->q_empty[i], 1);
    }
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&bars->ring_full[i], 1);
      mbar_init(&bars->ring_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_done[i], 256);
      mbar_init(&bars->y_full[i], 1);
      mbar_init(&bars->y_empty[i], 128);
      mbar_init(&bars->astat_full[i], 256);
      mbar_init(&bars->astat_empty[i], 1);
      mbar_init(&bars->lam_full[i], 1);
      mbar_init(&bars->lam_empty[i], 256);
    }
    for (int g = 0; g < 2; ++g)
      for (int i = 0; i < 2; ++i) mbar_init(&bars->grp[g][i], 4);   // one arrive per warp
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

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      prefetch_tensormap(&tmQ);
      prefetch_tensormap(&tmK);
      prefetch_tensormap(&tmV);
      const uint64_t keep = l2_evict_last(), stream = l2_evict_first();
      JobIter it;
      it.init(&sc, a.n);
      uint32_t slot = 0, ring_use = 0;   // ring_use counts loads
      int seg = 0, qissued = 0;
      bool ok = true;
      bool pend_v = false;
      int pv_j0 = 0, pv_u = 0;
      auto load = [&](const CUtensorMap* map, int j0, int u, uint64_t pol) -> bool {
        if (ring_use >= kRing &&
            !mbar_wait(&bars->ring_empty[slot], ((ring_use / kRing) - 1) & 1, abort_flag,
                       a.wait_budget))
          return false;
        uint8_t* dst = sm + kOffRing + slot * kTileBytes;
        mbar_expect_tx(&bars->ring_full[slot], kTileBytes);
        tma_load_3d(dst, map, &bars->ring_full[slot], 0, j0, u, pol);
        tma_load_3d(dst + kTileBytes / 2, map, &bars->ring_full[slot], 64, j0, u, pol);
        ++ring_use;
        slot = (slot + 1) % kRing;
        return true;
      };
      while (ok && it.next_block()) {
        for (; ok && it.has_job(); it.advance()) {
          const Job j = it.job();
          if (j.seg_first) {
            const int qs = seg % kQBuf;
            if (seg >= kQBuf) ok = mbar_wait(&bars->q_empty[qs], (seg / kQBuf - 1) & 1, abort_flag,
                                         a.wait_budget);
            if (!ok) break;
            ++qissued;
            mbar_expect_tx(&bars->q_full[qs], kTileBytes);
            uint8_t* dq = sm + kOffQ + qs * kTileBytes;
            tma_load_3d(dq, &tmQ, &bars->q_full[qs], 0, a.row0, j.u, keep);
            tma_load_3d(dq + kTileBytes / 2, &tmQ, &bars->q_full[qs], 64, a.row0, j.u, keep);
          }
          // the job's K, then the V of the previous pass-B job: V waits in the
          // ring through a tile's compute, so it is fetched one tile later
          ok = load(&tmK, j.j0, j.u, stream);
          if (ok && pend_v) {
            ok = load(&tmV, pv_j0, pv_u, stream);
            pend_v = false;
          }
          if (j.kind == 1) {
            pend_v = true;
            pv_j0 = j.j0;
            pv_u = j.u;
          }
          if (j.seg_last) ++seg;
        }
      }
      if (ok && pend_v) ok = load(&tmV, pv_j0, pv_u, stream);
      // let every issued load land before the CTA can exit (these waits
      // ignore the abort flag, and are bounded)
      volatile int no_abort = 0;
      for (uint32_t i = ring_use > kRing ? ring_use - kRing : 0; i < ring_use; ++i)
        mbar_wait(&bars->ring_full[i % kRing], (i / kRing) & 1, &no_abort, a.wait_budget);
      const int qloads = qissued;
      for (int i = qloads > kQBuf ? qloads - kQBuf : 0; i < qloads; ++i)
        mbar_wait(&bars->q_full[i % kQBuf], (i / kQBuf) & 1, &no_abort, a.wait_budget);
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(kRows, kTile, 0, 0);   // S = Q K^T, both K-major
      const uint32_t id_y = idesc_bf16(kRows, kD, 0, 1);      // Y += P V, V MN-major
      JobIter it;
      it.init(&sc, a.n);
      uint32_t slot = 0, ring_use = 0;
      int seg = 0, bseg = 0, i = 0;
      bool ok = true;
      // the pending pass-B job whose Y MMA is issued after the next S MMA
      bool pend = false;
      Job pj{};
      int p_i = 0, p_yb = 0;
      uint32_t p_vslot = 0, p_vuse = 0;
      int ybuf_uses[2] = {0, 0};
      while (ok && it.next_block()) {
        for (; ok && it.has_job(); it.advance()) {
          const Job j = it.job();
          const int b = i & 1, use = i >> 1;
          if (j.seg_first) {
            ok = mbar_wait(&bars->q_full[seg % kQBuf], (seg / kQBuf) & 1, abort_flag, a.wait_budget);
            if (!ok) break;
          }
          const uint32_t kslot = slot, kuse = ring_use;
          ok = mbar_wait(&bars->ring_full[kslot], (kuse / kRing) & 1, abort_flag, a.wait_budget);
          if (ok && use >= 1)
            ok = mbar_wait(&bars->s_done[b], (use - 1) & 1, abort_flag, a.wait_budget);
          if (!ok) break;
          tc_fence_after();
          const uint32_t qa = smem_u32(sm + kOffQ + (seg % kQBuf) * kTileBytes);
          const uint32_t ka = smem_u32(sm + kOffRing + kslot * kTileBytes);
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
            mma_bf16(tmem + kColS + b * kTile, sw128_desc(qa + off, 16, 1024),
                     sw128_desc(ka + off, 16, 1024), id_s, kk > 0);
          }
          mma_commit(&bars->ring_empty[kslot]);
          mma_commit(&bars->s_full[b]);
          ++ring_use;
          slot = (slot + 1) % kRing;
          if (j.seg_last) {
            mma_commit(&bars->q_empty[seg % kQBuf]);
            ++seg;
          }
          // Y MMA of the previous pass-B job (its P is ready once s_done fires);
          // its V is the load after this job's K
          if (pend) {
            p_vslot = slot;
            p_vuse = ring_use;
            ++ring_use;
            slot = (slot + 1) % kRing;
            const int pb = p_i & 1, puse = p_i >> 1;
            const int yb = p_yb;
            if (pj.seg_first && ybuf_uses[yb] >= 1)
              ok = mbar_wait(&bars->y_empty[yb], (ybuf_uses[yb] - 1) & 1, abort_flag,
                             a.wait_budget);
            if (ok) ok = mbar_wait(&bars->s_done[pb], puse & 1, abort_flag, a.wait_budget);
            if (ok)
              ok = mbar_wait(&bars->ring_full[p_vslot], (p_vuse / kRing) & 1, abort_flag,
                             a.wait_budget);
            if (!ok) break;
            tc_fence_after();
            const uint32_t va = smem_u32(sm + kOffRing + p_vslot * kTileBytes);
#pragma unroll
            for (int kk = 0; kk < kTile / 16; ++kk)
              mma_bf16_ts(tmem + kColY + yb * kD, tmem + kColS + pb * kTile + p_col(kk),
                          sw128_desc(va + kk * 2048, kTileBytes / 2, 1024), id_y,
                          (pj.seg_first && kk == 0) ? 0u : 1u);
            mma_commit(&bars->ring_empty[p_vslot]);
            if (pj.seg_last) {
              mma_commit(&bars->y_full[yb]);
              ++ybuf_uses[yb];
            }
            pend = false;
          }
          if (j.kind == 1) {
            pend = true;
            pj = j;
            p_i = i;
            if (j.seg_first) p_yb = bseg & 1;
            if (j.seg_last) ++bseg;
          }
          ++i;
        }
      }
      if (ok && pend) {
        p_vslot = slot;
        p_vuse = ring_use;
        const int pb = p_i & 1, puse = p_i >> 1;
        const int yb = p_yb;
        if (pj.seg_first && ybuf_uses[yb] >= 1)
          ok = mbar_wait(&bars->y_empty[yb], (ybuf_uses[yb] - 1) & 1, abort_flag, a.wait_budget);
        if (ok) ok = mbar_wait(&bars->s_done[pb], puse & 1, abort_flag, a.wait_budget);
        if (ok)
          ok = mbar_wait(&bars->ring_full[p_vslot], (p_vuse / kRing) & 1, abort_flag,
                         a.wait_budget);
        if (ok) {
          tc_fence_after();
          const uint32_t va = smem_u32(sm + kOffRing + p_vslot * kTileBytes);
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk)
            mma_bf16_ts(tmem + kColY + yb * kD, tmem + kColS + pb * kTile + p_col(kk),
                        sw128_desc(va + kk * 2048, kTileBytes / 2, 1024), id_y,
                        (pj.seg_first && kk == 0) ? 0u : 1u);
          mma_commit(&bars->ring_empty[p_vslot]);
          if (pj.seg_last) mma_commit(&bars->y_full[yb]);
        }
      }
      // every MMA issued so far completes before TMEM can be released (this
      // wait ignores the abort flag, and is bounded)
      mma_commit(&bars->drain);
      volatile int no_abort = 0;
      mbar_wait(&bars->drain, 0, &no_abort, a.wait_budget);
    }
  } else if (warp == 2) {
    // ----------------------------------------------- statistics publisher
    // Merges the two compute groups' row statistics of each pass-A segment
    // into the segment's global slot, then counts the slot as written.
    float2* astat = (float2*)(sm + kOffAstat);
    JobIter it;
    it.init(&sc, a.n);
    int aseg = 0;
    bool ok = true;
    while (ok && it.next_block()) {
      for (; ok && it.has_job(); it.advance()) {
        const Job j = it.job();
        if (!(j.seg_last && j.kind == 0)) continue;
        const int ab = aseg & 1;
        ok = mbar_wait_warp(&bars->astat_full[ab], (aseg >> 1) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        const int k = (int)blockIdx.x - sc.first_cta(j.u);
        // k < maxc always holds (the host sizes maxc from the same partition)
        if (k >= 0 && k < a.maxc) {
          float2* slot = a.pstats + ((size_t)j.u * a.maxc + k) * kRows;
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const int r = t * 32 + lane;
            slot[r] = stat_merge(astat[(ab * 2 + 0) * kRows + r], astat[(ab * 2 + 1) * kRows + r]);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->astat_empty[ab]);
        __threadfence();
        __syncwarp();
        if (lane == 0) atomicAdd(&a.unit_cnt[j.u], 1);
        ++aseg;
      }
    }
  } else if (warp == 3) {
    // ------------------------------------------------ statistics fetcher
    // Ahead of each pass-B segment: wait until every pass-A slot of the unit
    // is written, combine the slots, and leave every row's log2 normaliser in
    // shared memory.  The CTA that holds the unit's first tile also writes
    // the unit's row statistics.
    float* lam_s = (float*)(sm + kOffLam);
    JobIter it;
    it.init(&sc, a.n);
    int bseg = 0;
    bool ok = true;
    while (ok && it.next_block()) {
      for (; ok && it.has_job(); it.advance()) {
        const Job j = it.job();
        if (!(j.seg_first && j.kind == 1)) continue;
        const int lb = bseg & 1;
        if (bseg >= 2)
          ok = mbar_wait_warp(&bars->lam_empty[lb], ((bseg >> 1) - 1) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        const int need = sc.writers(j.u);
        const long long t0 = clock64();
        while (ld_acquire(&a.unit_cnt[j.u]) < need) {
          if (*abort_flag || clock64() - t0 > a.wait_budget) {
            *abort_flag = 1;
            ok = false;
            break;
          }
        }
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        const int ns = sc.nslots(j.u), c0 = sc.first_cta(j.u);
        const bool dense = sc.tiles(j.r) >= sc.G;   // every CTA holds tiles of the round
        float2 st[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) st[t] = make_float2(-INFINITY, 0.f);
        // eight slots per round trip: 32 independent loads in flight per lane
        for (int k0 = 0; k0 < ns; k0 += 8) {
          float2 pr[8][4];
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const bool use = k0 + kk < ns && (dense || !sc.empty(j.r, c0 + k0 + kk));
            const float2* sl = a.pstats + ((size_t)j.u * a.maxc + k0 + kk) * kRows;
#pragma unroll
            for (int t = 0; t < 4; ++t)
              pr[kk][t] = use ? __ldcg(sl + t * 32 + lane) : make_float2(-INFINITY, 0.f);
          }
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
#pragma unroll
            for (int t = 0; t < 4; ++t) st[t] = stat_merge(st[t], pr[kk][t]);
        }
        const bool first = (int)blockIdx.x == c0;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int r = t * 32 + lane;
          lam_s[lb * kRows + r] = (r < a.mr && st[t].y > 0.f) ? st[t].x + __log2f(st[t].y) : INFINITY;
          if (first && r < a.mr) {
            a.row_stats[((size_t)j.u * a.m + a.row0 + r) * 2 + 0] = st[t].x * 0.69314718055994531f;
            a.row_stats[((size_t)j.u * a.m + a.row0 + r) * 2 + 1] = st[t].y;
          }
        }
        __syncwarp();
        // GRKV_TEST_TIMEOUT: CTA 0 never announces its first pass-B
        // normalisers, so its compute groups' bounded wait expires
        if (lane == 0 && !(a.test_withhold && blockIdx.x == 0 && bseg == 0))
          mbar_arrive(&bars->lam_full[lb]);
        ++bseg;
      }
    }
  } else if (warp >= 12) {
    // ------------------------------------------------------- Y flusher
    // Each pass-B segment's Y partial (TMEM, one row per lane) is added to
    // the unit's Y with float4 atomics.
    const int q = warp & 3, row = q * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    JobIter it;
    it.init(&sc, a.n);
    int bseg = 0;
    bool ok = true;
    while (ok && it.next_block()) {
      for (; ok && it.has_job(); it.advance()) {
        const Job j = it.job();
        if (!(j.seg_last && j.kind == 1)) continue;
        const int yb = bseg & 1;
        ok = mbar_wait_warp(&bars->y_full[yb], (bseg >> 1) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t ybase = lane_addr + kColY + yb * kD;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(ybase + c * 32, v);
          tmem_ld_wait();
          if (row < a.mr && a.ypart) {
            // the segment's partial into its own slot, summed in slot order later
            const int k = (int)blockIdx.x - sc.first_cta(j.u);
            float4* dst = (float4*)(a.ypart + (((size_t)j.u * a.maxc + k) * a.m + a.row0 + row) *
                                                  kD + c * 32);
#pragma unroll
            for (int e = 0; e < 8; ++e)
              dst[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
          } else if (row < a.mr) {
            float4* dst = (float4*)(a.y + ((size_t)j.u * a.m + a.row0 + row) * kD + c * 32);
#pragma unroll
            for (int e = 0; e < 8; ++e)
              atomicAdd(dst + e, make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]));
          }
        }
        tc_fence_before();
        mbar_arrive(&bars->y_empty[yb]);
        ++bseg;
      }
    }
    if (!ok && row == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  } else if (warp >= 4) {
    // ------------------------------------------------------- compute groups
    const int wg = (warp - 4) >> 2, q = warp & 3;
    const int row = q * 32 + lane;
    const bool row_ok = row < a.mr;
    const int lim = a.causal ? a.n - a.w + (row_ok ? (a.row0 + row) % a.w : 0) : a.n - 1;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    float2* astat = (float2*)(sm + kOffAstat);
    const float* lam_s = (const float*)(sm + kOffLam);
    JobIter it;
    it.init(&sc, a.n);
    int i = 0, aseg = 0, bseg = 0;
    bool ok = true;
    float M = -INFINITY, L = 0.f;     // pass-A running stats (log2 units)
    float lam = INFINITY;             // pass-B log2 normaliser of this row
    while (ok && it.next_block()) {
      for (; ok && it.has_job(); it.advance(), ++i) {
        const Job j = it.job();
        const int b = i & 1;
        if (j.seg_first) {
          if (j.kind == 0) {
            M = -INFINITY;
            L = 0.f;
          } else {
            const int lb = bseg & 1;
            ok = mbar_wait_warp(&bars->lam_full[lb], (bseg >> 1) & 1, abort_flag, a.wait_budget);
            if (!ok) break;
            lam = lam_s[lb * kRows + row];
            mbar_arrive(&bars->lam_empty[lb]);
          }
        }
        {
          ok = mbar_wait_warp(&bars->s_full[b], (i >> 1) & 1, abort_flag, a.wait_budget);
          if (!ok) break;
          tc_fence_after();
          // this group's half of the tile: tokens 64 wg .. 64 wg + 63
          const int c0 = 2 * wg, t0 = j.j0 + 64 * wg;
          const uint32_t sbase = lane_addr + kColS + b * kTile;
          // halves away from the window and the end of the unit need no mask
          const bool full = row_ok && t0 + 63 <= lim && t0 + 64 <= a.n;
          float va[32], vb[32];
          tmem_ld32f(sbase + c0 * 32, va);
          tmem_wait32(va);
          tmem_ld32f(sbase + c0 * 32 + 32, vb);
          if (j.kind == 0) {
            stats_chunk(va, full, t0, lim, a.n, row_ok, a.sl2, M, L);
            tmem_wait32(vb);
            tc_fence_before();
            mbar_arrive(&bars->s_done[b]);   // S fully read
            stats_chunk(vb, full, t0 + 32, lim, a.n, row_ok, a.sl2, M, L);
          } else {
            float* rb = red + ((wg * 2 + (i & 1)) * 4) * kTile;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              float* v = h ? vb : va;
              if (h) tmem_wait32(vb);
              if (full) {
#pragma unroll
                for (int e = 0; e < 32; ++e) v[e] = fast_exp2(fmaf(v[e], a.sl2, -lam));
              } else {
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const int jj = t0 + h * 32 + e;
                  v[e] = (jj > lim || jj >= a.n || !row_ok) ? 0.f
                                                            : fast_exp2(fmaf(v[e], a.sl2, -lam));
                }
              }
              uint32_t pk[16];
#pragma unroll
              for (int e = 0; e < 16; ++e) pk[e] = pack_bf16(v[2 * e], v[2 * e + 1]);
              // chunk c0 + h packs into the 16 columns at 64 wg + 16 h
              tmem_st16(sbase + 64 * wg + 16 * h, pk);
              // transpose-reduce: lane t ends with the warp's sum for token 32h + t
#pragma unroll
              for (int hh = 16; hh >= 1; hh >>= 1) {
                const bool up = (lane & hh) != 0;
#pragma unroll
                for (int e = 0; e < hh; ++e) {
                  const float send = up ? v[e] : v[e + hh];
                  const float keep = up ? v[e + hh] : v[e];
                  v[e] = keep + __shfl_xor_sync(0xffffffffu, send, hh);
                }
              }
              rb[q * 64 + h * 32 + lane] = v[0];
            }
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(&bars->s_done[b]);
            // the group's four warps have written their sums (a bounded wait
            // where a barrier instruction could not give up)
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars->grp[wg][i & 1]);
            ok = mbar_wait_warp(&bars->grp[wg][i & 1], (i >> 1) & 1, abort_flag, a.wait_budget);
            if (!ok) break;
            if (q < 2) {
              const int jj = q * 32 + lane;
              const float cs = ((rb[jj] + rb[64 + jj]) + rb[128 + jj]) + rb[192 + jj];
              if (t0 + jj < a.P && 64 * wg + jj < j.len) {
                (a.acc ? a.scores2 : a.scores)[(size_t)j.u * a.P + t0 + jj] = cs;
              }
            }
          }
        }
        if (j.seg_last) {
          if (j.kind == 0) {
            const int ab = aseg & 1;
            if (aseg >= 2)
              ok = mbar_wait_warp(&bars->astat_empty[ab], ((aseg >> 1) - 1) & 1, abort_flag,
                             a.wait_budget);
            if (!ok) break;
            astat[(ab * 2 + wg) * kRows + row] = make_float2(M, L);
            mbar_arrive(&bars->astat_full[ab]);
            ++aseg;
          } else {
            ++bseg;
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

// scores += scores2: the second row block's prefix scores (m > 128) added
// once, instead of read-modify-written by the tiles of its pass B.
__global__ void k_add_scores(float* __restrict__ scores, const float* __restrict__ scores2,
                             size_t count) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
       i += (size_t)gridDim.x * blockDim.x)
    scores[i] += scores2[i];
}

// Deterministic mode: Y[u] = sum over the unit's slots k = 0 .. maxc-1 of the
// segment partials, in slot order (unwritten slots hold zeros).
__global__ void k_y_sum_slots(const float4* __restrict__ part, float4* __restrict__ y, int U,
                              int m, int maxc) {
  const size_t per_unit = (size_t)m * kD / 4;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < (size_t)U * per_unit;
       i += (size_t)gridDim.x * blockDim.x) {
    const size_t u = i / per_unit, r = i - u * per_unit;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k = 0; k < maxc; ++k) {
      const float4 x = __ldg(part + (u * maxc + k) * per_unit + r);
      acc.x += x.x;
      acc.y += x.y;
      acc.z += x.z;
      acc.w += x.w;
    }
    y[i] = acc;
  }
}

int g_num_sms[64] = {};

}  // namespace

// m <= 256: stacked rows past 128 run as a second pair of passes over the
// keys (row statistics and Y are per row; the prefix scores of the second
// pair are added to the first's).
bool score_tc_supported(const Shape& s) { return s.dtype == GRKV_BF16 && s.m <= 2 * kRows; }

size_t score_tc_pstats_bytes(const Shape& s, int* maxc, int* gu, int* rounds, int sms) {
  const int tpu = (s.n + kTile - 1) / kTile;
  const size_t unit_k = (size_t)s.n * kD * 2;
  const size_t budget = (size_t)64 << 20;   // K of two rounds resident in L2
  int g = (int)std::max<size_t>(1, budget / (2 * unit_k));
  g = std::min(g, s.U);
  const int R = (s.U + g - 1) / g;
  const int last = s.U - (R - 1) * g;
  const long long tmin = (long long)std::min(g, last) * tpu;
  const int mc = (int)std::min<long long>(sms, ((long long)tpu * sms + tmin - 1) / tmin + 2);
  *maxc = mc;
  *gu = g;
  *rounds = R;
  return (size_t)s.U * mc * kRows * sizeof(float2);
}

int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (!g_num_sms[dev] &&
      cudaDeviceGetAttribute(&g_num_sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    g_num_sms[dev] = 0;
  return g_num_sms[dev];
}

cudaError_t launch_score_tc(const Shape& s, const void* q, const void* k, const void* v,
                            float* scores, float* y, float* row_stats, char* ws,
                            const WsLayout& L, int mode, cudaStream_t st) {
  CUtensorMap mq, mk, mv;
  if (!encode_bf16_3d(&mq, q, kD, s.m, s.U, 64, kRows) ||
      !encode_bf16_3d(&mk, k, kD, s.n, s.U, 64, kTile) ||
      !encode_bf16_3d(&mv, v, kD, s.n, s.U, 64, kTile))
    return cudaErrorInvalidValue;
  const int G = sm_count();
  if (G <= 0 || G > kMaxScoreCtas) return cudaErrorInvalidDevice;
  Args a{};
  a.U = s.U;
  a.n = s.n;
  a.w = s.w;
  a.m = s.m;
  a.P = s.P;
  a.causal = s.causal;
  a.tpu = (s.n + kTile - 1) / kTile;
  int maxc, gu, rounds;
  score_tc_pstats_bytes(s, &maxc, &gu, &rounds, G);
  a.maxc = maxc;
  a.gu = gu;
  a.rounds = rounds;
  a.sl2 = (float)((double)s.scale * 1.4426950408889634);
  a.scores = scores;
  a.scores2 = (float*)(ws + L.pooled);   // unused until the selection
  a.y = y;
  a.row_stats = row_stats;
  a.pstats = (float2*)(ws + L.pstats_tc);
  a.unit_cnt = (int*)(ws + L.flags_tc);
  a.status = (int*)(ws + L.status);
  a.ypart = s.deterministic ? (float*)(ws + L.ypart_tc) : nullptr;
  a.test_withhold = s.test_timeout;
  a.wait_budget = s.test_timeout ? kTestWaitBudget : kWaitBudget;
  const size_t part_bytes = (size_t)s.U * maxc * s.m * kD * sizeof(float);
  cudaError_t e = a.ypart ? cudaMemsetAsync(a.ypart, 0, part_bytes, st)
                          : cudaMemsetAsync(y, 0, (size_t)s.U * s.m * kD * sizeof(float), st);
  if (e != cudaSuccess) return e;
  auto launch = [&](int md) {
    a.mode = md;
    a.gu = s.U;
    a.rounds = 1;
    auto kern = k_score_tc<kRingTwo, kQBufTwo>;
    const uint32_t smem = Layout<kRingTwo, kQBufTwo>::kSmemBytes;
    cudaError_t fe = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (fe != cudaSuccess) return fe;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(G);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    count_launches(1);
    return cudaLaunchKernelEx(&cfg, kern, mq, mk, mv, a);
  };
  (void)mode;
  for (int row0 = 0; row0 < s.m; row0 += kRows) {
    a.row0 = row0;
    a.mr = std::min(kRows, s.m - row0);
    a.acc = row0 > 0;
    e = cudaMemsetAsync(a.unit_cnt, 0, (size_t)s.U * sizeof(int), st);
    if (e != cudaSuccess) return e;
    e = launch(0);
    if (e == cudaSuccess) e = launch(1);
    if (e != cudaSuccess) return e;
  }
  if (s.m > kRows) {
    const size_t count = (size_t)s.U * s.P;
    const int blocks = (int)std::min<size_t>((count + 255) / 256, (size_t)G * 8);
    k_add_scores<<<blocks, 256, 0, st>>>(scores, a.scores2, count);
    count_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (a.ypart) {
    const size_t n4 = (size_t)s.U * s.m * kD / 4;
    const int blocks = (int)std::min<size_t>((n4 + 255) / 256, (size_t)G * 8);
    k_y_sum_slots<<<blocks, 256, 0, st>>>((const float4*)a.ypart, (float4*)y, s.U, s.m, maxc);
    count_launches(1);
    e = cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace grkv
