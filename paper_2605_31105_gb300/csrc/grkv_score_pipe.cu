// Window scoring with one read of the key cache from HBM (bf16, d = 128,
// stacked window rows in blocks of 128).
//
// For every unit the path needs the row statistics of the window logits over
// all n keys (pass A: M_r, L_r), and then, with those, the probabilities, the
// per-key prefix scores c_j = sum_r P_rj and the target Y = P V (pass B);
// Eq. 4 and Algorithm 1 of the paper.  The row normaliser depends on every
// key, so the keys are needed twice; this kernel reads them from HBM once and
// serves the second read from L2.
//
// Schedule.  The persistent grid (one CTA per SM) is split into ng groups; a
// group works on the units g, g + ng, g + 2 ng, ... one after another, each CTA
// of the group always on the same token range of the unit.  ng is chosen so
// that the keys of ng units fit in L2.  Phase p of a CTA interleaves pass A of
// the group's unit p with pass B of its unit p - 1: kLead A tiles first, then
// B and A tiles alternately, then the remaining B tiles.  So a unit's keys are
// fetched from HBM by pass A and re-read from L2 by pass B one phase later,
// while at any time about one unit's keys per group are held in L2.  Before
// its first B tile a CTA needs the unit's complete statistics: every CTA of
// the group publishes its rows' (max, sum) into a slot, the last one to
// arrive combines the slots into the rows' log2 normalisers and publishes
// them once; the lead gives the other CTAs of the group time to catch up.
//
// Roles (512 threads): warp 0 issues TMA loads (Q of the pass-B unit, the K
// tile of every job, each pass-B job's V tile right after its K) and L2
// prefetches a few jobs ahead; warp 1 issues the S MMAs of every job; warp 2
// issues the Y^T MMAs of the pass-B tiles (so that no S MMA waits behind a
// probability tile); warp 3 publishes pass-A statistics (and combines them
// in the last CTA) and fetches a unit's normalisers ahead of its pass-B
// tiles; warps 4-11 are two compute groups of 128 threads; warps 12-15 add
// the two groups' halves of every pass-B tile's column scores and flush each
// pass-B segment's Y partial.
//
// Pass A: S = Q K^T (window rows on TMEM lanes, Q as the A operand in TMEM,
// filled by the compute threads).  A compute thread owns one row; the two
// groups split the tile's 128 tokens; running max / sum in registers.
// Pass B, transposed: S^T = K Q^T (tokens on TMEM lanes, Q as the B operand
// in shared memory).  A compute thread owns one token; the two groups split
// the 128 rows.  p = exp2(l * s * log2 e - Lambda_r); the token's column
// score is a sum in registers (the two halves meet in shared memory); P^T is
// written as bf16 into the K tile's ring slot, which the S^T MMA has finished
// reading, and becomes the MN-major B operand of Y^T += V^T P^T.  Y^T (lanes
// = d, columns = rows) is added to the unit's Y with fp32 reductions at the
// end of the CTA's pass-B segment.
#include <algorithm>
#include <climits>
#include <cmath>

#include "grkv_internal.cuh"
#include "sm100.cuh"
#include "tmap.cuh"

namespace grkv {
namespace {

using namespace sm100;

constexpr int kTile = 128;      // tokens per tile
constexpr int kRows = 128;      // window rows per launch (row block)
constexpr int kThreads = 512;
constexpr int kRing = 5;        // K / V ring slots
constexpr int kSBufs = 2;       // S tiles in TMEM
constexpr int kLead = 8;        // pass-A tiles of a phase ahead of its first pass-B tile
constexpr int kRedBufs = 4;
constexpr int kPrefetch = 4;    // jobs whose K / V tiles are prefetched into L2 ahead of their loads     // column-score buffers (pass-B tiles in flight to the summers)
constexpr uint32_t kTileBytes = kTile * kD * 2;    // 32 KB
constexpr long long kWaitBudget = 1ll << 32;       // cycles (~2 s) before a wait gives up
constexpr long long kTestWaitBudget = 1ll << 22;   // ~2 ms: the budget of GRKV_TEST_TIMEOUT
constexpr size_t kL2KeyBudget = (size_t)72 << 20;  // keys of the units in flight

// Shared memory (offsets from a 1024-byte aligned base).
constexpr uint32_t kOffQ = 0;                                   // Q of the pass-B unit, 32 KB
constexpr uint32_t kOffRing = kOffQ + kTileBytes;               // kRing x 32 KB
constexpr uint32_t kOffRed = kOffRing + kRing * kTileBytes;     // [kRedBufs][2 wg][128] fp32
constexpr uint32_t kOffAstat = kOffRed + kRedBufs * 2 * kTile * 4;   // [2 buf][2 wg][128] float2
constexpr uint32_t kOffLam = kOffAstat + 2 * 2 * kRows * 8;     // [2 buf][128] fp32
constexpr uint32_t kOffBar = kOffLam + 2 * kRows * 4;
constexpr uint32_t kSmemBytes = kOffBar + 512 + 1024;           // + alignment slack
static_assert(kSmemBytes <= 227 * 1024, "shared memory");

// TMEM columns: two S buffers, the Y^T accumulator, two Q buffers of the
// pass-A unit (bf16 pairs, the A operand of S = Q K^T).
constexpr uint32_t kColS = 0, kColY = kSBufs * kTile, kColQ = kColY + kD;
static_assert(kColQ + 2 * 64 <= 512, "TMEM columns");

struct Args {
  int U, n, w, m, P, causal;
  int row0, mr;      // stacked rows row0 .. row0 + mr - 1 (mr <= 128) in this launch
  int acc;           // add the prefix scores to those of an earlier launch
  int tpu;           // tiles per unit
  int ng;            // CTA groups
  int maxgs;         // statistics slots per unit (largest group)
  float sl2;         // scale * log2(e)
  const __nv_bfloat16* q;   // [U][m][128]
  float* scores;     // [U][P]
  float* y;          // [U][m][128], zeroed by the host
  float* row_stats;  // [U][m][2]
  float2* pstats;    // [U][maxgs][128]  per-CTA (max in log2 units, sum)
  float* lam;        // [U][128]         combined log2 normalisers
  int* unit_cnt;     // [U] slots written (+1 once combined), zeroed by the host
  int* status;
  long long wait_budget;   // cycles before a bounded wait gives up
  int test_withhold;       // GRKV_TEST_TIMEOUT: CTA 0 withholds one arrive
};

// The group of CTA c, its index inside the group and the group's size: group
// g holds CTAs [G g / ng, G (g + 1) / ng).
struct Group {
  int g, i, size;
  __device__ Group(int c, int G, int ng) {
    g = (int)(((long long)(c + 1) * ng - 1) / G);
    const int b0 = (int)((long long)G * g / ng), b1 = (int)((long long)G * (g + 1) / ng);
    i = c - b0;
    size = b1 - b0;
  }
};

// First tile of CTA i's token range in a group of `size` CTAs.
__host__ __device__ __forceinline__ int range_begin(int tpu, int i, int size) {
  return (int)((long long)tpu * i / size);
}

struct Job {
  int kind;          // 0 = pass A, 1 = pass B
  int u;             // unit
  int j0, len;       // first token, tokens in the tile
  bool first, last;  // first / last tile of the CTA's segment of this unit
};

// The CTA's job sequence; every role walks the same one.
struct JobIter {
  int U, n, ng, g, t0, T, nu;
  int p, ia, ib;
  __device__ void init(const Args& a, const Group& gr) {
    U = a.U;
    n = a.n;
    ng = a.ng;
    g = gr.g;
    t0 = range_begin(a.tpu, gr.i, gr.size);
    T = range_begin(a.tpu, gr.i + 1, gr.size) - t0;
    nu = g < U ? (U - g + ng - 1) / ng : 0;
    p = 0;
    ia = ib = 0;
  }
  __device__ bool next(Job* j) {
    if (T <= 0) return false;
    int na, nb;
    while (true) {
      if (p > nu) return false;
      na = p < nu ? T : 0;
      nb = p >= 1 ? T : 0;
      if (ia + ib < na + nb) break;
      ++p;
      ia = ib = 0;
    }
    const bool take_a = ia < na && (ib >= nb || ia < kLead || ib > ia - kLead);
    const int ti = take_a ? ia++ : ib++;
    j->kind = take_a ? 0 : 1;
    j->u = g + ng * (take_a ? p : p - 1);
    j->j0 = (t0 + ti) * kTile;
    j->len = min(kTile, n - j->j0);
    j->first = ti == 0;
    j->last = ti == T - 1;
    return true;
  }
};

// mbar_wait for all 32 lanes of a warp with one answer: a lane that sees the
// abort flag makes the whole warp give up, so warp-collective instructions
// (tcgen05.ld / st, shuffles) that follow a wait are reached by all lanes or
// by none.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort,
                                               long long budget) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort, budget));
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

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

// Pass A on 32 logits of one row: online max / sum of exp2 in log2 units.
// The masked form (tiles at the window or the end of the unit, rows past m)
// is a separate instantiation, so the common path carries no mask.
template <bool kMasked>
__device__ __forceinline__ void stats_chunk(float* v, int j0, int lim, int n, bool row_ok,
                                            float sl2, float& M, float& L) {
  if (kMasked) {
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

// Pass B for this thread's token over 32 window rows r0 .. r0 + 31 (one TMEM
// load): v = exp2(l * s * log2 e - Lambda_r), and their sum.  Masked form:
// zero where the token is past the unit's end (!tok) or, causally, where
// r % w < thr = token - (n - w); am = r0 % w.
template <bool kMasked>
__device__ __forceinline__ float probs32(float* v, const float* lam, float sl2, bool tok, int thr,
                                         int am, int w) {
  float cs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e4 = 0; e4 < 8; ++e4) {
    const float4 l4 = *reinterpret_cast<const float4*>(lam + 4 * e4);
    const float lv[4] = {l4.x, l4.y, l4.z, l4.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float x = fast_exp2(fmaf(v[4 * e4 + e], sl2, -lv[e]));
      if (kMasked) {
        if (!tok || am < thr) x = 0.f;
        am = am + 1 == w ? 0 : am + 1;
      }
      v[4 * e4 + e] = x;
      cs[e] += x;
    }
  }
  return (cs[0] + cs[1]) + (cs[2] + cs[3]);
}

// 32 probabilities of this thread's token as bf16 into its P^T row: chunks
// c0 .. c0 + 3 (eight rows each) of the 128-byte row, 128-byte swizzle.
__device__ __forceinline__ void store_pt(uint32_t row_addr, int lr, int c0, const float* v) {
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    const uint32_t w0 = pack_bf16(v[8 * c], v[8 * c + 1]), w1 = pack_bf16(v[8 * c + 2], v[8 * c + 3]);
    const uint32_t w2 = pack_bf16(v[8 * c + 4], v[8 * c + 5]), w3 = pack_bf16(v[8 * c + 6], v[8 * c + 7]);
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                     row_addr + (((c0 + c) ^ (lr & 7)) << 4)),
                 "r"(w0), "r"(w1), "r"(w2), "r"(w3)
                 : "memory");
  }
}

// Merges two (max, sum) row statistics in log2 units.
__device__ __forceinline__ float2 stat_merge(float2 x, float2 y) {
  if (x.x == -INFINITY) return y;
  if (y.x == -INFINITY) return x;
  const float M = fmaxf(x.x, y.x);
  return make_float2(M, x.y * fast_exp2(x.x - M) + y.y * fast_exp2(y.x - M));
}

struct Bars {
  uint64_t ring_full[kRing], ring_empty[kRing];
  uint64_t q_full, q_empty;          // Q of the pass-B unit (shared memory)
  uint64_t qa_full[2], qa_empty[2];  // Q of the pass-A unit (TMEM)
  uint64_t s_full[kSBufs], s_done[kSBufs];
  uint64_t p_full[4];                // P^T written (pass-B tile nb uses nb % 4)
  uint64_t y_full, y_empty;
  uint64_t astat_full[2], astat_empty[2];
  uint64_t lam_full[2], lam_empty[2];
  uint64_t red_full[kRedBufs], red_empty[kRedBufs];  // column-score halves of a pass-B tile
  uint64_t drain, drain_y;
  uint32_t tmem;
  int abort;
};
static_assert(sizeof(Bars) <= 512, "barrier block");


__global__ void __launch_bounds__(kThreads, 1)
    k_score_pipe(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, Args a) {
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  Bars* bars = (Bars*)(sm + kOffBar);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const Group gr((int)blockIdx.x, (int)gridDim.x, a.ng);

  if (tid == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&bars->ring_full[i], 1);
      mbar_init(&bars->ring_empty[i], 1);
    }
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int i = 0; i < kSBufs; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_done[i], 256);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->qa_full[i], 256);
      mbar_init(&bars->qa_empty[i], 1);
      mbar_init(&bars->astat_full[i], 256);
      mbar_init(&bars->astat_empty[i], 1);
      mbar_init(&bars->lam_full[i], 1);
      mbar_init(&bars->lam_empty[i], 256);
    }
    // four P^T barriers, one per pass-B tile in flight: the ring holds the K
    // and V of at most two pass-B tiles whose Y^T MMA has not completed
    for (int i = 0; i < 4; ++i) mbar_init(&bars->p_full[i], 256);
    for (int i = 0; i < kRedBufs; ++i) {
      mbar_init(&bars->red_full[i], 256);
      mbar_init(&bars->red_empty[i], 128);
    }
    mbar_init(&bars->y_full, 1);
    mbar_init(&bars->y_empty, 128);
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->drain_y, 1);
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
  // statistics slots a unit receives: one per CTA of the group with tiles
  const int writers = min(gr.size, a.tpu);

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      prefetch_tensormap(&tmQ);
      prefetch_tensormap(&tmK);
      prefetch_tensormap(&tmV);
      // pass-A keys stay in L2 for their pass-B re-read; everything else streams
      const uint64_t keep = l2_evict_last(), stream = l2_evict_first(), normal = l2_evict_normal();
      JobIter it;
      it.init(a, gr);
      uint32_t slot = 0, ring_use = 0;
      int q_loads = 0;
      bool ok = true;
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
      // L2 prefetches run kPrefetch jobs ahead of the ring loads, so a load
      // that waited for its ring slot finds its tile in L2
      JobIter pf;
      pf.init(a, gr);
      int pf_ahead = 0;
      Job j, jp;
      while (ok && it.next(&j)) {
        for (; pf_ahead <= kPrefetch && pf.next(&jp); ++pf_ahead) {
          const uint64_t pol = jp.kind == 0 ? keep : normal;
          tma_prefetch_3d(&tmK, 0, jp.j0, jp.u, pol);
          tma_prefetch_3d(&tmK, 64, jp.j0, jp.u, pol);
          if (jp.kind == 1) {
            tma_prefetch_3d(&tmV, 0, jp.j0, jp.u, normal);
            tma_prefetch_3d(&tmV, 64, jp.j0, jp.u, normal);
          }
        }
        --pf_ahead;
        if (j.kind == 1 && j.first) {
          // Q of the pass-B unit, once the previous pass-B segment's MMAs are done
          if (q_loads >= 1)
            ok = mbar_wait(&bars->q_empty, (q_loads - 1) & 1, abort_flag, a.wait_budget);
          if (!ok) break;
          mbar_expect_tx(&bars->q_full, kTileBytes);
          tma_load_3d(sm + kOffQ, &tmQ, &bars->q_full, 0, a.row0, j.u, keep);
          tma_load_3d(sm + kOffQ + kTileBytes / 2, &tmQ, &bars->q_full, 64, a.row0, j.u, keep);
          ++q_loads;
        }
        // a pass-B job's V right after its K (both stay in the ring until
        // the job's Y^T MMA has read them)
        ok = load(&tmK, j.j0, j.u, j.kind == 0 ? keep : stream);
        if (ok && j.kind == 1) ok = load(&tmV, j.j0, j.u, stream);
      }
      // every issued load lands before the CTA can exit (these waits ignore
      // the abort flag, and are bounded)
      volatile int no_abort = 0;
      for (uint32_t i = ring_use > kRing ? ring_use - kRing : 0; i < ring_use; ++i)
        mbar_wait(&bars->ring_full[i % kRing], (i / kRing) & 1, &no_abort, a.wait_budget);
      if (q_loads > 0) mbar_wait(&bars->q_full, (q_loads - 1) & 1, &no_abort, a.wait_budget);
      if (!ok) set_status(a.status, GRKV_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------ S MMA issuer
    // S = Q K^T (pass A, Q in TMEM) or S^T = K Q^T (pass B, Q in shared
    // memory) of every job, as soon as the K tile has landed and the S
    // buffer is free; the Y^T MMAs are issued by warp 2, so an S MMA never
    // waits for a probability tile.
    if (lane == 0) {
      const uint32_t id_a = idesc_bf16(kRows, kTile, 0, 0);   // S = Q K^T
      const uint32_t id_b = idesc_bf16(kTile, kRows, 0, 0);   // S^T = K Q^T
      JobIter it;
      it.init(a, gr);
      uint32_t ring_use = 0;
      int i = 0, aseg = 0, bseg = 0;
      bool ok = true;
      Job j;
      while (ok && it.next(&j)) {
        const int b = i % kSBufs, use = i / kSBufs;
        const uint32_t kuse = ring_use, kslot = kuse % kRing;
        ring_use += j.kind == 1 ? 2 : 1;   // a pass-B job's V follows its K
        if (j.first) {
          if (j.kind == 0)
            ok = mbar_wait(&bars->qa_full[aseg & 1], (aseg >> 1) & 1, abort_flag, a.wait_budget);
          else
            ok = mbar_wait(&bars->q_full, bseg & 1, abort_flag, a.wait_budget);
        }
        if (ok) ok = mbar_wait(&bars->ring_full[kslot], (kuse / kRing) & 1, abort_flag, a.wait_budget);
        if (ok && use >= 1)
          ok = mbar_wait(&bars->s_done[b], (use - 1) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t ka = smem_u32(sm + kOffRing + kslot * kTileBytes);
        if (j.kind == 0) {
          const uint32_t qcol = tmem + kColQ + (aseg & 1) * 64;
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
            mma_bf16_ts(tmem + kColS + b * kTile, qcol + kk * 8, sw128_desc(ka + off, 16, 1024),
                        id_a, kk > 0);
          }
          mma_commit(&bars->ring_empty[kslot]);
          mma_commit(&bars->s_full[b]);
          if (j.last) {
            mma_commit(&bars->qa_empty[aseg & 1]);
            ++aseg;
          }
        } else {
          const uint32_t qa = smem_u32(sm + kOffQ);
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
            mma_bf16(tmem + kColS + b * kTile, sw128_desc(ka + off, 16, 1024),
                     sw128_desc(qa + off, 16, 1024), id_b, kk > 0);
          }
          // the K slot then takes the tile's P^T; warp 2 releases it
          mma_commit(&bars->s_full[b]);
          if (j.last) {
            mma_commit(&bars->q_empty);
            ++bseg;
          }
        }
        ++i;
      }
      // every MMA issued so far completes before TMEM can be released (this
      // wait ignores the abort flag, and is bounded)
      mma_commit(&bars->drain);
      volatile int no_abort = 0;
      mbar_wait(&bars->drain, 0, &no_abort, a.wait_budget);
      if (!ok) set_status(a.status, GRKV_ERR_TIMEOUT);
    }
  } else if (warp == 2) {
    // ---------------------------------------------------- Y^T MMA issuer
    // Y^T += V^T P^T of every pass-B tile once its P^T is written (into the
    // tile's K slot) and its V has landed; releases both slots.
    if (lane == 0) {
      const uint32_t id_y = idesc_bf16(kD, kRows, 1, 1);   // V^T and P^T both MN-major
      JobIter it;
      it.init(a, gr);
      uint32_t ring_use = 0;
      int nb = 0, y_uses = 0;
      bool ok = true;
      Job j;
      while (ok && it.next(&j)) {
        const uint32_t kuse = ring_use;
        ring_use += j.kind == 1 ? 2 : 1;
        if (j.kind != 1) continue;
        const uint32_t kslot = kuse % kRing, vuse = kuse + 1, vslot = vuse % kRing;
        if (j.first && y_uses >= 1)
          ok = mbar_wait(&bars->y_empty, (y_uses - 1) & 1, abort_flag, a.wait_budget);
        if (ok) ok = mbar_wait(&bars->p_full[nb & 3], (nb >> 2) & 1, abort_flag, a.wait_budget);
        if (ok) ok = mbar_wait(&bars->ring_full[vslot], (vuse / kRing) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t va = smem_u32(sm + kOffRing + vslot * kTileBytes);
        const uint32_t pa = smem_u32(sm + kOffRing + kslot * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk)
          mma_bf16(tmem + kColY, sw128_desc(va + kk * 2048, kTileBytes / 2, 1024),
                   sw128_desc(pa + kk * 2048, kTileBytes / 2, 1024), id_y,
                   (j.first && kk == 0) ? 0u : 1u);
        mma_commit(&bars->ring_empty[vslot]);
        mma_commit(&bars->ring_empty[kslot]);
        if (j.last) {
          mma_commit(&bars->y_full);
          ++y_uses;
        }
        ++nb;
      }
      mma_commit(&bars->drain_y);
      volatile int no_abort = 0;
      mbar_wait(&bars->drain_y, 0, &no_abort, a.wait_budget);
      if (!ok) set_status(a.status, GRKV_ERR_TIMEOUT);
    }
  } else if (warp == 3) {
    // ------------------------------------------------- row statistics
    // In job order: at the end of each pass-A segment, merges the two
    // compute groups' statistics into this CTA's slot of the unit and
    // counts it (the CTA whose count completes the unit combines all slots,
    // in slot order, into the rows' log2 normalisers and the row statistics,
    // then counts once more); ahead of each pass-B segment, waits (bounded)
    // until the unit's normalisers are published and leaves them in shared
    // memory.  A unit's pass-A segment precedes its pass-B segment in every
    // CTA's job order, so the two duties share one warp without waiting on
    // each other.
    const float2* astat = (const float2*)(sm + kOffAstat);
    float* lam_s = (float*)(sm + kOffLam);
    JobIter it;
    it.init(a, gr);
    int aseg = 0, bseg = 0;
    bool ok = true;
    Job j;
    while (ok && it.next(&j)) {
      if (j.kind == 0 && j.last) {
        const int ab = aseg & 1;
        ok = mbar_wait_warp(&bars->astat_full[ab], (aseg >> 1) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        float2* mine = a.pstats + ((size_t)j.u * a.maxgs + gr.i) * kRows;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int r = t * 32 + lane;
          mine[r] = stat_merge(astat[(ab * 2 + 0) * kRows + r], astat[(ab * 2 + 1) * kRows + r]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->astat_empty[ab]);
        __threadfence();
        __syncwarp();
        int old = 0;
        if (lane == 0) old = atomicAdd(&a.unit_cnt[j.u], 1);
        old = __shfl_sync(0xffffffffu, old, 0);
        if (old == writers - 1) {
          __threadfence();
          float2 st[4];
#pragma unroll
          for (int t = 0; t < 4; ++t) st[t] = make_float2(-INFINITY, 0.f);
          // eight slots per round trip: 32 independent loads in flight per lane
          for (int k0 = 0; k0 < gr.size; k0 += 8) {
            float2 pr[8][4];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const int k = k0 + kk;
              const bool use = k < gr.size && range_begin(a.tpu, k + 1, gr.size) >
                                                  range_begin(a.tpu, k, gr.size);
              const float2* sl = a.pstats + ((size_t)j.u * a.maxgs + (use ? k : 0)) * kRows;
#pragma unroll
              for (int t = 0; t < 4; ++t)
                pr[kk][t] = use ? __ldcg(sl + t * 32 + lane) : make_float2(-INFINITY, 0.f);
            }
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
#pragma unroll
              for (int t = 0; t < 4; ++t) st[t] = stat_merge(st[t], pr[kk][t]);
          }
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const int r = t * 32 + lane;
            const bool live = r < a.mr && st[t].y > 0.f;
            a.lam[(size_t)j.u * kRows + r] = live ? st[t].x + __log2f(st[t].y) : INFINITY;
            if (r < a.mr) {
              float* rs = a.row_stats + ((size_t)j.u * a.m + a.row0 + r) * 2;
              rs[0] = st[t].x * 0.69314718055994531f;
              rs[1] = st[t].y;
            }
          }
          __threadfence();
          __syncwarp();
          if (lane == 0) atomicAdd(&a.unit_cnt[j.u], 1);
        }
        ++aseg;
      } else if (j.kind == 1 && j.first) {
        const int lb = bseg & 1;
        if (bseg >= 2)
          ok = mbar_wait_warp(&bars->lam_empty[lb], ((bseg >> 1) - 1) & 1, abort_flag,
                              a.wait_budget);
        if (!ok) break;
        const long long t0 = clock64();
        while (ld_acquire(&a.unit_cnt[j.u]) < writers + 1) {
          if (*abort_flag || clock64() - t0 > a.wait_budget) {
            *abort_flag = 1;
            ok = false;
            break;
          }
          __nanosleep(64);
        }
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
#pragma unroll
        for (int t = 0; t < 4; ++t)
          lam_s[lb * kRows + t * 32 + lane] = __ldcg(a.lam + (size_t)j.u * kRows + t * 32 + lane);
        __syncwarp();
        // GRKV_TEST_TIMEOUT: CTA 0 never announces its first pass-B
        // normalisers, so its compute groups' bounded wait expires
        if (lane == 0 && !(a.test_withhold && blockIdx.x == 0 && bseg == 0))
          mbar_arrive(&bars->lam_full[lb]);
        ++bseg;
      }
    }
    if (!ok && lane == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  } else if (warp >= 12) {
    // ------------------------------------------- column scores and Y^T flush
    // Thread t (token t of a tile, d = t of Y^T): for every pass-B tile, adds
    // the two compute groups' halves of the token's column score (group 0's
    // rows first) and writes the score; at the end of each pass-B segment,
    // adds the segment's 128 Y^T row columns to Y[u][row][d] with fp32
    // reductions (consecutive d per warp).
    const int q = warp & 3, t = q * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    const float* red = (const float*)(sm + kOffRed);
    JobIter it;
    it.init(a, gr);
    int bseg = 0, nb = 0;
    bool ok = true;
    Job j;
    while (ok && it.next(&j)) {
      if (j.kind != 1) continue;
      const int rb = nb % kRedBufs;
      ok = mbar_wait_warp(&bars->red_full[rb], (nb / kRedBufs) & 1, abort_flag, a.wait_budget);
      if (!ok) break;
      const float c2 = red[(rb * 2) * kTile + t] + red[(rb * 2 + 1) * kTile + t];
      mbar_arrive(&bars->red_empty[rb]);
      ++nb;
      const int jt = j.j0 + t;
      if (t < j.len && jt < a.P) {
        float* dst = a.scores + (size_t)j.u * a.P + jt;
        *dst = a.acc ? *dst + c2 : c2;
      }
      if (!j.last) continue;
      ok = mbar_wait_warp(&bars->y_full, bseg & 1, abort_flag, a.wait_budget);
      if (!ok) break;
      tc_fence_after();
      float* yu = a.y + ((size_t)j.u * a.m + a.row0) * kD + t;
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(lane_addr + kColY + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (c * 32 + e < a.mr) atomicAdd(yu + (size_t)(c * 32 + e) * kD, v[e]);
      }
      tc_fence_before();
      mbar_arrive(&bars->y_empty);
      ++bseg;
    }
    if (!ok && lane == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  } else if (warp >= 4) {
    // ------------------------------------------------------- compute groups
    const int wg = (warp - 4) >> 2, q = warp & 3;
    const int lr = q * 32 + lane;   // TMEM lane: a window row in pass A, a token in pass B
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    float2* astat = (float2*)(sm + kOffAstat);
    const float* lam_s = (const float*)(sm + kOffLam);
    float* red = (float*)(sm + kOffRed);
    const bool row_ok = lr < a.mr;
    const int lim = a.causal ? a.n - a.w + (row_ok ? (a.row0 + lr) % a.w : 0) : a.n - 1;
    JobIter it;
    it.init(a, gr);
    bool ok = true;
    // Q of pass-A segment s into TMEM buffer s & 1: this thread's row, this
    // group's half of d, as packed bf16 pairs (the MMA's A-operand layout)
    auto fill_q = [&](int s) -> bool {
      const int buf = s & 1;
      if (s >= 2 &&
          !mbar_wait_warp(&bars->qa_empty[buf], ((s >> 1) - 1) & 1, abort_flag, a.wait_budget))
        return false;
      tc_fence_after();
      const int u = gr.g + a.ng * s;
      uint32_t wv[32];
      if (row_ok) {
        const uint4* src =
            reinterpret_cast<const uint4*>(a.q + ((size_t)u * a.m + a.row0 + lr) * kD + 64 * wg);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint4 x = __ldg(src + c);
          wv[4 * c] = x.x;
          wv[4 * c + 1] = x.y;
          wv[4 * c + 2] = x.z;
          wv[4 * c + 3] = x.w;
        }
      } else {
#pragma unroll
        for (int c = 0; c < 32; ++c) wv[c] = 0u;
      }
      const uint32_t qcol = lane_addr + kColQ + buf * 64 + 32 * wg;
      tmem_st16(qcol, wv);
      tmem_st16(qcol + 16, wv + 16);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&bars->qa_full[buf]);
      return true;
    };
    if (it.T > 0 && it.nu > 0) ok = fill_q(0);
    int i = 0, aseg = 0, bseg = 0, nb = 0;
    uint32_t ring_use = 0;
    // causal visibility of this thread's token in pass B: row r sees it iff
    // r % w >= token - (n - w); am0 / am1 = first row of each 32-row half mod w
    const int am0 = (a.row0 + 64 * wg) % a.w, am1 = (a.row0 + 64 * wg + 32) % a.w;
    float M = -INFINITY, L = 0.f;   // pass-A running stats of this row (log2 units)
    Job j;
    while (ok && it.next(&j)) {
      const int b = i % kSBufs, sp = (i / kSBufs) & 1;
      // ring slot of this job's K tile (the producer's count: a pass-B job's V
      // follows its K); a pass-B tile's P^T goes into its K slot
      const uint32_t kslot = ring_use % kRing;
      ring_use += j.kind == 1 ? 2 : 1;
      if (j.kind == 0) {
        // ---- pass A: this thread's row over the group's 64 tokens
        if (j.first) {
          M = -INFINITY;
          L = 0.f;
          if (aseg + 1 < it.nu && !(ok = fill_q(aseg + 1))) break;
        }
        ok = mbar_wait_warp(&bars->s_full[b], sp, abort_flag, a.wait_budget);
        if (!ok) break;
        tc_fence_after();
        const int t0 = j.j0 + 64 * wg;
        const uint32_t sbase = lane_addr + kColS + b * kTile + 64 * wg;
        // halves away from the window and the end of the unit need no mask
        const bool full = row_ok && t0 + 63 <= lim && t0 + 64 <= a.n;
        float va[32], vb[32];
        tmem_ld32f(sbase, va);
        tmem_wait32(va);
        tmem_ld32f(sbase + 32, vb);
        if (full) stats_chunk<false>(va, t0, lim, a.n, row_ok, a.sl2, M, L);
        else stats_chunk<true>(va, t0, lim, a.n, row_ok, a.sl2, M, L);
        tmem_wait32(vb);
        tc_fence_before();
        mbar_arrive(&bars->s_done[b]);   // S fully read
        if (full) stats_chunk<false>(vb, t0 + 32, lim, a.n, row_ok, a.sl2, M, L);
        else stats_chunk<true>(vb, t0 + 32, lim, a.n, row_ok, a.sl2, M, L);
        if (j.last) {
          const int ab = aseg & 1;
          if (aseg >= 2)
            ok = mbar_wait_warp(&bars->astat_empty[ab], ((aseg >> 1) - 1) & 1, abort_flag,
                           a.wait_budget);
          if (!ok) break;
          astat[(ab * 2 + wg) * kRows + lr] = make_float2(M, L);
          mbar_arrive(&bars->astat_full[ab]);
          ++aseg;
        }
      } else {
        // ---- pass B: this thread's token over the group's 64 rows
        const int lb = bseg & 1;
        if (j.first) {
          ok = mbar_wait_warp(&bars->lam_full[lb], (bseg >> 1) & 1, abort_flag, a.wait_budget);
          if (!ok) break;
        }
        ok = mbar_wait_warp(&bars->s_full[b], sp, abort_flag, a.wait_budget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t sbase = lane_addr + kColS + b * kTile + 64 * wg;
        const int jt = j.j0 + lr;
        const bool tok = lr < j.len;
        // tokens before the window are seen by every row (rows past mr have
        // Lambda = +inf and give 0)
        const bool full = tok && (!a.causal || jt <= a.n - a.w);
        const int thr = a.causal ? jt - (a.n - a.w) : INT_MIN;
        const float* lam = lam_s + lb * kRows + 64 * wg;
        // P^T row of this token (MN-major, 128-byte swizzle: half wg holds
        // rows 64 wg .. 64 wg + 63)
        const uint32_t pT =
            smem_u32(sm + kOffRing + kslot * kTileBytes) + wg * (kTileBytes / 2) + lr * 128;
        float va[32], vb[32], csum;
        tmem_ld32f(sbase, va);
        tmem_wait32(va);
        tmem_ld32f(sbase + 32, vb);
        csum = full ? probs32<false>(va, lam, a.sl2, tok, thr, am0, a.w)
                    : probs32<true>(va, lam, a.sl2, tok, thr, am0, a.w);
        store_pt(pT, lr, 0, va);
        tmem_wait32(vb);
        tc_fence_before();
        mbar_arrive(&bars->s_done[b]);   // S^T fully read
        csum += full ? probs32<false>(vb, lam + 32, a.sl2, tok, thr, am1, a.w)
                     : probs32<true>(vb, lam + 32, a.sl2, tok, thr, am1, a.w);
        store_pt(pT, lr, 4, vb);
        fence_proxy_async_smem();
        mbar_arrive(&bars->p_full[nb & 3]);
        // this group's half of the token's column score, for the summers
        const int rb = nb % kRedBufs;
        if (nb >= kRedBufs)
          ok = mbar_wait_warp(&bars->red_empty[rb], ((nb / kRedBufs) - 1) & 1, abort_flag, a.wait_budget);
        if (!ok) break;
        red[(rb * 2 + wg) * kTile + lr] = csum;
        mbar_arrive(&bars->red_full[rb]);
        ++nb;
        if (j.last) {
          mbar_arrive(&bars->lam_empty[lb]);
          ++bseg;
        }
      }
      ++i;
    }
    if (!ok && lr == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

}  // namespace

// Groups and group size for a grid of at most G CTAs.  At most
// kL2KeyBudget of keys may be in flight (one unit per group); within that,
// the plan minimises the modelled time: phases (units per group + 1) x
// (tiles per CTA and phase + two tiles' worth of statistics exchange), where
// a group whose CTAs hold unequal tile counts pays 15% (every CTA of a group
// waits for its slowest one at each phase).
PipePlan score_pipe_plan(const Shape& s, int G) {
  const int tpu = (s.n + kTile - 1) / kTile;
  const size_t unit_k = (size_t)s.n * kD * 2;
  const int ng_max = (int)std::min<size_t>(std::max<size_t>(1, kL2KeyBudget / unit_k),
                                           (size_t)std::max(1, std::min(s.U, G)));
  PipePlan best{1, std::max(1, G)};
  double best_t = 1e300;
  for (int ng = 1; ng <= ng_max; ++ng) {
    for (int gs = 1; gs * ng <= G; ++gs) {
      const double t = (double)((s.U + ng - 1) / ng + 1) *
                       ((tpu + gs - 1) / gs * (tpu % gs == 0 || tpu < gs ? 1.0 : 1.15) + 2.0);
      if (t < best_t * (1 - 1e-9) || (t <= best_t * (1 + 1e-9) && ng * gs > best.ng * best.gs)) {
        best_t = t;
        best = PipePlan{ng, gs};
      }
    }
  }
  return best;
}

size_t score_pipe_slot_bytes(const Shape& s) {
  const int G = sm_count();
  const PipePlan pl = score_pipe_plan(s, G > 0 ? G : kMaxScoreCtas);
  return (size_t)s.U * pl.gs * kRows * sizeof(float2);
}

cudaError_t launch_score_pipe(const Shape& s, const void* q, const void* k, const void* v,
                              float* scores, float* y, float* row_stats, char* ws,
                              const WsLayout& L, cudaStream_t st) {
  CUtensorMap mq, mk, mv;
  if (!encode_bf16_3d(&mq, q, kD, s.m, s.U, 64, kRows) ||
      !encode_bf16_3d(&mk, k, kD, s.n, s.U, 64, kTile) ||
      !encode_bf16_3d(&mv, v, kD, s.n, s.U, 64, kTile))
    return cudaErrorInvalidValue;
  const int sms = sm_count();
  if (sms <= 0 || sms > kMaxScoreCtas) return cudaErrorInvalidDevice;
  const PipePlan pl = score_pipe_plan(s, sms);
  const int G = pl.ng * pl.gs;   // the grid: ng groups of gs CTAs
  Args a{};
  a.U = s.U;
  a.n = s.n;
  a.w = s.w;
  a.m = s.m;
  a.P = s.P;
  a.causal = s.causal;
  a.tpu = (s.n + kTile - 1) / kTile;
  a.ng = pl.ng;
  a.maxgs = pl.gs;
  a.sl2 = (float)((double)s.scale * 1.4426950408889634);
  a.q = (const __nv_bfloat16*)q;
  a.scores = scores;
  a.y = y;
  a.row_stats = row_stats;
  a.pstats = (float2*)(ws + L.pstats_tc);
  a.lam = (float*)(ws + L.lam_tc);
  a.unit_cnt = (int*)(ws + L.flags_tc);
  a.status = (int*)(ws + L.status);
  a.test_withhold = s.test_timeout;
  a.wait_budget = s.test_timeout ? kTestWaitBudget : kWaitBudget;
  cudaError_t e = cudaMemsetAsync(y, 0, (size_t)s.U * s.m * kD * sizeof(float), st);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_score_pipe, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)kSmemBytes);
  if (e != cudaSuccess) return e;
  for (int row0 = 0; row0 < s.m; row0 += kRows) {
    a.row0 = row0;
    a.mr = std::min(kRows, s.m - row0);
    a.acc = row0 > 0;
    e = cudaMemsetAsync(a.unit_cnt, 0, (size_t)s.U * sizeof(int), st);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(G);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = st;
    // the CTAs of a group wait for one another: all of them must be resident
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    count_launches(1);
    e = cudaLaunchKernelEx(&cfg, k_score_pipe, mq, mk, mv, a);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace grkv
