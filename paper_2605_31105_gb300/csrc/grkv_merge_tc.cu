// GRKV value step on the tensor cores (bf16, d = 128, m <= 128, B <= 32768).
//
// One CTA per unit; Algorithm 1's value step in dual form (Sec. 3.4,
// App. D.1) with the fixed tokens of App. D.3:
//   phase 1  row max / sum of the retained logits l = s Q K0^T  (K0 gathered
//            with TMA gather4 from the positions idx);
//   phase 2  X = softmax over the retained keys; R~ += Xh V0 and the Gram
//            G += XGh XGh^T + (2 XGl) XGh^T on the tensor cores, where Xh, Xl
//            are the bf16 high / low parts of X and XG is X with the fixed
//            columns zeroed (N = (G + G^T) / 2 restores all three cross terms);
//   phase 3  in shared memory, fp32: N = sym(G) + lambda I, blocked Cholesky,
//            R = Y - R~, Z = N^-1 R by blocked triangular solves; Z^T (high and
//            low bf16 parts) goes to TMEM as an MMA operand;
//   phase 4  per tile D = Zh^T XGh + Zl^T XGh + Zh^T XGl = (dV)^T on the tensor
//            cores, and V_out = V0 + dV (fixed rows get exactly V0, their XG
//            columns are zero), K_out = K0.
// Roles (384 threads): warp 0 TMA, warp 1 MMA issue, warps 4-7 one thread per
// window row (TMEM lane), warps 8-11 the output epilogue; all warps share the
// shared-memory solve.
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
constexpr int kRing = 3;
constexpr int kThreads = 384;
constexpr uint32_t kTileBytes = kTile * kD * 2;   // 32 KB
constexpr int kMaxB = 32768;
constexpr long long kBudget = 1ll << 32;

constexpr int kLD = 129;   // fp32 row stride of N, R/Z and the epilogue stage

// Shared memory (offsets from a 1024-byte aligned base).
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffRing = kOffQ + kTileBytes;              // 3 x 32 KB gathered tiles
constexpr uint32_t kOffXG = kOffRing + kRing * kTileBytes;     // 2 x 32 KB
constexpr uint32_t kOffStage = kOffXG + 2 * kTileBytes;        // 32 tokens x 129 fp32
constexpr uint32_t kOffMask = kOffStage + 32 * kLD * 4;        // fixed-token bits
constexpr uint32_t kOffMisc = kOffMask + kMaxB / 8;            // hist[256], sh[64]
constexpr uint32_t kOffBar = kOffMisc + (256 + 64) * 4;
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;
// The solve phase reuses the ring and XG region for N and R/Z.
constexpr uint32_t kOffN = kOffRing;
constexpr uint32_t kOffR = kOffN + kRows * kLD * 4;
static_assert(kOffR + kRows * kLD * 4 <= kOffStage, "solve buffers overlap the stage");

// TMEM columns.
constexpr uint32_t kColS = 0;     // two S buffers (128 each)
constexpr uint32_t kColR = 256;   // phase 2: R~ accumulator; phase 4: Zh^T (64) | Zl^T (64)
constexpr uint32_t kColG = 384;   // phase 2: Gram accumulator; phase 4: D = dV^T

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
  int* status;
};

struct MBars {
  uint64_t ring_full[kRing], ring_empty[kRing];
  uint64_t q_full;
  uint64_t s_full[2], s_done[2];
  uint64_t xg_full[2], xg_empty[2];
  uint64_t acc_done;
  uint64_t d_full, d_empty;
  uint64_t drain;
  uint32_t tmem;
  int abort;
  int fail;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ float bf16_round(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
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

// Gathers the 128 retained rows of tile t (clamped to the last retained row
// past B) of one unit's [n][128] matrix into a swizzled 32 KB tile.
__device__ __forceinline__ void gather_tile(uint8_t* dst, const CUtensorMap* map, uint64_t* bar,
                                            const int32_t* idx_u, int B, int row0, int t) {
  mbar_expect_tx(bar, kTileBytes);
  for (int g = 0; g < kTile / 4; ++g) {
    int r[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) r[e] = row0 + __ldg(idx_u + min(t * kTile + 4 * g + e, B - 1));
    tma_gather4(dst + g * 512, map, bar, 0, r[0], r[1], r[2], r[3]);
    tma_gather4(dst + kTileBytes / 2 + g * 512, map, bar, 64, r[0], r[1], r[2], r[3]);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    k_merge_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, MArgs a) {
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = (uint8_t*)(((uintptr_t)smraw + 1023) & ~(uintptr_t)1023);
  MBars* bars = (MBars*)(sm + kOffBar);
  uint32_t* mask = (uint32_t*)(sm + kOffMask);
  int* hist = (int*)(sm + kOffMisc);
  int* sh = hist + 256;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x, B = a.B, T = (B + kTile - 1) / kTile;
  const int32_t* idx_u = a.idx + (size_t)u * B;
  const float* sc_u = a.scores + (size_t)u * a.P;

  if (tid == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&bars->ring_full[i], 1);
      mbar_init(&bars->ring_empty[i], 1);
    }
    mbar_init(&bars->q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_done[i], 128);
      mbar_init(&bars->xg_full[i], 128);
      mbar_init(&bars->xg_empty[i], 1);
    }
    mbar_init(&bars->acc_done, 1);
    mbar_init(&bars->d_full, 1);
    mbar_init(&bars->d_empty, 128);
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    bars->fail = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem, 512);
    tmem_relinquish();
  }
  // ---- fixed tokens: retained sinks, the window, and the n_fix retained
  // prefix non-sink tokens with the largest scores (ties: smaller position)
  for (int i = tid; i < (B + 31) / 32; i += kThreads) mask[i] = 0;
  __syncthreads();
  auto cand = [&](int i) {
    const int j = __ldg(idx_u + i);
    return j >= a.n_sink && j < a.P;
  };
  int nc = 0;
  for (int i = tid; i < B; i += kThreads) {
    if (!cand(i)) atomicOr(&mask[i >> 5], 1u << (i & 31));
    else ++nc;
  }
  int ncand;
  (void)block_exclusive_scan(nc, sh + 8, &ncand);
  const int nf = min(a.n_fix, ncand);
  if (nf > 0) {
    auto get = [&](int i, uint32_t* key) {
      if (!cand(i)) return false;
      *key = order_key(__ldg(sc_u + __ldg(idx_u + i)));
      return true;
    };
    block_topk_mark(get, [&](int i, int) { atomicOr(&mask[i >> 5], 1u << (i & 31)); }, B, nf,
                    hist, sh);
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem;
  volatile int* abort_flag = &bars->abort;
  const int row0 = u * a.n;   // first row of this unit in the 2-D K / V maps
  float lam = INFINITY;        // log2 normaliser of the retained softmax (compute rows)

  // Job k: k < T: phase 1 tile k; T <= k < 2T: phase 2 tile k - T;
  // 2T <= k < 3T: phase 4 tile k - 2T.  S buffer k & 1, ring loads in order.
  // ================================================= phases 1 and 2
  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&tmQ);
      prefetch_tensormap(&tmK);
      prefetch_tensormap(&tmV);
      mbar_expect_tx(&bars->q_full, kTileBytes);
      const uint64_t pol = l2_evict_last();
      tma_load_3d(sm + kOffQ, &tmQ, &bars->q_full, 0, 0, u, pol);
      tma_load_3d(sm + kOffQ + kTileBytes / 2, &tmQ, &bars->q_full, 64, 0, u, pol);
      uint32_t use = 0;
      bool ok = true;
      for (int k = 0; k < 2 * T && ok; ++k) {
        const int t = k < T ? k : k - T;
        for (int l = 0; l < (k < T ? 1 : 2) && ok; ++l) {
          const uint32_t slot = use % kRing;
          if (use >= kRing)
            ok = mbar_wait(&bars->ring_empty[slot], (use / kRing - 1) & 1, abort_flag, kBudget);
          if (!ok) break;
          gather_tile(sm + kOffRing + slot * kTileBytes, l == 0 ? &tmK : &tmV,
                      &bars->ring_full[slot], idx_u, B, row0, t);
          ++use;
        }
      }
      // let every issued gather land before the region is reused
      for (uint32_t i = use > kRing ? use - kRing : 0; i < use; ++i)
        mbar_wait(&bars->ring_full[i % kRing], (i / kRing) & 1, abort_flag, kBudget);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(kRows, kTile, 0, 0);
      const uint32_t id_r = idesc_bf16(kRows, kD, 0, 1);     // R~ += Xh V0 (V0 MN-major)
      const uint32_t id_g = idesc_bf16(kRows, kRows, 0, 0);  // G += A XGh^T
      bool ok = mbar_wait(&bars->q_full, 0, abort_flag, kBudget);
      const uint32_t qa = smem_u32(sm + kOffQ);
      uint32_t use = 0;
      int pend = -1;
      uint32_t pend_v = 0;
      auto issue_rg = [&](int kp, uint32_t vuse) -> bool {
        const int t = kp - T, b = kp & 1, xb = t & 1;
        bool w = mbar_wait(&bars->s_done[b], (kp >> 1) & 1, abort_flag, kBudget);
        if (w) w = mbar_wait(&bars->xg_full[xb], (t >> 1) & 1, abort_flag, kBudget);
        if (w)
          w = mbar_wait(&bars->ring_full[vuse % kRing], (vuse / kRing) & 1, abort_flag, kBudget);
        if (!w) return false;
        tc_fence_after();
        const uint32_t va = smem_u32(sm + kOffRing + (vuse % kRing) * kTileBytes);
        const uint32_t xa = smem_u32(sm + kOffXG + xb * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk)
          mma_ts(tmem + kColR, tmem + kColS + b * kTile + kk * 8,
                 sw128_desc(va + kk * 2048, kTileBytes / 2, 1024), id_r, (t > 0 || kk > 0));
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_bf16(tmem + kColG, sw128_desc(xa + off, 16, 1024), sw128_desc(xa + off, 16, 1024),
                   id_g, (t > 0 || kk > 0));
        }
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_ts(tmem + kColG, tmem + kColS + b * kTile + 64 + kk * 8,
                 sw128_desc(xa + off, 16, 1024), id_g, 1);
        }
        mma_commit(&bars->ring_empty[vuse % kRing]);
        mma_commit(&bars->xg_empty[xb]);
        return true;
      };
      for (int k = 0; k < 2 * T && ok; ++k) {
        const int b = k & 1;
        const uint32_t kuse = use++;
        ok = mbar_wait(&bars->ring_full[kuse % kRing], (kuse / kRing) & 1, abort_flag, kBudget);
        if (ok && k >= 2) ok = mbar_wait(&bars->s_done[b], ((k >> 1) - 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t ka = smem_u32(sm + kOffRing + (kuse % kRing) * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
          mma_bf16(tmem + kColS + b * kTile, sw128_desc(qa + off, 16, 1024),
                   sw128_desc(ka + off, 16, 1024), id_s, kk > 0);
        }
        mma_commit(&bars->ring_empty[kuse % kRing]);
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
    }
  } else if (warp >= 4 && warp < 8) {
    const int q = warp & 3, row = q * 32 + lane;
    const bool row_ok = row < a.m;
    const int lim = a.causal ? a.n - a.w + (row_ok ? row % a.w : 0) : a.n - 1;
    const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
    float M = -INFINITY, L = 0.f;
    bool ok = true;
    for (int k = 0; k < 2 * T && ok; ++k) {
      const int b = k & 1, t = k < T ? k : k - T;
      ok = mbar_wait(&bars->s_full[b], (k >> 1) & 1, abort_flag, kBudget);
      if (!ok) break;
      tc_fence_after();
      const uint32_t sbase = lane_addr + kColS + b * kTile;
      if (k < T) {
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(sbase + c * 32, v);
          tmem_ld_wait();
          float vmax = -INFINITY;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int i = t * kTile + c * 32 + e;
            if (i >= B || !row_ok || __ldg(idx_u + i) > lim) v[e] = -INFINITY;
            vmax = fmaxf(vmax, v[e]);
          }
          if (vmax == -INFINITY) continue;
          const float cm = vmax * a.sl2;
          if (cm > M) {
            L *= fast_exp2(M - cm);
            M = cm;
          }
          float s = 0.f;
#pragma unroll
          for (int e = 0; e < 32; ++e) s += fast_exp2(fmaf(v[e], a.sl2, -M));
          L += s;
        }
        tc_fence_before();
        mbar_arrive(&bars->s_done[b]);
        if (k == T - 1) lam = (row_ok && L > 0.f) ? M + __log2f(L) : INFINITY;
      } else {
        const int xb = t & 1;
        if (t >= 2) ok = mbar_wait(&bars->xg_empty[xb], ((t >> 1) - 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        uint8_t* xg = sm + kOffXG + xb * kTileBytes;
        // 2 (X - Xh) goes to TMEM columns 64..127, which hold S chunks 2 and 3:
        // chunks 0 and 1 are written once chunk 2 is read, chunk 2 once chunk 3 is
        uint32_t lo2[3][16];
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(sbase + c * 32, v);
          tmem_ld_wait();
          uint32_t hi[16], lo[16], ghi[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float x[2], g[2], l2[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int i = t * kTile + c * 32 + e + h;
              const bool vis = i < B && row_ok && __ldg(idx_u + i) <= lim;
              x[h] = vis ? fast_exp2(fmaf(v[e + h], a.sl2, -lam)) : 0.f;
              const bool fixed = i >= B || ((mask[i >> 5] >> (i & 31)) & 1u);
              const float xh = bf16_round(x[h]);
              g[h] = fixed ? 0.f : xh;
              l2[h] = fixed ? 0.f : 2.f * (x[h] - xh);
            }
            hi[e / 2] = pack_bf16(x[0], x[1]);
            ghi[e / 2] = pack_bf16(g[0], g[1]);
            lo[e / 2] = pack_bf16(l2[0], l2[1]);
          }
          tmem_st16(sbase + c * 16, hi);
          // XGh row `row`, tokens 32c..32c+31: token block c/2, 16-byte chunks (c&1)*4..+3
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) {
            const uint4 val = make_uint4(ghi[4 * qq], ghi[4 * qq + 1], ghi[4 * qq + 2],
                                         ghi[4 * qq + 3]);
            *(uint4*)(xg + (c >> 1) * (kTileBytes / 2) + sw128_offset(row, (c & 1) * 4 + qq)) = val;
          }
          if (c < 3) {
#pragma unroll
            for (int e = 0; e < 16; ++e) lo2[c][e] = lo[e];
          }
          if (c == 2) {
            tmem_st16(sbase + 64, lo2[0]);
            tmem_st16(sbase + 64 + 16, lo2[1]);
          } else if (c == 3) {
            tmem_st16(sbase + 64 + 32, lo2[2]);
            tmem_st16(sbase + 64 + 48, lo);
          }
        }
        tmem_st_wait();
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&bars->s_done[b]);
        mbar_arrive(&bars->xg_full[xb]);
      }
    }
    // R = Y - R~ and the raw Gram rows into shared memory (fp32)
    if (ok) ok = mbar_wait(&bars->acc_done, 0, abort_flag, kBudget);
    tc_fence_after();
    float* N = (float*)(sm + kOffN);
    float* R = (float*)(sm + kOffR);
    if (ok) {
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(lane_addr + kColR + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int col = c * 32 + e;
          R[row * kLD + col] =
              row_ok ? a.y[((size_t)u * a.m + row) * kD + col] - v[e] : 0.f;
        }
        tmem_ld32(lane_addr + kColG + c * 32, v);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e) N[row * kLD + c * 32 + e] = v[e];
      }
    }
    if (!ok && row == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // ================================================= phase 3: solve (fp32)
  float* N = (float*)(sm + kOffN);
  float* R = (float*)(sm + kOffR);
  const bool aborted = *abort_flag != 0;
  if (!aborted) {
    // N = (G + G^T) / 2 + lambda I on the window rows; identity on padding
    for (int p = tid; p < kRows * kRows; p += kThreads) {
      const int i = p / kRows, j = p % kRows;
      if (j > i) continue;
      float val;
      if (i >= a.m || j >= a.m) val = (i == j) ? 1.f : 0.f;
      else if (i == j) val = N[i * kLD + i] + a.lambda;
      else val = 0.5f * (N[i * kLD + j] + N[j * kLD + i]);
      N[i * kLD + j] = val;
    }
    __syncthreads();
    for (int kb = 0; kb < kRows / 32 && !a.lambda_inf; ++kb) {
      const int k0 = kb * 32;
      if (warp == 0) {   // diagonal block, one warp
        for (int k = k0; k < k0 + 32; ++k) {
          if (lane == 0) {
            const float dkk = N[k * kLD + k];
            if (!(dkk > 0.f)) bars->fail = 1;
            N[k * kLD + k] = sqrtf(fmaxf(dkk, 0.f));
          }
          __syncwarp();
          const int i = k0 + lane;
          const float piv = N[k * kLD + k];
          if (i > k) N[i * kLD + k] = piv > 0.f ? N[i * kLD + k] / piv : 0.f;
          __syncwarp();
          if (i > k)
            for (int j = k + 1; j <= i; ++j) N[i * kLD + j] -= N[i * kLD + k] * N[j * kLD + k];
          __syncwarp();
        }
      }
      __syncthreads();
      // panel below the diagonal block: L_ij = (N_ij - sum_p L_ip L_jp) / L_jj
      for (int i = k0 + 32 + tid; i < kRows; i += kThreads) {
        for (int j = k0; j < k0 + 32; ++j) {
          float s = N[i * kLD + j];
          for (int p = k0; p < j; ++p) s -= N[i * kLD + p] * N[j * kLD + p];
          const float piv = N[j * kLD + j];
          N[i * kLD + j] = piv > 0.f ? s / piv : 0.f;
        }
      }
      __syncthreads();
      // trailing update of the lower triangle
      const int rest = kRows - (k0 + 32);
      for (int p = tid; p < rest * rest; p += kThreads) {
        const int i = k0 + 32 + p / rest, j = k0 + 32 + p % rest;
        if (j > i) continue;
        float s = N[i * kLD + j];
#pragma unroll 8
        for (int pp = k0; pp < k0 + 32; ++pp) s -= N[i * kLD + pp] * N[j * kLD + pp];
        N[i * kLD + j] = s;
      }
      __syncthreads();
    }
    const bool fail = bars->fail != 0 || a.lambda_inf;
    if (bars->fail && !a.lambda_inf && tid == 0) set_status(a.status, GRKV_ERR_NUMERIC);
    if (fail) {   // values stay V0
      for (int p = tid; p < kRows * kLD; p += kThreads) R[p] = 0.f;
      __syncthreads();
    } else {
      // forward: L W = R, 32-row blocks
      for (int ib = 0; ib < kRows / 32; ++ib) {
        const int i0 = ib * 32;
        if (tid < kD) {
          for (int i = i0; i < i0 + 32; ++i) {
            float s = R[i * kLD + tid];
            for (int kx = i0; kx < i; ++kx) s -= N[i * kLD + kx] * R[kx * kLD + tid];
            R[i * kLD + tid] = s / N[i * kLD + i];
          }
        }
        __syncthreads();
        const int rest = kRows - (i0 + 32);
        for (int p = tid; p < rest * kD; p += kThreads) {
          const int i = i0 + 32 + p / kD, e = p % kD;
          float s = R[i * kLD + e];
#pragma unroll 8
          for (int kx = i0; kx < i0 + 32; ++kx) s -= N[i * kLD + kx] * R[kx * kLD + e];
          R[i * kLD + e] = s;
        }
        __syncthreads();
      }
      // backward: L^T Z = W
      for (int ib = kRows / 32 - 1; ib >= 0; --ib) {
        const int i0 = ib * 32;
        if (tid < kD) {
          for (int i = i0 + 31; i >= i0; --i) {
            float s = R[i * kLD + tid];
            for (int kx = i + 1; kx < i0 + 32; ++kx) s -= N[kx * kLD + i] * R[kx * kLD + tid];
            R[i * kLD + tid] = s / N[i * kLD + i];
          }
        }
        __syncthreads();
        for (int p = tid; p < i0 * kD; p += kThreads) {
          const int i = p / kD, e = p % kD;
          float s = R[i * kLD + e];
#pragma unroll 8
          for (int kx = i0; kx < i0 + 32; ++kx) s -= N[kx * kLD + i] * R[kx * kLD + e];
          R[i * kLD + e] = s;
        }
        __syncthreads();
      }
    }
    // Z^T into TMEM as MMA operands: lane = column e of Z, packed row pairs
    if (warp >= 4 && warp < 8) {
      const int q = warp & 3, e = q * 32 + lane;
      const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
      for (int rc = 0; rc < 4; ++rc) {
        uint32_t zh[16], zl[16];
#pragma unroll
        for (int p = 0; p < 16; ++p) {
          const float z0 = R[(rc * 32 + 2 * p) * kLD + e], z1 = R[(rc * 32 + 2 * p + 1) * kLD + e];
          const float h0 = bf16_round(z0), h1 = bf16_round(z1);
          zh[p] = pack_bf16(h0, h1);
          zl[p] = pack_bf16(z0 - h0, z1 - h1);
        }
        tmem_st16(lane_addr + kColR + rc * 16, zh);
        tmem_st16(lane_addr + kColR + 64 + rc * 16, zl);
      }
      tmem_st_wait();
    }
  }
  fence_proxy_async_smem();   // the solve buffers are TMA destinations again
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // ================================================= phase 4: dV and outputs
  if (!aborted) {
    if (warp == 0) {
      if (lane == 0) {
        uint32_t use = 3u * T;   // loads of phases 1 and 2
        bool ok = true;
        for (int t = 0; t < T && ok; ++t) {
          const uint32_t slot = use % kRing;
          if (use >= kRing)
            ok = mbar_wait(&bars->ring_empty[slot], (use / kRing - 1) & 1, abort_flag, kBudget);
          if (!ok) break;
          gather_tile(sm + kOffRing + slot * kTileBytes, &tmK, &bars->ring_full[slot], idx_u, B,
                      row0, t);
          ++use;
        }
        for (uint32_t i = use > kRing ? use - kRing : 0; i < use; ++i)
          mbar_wait(&bars->ring_full[i % kRing], (i / kRing) & 1, abort_flag, kBudget);
      }
    } else if (warp == 1) {
      if (lane == 0) {
        const uint32_t id_s = idesc_bf16(kRows, kTile, 0, 0);
        const uint32_t id_d = idesc_bf16(kD, kTile, 0, 1);   // D = Z^T XG (XG MN-major)
        const uint32_t qa = smem_u32(sm + kOffQ);
        uint32_t use = 3u * T;
        bool ok = true;
        auto issue_d = [&](int t) -> bool {
          const int k = 2 * T + t, b = k & 1;
          bool w = mbar_wait(&bars->xg_full[0], (t + ((T + 1) >> 1)) & 1, abort_flag, kBudget);
          if (w && t >= 1) w = mbar_wait(&bars->d_empty, (t - 1) & 1, abort_flag, kBudget);
          (void)b;
          if (!w) return false;
          tc_fence_after();
          const uint32_t xh = smem_u32(sm + kOffXG), xl = xh + kTileBytes;
#pragma unroll
          for (int kk = 0; kk < kRows / 16; ++kk)
            mma_ts(tmem + kColG, tmem + kColR + kk * 8,
                   sw128_desc(xh + kk * 2048, kTileBytes / 2, 1024), id_d, kk > 0);
#pragma unroll
          for (int kk = 0; kk < kRows / 16; ++kk)
            mma_ts(tmem + kColG, tmem + kColR + 64 + kk * 8,
                   sw128_desc(xh + kk * 2048, kTileBytes / 2, 1024), id_d, 1);
#pragma unroll
          for (int kk = 0; kk < kRows / 16; ++kk)
            mma_ts(tmem + kColG, tmem + kColR + kk * 8,
                   sw128_desc(xl + kk * 2048, kTileBytes / 2, 1024), id_d, 1);
          mma_commit(&bars->xg_empty[0]);
          mma_commit(&bars->d_full);
          return true;
        };
        for (int t = 0; t < T && ok; ++t) {
          const int k = 2 * T + t, b = k & 1;
          const uint32_t kuse = use++;
          ok = mbar_wait(&bars->ring_full[kuse % kRing], (kuse / kRing) & 1, abort_flag, kBudget);
          if (ok) ok = mbar_wait(&bars->s_done[b], ((k >> 1) - 1) & 1, abort_flag, kBudget);
          if (!ok) break;
          tc_fence_after();
          const uint32_t ka = smem_u32(sm + kOffRing + (kuse % kRing) * kTileBytes);
#pragma unroll
          for (int kk = 0; kk < kD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (kTileBytes / 2) + (kk & 3) * 32;
            mma_bf16(tmem + kColS + b * kTile, sw128_desc(qa + off, 16, 1024),
                     sw128_desc(ka + off, 16, 1024), id_s, kk > 0);
          }
          mma_commit(&bars->ring_empty[kuse % kRing]);
          mma_commit(&bars->s_full[b]);
          if (t >= 1) ok = issue_d(t - 1);
        }
        if (ok && T >= 1) ok = issue_d(T - 1);
        mma_commit(&bars->drain);
        mbar_wait(&bars->drain, 0, abort_flag, kBudget);
      }
    } else if (warp >= 4 && warp < 8) {
      const int q = warp & 3, row = q * 32 + lane;
      const bool row_ok = row < a.m;
      const int lim = a.causal ? a.n - a.w + (row_ok ? row % a.w : 0) : a.n - 1;
      const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
      bool ok = true;
      uint8_t* xh = sm + kOffXG;
      uint8_t* xl = xh + kTileBytes;
      // xg_empty[0] / xg_full[0] keep counting from phase 2 (tiles t with t&1 == 0)
      const int base_uses = (T + 1) >> 1;
      for (int t = 0; t < T && ok; ++t) {
        const int k = 2 * T + t, b = k & 1;
        ok = mbar_wait(&bars->s_full[b], (k >> 1) & 1, abort_flag, kBudget);
        if (ok && base_uses + t >= 1)
          ok = mbar_wait(&bars->xg_empty[0], (base_uses + t - 1) & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
        const uint32_t sbase = lane_addr + kColS + b * kTile;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(sbase + c * 32, v);
          tmem_ld_wait();
          uint32_t ghi[16], glo[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float g[2], l[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int i = t * kTile + c * 32 + e + h;
              const bool vis = i < B && row_ok && __ldg(idx_u + i) <= lim;
              const float x = vis ? fast_exp2(fmaf(v[e + h], a.sl2, -lam)) : 0.f;
              const bool fixed = i >= B || ((mask[i >> 5] >> (i & 31)) & 1u);
              const float xhv = bf16_round(x);
              g[h] = fixed ? 0.f : xhv;
              l[h] = fixed ? 0.f : x - xhv;
            }
            ghi[e / 2] = pack_bf16(g[0], g[1]);
            glo[e / 2] = pack_bf16(l[0], l[1]);
          }
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) {
            const uint32_t off = (c >> 1) * (kTileBytes / 2) + sw128_offset(row, (c & 1) * 4 + qq);
            *(uint4*)(xh + off) = make_uint4(ghi[4 * qq], ghi[4 * qq + 1], ghi[4 * qq + 2],
                                             ghi[4 * qq + 3]);
            *(uint4*)(xl + off) = make_uint4(glo[4 * qq], glo[4 * qq + 1], glo[4 * qq + 2],
                                             glo[4 * qq + 3]);
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&bars->s_done[b]);
        mbar_arrive(&bars->xg_full[0]);
      }
      if (!ok && row == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
    } else if (warp >= 8) {
      // epilogue: D = dV^T, lane = column e of V; staged through shared memory
      const int q = warp & 3, e = q * 32 + lane, et = tid - 256;
      const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
      float* stage = (float*)(sm + kOffStage);
      bool ok = true;
      for (int t = 0; t < T && ok; ++t) {
        ok = mbar_wait(&bars->d_full, t & 1, abort_flag, kBudget);
        if (!ok) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(lane_addr + kColG + c * 32, v);
          tmem_ld_wait();
          if (c == 3) {
            tc_fence_before();
            mbar_arrive(&bars->d_empty);
          }
#pragma unroll
          for (int tk = 0; tk < 32; ++tk) stage[tk * kLD + e] = v[tk];
          named_bar(3, 128);
          // a warp takes 32 tokens of one 32-column block
          const int tk = et & 31, c0 = (et >> 5) * 32, i = t * kTile + c * 32 + tk;
          if (i < B) {
            const size_t src = ((size_t)u * a.n + __ldg(idx_u + i)) * kD + c0;
            const size_t dst = ((size_t)u * B + i) * kD + c0;
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const uint4 v0 = *(const uint4*)(a.v + src + 8 * h);
              const uint4 k0 = *(const uint4*)(a.k + src + 8 * h);
              const __nv_bfloat16* pv = (const __nv_bfloat16*)&v0;
              uint32_t o[4];
#pragma unroll
              for (int z = 0; z < 4; ++z)
                o[z] = pack_bf16(__bfloat162float(pv[2 * z]) + stage[tk * kLD + c0 + 8 * h + 2 * z],
                                 __bfloat162float(pv[2 * z + 1]) +
                                     stage[tk * kLD + c0 + 8 * h + 2 * z + 1]);
              *(uint4*)(a.v_out + dst + 8 * h) = make_uint4(o[0], o[1], o[2], o[3]);
              *(uint4*)(a.k_out + dst + 8 * h) = k0;
            }
          }
          named_bar(3, 128);
        }
      }
      if (!ok && e == 0) set_status(a.status, GRKV_ERR_TIMEOUT);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

}  // namespace

bool merge_tc_supported(const Shape& s) {
  return s.dtype == GRKV_BF16 && s.m <= kRows && s.B <= kMaxB && s.B >= 1;
}

cudaError_t launch_merge_tc(const Shape& s, const void* q, const void* k, const void* v,
                            const float* scores, const float* y, const int32_t* idx, void* k_out,
                            void* v_out, char* ws, const WsLayout& L, cudaStream_t st) {
  CUtensorMap mq, mk, mv;
  if (!encode_bf16_3d(&mq, q, kD, s.m, s.U, 64, kRows) ||
      !encode_bf16_2d_rows(&mk, k, kD, (uint64_t)s.U * s.n) ||
      !encode_bf16_2d_rows(&mv, v, kD, (uint64_t)s.U * s.n))
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
  a.status = (int*)(ws + L.status);
  cudaError_t e =
      cudaFuncSetAttribute(k_merge_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (e != cudaSuccess) return e;
  k_merge_tc<<<s.U, kThreads, kSmemBytes, st>>>(mq, mk, mv, a);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace grkv
