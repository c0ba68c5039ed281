// Key step of Algorithm 1 at t = 0 (Sec. 3.4 "Key step", App. D.2): fp32 on
// CUDA cores, with the CG products on the tensor cores (three-part bf16
// splits of the fp32 operands) when m <= 128.  One CTA per unit, or, when
// units are few, a cluster of up to 8 CTAs per unit that split the CG
// products by retained columns (KPart).
//
// With the merged values V* of the value step fixed, f(K) = softmax(s Q K^T) V*
// is linearised at K0 and the local ridge problem is solved in its dual form:
//     e = vec(Y - X V*),   (J_G J_G^T + lambda_k I) alpha = e,
//     K*_G = K0_G + J_G^T alpha,   K*_F = K0_F,
// where X is the (masked) retained attention at K0 and J_G the Jacobian of f
// with respect to the free retained rows.  The operator is applied without
// forming J: J^T W (vector-Jacobian product) is
//     dA = W V*^T,  dS = X o (dA - rowsum(X o dA)),  dK = s dS^T Q,
// with the fixed rows of dK zeroed, and J dK (Jacobian-vector product) is
//     dS = s Q dK^T,  dA = X o (dS - rowsum(X o dS)),  df = dA V*.
// Inside CG the two meet as s Q dK^T = (s^2 Q Q^T) dS on the free columns,
// so an iteration is three GEMMs (m x B x d, m x m x B, m x B x d).
// Conjugate gradients start from alpha = 0 and run at most cg_iters
// iterations, stopping once ||r|| <= cg_tol ||e|| or the search direction
// vanishes.  Each product is a tiled GEMM over the unit's m x B, B x d and
// m x d matrices, staged in the workspace; with m <= 128 the three products
// of a CG iteration run on tcgen05 (tc_gemm).
//
// V* is read from v_out as written by the value step (rounded to the input
// dtype), K0 from k_out (the value step copies K0 there), and the fixed set is
// recomputed from the prefix scores exactly as the value step defines it.
//
// With S > 1 steps (Algorithm 1's outer loop), k_alternate_step runs steps
// t = 1 .. S-1: the value step from V0 with X at the current keys K^(t)
// (dual form, X_G X_G^T + lambda_v I factored by Cholesky in fp32), then the
// key step linearised at K^(t), whose right-hand side gains J_G (K^(t) - K0);
// K^(t) and V^(t) are carried in fp32 between steps.
#include <cmath>

#include "block_select.cuh"
#include "grkv_internal.cuh"
#include "sm100.cuh"

namespace grkv {
namespace {

using namespace sm100;

constexpr int kKT = 256;                  // threads per CTA
constexpr int kTM = 64, kTN = 64, kTK = 16;
constexpr long long kWaitBudget = 1ll << 32;   // clock cycles of a bounded wait

struct KArgs {
  int n, w, m, B, P, n_sink, n_fix, causal, dtype, iters;
  float scale, lambda_k, tol;
  float lambda_v, step_tol;
  int lambda_inf;
  int vt_valid;           // Vt holds V^(t) (false at t = 1: V^(1) is only in v_out)
  int use_tc;             // m <= 128: the CG products run on the tensor cores
  int cluster;            // C: CTAs per unit in k_key_step's CG (one cluster each)
  const void* k;          // [U][n][d]  full caches (K0, V0 gathers of steps t >= 1)
  const void* v;
  float* Kt;              // [U][B][d]  fp32 K^(t) of the alternation, or null
  float* Vt;              // [U][B][d]  fp32 V^(t) of the alternation (t >= 2)
  float* G;               // [U][m][m]  value step: X_G X_G^T + lambda_v I, then its factor
  float* RZ;              // [U][m][d]  value step: R, then Z
  int* done;              // [U]        the unit met the alternation's stop test
  int* status;
  const void* q;          // [U][m][d]
  const float* y;         // [U][m][d]
  const float* scores;    // [U][P]
  const int32_t* idx;     // [U][B]
  void* v_out;            // [U][B][d]  merged values V* (rewritten by steps t >= 1)
  void* k_out;            // [U][B][d]  holds K0 on entry, K* on exit
  float* X;               // [U][m][B]
  float* T;               // [U][m][B]
  float* dK;              // [U][B][d]
  float* T2;              // [U][m][B]
  float* GQ;              // [U][m][m]
  float* vec;             // [U][C][5][m][d]: r, p, Ap, alpha, X V* of each CTA
  float* app;             // [U][C][m][d]  per-CTA partial products (C > 1)
  float* rho2p;           // [U][C][128]   per-CTA partial row sums (C > 1)
  int* cnt;               // [U]           barrier counters (C > 1, zeroed per launch)
  uint8_t* fixed;         // [U][B]
};

__device__ __forceinline__ float ldv(const void* p, size_t i, int dtype) {
  return dtype == GRKV_F32 ? ((const float*)p)[i]
                           : __bfloat162float(((const __nv_bfloat16*)p)[i]);
}

// Shared-memory k slabs of one block_gemm tile.
struct GemmSmem {
  alignas(16) float As[kTK][kTM + 4];
  alignas(16) float Bs[kTK][kTN + 4];
};

// C(i, j) = sum_k a(i, k) b(k, j) for i < M, j < N; store(i, j, value).
// 64 x 64 output tiles, 16-deep k slabs in shared memory, 4 x 4 per thread.
// The next slab is fetched into registers while the current one is used.
// Each thread fetches four elements of each operand; kAIFast / kBKFast pick
// the index that runs fastest across threads (i for A, k for B), so that the
// loads are coalesced for operands stored with that index contiguous.
template <bool kAIFast = false, bool kBKFast = false, class FA, class FB, class FS>
__device__ void block_gemm(GemmSmem& g, int M, int N, int K, FA a, FB b, FS store) {
  constexpr int kAL = kTM * kTK / kKT, kBL = kTN * kTK / kKT;
  static_assert(kAL * kKT == kTM * kTK && kBL * kKT == kTN * kTK, "slab split");
  auto& As = g.As;
  auto& Bs = g.Bs;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  auto a_at = [&](int l, int& ii, int& kk) {
    const int e = threadIdx.x + l * kKT;
    ii = kAIFast ? e % kTM : e / kTK;
    kk = kAIFast ? e / kTM : e % kTK;
  };
  auto b_at = [&](int l, int& jj, int& kk) {
    const int e = threadIdx.x + l * kKT;
    jj = kBKFast ? e / kTK : e % kTN;
    kk = kBKFast ? e % kTK : e / kTN;
  };
  for (int i0 = 0; i0 < M; i0 += kTM)
    for (int j0 = 0; j0 < N; j0 += kTN) {
      float acc[4][4];
#pragma unroll
      for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int u = 0; u < 4; ++u) acc[t][u] = 0.f;
      float ra[kAL], rb[kBL];
      auto fetch = [&](int k0) {
#pragma unroll
        for (int l = 0; l < kAL; ++l) {
          int ii, kk;
          a_at(l, ii, kk);
          ra[l] = (i0 + ii < M && k0 + kk < K) ? a(i0 + ii, k0 + kk) : 0.f;
        }
#pragma unroll
        for (int l = 0; l < kBL; ++l) {
          int jj, kk;
          b_at(l, jj, kk);
          rb[l] = (j0 + jj < N && k0 + kk < K) ? b(k0 + kk, j0 + jj) : 0.f;
        }
      };
      fetch(0);
      for (int k0 = 0; k0 < K; k0 += kTK) {
#pragma unroll
        for (int l = 0; l < kAL; ++l) {
          int ii, kk;
          a_at(l, ii, kk);
          As[kk][ii] = ra[l];
        }
#pragma unroll
        for (int l = 0; l < kBL; ++l) {
          int jj, kk;
          b_at(l, jj, kk);
          Bs[kk][jj] = rb[l];
        }
        __syncthreads();
        if (k0 + kTK < K) fetch(k0 + kTK);
#pragma unroll
        for (int kk = 0; kk < kTK; ++kk) {
          // rows of 68 floats keep every 4-float group 16-byte aligned
          const float4 a4 = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
          const float4 b4 = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
          const float av[4] = {a4.x, a4.y, a4.z, a4.w}, bv[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
          for (int t = 0; t < 4; ++t)
#pragma unroll
            for (int u = 0; u < 4; ++u) acc[t][u] = fmaf(av[t], bv[u], acc[t][u]);
        }
        __syncthreads();
      }
#pragma unroll
      for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = i0 + ty * 4 + t, j = j0 + tx * 4 + u;
          if (i < M && j < N) store(i, j, acc[t][u]);
        }
    }
  __syncthreads();
}

// ----------------------------------------------------- tensor-core products
// The CG products on tcgen05.  An fp32 operand is split into three bf16 parts
// x = h + m + l (h = bf16(x), m = bf16(x - h), l = bf16(x - h - m)); keeping
// the six part products of combined order <= 2 (h.h, h.m, m.h, h.l, m.m, l.h)
// reproduces the fp32 product to about 2^-24 of its terms, so CG sees fp32
// products.  An operand exact in bf16 (V* of a bf16 cache) takes one part and
// three products.  One 128 x 128 output tile at a time: 64-deep slabs of A
// (K-major) and B (K-major or MN-major) staged by all threads into
// 128-byte-swizzled shared memory, the MMAs issued by one thread into a
// 128-column TMEM accumulator, then the tile staged through shared memory so
// that warps write rows with coalesced stores.
constexpr int kTP = 3;                          // parts of an fp32 operand
constexpr uint32_t kSlab = 128 * 64 * 2;        // one part of a 128 x 64 bf16 slab
constexpr uint32_t kTcSmem = 2 * kTP * kSlab + 1024;
constexpr int kTLD = 129;                       // fp32 row stride of the staged output tile
static_assert(128 * kTLD * 4 <= 2 * kTP * kSlab, "output tile fits the slabs");

struct TcCtx {
  uint8_t* sm;        // 1024-byte aligned: A parts, then B parts
  uint32_t tmem;      // 128 fp32 columns
  uint64_t* bar;      // MMA completion
  uint32_t phase;
  int* status;
};

__device__ __forceinline__ float bf_lo(uint32_t h) { return __uint_as_float(h << 16); }
__device__ __forceinline__ float bf_hi(uint32_t h) { return __uint_as_float(h & 0xFFFF0000u); }

// x[0..8) = p[0..nv), zero past nv: two 16-byte loads when the chunk is whole
// and aligned, element loads otherwise.
__device__ __forceinline__ void ld8(const float* p, int nv, float* x) {
  if (nv == 8 && ((uintptr_t)p & 15) == 0) {
    const float4 a = *(const float4*)p, b = *(const float4*)(p + 4);
    x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
    x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) x[e] = e < nv ? p[e] : 0.f;
  }
}
__device__ __forceinline__ void ld8(const __nv_bfloat16* p, int nv, float* x) {
  if (nv == 8 && ((uintptr_t)p & 15) == 0) {
    const uint4 a = *(const uint4*)p;
    const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      x[2 * e] = bf_lo(w[e]);
      x[2 * e + 1] = bf_hi(w[e]);
    }
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) x[e] = e < nv ? __bfloat162float(p[e]) : 0.f;
  }
}

// Eight values into their three bf16 parts, four packed pairs each.
__device__ __forceinline__ void split3(const float* x, uint4* part) {
  uint32_t p[3][4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float a0 = x[2 * e], a1 = x[2 * e + 1];
    const uint32_t h = pack_bf16(a0, a1);
    const float r0 = a0 - bf_lo(h), r1 = a1 - bf_hi(h);
    const uint32_t mm = pack_bf16(r0, r1);
    p[0][e] = h;
    p[1][e] = mm;
    p[2][e] = pack_bf16(r0 - bf_lo(mm), r1 - bf_hi(mm));
  }
#pragma unroll
  for (int q = 0; q < 3; ++q) part[q] = make_uint4(p[q][0], p[q][1], p[q][2], p[q][3]);
}

// C = A B for A [M][K] (M <= 128) and B [K][N], B staged K-major ([N] rows of
// K, kBK) or MN-major ([K] rows of N); parts_b = 1 when B is exact in bf16.
// Operands come in chunks of eight along their contiguous index:
// a8(i, k, nv, x) fills x with A[i][k .. k+nv) (nv <= 8, zeros after), b8(k,
// j, nv, x) with B[k .. k+nv)[j] (kBK) or B[k][j .. j+nv).  Every thread
// loads all its chunks of a slab before it stores any to shared memory, and
// loads the next slab of the same output tile while the MMAs of the
// current one run.  The epilogue takes a warp's rows four
// at a time: pre(i, j) for all of them first, then store(i, j, v, pre(i, j))
// for every output element, whose results are summed per row and handed to
// rowsum(i, s) once per 128-column tile.  All threads of the CTA call it.
template <bool kBK, class FA, class FB, class FP, class FS, class FR>
__device__ void tc_gemm(TcCtx& c, int M, int N, int K, int parts_b, FA a, FB b, FP pre, FS store,
                        FR rowsum) {
  constexpr int kCh = 128 * 8 / kKT;     // chunks of each operand a thread stages per slab
  constexpr int kRows = kKT / 32;        // rows apart in a warp's epilogue batch
  static_assert(kCh * kKT == 128 * 8 && kCh * kKT == 64 * 16, "slab split");
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint8_t* As = c.sm;
  uint8_t* Bs = c.sm + kTP * kSlab;
  const uint32_t as = smem_u32(As), bs = smem_u32(Bs);
  const uint32_t idesc = idesc_bf16(128, 128, 0, kBK ? 0 : 1);
  volatile int no_abort = 0;
  const int nk = max(1, (K + 63) / 64), nt = (N + 127) / 128 * nk;
  float xa[kCh][8], xb[kCh][8];
  auto fetch = [&](int sl) {
    const int j0 = sl / nk * 128, k0 = sl % nk * 64;
#pragma unroll
    for (int l = 0; l < kCh; ++l) {
      const int ch = tid + l * kKT, r = ch >> 3, kk = k0 + (ch & 7) * 8;
      a(r, kk, r < M ? max(0, min(8, K - kk)) : 0, xa[l]);
    }
#pragma unroll
    for (int l = 0; l < kCh; ++l) {
      const int ch = tid + l * kKT;
      if (kBK) {
        const int r = ch >> 3, kk = k0 + (ch & 7) * 8;
        b(kk, j0 + r, j0 + r < N ? max(0, min(8, K - kk)) : 0, xb[l]);
      } else {
        // [64 rows of K][128 of N] as two halves of 64 columns (8 KB each)
        const int kr = ch >> 4, jj = j0 + (ch & 15) * 8;
        b(k0 + kr, jj, k0 + kr < K ? max(0, min(8, N - jj)) : 0, xb[l]);
      }
    }
  };
  if (nt > 0) fetch(0);
  for (int sl = 0; sl < nt; ++sl) {
    const int j0 = sl / nk * 128, kt = sl % nk;
#pragma unroll
    for (int l = 0; l < kCh; ++l) {
      const int ch = tid + l * kKT;
      uint4 pt[3];
      split3(xa[l], pt);
      const uint32_t off = sw128_offset(ch >> 3, ch & 7);
#pragma unroll
      for (int q = 0; q < kTP; ++q) *(uint4*)(As + q * kSlab + off) = pt[q];
    }
#pragma unroll
    for (int l = 0; l < kCh; ++l) {
      const int ch = tid + l * kKT;
      uint4 pt[3];
      split3(xb[l], pt);
      const uint32_t off = kBK ? sw128_offset(ch >> 3, ch & 7)
                               : ((ch & 15) >> 3) * (kSlab / 2) + sw128_offset(ch >> 4, ch & 7);
      for (int q = 0; q < parts_b; ++q) *(uint4*)(Bs + q * kSlab + off) = pt[q];
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      bool acc = kt > 0;
      for (int pa = 0; pa < kTP; ++pa)
        for (int pb = 0; pb < parts_b; ++pb) {
          if (pa + pb > 2) continue;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t ad = sw128_desc(as + pa * kSlab + kk * 32, 16, 1024);
            const uint64_t bd = kBK ? sw128_desc(bs + pb * kSlab + kk * 32, 16, 1024)
                                    : sw128_desc(bs + pb * kSlab + kk * 2048, kSlab / 2, 1024);
            mma_bf16(c.tmem, ad, bd, idesc, acc ? 1u : 0u);
            acc = true;
          }
        }
      mma_commit(c.bar);
    }
    if (sl + 1 < nt && kt + 1 < nk) fetch(sl + 1);
    if (!mbar_wait(c.bar, c.phase, &no_abort, kWaitBudget) && tid == 0)
      set_status(c.status, GRKV_ERR_TIMEOUT);
    c.phase ^= 1;
    tc_fence_after();
    if (kt != nk - 1) continue;
    // the tile through shared memory (the slabs are free: every MMA has completed)
    float* tile = (float*)c.sm;
    if (warp < 4) {
      const uint32_t la = c.tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
      for (int cc = 0; cc < 4; ++cc) {
        float v[32];
        tmem_ld32f(la + cc * 32, v);
        tmem_wait32(v);
#pragma unroll
        for (int e = 0; e < 32; ++e) tile[(warp * 32 + lane) * kTLD + cc * 32 + e] = v[e];
      }
    }
    tc_fence_before();
    __syncthreads();
    for (int i0 = warp; i0 < M; i0 += 4 * kRows) {
      float pv[4][4], tv[4][4];
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int i = i0 + rr * kRows;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int j = j0 + q * 32 + lane;
          const bool ok = i < M && j < N;
          pv[rr][q] = ok ? pre(i, j) : 0.f;
          tv[rr][q] = ok ? tile[i * kTLD + q * 32 + lane] : 0.f;
        }
      }
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int i = i0 + rr * kRows;
        if (i >= M) break;
        float sum = 0.f;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int j = j0 + q * 32 + lane;
          if (j < N) sum += store(i, j, tv[rr][q], pv[rr][q]);
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0) rowsum(i, sum);
      }
    }
    __syncthreads();
    if (sl + 1 < nt) fetch(sl + 1);
  }
}

// Sum over the block of one value per thread (all threads return it).
__device__ float block_sum(float v, float* sh) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (lane == 0) sh[wid] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < kKT / 32; ++i) t += sh[i];
  __syncthreads();
  return t;
}

// T <- X o (T - rowsum(X o T)), one warp per row.
__device__ void softmax_jacobian_rows(const float* X, float* T, int m, int B) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int r = wid; r < m; r += kKT / 32) {
    const float* x = X + (size_t)r * B;
    float* t = T + (size_t)r * B;
    float rho = 0.f;
    for (int j = lane; j < B; j += 32) rho = fmaf(x[j], t[j], rho);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) rho += __shfl_xor_sync(0xffffffffu, rho, o);
    for (int j = lane; j < B; j += 32) t[j] = x[j] * (t[j] - rho);
  }
  __syncthreads();
}

// Per-unit working set of the key step and of the alternation; r is the
// CTA's rank among the unit's C CTAs, whose m x d vectors are its own.
struct KUnit {
  int u, m, B;
  const int32_t* idx;
  const void* q;
  size_t kv_off;          // u * B * d
  const float* Y;
  float *X, *T, *dK, *T2, *GQ, *R, *Pd, *AP, *AL, *XV;
  float* E;               // rank 0's r: the right-hand side e on entry to CG
  uint8_t* fixed;
  __device__ KUnit(const KArgs& a, int u_, int r_ = 0) : u(u_), m(a.m), B(a.B) {
    idx = a.idx + (size_t)u * B;
    q = (const char*)a.q + (size_t)u * m * kD * (a.dtype == GRKV_F32 ? 4 : 2);
    kv_off = (size_t)u * B * kD;
    Y = a.y + (size_t)u * m * kD;
    X = a.X + (size_t)u * m * B;
    T = a.T + (size_t)u * m * B;
    dK = a.dK + kv_off;
    T2 = a.T2 + (size_t)u * m * B;
    GQ = a.GQ + (size_t)u * m * m;
    const size_t md = (size_t)m * kD;
    E = a.vec + (size_t)u * a.cluster * 5 * md;
    R = E + (size_t)r_ * 5 * md;
    Pd = R + md;
    AP = Pd + md;
    AL = AP + md;
    XV = AL + md;
    fixed = a.fixed + (size_t)u * B;
  }
};

__device__ __forceinline__ int kpos(const KArgs& a, const KUnit& k, int i) {
  const int j = k.idx[i];
  return (unsigned)j < (unsigned)a.n ? j : 0;
}

// Fixed set: retained sinks, the window, and the n_fix best-scored remaining
// retained prefix tokens (ties to the smaller position); k.T is scratch.
__device__ void fixed_set(const KArgs& a, const KUnit& k, int* hist, int* sh) {
  const int B = k.B;
  uint32_t* key = (uint32_t*)k.T;
  int nc = 0;
  for (int i = threadIdx.x; i < B; i += kKT) {
    const int j = kpos(a, k, i);
    const bool cand = j >= a.n_sink && j < a.P;
    key[i] = cand ? max(order_key(a.scores[(size_t)k.u * a.P + j]), 1u) : 0u;
    k.fixed[i] = cand ? 0 : 1;
    nc += cand;
  }
  __syncthreads();
  int ncand;
  (void)block_exclusive_scan(nc, sh + 8, &ncand);
  const int nf = min(a.n_fix, ncand);
  if (nf > 0) {
    auto get = [&](int i, uint32_t* kk) {
      *kk = key[i];
      return *kk != 0u;
    };
    auto mark = [&](int i, int) { k.fixed[i] = 1; };
    block_topk_mark(get, mark, B, nf, hist, sh);
  }
  __syncthreads();
}

// X = softmax over the retained keys of s q_r . k_j with the causal rule of
// the retained positions; kget(j, t) is element t of retained key j.
template <class FK>
__device__ void retained_softmax(const KArgs& a, const KUnit& k, GemmSmem& gs, FK kget) {
  const int m = k.m, B = k.B, dt = a.dtype;
  const float s = a.scale;
  block_gemm<false, true>(gs,
      m, B, kD, [&](int r, int t) { return ldv(k.q, (size_t)r * kD + t, dt); },
      [&](int t, int j) { return kget(j, t); },
      [&](int r, int j, float v) { k.X[(size_t)r * B + j] = s * v; });
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int r = wid; r < m; r += kKT / 32) {
    float* x = k.X + (size_t)r * B;
    const int lim = a.causal ? a.n - a.w + r % a.w : a.n - 1;
    float mx = -INFINITY;
    for (int j = lane; j < B; j += 32)
      if (kpos(a, k, j) <= lim) mx = fmaxf(mx, x[j]);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
    for (int j = lane; j < B; j += 32) {
      const float e = kpos(a, k, j) <= lim ? expf(x[j] - mx) : 0.f;
      x[j] = e;
      sum += e;
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const float inv = sum > 0.f ? 1.f / sum : 0.f;
    for (int j = lane; j < B; j += 32) x[j] *= inv;
  }
  __syncthreads();
}

// dK <- J_G^T W (fixed rows zero) with the values vget(j, t).
template <class FV>
__device__ void key_vjp(const KArgs& a, const KUnit& k, GemmSmem& gs, const float* W, FV vget) {
  const int m = k.m, B = k.B, dt = a.dtype;
  const float s = a.scale;
  block_gemm<false, true>(gs,
      m, B, kD, [&](int r, int t) { return W[(size_t)r * kD + t]; },
      [&](int t, int j) { return vget(j, t); },
      [&](int r, int j, float v) { k.T[(size_t)r * B + j] = v; });
  softmax_jacobian_rows(k.X, k.T, m, B);
  block_gemm<true, false>(gs,
      B, kD, m, [&](int j, int r) { return k.T[(size_t)r * B + j]; },
      [&](int r, int t) { return ldv(k.q, (size_t)r * kD + t, dt); },
      [&](int j, int t, float v) { k.dK[(size_t)j * kD + t] = k.fixed[j] ? 0.f : s * v; });
}

// Conjugate gradients on (J_G J_G^T + lambda_k I) alpha = e from alpha = 0,
// with e in k.R on entry; alpha ends in k.AL.  The operator is applied as
// three GEMMs through the query Gram (see the file comment).
template <class FV>
__device__ void key_cg(const KArgs& a, const KUnit& k, GemmSmem& gs, float* red, FV vget) {
  const int m = k.m, B = k.B, dt = a.dtype, md = m * kD;
  const float s = a.scale;
  block_gemm<false, true>(gs,
      m, m, kD, [&](int r, int t) { return ldv(k.q, (size_t)r * kD + t, dt); },
      [&](int t, int r2) { return ldv(k.q, (size_t)r2 * kD + t, dt); },
      [&](int r, int r2, float v) { k.GQ[(size_t)r * m + r2] = s * s * v; });
  float rs = 0.f;
  for (int i = threadIdx.x; i < md; i += kKT) {
    k.Pd[i] = k.R[i];
    k.AL[i] = 0.f;
    rs = fmaf(k.R[i], k.R[i], rs);
  }
  rs = block_sum(rs, red);
  const float stop = a.tol * a.tol * rs;
  for (int it = 0; it < a.iters; ++it) {
    if (!(rs > stop) || !(rs > 0.f)) break;
    // Ap = J_G (J_G^T p) + lambda p without forming dK: with dS = X o (dA -
    // rowsum(X o dA)), dA = p V^T, the JVP of dK = s dS^T Q (free rows) is
    // s Q dK^T = (s^2 Q Q^T) dS on the free columns and 0 on the fixed ones.
    block_gemm<false, true>(gs,
        m, B, kD, [&](int r, int t) { return k.Pd[(size_t)r * kD + t]; },
        [&](int t, int j) { return vget(j, t); },
        [&](int r, int j, float v) { k.T[(size_t)r * B + j] = v; });
    softmax_jacobian_rows(k.X, k.T, m, B);
    block_gemm(gs,
        m, B, m, [&](int r, int r2) { return k.GQ[(size_t)r * m + r2]; },
        [&](int r2, int j) { return k.T[(size_t)r2 * B + j]; },
        [&](int r, int j, float v) { k.T2[(size_t)r * B + j] = k.fixed[j] ? 0.f : v; });
    softmax_jacobian_rows(k.X, k.T2, m, B);
    block_gemm(gs,
        m, kD, B, [&](int r, int j) { return k.T2[(size_t)r * B + j]; },
        [&](int j, int t) { return vget(j, t); },
        [&](int r, int t, float v) {
          const size_t o = (size_t)r * kD + t;
          k.AP[o] = v + a.lambda_k * k.Pd[o];
        });
    float pap = 0.f;
    for (int i = threadIdx.x; i < md; i += kKT) pap = fmaf(k.Pd[i], k.AP[i], pap);
    pap = block_sum(pap, red);
    if (!(pap > 0.f)) break;   // the direction has vanished
    const float al = rs / pap;
    float rn = 0.f;
    for (int i = threadIdx.x; i < md; i += kKT) {
      k.AL[i] = fmaf(al, k.Pd[i], k.AL[i]);
      const float r = fmaf(-al, k.AP[i], k.R[i]);
      k.R[i] = r;
      rn = fmaf(r, r, rn);
    }
    rn = block_sum(rn, red);
    const float beta = rn / rs;
    for (int i = threadIdx.x; i < md; i += kKT) k.Pd[i] = fmaf(beta, k.Pd[i], k.R[i]);
    rs = rn;
    __syncthreads();
  }
}

// The share of a unit's CG that one CTA carries.  With C > 1 CTAs per unit
// (launched as one cluster, so they run together), rank r takes the
// retained columns [c0, c0 + nc) of the three products; the row sums rho2
// and the product J_G (J_G^T p) are summed over the ranks through the
// workspace, always in rank order, and every rank keeps its own copy of the
// m x d vectors and updates all of it.  Every rank therefore holds the same
// bits, takes the same branches and meets the same barriers.
struct KPart {
  int C, r, c0, nc;
  float* app;       // [C][m][d] partial products, one slot per rank (k.AP when C == 1)
  float* rho2p;     // [C][128] partial row sums (C > 1)
  int* cnt;         // barrier counter of the unit (C > 1)
  int nb;           // barriers passed
  int* flag;        // shared: the last barrier completed
};

__device__ __forceinline__ int ld_acquire_gpu(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Barrier of the C CTAs of a unit on its counter in global memory (zeroed
// before the launch).  Each CTA's earlier global writes are visible to the
// others' L2 loads (__ldcg) once it returns.  The wait is bounded: when the
// peers have not all arrived within the budget it sets the status and
// returns false, and the caller stops exchanging.
__device__ bool part_barrier(KPart& kp, int* status) {
  __syncthreads();
  ++kp.nb;
  if (threadIdx.x == 0) {
    int ok = 1;
    __threadfence();
    atomicAdd(kp.cnt, 1);
    const int target = kp.nb * kp.C;
    if (ld_acquire_gpu(kp.cnt) < target) {
      const long long t0 = clock64();
      while (ld_acquire_gpu(kp.cnt) < target)
        if (clock64() - t0 > kWaitBudget) {
          ok = 0;
          set_status(status, GRKV_ERR_TIMEOUT);
          break;
        }
    }
    __threadfence();
    *kp.flag = ok;
  }
  __syncthreads();
  return *kp.flag != 0;
}

// The m x d vectors of the tensor-core CG are walked by rows: warp w takes
// rows w, w + 8, ..., lane l the four columns 4l .. 4l+3 of each (one float4).
// Each loop loads a batch of rows before it stores anything, so that the
// loads of a batch are in flight together.
constexpr int kWarps = kKT / 32;

__device__ __forceinline__ float dot4(float4 a, float4 b, float acc) {
  acc = fmaf(a.x, b.x, acc);
  acc = fmaf(a.y, b.y, acc);
  acc = fmaf(a.z, b.z, acc);
  return fmaf(a.w, b.w, acc);
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
// Sum of float4 i over the kC partial slots (md floats apart), in rank order.
template <int kC>
__device__ __forceinline__ float4 sum_parts(const float* app, size_t md, int i) {
  float4 t[kC];
#pragma unroll
  for (int q = 0; q < kC; ++q) t[q] = __ldcg((const float4*)(app + (size_t)q * md) + i);
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int q = 0; q < kC; ++q) {
    v.x += t[q].x;
    v.y += t[q].y;
    v.z += t[q].z;
    v.w += t[q].w;
  }
  return v;
}

// Start of CG: X V* = sum of the partials, r = p = e (rank 0's r), alpha = 0,
// rho1 = rowsum(p o X V*); returns the thread's share of ||e||^2.
template <int kC>
__device__ float cg_start(const KUnit& k, const KPart& kp, float* rho1) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, m = k.m;
  const size_t md = (size_t)m * kD;
  float rs = 0.f;
  for (int r0 = warp; r0 < m; r0 += 2 * kWarps) {
    float4 xv[2], e[2];
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      const int r = r0 + b * kWarps, i = r * 32 + lane;
      xv[b] = r < m ? sum_parts<kC>(kp.app, md, i) : make_float4(0.f, 0.f, 0.f, 0.f);
      e[b] = r < m ? __ldcg((const float4*)k.E + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      const int r = r0 + b * kWarps, i = r * 32 + lane;
      if (r >= m) break;
      ((float4*)k.R)[i] = e[b];
      ((float4*)k.Pd)[i] = e[b];
      ((float4*)k.AL)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      rs = dot4(e[b], e[b], rs);
      ((float4*)k.XV)[i] = xv[b];
      const float d = warp_sum(dot4(e[b], xv[b], 0.f));
      if (lane == 0) rho1[r] = d;
    }
  }
  return rs;
}

// Ap = (sum of the partial products) + lambda p; returns the share of p . Ap.
template <int kC>
__device__ float cg_ap(const KUnit& k, const KPart& kp, float lambda) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, m = k.m;
  const size_t md = (size_t)m * kD;
  float pap = 0.f;
  for (int r0 = warp; r0 < m; r0 += 2 * kWarps) {
    float4 v[2], pd[2];
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      const int r = r0 + b * kWarps, i = r * 32 + lane;
      v[b] = r < m ? sum_parts<kC>(kp.app, md, i) : make_float4(0.f, 0.f, 0.f, 0.f);
      pd[b] = r < m ? ((const float4*)k.Pd)[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      const int r = r0 + b * kWarps, i = r * 32 + lane;
      if (r >= m) break;
      float4 ap = v[b];
      ap.x = fmaf(lambda, pd[b].x, ap.x);
      ap.y = fmaf(lambda, pd[b].y, ap.y);
      ap.z = fmaf(lambda, pd[b].z, ap.z);
      ap.w = fmaf(lambda, pd[b].w, ap.w);
      ((float4*)k.AP)[i] = ap;
      pap = dot4(pd[b], ap, pap);
    }
  }
  return pap;
}

// alpha += al p, r -= al Ap; returns the share of ||r||^2.
__device__ float cg_step(const KUnit& k, float al) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, m = k.m;
  float rn = 0.f;
  for (int r0 = warp; r0 < m; r0 += 4 * kWarps) {
    float4 pd[4], alp[4], ap[4], rr[4];
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int r = min(r0 + b * kWarps, m - 1), i = r * 32 + lane;
      pd[b] = ((const float4*)k.Pd)[i];
      alp[b] = ((const float4*)k.AL)[i];
      ap[b] = ((const float4*)k.AP)[i];
      rr[b] = ((const float4*)k.R)[i];
    }
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int r = r0 + b * kWarps, i = r * 32 + lane;
      if (r >= m) break;
      float4 a4 = alp[b], r4 = rr[b];
      a4.x = fmaf(al, pd[b].x, a4.x);
      a4.y = fmaf(al, pd[b].y, a4.y);
      a4.z = fmaf(al, pd[b].z, a4.z);
      a4.w = fmaf(al, pd[b].w, a4.w);
      r4.x = fmaf(-al, ap[b].x, r4.x);
      r4.y = fmaf(-al, ap[b].y, r4.y);
      r4.z = fmaf(-al, ap[b].z, r4.z);
      r4.w = fmaf(-al, ap[b].w, r4.w);
      ((float4*)k.AL)[i] = a4;
      ((float4*)k.R)[i] = r4;
      rn = dot4(r4, r4, rn);
    }
  }
  return rn;
}

// p = r + beta p and the next iteration's rho1 = rowsum(p o X V*).
__device__ void cg_dir(const KUnit& k, float beta, float* rho1) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, m = k.m;
  for (int r0 = warp; r0 < m; r0 += 4 * kWarps) {
    float4 pd[4], rr[4], xv[4];
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int r = min(r0 + b * kWarps, m - 1), i = r * 32 + lane;
      pd[b] = ((const float4*)k.Pd)[i];
      rr[b] = ((const float4*)k.R)[i];
      xv[b] = ((const float4*)k.XV)[i];
    }
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int r = r0 + b * kWarps, i = r * 32 + lane;
      if (r >= m) break;
      float4 p4 = rr[b];
      p4.x = fmaf(beta, pd[b].x, p4.x);
      p4.y = fmaf(beta, pd[b].y, p4.y);
      p4.z = fmaf(beta, pd[b].z, p4.z);
      p4.w = fmaf(beta, pd[b].w, p4.w);
      ((float4*)k.Pd)[i] = p4;
      const float d = warp_sum(dot4(p4, xv[b], 0.f));
      if (lane == 0) rho1[r] = d;
    }
  }
}

// key_cg with the three products of an iteration on the tensor cores
// (m <= 128), over the CTA's columns of kp.  The softmax Jacobians are
// applied as the next product stages its operand.  Their row sums are
//   rho1 = rowsum(X o (P V*^T)) = rowsum(P o (X V*)),  with X V* formed once,
//   rho2 = rowsum(X o T2), taken in the epilogue of the product writing T2,
// so that rho1 needs neither a pass over X nor, for a split unit, an exchange.
// X, the query Gram and the fixed flags are written by rank 0 before the
// first barrier and never again, and no other SM has read them before it,
// so plain (L1-cached) loads see them; the partials, rewritten every
// iteration by other CTAs, are read through L2 (__ldcg).
template <class FV8>
__device__ void key_cg_tc(const KArgs& a, const KUnit& k, GemmSmem& gs, float* red, TcCtx& c,
                          KPart& kp, float* rho1, float* rho2, int parts_v, FV8 vget8) {
  const int m = k.m, B = k.B, dt = a.dtype, md = m * kD;
  const int C = kp.C, c0 = kp.c0, nc = kp.nc;
  const float s = a.scale;
  float* mine = kp.app + (size_t)kp.r * md;
  if (kp.r == 0)
    block_gemm<false, true>(gs,
        m, m, kD, [&](int r, int t) { return ldv(k.q, (size_t)r * kD + t, dt); },
        [&](int t, int r2) { return ldv(k.q, (size_t)r2 * kD + t, dt); },
        [&](int r, int r2, float v) { k.GQ[(size_t)r * m + r2] = s * s * v; });
  const bool split = C > 1;
  bool ok = !split || part_barrier(kp, a.status);
  // X V* over the CTA's columns, summed over the ranks in cg_start
  tc_gemm<false>(c, m, kD, nc, parts_v,
      [&](int r, int j, int nv, float* x) { ld8(k.X + (size_t)r * B + c0 + j, nv, x); },
      [&](int j, int t, int nv, float* x) { vget8(c0 + j, t, nv, x); },
      [](int, int) { return 0.f; },
      [&](int r, int t, float v, float) {
        mine[(size_t)r * kD + t] = v;
        return 0.f;
      }, [](int, float) {});
  if (split && ok) ok = part_barrier(kp, a.status);
  float rs = C == 8 ? cg_start<8>(k, kp, rho1)
           : C == 4 ? cg_start<4>(k, kp, rho1)
           : C == 2 ? cg_start<2>(k, kp, rho1) : cg_start<1>(k, kp, rho1);
  rs = block_sum(rs, red);
  const float stop = a.tol * a.tol * rs;
  auto add2 = [&](int i, float v) { rho2[i] += v; };
  for (int it = 0; it < a.iters && ok; ++it) {
    if (!(rs > stop) || !(rs > 0.f)) break;
    if (threadIdx.x < 128) rho2[threadIdx.x] = 0.f;
    __syncthreads();
    // T = P V*^T
    tc_gemm<true>(c, m, nc, kD, parts_v,
        [&](int r, int t, int nv, float* x) { ld8(k.Pd + (size_t)r * kD + t, nv, x); },
        [&](int t, int j, int nv, float* x) { vget8(c0 + j, t, nv, x); },
        [](int, int) { return 0.f; },
        [&](int r, int j, float v, float) {
          k.T[(size_t)r * B + c0 + j] = v;
          return 0.f;
        }, [](int, float) {});
    // T2 = (s^2 Q Q^T) dS on the free columns, dS = X o (T - rho1)
    tc_gemm<false>(c, m, nc, m, kTP,
        [&](int r, int r2, int nv, float* x) { ld8(k.GQ + (size_t)r * m + r2, nv, x); },
        [&](int r2, int j, int nv, float* x) {
          float t[8];
          const size_t o = (size_t)r2 * B + c0 + j;
          ld8(k.X + o, nv, x);
          ld8(k.T + o, nv, t);
          const float rh = nv > 0 ? rho1[r2] : 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] *= t[e] - rh;
        },
        // X (a probability, >= 0) of a free column, -1 for a fixed one
        [&](int r, int j) {
          return k.fixed[c0 + j] ? -1.f : k.X[(size_t)r * B + c0 + j];
        },
        [&](int r, int j, float v, float x) {
          const float t2 = x < 0.f ? 0.f : v;
          k.T2[(size_t)r * B + c0 + j] = t2;
          return x < 0.f ? 0.f : x * t2;
        }, add2);
    if (C > 1) {
      if (threadIdx.x < m) kp.rho2p[(size_t)kp.r * 128 + threadIdx.x] = rho2[threadIdx.x];
      ok = part_barrier(kp, a.status);
      if (threadIdx.x < m) {
        float v = 0.f;
        for (int q = 0; q < C; ++q) v += __ldcg(kp.rho2p + (size_t)q * 128 + threadIdx.x);
        rho2[threadIdx.x] = v;
      }
      __syncthreads();
      if (!ok) break;
    }
    // the CTA's share of J_G (J_G^T p) = dS2 V*, dS2 = X o (T2 - rho2)
    tc_gemm<false>(c, m, kD, nc, parts_v,
        [&](int r, int j, int nv, float* x) {
          float t[8];
          const size_t o = (size_t)r * B + c0 + j;
          ld8(k.X + o, nv, x);
          ld8(k.T2 + o, nv, t);
          const float rh = nv > 0 ? rho2[r] : 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] *= t[e] - rh;
        },
        [&](int j, int t, int nv, float* x) { vget8(c0 + j, t, nv, x); },
        [](int, int) { return 0.f; },
        [&](int r, int t, float v, float) {
          mine[(size_t)r * kD + t] = v;
          return 0.f;
        }, [](int, float) {});
    if (C > 1 && !(ok = part_barrier(kp, a.status))) break;
    // Ap = J_G (J_G^T p) + lambda p
    float pap = C == 8 ? cg_ap<8>(k, kp, a.lambda_k)
              : C == 4 ? cg_ap<4>(k, kp, a.lambda_k)
              : C == 2 ? cg_ap<2>(k, kp, a.lambda_k) : cg_ap<1>(k, kp, a.lambda_k);
    pap = block_sum(pap, red);
    if (!(pap > 0.f)) break;   // the direction has vanished
    const float al = rs / pap;
    const float rn = block_sum(cg_step(k, al), red);
    cg_dir(k, rn / rs, rho1);
    rs = rn;
    __syncthreads();
  }
}

// Tensor-core context of a key-step CTA: dynamic shared memory for the
// slabs, a 128-column TMEM accumulator (allocated by warp 0) and the MMA
// barrier.  tc_release frees the TMEM once every thread is done with it.
__device__ void tc_setup(TcCtx& c, uint8_t* dyn, uint32_t* tmem_s, uint64_t* bar, int* status) {
  c.sm = (uint8_t*)(((uintptr_t)dyn + 1023) & ~(uintptr_t)1023);
  c.bar = bar;
  c.phase = 0;
  c.status = status;
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  if (threadIdx.x < 32) {
    tmem_alloc(tmem_s, 128);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  c.tmem = *tmem_s;
}
__device__ void tc_release(const TcCtx& c) {
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x < 32) tmem_dealloc(c.tmem, 128);
}

__device__ __forceinline__ void stv(void* p, size_t i, int dtype, float v) {
  if (dtype == GRKV_F32)
    ((float*)p)[i] = v;
  else
    ((__nv_bfloat16*)p)[i] = __float2bfloat16_rn(v);
}

// Key step of Algorithm 1 at t = 0: linearised at K0 (k_out on entry) with
// V* = v_out; K* to k_out (and, for an alternation, in fp32 to Kt).
__global__ void __launch_bounds__(kKT, 2) k_key_step(KArgs a) {
  __shared__ int hist[256], sh[64];
  __shared__ float red[kKT / 32];
  __shared__ GemmSmem gs;
  __shared__ float rho[2][128];
  __shared__ uint64_t tc_bar;
  __shared__ uint32_t tc_tmem;
  __shared__ int part_flag;
  extern __shared__ uint8_t tc_dyn[];
  const int C = a.cluster, u = blockIdx.x / C, rank = blockIdx.x - u * C;
  const KUnit k(a, u, rank);
  const int B = k.B, dt = a.dtype;
  TcCtx tc{};
  if (a.use_tc) tc_setup(tc, tc_dyn, &tc_tmem, &tc_bar, a.status);
  auto vget = [&](int j, int t) { return ldv(a.v_out, k.kv_off + (size_t)j * kD + t, dt); };
  if (rank == 0) {
    fixed_set(a, k, hist, sh);
    retained_softmax(a, k, gs, [&](int j, int t) { return ldv(a.k_out, k.kv_off + (size_t)j * kD + t, dt); });
    // e = Y - X V*
    block_gemm(gs,
        k.m, kD, B, [&](int r, int j) { return k.X[(size_t)r * B + j]; }, vget,
        [&](int r, int t, float v) { k.R[(size_t)r * kD + t] = k.Y[(size_t)r * kD + t] - v; });
  }
  if (a.use_tc) {
    // V* row j, columns t .. t+nv
    auto vget8 = [&](int j, int t, int nv, float* x) {
      const size_t o = k.kv_off + (size_t)j * kD + t;
      if (dt == GRKV_BF16)
        ld8((const __nv_bfloat16*)a.v_out + o, nv, x);
      else
        ld8((const float*)a.v_out + o, nv, x);
    };
    // rank r carries columns [r * Bc, r * Bc + Bc) (the last rank the rest)
    const int Bc = ((B + C - 1) / C + 7) / 8 * 8;
    KPart kp{};
    kp.C = C;
    kp.r = rank;
    kp.c0 = min(B, rank * Bc);
    kp.nc = min(B, kp.c0 + Bc) - kp.c0;
    kp.app = C > 1 ? a.app + (size_t)u * C * k.m * kD : k.AP;
    kp.rho2p = C > 1 ? a.rho2p + (size_t)u * C * 128 : nullptr;
    kp.cnt = C > 1 ? a.cnt + u : nullptr;
    kp.flag = &part_flag;
    key_cg_tc(a, k, gs, red, tc, kp, rho[0], rho[1], dt == GRKV_BF16 ? 1 : kTP, vget8);
    tc_release(tc);
    if (rank != 0) return;
  } else {
    key_cg(a, k, gs, red, vget);
  }
  // K*_G = K0_G + J_G^T alpha; fixed rows keep K0
  key_vjp(a, k, gs, k.AL, vget);
  for (int i = threadIdx.x; i < B * kD; i += kKT) {
    const int j = i / kD;
    const size_t o = k.kv_off + i;
    const float k0 = ldv(a.k_out, o, dt);
    const float v = k.fixed[j] ? k0 : k0 + k.dK[i];
    if (a.Kt) a.Kt[o] = v;
    if (!k.fixed[j]) stv(a.k_out, o, dt, v);
  }
}

// In-place Cholesky of the m x m matrix G (row-major, lower triangle used)
// by one CTA; returns false on a non-positive pivot.
__device__ bool block_cholesky(float* G, int m, int* flag) {
  if (threadIdx.x == 0) *flag = 0;
  __syncthreads();
  for (int c = 0; c < m; ++c) {
    if (threadIdx.x == 0) {
      const float d = G[(size_t)c * m + c];
      if (!(d > 0.f)) *flag = 1;
      G[(size_t)c * m + c] = d > 0.f ? sqrtf(d) : 1.f;
    }
    __syncthreads();
    const float inv = 1.f / G[(size_t)c * m + c];
    for (int i = c + 1 + threadIdx.x; i < m; i += kKT) G[(size_t)i * m + c] *= inv;
    __syncthreads();
    const int rem = m - c - 1;
    for (int e = threadIdx.x; e < rem * rem; e += kKT) {
      const int i = c + 1 + e / rem, j = c + 1 + e % rem;
      if (j <= i) G[(size_t)i * m + j] -= G[(size_t)i * m + c] * G[(size_t)j * m + c];
    }
    __syncthreads();
  }
  return *flag == 0;
}

// One step t >= 1 of Algorithm 1's alternation for every unit still running:
// the value step from V0 with X at the current keys K^(t) (Kt), then the key
// step linearised at K^(t) (right-hand side e + J_G (K^(t) - K0)).  Writes
// V^(t+1), K^(t+1) to v_out / k_out (rounded) and to Vt / Kt (fp32), and
// marks the unit done once both changes are <= step_tol.
__global__ void __launch_bounds__(kKT, 2) k_alternate_step(KArgs a) {
  __shared__ int hist[256], sh[64];
  __shared__ float red[kKT / 32];
  __shared__ GemmSmem gs;
  __shared__ int flag;
  __shared__ float rho[2][128];
  __shared__ uint64_t tc_bar;
  __shared__ uint32_t tc_tmem;
  extern __shared__ uint8_t tc_dyn[];
  const KUnit k(a, blockIdx.x);
  if (a.done[k.u]) return;
  const int m = k.m, B = k.B, dt = a.dtype;
  const size_t un = (size_t)k.u * a.n;
  auto k0 = [&](int j, int t) { return ldv(a.k, (un + kpos(a, k, j)) * kD + t, dt); };
  auto v0 = [&](int j, int t) { return ldv(a.v, (un + kpos(a, k, j)) * kD + t, dt); };
  fixed_set(a, k, hist, sh);
  retained_softmax(a, k, gs, [&](int j, int t) { return a.Kt[k.kv_off + (size_t)j * kD + t]; });

  // ---- value step: V = V0 + X_G^T (X_G X_G^T + lambda_v I)^-1 (Y - X V0)
  float* G = a.G + (size_t)k.u * m * m;
  float* Z = a.RZ + (size_t)k.u * m * kD;
  bool solved = false;
  if (!a.lambda_inf) {
    block_gemm<false, true>(gs,
        m, m, B, [&](int r, int j) { return k.fixed[j] ? 0.f : k.X[(size_t)r * B + j]; },
        [&](int j, int r2) { return k.fixed[j] ? 0.f : k.X[(size_t)r2 * B + j]; },
        [&](int r, int r2, float v) { G[(size_t)r * m + r2] = v + (r == r2 ? a.lambda_v : 0.f); });
    block_gemm(gs,
        m, kD, B, [&](int r, int j) { return k.X[(size_t)r * B + j]; }, v0,
        [&](int r, int t, float v) { Z[(size_t)r * kD + t] = k.Y[(size_t)r * kD + t] - v; });
    solved = block_cholesky(G, m, &flag);
    if (!solved && threadIdx.x == 0) set_status(a.status, GRKV_ERR_NUMERIC);
    if (solved) {
      for (int c = 0; c < m; ++c) {   // L W = R
        const float inv = 1.f / G[(size_t)c * m + c];
        for (int t = threadIdx.x; t < kD; t += kKT) Z[(size_t)c * kD + t] *= inv;
        __syncthreads();
        for (int e = threadIdx.x; e < (m - c - 1) * kD; e += kKT) {
          const int i = c + 1 + e / kD, t = e % kD;
          Z[(size_t)i * kD + t] -= G[(size_t)i * m + c] * Z[(size_t)c * kD + t];
        }
        __syncthreads();
      }
      for (int c = m - 1; c >= 0; --c) {   // L^T Z = W
        const float inv = 1.f / G[(size_t)c * m + c];
        for (int t = threadIdx.x; t < kD; t += kKT) Z[(size_t)c * kD + t] *= inv;
        __syncthreads();
        for (int e = threadIdx.x; e < c * kD; e += kKT) {
          const int i = e / kD, t = e % kD;
          Z[(size_t)i * kD + t] -= G[(size_t)c * m + i] * Z[(size_t)c * kD + t];
        }
        __syncthreads();
      }
    }
  }
  // V^(t+1) (fp32 in dK as scratch), its largest change, then v_out / Vt
  if (solved) {
    block_gemm<true, false>(gs,
        B, kD, m, [&](int j, int r) { return k.fixed[j] ? 0.f : k.X[(size_t)r * B + j]; },
        [&](int r, int t) { return Z[(size_t)r * kD + t]; },
        [&](int j, int t, float v) { k.dK[(size_t)j * kD + t] = v0(j, t) + v; });
  } else {
    for (int i = threadIdx.x; i < B * kD; i += kKT) k.dK[i] = v0(i / kD, i % kD);
    __syncthreads();
  }
  float dv = 0.f;
  for (int i = threadIdx.x; i < B * kD; i += kKT) {
    const size_t o = k.kv_off + i;
    const float prev = a.vt_valid ? a.Vt[o] : ldv(a.v_out, o, dt);
    dv = fmaxf(dv, fabsf(k.dK[i] - prev));
  }
  __syncthreads();
  for (int i = threadIdx.x; i < B * kD; i += kKT) {
    const size_t o = k.kv_off + i;
    a.Vt[o] = k.dK[i];
    stv(a.v_out, o, dt, k.dK[i]);
  }
  __syncthreads();

  // ---- key step at K^(t) against V^(t+1) (fp32, Vt)
  auto vget = [&](int j, int t) { return a.Vt[k.kv_off + (size_t)j * kD + t]; };
  // e = Y - X V, then + J_G g with g = K^(t) - K0 on the free rows:
  // dS = s Q g^T, dA = X o (dS - rowsum(X o dS)), df = dA V
  block_gemm(gs,
      m, kD, B, [&](int r, int j) { return k.X[(size_t)r * B + j]; }, vget,
      [&](int r, int t, float v) { k.R[(size_t)r * kD + t] = k.Y[(size_t)r * kD + t] - v; });
  block_gemm<false, true>(gs,
      m, B, kD, [&](int r, int t) { return ldv(k.q, (size_t)r * kD + t, dt); },
      [&](int t, int j) {
        return k.fixed[j] ? 0.f : a.Kt[k.kv_off + (size_t)j * kD + t] - k0(j, t);
      },
      [&](int r, int j, float v) { k.T[(size_t)r * B + j] = a.scale * v; });
  softmax_jacobian_rows(k.X, k.T, m, B);
  block_gemm(gs,
      m, kD, B, [&](int r, int j) { return k.T[(size_t)r * B + j]; }, vget,
      [&](int r, int t, float v) { k.R[(size_t)r * kD + t] += v; });
  if (a.use_tc) {
    TcCtx tc{};
    tc_setup(tc, tc_dyn, &tc_tmem, &tc_bar, a.status);
    auto vget8 = [&](int j, int t, int nv, float* x) {
      ld8(a.Vt + k.kv_off + (size_t)j * kD + t, nv, x);
    };
    KPart kp{};
    kp.C = 1;
    kp.nc = B;
    kp.app = k.AP;
    kp.flag = &flag;
    key_cg_tc(a, k, gs, red, tc, kp, rho[0], rho[1], kTP, vget8);
    tc_release(tc);
  } else {
    key_cg(a, k, gs, red, vget);
  }
  key_vjp(a, k, gs, k.AL, vget);
  float dkmax = 0.f;
  for (int i = threadIdx.x; i < B * kD; i += kKT) {
    const int j = i / kD;
    const size_t o = k.kv_off + i;
    const float base = k0(j, i % kD);
    const float v = k.fixed[j] ? base : base + k.dK[i];
    dkmax = fmaxf(dkmax, fabsf(v - a.Kt[o]));
    a.Kt[o] = v;
    stv(a.k_out, o, dt, v);
  }
  // the stop test: both changes within step_tol
  float ch = fmaxf(dkmax, dv);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) ch = fmaxf(ch, __shfl_xor_sync(0xffffffffu, ch, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ch;
  __syncthreads();
  if (threadIdx.x == 0) {
    float mx = 0.f;
    for (int i = 0; i < kKT / 32; ++i) mx = fmaxf(mx, red[i]);
    if (mx <= a.step_tol) a.done[k.u] = 1;
  }
}

}  // namespace

// CTAs per unit in k_key_step: with few units, a unit's CG products are split
// over up to 8 CTAs (at least 64 retained columns each) while the units
// times the split stay within one CTA per SM of a GB300 (152 SMs).
constexpr int kKeySms = 152;
int key_cluster(const Shape& s) {
  if (s.m > 128) return 1;   // the fp32 CUDA-core CG runs one CTA per unit
  int c = 1;
  while (c < 8 && (long long)s.U * 2 * c <= kKeySms && s.B >= 2 * c * 64) c *= 2;
  return c;
}

namespace {
size_t a256(size_t x) { return (x + 255) & ~(size_t)255; }

// Regions of the key step's workspace (offsets from its base, 256-aligned).
struct KeyLayout {
  size_t vec, app, rho2p, cnt, X, T, dK, T2, GQ, fixed, alt, total;
};
KeyLayout key_layout(const Shape& s, int C) {
  const size_t U = (size_t)s.U, m = (size_t)s.m, B = (size_t)s.B, d = (size_t)kD;
  KeyLayout l{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = a256(off + bytes);
    return o;
  };
  l.vec = take(U * C * 5 * m * d * 4);
  l.app = take(C > 1 ? U * C * m * d * 4 : 0);
  l.rho2p = take(C > 1 ? U * C * 128 * 4 : 0);
  l.cnt = take(C > 1 ? U * 4 : 0);
  l.X = take(U * m * B * 4);
  l.T = take(U * m * B * 4);
  l.dK = take(U * B * d * 4);
  l.T2 = take(U * m * B * 4);
  l.GQ = take(U * m * m * 4);
  l.fixed = take(U * B);
  l.alt = take(s.steps > 1 ? U * (2 * B * d * 4 + m * m * 4 + m * d * 4 + 4) + 1024 : 0);
  l.total = off;
  return l;
}
}  // namespace

size_t key_ws_bytes(const Shape& s) { return key_layout(s, key_cluster(s)).total + 256; }

cudaError_t launch_key_step(const Shape& s, const void* q, const void* k, const void* v,
                            const float* y, const float* scores, const int32_t* idx,
                            void* v_out, void* k_out, char* ws, const WsLayout& L,
                            cudaStream_t st) {
  const size_t U = (size_t)s.U, m = (size_t)s.m, B = (size_t)s.B, d = (size_t)kD;
  char* base = (char*)(((uintptr_t)(ws + L.key) + 255) & ~(uintptr_t)255);
  KArgs a{};
  a.n = s.n;
  a.w = s.w;
  a.m = s.m;
  a.B = s.B;
  a.P = s.P;
  a.n_sink = s.n_sink;
  a.n_fix = s.n_fix;
  a.causal = s.causal;
  a.dtype = s.dtype;
  a.iters = s.cg_iters;
  a.scale = s.scale;
  a.lambda_k = s.lambda_k;
  a.tol = s.cg_tol;
  a.lambda_v = s.lambda;
  a.lambda_inf = s.lambda_inf;
  a.step_tol = s.step_tol;
  a.q = q;
  a.k = k;
  a.v = v;
  a.y = y;
  a.scores = scores;
  a.idx = idx;
  a.v_out = v_out;
  a.k_out = k_out;
  a.status = (int*)(ws + L.status);
  a.use_tc = s.m <= 128;
  const uint32_t dyn = a.use_tc ? kTcSmem : 0;
  cudaError_t e = cudaFuncSetAttribute(k_key_step, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kTcSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_alternate_step, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kTcSmem);
  if (e != cudaSuccess) return e;
  // the split the workspace was sized for, halved while the device cannot
  // hold a cluster of that many CTAs
  int C = key_cluster(s);
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.blockDim = dim3(kKT);
  cfg.dynamicSmemBytes = dyn;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  for (; C > 1; C /= 2) {
    cfg.gridDim = dim3((unsigned)(U * C));
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    int nclusters = 0;
    if (cudaOccupancyMaxActiveClusters(&nclusters, k_key_step, &cfg) == cudaSuccess &&
        nclusters > 0)
      break;
    (void)cudaGetLastError();
  }
  const KeyLayout kl = key_layout(s, C);
  a.cluster = C;
  a.vec = (float*)(base + kl.vec);
  a.app = (float*)(base + kl.app);
  a.rho2p = (float*)(base + kl.rho2p);
  a.cnt = (int*)(base + kl.cnt);
  a.X = (float*)(base + kl.X);
  a.T = (float*)(base + kl.T);
  a.dK = (float*)(base + kl.dK);
  a.T2 = (float*)(base + kl.T2);
  a.GQ = (float*)(base + kl.GQ);
  a.fixed = (uint8_t*)(base + kl.fixed);
  if (s.steps > 1) {
    char* alt = base + kl.alt;
    a.Kt = (float*)alt;
    a.Vt = a.Kt + U * B * d;
    a.G = a.Vt + U * B * d;
    a.RZ = a.G + U * m * m;
    a.done = (int*)(a.RZ + U * m * d);
    e = cudaMemsetAsync(a.done, 0, U * sizeof(int), st);
    if (e != cudaSuccess) return e;
  }
  count_launches(1);
  if (C > 1) {
    e = cudaMemsetAsync(a.cnt, 0, U * sizeof(int), st);
    if (e != cudaSuccess) return e;
    cfg.gridDim = dim3((unsigned)(U * C));
    attr[0].val.clusterDim.x = C;
    e = cudaLaunchKernelEx(&cfg, k_key_step, a);
  } else {
    k_key_step<<<s.U, kKT, dyn, st>>>(a);
    e = cudaGetLastError();
  }
  for (int t = 1; t < s.steps && e == cudaSuccess; ++t) {
    a.vt_valid = t > 1;   // V^(1) exists only as written to v_out (rounded)
    count_launches(1);
    k_alternate_step<<<s.U, kKT, dyn, st>>>(a);
    e = cudaGetLastError();
  }
  return e;
}

}  // namespace grkv
