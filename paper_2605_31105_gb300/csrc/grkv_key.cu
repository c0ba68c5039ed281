// Key step of Algorithm 1 at t = 0 (Sec. 3.4 "Key step", App. D.2), one CTA
// per unit: fp32 on CUDA cores, with the CG products on the tensor cores
// (three-part bf16 splits of the fp32 operands) when m <= 128.
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
  float* vec;             // [U][4][m][d]: r, p, Ap, alpha
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
// j, nv, x) with B[k .. k+nv)[j] (kBK) or B[k][j .. j+nv).  For every output
// element store(i, j, v) returns a value summed per row and handed to
// rowsum(i, s) once per 128-column tile.  All threads of the CTA call it.
template <bool kBK, class FA, class FB, class FS, class FR>
__device__ void tc_gemm(TcCtx& c, int M, int N, int K, int parts_b, FA a, FB b, FS store,
                        FR rowsum) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint8_t* As = c.sm;
  uint8_t* Bs = c.sm + kTP * kSlab;
  const uint32_t as = smem_u32(As), bs = smem_u32(Bs);
  const uint32_t idesc = idesc_bf16(128, 128, 0, kBK ? 0 : 1);
  volatile int no_abort = 0;
  for (int j0 = 0; j0 < N; j0 += 128) {
    for (int k0 = 0; k0 < K; k0 += 64) {
      for (int ch = tid; ch < 128 * 8; ch += kKT) {
        const int r = ch >> 3, c8 = ch & 7, kk = k0 + c8 * 8;
        float x[8];
        a(r, kk, r < M ? max(0, min(8, K - kk)) : 0, x);
        uint4 pt[3];
        split3(x, pt);
        const uint32_t off = sw128_offset(r, c8);
#pragma unroll
        for (int q = 0; q < kTP; ++q) *(uint4*)(As + q * kSlab + off) = pt[q];
      }
      if (kBK) {
        for (int ch = tid; ch < 128 * 8; ch += kKT) {
          const int r = ch >> 3, c8 = ch & 7, kk = k0 + c8 * 8;
          float x[8];
          b(kk, j0 + r, j0 + r < N ? max(0, min(8, K - kk)) : 0, x);
          uint4 pt[3];
          split3(x, pt);
          const uint32_t off = sw128_offset(r, c8);
          for (int q = 0; q < parts_b; ++q) *(uint4*)(Bs + q * kSlab + off) = pt[q];
        }
      } else {
        // [64 rows of K][128 of N] as two halves of 64 columns (8 KB each)
        for (int ch = tid; ch < 64 * 16; ch += kKT) {
          const int kr = ch >> 4, nc = ch & 15, hf = nc >> 3, c8 = nc & 7, jj = j0 + nc * 8;
          float x[8];
          b(k0 + kr, jj, k0 + kr < K ? max(0, min(8, N - jj)) : 0, x);
          uint4 pt[3];
          split3(x, pt);
          const uint32_t off = hf * (kSlab / 2) + sw128_offset(kr, c8);
          for (int q = 0; q < parts_b; ++q) *(uint4*)(Bs + q * kSlab + off) = pt[q];
        }
      }
      fence_proxy_async_smem();
      __syncthreads();
      if (tid == 0) {
        tc_fence_after();
        bool acc = k0 > 0;
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
      if (!mbar_wait(c.bar, c.phase, &no_abort, kWaitBudget) && tid == 0)
        set_status(c.status, GRKV_ERR_TIMEOUT);
      c.phase ^= 1;
      tc_fence_after();
    }
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
    for (int i = warp; i < M; i += kKT / 32) {
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int jj = q * 32 + lane, j = j0 + jj;
        if (j < N) sum += store(i, j, tile[i * kTLD + jj]);
      }
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      if (lane == 0) rowsum(i, sum);
    }
    __syncthreads();
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

// Per-unit working set of the key step and of the alternation.
struct KUnit {
  int u, m, B;
  const int32_t* idx;
  const void* q;
  size_t kv_off;          // u * B * d
  const float* Y;
  float *X, *T, *dK, *T2, *GQ, *R, *Pd, *AP, *AL;
  uint8_t* fixed;
  __device__ KUnit(const KArgs& a, int u_) : u(u_), m(a.m), B(a.B) {
    idx = a.idx + (size_t)u * B;
    q = (const char*)a.q + (size_t)u * m * kD * (a.dtype == GRKV_F32 ? 4 : 2);
    kv_off = (size_t)u * B * kD;
    Y = a.y + (size_t)u * m * kD;
    X = a.X + (size_t)u * m * B;
    T = a.T + (size_t)u * m * B;
    dK = a.dK + kv_off;
    T2 = a.T2 + (size_t)u * m * B;
    GQ = a.GQ + (size_t)u * m * m;
    R = a.vec + (size_t)u * 4 * m * kD;
    Pd = R + (size_t)m * kD;
    AP = Pd + (size_t)m * kD;
    AL = AP + (size_t)m * kD;
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

// key_cg with the three products of an iteration on the tensor cores
// (m <= 128).  The softmax Jacobians are applied as the next product stages
// its operand: the row sums rho1 = rowsum(X o T) and rho2 = rowsum(X o T2)
// are taken in the epilogues of the products that write T and T2.
template <class FV, class FV8>
__device__ void key_cg_tc(const KArgs& a, const KUnit& k, GemmSmem& gs, float* red, TcCtx& c,
                          float* rho1, float* rho2, int parts_v, FV vget, FV8 vget8) {
  (void)vget;
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
  auto add1 = [&](int i, float v) { rho1[i] += v; };
  auto add2 = [&](int i, float v) { rho2[i] += v; };
  for (int it = 0; it < a.iters; ++it) {
    if (!(rs > stop) || !(rs > 0.f)) break;
    if (threadIdx.x < 128) rho1[threadIdx.x] = rho2[threadIdx.x] = 0.f;
    __syncthreads();
    // T = P V*^T
    tc_gemm<true>(c, m, B, kD, parts_v,
        [&](int r, int t, int nv, float* x) { ld8(k.Pd + (size_t)r * kD + t, nv, x); },
        [&](int t, int j, int nv, float* x) { vget8(j, t, nv, x); },
        [&](int r, int j, float v) {
          k.T[(size_t)r * B + j] = v;
          return k.X[(size_t)r * B + j] * v;
        }, add1);
    // T2 = (s^2 Q Q^T) dS on the free columns, dS = X o (T - rho1)
    tc_gemm<false>(c, m, B, m, kTP,
        [&](int r, int r2, int nv, float* x) { ld8(k.GQ + (size_t)r * m + r2, nv, x); },
        [&](int r2, int j, int nv, float* x) {
          float t[8];
          const size_t o = (size_t)r2 * B + j;
          ld8(k.X + o, nv, x);
          ld8(k.T + o, nv, t);
          const float rh = nv > 0 ? rho1[r2] : 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] *= t[e] - rh;
        },
        [&](int r, int j, float v) {
          const float t2 = k.fixed[j] ? 0.f : v;
          k.T2[(size_t)r * B + j] = t2;
          return k.X[(size_t)r * B + j] * t2;
        }, add2);
    // Ap = dS2 V* + lambda p, dS2 = X o (T2 - rho2)
    tc_gemm<false>(c, m, kD, B, parts_v,
        [&](int r, int j, int nv, float* x) {
          float t[8];
          const size_t o = (size_t)r * B + j;
          ld8(k.X + o, nv, x);
          ld8(k.T2 + o, nv, t);
          const float rh = nv > 0 ? rho2[r] : 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] *= t[e] - rh;
        },
        [&](int j, int t, int nv, float* x) { vget8(j, t, nv, x); },
        [&](int r, int t, float v) {
          const size_t o = (size_t)r * kD + t;
          k.AP[o] = v + a.lambda_k * k.Pd[o];
          return 0.f;
        }, [](int, float) {});
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
__global__ void __launch_bounds__(kKT) k_key_step(KArgs a) {
  __shared__ int hist[256], sh[64];
  __shared__ float red[kKT / 32];
  __shared__ GemmSmem gs;
  __shared__ float rho[2][128];
  __shared__ uint64_t tc_bar;
  __shared__ uint32_t tc_tmem;
  extern __shared__ uint8_t tc_dyn[];
  const KUnit k(a, blockIdx.x);
  const int B = k.B, dt = a.dtype;
  TcCtx tc{};
  if (a.use_tc) tc_setup(tc, tc_dyn, &tc_tmem, &tc_bar, a.status);
  fixed_set(a, k, hist, sh);
  retained_softmax(a, k, gs, [&](int j, int t) { return ldv(a.k_out, k.kv_off + (size_t)j * kD + t, dt); });
  auto vget = [&](int j, int t) { return ldv(a.v_out, k.kv_off + (size_t)j * kD + t, dt); };
  // e = Y - X V*
  block_gemm(gs,
      k.m, kD, B, [&](int r, int j) { return k.X[(size_t)r * B + j]; }, vget,
      [&](int r, int t, float v) { k.R[(size_t)r * kD + t] = k.Y[(size_t)r * kD + t] - v; });
  if (a.use_tc) {
    // V* row j, columns t .. t+nv
    auto vget8 = [&](int j, int t, int nv, float* x) {
      const size_t o = k.kv_off + (size_t)j * kD + t;
      if (dt == GRKV_BF16)
        ld8((const __nv_bfloat16*)a.v_out + o, nv, x);
      else
        ld8((const float*)a.v_out + o, nv, x);
    };
    key_cg_tc(a, k, gs, red, tc, rho[0], rho[1], dt == GRKV_BF16 ? 1 : kTP, vget, vget8);
    tc_release(tc);
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
__global__ void __launch_bounds__(kKT) k_alternate_step(KArgs a) {
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
    key_cg_tc(a, k, gs, red, tc, rho[0], rho[1], kTP, vget, vget8);
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

size_t key_ws_bytes(const Shape& s) {
  const size_t U = (size_t)s.U, m = (size_t)s.m, B = (size_t)s.B, d = (size_t)kD;
  size_t bytes = U * (3 * m * B * 4 + B * d * 4 + 4 * m * d * 4 + m * m * 4 + B) + 1024;
  if (s.steps > 1) bytes += U * (2 * B * d * 4 + m * m * 4 + m * d * 4 + 4) + 1024;
  return bytes;
}

cudaError_t launch_key_step(const Shape& s, const void* q, const void* k, const void* v,
                            const float* y, const float* scores, const int32_t* idx,
                            void* v_out, void* k_out, char* ws, const WsLayout& L,
                            cudaStream_t st) {
  const size_t U = (size_t)s.U, m = (size_t)s.m, B = (size_t)s.B, d = (size_t)kD;
  char* base = ws + L.key;
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
  a.X = (float*)base;
  a.T = a.X + U * m * B;
  a.dK = a.T + U * m * B;
  a.vec = a.dK + U * B * d;
  a.T2 = a.vec + U * 4 * m * d;
  a.GQ = a.T2 + U * m * B;
  a.fixed = (uint8_t*)(a.GQ + U * m * m);
  if (s.steps > 1) {
    char* alt = (char*)(((uintptr_t)(a.fixed + U * B) + 255) & ~(uintptr_t)255);
    a.Kt = (float*)alt;
    a.Vt = a.Kt + U * B * d;
    a.G = a.Vt + U * B * d;
    a.RZ = a.G + U * m * m;
    a.done = (int*)(a.RZ + U * m * d);
    cudaError_t e = cudaMemsetAsync(a.done, 0, U * sizeof(int), st);
    if (e != cudaSuccess) return e;
  }
  a.use_tc = s.m <= 128;
  const uint32_t dyn = a.use_tc ? kTcSmem : 0;
  cudaError_t e = cudaFuncSetAttribute(k_key_step, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kTcSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_alternate_step, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kTcSmem);
  if (e != cudaSuccess) return e;
  count_launches(1);
  k_key_step<<<s.U, kKT, dyn, st>>>(a);
  e = cudaGetLastError();
  for (int t = 1; t < s.steps && e == cudaSuccess; ++t) {
    a.vt_valid = t > 1;   // V^(1) exists only as written to v_out (rounded)
    count_launches(1);
    k_alternate_step<<<s.U, kKT, dyn, st>>>(a);
    e = cudaGetLastError();
  }
  return e;
}

}  // namespace grkv
