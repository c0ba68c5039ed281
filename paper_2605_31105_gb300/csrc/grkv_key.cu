// Key step of Algorithm 1 at t = 0 (Sec. 3.4 "Key step", App. D.2) on CUDA
// cores in fp32, one CTA per unit.
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
// vanishes.  Each product is a small tiled GEMM over the unit's
// m x B, B x d and m x d matrices, staged in the workspace (L2-resident).
//
// V* is read from v_out as written by the value step (rounded to the input
// dtype), K0 from k_out (the value step copies K0 there), and the fixed set is
// recomputed from the prefix scores exactly as the value step defines it.
#include <cmath>

#include "block_select.cuh"
#include "grkv_internal.cuh"

namespace grkv {
namespace {

constexpr int kKT = 256;                  // threads per CTA
constexpr int kTM = 64, kTN = 64, kTK = 16;

struct KArgs {
  int n, w, m, B, P, n_sink, n_fix, causal, dtype, iters;
  float scale, lambda_k, tol;
  const void* q;          // [U][m][d]
  const float* y;         // [U][m][d]
  const float* scores;    // [U][P]
  const int32_t* idx;     // [U][B]
  const void* v_out;      // [U][B][d]  merged values V*
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
template <class FA, class FB, class FS>
__device__ void block_gemm(GemmSmem& g, int M, int N, int K, FA a, FB b, FS store) {
  auto& As = g.As;
  auto& Bs = g.Bs;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  for (int i0 = 0; i0 < M; i0 += kTM)
    for (int j0 = 0; j0 < N; j0 += kTN) {
      float acc[4][4];
#pragma unroll
      for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int u = 0; u < 4; ++u) acc[t][u] = 0.f;
      for (int k0 = 0; k0 < K; k0 += kTK) {
        for (int e = threadIdx.x; e < kTM * kTK; e += kKT) {
          const int ii = e / kTK, kk = e % kTK;
          As[kk][ii] = (i0 + ii < M && k0 + kk < K) ? a(i0 + ii, k0 + kk) : 0.f;
        }
        for (int e = threadIdx.x; e < kTN * kTK; e += kKT) {
          const int jj = e % kTN, kk = e / kTN;
          Bs[kk][jj] = (j0 + jj < N && k0 + kk < K) ? b(k0 + kk, j0 + jj) : 0.f;
        }
        __syncthreads();
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

__global__ void __launch_bounds__(kKT) k_key_step(KArgs a) {
  __shared__ int hist[256], sh[64];
  __shared__ float red[kKT / 32];
  __shared__ GemmSmem gs;
  const int u = blockIdx.x, m = a.m, B = a.B, dt = a.dtype;
  const int32_t* idx = a.idx + (size_t)u * B;
  const void* q = (const char*)a.q + (size_t)u * m * kD * (dt == GRKV_F32 ? 4 : 2);
  const size_t kv_off = (size_t)u * B * kD;
  const float* Y = a.y + (size_t)u * m * kD;
  float* X = a.X + (size_t)u * m * B;
  float* T = a.T + (size_t)u * m * B;
  float* dK = a.dK + kv_off;
  float* T2 = a.T2 + (size_t)u * m * B;
  float* GQ = a.GQ + (size_t)u * m * m;
  float* R = a.vec + (size_t)u * 4 * m * kD;
  float* Pd = R + (size_t)m * kD;
  float* AP = Pd + (size_t)m * kD;
  float* AL = AP + (size_t)m * kD;
  uint8_t* fixed = a.fixed + (size_t)u * B;
  const float s = a.scale;
  auto pos = [&](int i) {
    const int j = idx[i];
    return (unsigned)j < (unsigned)a.n ? j : 0;
  };

  // ---- fixed set: retained sinks, the window, and the n_fix best-scored
  // remaining retained prefix tokens (ties to the smaller position)
  uint32_t* key = (uint32_t*)T;   // scratch, B words
  int nc = 0;
  for (int i = threadIdx.x; i < B; i += kKT) {
    const int j = pos(i);
    const bool cand = j >= a.n_sink && j < a.P;
    key[i] = cand ? max(order_key(a.scores[(size_t)u * a.P + j]), 1u) : 0u;
    fixed[i] = cand ? 0 : 1;
    nc += cand;
  }
  __syncthreads();
  int ncand;
  (void)block_exclusive_scan(nc, sh + 8, &ncand);
  const int nf = min(a.n_fix, ncand);
  if (nf > 0) {
    auto get = [&](int i, uint32_t* k) {
      *k = key[i];
      return *k != 0u;
    };
    auto mark = [&](int i, int) { fixed[i] = 1; };
    block_topk_mark(get, mark, B, nf, hist, sh);
  }
  __syncthreads();

  // ---- X = softmax over the retained keys of s q_r . k_j (causal rule)
  block_gemm(gs,
      m, B, kD, [&](int r, int t) { return ldv(q, (size_t)r * kD + t, dt); },
      [&](int t, int j) { return ldv(a.k_out, kv_off + (size_t)j * kD + t, dt); },
      [&](int r, int j, float v) { X[(size_t)r * B + j] = s * v; });
  {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int r = wid; r < m; r += kKT / 32) {
      float* x = X + (size_t)r * B;
      const int lim = a.causal ? a.n - a.w + r % a.w : a.n - 1;
      float mx = -INFINITY;
      for (int j = lane; j < B; j += 32)
        if (pos(j) <= lim) mx = fmaxf(mx, x[j]);
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      float sum = 0.f;
      for (int j = lane; j < B; j += 32) {
        const float e = pos(j) <= lim ? expf(x[j] - mx) : 0.f;
        x[j] = e;
        sum += e;
      }
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      const float inv = sum > 0.f ? 1.f / sum : 0.f;
      for (int j = lane; j < B; j += 32) x[j] *= inv;
    }
  }
  __syncthreads();

  const int md = m * kD;
  // ---- GQ = s^2 Q Q^T (the Gram of the window queries)
  block_gemm(gs,
      m, m, kD, [&](int r, int t) { return ldv(q, (size_t)r * kD + t, dt); },
      [&](int t, int r2) { return ldv(q, (size_t)r2 * kD + t, dt); },
      [&](int r, int r2, float v) { GQ[(size_t)r * m + r2] = s * s * v; });
  // ---- r = e = Y - X V*, p = r, alpha = 0
  block_gemm(gs,
      m, kD, B, [&](int r, int j) { return X[(size_t)r * B + j]; },
      [&](int j, int t) { return ldv(a.v_out, kv_off + (size_t)j * kD + t, dt); },
      [&](int r, int t, float v) {
        const size_t o = (size_t)r * kD + t;
        const float e = Y[o] - v;
        R[o] = e;
        Pd[o] = e;
        AL[o] = 0.f;
      });
  float rs = 0.f;
  for (int i = threadIdx.x; i < md; i += kKT) rs = fmaf(R[i], R[i], rs);
  rs = block_sum(rs, red);
  const float stop = a.tol * a.tol * rs;

  // dK <- J_G^T W (fixed rows zero)
  auto vjp = [&](const float* W) {
    block_gemm(gs,
        m, B, kD, [&](int r, int t) { return W[(size_t)r * kD + t]; },
        [&](int t, int j) { return ldv(a.v_out, kv_off + (size_t)j * kD + t, dt); },
        [&](int r, int j, float v) { T[(size_t)r * B + j] = v; });
    softmax_jacobian_rows(X, T, m, B);
    block_gemm(gs,
        B, kD, m, [&](int j, int r) { return T[(size_t)r * B + j]; },
        [&](int r, int t) { return ldv(q, (size_t)r * kD + t, dt); },
        [&](int j, int t, float v) { dK[(size_t)j * kD + t] = fixed[j] ? 0.f : s * v; });
  };

  for (int it = 0; it < a.iters; ++it) {
    if (!(rs > stop) || !(rs > 0.f)) break;
    // Ap = J_G (J_G^T p) + lambda p without forming dK: with dS = X o (dA -
    // rowsum(X o dA)), dA = p V*^T, the JVP of dK = s dS^T Q (free rows) is
    // s Q dK^T = (s^2 Q Q^T) dS on the free columns and 0 on the fixed ones.
    block_gemm(gs,
        m, B, kD, [&](int r, int t) { return Pd[(size_t)r * kD + t]; },
        [&](int t, int j) { return ldv(a.v_out, kv_off + (size_t)j * kD + t, dt); },
        [&](int r, int j, float v) { T[(size_t)r * B + j] = v; });
    softmax_jacobian_rows(X, T, m, B);
    block_gemm(gs,
        m, B, m, [&](int r, int r2) { return GQ[(size_t)r * m + r2]; },
        [&](int r2, int j) { return T[(size_t)r2 * B + j]; },
        [&](int r, int j, float v) { T2[(size_t)r * B + j] = fixed[j] ? 0.f : v; });
    softmax_jacobian_rows(X, T2, m, B);
    block_gemm(gs,
        m, kD, B, [&](int r, int j) { return T2[(size_t)r * B + j]; },
        [&](int j, int t) { return ldv(a.v_out, kv_off + (size_t)j * kD + t, dt); },
        [&](int r, int t, float v) {
          const size_t o = (size_t)r * kD + t;
          AP[o] = v + a.lambda_k * Pd[o];
        });
    float pap = 0.f;
    for (int i = threadIdx.x; i < md; i += kKT) pap = fmaf(Pd[i], AP[i], pap);
    pap = block_sum(pap, red);
    if (!(pap > 0.f)) break;   // the direction has vanished
    const float al = rs / pap;
    float rn = 0.f;
    for (int i = threadIdx.x; i < md; i += kKT) {
      AL[i] = fmaf(al, Pd[i], AL[i]);
      const float r = fmaf(-al, AP[i], R[i]);
      R[i] = r;
      rn = fmaf(r, r, rn);
    }
    rn = block_sum(rn, red);
    const float beta = rn / rs;
    for (int i = threadIdx.x; i < md; i += kKT) Pd[i] = fmaf(beta, Pd[i], R[i]);
    rs = rn;
    __syncthreads();
  }

  // ---- K*_G = K0_G + J_G^T alpha; fixed rows keep K0
  vjp(AL);
  for (int i = threadIdx.x; i < B * kD; i += kKT) {
    const int j = i / kD;
    if (fixed[j]) continue;
    const size_t o = kv_off + i;
    const float v = ldv(a.k_out, o, dt) + dK[i];
    if (dt == GRKV_F32)
      ((float*)a.k_out)[o] = v;
    else
      ((__nv_bfloat16*)a.k_out)[o] = __float2bfloat16_rn(v);
  }
}

}  // namespace

size_t key_ws_bytes(const Shape& s) {
  const size_t U = (size_t)s.U, m = (size_t)s.m, B = (size_t)s.B, d = (size_t)kD;
  return U * (3 * m * B * 4 + B * d * 4 + 4 * m * d * 4 + m * m * 4 + B) + 1024;
}

cudaError_t launch_key_step(const Shape& s, const void* q, const float* y, const float* scores,
                            const int32_t* idx, const void* v_out, void* k_out, char* ws,
                            const WsLayout& L, cudaStream_t st) {
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
  a.q = q;
  a.y = y;
  a.scores = scores;
  a.idx = idx;
  a.v_out = v_out;
  a.k_out = k_out;
  a.X = (float*)base;
  a.T = a.X + U * m * B;
  a.dK = a.T + U * m * B;
  a.vec = a.dK + U * B * d;
  a.T2 = a.vec + U * 4 * m * d;
  a.GQ = a.T2 + U * m * B;
  a.fixed = (uint8_t*)(a.GQ + U * m * m);
  count_launches(1);
  k_key_step<<<s.U, kKT, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace grkv
