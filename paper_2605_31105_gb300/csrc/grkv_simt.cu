// Portable CUDA-core kernels of the GRKV compression path.
//
// These run for fp32 inputs, and for bf16 when GRKV_FORCE_SIMT is set.  They
// favour plain, checkable arithmetic over speed: every logit is an fp32 FMA
// chain over the head dimension, probabilities use expf and an IEEE divide,
// and every reduction runs in a fixed order, so results are deterministic.
// The value-step solve accumulates in double for fp32 inputs.
#include <cfloat>
#include <cmath>
#include <type_traits>

#include "block_select.cuh"
#include "grkv_internal.cuh"

namespace grkv {
namespace {

constexpr int QP = kD + 1;  // padded row stride (floats) of q / key tiles in shared memory

// Float count rounded up to a multiple of 4, so the next shared-memory region
// starts on a 16-byte boundary.
__host__ __device__ constexpr int pad4(int n) { return (n + 3) & ~3; }

__device__ __forceinline__ float ldv(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ldv(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void stv(float* p, size_t i, double x) { p[i] = (float)x; }
__device__ __forceinline__ void stv(__nv_bfloat16* p, size_t i, float x) {
  p[i] = __float2bfloat16_rn(x);
}

// Window slot a = r mod w sits at position n - w + a and sees keys j <= n - w + a.
__device__ __forceinline__ bool visible(const Shape& s, int r, int j) {
  return !s.causal || j <= s.n - s.w + (r % s.w);
}

// ---------------------------------------------------------------- pass A --
// Row statistics of one chunk of keys: (max_j l_rj, sum_j exp(l_rj - max)).
template <typename T>
__global__ void __launch_bounds__(256) k_stats_chunk(const T* __restrict__ q,
                                                     const T* __restrict__ k, Shape s, int chunk,
                                                     int nchunk, float2* __restrict__ pstats) {
  extern __shared__ __align__(16) float sm[];
  float* qs = sm;                          // [m][QP], padded to 16 bytes
  float* ks = qs + pad4(s.m * QP);         // [64][kD]
  float2* red = (float2*)(ks + 64 * kD);   // [256], 8-byte aligned
  const int u = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
  const int j0 = c * chunk, j1 = min(s.n, j0 + chunk);
  const T* qu = q + (size_t)u * s.m * kD;
  const T* ku = k + (size_t)u * s.n * kD;
  for (int i = tid; i < s.m * kD; i += blockDim.x) qs[(i / kD) * QP + i % kD] = ldv(qu, i);
  const int tpr = max(1, (int)blockDim.x / s.m);
  const int r = tid / tpr, sub = tid % tpr;
  const bool active = r < s.m;
  float M = -INFINITY, L = 0.f;
  for (int base = j0; base < j1; base += 64) {
    const int len = min(64, j1 - base);
    __syncthreads();
    for (int i = tid; i < len * kD; i += blockDim.x) ks[i] = ldv(ku, (size_t)base * kD + i);
    __syncthreads();
    if (!active) continue;
    for (int jj = sub; jj < len; jj += tpr) {
      const int j = base + jj;
      if (!visible(s, r, j)) continue;
      float acc = 0.f;
#pragma unroll 8
      for (int t = 0; t < kD; ++t) acc = fmaf(qs[r * QP + t], ks[jj * kD + t], acc);
      const float l = s.scale * acc;
      if (l > M) {
        L = L * expf(M - l) + 1.f;
        M = l;
      } else {
        L += expf(l - M);
      }
    }
  }
  red[tid] = make_float2(M, L);
  __syncthreads();
  if (active && sub == 0) {
    float Mr = -INFINITY, Lr = 0.f;
    for (int t = 0; t < tpr; ++t) {
      const float2 pr = red[r * tpr + t];
      if (pr.x == -INFINITY) continue;
      if (pr.x > Mr) {
        Lr = Lr * expf(Mr - pr.x) + pr.y;
        Mr = pr.x;
      } else {
        Lr += pr.y * expf(pr.x - Mr);
      }
    }
    pstats[((size_t)u * nchunk + c) * s.m + r] = make_float2(Mr, Lr);
  }
}

__global__ void k_stats_reduce(const float2* __restrict__ pstats, Shape s, int nchunk,
                               float* __restrict__ row_stats) {
  const int u = blockIdx.x;
  for (int r = threadIdx.x; r < s.m; r += blockDim.x) {
    float M = -INFINITY, L = 0.f;
    for (int c = 0; c < nchunk; ++c) {
      const float2 pr = pstats[((size_t)u * nchunk + c) * s.m + r];
      if (pr.x == -INFINITY) continue;
      if (pr.x > M) {
        L = L * expf(M - pr.x) + pr.y;
        M = pr.x;
      } else {
        L += pr.y * expf(pr.x - M);
      }
    }
    row_stats[((size_t)u * s.m + r) * 2 + 0] = M;
    row_stats[((size_t)u * s.m + r) * 2 + 1] = L;
  }
}

// ---------------------------------------------------------------- pass B --
// Probabilities of one chunk: prefix scores (column sums over the m rows, in
// row order) and the chunk's share of Y = P V.
template <typename T, int RPT>
__global__ void __launch_bounds__(512) k_prob_chunk(const T* __restrict__ q,
                                                    const T* __restrict__ k,
                                                    const T* __restrict__ v, Shape s, int chunk,
                                                    int nchunk, const float* __restrict__ row_stats,
                                                    float* __restrict__ scores,
                                                    float* __restrict__ ypart) {
  extern __shared__ __align__(16) float sm[];
  float* qs = sm;                 // [m][QP]
  float* ks = qs + s.m * QP;      // [32][QP]
  float* vs = ks + 32 * QP;       // [32][kD]
  float* ps = vs + 32 * kD;       // [m][33]
  float* st = ps + s.m * 33;      // [m][2]  (M_r, L_r)
  const int u = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
  const int j0 = c * chunk, j1 = min(s.n, j0 + chunk);
  const T* qu = q + (size_t)u * s.m * kD;
  const T* ku = k + (size_t)u * s.n * kD;
  const T* vu = v + (size_t)u * s.n * kD;
  for (int i = tid; i < s.m * kD; i += blockDim.x) qs[(i / kD) * QP + i % kD] = ldv(qu, i);
  for (int i = tid; i < s.m * 2; i += blockDim.x) st[i] = row_stats[(size_t)u * s.m * 2 + i];
  const int e = tid & (kD - 1), rq = tid >> 7;  // 4 row phases of 128 columns
  float acc[RPT];
#pragma unroll
  for (int i = 0; i < RPT; ++i) acc[i] = 0.f;
  for (int base = j0; base < j1; base += 32) {
    const int len = min(32, j1 - base);
    __syncthreads();
    for (int i = tid; i < 32 * kD; i += blockDim.x) {
      const int jj = i / kD, t = i % kD;
      const bool in = jj < len;
      ks[jj * QP + t] = in ? ldv(ku, (size_t)(base + jj) * kD + t) : 0.f;
      vs[i] = in ? ldv(vu, (size_t)(base + jj) * kD + t) : 0.f;
    }
    __syncthreads();
    for (int pr = tid; pr < s.m * 32; pr += blockDim.x) {
      const int r = pr >> 5, jj = pr & 31, j = base + jj;
      float p = 0.f;
      if (jj < len && visible(s, r, j)) {
        float a = 0.f;
#pragma unroll 8
        for (int t = 0; t < kD; ++t) a = fmaf(qs[r * QP + t], ks[jj * QP + t], a);
        p = expf(s.scale * a - st[2 * r]) / st[2 * r + 1];
      }
      ps[r * 33 + jj] = p;
    }
    __syncthreads();
    if (tid < len && base + tid < s.P) {
      float cs = 0.f;
      for (int r = 0; r < s.m; ++r) cs += ps[r * 33 + tid];
      scores[(size_t)u * s.P + base + tid] = cs;
    }
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      const int r = rq + 4 * i;
      if (r < s.m) {
        float a = acc[i];
        for (int jj = 0; jj < 32; ++jj) a = fmaf(ps[r * 33 + jj], vs[jj * kD + e], a);
        acc[i] = a;
      }
    }
  }
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const int r = rq + 4 * i;
    if (r < s.m) ypart[(((size_t)u * nchunk + c) * s.m + r) * kD + e] = acc[i];
  }
}

__global__ void k_y_reduce(const float* __restrict__ ypart, Shape s, int nchunk,
                           float* __restrict__ y) {
  const int u = blockIdx.x;
  const size_t md = (size_t)s.m * kD;
  for (size_t i = threadIdx.x; i < md; i += blockDim.x) {
    float a = 0.f;
    for (int c = 0; c < nchunk; ++c) a += ypart[((size_t)u * nchunk + c) * md + i];
    y[(size_t)u * md + i] = a;
  }
}

// ------------------------------------------------------------- selection --
__global__ void __launch_bounds__(1024) k_select(const float* __restrict__ scores, Shape s,
                                                 float* __restrict__ pooled,
                                                 int32_t* __restrict__ idx) {
  __shared__ int hist[256];
  __shared__ int sh[48];
  const int u = blockIdx.x, tid = threadIdx.x, P = s.P, h = s.pool_k / 2;
  const float* c = scores + (size_t)u * P;
  float* pl = pooled + (size_t)u * P;
  int32_t* out = idx + (size_t)u * s.B;
  // four positions per step, the neighbour offset outermost, so that each
  // step's loads are independent of one another
  for (int j0 = tid; j0 < P; j0 += 4 * blockDim.x) {
    int j[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) j[q] = j0 + q * blockDim.x;
    if (s.pool_type == GRKV_POOL_MAX) {
      float mx[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) mx[q] = j[q] < P ? c[j[q]] : 0.f;
      for (int t = 1; t <= h; ++t) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (j[q] >= P) continue;
          if (j[q] - t >= 0) mx[q] = fmaxf(mx[q], c[j[q] - t]);
          if (j[q] + t < P) mx[q] = fmaxf(mx[q], c[j[q] + t]);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (j[q] < P) pl[j[q]] = mx[q];
    } else {
      double a[4] = {0.0, 0.0, 0.0, 0.0};   // left to right, zero padding, divisor k
      for (int t = -h; t <= h; ++t) {
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (j[q] < P && j[q] + t >= 0 && j[q] + t < P) a[q] += (double)c[j[q] + t];
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
        if (j[q] < P) pl[j[q]] = (float)(a[q] / (double)s.pool_k);
    }
  }
  __syncthreads();
  if (s.kk >= P) {
    for (int j = tid; j < P; j += blockDim.x) out[j] = j;
  } else if (s.kk > 0) {
    auto get = [&](int i, uint32_t* key) {
      *key = order_key(pl[i]);
      return true;
    };
    // positions: count the marks of earlier segments first
    const int seg = (P + blockDim.x - 1) / blockDim.x;
    const int lo = min(P, tid * seg), hi = min(P, lo + seg);
    uint32_t tau;
    int need_eq;
    block_kth_largest(get, P, s.kk, hist, sh, &tau, &need_eq);
    // the segment's keys in chunks of eight loaded together
    auto seg_keys = [&](int i0, uint32_t* kk) {
#pragma unroll
      for (int q = 0; q < 8; ++q) kk[q] = i0 + q < hi ? order_key(pl[i0 + q]) : 0u;
    };
    int eq = 0;
    for (int i0 = lo; i0 < hi; i0 += 8) {
      uint32_t kk[8];
      seg_keys(i0, kk);
#pragma unroll
      for (int q = 0; q < 8; ++q) eq += (i0 + q < hi && kk[q] == tau);
    }
    int tot;
    const int er0 = block_exclusive_scan(eq, sh + 8, &tot);
    int sel = 0, er = er0;
    for (int i0 = lo; i0 < hi; i0 += 8) {
      uint32_t kk[8];
      seg_keys(i0, kk);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (i0 + q >= hi) continue;
        if (kk[q] > tau) {
          ++sel;
        } else if (kk[q] == tau) {
          if (er < need_eq) ++sel;
          ++er;
        }
      }
    }
    int pos = block_exclusive_scan(sel, sh + 8, &tot);
    er = er0;
    for (int i0 = lo; i0 < hi; i0 += 8) {
      uint32_t kk[8];
      seg_keys(i0, kk);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (i0 + q >= hi) continue;
        if (kk[q] > tau) {
          out[pos++] = i0 + q;
        } else if (kk[q] == tau) {
          if (er < need_eq) out[pos++] = i0 + q;
          ++er;
        }
      }
    }
  }
  for (int a = tid; a < s.w; a += blockDim.x) out[s.kk + a] = P + a;
}

// Selection with the unit's keys resident in shared memory (n - w <= 32768):
// one 1024-thread CTA per unit.  The scores are staged once; thread t owns the
// 32 contiguous positions 32t .. 32t+31 and pools them into order-preserving
// keys held in its registers (max pooling of width 7 as a sliding window over
// the 38 scores around the segment); the (B - w)-th largest key is found by
// four 8-bit radix passes over per-warp histograms, and the positions are
// compacted in order from the same segments.  Same result as k_select.
// Shared-memory words are padded by one per 32 (index j + j / 32) so that
// both the strided staging and the segment reads are free of bank conflicts.
constexpr int kSelThreads = 1024, kSelPer = 32, kSelMaxP = kSelThreads * kSelPer;

__host__ __device__ __forceinline__ int sel_pad(int j) { return j + (j >> 5); }

size_t select_smem_bytes(int P) {
  return ((size_t)sel_pad(P) + 4) * 4 + (size_t)32 * 256 * 4;
}

__global__ void __launch_bounds__(kSelThreads, 1) k_select_smem(const float* __restrict__ scores,
                                                                Shape s,
                                                                int32_t* __restrict__ idx) {
  extern __shared__ uint32_t skey[];   // [sel_pad(P)] scores, then keys
  __shared__ int hist[256];
  __shared__ int sh[48];
  const int u = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int P = s.P, h = s.pool_k / 2;
  int* whist = (int*)(skey + ((sel_pad(P) + 4) & ~3));   // [32][256]
  const float* c = scores + (size_t)u * P;
  int32_t* out = idx + (size_t)u * s.B;
#pragma unroll 8
  for (int e = 0; e < kSelPer; ++e) {
    const int j = tid + e * kSelThreads;
    if (j < P) skey[sel_pad(j)] = __float_as_uint(__ldg(c + j));
  }
  __syncthreads();
  auto cs = [&](int j) { return __uint_as_float(skey[sel_pad(j)]); };
  const int lo = tid * kSelPer;   // this thread's segment lo .. lo + 31
  uint32_t kr[kSelPer];
  if (s.pool_type == GRKV_POOL_MAX && h == 3) {
    // w[i] = score at lo - 3 + i (cells outside [0, P) are ignored: -inf);
    // the window max over w[e .. e + 6] from pairs and quadruples
    float w[kSelPer + 6];
#pragma unroll
    for (int i = 0; i < kSelPer + 6; ++i) {
      const int j = lo - 3 + i;
      w[i] = (j >= 0 && j < P) ? cs(j) : -INFINITY;
    }
    float m2[kSelPer + 5], m4[kSelPer + 3];
#pragma unroll
    for (int i = 0; i < kSelPer + 5; ++i) m2[i] = fmaxf(w[i], w[i + 1]);
#pragma unroll
    for (int i = 0; i < kSelPer + 3; ++i) m4[i] = fmaxf(m2[i], m2[i + 2]);
#pragma unroll
    for (int e = 0; e < kSelPer; ++e)
      kr[e] = lo + e < P ? order_key(fmaxf(fmaxf(m4[e], m2[e + 4]), w[e + 6])) : 0u;
  } else {
#pragma unroll
    for (int e = 0; e < kSelPer; ++e) {
      const int j = lo + e;
      kr[e] = 0u;
      if (j < P) {
        float pv;
        if (s.pool_type == GRKV_POOL_MAX) {
          pv = cs(j);
          for (int t = 1; t <= h; ++t) {
            if (j - t >= 0) pv = fmaxf(pv, cs(j - t));
            if (j + t < P) pv = fmaxf(pv, cs(j + t));
          }
        } else {
          double acc = 0.0;   // left to right, zero padding, divisor k
          for (int t = -h; t <= h; ++t)
            if (j + t >= 0 && j + t < P) acc += (double)cs(j + t);
          pv = (float)(acc / (double)s.pool_k);
        }
        kr[e] = order_key(pv);
      }
    }
  }
  if (s.kk >= P) {
    for (int j = tid; j < P; j += kSelThreads) out[j] = j;
  } else if (s.kk > 0) {
    // (kk)-th largest key: four 8-bit digits, most significant first
    uint32_t prefix = 0, mask = 0;
    int rem = s.kk;
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = tid; i < 32 * 256; i += kSelThreads) whist[i] = 0;
      __syncthreads();
#pragma unroll
      for (int e = 0; e < kSelPer; ++e) {
        if (lo + e < P && (kr[e] & mask) == prefix)
          atomicAdd(&whist[warp * 256 + ((kr[e] >> shift) & 255u)], 1);
      }
      __syncthreads();
      if (tid < 256) {
        int a = 0;
#pragma unroll 8
        for (int w = 0; w < 32; ++w) a += whist[w * 256 + tid];
        hist[tid] = a;
      }
      __syncthreads();
      if (warp == 0) {
        // digit search from 255 down: lane l owns bins 8l..8l+7
        int cnt[8], own = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          cnt[q] = hist[8 * lane + q];
          own += cnt[q];
        }
        int suf = own;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_down_sync(0xffffffffu, suf, o);
          if (lane + o < 32) suf += y;
        }
        int above = suf - own, dg = -1, left = 0;
#pragma unroll
        for (int q = 7; q >= 0; --q) {
          if (dg < 0 && (above + cnt[q] >= rem || (lane == 0 && q == 0))) {
            dg = 8 * lane + q;
            left = rem - above;
          }
          above += cnt[q];
        }
        const unsigned found = __ballot_sync(0xffffffffu, dg >= 0);
        const int srcl = 31 - __clz(found);
        const int dsel = __shfl_sync(0xffffffffu, dg, srcl), lsel = __shfl_sync(0xffffffffu, left, srcl);
        if (lane == 0) {
          sh[0] = dsel;
          sh[1] = lsel;
        }
      }
      __syncthreads();
      prefix |= (uint32_t)sh[0] << shift;
      mask |= 255u << shift;
      rem = sh[1];
      __syncthreads();
    }
    const uint32_t tau = prefix;
    const int need_eq = rem;
    // compaction in position order over the same segments
    int eq = 0;
#pragma unroll
    for (int e = 0; e < kSelPer; ++e) eq += (lo + e < P && kr[e] == tau);
    int tot;
    const int er0 = block_exclusive_scan(eq, sh + 8, &tot);
    int sel = 0, er = er0;
#pragma unroll
    for (int e = 0; e < kSelPer; ++e) {
      if (lo + e >= P) continue;
      if (kr[e] > tau) {
        ++sel;
      } else if (kr[e] == tau) {
        if (er < need_eq) ++sel;
        ++er;
      }
    }
    int pos = block_exclusive_scan(sel, sh + 8, &tot);
    er = er0;
#pragma unroll
    for (int e = 0; e < kSelPer; ++e) {
      if (lo + e >= P) continue;
      if (kr[e] > tau) {
        out[pos++] = lo + e;
      } else if (kr[e] == tau) {
        if (er < need_eq) out[pos++] = lo + e;
        ++er;
      }
    }
  }
  for (int a = tid; a < s.w; a += kSelThreads) out[s.kk + a] = P + a;
}

// ------------------------------------------------------------------ merge --
// One CTA per unit.  A is the accumulation type of the regression (double for
// fp32 inputs, float for bf16).  phase 0 runs the whole value step; phase 1
// stops once R and N are in the workspace and phase 2 starts from Z there
// (the fp32 solve between them is k_solve_dense).
template <typename T, typename A>
__global__ void __launch_bounds__(512) k_merge(
    const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
    const float* __restrict__ scores, const float* __restrict__ y, const int32_t* __restrict__ idx,
    T* __restrict__ k_out, T* __restrict__ v_out, Shape s, float* __restrict__ xbuf,
    uint8_t* __restrict__ flags, A* __restrict__ gram, A* __restrict__ rz, int* status,
    int phase) {
  extern __shared__ __align__(16) float sm[];
  __shared__ int hist[256];
  __shared__ int sh[48];
  const int u = blockIdx.x, tid = threadIdx.x, m = s.m, B = s.B;
  const int nthr = blockDim.x;
  float* qs = sm;               // [m][QP]
  float* tile = qs + m * QP;    // [32][QP]
  float* xt = tile + 32 * QP;   // [m][33]
  const int32_t* id = idx + (size_t)u * B;
  // retained position of slot i; an entry outside [0, n) is reported and read as 0
  auto pos = [&](int i) {
    const int j = id[i];
    return (unsigned)j < (unsigned)s.n ? j : 0;
  };
  float* X = xbuf + (size_t)u * m * B;
  uint8_t* F = flags + (size_t)u * B;
  A* N = gram + (size_t)u * m * m;
  A* RZ = rz + (size_t)u * m * kD;
  const T* ku = k + (size_t)u * s.n * kD;
  const T* vu = v + (size_t)u * s.n * kD;
  T* ko = k_out + (size_t)u * B * kD;
  T* vo = v_out + (size_t)u * B * kD;
  const float* yu = y + (size_t)u * m * kD;
  const float* cu = scores + (size_t)u * s.P;
  if (phase == 2 && s.lambda_inf) return;   // phase 1 wrote V_out = V0
  if (phase != 2) {
  for (int i = tid; i < B; i += nthr)
    if ((unsigned)id[i] >= (unsigned)s.n) set_status(status, GRKV_ERR_INVALID_ARG);

  for (int i = tid; i < m * kD; i += nthr)
    qs[(i / kD) * QP + i % kD] = ldv(q + (size_t)u * m * kD, i);
  // K_out = K0 (the key step is not applied)
  for (int i = tid; i < B * kD; i += nthr) ko[i] = ku[(size_t)pos(i / kD) * kD + i % kD];

  // Fixed set: retained sinks, the window, and the n_fix best-scored
  // retained prefix non-sink tokens.
  auto cand = [&](int i) {
    const int j = pos(i);
    return j >= s.n_sink && j < s.P;
  };
  int nc = 0;
  for (int i = tid; i < B; i += nthr) {
    F[i] = cand(i) ? 0 : 1;
    nc += cand(i) ? 1 : 0;
  }
  int ncand;
  (void)block_exclusive_scan(nc, sh + 8, &ncand);
  const int nf = min(s.n_fix, ncand);
  if (nf > 0) {
    auto get = [&](int i, uint32_t* key) {
      if (!cand(i)) return false;
      *key = order_key(cu[pos(i)]);
      return true;
    };
    block_topk_mark(get, [&](int i, int) { F[i] = 1; }, B, nf, hist, sh);
  }
  __syncthreads();

  // Retained logits, then row softmax over the retained keys -> X.
  for (int base = 0; base < B; base += 32) {
    const int len = min(32, B - base);
    __syncthreads();
    for (int i = tid; i < 32 * kD; i += nthr) {
      const int jj = i / kD, t = i % kD;
      tile[jj * QP + t] = jj < len ? ldv(ku, (size_t)pos(base + jj) * kD + t) : 0.f;
    }
    __syncthreads();
    for (int pr = tid; pr < m * 32; pr += nthr) {
      const int r = pr >> 5, jj = pr & 31;
      if (jj >= len) continue;
      const int j = pos(base + jj);
      float l = -INFINITY;
      if (visible(s, r, j)) {
        float a = 0.f;
#pragma unroll 8
        for (int t = 0; t < kD; ++t) a = fmaf(qs[r * QP + t], tile[jj * QP + t], a);
        l = s.scale * a;
      }
      X[(size_t)r * B + base + jj] = l;
    }
  }
  __syncthreads();
  {
    const int lane = tid & 31, wid = tid >> 5, nw = nthr >> 5;
    for (int r = wid; r < m; r += nw) {
      float* xr = X + (size_t)r * B;
      float M = -INFINITY;
      for (int i = lane; i < B; i += 32) M = fmaxf(M, xr[i]);
      for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      float L = 0.f;
      for (int i = lane; i < B; i += 32) L += expf(xr[i] - M);
      for (int o = 16; o; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
      for (int i = lane; i < B; i += 32) xr[i] = expf(xr[i] - M) / L;
    }
  }
  __syncthreads();
  if (s.lambda_inf) {
    for (int i = tid; i < B * kD; i += nthr) vo[i] = vu[(size_t)pos(i / kD) * kD + i % kD];
    return;
  }

  // R = Y - X V0, 16 rows per thread per pass.
  const int e = tid & (kD - 1), rq = tid >> 7, nrq = nthr >> 7;
  constexpr int RPP = 16;
  for (int r0 = 0; r0 < m; r0 += RPP * nrq) {
    A acc[RPP];
#pragma unroll
    for (int i = 0; i < RPP; ++i) acc[i] = 0;
    for (int base = 0; base < B; base += 32) {
      const int len = min(32, B - base);
      __syncthreads();
      for (int i = tid; i < 32 * kD; i += nthr) {
        const int jj = i / kD, t = i % kD;
        tile[jj * QP + t] = jj < len ? ldv(vu, (size_t)pos(base + jj) * kD + t) : 0.f;
      }
      for (int i = tid; i < m * 32; i += nthr) {
        const int r = i >> 5, jj = i & 31;
        xt[r * 33 + jj] = jj < len ? X[(size_t)r * B + base + jj] : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int i = 0; i < RPP; ++i) {
        const int r = r0 + rq + nrq * i;
        if (r < m) {
          A a = acc[i];
          for (int jj = 0; jj < len; ++jj) a += (A)xt[r * 33 + jj] * (A)tile[jj * QP + e];
          acc[i] = a;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < RPP; ++i) {
      const int r = r0 + rq + nrq * i;
      if (r < m) RZ[(size_t)r * kD + e] = (A)yu[(size_t)r * kD + e] - acc[i];
    }
  }

  // Gram of the free columns: N = X_G X_G^T + lambda I, 32 entries per thread per pass.
  constexpr int GPP = 32;
  for (int p0 = 0; p0 < m * m; p0 += GPP * nthr) {
    A g[GPP];
#pragma unroll
    for (int i = 0; i < GPP; ++i) g[i] = 0;
    for (int base = 0; base < B; base += 32) {
      const int len = min(32, B - base);
      __syncthreads();
      for (int i = tid; i < m * 32; i += nthr) {
        const int r = i >> 5, jj = i & 31;
        xt[r * 33 + jj] = (jj < len && !F[base + jj]) ? X[(size_t)r * B + base + jj] : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int i = 0; i < GPP; ++i) {
        const int p = p0 + tid + nthr * i;
        if (p < m * m) {
          const int r1 = p / m, r2 = p % m;
          A a = g[i];
          for (int jj = 0; jj < len; ++jj) a += (A)xt[r1 * 33 + jj] * (A)xt[r2 * 33 + jj];
          g[i] = a;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < GPP; ++i) {
      const int p = p0 + tid + nthr * i;
      if (p < m * m) N[p] = g[i] + ((p / m == p % m) ? (A)s.lambda : (A)0);
    }
  }
  __syncthreads();
  if (phase == 1) return;

  // Cholesky N = L L^T in place (lower triangle), right-looking.
  for (int c = 0; c < m; ++c) {
    if (tid == 0) {
      const A dkk = N[(size_t)c * m + c];
      sh[0] = (dkk > (A)0) ? 0 : 1;
      if (dkk > (A)0) N[(size_t)c * m + c] = sqrt(dkk);
    }
    __syncthreads();
    if (sh[0]) {  // singular dual system: report it and leave V0 in place
      if (tid == 0) set_status(status, GRKV_ERR_NUMERIC);
      for (int i = tid; i < B * kD; i += nthr) vo[i] = vu[(size_t)pos(i / kD) * kD + i % kD];
      return;
    }
    const A piv = N[(size_t)c * m + c];
    for (int i = c + 1 + tid; i < m; i += nthr) N[(size_t)i * m + c] /= piv;
    __syncthreads();
    const int rest = m - c - 1;
    for (int p = tid; p < rest * rest; p += nthr) {
      const int i = c + 1 + p / rest, j = c + 1 + p % rest;
      if (j <= i) N[(size_t)i * m + j] -= N[(size_t)i * m + c] * N[(size_t)j * m + c];
    }
    __syncthreads();
  }
  // Z = N^-1 R: forward then backward substitution, one column per thread.
  if (tid < kD) {
    for (int i = 0; i < m; ++i) {
      A z = RZ[(size_t)i * kD + tid];
      for (int c = 0; c < i; ++c) z -= N[(size_t)i * m + c] * RZ[(size_t)c * kD + tid];
      RZ[(size_t)i * kD + tid] = z / N[(size_t)i * m + i];
    }
    for (int i = m - 1; i >= 0; --i) {
      A z = RZ[(size_t)i * kD + tid];
      for (int c = i + 1; c < m; ++c) z -= N[(size_t)c * m + i] * RZ[(size_t)c * kD + tid];
      RZ[(size_t)i * kD + tid] = z / N[(size_t)i * m + i];
    }
  }
  __syncthreads();

  }   // phase != 2

  // V_out[G] = V0[G] + X_G^T Z, V_out[F] = V0[F].
  for (int base = 0; base < B; base += 32) {
    const int len = min(32, B - base);
    __syncthreads();
    for (int i = tid; i < m * 32; i += nthr) {
      const int r = i >> 5, jj = i & 31;
      xt[r * 33 + jj] = jj < len ? X[(size_t)r * B + base + jj] : 0.f;
    }
    __syncthreads();
    for (int p = tid; p < len * kD; p += nthr) {
      const int jj = p / kD, c = p % kD, i = base + jj;
      const size_t src = (size_t)pos(i) * kD + c;
      if (F[i]) {
        vo[(size_t)i * kD + c] = vu[src];
      } else {
        A a = 0;
        for (int r = 0; r < m; ++r) a += (A)xt[r * 33 + jj] * RZ[(size_t)r * kD + c];
        stv(vo, (size_t)i * kD + c, (A)ldv(vu, src) + a);
      }
    }
  }
}

template <typename T>
cudaError_t score_impl(const Shape& s, const T* q, const T* k, const T* v, float* scores,
                       float* y, float* row_stats, char* ws, const WsLayout& L,
                       cudaStream_t st) {
  float2* pstats = (float2*)(ws + L.pstats);
  float* ypart = (float*)(ws + L.ypart);
  const size_t smA = ((size_t)pad4(s.m * QP) + 64 * kD) * 4 + 256 * sizeof(float2);
  cudaError_t e = cudaFuncSetAttribute(k_stats_chunk<T>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smA);
  if (e != cudaSuccess) return e;
  dim3 grid(L.nchunk, s.U);
  k_stats_chunk<T><<<grid, 256, smA, st>>>(q, k, s, L.chunk, L.nchunk, pstats);
  k_stats_reduce<<<s.U, 256, 0, st>>>(pstats, s, L.nchunk, row_stats);
  const size_t smB = ((size_t)s.m * QP + 32 * QP + 32 * kD + (size_t)s.m * 33 + s.m * 2) * 4;
  auto launchB = [&](auto kern) {
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smB);
    if (err != cudaSuccess) return err;
    kern<<<grid, 512, smB, st>>>(q, k, v, s, L.chunk, L.nchunk, row_stats, scores, ypart);
    return cudaGetLastError();
  };
  const int rpt = (s.m + 3) / 4;
  if (rpt <= 8) e = launchB(k_prob_chunk<T, 8>);
  else if (rpt <= 16) e = launchB(k_prob_chunk<T, 16>);
  else if (rpt <= 32) e = launchB(k_prob_chunk<T, 32>);
  else e = launchB(k_prob_chunk<T, 64>);
  if (e != cudaSuccess) return e;
  k_y_reduce<<<s.U, 512, 0, st>>>(ypart, s, L.nchunk, y);
  count_launches(4);
  return cudaGetLastError();
}

template <typename T, typename A>
cudaError_t merge_impl(const Shape& s, const T* q, const T* k, const T* v, const float* scores,
                       const float* y, const int32_t* idx, T* k_out, T* v_out, char* ws,
                       const WsLayout& L, cudaStream_t st) {
  const size_t sm = ((size_t)s.m * QP + 32 * QP + (size_t)s.m * 33) * 4;
  cudaError_t e = cudaFuncSetAttribute(k_merge<T, A>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sm);
  if (e != cudaSuccess) return e;
  auto run = [&](int phase) {
    k_merge<T, A><<<s.U, 512, sm, st>>>(q, k, v, scores, y, idx, k_out, v_out, s,
                                        (float*)(ws + L.xbuf), (uint8_t*)(ws + L.flags),
                                        (A*)(ws + L.gram), (A*)(ws + L.rz), (int*)(ws + L.status),
                                        phase);
    count_launches(1);
    return cudaGetLastError();
  };
  // fp32 inputs keep the double-precision solve inside the kernel; bf16 inputs
  // take the blocked shared-memory solve between two phases
  if (!std::is_same<A, float>::value) return run(0);
  if ((e = run(1)) != cudaSuccess) return e;
  if (!s.lambda_inf &&
      (e = launch_solve_dense(s.U, s.m, s.m, 0, 0.f, 0, (const float*)(ws + L.gram),
                              (float*)(ws + L.rz), (int*)(ws + L.status), st)) != cudaSuccess)
    return e;
  return run(2);
}

}  // namespace

cudaError_t launch_score_simt(const Shape& s, const void* q, const void* k, const void* v,
                              float* scores, float* y, float* row_stats, char* ws,
                              const WsLayout& L, cudaStream_t st) {
  if (s.dtype == GRKV_F32)
    return score_impl<float>(s, (const float*)q, (const float*)k, (const float*)v, scores, y,
                             row_stats, ws, L, st);
  return score_impl<__nv_bfloat16>(s, (const __nv_bfloat16*)q, (const __nv_bfloat16*)k,
                                   (const __nv_bfloat16*)v, scores, y, row_stats, ws, L, st);
}

bool select_uses_pooled_buffer(const Shape& s) { return s.P > kSelMaxP; }

cudaError_t launch_select_pooled(const Shape& s, const float* scores, int32_t* idx,
                                 float* pooled, cudaStream_t st) {
  if (!select_uses_pooled_buffer(s)) {
    const size_t bytes = select_smem_bytes(s.P);
    cudaError_t e =
        cudaFuncSetAttribute(k_select_smem, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    k_select_smem<<<s.U, kSelThreads, bytes, st>>>(scores, s, idx);
  } else {
    k_select<<<s.U, 1024, 0, st>>>(scores, s, pooled, idx);
  }
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_select(const Shape& s, const float* scores, int32_t* idx, char* ws,
                          const WsLayout& L, cudaStream_t st) {
  return launch_select_pooled(s, scores, idx, (float*)(ws + L.pooled), st);
}

cudaError_t launch_merge_simt(const Shape& s, const void* q, const void* k, const void* v,
                              const float* scores, const float* y, const int32_t* idx,
                              void* k_out, void* v_out, char* ws, const WsLayout& L,
                              cudaStream_t st) {
  if (s.dtype == GRKV_F32)
    return merge_impl<float, double>(s, (const float*)q, (const float*)k, (const float*)v,
                                     scores, y, idx, (float*)k_out, (float*)v_out, ws, L, st);
  return merge_impl<__nv_bfloat16, float>(
      s, (const __nv_bfloat16*)q, (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, scores, y,
      idx, (__nv_bfloat16*)k_out, (__nv_bfloat16*)v_out, ws, L, st);
}

}  // namespace grkv
