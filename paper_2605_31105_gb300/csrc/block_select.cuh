// Block-wide selection helpers shared by the selection and merge kernels:
// an exclusive scan, a radix k-th-largest over order-preserving uint32 keys,
// and top-k marking in index order (ties to the smaller index).
#pragma once

#include <stdint.h>

namespace grkv {
namespace {

// Exclusive scan over the block (blockDim.x a multiple of 32, <= 1024).
__device__ int block_exclusive_scan(int v, int* sh, int* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[wid] = x;
  __syncthreads();
  if (wid == 0) {
    int t = lane < nw ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    sh[lane] = t;
  }
  __syncthreads();
  const int pre = (wid > 0 ? sh[wid - 1] : 0) + x - v;
  *total = sh[nw - 1];
  __syncthreads();
  return pre;
}

// k-th largest (1 <= k <= #valid) of the keys get(i) -> (valid, key), i < count,
// by four 8-bit radix passes.  Returns the key tau and how many keys equal to
// tau belong to the top k (the rest of the top k is strictly above tau).
template <typename Get>
__device__ void block_kth_largest(Get get, int count, int k, int* hist, int* sh,
                                  uint32_t* tau, int* need_eq) {
  uint32_t prefix = 0, mask = 0;
  int rem = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    // eight keys fetched per step, so that their loads are in flight together
    for (int i0 = threadIdx.x; i0 < count; i0 += 8 * blockDim.x) {
      uint32_t key[8];
      bool ok[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int i = i0 + q * blockDim.x;
        ok[q] = i < count && get(i, &key[q]);
      }
#pragma unroll
      for (int q = 0; q < 8; ++q)
        if (ok[q] && (key[q] & mask) == prefix) atomicAdd(&hist[(key[q] >> shift) & 255u], 1);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // digit search from 255 down: lane l owns bins 8l..8l+7, a suffix sum
      // over the lanes gives each lane the count above its bins
      const int lane = threadIdx.x;
      int c[8], own = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        c[q] = hist[8 * lane + q];
        own += c[q];
      }
      int suf = own;   // inclusive suffix sum over lanes >= lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_down_sync(0xffffffffu, suf, o);
        if (lane + o < 32) suf += y;
      }
      int above = suf - own, dg = -1, left = 0;
#pragma unroll
      for (int q = 7; q >= 0; --q) {
        if (dg < 0 && (above + c[q] >= rem || (lane == 0 && q == 0))) {
          dg = 8 * lane + q;
          left = rem - above;
        }
        above += c[q];
      }
      // the largest digit whose suffix count reaches rem (digit 0 otherwise)
      const unsigned found = __ballot_sync(0xffffffffu, dg >= 0);
      const int src = 31 - __clz(found);
      const int dsel = __shfl_sync(0xffffffffu, dg, src), lsel = __shfl_sync(0xffffffffu, left, src);
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
  *tau = prefix;
  *need_eq = rem;
}

// Marks, in index order, the top-k of the valid keys (ties to the smaller
// index): calls mark(i) for each.  Each thread owns one contiguous segment.
template <typename Get, typename Mark>
__device__ void block_topk_mark(Get get, Mark mark, int count, int k, int* hist, int* sh) {
  uint32_t tau;
  int need_eq;
  block_kth_largest(get, count, k, hist, sh, &tau, &need_eq);
  const int seg = (count + blockDim.x - 1) / blockDim.x;
  const int lo = min(count, (int)threadIdx.x * seg), hi = min(count, lo + seg);
  int eq = 0;
  for (int i = lo; i < hi; ++i) {
    uint32_t key;
    if (get(i, &key) && key == tau) ++eq;
  }
  int tot;
  int er = block_exclusive_scan(eq, sh + 8, &tot);
  int sel = 0;
  for (int i = lo; i < hi; ++i) {
    uint32_t key;
    if (!get(i, &key)) continue;
    if (key > tau) {
      mark(i, sel++);
    } else if (key == tau) {
      if (er < need_eq) mark(i, sel++);
      ++er;
    }
  }
}

}  // namespace
}  // namespace grkv
