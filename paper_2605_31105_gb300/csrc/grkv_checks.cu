// Device-side argument checks of GRKV_CHECKS: every input value finite and
// the idx contract of grkv_merge (each entry in [0, n), ascending, the window
// n-w .. n-1 in the last w slots).  Violations are written to the status word
// (the first error of a call wins); the kernels that follow still run and
// read only in-range rows, and their outputs are then unspecified.
#include <algorithm>

#include "grkv_internal.cuh"

namespace grkv {
namespace {

template <typename T>
__device__ __forceinline__ bool finite_val(T x) {
  return isfinite(static_cast<float>(x));
}

template <typename T>
__global__ void k_check_finite(const T* __restrict__ a, size_t count, int* status) {
  bool bad = false;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
       i += (size_t)gridDim.x * blockDim.x)
    bad |= !finite_val(a[i]);
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0)
    set_status(status, GRKV_ERR_INVALID_ARG);
}

__global__ void k_check_idx(const int32_t* __restrict__ idx, int U, int n, int w, int B,
                            int* status) {
  const size_t total = (size_t)U * B;
  bool bad = false;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const int slot = (int)(i % B);
    const int j = idx[i];
    bad |= (unsigned)j >= (unsigned)n;
    if (slot > 0) bad |= idx[i - 1] >= j;
    if (slot >= B - w) bad |= j != n - w + (slot - (B - w));
  }
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) set_status(status, GRKV_ERR_BOUNDS);
}

int grid_for(size_t count) { return (int)std::min<size_t>((count + 255) / 256, 4096); }

}  // namespace

cudaError_t launch_check_inputs(const Shape& s, const void* q, const void* k, const void* v,
                                int* status, cudaStream_t st) {
  const size_t nq = (size_t)s.U * s.m * kD, nkv = (size_t)s.U * s.n * kD;
  if (s.dtype == GRKV_F32) {
    k_check_finite<<<grid_for(nq), 256, 0, st>>>((const float*)q, nq, status);
    k_check_finite<<<grid_for(nkv), 256, 0, st>>>((const float*)k, nkv, status);
    k_check_finite<<<grid_for(nkv), 256, 0, st>>>((const float*)v, nkv, status);
  } else {
    k_check_finite<<<grid_for(nq), 256, 0, st>>>((const __nv_bfloat16*)q, nq, status);
    k_check_finite<<<grid_for(nkv), 256, 0, st>>>((const __nv_bfloat16*)k, nkv, status);
    k_check_finite<<<grid_for(nkv), 256, 0, st>>>((const __nv_bfloat16*)v, nkv, status);
  }
  count_launches(3);
  return cudaGetLastError();
}

cudaError_t launch_check_idx(const Shape& s, const int32_t* idx, int* status, cudaStream_t st) {
  const size_t total = (size_t)s.U * s.B;
  k_check_idx<<<grid_for(total), 256, 0, st>>>(idx, s.U, s.n, s.w, s.B, status);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace grkv
