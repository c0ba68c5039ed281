// grkv_select_noalloc: the selection step (pooling + top-(B-w) + window)
// with its scratch in a fixed device array instead of a caller workspace.
//
// Some callers cannot hand the library device memory for scratch: for
// example a plugin inside an inference engine that owns every byte of device
// memory through its own pool and gives plugins no workspace, or a serving
// loop that forbids cudaMalloc on the request path because it synchronises
// the device and can fail once the pool has taken the free memory.  This
// entry point needs no workspace and allocates nothing: the pooled scores
// live in `g_pooled_scratch` below, which every GPU that loads the library
// holds (16 MiB) until the process exits.
#include <mutex>

#include "grkv_internal.cuh"

namespace {

constexpr size_t kScratchFloats = (size_t)1 << 22;   // 4 Mi floats = 16 MiB

// Pooled prefix scores [U][n-w] of the most recent call on this device.
static __device__ __align__(256) float g_pooled_scratch[kScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device.  The host-side
// name g_pooled_scratch is only a stand-in, so the address is looked up with
// cudaGetSymbolAddress once per device, with that device current, and cached.
int scratch_for_current_device(float** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return GRKV_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return GRKV_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_pooled_scratch) != cudaSuccess || !ptr)
      return GRKV_ERR_CUDA;
    g_scratch_ptr[dev] = (float*)ptr;
  }
  *out = g_scratch_ptr[dev];
  return GRKV_OK;
}

}  // namespace

extern "C" int grkv_select_noalloc(const grkv_params* p, const float* scores, int32_t* idx,
                                   void* stream) {
  grkv::Shape s;
  const int rc = grkv::make_shape(p, &s);
  if (rc != GRKV_OK) return rc;
  // prefixes up to 32768 positions are selected in shared memory and never
  // touch the array, so only longer ones are held to its size
  if (grkv::select_uses_pooled_buffer(s) && (size_t)s.U * (size_t)s.P > kScratchFloats)
    return GRKV_ERR_WORKSPACE_TOO_SMALL;
  if (((size_t)s.U * s.P && !scores) || ((size_t)s.U * s.B && !idx)) return GRKV_ERR_INVALID_ARG;
  if (((uintptr_t)scores & 15u) || ((uintptr_t)idx & 15u)) return GRKV_ERR_MISALIGNED;
  if (s.U == 0) return GRKV_OK;
  float* pooled = nullptr;
  const int src = scratch_for_current_device(&pooled);
  if (src != GRKV_OK) return src;
  return grkv::launch_select_pooled(s, scores, idx, pooled, (cudaStream_t)stream) == cudaSuccess
             ? GRKV_OK
             : GRKV_ERR_CUDA;
}
