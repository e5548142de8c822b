// wise_full_attn_accumulate_noalloc: the block-mass attention of
// wise_full_attn_accumulate for callers that cannot let the library allocate
// device memory.  Its per-CTA scratch (the log2 partial masses of each query
// row, one row of nKB floats per row of the query tile) lives in a fixed
// array compiled into the library instead of a buffer obtained with
// cudaMalloc.
#include <mutex>

#include "internal.cuh"

// Shared by every call on a device and kept by that device until the process
// exits.  Each call writes every entry it later reads, so nothing has to be
// cleared between calls.
static __device__ __align__(256) float wise_noalloc_scratch[WISE_NOALLOC_SCRATCH_BYTES / sizeof(float)];

namespace wise {

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mutex;
float* g_noalloc_scratch_ptr[kMaxDevices];
}  // namespace

// In host code the array's name only stands for the symbol; the address a
// kernel can use is looked up once per device, with that device current, and
// cached.  The cache is not invalidated: calls must not span a
// cudaDeviceReset of the device (which unloads the module holding the array).
int noalloc_scratch_address(float** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return WISE_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (!g_noalloc_scratch_ptr[dev]) {
    float* ptr = nullptr;
    if (cudaGetSymbolAddress((void**)&ptr, wise_noalloc_scratch) != cudaSuccess || !ptr) return WISE_ERR_CUDA;
    g_noalloc_scratch_ptr[dev] = ptr;
  }
  *out = g_noalloc_scratch_ptr[dev];
  return WISE_OK;
}

}  // namespace wise

extern "C" int wise_full_attn_accumulate_noalloc(const wise_shape_t* shape, const void* Q, const void* K,
                                                 const void* V, void* O, float* blockmass, int step,
                                                 cudaStream_t stream) {
  // The shape, pointers and device are checked exactly as for
  // wise_full_attn_accumulate before the array's address is resolved.
  if (!blockmass) return WISE_ERR_INVALID_ARG;
  return wise::launch_attention(shape, Q, K, V, O, wise::kDenseMass, blockmass, step, nullptr, nullptr, 0, stream,
                                /*fixed_scratch=*/true);
}
