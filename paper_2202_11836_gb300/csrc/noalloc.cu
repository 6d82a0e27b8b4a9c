// Column sum (bias gradient) without any device allocation.
//
// sky_column_sum needs a scratch buffer for its per-CTA partial sums, which
// the caller allocates.  Some callers cannot: code that draws all device
// memory from a fixed pool owned by someone else (a framework's caching
// allocator, a pre-sized arena) must not call cudaMalloc behind the pool's
// back, and code whose hot loop has to run without allocation calls at all
// (allocation can synchronise the device) cannot make one per call.  This
// entry point serves them: its scratch is a file-scope device array that
// exists from the moment the library is loaded on a device until the process
// exits, so nothing is allocated or freed per call.
#include "common.cuh"
#include "rowwise.h"

namespace sky {
namespace {

constexpr size_t kScratchBytes = size_t(1) << 20;  // 1 MiB per device
static __device__ __align__(256) unsigned char g_colsum_scratch[kScratchBytes];

// Device address of the scratch array on the current device.  Host code only
// sees a host-side stand-in under the array's name, so the address is looked
// up with the device current.  The lookup is repeated on every call (it is
// cheap and enqueues nothing): an address cached across calls would dangle
// after a device reset unloads the module.
sky_status scratch_on_current_device(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_colsum_scratch);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(column-sum scratch)");
  *out = p;
  return SKY_OK;
}

}  // namespace
}  // namespace sky

using namespace sky;

extern "C" sky_status sky_column_sum_noalloc(const void* x, int32_t T, int32_t N, sky_dtype dtype,
                                             float* out, void* stream) {
  try {
    SKY_CHECK(x && out, SKY_ERR_INVALID_ARG, "null argument");
    SKY_CHECK(T > 0 && N > 0, SKY_ERR_INVALID_ARG, "bad sizes");
    const size_t need = column_sum_ws(T, N);
    SKY_CHECK(need <= kScratchBytes, SKY_ERR_INVALID_ARG,
              "sky_column_sum_noalloc: T=%d, N=%d needs %zu bytes of scratch, above its fixed "
              "%zu-byte buffer; use sky_column_sum with a caller workspace",
              T, N, need, kScratchBytes);
    void* ws = nullptr;
    const sky_status st = scratch_on_current_device(&ws);
    if (st != SKY_OK) return st;
    // Every partial the reduction reads is written first by the same call,
    // so the buffer needs no clearing.
    return column_sum(x, T, N, dtype, out, ws, kScratchBytes, static_cast<cudaStream_t>(stream));
  } catch (...) {
    set_error("internal error");
    return SKY_ERR_CUDA;
  }
}
