// LinearShift (Eq. 3) for callers that cannot allocate device memory.
//
// ds_linear_shift needs two 32-bit words of device scratch (amax_io): the
// max|x| written by its pre-pass and read by the kernel to prove that 32-bit
// accumulation is exact.  Some callers cannot provide them: code that runs
// where cudaMalloc is not allowed or not wanted (inside a host callback, a
// plugin handed only input/output buffers by its host framework, a real-time
// path that must never enter the allocator).  This file gives them one entry
// point whose scratch lives in a file-scope static device array instead.
#include <mutex>

#include "ds_common.cuh"

namespace {

// Static scratch: 64 words (256 bytes) per device that loads this library,
// held until the process exits.  A call uses words [0, 2).
constexpr int kStaticScratchWords = 64;
constexpr int kWordsPerCall = 2;
static __device__ __align__(256) uint32_t g_static_scratch[kStaticScratchWords];

// The address is cached per device ordinal so that it is right for whichever
// device is current.  The rest of the library still serves one device per
// process (deepshift.h, "Devices"): the grid heuristics read the SM count of
// the first device once, so use this entry point on one device per process.
constexpr int kMaxDevices = 64;
std::mutex g_mutex;
uint32_t* g_scratch_addr[kMaxDevices] = {nullptr};

// Device address of the static array on the current device.  The array's
// name in host code is only a host-side stand-in, so the address is looked up
// once per device (with that device current) and cached.
ds_status static_scratch_address(uint32_t** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return ds::cuda_check(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices)
    return ds::fail(DS_ERR_UNSUPPORTED, "device ordinal %d beyond %d", dev, kMaxDevices);
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return ds::cuda_check(e, "cudaGetSymbolAddress(static scratch)");
    g_scratch_addr[dev] = static_cast<uint32_t*>(p);
  }
  *out = g_scratch_addr[dev];
  return DS_OK;
}

}  // namespace

extern "C" ds_status ds_linear_shift_static_scratch(const int32_t* x, const ds_weights* w,
                                                    const int32_t* bias, int32_t* y, int64_t M,
                                                    int64_t K, int64_t N, uint32_t flags,
                                                    void* stream) {
  ds::clear_error();
  if (flags & (DS_AMAX_IN | DS_AMAX_OUT))
    return ds::fail(DS_ERR_INVALID_ARG,
                    "DS_AMAX_IN / DS_AMAX_OUT need caller scratch: use ds_linear_shift");
  // Every problem size accepted by ds_linear_shift needs the same two words;
  // the guard keeps that true if either constant is ever changed.
  if (kWordsPerCall > kStaticScratchWords)
    return ds::fail(DS_ERR_UNSUPPORTED, "a call needs %d scratch words, the static array holds %d",
                    kWordsPerCall, kStaticScratchWords);
  uint32_t* scratch = nullptr;
  ds_status r = static_scratch_address(&scratch);
  if (r != DS_OK) return r;
  // The pre-pass of ds_linear_shift zeroes scratch[0] before it writes max|x|,
  // so nothing left by an earlier call is read.
  return ds_linear_shift(x, w, bias, y, M, K, N, flags, scratch, stream);
}
