// The projection op for callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc once they are running: a real-time robot controller
// that has finished start-up must not block on an allocation (cudaMalloc can take unbounded
// time and synchronize the device, stalling the control loop), and a host framework whose
// caching allocator has already reserved the GPU's memory would see a stray allocation fail
// or fragment its pool. uad_linear_static_scratch serves them: its split-K scratch is a
// fixed array in the library's device image instead of memory allocated at run time.
#include <cstdio>
#include <mutex>

#include "../../include/uad.h"
#include "uad_internal.cuh"

namespace uad {
int launch_linear(const void* x, const void* w_tiled, const float* bias, float* out, int M, int N, int K,
                  float* acc, int* counters, int* err, cudaStream_t s);
int linear_tiles(int M, int N);
}  // namespace uad

namespace {

constexpr size_t kAccFloats = (size_t)UAD_LINEAR_STATIC_MAX_ELEMS;  // fp32 accumulator, M * N values
constexpr size_t kCounters = (size_t)UAD_LINEAR_STATIC_MAX_TILES;   // one arrival counter per tile
constexpr size_t kScratchBytes = kAccFloats * 4 + kCounters * 4 + 256;

// Split-K scratch shared by every call: accumulator, tile counters, then one error word.
// It is part of the library's device image, so every GPU that loads the library holds these
// ~4 MiB until the process exits.
static __device__ __align__(256) unsigned char g_linear_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned char* g_scratch_addr[kMaxDevices] = {};

// Device address of g_linear_scratch on the current device. In host code the array's name
// only stands in for the symbol, so the address is looked up once per device, with that
// device current.
int scratch_on_current_device(unsigned char** base) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UAD_ECUDA;
  if (dev < 0 || dev >= kMaxDevices) return UAD_EINVAL;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_linear_scratch);
    if (e != cudaSuccess) {
      fprintf(stderr, "uad_linear_static_scratch: cudaGetSymbolAddress failed: %s\n", cudaGetErrorString(e));
      return UAD_ECUDA;
    }
    g_scratch_addr[dev] = static_cast<unsigned char*>(p);
  }
  *base = g_scratch_addr[dev];
  return UAD_OK;
}

}  // namespace

extern "C" int uad_linear_static_scratch(const void* x, const void* w_tiled, const float* bias, float* out,
                                         int32_t M, int32_t N, int32_t K, void* stream) {
  if (!x || !w_tiled || !out || M < 1 || N < 128 || N % 128 || K < 64 || K % 64) return UAD_EINVAL;
  const int tiles = uad::linear_tiles(M, N);
  if ((size_t)M * (size_t)N > kAccFloats || (size_t)tiles > kCounters) {
    fprintf(stderr,
            "uad_linear_static_scratch: M*N = %lld exceeds the static scratch (max %d values, %d tiles)\n",
            (long long)M * N, UAD_LINEAR_STATIC_MAX_ELEMS, UAD_LINEAR_STATIC_MAX_TILES);
    return UAD_ETOOBIG;
  }
  unsigned char* base = nullptr;
  const int rc = scratch_on_current_device(&base);
  if (rc) return rc;
  float* acc = reinterpret_cast<float*>(base);
  int* counters = reinterpret_cast<int*>(base + kAccFloats * 4);
  int* err = counters + kCounters;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The array keeps whatever the previous call left; the kernel needs a zero accumulator,
  // zero counters and a clear error word, so clear the part this call uses. Wide tiles (many
  // rows) have no K split and never touch the accumulator or the counters.
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UAD_ECUDA;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const bool split_scratch = uad::gemm_tc_use_wide(M, N, sms) == 0;
  if ((split_scratch && (cudaMemsetAsync(acc, 0, (size_t)M * N * 4, s) != cudaSuccess ||
                         cudaMemsetAsync(counters, 0, (size_t)tiles * 4, s) != cudaSuccess)) ||
      cudaMemsetAsync(err, 0, 4, s) != cudaSuccess)
    return UAD_ECUDA;
  return uad::launch_linear(x, w_tiled, bias, out, M, N, K, acc, counters, err, s);
}
