// Kernel-level entry points: the step loop's tensor-core projection GEMM on caller buffers.
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/uad.h"
#include "uad_internal.cuh"

using namespace uad;

namespace {

constexpr int kTileN = 128, kTileK = 64;

// Split-K scratch of uad_linear, allocated by the library on first use on each device and
// grown on demand: fp32 accumulator [M][N] and per-tile arrival counters, both all-zero
// between launches (the last CTA of every tile clears its part).
struct Scratch {
  float* acc = nullptr;
  size_t acc_floats = 0;
  int* counters = nullptr;
  int n_counters = 0;
  int* err = nullptr;
};
std::mutex g_mu;
std::vector<Scratch> g_scratch;

uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x7fffffu)) return (uint16_t)((u >> 16) | 0x40);  // NaN
  const uint32_t lsb = (u >> 16) & 1u;
  return (uint16_t)((u + 0x7fffu + lsb) >> 16);
}

int check_linear_args(const void* x, const void* w, const float* out, int32_t M, int32_t N, int32_t K) {
  if (!x || !w || !out) return UAD_EINVAL;
  if (M < 1 || N < kTileN || N % kTileN || K < kTileK || K % kTileK) return UAD_EINVAL;
  return UAD_OK;
}

}  // namespace

namespace uad {

// Shared by uad_linear and its caller-scratch variants: launch the projection kernel with
// out[M][N] = x[M][K] w^T (+ bias), fp32 output, the given split-K scratch.
int launch_linear(const void* x, const void* w_tiled, const float* bias, float* out, int M, int N, int K,
                  float* acc, int* counters, int* err, cudaStream_t s) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UAD_ECUDA;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  CUtensorMap tm;
  if (encode_act_tmap(&tm, x, K, M)) return UAD_ECUDA;
  TcGemmArgs a;
  a.w_tiled = w_tiled; a.M = M; a.N = N; a.K = K;
  gemm_tc_plan(M, N, K, sms, EPI_STORE, &a);   // the tile selection of the velocity network's projections
  a.epi = EPI_STORE; a.out = out; a.ldo = N; a.out_dtype = F32; a.bias = bias;
  a.acc = acc; a.counters = counters; a.err = err;
  gemm_tc_prepare();
  launch_gemm_tc(&tm, a, s);
  return cudaGetLastError() == cudaSuccess ? UAD_OK : UAD_ECUDA;
}

int linear_tiles(int M, int N) { return (N / kTileN) * ((M + 63) / 64); }

}  // namespace uad

extern "C" {

int uad_tile_weight(const float* w, int32_t K, int32_t N, uint16_t* out) {
  if (!w || !out || N < kTileN || N % kTileN || K < kTileK || K % kTileK) return UAD_EINVAL;
  const int KC = K / kTileK;
  for (int n = 0; n < N; ++n)
    for (int k = 0; k < K; ++k) {
      const int rr = n % kTileN, kk = k % kTileK;
      const size_t tile = (size_t)(n / kTileN) * KC + k / kTileK;
      const int gran = (kk >> 3) ^ (rr & 7);
      out[tile * kTileN * kTileK + rr * kTileK + gran * 8 + (kk & 7)] = f32_to_bf16_rne(w[(size_t)k * N + n]);
    }
  return UAD_OK;
}

int uad_linear(const void* x, const void* w_tiled, const float* bias, float* out, int32_t M, int32_t N,
               int32_t K, void* stream) {
  int rc = check_linear_args(x, w_tiled, out, M, N, K);
  if (rc) return rc;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UAD_ECUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if ((int)g_scratch.size() <= dev) g_scratch.resize(dev + 1);
  Scratch& sc = g_scratch[dev];
  const size_t need = (size_t)((M + 63) / 64) * 64 * N;
  const int tiles = linear_tiles(M, N);
  if (sc.acc_floats < need) {
    if (sc.acc) cudaFree(sc.acc);
    sc.acc = nullptr;
    sc.acc_floats = 0;
    if (cudaMalloc(&sc.acc, need * 4) != cudaSuccess) return UAD_ENOMEM;
    if (cudaMemset(sc.acc, 0, need * 4) != cudaSuccess) return UAD_ECUDA;
    sc.acc_floats = need;
  }
  if (sc.n_counters < tiles) {
    if (sc.counters) cudaFree(sc.counters);
    sc.counters = nullptr;
    sc.n_counters = 0;
    if (cudaMalloc(&sc.counters, (size_t)tiles * 4) != cudaSuccess) return UAD_ENOMEM;
    if (cudaMemset(sc.counters, 0, (size_t)tiles * 4) != cudaSuccess) return UAD_ECUDA;
    sc.n_counters = tiles;
  }
  if (!sc.err) {
    if (cudaMalloc(&sc.err, 4) != cudaSuccess) return UAD_ENOMEM;
    if (cudaMemset(sc.err, 0, 4) != cudaSuccess) return UAD_ECUDA;
  }
  return launch_linear(x, w_tiled, bias, out, M, N, K, sc.acc, sc.counters, sc.err,
                       static_cast<cudaStream_t>(stream));
}

}  // extern "C"
