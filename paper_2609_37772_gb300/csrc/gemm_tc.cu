// Tensor-core projection GEMM for sm_103a: out[m][n] = epi(sum_k X[m][k] * Wt[n][k]).
//
// Swap-AB tiling for few tokens: 128 weight rows form the MMA's M side, 64 tokens its N
// side, so one CTA computes a 128 x 64 fp32 tile in tensor memory (TMEM). Weights are
// pre-tiled at init into 128 x 64 bf16 blocks already in the 128-byte-swizzled K-major
// shared-memory layout, so each block arrives with one 16 KB bulk copy (cp.async.bulk);
// activation tiles come through a 2-D TMA tensor map (cp.async.bulk.tensor) with the same
// swizzle and zero fill past the last row. One thread issues tcgen05.mma, one thread feeds
// the TMA ring, four warps drain TMEM with tcgen05.ld.
//
// Split-K: CTAs sharing an output tile each own a K range; they add their partial tile into
// an fp32 accumulator in L2 (red.global.add) and the last one to arrive (per-tile counter)
// applies the epilogue, then clears the accumulator and counter for the next launch. The
// residual projections instead write each split's tile to a plane of its own (EPI_PARTIAL):
// the norm that follows sums the planes in a fixed order as part of the residual update.
// Every wait is bounded: on timeout the kernel records an error code and winds down.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "uad_internal.cuh"
#include "ptx.cuh"

namespace uad {

using namespace ptx;

namespace {

constexpr int kBM = 128, kBN = 64, kBK = 64;
constexpr int kStageA = kBM * kBK * 2;  // 16 KB
constexpr int kStageB = kBN * kBK * 2;  // 8 KB
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s bound on any wait

__device__ __forceinline__ bool mbar_wait(uint64_t* b, uint32_t parity, int* err, int code) {
  return ptx::mbar_wait(b, parity, err, code, kWaitNs);
}

// Instruction descriptor, kind::f16: bf16 x bf16 -> fp32, both K-major, M = 128, N = 64.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kBN >> 3) << 17) |
                            ((uint32_t)(kBM >> 4) << 24);
__device__ __forceinline__ void mma_bf16(uint32_t d, uint64_t a, uint64_t b, uint32_t accum) {
  ptx::mma_bf16(d, a, b, kIdesc, accum);
}

__device__ __forceinline__ float gelu_tanh_f(float x) {
  const float k0 = 0.7978845608028654f;
  return 0.5f * x * (1.f + tanhf(k0 * (x + 0.044715f * x * x * x)));
}
// The same with the hardware tanh (MUFU), for outputs rounded to bf16 next: its error is far
// below bf16's.
__device__ __forceinline__ float gelu_tanh_fast(float x) {
  const float k0 = 0.7978845608028654f;
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(k0 * (x + 0.044715f * x * x * x)));
  return 0.5f * x * (1.f + t);
}

__device__ __forceinline__ void store_out(void* out, long long i, float v, int dt) {
  if (dt == BF16) static_cast<__nv_bfloat16*>(out)[i] = __float2bfloat16_rn(v);
  else static_cast<float*>(out)[i] = v;
}


// Shared-memory plan: [pipeline stages, at least 32 KB (reused as the split-K staging tile)]
// [mbarriers, TMEM slot, flag].
__host__ __device__ __forceinline__ int tc_stages(int nch, int epi) {
  (void)epi;
  return nch < kTcMaxStages ? nch : kTcMaxStages;
}
__host__ __device__ __forceinline__ size_t tc_pipe_bytes(int stages) {
  const size_t b = (size_t)stages * (kStageA + kStageB);
  return b < 32768 ? 32768 : b;
}


// Epilogue of one tile slice: T[j][row] holds the fp32 accumulator of token m0 + j (j < mcount)
// for output row n = this thread's row; `plane` is the K split (partial epilogue). Small rolled
// loops keep the code compact.
__device__ __forceinline__ void tile_epilogue(const TcGemmArgs& p, const float* T, int plane, int m0, int mcount,
                                              int n, int row, int lane) {
  const float b = p.bias ? p.bias[n] : 0.f;
  const float* Tr = T + row;
  switch (p.epi) {
    case EPI_PARTIAL: {
      // this split's fp32 partial tile into its own plane [split][M][N]; the consumer sums
      float* dst = static_cast<float*>(p.out) + (size_t)plane * p.M * p.N;
#pragma unroll 4
      for (int j = 0; j < mcount; ++j) dst[(size_t)(m0 + j) * p.N + n] = Tr[j * kBM];
      break;
    }
    case EPI_GEGLU: {
      // rows 2i (gate) and 2i + 1 (up) give output i: tokens over the warps, lane owns rows
      // 4 lane .. 4 lane + 3 (outputs 2 lane, 2 lane + 1 of the tile), so that a warp writes one
      // token's 64 outputs as one contiguous run
      const int o0 = (n - row) / 2 + 2 * lane;
      const bool fast = p.out_dtype == BF16;
      for (int j = row >> 5; j < mcount; j += kBM / 32) {
        const float4 v = *reinterpret_cast<const float4*>(T + j * kBM + 4 * lane);
        const size_t off = (size_t)(m0 + j) * p.ldo + o0;
        if (fast) {
          *reinterpret_cast<__nv_bfloat162*>(static_cast<__nv_bfloat16*>(p.out) + off) =
              __floats2bfloat162_rn(gelu_tanh_fast(v.x) * v.y, gelu_tanh_fast(v.z) * v.w);
        } else {
          store_out(p.out, off, gelu_tanh_f(v.x) * v.y, p.out_dtype);
          store_out(p.out, off + 1, gelu_tanh_f(v.z) * v.w, p.out_dtype);
        }
      }
      break;
    }
    case EPI_BIAS_GELU:
#pragma unroll 4
      for (int j = 0; j < mcount; ++j)
        store_out(p.out, (size_t)(m0 + j) * p.ldo + n, gelu_tanh_f(Tr[j * kBM] + b), p.out_dtype);
      break;
    case EPI_QKV_TC: {
      const QkvTcOut& o = p.qkv;
      const int n0 = n - row;   // the tile's first output row; q, k and v each span whole tiles
      if (n0 < o.qd + o.kvd) {
        // q or k rows: tokens over the warps, lane owns 4 consecutive rows (two RoPE pairs, with
        // rows 2j, 2j + 1 of a head holding dims j and j + dh/2), so that each token's features
        // go out as contiguous runs; (cos, sin) of the token's position from the table
        const bool isq = n0 < o.qd;
        const int sn = (isq ? n0 : n0 - o.qd) + 4 * lane;
        const int h = sn / o.dh, r = sn % o.dh, half = o.dh / 2;
        __nv_bfloat16* base = isq ? o.q + ((size_t)(h / o.G) * o.G + (h % o.G)) * o.H * o.dh
                                  : o.kcache + (((size_t)o.layer * o.Hkv + h) * o.NK + o.P) * o.dh;
        const size_t sb = isq ? (size_t)o.Hkv * o.G * o.H * o.dh : (size_t)o.L * o.Hkv * o.NK * o.dh;
        for (int j = row >> 5; j < mcount; j += kBM / 32) {
          const int m = m0 + j, bi = m / o.H, ii = m - bi * o.H;
          const float4 v = *reinterpret_cast<const float4*>(T + j * kBM + 4 * lane);
          __nv_bfloat16* dst = base + bi * sb + (size_t)ii * o.dh;
          if (o.rope) {
            const float4 cs = *reinterpret_cast<const float4*>(o.rope + (size_t)ii * o.dh + r);
            const int d = r >> 1;
            *reinterpret_cast<__nv_bfloat162*>(dst + d) =
                __floats2bfloat162_rn(v.x * cs.x - v.y * cs.y, v.z * cs.z - v.w * cs.w);
            *reinterpret_cast<__nv_bfloat162*>(dst + d + half) =
                __floats2bfloat162_rn(v.y * cs.x + v.x * cs.y, v.w * cs.z + v.z * cs.w);
          } else {
            *reinterpret_cast<__nv_bfloat162*>(dst + r) = __floats2bfloat162_rn(v.x, v.y);
            *reinterpret_cast<__nv_bfloat162*>(dst + r + 2) = __floats2bfloat162_rn(v.z, v.w);
          }
        }
      } else {
        // v rows: lane owns a token and reads 4 head dims of it at once; each store instruction
        // then writes 32 consecutive keys of one head dim of Vt (keys contiguous)
        const int sv0 = n0 - o.qd - o.kvd;   // the tile's first v feature
        const size_t sb = (size_t)o.L * o.Hkv * o.dh * o.NKp;
        for (int it = row >> 5; it < (kBM / 4) * 2; it += kBM / 32) {
          const int r4 = 4 * (it >> 1), j = 32 * (it & 1) + lane;
          if (j >= mcount) continue;
          const int m = m0 + j, bi = m / o.H, ii = m - bi * o.H;
          const float4 v = *reinterpret_cast<const float4*>(T + j * kBM + r4);
          const int sn = sv0 + r4, g = sn / o.dh, d = sn % o.dh;   // 4 dims of one head
          __nv_bfloat16* dst = o.vtcache + bi * sb + (((size_t)o.layer * o.Hkv + g) * o.dh + d) * o.NKp + o.P + ii;
          dst[0] = __float2bfloat16_rn(v.x);
          dst[o.NKp] = __float2bfloat16_rn(v.y);
          dst[2 * (size_t)o.NKp] = __float2bfloat16_rn(v.z);
          dst[3 * (size_t)o.NKp] = __float2bfloat16_rn(v.w);
        }
      }
      break;
    }
    default:
#pragma unroll 4
      for (int j = 0; j < mcount; ++j)
        store_out(p.out, (size_t)(m0 + j) * p.ldo + n, Tr[j * kBM] + b, p.out_dtype);
      break;
  }
}

// Optional phase timestamps (TcGemmArgs::trace): slot i of this CTA's 16.
#define TC_TRACE(i)                                                                                  \
  do {                                                                                               \
    if (p.trace)                                                                                     \
      p.trace[((size_t)(blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x) * 16 + (i)] = gtime(); \
  } while (0)

__global__ void __launch_bounds__(128, 1) gemm_tc_kernel(const __grid_constant__ CUtensorMap tmx, TcGemmArgs p) {
  extern __shared__ uint8_t smem_raw[];
  if (threadIdx.x == 0) TC_TRACE(0);
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int t = blockIdx.x, mt = blockIdx.y, s = blockIdx.z;
  const int KC = p.K / kBK;
  const int c0 = s * KC / p.splits, c1 = (s + 1) * KC / p.splits, nch = c1 - c0;
  const int stages = tc_stages(nch, p.epi);
  const bool partial = p.epi == EPI_PARTIAL;
  uint8_t* sA = smem;
  uint8_t* sB = smem + (size_t)stages * kStageA;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + tc_pipe_bytes(stages));
  uint64_t* empty = full + kTcMaxStages;
  uint64_t* done = empty + kTcMaxStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  int* last_flag = reinterpret_cast<int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = mt * kBN;
  const int mcount = p.M - m0 < kBN ? p.M - m0 : kBN;

  if (threadIdx.x == 0) {
    for (int i = 0; i < stages; ++i) {
      mbar_init(full + i, 1);
      mbar_init(empty + i, 1);
    }
    mbar_init(done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)), "r"(kBN));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (threadIdx.x == 0) TC_TRACE(1);

  pdl_trigger();
  if (threadIdx.x == 0) {
    // ---- producer: weight block (bulk copy) + activation tile (tensor map) per K chunk.
    //      Weights are constant: the first ring's worth is requested before waiting for the
    //      kernel that produces the activations. ----
    const uint64_t pol = policy_evict_first();
    const uint8_t* wt = static_cast<const uint8_t*>(p.w_tiled) + ((size_t)t * KC + c0) * kStageA;
    const int first = nch < stages ? nch : stages;
    for (int i = 0; i < first; ++i) {
      mbar_expect_tx(full + i, kStageA + kStageB);
      bulk_g2s(sA + (size_t)i * kStageA, wt + (size_t)i * kStageA, kStageA, full + i, pol);
    }
    TC_TRACE(2);
    pdl_wait();
    TC_TRACE(3);
    for (int i = 0; i < first; ++i) tma_2d(sB + (size_t)i * kStageB, &tmx, (c0 + i) * kBK, mt * kBN, full + i);
    int issued = first;
    for (int i = first; i < nch; ++i) {
      const int st = i % stages, round = i / stages;
      if (!mbar_wait(empty + st, (round - 1) & 1, p.err, 11)) break;
      mbar_expect_tx(full + st, kStageA + kStageB);
      bulk_g2s(sA + (size_t)st * kStageA, wt + (size_t)i * kStageA, kStageA, full + st, pol);
      tma_2d(sB + (size_t)st * kStageB, &tmx, (c0 + i) * kBK, mt * kBN, full + st);
      ++issued;
    }
    // do not leave copies in flight into shared memory of an exiting CTA
    for (int i = issued - stages > 0 ? issued - stages : 0; i < issued; ++i)
      mbar_wait(full + i % stages, (i / stages) & 1, p.err, 12);
  } else if (threadIdx.x == 32) {
    // ---- MMA issuer ----
    bool ok = true;
    for (int i = 0; i < nch && ok; ++i) {
      const int st = i % stages, round = i / stages;
      ok = mbar_wait(full + st, round & 1, p.err, 13);
      if (!ok) break;
      if (i == 0) TC_TRACE(4);
      tc_fence_after();
      const uint32_t a0 = su32(sA + (size_t)st * kStageA), b0 = su32(sB + (size_t)st * kStageB);
#pragma unroll
      for (int k = 0; k < kBK / 16; ++k)
        mma_bf16(tmem, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), (i > 0 || k > 0) ? 1u : 0u);
      mma_commit(empty + st);
    }
    TC_TRACE(5);
    mma_commit(done);
  }
  __syncwarp();

  // ---- epilogue: TMEM -> registers, one weight row (output feature) per thread ----
  pdl_wait();
  const bool ok = mbar_wait(done, 0, p.err, 14);
  if (threadIdx.x == 64) TC_TRACE(6);
  tc_fence_after();
  const int row = warp * 32 + lane;
  const int n = t * kBM + row;
  float v[kBN];
  __syncwarp();
  tmem_ld64(tmem + ((uint32_t)(warp * 32) << 16), v);
  bool have = ok && nch > 0;
  // Stage the accumulator tile in shared memory, T[token j][row]: the epilogues below are
  // compact loops over it (neighbouring rows -- GeGLU and RoPE partners -- are one column
  // apart), which keeps the kernel's code small.
  float* T = reinterpret_cast<float*>(smem);                         // pipeline region is idle
#pragma unroll
  for (int j = 0; j < kBN; ++j) T[j * kBM + row] = v[j];
  __syncthreads();
  if (threadIdx.x == 0) TC_TRACE(7);
  if (p.splits > 1 && !partial) {
    // add the partial tile into the L2 accumulator with 16-byte reds; the last CTA of the tile
    // reads the sum back (independent 16-byte loads) and clears it for the next launch
    float* acc = p.acc + (size_t)m0 * p.N + t * kBM;
    if (have) {
      for (int idx = threadIdx.x; idx < mcount * (kBM / 4); idx += 128) {
        const int j = idx / (kBM / 4), c4 = idx % (kBM / 4);
        red_add_v4(acc + (size_t)j * p.N + c4 * 4, *reinterpret_cast<const float4*>(T + j * kBM + c4 * 4));
      }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      TC_TRACE(8);
      const int prev = atomicAdd(p.counters + mt * gridDim.x + t, 1);
      *last_flag = prev == p.splits - 1;
      TC_TRACE(9);
    }
    __syncthreads();
    const bool last = *last_flag;
    have = have && last;
    if (last) {
      __threadfence();
      float4 q[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int idx = threadIdx.x + u * 128;
        if (idx < mcount * (kBM / 4))
          q[u] = __ldcg(reinterpret_cast<const float4*>(acc + (size_t)(idx / (kBM / 4)) * p.N + (idx % (kBM / 4)) * 4));
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int idx = threadIdx.x + u * 128;
        if (idx < mcount * (kBM / 4)) {
          const int j = idx / (kBM / 4), c4 = idx % (kBM / 4);
          __stcg(reinterpret_cast<float4*>(acc + (size_t)j * p.N + c4 * 4), make_float4(0.f, 0.f, 0.f, 0.f));
          *reinterpret_cast<float4*>(T + j * kBM + c4 * 4) = q[u];
        }
      }
      if (threadIdx.x == 0) p.counters[mt * gridDim.x + t] = 0;
    }
    __syncthreads();
    if (threadIdx.x == 0 && last) TC_TRACE(10);
  }
  if (partial) {
    // plane s of [splits][M][N]: whole rows of the tile as 16-byte stores
    if (have) {
      float* dst = static_cast<float*>(p.out) + (size_t)s * p.M * p.N + (size_t)m0 * p.N + t * kBM;
      for (int idx = threadIdx.x; idx < mcount * (kBM / 4); idx += 128) {
        const int j = idx / (kBM / 4), c4 = idx % (kBM / 4);
        *reinterpret_cast<float4*>(dst + (size_t)j * p.N + c4 * 4) = *reinterpret_cast<const float4*>(T + j * kBM + c4 * 4);
      }
    }
  } else if (have) {
    tile_epilogue(p, T, s, m0, mcount, n, row, lane);
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) TC_TRACE(11);
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kBN));
}


// TN tokens per tile (MMA N = 128 or 256); STAGES pipeline stages of 16 KB + TN x 128 B; MINB CTAs
// per SM (more than one: one CTA's epilogue overlaps another's main loop, which pays when there
// are at least as many tiles as SMs).
template <int TN, int STAGES, int MINB>
__global__ void __launch_bounds__(128, MINB) gemm_tc_wide_kernel(const __grid_constant__ CUtensorMap tmx, TcGemmArgs p) {
  constexpr int kWN = TN;
  constexpr int kWStages = STAGES;
  constexpr int kWStageB = kWN * kBK * 2;
  constexpr uint32_t kIdescWide = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kWN >> 3) << 17) |
                                  ((uint32_t)(kBM >> 4) << 24);
  static_assert(STAGES * (kStageA + kWStageB) >= kBM * kBN * 4, "the stage area holds the epilogue slice");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const int t = blockIdx.x, mt = blockIdx.y;
  const int KC = p.K / kBK;
  const int stages = KC < kWStages ? KC : kWStages;
  uint8_t* sA = smem;                                        // stages x 16 KB weights
  uint8_t* sB = smem + (size_t)kWStages * kStageA;           // stages x 32 KB activations
  // after the main loop the stage area holds the epilogue slice T (32 KB)
  float* T = reinterpret_cast<float*>(smem);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)kWStages * (kStageA + kWStageB));
  uint64_t* empty = full + kWStages;
  uint64_t* done = empty + kWStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kWStages; ++i) {
      mbar_init(full + i, 1);
      mbar_init(empty + i, 1);
    }
    mbar_init(done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)), "r"(kWN));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  if (threadIdx.x == 0) {
    const uint64_t pol = policy_evict_first();
    const uint8_t* wt = static_cast<const uint8_t*>(p.w_tiled) + (size_t)t * KC * kStageA;
    const int first = stages;
    for (int i = 0; i < first; ++i) {
      mbar_expect_tx(full + i, kStageA + kWStageB);
      bulk_g2s(sA + (size_t)i * kStageA, wt + (size_t)i * kStageA, kStageA, full + i, pol);
    }
    pdl_wait();
    for (int i = 0; i < first; ++i)
      for (int q = 0; q < kWN / kBN; ++q)
        tma_2d(sB + (size_t)i * kWStageB + q * kStageB, &tmx, i * kBK, mt * kWN + q * kBN, full + i);
    int issued = first;
    for (int i = first; i < KC; ++i) {
      const int st = i % stages, round = i / stages;
      if (!mbar_wait(empty + st, (round - 1) & 1, p.err, 31)) break;
      mbar_expect_tx(full + st, kStageA + kWStageB);
      bulk_g2s(sA + (size_t)st * kStageA, wt + (size_t)i * kStageA, kStageA, full + st, pol);
      for (int q = 0; q < kWN / kBN; ++q)
        tma_2d(sB + (size_t)st * kWStageB + q * kStageB, &tmx, i * kBK, mt * kWN + q * kBN, full + st);
      ++issued;
    }
    for (int i = issued - stages > 0 ? issued - stages : 0; i < issued; ++i)
      mbar_wait(full + i % stages, (i / stages) & 1, p.err, 32);
  } else if (threadIdx.x == 32) {
    bool ok = true;
    for (int i = 0; i < KC && ok; ++i) {
      const int st = i % stages, round = i / stages;
      ok = mbar_wait(full + st, round & 1, p.err, 33);
      if (!ok) break;
      tc_fence_after();
      const uint32_t a0 = su32(sA + (size_t)st * kStageA), b0 = su32(sB + (size_t)st * kWStageB);
#pragma unroll
      for (int k = 0; k < kBK / 16; ++k)
        ptx::mma_bf16(tmem, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), kIdescWide, (i > 0 || k > 0) ? 1u : 0u);
      mma_commit(empty + st);
    }
    mma_commit(done);
  }
  __syncwarp();
  pdl_wait();
  const bool ok = mbar_wait(done, 0, p.err, 34);
  tc_fence_after();
  const int row = warp * 32 + lane;
  const int n = t * kBM + row;
  // epilogue in four slices of 64 tokens (TMEM columns [64 q, 64 q + 64))
  for (int q = 0; q < kWN / kBN; ++q) {
    const int m0 = mt * kWN + q * kBN;
    if (m0 >= p.M) break;
    const int mcount = p.M - m0 < kBN ? p.M - m0 : kBN;
    float v[kBN];
    __syncwarp();
    tmem_ld64(tmem + ((uint32_t)(warp * 32) << 16) + q * kBN, v);
#pragma unroll
    for (int j = 0; j < kBN; ++j) T[j * kBM + row] = v[j];
    __syncthreads();
    if (ok) tile_epilogue(p, T, 0, m0, mcount, n, row, lane);
    __syncthreads();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kWN));
}

// ---- weight re-layout into 128 x 64 swizzled blocks --------------------------------------
__global__ void relayout_tiled_kernel(const float* src, int K, int N, __nv_bfloat16* dst, int mult, long long off,
                                      int rope_dh) {
  __shared__ float tt[32][33];
  const int k0 = blockIdx.y * 32, n0 = blockIdx.x * 32;
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int k = k0 + r, n = n0 + threadIdx.x;
    tt[r][threadIdx.x] = (k < K && n < N) ? src[(long long)k * N + n] : 0.f;
  }
  __syncthreads();
  const int KC = K / kBK;
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int n = n0 + r, k = k0 + threadIdx.x;
    if (n >= N || k >= K) continue;
    int nn = n;
    if (rope_dh > 0) {
      const int h = n / rope_dh, d = n % rope_dh, half = rope_dh / 2;
      nn = h * rope_dh + (d < half ? 2 * d : 2 * (d - half) + 1);
    }
    const long long row = (long long)nn * mult + off;
    const long long tile = (row / kBM) * KC + k / kBK;
    const int rr = (int)(row % kBM), kk = k % kBK;
    const int gran = (kk >> 3) ^ (rr & 7);
    dst[tile * (kBM * kBK) + rr * kBK + gran * 8 + (kk & 7)] = __float2bfloat16_rn(tt[threadIdx.x][r]);
  }
}

}  // namespace

static PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

int encode_act_tmap(CUtensorMap* m, const void* base, int K, int rows) {
  auto enc = tmap_encoder();
  if (!enc) return -1;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {kBK, kBN};
  const cuuint32_t es[2] = {1, 1};
  const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

size_t gemm_tc_smem_bytes(int stages, int epi, int M) {
  (void)epi;
  (void)M;
  return 1024 + tc_pipe_bytes(stages) + (2 * kTcMaxStages + 1) * 8 + 16;
}

static size_t gemm_tc_wide_smem_bytes(int tn, int stages) {
  return 1024 + (size_t)stages * (kStageA + (size_t)tn * kBK * 2) + (2 * stages + 2) * 8 + 16;
}

void gemm_tc_prepare() {
  const size_t a = gemm_tc_smem_bytes(kTcMaxStages, EPI_STORE, kBN);
  cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)a);
  cudaFuncSetAttribute(gemm_tc_wide_kernel<256, 4, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemm_tc_wide_smem_bytes(256, 4));
  cudaFuncSetAttribute(gemm_tc_wide_kernel<256, 2, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemm_tc_wide_smem_bytes(256, 2));
  cudaFuncSetAttribute(gemm_tc_wide_kernel<128, 4, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemm_tc_wide_smem_bytes(128, 4));
  cudaFuncSetAttribute(gemm_tc_wide_kernel<128, 3, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemm_tc_wide_smem_bytes(128, 3));
}

// Wide tiles (MMA N = 256 or 128 tokens) run the tensor cores near their rate (N = 64 runs at a
// third of it) and cut L2 re-reads of the weights. Returns 0 (narrow 128 x 64 tiles with K
// splits), or the wide form: 1 = 256 tokens, four stages, one CTA per SM; 2 = 256 tokens, two
// stages, two CTAs per SM (with at least as many tiles as SMs, one CTA's epilogue overlaps the
// other's main loop); 3 = 128 tokens, four stages, one CTA per SM; 4 = 128 tokens, three stages,
// two CTAs per SM. 256-token tiles while they fill 60% of the SMs, else 128-token tiles while
// those fill half of them (measured on the pi0-like projections from 200 to 3200 tokens: with
// fewer than 256 tokens the narrow tiles win).
int gemm_tc_use_wide(int M, int N, int sms) {
  if (M < 256 || N > 8192) return 0;
  const int t256 = (N / kBM) * ((M + 255) / 256), t128 = (N / kBM) * ((M + 127) / 128);
  if (t256 >= sms) return 2;
  if (t256 * 5 >= sms * 3) return 1;
  if (t128 >= sms) return 4;
  if (t128 * 2 >= sms) return 3;
  return 0;
}
int gemm_tc_wide_tokens(int wide) { return wide >= 3 ? 128 : 256; }

// K splits per output tile: one CTA per SM. Partial-plane epilogues (the consumer sums the
// planes) take more splits, up to two CTAs per SM, so that every CTA holds its whole K range in
// flight (one HBM round trip); where the kernel reduces in L2, extra splits cost more than they
// save.
int gemm_tc_splits(int M, int N, int K, int sms, int epi) {
  const int tiles = (N / kBM) * ((M + kBN - 1) / kBN);
  const int KC = K / kBK;
  const int cap = kTcMaxStages;
  int s = sms / tiles;
  if (s < 1) s = 1;
  if (epi == EPI_PARTIAL && (KC + s - 1) / s > cap) {
    const int need = (KC + cap - 1) / cap;
    const int most = 2 * sms / tiles;
    s = need < most ? need : (most > s ? most : s);
  }
  if (s > KC) s = KC;
  return s;
}

void launch_gemm_tc(const CUtensorMap* tmx, const TcGemmArgs& a, cudaStream_t s) {
  if (a.wide) {
    const int tn = gemm_tc_wide_tokens(a.wide);
    const dim3 grid(a.N / kBM, (a.M + tn - 1) / tn);
    switch (a.wide) {
      case 1: launch_k(gemm_tc_wide_kernel<256, 4, 1>, grid, dim3(128), gemm_tc_wide_smem_bytes(256, 4), s, *tmx, a); break;
      case 2: launch_k(gemm_tc_wide_kernel<256, 2, 2>, grid, dim3(128), gemm_tc_wide_smem_bytes(256, 2), s, *tmx, a); break;
      case 3: launch_k(gemm_tc_wide_kernel<128, 4, 1>, grid, dim3(128), gemm_tc_wide_smem_bytes(128, 4), s, *tmx, a); break;
      default: launch_k(gemm_tc_wide_kernel<128, 3, 2>, grid, dim3(128), gemm_tc_wide_smem_bytes(128, 3), s, *tmx, a); break;
    }
    return;
  }
  const int KC = a.K / kBK;
  const int per = (KC + a.splits - 1) / a.splits;
  dim3 grid(a.N / kBM, (a.M + kBN - 1) / kBN, a.splits);
  launch_k(gemm_tc_kernel, grid, dim3(128), gemm_tc_smem_bytes(tc_stages(per, a.epi), a.epi, a.M), s, *tmx, a);
}

void launch_relayout_tiled(const float* src, int K, int N, void* dst, int mult, long long off, int rope_dh,
                           cudaStream_t s) {
  dim3 grid((N + 31) / 32, (K + 31) / 32);
  relayout_tiled_kernel<<<grid, dim3(32, 8), 0, s>>>(src, K, N, static_cast<__nv_bfloat16*>(dst), mult, off, rope_dh);
}

}  // namespace uad
