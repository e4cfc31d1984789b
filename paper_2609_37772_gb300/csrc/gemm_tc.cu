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
// Many tokens (a batch of robots) take the persistent wide form instead: one CTA per SM walks
// units of up to 256 tokens x 128 weight rows with two tensor-memory accumulators, so that the
// epilogue of one unit overlaps the main loop of the next.
// Every wait is bounded: on timeout the kernel records an error code and winds down.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <array>
#include <cstdlib>
#include <map>

#include "uad_internal.cuh"
#include "ptx.cuh"

namespace uad {

using namespace ptx;

namespace {

constexpr int kBM = 128, kBN = 64, kBK = 64;
constexpr int kStageA = kBM * kBK * 2;  // 16 KB
constexpr int kStageB = kBN * kBK * 2;  // 8 KB
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s bound on any wait
// persistent form: tokens per epilogue slice, epilogue groups (four warps each), staging pitch
// in floats (132: a float4 column read across 8 tokens touches all 32 banks once), threads
constexpr int kPersSlice = 16, kPersGroups = 4, kPersPitch = kBM + 4;
constexpr int kPersThreads = 64 + kPersGroups * 128;

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


// Epilogue of one tile slice: T[j * pitch + row] holds the fp32 accumulator of token m0 + j
// (j < mcount) for output row n = this thread's row (row = 32 w + lane over the four warps w of
// the slice's group). Partial-plane epilogues (EPI_PARTIAL) are written by the kernels themselves
// as whole-row 16-byte stores. Small rolled loops keep the code compact.
__device__ __forceinline__ void tile_epilogue(const TcGemmArgs& p, const float* T, int pitch, int m0,
                                              int mcount, int n, int row, int lane) {
  const float b = p.bias && (p.n_store <= 0 || n < p.n_store) ? p.bias[n] : 0.f;
  const float* Tr = T + row;
  switch (p.epi) {
    case EPI_GEGLU: {
      // rows 2i (gate) and 2i + 1 (up) give output i: tokens over the warps, lane owns rows
      // 4 lane .. 4 lane + 3 (outputs 2 lane, 2 lane + 1 of the tile), so that a warp writes one
      // token's 64 outputs as one contiguous run
      const int o0 = (n - row) / 2 + 2 * lane;
      const bool fast = p.out_dtype == BF16;
      for (int j = row >> 5; j < mcount; j += kBM / 32) {
        const float4 v = *reinterpret_cast<const float4*>(T + j * pitch + 4 * lane);
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
        store_out(p.out, (size_t)(m0 + j) * p.ldo + n, gelu_tanh_f(Tr[j * pitch] + b), p.out_dtype);
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
        // four tokens at a time (a warp's tokens j, j + 4, ...): every (cos, sin) load of the four
        // is issued before the first use, so that the table's L2 round trips overlap
        constexpr int kStep = kBM / 32, kU = 4;
        for (int j0 = row >> 5; j0 < mcount; j0 += kStep * kU) {
          float4 v[kU], cs[kU];
          int ii[kU];
          __nv_bfloat16* dst[kU];
#pragma unroll
          for (int u = 0; u < kU; ++u) {
            const int j = j0 + kStep * u;
            if (j >= mcount) continue;
            const int m = m0 + j, bi = m / o.H;
            ii[u] = m - bi * o.H;
            dst[u] = base + bi * sb + (size_t)ii[u] * o.dh;
            v[u] = *reinterpret_cast<const float4*>(T + j * pitch + 4 * lane);
            if (o.rope) cs[u] = __ldg(reinterpret_cast<const float4*>(o.rope + (size_t)ii[u] * o.dh + r));
          }
#pragma unroll
          for (int u = 0; u < kU; ++u) {
            if (j0 + kStep * u >= mcount) continue;
            if (o.rope) {
              const int d = r >> 1;
              *reinterpret_cast<__nv_bfloat162*>(dst[u] + d) =
                  __floats2bfloat162_rn(v[u].x * cs[u].x - v[u].y * cs[u].y, v[u].z * cs[u].z - v[u].w * cs[u].w);
              *reinterpret_cast<__nv_bfloat162*>(dst[u] + d + half) =
                  __floats2bfloat162_rn(v[u].y * cs[u].x + v[u].x * cs[u].y, v[u].w * cs[u].z + v[u].z * cs[u].w);
            } else {
              *reinterpret_cast<__nv_bfloat162*>(dst[u] + r) = __floats2bfloat162_rn(v[u].x, v[u].y);
              *reinterpret_cast<__nv_bfloat162*>(dst[u] + r + 2) = __floats2bfloat162_rn(v[u].z, v[u].w);
            }
          }
        }
      } else {
        // v rows: item (row quad rq, token j), tokens fastest: a thread reads 4 head dims of one
        // token at once and each store instruction writes consecutive keys of one head dim of Vt
        // (keys contiguous)
        const int sv0 = n0 - o.qd - o.kvd;   // the tile's first v feature
        const size_t sb = (size_t)o.L * o.Hkv * o.dh * o.NKp;
        for (int it = row; it < (kBM / 4) * mcount; it += kBM) {
          const int r4 = 4 * (it / mcount), j = it - (it / mcount) * mcount;
          const int m = m0 + j, bi = m / o.H, ii = m - bi * o.H;
          const float4 v = *reinterpret_cast<const float4*>(T + j * pitch + r4);
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
      if (p.n_store > 0 && n >= p.n_store) break;   // padding rows of a narrow projection
#pragma unroll 4
      for (int j = 0; j < mcount; ++j)
        store_out(p.out, (size_t)(m0 + j) * p.ldo + n, Tr[j * pitch] + b, p.out_dtype);
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
    tile_epilogue(p, T, kBM, m0, mcount, n, row, lane);
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) TC_TRACE(11);
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kBN));
}


// Persistent form for many tokens: one CTA per SM walks the work units u = blockIdx.x,
// blockIdx.x + gridDim.x, ... Unit u is (token tile mt of p.tn <= TN tokens, weight tile nt, K
// split sp) with mt fastest, so the CTAs running side by side share a weight tile in L2. Warp 0
// feeds the ring of STAGES (weights 16 KB + up to TN x 128 B of tokens) without stopping at unit
// boundaries; warp 1 issues the MMAs into one of two TMEM accumulators (2 x TN columns) while
// four groups of four warps (2-5, 6-9, 10-13, 14-17) drain the other one in 16-token slices,
// slice q to group q % 4, each group through a staging slice of its own, so a unit's epilogue
// overlaps the next unit's main loop. A ragged last token tile loads and multiplies only its
// 64-token boxes. K splits (residual projections only) write planes of their own, summed by the
// norm that follows.
template <int TN, int STAGES>
__global__ void __launch_bounds__(kPersThreads, 1) gemm_tc_pers_kernel(const __grid_constant__ CUtensorMap tmx,
                                                                       TcGemmArgs p) {
  constexpr int kStageBw = TN * kBK * 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;                                        // STAGES x 16 KB weights
  uint8_t* sB = smem + (size_t)STAGES * kStageA;             // STAGES x TN x 128 B tokens
  float* T = reinterpret_cast<float*>(smem + (size_t)STAGES * (kStageA + kStageBw));  // groups x 16 x pitch
  uint64_t* full = reinterpret_cast<uint64_t*>(T + kPersGroups * kPersSlice * kPersPitch);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;    // accumulator b complete
  uint64_t* tempty = tfull + 2;        // accumulator b drained (one arrival per epilogue thread)
  uint64_t* done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tn = p.tn;
  const int n_nt = p.N / kBM, n_mt = (p.M + tn - 1) / tn, S = p.splits, KC = p.K / kBK;
  const int per = (KC + S - 1) / S;
  const int units = n_nt * n_mt * S;

  if (threadIdx.x == 0) {
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(full + i, 1);
      mbar_init(empty + i, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull + b, 1);
      mbar_init(tempty + b, kPersGroups * 128);
    }
    mbar_init(done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)), "r"(2 * TN));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ---- producer ----
      pdl_wait();
      int it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        const int mt = u % n_mt, r = u / n_mt, nt = r % n_nt, sp = r / n_nt;
        const int k0 = sp * per, k1 = k0 + per < KC ? k0 + per : KC;
        const int left = p.M - mt * tn;
        const int nb = ((left < tn ? left : tn) + kBN - 1) / kBN;
        const uint8_t* wt = static_cast<const uint8_t*>(p.w_tiled) + (size_t)nt * KC * kStageA;
        for (int kb = k0; kb < k1; ++kb, ++it) {
          const int st = it % STAGES, round = it / STAGES;
          if (round > 0 && !mbar_wait(empty + st, (round - 1) & 1, p.err, 61)) { ok = false; break; }
          mbar_expect_tx(full + st, kStageA + nb * kStageB);
          bulk_g2s_nohint(sA + (size_t)st * kStageA, wt + (size_t)kb * kStageA, kStageA, full + st);
          for (int q = 0; q < nb; ++q)
            tma_2d(sB + (size_t)st * kStageBw + q * kStageB, &tmx, kb * kBK, mt * tn + q * kBN, full + st);
        }
      }
      // do not leave copies in flight into shared memory of an exiting CTA
      for (int i = it - STAGES > 0 ? it - STAGES : 0; i < it; ++i)
        mbar_wait(full + i % STAGES, (i / STAGES) & 1, p.err, 62);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issuer ----
      const uint32_t tmem = *tmem_slot;
      int it = 0, j = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++j) {
        const int mt = u % n_mt, sp = u / n_mt / n_nt;
        const int k0 = sp * per, k1 = k0 + per < KC ? k0 + per : KC;
        const int left = p.M - mt * tn;
        const int nb = ((left < tn ? left : tn) + kBN - 1) / kBN;
        const uint32_t idesc = idesc_m128(nb * kBN);
        const int b = j & 1;
        if (j >= 2 && !mbar_wait(tempty + b, ((j >> 1) - 1) & 1, p.err, 63)) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * TN);
        for (int kb = k0; kb < k1; ++kb, ++it) {
          const int st = it % STAGES, round = it / STAGES;
          if (!mbar_wait(full + st, round & 1, p.err, 64)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = su32(sA + (size_t)st * kStageA), b0 = su32(sB + (size_t)st * kStageBw);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            ptx::mma_bf16(d, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc, (kb > k0 || k > 0) ? 1u : 0u);
          mma_commit(empty + st);
        }
        if (ok) mma_commit(tfull + b);
      }
      mma_commit(done);
      mbar_wait(done, 0, p.err, 65);
    }
  } else {
    // ---- epilogue: group g = warps 2 + 4g .. 5 + 4g takes slices g, g + 4, ...; warp w reads
    //      tensor-memory lanes 32 (w % 4) .. + 31 ----
    const int g = (warp - 2) >> 2;
    const int q4 = warp & 3, row = q4 * 32 + lane;
    float* Tg = T + g * kPersSlice * kPersPitch;
    pdl_wait();
    int j = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++j) {
      const int mt = u % n_mt, r = u / n_mt, nt = r % n_nt, sp = r / n_nt;
      const int left = p.M - mt * tn;
      const int nsl = ((left < tn ? left : tn) + kPersSlice - 1) / kPersSlice;
      const int mylast = g < nsl ? g + kPersGroups * ((nsl - 1 - g) / kPersGroups) : -1;  // this group's last slice
      const int b = j & 1;
      // one decision for the group, so that none of its warps is left alone at a named barrier
      if (!named_and(1 + g, 128, mbar_wait(tfull + b, (j >> 1) & 1, p.err, 66))) break;
      tc_fence_after();
      if (mylast < 0) {
        tc_fence_before();
        mbar_arrive(tempty + b);
      }
      const uint32_t tb = tmem_base_after_wait(tmem_slot) + (uint32_t)(b * TN) + ((uint32_t)(q4 * 32) << 16);
      const int n = nt * kBM + row;
      for (int q = g; q < nsl; q += kPersGroups) {
        const int m0 = mt * tn + q * kPersSlice;
        const int mcount = p.M - m0 < kPersSlice ? p.M - m0 : kPersSlice;
        float v[kPersSlice];
        tmem_ld16(tb + q * kPersSlice, v);
        if (q == mylast) {
          // the group's share of the accumulator is in registers: hand it back
          tc_fence_before();
          mbar_arrive(tempty + b);
        }
        named_sync(1 + g, 128);   // the previous slice's readers are done with Tg
#pragma unroll
        for (int jj = 0; jj < kPersSlice; ++jj) Tg[jj * kPersPitch + row] = v[jj];
        named_sync(1 + g, 128);
        if (p.epi == EPI_PARTIAL) {
          // plane sp of [splits][M][N]: whole rows of the slice as 16-byte stores
          float* dst = static_cast<float*>(p.out) + (size_t)sp * p.M * p.N + (size_t)m0 * p.N + nt * kBM;
          for (int idx = row; idx < mcount * (kBM / 4); idx += 128) {
            const int jr = idx / (kBM / 4), c4 = idx % (kBM / 4);
            *reinterpret_cast<float4*>(dst + (size_t)jr * p.N + c4 * 4) =
                *reinterpret_cast<const float4*>(Tg + jr * kPersPitch + c4 * 4);
          }
        } else {
          tile_epilogue(p, Tg, kPersPitch, m0, mcount, n, row, lane);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(*tmem_slot), "r"(2 * TN));
  }
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

constexpr int kPersStages256 = 4, kPersStages128 = 6;   // 192 KB of ring either way
// tn: the instantiation's tile capacity (256 or 128)
static size_t gemm_tc_pers_smem_bytes(int tn) {
  const int st = tn == 256 ? kPersStages256 : kPersStages128;
  return 1024 + (size_t)st * (kStageA + (size_t)tn * kBK * 2) + (size_t)kPersGroups * kPersSlice * kPersPitch * 4 +
         (2 * st + 5) * 8 + 16;
}

void gemm_tc_prepare() {
  static bool done = false;
  if (done) return;
  done = true;
  cudaFuncSetAttribute(gemm_tc_pers_kernel<256, kPersStages256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)gemm_tc_pers_smem_bytes(256));
  cudaFuncSetAttribute(gemm_tc_pers_kernel<128, kPersStages128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)gemm_tc_pers_smem_bytes(128));
  cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)gemm_tc_smem_bytes(kTcMaxStages, EPI_STORE, kBN));
}

// Wide tiles (MMA N up to 256 tokens) run the tensor cores near their rate (N = 64 runs at a
// third of it) and cut L2 re-reads of the weights: 1 = the persistent wide form, 0 = narrow
// 128 x 64 tiles with K splits. Wide from 512 tokens, or while 256-token tiles fill 60% of the
// SMs or 128-token tiles fill half of them (measured on the pi0-like projections from 200 to 3200
// tokens: with fewer than 256 tokens the narrow tiles win; at 800 tokens the wide form with K
// split planes wins for the 1024-row o and down projections too).
int gemm_tc_use_wide(int M, int N, int sms) {
  if (M < 256 || N > 8192) return 0;
  const int t256 = (N / kBM) * ((M + 255) / 256), t128 = (N / kBM) * ((M + 127) / 128);
  return M >= 512 || t256 * 5 >= sms * 3 || t128 * 2 >= sms ? 1 : 0;
}

// The persistent form's plan: tokens per tile (256, 192 or 128) and, for partial-plane
// epilogues, K splits. Units go to the CTAs round robin; the plan minimises the busiest CTA's
// work, counted in k-blocks of a 256-token tile: a k-block of nb 64-token boxes costs half by
// its MMA time (nb / 4) and half by its bytes ((2 + nb) / 6, weights 16 KB + 8 KB a box), plus
// half a k-block per unit and, per extra plane, the cost of writing and reading it once more.
void gemm_tc_pers_plan(int M, int N, int K, int sms, int epi, int* tn, int* splits) {
  const int KC = K / kBK, n_nt = N / kBM;
  double best = 1e30;
  *tn = 256;
  *splits = 1;
  for (int t = 256; t >= 128; t -= 64) {
    const int n_mt = (M + t - 1) / t;
    const int smax = epi == EPI_PARTIAL ? 8 : 1;
    for (int sp = 1; sp <= smax && sp <= KC; ++sp) {
      const int per = (KC + sp - 1) / sp;
      if ((sp - 1) * per >= KC) continue;
      const int units = n_nt * n_mt * sp;
      const int ctas = units < sms ? units : sms;
      double worst = 0;
      for (int c = 0; c < ctas; ++c) {
        double w = 0;
        for (int u = c; u < units; u += ctas) {
          const int mt = u % n_mt, s = u / n_mt / n_nt;
          const int kb = (s + 1) * per < KC ? per : KC - s * per;
          const int left = M - mt * t;
          const int nb = ((left < t ? left : t) + kBN - 1) / kBN;
          w += kb * (0.5 * nb / 4.0 + 0.5 * (2 + nb) / 6.0) + 0.5;
        }
        worst = w > worst ? w : worst;
      }
      const double plane = 8.0 * M * N / 6.5e12 / 0.3e-6;   // extra plane written and read, in k-blocks
      const double cost = worst + (sp - 1) * plane;
      if (cost < best - 1e-9) {
        best = cost;
        *tn = t;
        *splits = sp;
      }
    }
  }
}

// K splits per output tile: one CTA per SM. Partial-plane epilogues (the consumer sums the
// planes), and any epilogue when all tokens fit one 64-token tile, take more splits, up to two
// CTAs per SM, so that every CTA holds its whole K range in flight (one HBM round trip). Where the
// kernel reduces several token tiles in L2 extra splits cost more than they save (measured:
// pi0-like qkv at 200 tokens 19.6 -> 20.2 us per layer; DiT qkv and MLP up at 16 tokens gain,
// 1.134 -> 1.103 ms per evaluation).
int gemm_tc_splits(int M, int N, int K, int sms, int epi) {
  const int tiles = (N / kBM) * ((M + kBN - 1) / kBN);
  const int KC = K / kBK;
  const int cap = kTcMaxStages;
  int s = sms / tiles;
  if (s < 1) s = 1;
  if ((epi == EPI_PARTIAL || M <= kBN) && (KC + s - 1) / s > cap) {
    const int need = (KC + cap - 1) / cap;
    const int most = 2 * sms / tiles;
    s = need < most ? need : (most > s ? most : s);
  }
  if (s > KC) s = KC;
  return s;
}

void gemm_tc_plan(int M, int N, int K, int sms, int epi, TcGemmArgs* a) {
  a->wide = gemm_tc_use_wide(M, N, sms);
  a->tn = 0;
  a->splits = 1;
  if (a->wide) {
    // the plan search walks every unit: remember its answers
    thread_local std::map<std::array<int, 5>, std::pair<int, int>> memo;
    const std::array<int, 5> key{M, N, K, sms, epi == EPI_PARTIAL};
    auto it = memo.find(key);
    if (it == memo.end()) {
      std::pair<int, int> v;
      gemm_tc_pers_plan(M, N, K, sms, epi, &v.first, &v.second);
      it = memo.emplace(key, v).first;
    }
    a->tn = it->second.first;
    a->splits = it->second.second;
  } else {
    a->splits = gemm_tc_splits(M, N, K, sms, epi);
  }
}

void launch_gemm_tc(const CUtensorMap* tmx, const TcGemmArgs& a, cudaStream_t s) {
  if (a.wide) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int units = (a.N / kBM) * ((a.M + a.tn - 1) / a.tn) * a.splits;
    const dim3 grid(units < sms ? units : sms);
    if (a.tn > 128)
      launch_k(gemm_tc_pers_kernel<256, kPersStages256>, grid, dim3(kPersThreads), gemm_tc_pers_smem_bytes(256), s,
               *tmx, a);
    else
      launch_k(gemm_tc_pers_kernel<128, kPersStages128>, grid, dim3(kPersThreads), gemm_tc_pers_smem_bytes(128), s,
               *tmx, a);
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
