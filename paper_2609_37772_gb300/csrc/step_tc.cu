// Persistent evaluation kernel: one velocity evaluation v = F_theta(u, tau) of an adaRMS action
// expert with few tokens in a single launch, one CTA per SM.
//
// With few tokens an evaluation is a chain of dependent steps per layer, each far too small to
// fill the GPU; its cost is the latency of that chain, not the weight bytes. The kernel keeps the
// chain short: every elementwise step is fused into the epilogue of the projection that produces
// its input, and the phases of a layer wait on completion counts rather than grid barriers. One producer thread per CTA streams this CTA's share of
// every projection weight through a shared-memory ring without waiting for the barriers (the
// weights do not depend on the activations).
//
// Factored adaptive RMSNorm. With y = RMSNorm(h) (1 + scale) + shift (per-token modulation of
// the token's flow time), a projection of y splits as
//     y W^T = rstd(h) * ((h (1 + scale)) W^T) + shift W^T,
// so the producer of h writes z = h (1 + scale) (bf16) without waiting for the row norm, and the
// shift vectors of the step's distinct flow times ride along as extra rows of z (rows M..M+S-1).
// The consumer of the projection applies rstd (from row sums of squares accumulated by the
// producers of h) and adds the shift row of the token's flow time.
//
// Phases (the CTAs that add into an output block of a projection count their arrivals on the
// block; each of them then runs the block's epilogue for a share of its rows):
//   in       row m: h = W_in u + b_in, sum h^2, z = h (1 + scale1); shift rows of layer 0
//   qkv      acc += z W_qkv^T;  block epilogue: rstd * acc + shift row, RoPE, q -> Q, k -> K
//            cache, v -> Vt cache
//   attn     items (robot-group, 128 query rows, 64 keys): S = Q K^T, P = exp(S - max),
//            O = P V on tcgen05 -> partial O rows and (max, sum)
//   combine  query rows: log-sum-exp merge of the key chunks -> o (bf16)
//   o        acc += o W_o^T;  block epilogue: h += gate1 * acc, sum h^2, z = h (1 + scale2),
//            shift rows of norm 2
//   gate_up  acc += z W_gu^T;  block epilogue: rstd * acc + shift row, act = gelu_tanh(gate) up
//   down     acc += act W_d^T;  block epilogue: h += gate2 * acc, sum h^2, z for the next
//            layer's norm 1
// then the final norm and the action-out projection v = W_out y + b_out (row m). The epilogue
// that reads an accumulator block clears it, so the next use starts from zero.
//
// Warps: 0-7 = consumers (tensor-memory readout, epilogues, row steps, chunk merges), 8 = weight
// producer (lane 0), 9 = tcgen05 issuer and TMA loads of activations and attention operands (lane 0).
// Every wait is bounded: on timeout the kernel records an error code, skips the remaining
// work, waits (bounded) for its copies in flight and frees its tensor memory.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "uad_internal.cuh"
#include "ptx.cuh"
#include "euler.cuh"

namespace uad {

using namespace ptx;

namespace {

constexpr int kSlot = 16384;         // weight tile: 128 rows x 64 bf16, 128-byte swizzled
constexpr int kATile = 8192;         // activation tile: 64 tokens x 64 bf16
constexpr int kQT = 128, kKC = 64;   // attention: query rows per tile, keys per chunk
constexpr int kConsWarps = 8;                      // consumer warps 0-7
constexpr int kCons = 32 * kConsWarps;              // consumer threads
constexpr int kProdWarp = kConsWarps;               // weight producer (lane 0)
constexpr int kMmaThread = 32 * (kConsWarps + 1);   // tcgen05 issuer and TMA loads (lane 0 of the last warp)
constexpr int kThreads = kMmaThread + 32;
constexpr int kSyncThreads = kCons + 32;            // consumers and the issuer's warp
constexpr int kMaxRows = kStepMaxRows;   // tokens per evaluation (the N side of every MMA)
constexpr int kMaxATiles = kStepMaxATiles;
constexpr int kMaxRing = kStepMaxRing;
constexpr uint32_t kTmemCols = 512;  // projection segments at 64-column steps; attention S at 0, O at 256
constexpr unsigned long long kDrainNs = 200000000ull;   // waiting for own copies before exit

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ float gelu_tanh(float x) {
  const float k0 = 0.7978845608028654f;
  return 0.5f * x * (1.f + tanh_approx(k0 * (x + 0.044715f * x * x * x)));
}

__device__ __forceinline__ void st_bf16x4(__nv_bfloat16* dst, float a, float b, float c, float d) {
  uint2 pk;
  pk.x = pack_bf16(a, b);
  pk.y = pack_bf16(c, d);
  *reinterpret_cast<uint2*>(dst) = pk;
}

// Shared-memory plan (1024-aligned base): [weight ring: ring x 16 KB][work area X][mbarriers,
// TMEM slot, flags, reduction scratch]. X holds, by step, the activation tiles of a projection,
// the staged accumulator tile and the operands of its block epilogue, the attention operands
// Q | K | Vt | P and the staged partial O rows, or the partial rows of a combine.
constexpr size_t kEpiBytes = (size_t)kMaxRows * 512 * 2 + (size_t)3 * kStepMaxShift * 512;
__host__ __device__ constexpr size_t step_x_bytes(int dh) {
  const size_t a = (size_t)kMaxATiles * kATile;
  const size_t att = (size_t)dh * kQT * 2 + 2 * (size_t)dh * kKC * 2 + (size_t)kQT * kKC * 2;
  const size_t ost = (size_t)kQT * (dh * 2 + 16);
  size_t m = a > att ? a : att;
  m = m > ost ? m : ost;
  return m > kEpiBytes ? m : kEpiBytes;
}
constexpr size_t kTailBytes = 512;   // mbarriers (<= 2 * 12 + 8), TMEM slot, flags, scratch

// Projection j of a layer: 0 = qkv, 1 = o, 2 = gate/up, 3 = down.
__device__ __forceinline__ void proj_shape(const StepArgs& __restrict__ p, int j, int& N, int& K) {
  switch (j) {
    case 0: N = p.qkvd; K = p.W; break;
    case 1: N = p.W; K = p.qd; break;
    case 2: N = 2 * p.F; K = p.W; break;
    default: N = p.W; K = p.F; break;
  }
}

// Tiles of this CTA in a projection of NB output blocks x KT k-blocks: the CTAs are split into
// NB contiguous groups (rotated from projection to projection), group b shares block b's KT
// k-blocks. Every CTA's tiles lie in one output block, so each CTA adds one accumulator tile.
struct Tiles {
  int b, k0, k1, contrib;   // output block, k-block range, CTAs that add into block b
  int idx;                  // this CTA's index among them (its share of the block's epilogue)
};
__host__ __device__ __forceinline__ Tiles assign_tiles(int cta, int G, int NB, int KT, int rot) {
  const int v = (cta + rot) % G;
  const int b = v * NB / G;
  const int first = (b * G + NB - 1) / NB, next = ((b + 1) * G + NB - 1) / NB;
  const int cb = next - first, i = v - first;
  Tiles t;
  t.b = b;
  t.k0 = i * KT / cb;
  t.k1 = (i + 1) * KT / cb;
  t.contrib = cb < KT ? cb : KT;
  t.idx = cb <= KT ? i : t.k0;   // with more CTAs than k-blocks, each non-empty range is one k-block
  return t;
}
__host__ __device__ __forceinline__ int proj_rot(int j) { return 41 * j; }
// Epilogue shares of a projection: the sum over output blocks of their contributing CTAs.
__host__ __device__ __forceinline__ int proj_shares(int G, int NB, int KT) {
  int n = 0;
  for (int b = 0; b < NB; ++b) {
    const int cb = ((b + 1) * G + NB - 1) / NB - (b * G + NB - 1) / NB;
    n += cb < KT ? cb : KT;
  }
  return n;
}

struct Smem {
  uint8_t* ring;
  uint8_t* X;
  uint64_t *full, *empty;   // [ring]
  uint64_t *a_full, *g_done, *q_full, *v_full, *s_full, *p_full, *o_done, *fin;
  uint32_t* tmem_slot;
  int* flag;
  int* last;
  float* red;               // [8]
  uint64_t* cbar;           // [kConsWarps] per consumer warp: staging of a combine's partial rows
};

__device__ __forceinline__ Smem smem_plan(int R, size_t xbytes) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  Smem S;
  S.ring = base;
  S.X = base + (size_t)R * kSlot;
  uint64_t* bars = reinterpret_cast<uint64_t*>(S.X + xbytes);
  S.full = bars;
  S.empty = bars + R;
  S.a_full = bars + 2 * R;
  S.g_done = S.a_full + 1;
  S.q_full = S.a_full + 2;
  S.v_full = S.a_full + 3;
  S.s_full = S.a_full + 4;
  S.p_full = S.a_full + 5;
  S.o_done = S.a_full + 6;
  S.fin = S.a_full + 7;
  S.tmem_slot = reinterpret_cast<uint32_t*>(S.a_full + 8);
  S.flag = reinterpret_cast<int*>(S.tmem_slot + 1);
  S.last = S.flag + 1;
  S.red = reinterpret_cast<float*>(S.tmem_slot + 4);
  S.cbar = reinterpret_cast<uint64_t*>(S.red + 8);
  return S;
}

// Per-thread position in the CTA's barrier and ring sequences (issuer and consumers advance
// the same sequences in the same order).
struct Role {
  int slot = 0;                      // weight ring slot and its phase parity
  uint32_t par = 0;
  uint32_t apar = 0, gpar = 0, ipar = 0;   // a_full, g_done, per-attention-item barriers
  int a_uses = 0, i_uses = 0;        // loads issued on a_full and on q_full / v_full
  uint32_t cpar = 0;                 // this consumer warp's combine barrier
  int c_uses = 0;
};

// Step values shared by the CTA's threads: this step's distinct flow times and each token's.
struct StepShared {
  StepArgs p;
  int nsh;                           // distinct flow times (shift rows of z)
  int srow[kStepMaxShift];           // their modulation-table rows
  int sidx[kMaxRows];                // token -> index of its flow time
  uint8_t row_b[kMaxRows];           // token -> its robot (row / H)
  uint8_t row_i[kMaxRows];           // token -> its position in the chunk (row % H)
  Tiles tiles[4];                    // this CTA's tiles of the qkv, o, gate/up, down projections
  int fused_combine;                 // idle CTAs of the attention step merge the key chunks; the
                                     // phases of a layer then wait on counts, not grid barriers
  unsigned shares[4];                // epilogue shares of qkv, o, gate/up; [3] = merging CTAs
};

// A function's working copy of the caller's Role, written back when the function returns (kept in
// registers instead of being read and written through a reference in local memory).
struct RoleCopy {
  Role& ref;
  Role v;
  __device__ __forceinline__ explicit RoleCopy(Role& r) : ref(r), v(r) {}
  __device__ __forceinline__ ~RoleCopy() { ref = v; }
};

// Grid barrier among the consumer warps and the issuer's warp of every CTA: every CTA arrives (also
// after an error, so that no CTA waits for it), then the issuer thread spins on the counter. Returns false once any error is
// recorded, so that the remaining steps are skipped.
__device__ __noinline__ bool grid_sync(unsigned* ctr, bool ok, int* err, const Smem& S, unsigned long long lim,
                                       unsigned extra = 0) {
  tc_fence_before();
  __syncwarp();
  named_sync(1, kSyncThreads);
  if (threadIdx.x == kMmaThread) {
    bool good = ok && *reinterpret_cast<volatile int*>(err) == 0;
    // release arrival: the CTA's writes (ordered before this thread by the named barrier)
    // are visible at GPU scope to whoever observes the count
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
    if (good) {
      const unsigned target = gridDim.x + extra;
      unsigned long long t0 = 0;
      for (uint32_t it = 0;; ++it) {
        if (ld_acquire(ctr) >= target) break;
        if ((it & 63) == 63) {
          if (*reinterpret_cast<volatile int*>(err) != 0) { good = false; break; }
          const unsigned long long t = gtime();
          if (t0 == 0) t0 = t;
          else if (t - t0 > lim) {
            atomicCAS(err, 0, 51);
            good = false;
            break;
          }
        }
      }
    }
    // activations written by other CTAs are read next by this thread's tensor-map loads
    asm volatile("fence.proxy.async.global;" ::: "memory");
    *S.flag = good ? 1 : 0;
  }
  __syncwarp();
  named_sync(1, kSyncThreads);
  tc_fence_after();
  return *reinterpret_cast<volatile int*>(S.flag) != 0;
}

// Bounded wait until *ctr >= target (acquire); false (error 52 recorded) on timeout or once any
// error is recorded.
__device__ __noinline__ int count_wait(const unsigned* ctr, unsigned target, int* err, unsigned long long lim) {
  return ptx::count_wait(ctr, target, err, 52, lim);
}

// Phase boundary inside a layer when the phases wait on counts: the CTA's consumers and issuer
// meet (tensor memory and the work area are free again), the issuer waits until *ctr reaches
// `target` (acquire: the outputs this phase reads), then they meet again, so that every thread's
// loads come after the acquire. Returns false once any error is recorded.
__device__ __noinline__ bool phase_wait(const unsigned* ctr, unsigned target, bool ok, int* err, const Smem& S,
                                        unsigned long long lim) {
  tc_fence_before();
  __syncwarp();
  named_sync(1, kSyncThreads);
  if (threadIdx.x == kMmaThread) {
    bool good = ok && *reinterpret_cast<volatile int*>(err) == 0;
    if (good) good = count_wait(ctr, target, err, lim) != 0;
    // outputs written by other CTAs are read next by this thread's tensor-map loads
    asm volatile("fence.proxy.async.global;" ::: "memory");
    *S.flag = good ? 1 : 0;
  }
  __syncwarp();
  named_sync(1, kSyncThreads);
  tc_fence_after();
  return *reinterpret_cast<volatile int*>(S.flag) != 0;
}

// Sum over the consumer threads; every consumer gets the total.
__device__ __forceinline__ float cons_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = v;
  named_sync(2, kCons);
  float t = 0.f;
#pragma unroll
  for (int i = 0; i < kConsWarps; ++i) t += red[i];
  named_sync(2, kCons);
  return t;
}

__device__ __forceinline__ float* sumsq_slot(const StepArgs& __restrict__ p, int l, int which) {
  return reinterpret_cast<float*>(p.sync + (1 + kStepBarriersPerLayer * p.L) + (size_t)p.L * 4 * kStepMaxNB) +
         (size_t)(2 * l + which) * kMaxRows;
}
// Count of finished key chunks of query tile t (robot-group x 128-row tile) in layer l.
__device__ __forceinline__ unsigned* qtile_ctr(const StepArgs& __restrict__ p, int l, int t) {
  return p.sync + (1 + kStepBarriersPerLayer * p.L) + (size_t)p.L * 4 * kStepMaxNB + (size_t)(p.L + 1) * 2 * kMaxRows +
         (size_t)l * kStepMaxQTiles + t;
}
// Count of finished epilogue shares of projection j (0 qkv, 1 o, 2 gate/up) of layer l; j = 3:
// count of CTAs that finished their chunk merges.
__device__ __forceinline__ unsigned* done_ctr(const StepArgs& __restrict__ p, int l, int j) {
  return p.sync + (1 + kStepBarriersPerLayer * p.L) + (size_t)p.L * 4 * kStepMaxNB + (size_t)(p.L + 1) * 2 * kMaxRows +
         (size_t)p.L * kStepMaxQTiles + (size_t)l * 4 + j;
}
__device__ __forceinline__ const float* mod_row(const StepArgs& __restrict__ p, int row) {
  return p.tab + (size_t)row * p.rowlen;
}

// ---- phase "in": rows of layer 0 ------------------------------------------------------------
// Token row m (CTA m < M): h = W_in u + b_in, the row's sum of squares, z = h (1 + scale1).
// CTA M + j < M + nsh: shift row j of layer 0's first norm.
__device__ __noinline__ void in_rows(const StepShared& __restrict__ sh, float* red) {
  const StepArgs& p = sh.p;
  const int c = blockIdx.x, tid = threadIdx.x, W = p.W;
  if (c < p.M) {
    const float* mod = mod_row(p, p.tau_row[c]);
    const float* u = p.u + (size_t)c * p.D;
    const uint4* wi = static_cast<const uint4*>(p.w_in);
    const int D8 = p.D / 8;
    float ss = 0.f;
#pragma unroll 1
    for (int c4 = tid; c4 < W / 4; c4 += kCons) {
      const float4 b = __ldg(reinterpret_cast<const float4*>(p.b_in) + c4);
      float o[4] = {b.x, b.y, b.z, b.w};
#pragma unroll 1
      for (int k8 = 0; k8 < D8; ++k8) {
        const float4 u0 = __ldg(reinterpret_cast<const float4*>(u) + 2 * k8);
        const float4 u1 = __ldg(reinterpret_cast<const float4*>(u) + 2 * k8 + 1);
        const float uk[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const uint4 wv = __ldg(wi + (size_t)(4 * c4 + r) * D8 + k8);
          const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&wv);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 f = __bfloat1622float2(w2[q]);
            o[r] = fmaf(uk[2 * q], f.x, fmaf(uk[2 * q + 1], f.y, o[r]));
          }
        }
      }
      const float4 x = make_float4(o[0], o[1], o[2], o[3]);
      reinterpret_cast<float4*>(p.h + (size_t)c * W)[c4] = x;
      ss = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, fmaf(x.w, x.w, ss))));
      const float4 s = __ldg(reinterpret_cast<const float4*>(mod) + c4);
      st_bf16x4(p.z + (size_t)c * W + 4 * c4, x.x * (1.f + s.x), x.y * (1.f + s.y), x.z * (1.f + s.z),
                x.w * (1.f + s.w));
    }
    ss = cons_sum(ss, red);
    if (tid == 0) sumsq_slot(p, 0, 0)[c] = ss;
  } else if (c < p.M + sh.nsh) {
    const float* shift = mod_row(p, sh.srow[c - p.M]) + W;
#pragma unroll 1
    for (int c4 = tid; c4 < W / 4; c4 += kCons) {
      const float4 s = __ldg(reinterpret_cast<const float4*>(shift) + c4);
      st_bf16x4(p.z + (size_t)c * W + 4 * c4, s.x, s.y, s.z, s.w);
    }
  }
}

// ---- block epilogues --------------------------------------------------------------------------
// Every CTA that added into output block b finishes its share of the block's token rows,
// [r0, r1), once all of them have arrived. A[m][128] (row m of the block at A + 128 m) holds the
// staged accumulator rows; each CTA clears the rows it read. The shift rows M..M+nsh-1, which
// every share reads, are cleared in a later phase (clear_shift_rows).
__device__ __forceinline__ void stage_rows(float* A, const float* src, int N, int c0, int r0, int r1) {
#pragma unroll 1
  for (int i = threadIdx.x; i < (r1 - r0) * 32; i += kCons) {
    const int m = r0 + (i >> 5);
    cp16(A + m * 128 + (i & 31) * 4, src + (size_t)m * N + c0 + (i & 31) * 4);
  }
}
__device__ __forceinline__ void clear_rows(float* acc, int N, int c0, int r0, int r1) {
#pragma unroll 1
  for (int i = threadIdx.x; i < (r1 - r0) * 32; i += kCons)
    __stcg(reinterpret_cast<float4*>(acc + (size_t)(r0 + (i >> 5)) * N + c0) + (i & 31), make_float4(0.f, 0.f, 0.f, 0.f));
}
// Clears the shift rows of the qkv accumulator (this layer) and of the gate/up accumulator
// (previous layer); every CTA's consumers take a strided share.
__device__ __forceinline__ void clear_shift_rows(const StepShared& __restrict__ sh, bool qkv, bool gu) {
  const StepArgs& p = sh.p;
  const int nq = qkv ? sh.nsh * p.qkvd / 4 : 0, ng = gu ? sh.nsh * 2 * p.F / 4 : 0;
  const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
  for (int i = blockIdx.x * kCons + threadIdx.x; i < nq + ng; i += gridDim.x * kCons) {
    if (i < nq) __stcg(reinterpret_cast<float4*>(p.acc_qkv + (size_t)p.M * p.qkvd) + i, zero);
    else __stcg(reinterpret_cast<float4*>(p.acc_gu + (size_t)p.M * 2 * p.F) + (i - nq), zero);
  }
}

// qkv block b, rows [r0, r1): value = rstd(h_m) * acc[m] + acc[M + sidx[m]]; RoPE on q/k
// pairs; q -> Q, k -> K cache, v -> Vt cache (bf16). Lane owns 4 consecutive features (two
// RoPE pairs), whose (cos, sin) are staged per row next to the accumulator rows. DH = head dim.
template <int DH>
__device__ __noinline__ void epi_qkv(const StepShared& __restrict__ sh, int l, int b, int r0, int r1, uint8_t* X) {
  const StepArgs& p = sh.p;
  const int M = p.M, warp = threadIdx.x >> 5, lane = threadIdx.x & 31, c0 = b * 128;
  float* A = reinterpret_cast<float*>(X);
  float* CS = A + kMaxRows * 128;           // [m][lane][cos0, sin0, cos1, sin1]
  float* rs = CS + kMaxRows * 128;
  stage_rows(A, p.acc_qkv, p.qkvd, c0, r0, r1);
  stage_rows(A, p.acc_qkv, p.qkvd, c0, M, M + sh.nsh);
  constexpr int half = DH / 2;
  const int n = c0 + 4 * lane;
  const bool qk = n < p.qd + p.kvd, isq = n < p.qd;
  const int sn = isq ? n : n - p.qd;             // feature within q, or within k
  const int hh = sn / DH, rr0 = sn % DH;         // head and dim of the lane's first feature
  const int ev = n - p.qd - p.kvd;               // feature within v
  if (qk && p.rope) {
#pragma unroll 1
    for (int m = r0 + warp; m < r1; m += kConsWarps)
      cp16(CS + m * 128 + 4 * lane, p.rope_cs + (size_t)sh.row_i[m] * DH + (rr0 >> 1) * 2);
  }
  const float* s1 = sumsq_slot(p, l, 0);
  for (int m = r0 + threadIdx.x; m < r1; m += kCons) rs[m] = rsqrtf(__ldcg(s1 + m) / p.W + 1e-6f);
  cp_wait_all();
  clear_rows(p.acc_qkv, p.qkvd, c0, r0, r1);
  named_sync(2, kCons);
#pragma unroll 1
  for (int m = r0 + warp; m < r1; m += kConsWarps) {
    const float r = rs[m];
    const float4 a = *reinterpret_cast<const float4*>(A + m * 128 + 4 * lane);
    const float4 s = *reinterpret_cast<const float4*>(A + (M + sh.sidx[m]) * 128 + 4 * lane);
    const float v[4] = {fmaf(r, a.x, s.x), fmaf(r, a.y, s.y), fmaf(r, a.z, s.z), fmaf(r, a.w, s.w)};
    const int rb = sh.row_b[m], i = sh.row_i[m];
    if (qk) {
      __nv_bfloat16* dst = isq ? p.q + (((size_t)rb * p.n_heads + hh) * p.H + i) * DH
                               : p.kcache + ((((size_t)rb * p.L + l) * p.n_kv_heads + hh) * p.n_keys + p.P + i) * DH;
      const float4 cs = p.rope ? *reinterpret_cast<const float4*>(CS + m * 128 + 4 * lane) : make_float4(1.f, 0.f, 1.f, 0.f);
#pragma unroll
      for (int e = 0; e < 4; e += 2) {
        const int rr = rr0 + e;   // the lane's 4 features lie in one head (DH is a multiple of 4)
        const float c = e ? cs.z : cs.x, si = e ? cs.w : cs.y;
        // with RoPE, rows 2j, 2j+1 of a head hold dims j and j + DH/2 (pair-interleaved weights)
        const int d0 = p.rope ? (rr >> 1) : rr, d1 = p.rope ? (rr >> 1) + half : rr + 1;
        dst[d0] = __float2bfloat16_rn(v[e] * c - v[e + 1] * si);
        dst[d1] = __float2bfloat16_rn(v[e + 1] * c + v[e] * si);
      }
    } else {
      const int g = ev / DH, d = ev % DH;   // the lane's 4 features lie in one head
      __nv_bfloat16* dst = p.vtcache + ((((size_t)rb * p.L + l) * p.n_kv_heads + g) * DH + d) * p.nk_pad + p.P + i;
#pragma unroll
      for (int e = 0; e < 4; ++e) dst[(size_t)e * p.nk_pad] = __float2bfloat16_rn(v[e]);
    }
  }
}

// gate/up block b (rows interleaved gate_j, up_j), rows [r0, r1): act[m][j] = gelu_tanh(gate) * up
// with gate, up = rstd(h_m) * acc[m] + acc[M + sidx[m]].
__device__ __noinline__ void epi_geglu(const StepShared& __restrict__ sh, int l, int b, int r0, int r1, uint8_t* X) {
  const StepArgs& p = sh.p;
  const int M = p.M, warp = threadIdx.x >> 5, lane = threadIdx.x & 31, c0 = b * 128;
  float* A = reinterpret_cast<float*>(X);
  float* rs = A + kMaxRows * 128;
  stage_rows(A, p.acc_gu, 2 * p.F, c0, r0, r1);
  stage_rows(A, p.acc_gu, 2 * p.F, c0, M, M + sh.nsh);
  const float* s2 = sumsq_slot(p, l, 1);
  for (int m = r0 + threadIdx.x; m < r1; m += kCons) rs[m] = rsqrtf(__ldcg(s2 + m) / p.W + 1e-6f);
  cp_wait_all();
  clear_rows(p.acc_gu, 2 * p.F, c0, r0, r1);
  named_sync(2, kCons);
#pragma unroll 1
  for (int m = r0 + warp; m < r1; m += kConsWarps) {
    const float r = rs[m];
    const float4 a = *reinterpret_cast<const float4*>(A + m * 128 + 4 * lane);
    const float4 s = *reinterpret_cast<const float4*>(A + (M + sh.sidx[m]) * 128 + 4 * lane);
    const float g0 = fmaf(r, a.x, s.x), u0 = fmaf(r, a.y, s.y), g1 = fmaf(r, a.z, s.z), u1 = fmaf(r, a.w, s.w);
    reinterpret_cast<uint32_t*>(p.act + (size_t)m * p.F + b * 64)[lane] = pack_bf16(gelu_tanh(g0) * u0, gelu_tanh(g1) * u1);
  }
}

// o / down block b, rows [r0, r1): h[m] += gate(tau_m) * acc[m] on the block's 128 features, the
// rows' partial sums of squares into `ss_out`, and (unless next_mod < 0) z[m] = h (1 + scale); the
// first share also writes the block's shift rows of the next norm (modulation offsets next_mod =
// scale, next_mod + W = shift).
__device__ __noinline__ void epi_resid(const StepShared& __restrict__ sh, float* acc, int gate_off, int next_mod,
                                       float* ss_out, int b, int r0, int r1, bool first, uint8_t* X) {
  const StepArgs& p = sh.p;
  const int M = p.M, W = p.W, nsh = sh.nsh, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* A = reinterpret_cast<float*>(X);
  float* Hs = A + kMaxRows * 128;
  float* G = Hs + kMaxRows * 128;           // [nsh][128] gates, then scales, then shifts
  float* Sc = G + kStepMaxShift * 128;
  float* Sh = Sc + kStepMaxShift * 128;
  const int tid = threadIdx.x, c0 = b * 128;
  stage_rows(A, acc, W, c0, r0, r1);
  stage_rows(Hs, p.h, W, c0, r0, r1);
  const int nv = next_mod >= 0 ? 3 : 1;
#pragma unroll 1
  for (int i = tid; i < nv * nsh * 32; i += kCons) {
    const int kind = i / (nsh * 32), j = (i / 32) % nsh, q = i & 31;
    const int off = kind == 0 ? gate_off : next_mod + (kind - 1) * W;
    cp16(G + (kind * kStepMaxShift + j) * 128 + q * 4, mod_row(p, sh.srow[j]) + off + c0 + q * 4);
  }
  cp_wait_all();
  clear_rows(acc, W, c0, r0, r1);
  named_sync(2, kCons);
#pragma unroll 1
  for (int m = r0 + warp; m < r1; m += kConsWarps) {
    const int j = sh.sidx[m];
    const float4 a = *reinterpret_cast<const float4*>(A + m * 128 + 4 * lane);
    float4 h = *reinterpret_cast<const float4*>(Hs + m * 128 + 4 * lane);
    const float4 g = *reinterpret_cast<const float4*>(G + j * 128 + 4 * lane);
    h.x = fmaf(g.x, a.x, h.x);
    h.y = fmaf(g.y, a.y, h.y);
    h.z = fmaf(g.z, a.z, h.z);
    h.w = fmaf(g.w, a.w, h.w);
    reinterpret_cast<float4*>(p.h + (size_t)m * W + c0)[lane] = h;
    const float ss = warp_sum(fmaf(h.x, h.x, fmaf(h.y, h.y, fmaf(h.z, h.z, h.w * h.w))));
    if (lane == 0) atomicAdd(ss_out + m, ss);
    if (next_mod >= 0) {
      const float4 s = *reinterpret_cast<const float4*>(Sc + j * 128 + 4 * lane);
      st_bf16x4(p.z + (size_t)m * W + c0 + 4 * lane, h.x * (1.f + s.x), h.y * (1.f + s.y), h.z * (1.f + s.z),
                h.w * (1.f + s.w));
    }
  }
  if (next_mod >= 0 && first) {
#pragma unroll 1
    for (int j = warp; j < nsh; j += kConsWarps) {
      const float4 s = *reinterpret_cast<const float4*>(Sh + j * 128 + 4 * lane);
      st_bf16x4(p.z + (size_t)(M + j) * W + c0 + 4 * lane, s.x, s.y, s.z, s.w);
    }
  }
}

// Merge the key chunks of query rows (one warp): lane c < n_chunks copies chunk c's partial row
// into shared memory with one bulk copy (up to two rows at once), the weights exp(max_c - max)
// and the total sum are formed meanwhile, then each lane loads its dims of every chunk before
// accumulating. Lane owns dims 2 lane + 64 e, e < DH / 64. Rows r0, r0 + step, ... < r1 of
// robot-group bg.
template <int DH>
__device__ __forceinline__ void combine_rows_warp(const StepArgs& __restrict__ p, int bg, int r0, int r1, int step,
                                                  __nv_bfloat16* buf, uint64_t* bar, Role& st) {
  constexpr int E = DH / 64, kG = 8;
  // the arguments this routine uses, in registers (the asm statements below clobber memory, which
  // would otherwise make every use reload them)
  const int lane = threadIdx.x & 31, nck = p.n_chunks, r_pad = p.r_pad, H = p.H, qd = p.qd;
  const int nkv = p.n_kv_heads, group = p.group;
  const float scale_log2 = p.scale_log2;
  const __nv_bfloat16* __restrict__ part_o = p.part_o;
  const float* __restrict__ part_ml = p.part_ml;
  __nv_bfloat16* __restrict__ o_out = p.o;
  int* err = p.err;
  const unsigned long long wait_ns = p.wait_ns;
  constexpr int kRows = 2;                  // rows staged at once (two when n_chunks <= 16)
  const int batch = nck * kRows <= kStepMaxChunks ? kRows : 1;
#pragma unroll 1
  for (int rb = r0; rb < r1; rb += batch * step) {
    int nr = 0;
    for (int r = rb; r < r1 && nr < batch; r += step) ++nr;
    if (lane == 0) mbar_expect_tx(bar, (uint32_t)(nr * nck * DH * 2));
    __syncwarp();
    if (lane < nck) {
      // partial rows written by other CTAs (acquired through the chunk count) are read next by
      // this lane's bulk copies
      asm volatile("fence.proxy.async.global;" ::: "memory");
      for (int k = 0; k < nr; ++k) {
        const __nv_bfloat16* src = part_o + (((size_t)bg * nck + lane) * r_pad + rb + k * step) * DH;
        asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                     ::"r"(su32(buf + ((size_t)k * nck + lane) * DH)), "l"(src), "r"(DH * 2), "r"(su32(bar)) : "memory");
      }
    }
    ++st.c_uses;
    float mc[kRows], lc[kRows];
#pragma unroll
    for (int k = 0; k < kRows; ++k) {
      mc[k] = -INFINITY;
      lc[k] = 0.f;
      if (k < nr && lane < nck) {
        const size_t pi = ((size_t)bg * nck + lane) * r_pad + rb + k * step;
        mc[k] = __ldcg(part_ml + pi * 2);
        lc[k] = __ldcg(part_ml + pi * 2 + 1);
      }
    }
    float wgt[kRows], invL[kRows];
#pragma unroll
    for (int k = 0; k < kRows; ++k) {
      const float M = warp_max(mc[k]);
      wgt[k] = lane < nck && k < nr ? exp2f((mc[k] - M) * scale_log2) : 0.f;
      invL[k] = 1.f / warp_sum(wgt[k] * lc[k]);
    }
    const bool ok = mbar_wait(bar, st.cpar, err, 53, wait_ns);
    st.cpar ^= 1u;
#pragma unroll 1
    for (int k = 0; k < nr && ok; ++k) {
      const int r = rb + k * step;
      const __nv_bfloat16* row = buf + (size_t)k * nck * DH;
      const float wk = k ? wgt[1] : wgt[0], ik = k ? invL[1] : invL[0];
      float2 acc[E];
#pragma unroll
      for (int e = 0; e < E; ++e) acc[e] = make_float2(0.f, 0.f);
#pragma unroll 1
      for (int c0 = 0; c0 < nck; c0 += kG) {
        __nv_bfloat162 v[kG][E];
#pragma unroll
        for (int g = 0; g < kG; ++g)
#pragma unroll
          for (int e = 0; e < E; ++e)
            v[g][e] = c0 + g < nck ? *reinterpret_cast<const __nv_bfloat162*>(row + (c0 + g) * DH + 64 * e + 2 * lane)
                                   : __floats2bfloat162_rn(0.f, 0.f);
#pragma unroll
        for (int g = 0; g < kG; ++g) {
          const float wc = __shfl_sync(0xffffffffu, wk, (c0 + g) & 31);
#pragma unroll
          for (int e = 0; e < E; ++e) {
            const float2 f = __bfloat1622float2(v[g][e]);
            acc[e].x = fmaf(wc, f.x, acc[e].x);
            acc[e].y = fmaf(wc, f.y, acc[e].y);
          }
        }
      }
      const int b = bg / nkv, g = bg % nkv, j = r / H, i = r % H;
      __nv_bfloat16* dst = o_out + ((size_t)b * H + i) * qd + (size_t)(g * group + j) * DH;
#pragma unroll
      for (int e = 0; e < E; ++e)
        *reinterpret_cast<uint32_t*>(dst + 64 * e + 2 * lane) = pack_bf16(acc[e].x * ik, acc[e].y * ik);
    }
    __syncwarp();
    if (!ok) break;
  }
}

// Combine step (when the attention step does not merge the chunks itself): query rows over all
// consumer warps of the grid.
template <int DH>
__device__ __noinline__ void combine_rows(const StepArgs& __restrict__ p, uint8_t* X, uint64_t* bar, Role& st) {
  const int w = threadIdx.x >> 5, gw = blockIdx.x * kConsWarps + w, nw = gridDim.x * kConsWarps;
  __nv_bfloat16* buf = reinterpret_cast<__nv_bfloat16*>(X) + (size_t)w * kStepMaxChunks * DH;
  const int total = p.B * p.n_kv_heads * p.rows;
#pragma unroll 1
  for (int idx = gw; idx < total; idx += nw) combine_rows_warp<DH>(p, idx / p.rows, idx % p.rows, idx % p.rows + 1, 1, buf, bar, st);
}

struct ConsSync {
  __device__ void operator()() const { named_sync(2, kCons); }
};

}  // namespace

// ---- projection step: acc[m][n] += sum over this CTA's weight tiles of A[m][k] W[n][k] -----
// The issuer thread loads the activation tiles (tensor map) and issues the MMAs against the weight
// ring; the consumer warps add the finished 128 x 64 tile into `acc` (fp32, L2) with 16-byte
// reds and count the block's arrival; once every CTA of the block has arrived, each runs the
// block's epilogue for its share of the rows.
template <int DH>
__device__ __noinline__ void projection_step(const StepShared& __restrict__ sh, const CUtensorMap* amap, int l, int j,
                                             uint32_t tmem, size_t xbytes, Role& st_) {
  RoleCopy rc_(st_);
  Role& st = rc_.v;
  const StepArgs& p = sh.p;
  const Smem S = smem_plan(p.ring, xbytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool mma = threadIdx.x == kMmaThread, cons = warp < kConsWarps;
  const Tiles tl = sh.tiles[j];
  const int nt = tl.k1 - tl.k0;
  if (nt <= 0) return;
  const int N = j == 0 ? p.qkvd : j == 2 ? 2 * p.F : p.W;
  float* acc = j == 0 ? p.acc_qkv : j == 1 ? p.acc_o : j == 2 ? p.acc_gu : p.acc_d;
  const int R = (j == 0 || j == 2) ? p.M + sh.nsh : p.M;   // rows added: tokens (+ shift rows)
  if (mma) {
    mbar_expect_tx(S.a_full, (uint32_t)nt * kATile);
    for (int i = 0; i < nt; ++i) tma_2d(S.X + (size_t)i * kATile, amap, (tl.k0 + i) * 64, 0, S.a_full);
    ++st.a_uses;
    // the next weight tile's barrier is tested (without blocking) before the current tile's MMAs
    // are issued, so that the test's latency overlaps the issue
    bool ready = mbar_peek(S.full + st.slot, st.par);
    bool good = mbar_wait(S.a_full, st.apar, p.err, 42, p.wait_ns);
    for (int i = 0; i < nt && good; ++i) {
      if (!ready) {
        good = mbar_wait(S.full + st.slot, st.par, p.err, 43, p.wait_ns);
        if (!good) break;
      }
      tc_fence_after();
      const int cur = st.slot;
      if (++st.slot == p.ring) { st.slot = 0; st.par ^= 1u; }
      ready = i + 1 < nt && mbar_peek(S.full + st.slot, st.par);
      const uint32_t a0 = su32(S.ring + (size_t)cur * kSlot), b0 = su32(S.X + (size_t)i * kATile);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_bf16(tmem, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc_m128(64), (i | k) ? 1u : 0u);
      mma_commit(S.empty + cur);
    }
    mma_commit(S.g_done);
  }
  st.apar ^= 1u;
  if (cons) {
    const bool good = mbar_wait(S.g_done, st.gpar, p.err, 44, p.wait_ns);
    tc_fence_after();
    const uint32_t tm = tmem_base_after_wait(S.tmem_slot);
    const int quad = warp & 3, row = quad * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    // the tile goes through shared memory (T[token][row], over the activation tiles, which the
    // finished MMAs no longer read) so that the adds into L2 are 16-byte reds along the features
    float* T = reinterpret_cast<float*>(S.X);
#pragma unroll 1
    for (int q = (warp >> 2) * 32; q < R; q += 64) {   // warps 4-7 take tokens 32-63
      float v[32];
      __syncwarp();
      tmem_ld32(tm + lane_base + q, v);
#pragma unroll
      for (int e = 0; e < 32; ++e) T[(q + e) * 128 + row] = v[e];
    }
    named_sync(2, kCons);
    if (good) {
      float* dst = acc + tl.b * 128;
#pragma unroll 4
      for (int idx = threadIdx.x; idx < R * 32; idx += kCons) {
        const int m = idx >> 5, c4 = idx & 31;
        red_add_v4(dst + (size_t)m * N + 4 * c4, *reinterpret_cast<const float4*>(T + m * 128 + 4 * c4));
      }
    }
    named_sync(2, kCons);
    if (threadIdx.x == 0) {
      // arrive on the block (release: this CTA's reds, ordered before by the named barrier), then
      // wait until every CTA of the block has arrived (acquire: their reds)
      int go = 0;
      if (good) {
        unsigned* ctr = p.sync + (1 + kStepBarriersPerLayer * p.L) + (size_t)(4 * l + j) * kStepMaxNB + tl.b;
        asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
        go = count_wait(ctr, (unsigned)tl.contrib, p.err, p.wait_ns);
      }
      *S.last = go;
    }
    named_sync(2, kCons);
    if (*reinterpret_cast<volatile int*>(S.last)) {
      const int W6 = 6 * p.W, b6 = l * W6, M = p.M;
      const int r0 = tl.idx * M / tl.contrib, r1 = (tl.idx + 1) * M / tl.contrib;
      if (j == 0) epi_qkv<DH>(sh, l, tl.b, r0, r1, S.X);
      else if (j == 2) epi_geglu(sh, l, tl.b, r0, r1, S.X);
      else if (j == 1) epi_resid(sh, p.acc_o, b6 + 2 * p.W, b6 + 3 * p.W, sumsq_slot(p, l, 1), tl.b, r0, r1, tl.idx == 0, S.X);
      else epi_resid(sh, p.acc_d, b6 + 5 * p.W, l + 1 < p.L ? b6 + W6 : -1, sumsq_slot(p, l + 1, 0), tl.b, r0, r1,
                     tl.idx == 0, S.X);
      if (j < 3) {
        // count this share (release: every consumer's epilogue stores, ordered before by the
        // named barrier) for the phase that reads the projection's output
        named_sync(2, kCons);
        if (threadIdx.x == 0) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(done_ctr(p, l, j)) : "memory");
      }
    }
  }
  st.gpar ^= 1u;
}

// ---- attention step: items (robot-group bg, 128-row query tile qt, 64-key chunk kc) ---------
template <int DH>
__device__ __noinline__ void attention_step(const StepArgs& __restrict__ p, const CUtensorMap* t_q, const CUtensorMap* t_k,
                                            const CUtensorMap* t_vt, int l, uint32_t tmem, Role& st_, bool fused) {
  RoleCopy rc_(st_);
  Role& st = rc_.v;
  constexpr int NC = DH / 64;
  constexpr uint32_t QB = DH * kQT * 2, KB = DH * kKC * 2, VB = DH * kKC * 2;
  const Smem S = smem_plan(p.ring, step_x_bytes(DH));
  uint8_t* sQ = S.X;
  uint8_t* sK = sQ + QB;
  uint8_t* sV = sK + KB;
  uint8_t* sP = sV + VB;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool mma = threadIdx.x == kMmaThread, cons = warp < kConsWarps;
  const int nck = p.n_chunks, nqt = p.r_pad / kQT;
  const int items = p.B * p.n_kv_heads * nqt * nck;
  if (fused && (int)blockIdx.x >= items) {
    // CTAs without an item merge the key chunks: each takes a share of one query tile's rows
    // and starts once all chunks of that tile have finished
    if (cons) {
      const int ncomb = gridDim.x - items, ci = (int)blockIdx.x - items, QT = p.B * p.n_kv_heads * nqt;
      const int t = ci * QT / ncomb, first = (t * ncomb + QT - 1) / QT, next = ((t + 1) * ncomb + QT - 1) / QT;
      const int bg = t / nqt, qt = t % nqt, rows = min(kQT, p.rows - qt * kQT);
      const int r0 = qt * kQT + (ci - first) * rows / (next - first), r1 = qt * kQT + (ci - first + 1) * rows / (next - first);
      if (threadIdx.x == 0) *S.last = count_wait(qtile_ctr(p, l, t), (unsigned)nck, p.err, p.wait_ns);
      named_sync(2, kCons);
      if (*reinterpret_cast<volatile int*>(S.last)) {
        __nv_bfloat16* buf = reinterpret_cast<__nv_bfloat16*>(S.X) + (size_t)warp * kStepMaxChunks * DH;
        combine_rows_warp<DH>(p, bg, r0 + warp, r1, kConsWarps, buf, S.cbar + warp, st);
        named_sync(2, kCons);
        if (threadIdx.x == 0) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(done_ctr(p, l, 3)) : "memory");
      }
    }
    return;
  }
  for (int it = blockIdx.x; it < items; it += gridDim.x) {
    const int kc = it % nck, qt = (it / nck) % nqt, bg = it / (nck * nqt);
    const int b = bg / p.n_kv_heads, g = bg % p.n_kv_heads;
    const int kvz = (b * p.L + l) * p.n_kv_heads + g;
    if (mma) {
      const uint64_t pol = policy_evict_last();
      mbar_expect_tx(S.q_full, QB + KB);
#pragma unroll
      for (int cc = 0; cc < NC; ++cc) {
        tma_3d(sQ + cc * (kQT * 128), t_q, cc * 64, qt * kQT, bg, S.q_full, pol);
        tma_3d(sK + cc * (kKC * 128), t_k, cc * 64, kc * kKC, kvz, S.q_full, pol);
      }
      mbar_expect_tx(S.v_full, VB);
      tma_3d(sV, t_vt, kc * kKC, 0, kvz, S.v_full, pol);
      ++st.i_uses;
      bool good = mbar_wait(S.q_full, st.ipar, p.err, 45, p.wait_ns);
      if (good) {
        tc_fence_after();
        const uint32_t q0 = su32(sQ), k0 = su32(sK);
#pragma unroll
        for (int cc = 0; cc < NC; ++cc)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_bf16(tmem, sw128_desc(q0 + cc * (kQT * 128) + 32 * k), sw128_desc(k0 + cc * (kKC * 128) + 32 * k),
                     idesc_m128(kKC), (cc | k) ? 1u : 0u);
      }
      mma_commit(S.s_full);
      good = good && mbar_wait(S.p_full, st.ipar, p.err, 46, p.wait_ns) && mbar_wait(S.v_full, st.ipar, p.err, 47, p.wait_ns);
      if (good) {
        tc_fence_after();
        const uint32_t p0 = su32(sP), v0 = su32(sV);
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16(tmem + 256, sw128_desc(p0 + 32 * k), sw128_desc(v0 + 32 * k), idesc_m128(DH), k ? 1u : 0u);
      }
      mma_commit(S.o_done);
    }
    if (cons) {
      // warps 0-3: softmax over the chunk's 64 keys, one query row per thread; all warps then
      // read out O, warps 0-3 the first half of its columns and warps 4-7 the second
      const int quad = warp & 3, half = warp >> 2, row = quad * 32 + lane;
      const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
      bool ok_s = true;
      float mx = -INFINITY, l_sum = 0.f;
      if (half == 0) {
        ok_s = mbar_wait(S.s_full, st.ipar, p.err, 48, p.wait_ns);
        tc_fence_after();
        const uint32_t tS = tmem_base_after_wait(S.tmem_slot);
        const int key0 = kc * kKC;
        const int nvalid = p.n_keys - key0 < kKC ? p.n_keys - key0 : kKC;
        float sv[64];
        __syncwarp();
        tmem_ld64(tS + lane_base, sv);
        if (nvalid < 64) {   // keys past the end: excluded from the maximum, P = 2^-inf = 0
#pragma unroll
          for (int i = 0; i < 64; ++i)
            if (i >= nvalid) sv[i] = -INFINITY;
        }
#pragma unroll
        for (int i = 0; i < 64; ++i) mx = fmaxf(mx, sv[i]);
        const float mxs = mx * p.scale_log2;
        const int r8 = row & 7;
        uint8_t* prow = sP + row * 128;
#pragma unroll
        for (int gi = 0; gi < 8; ++gi) {
          uint32_t pk[4];
#pragma unroll
          for (int e = 0; e < 8; e += 2) {
            const int i0 = gi * 8 + e;
            const float e0 = ex2_approx(fmaf(sv[i0], p.scale_log2, -mxs));
            const float e1 = ex2_approx(fmaf(sv[i0 + 1], p.scale_log2, -mxs));
            const __nv_bfloat162 h = __floats2bfloat162_rn(e0, e1);
            const float2 hf = __bfloat1622float2(h);
            l_sum += hf.x + hf.y;   // normalise by what the MMA sums
            pk[e / 2] = *reinterpret_cast<const uint32_t*>(&h);
          }
          *reinterpret_cast<uint4*>(prow + ((gi ^ r8) * 16)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(S.p_full);
      }
      const bool ok_o = mbar_wait(S.o_done, st.ipar, p.err, 49, p.wait_ns);
      tc_fence_after();
      const uint32_t tO = tmem_base_after_wait(S.tmem_slot) + 256;
      // unnormalised O row in bf16: staged in shared memory (the operand tiles are free once O
      // is complete; rows padded by 16 bytes against bank conflicts), then written by one bulk
      // copy per row, complete before the chunk is counted
      const int qrow = qt * kQT + row;
      const size_t pi = ((size_t)bg * nck + kc) * p.r_pad + qrow;
      constexpr uint32_t pitch = DH * 2 + 16;
      uint8_t* srow = S.X + (size_t)row * pitch;
#pragma unroll 1
      for (int q = half * (DH / 2); q < (half + 1) * (DH / 2); q += 32) {
        float ov[32];
        __syncwarp();
        tmem_ld32(tO + lane_base + q, ov);
#pragma unroll
        for (int e = 0; e < 32; e += 8)
          *reinterpret_cast<uint4*>(srow + (q + e) * 2) = make_uint4(pack_bf16(ov[e], ov[e + 1]), pack_bf16(ov[e + 2], ov[e + 3]),
                                                                     pack_bf16(ov[e + 4], ov[e + 5]), pack_bf16(ov[e + 6], ov[e + 7]));
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      named_sync(2, kCons);   // both halves of every row staged
      if (half == 0 && ok_s && ok_o && qrow < p.rows) {
        bulk_s2g(p.part_o + pi * DH, srow, DH * 2);
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        p.part_ml[pi * 2] = mx;
        p.part_ml[pi * 2 + 1] = l_sum;
        asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
        asm volatile("fence.proxy.async.global;" ::: "memory");
      }
      // count the chunk for its query tile (release: every consumer's rows, ordered before by the
      // named barrier)
      named_sync(2, kCons);
      if (threadIdx.x == 0 && ok_s && ok_o)
        asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(qtile_ctr(p, l, bg * nqt + qt)) : "memory");
    }
    st.ipar ^= 1u;
    // the next item's operand loads overwrite this item's operands and P
    tc_fence_before();
    __syncwarp();
    named_sync(1, kSyncThreads);
    tc_fence_after();
  }
}

// Final norm and action-out projection of row m: y = RMSNorm(h) (1 + scale) + shift (rounded to
// bf16 like every projection input), v[m] = W_out y + b_out.
__device__ __noinline__ void final_row(const StepArgs& __restrict__ p, int m, float* ys) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, W = p.W;
  const float* mod = mod_row(p, p.tau_row[m]) + (size_t)p.L * 6 * W;
  const float rstd = rsqrtf(__ldcg(sumsq_slot(p, p.L, 0) + m) / W + 1e-6f);
#pragma unroll 1
  for (int c4 = tid; c4 < W / 4; c4 += kCons) {
    const float4 h = __ldcg(reinterpret_cast<const float4*>(p.h + (size_t)m * W) + c4);
    const float4 sc = __ldg(reinterpret_cast<const float4*>(mod) + c4);
    const float4 sf = __ldg(reinterpret_cast<const float4*>(mod + W) + c4);
    const __nv_bfloat162 lo = __floats2bfloat162_rn(fmaf(h.x * rstd, 1.f + sc.x, sf.x), fmaf(h.y * rstd, 1.f + sc.y, sf.y));
    const __nv_bfloat162 hi = __floats2bfloat162_rn(fmaf(h.z * rstd, 1.f + sc.z, sf.z), fmaf(h.w * rstd, 1.f + sc.w, sf.w));
    reinterpret_cast<float4*>(ys)[c4] = make_float4(__low2float(lo), __high2float(lo), __low2float(hi), __high2float(hi));
  }
  named_sync(2, kCons);
  const __nv_bfloat16* wo = static_cast<const __nv_bfloat16*>(p.w_out);
#pragma unroll 1
  for (int d = warp; d < p.D; d += kConsWarps) {
    float a = 0.f;
#pragma unroll 4
    for (int k = 2 * lane; k < W; k += 64) {
      const float2 wv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(wo + (size_t)d * W + k));
      a = fmaf(ys[k], wv.x, fmaf(ys[k + 1], wv.y, a));
    }
    a = warp_sum(a);
    if (lane == 0) p.v[(size_t)m * p.D + d] = a + p.b_out[d];
  }
}

template <int DH>
__global__ void __launch_bounds__(kThreads, 1)
    step_kernel(const __grid_constant__ CUtensorMap t_z, const __grid_constant__ CUtensorMap t_o,
                const __grid_constant__ CUtensorMap t_act, const __grid_constant__ CUtensorMap t_q,
                const __grid_constant__ CUtensorMap t_k, const __grid_constant__ CUtensorMap t_vt,
                const __grid_constant__ StepArgs p_in) {
  constexpr size_t XB = step_x_bytes(DH);
  // the arguments and this step's flow-time rows live in shared memory for the whole launch
  __shared__ StepShared sh;
  const int R = p_in.ring;
  const Smem S = smem_plan(R, XB);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    sh.p = p_in;
    int n = __ldg(p_in.sinfo);
    n = n < kStepMaxShift ? n : kStepMaxShift;
    n = n < kMaxRows - p_in.M ? n : kMaxRows - p_in.M;
    sh.nsh = n > 0 ? n : 0;
    for (int i = 0; i < kStepMaxShift; ++i) sh.srow[i] = __ldg(p_in.sinfo + 1 + i);
    for (int i = 0; i < R; ++i) {
      mbar_init(S.full + i, 1);
      mbar_init(S.empty + i, 1);
    }
    for (int i = 0; i < 8; ++i) mbar_init(S.a_full + i, i == 5 ? 4 : 1);   // p_full: one arrive per consumer warp
    for (int i = 0; i < kConsWarps; ++i) mbar_init(S.cbar + i, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (threadIdx.x < kMaxRows) {
    const int si = threadIdx.x < p_in.M ? __ldg(p_in.sidx + threadIdx.x) : 0;
    sh.sidx[threadIdx.x] = si >= 0 && si < kStepMaxShift ? si : 0;
    sh.row_b[threadIdx.x] = (uint8_t)(threadIdx.x / p_in.H);
    sh.row_i[threadIdx.x] = (uint8_t)(threadIdx.x % p_in.H);
  }
  if (threadIdx.x == 68) {
    const int items = p_in.B * p_in.n_kv_heads * (p_in.r_pad / kQT) * p_in.n_chunks;
    const int qtiles = p_in.B * p_in.n_kv_heads * (p_in.r_pad / kQT);
    sh.fused_combine = (int)gridDim.x - items >= (qtiles > 16 ? qtiles : 16) ? 1 : 0;
    sh.shares[3] = (unsigned)((int)gridDim.x - items);
  }
  if (threadIdx.x >= 72 && threadIdx.x < 75) {
    const int j = threadIdx.x - 72;
    int N, K;
    proj_shape(p_in, j, N, K);
    sh.shares[j] = (unsigned)proj_shares(gridDim.x, N / 128, K / 64);
  }
  if (threadIdx.x >= 64 && threadIdx.x < 68) {
    const int j = threadIdx.x - 64;
    int N, K;
    proj_shape(p_in, j, N, K);
    sh.tiles[j] = assign_tiles(blockIdx.x, gridDim.x, N / 128, K / 64, proj_rot(j));
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(S.tmem_slot)), "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const StepArgs& p = sh.p;
  const uint32_t tmem = *S.tmem_slot;

  if (warp == kProdWarp) {
    // ---- weight producer: this CTA's tiles of every projection, in consumption order ----
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int slot = 0, issued = 0;
      uint32_t par = 0;
      bool ok = true;
      for (int l = 0; l < p.L && ok; ++l)
        for (int j = 0; j < 4 && ok; ++j) {
          int N, K;
          proj_shape(p, j, N, K);
          const Tiles tl = sh.tiles[j];
          const uint8_t* w = static_cast<const uint8_t*>(p.wl[4 * l + j]) + ((size_t)tl.b * (K / 64) + tl.k0) * kSlot;
          for (int t = 0; t < tl.k1 - tl.k0; ++t) {
            if (!mbar_wait(S.empty + slot, par ^ 1u, p.err, 41, p.wait_ns)) { ok = false; break; }
            mbar_expect_tx(S.full + slot, kSlot);
            bulk_g2s(S.ring + (size_t)slot * kSlot, w + (size_t)t * kSlot, kSlot, S.full + slot, pol);
            ++issued;
            if (++slot == R) { slot = 0; par ^= 1u; }
          }
        }
      // copies still in flight land before the CTA exits
      for (int i = issued - R > 0 ? issued - R : 0; i < issued; ++i) mbar_drain(S.full + i % R, (uint32_t)(i / R) & 1u, kDrainNs);
    }
    __syncwarp();
  } else {
    // ---- consumer warps; the last warp: tcgen05 issuer (its lane 0) ----
    const bool mma = threadIdx.x == kMmaThread, cons = warp < kConsWarps;
    Role st;
    bool ok = true;
    unsigned* bar = p.sync;
    if (cons) in_rows(sh, S.red);
    ok = grid_sync(bar++, ok, p.err, S, p.wait_ns, p.unreachable);
    for (int l = 0; l < p.L; ++l) {
      const bool df = sh.fused_combine != 0;   // phases inside the layer wait on counts
      if (ok) projection_step<DH>(sh, &t_z, l, 0, tmem, XB, st);
      ok = df ? phase_wait(done_ctr(p, l, 0), sh.shares[0], ok, p.err, S, p.wait_ns) : grid_sync(bar++, ok, p.err, S, p.wait_ns);
      if (ok) attention_step<DH>(p, &t_q, &t_k, &t_vt, l, tmem, st, df);
      if (df) {
        ok = phase_wait(done_ctr(p, l, 3), sh.shares[3], ok, p.err, S, p.wait_ns);
      } else {
        ok = grid_sync(bar++, ok, p.err, S, p.wait_ns);
        if (ok && cons) combine_rows<DH>(p, S.X, S.cbar + warp, st);
        ok = grid_sync(bar++, ok, p.err, S, p.wait_ns);
      }
      if (ok) projection_step<DH>(sh, &t_o, l, 1, tmem, XB, st);
      ok = df ? phase_wait(done_ctr(p, l, 1), sh.shares[1], ok, p.err, S, p.wait_ns) : grid_sync(bar++, ok, p.err, S, p.wait_ns);
      if (ok) projection_step<DH>(sh, &t_z, l, 2, tmem, XB, st);
      ok = df ? phase_wait(done_ctr(p, l, 2), sh.shares[2], ok, p.err, S, p.wait_ns) : grid_sync(bar++, ok, p.err, S, p.wait_ns);
      // the shift rows of this layer's qkv and gate/up sums have been read by now
      if (ok && cons) clear_shift_rows(sh, true, true);
      if (ok) projection_step<DH>(sh, &t_act, l, 3, tmem, XB, st);
      ok = grid_sync(bar++, ok, p.err, S, p.wait_ns);
    }
    if (cons) {
      if (ok && (int)blockIdx.x < p.M) final_row(p, blockIdx.x, reinterpret_cast<float*>(S.X));
      // the step epilogue (Sec. 4.2-4.4) runs on the last CTA to finish: the count's acquire makes
      // every CTA's velocity rows visible to it
      named_sync(2, kCons);
      if (threadIdx.x == 0) {
        unsigned prev;
        asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;"
                     : "=r"(prev) : "l"(p.sync + step_sync_words(p.L) - 1) : "memory");
        *S.last = ok && prev == gridDim.x - 1u && *reinterpret_cast<volatile int*>(p.err) == 0;
      }
      named_sync(2, kCons);
      if (*reinterpret_cast<volatile int*>(S.last)) {
        float* base = reinterpret_cast<float*>(S.X);
        const EulerSmem es{base + 96, base, base + 64, reinterpret_cast<int*>(S.tmem_slot + 3)};
        for (int b = 0; b < p.eu.B; ++b) euler_robot(p.eu, b, threadIdx.x, kCons, es, ConsSync());
      }
    }
    // a consumer warp exits only after its last combine copies have landed
    if (cons && st.c_uses) mbar_drain(S.cbar + warp, (uint32_t)(st.c_uses - 1) & 1u, kDrainNs);
    if (mma) {
      // tensor memory is freed only after every MMA of this thread has completed, and the CTA
      // exits only after its last operand loads have landed (they are waited for on the normal
      // path; this matters only after an error)
      mma_commit(S.fin);
      mbar_drain(S.fin, 0, kDrainNs);
      if (st.a_uses) mbar_drain(S.a_full, (uint32_t)(st.a_uses - 1) & 1u, kDrainNs);
      if (st.i_uses) {
        mbar_drain(S.q_full, (uint32_t)(st.i_uses - 1) & 1u, kDrainNs);
        mbar_drain(S.v_full, (uint32_t)(st.i_uses - 1) & 1u, kDrainNs);
      }
    }
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

size_t step_smem_bytes(int dh, int ring) { return 1024 + (size_t)ring * kSlot + step_x_bytes(dh) + kTailBytes; }

int step_ring_slots(int dh, int smem_optin) {
  // the kernel's static shared memory (arguments and flow-time rows) comes off the top
  const long long left = (long long)smem_optin - (long long)sizeof(StepShared) - 1024 - (long long)step_x_bytes(dh) -
                         (long long)kTailBytes;
  long long r = left / kSlot;
  if (r > kMaxRing) r = kMaxRing;
  return (int)r;
}

int step_max_tiles(int ctas, const int (*shapes)[2], int n) {
  int most = 0;
  for (int s = 0; s < n; ++s) {
    const int NB = shapes[s][0] / 128, KT = shapes[s][1] / 64;
    if (NB < 1 || NB > ctas || NB > kStepMaxNB) return 0;
    for (int c = 0; c < ctas; ++c) {
      const Tiles t = assign_tiles(c, ctas, NB, KT, 0);
      most = t.k1 - t.k0 > most ? t.k1 - t.k0 : most;
    }
  }
  return most;
}

int step_prepare(int dh, int ring, int* blocks_per_sm) {
  const int smem = (int)step_smem_bytes(dh, ring);
  cudaError_t e = cudaErrorInvalidValue;
  *blocks_per_sm = 0;
  if (dh == 64) {
    e = cudaFuncSetAttribute(step_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, step_kernel<64>, kThreads, smem);
  } else if (dh == 128) {
    e = cudaFuncSetAttribute(step_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, step_kernel<128>, kThreads, smem);
  } else if (dh == 256) {
    e = cudaFuncSetAttribute(step_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, step_kernel<256>, kThreads, smem);
  }
  return e == cudaSuccess ? 0 : -1;
}

// One CTA per SM. The grid barriers need every CTA resident at once: the shared-memory plan
// admits one CTA per SM (checked at set-up with the occupancy calculator) and the kernel is
// launched after the previous kernel has drained, so all `grid` CTAs start together. The
// launch is not marked cooperative because the kernel needs none of its semantics (the same
// kernel launched cooperatively gives the same results). Should the CTAs ever not all be
// resident, the bounded barrier wait reports an error instead of hanging.
int launch_step(const StepMaps& m, const StepArgs& a, int grid, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = step_smem_bytes(a.dh, a.ring);
  cfg.stream = s;
  cfg.attrs = nullptr;
  cfg.numAttrs = 0;
  cudaError_t e = cudaErrorInvalidValue;
  if (a.dh == 64) e = cudaLaunchKernelEx(&cfg, step_kernel<64>, m.z, m.o, m.act, m.q, m.k, m.vt, a);
  if (a.dh == 128) e = cudaLaunchKernelEx(&cfg, step_kernel<128>, m.z, m.o, m.act, m.q, m.k, m.vt, a);
  if (a.dh == 256) e = cudaLaunchKernelEx(&cfg, step_kernel<256>, m.z, m.o, m.act, m.q, m.k, m.vt, a);
  return e == cudaSuccess ? 0 : -1;
}

}  // namespace uad
