// Tensor-core attention of chunk queries over [prefix keys ; chunk keys] (grouped KV heads),
// for bf16 experts with joint attention over the observation prefix.
//
// Layouts (written by the QKV projection epilogue and, for the prefix, by set_prefix):
//   Q  [B][Hkv][G][H][dh]       queries of one KV group are the R = G*H rows of one matrix
//   K  [B][L][Hkv][NK][dh]      keys: P prefix rows then H chunk rows (NK = P + H)
//   Vt [B][L][Hkv][dh][NKp]     values transposed (keys contiguous), NKp = NK rounded up to 8
// Few query tiles (split-KV): one CTA = one 128-row query tile x one 128-key chunk of one
//   (robot, group): TMA loads Q, K, Vt tiles (128-byte swizzle); S = Q K^T on tcgen05 into TMEM;
//   four warps read S rows, apply the 1/sqrt(dh) scale and key mask, write P = exp(S - rowmax) in
//   bf16 into shared memory in the K-major swizzled layout; O = P Vt^T on tcgen05; O rows
//   (unnormalised) and per-row (max, sum) go to a workspace. attn_combine merges the key chunks
//   (the usual log-sum-exp rescaling) and writes o [B*H][Hq*dh] in bf16 for the O projection.
// Many query tiles (attn_tc2_kernel): one CTA per query tile walks all key chunks in one pass,
//   O accumulating in TMEM, and writes o itself; with at most half as many tiles as SMs, two CTAs
//   per tile, one per half of the head dims.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "uad_internal.cuh"
#include "ptx.cuh"

namespace uad {

using namespace ptx;

namespace {

constexpr int kQT = 128, kKT = 128;
constexpr int kMaxKeyChunks = 16;   // keys per (robot, layer) <= 2048
constexpr uint32_t kTmemCols = 256; // S (128 columns) then O (dh <= 256 columns) in the same columns
constexpr unsigned long long kWaitNs = 2000000000ull;

__device__ __forceinline__ bool mbar_wait(uint64_t* b, uint32_t parity, int* err, int code) {
  return ptx::mbar_wait(b, parity, err, code, kWaitNs);
}
__device__ __forceinline__ float ex2_fast(float x) { return ptx::ex2_approx(x); }


// smem plan for head dim dh: Q tiles (dh/64 blocks of 128 x 64), K tiles (same), Vt tiles
// (2 blocks of dh x 64 keys), P (2 blocks of 128 x 64, aliased on Q when Q is >= 32 KB).
__host__ __device__ __forceinline__ size_t attn_q_bytes(int dh) { return (size_t)dh * kQT * 2; }
__host__ __device__ __forceinline__ size_t attn_p_extra(int dh) { return attn_q_bytes(dh) >= 32768 ? 0 : 32768; }

template <int DH>
__global__ void __launch_bounds__(128, 1) attn_tc_kernel(const __grid_constant__ CUtensorMap tq,
                                                         const __grid_constant__ CUtensorMap tk,
                                                         const __grid_constant__ CUtensorMap tv, AttnTcArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  constexpr int NC = DH / 64;
  constexpr uint32_t QB = DH * kQT * 2, KB = DH * kKT * 2, VB = DH * kKT * 2;
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + QB;
  uint8_t* sV = sK + KB;
  uint8_t* sP = attn_p_extra(DH) ? sV + VB : sQ;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + VB + attn_p_extra(DH));
  uint64_t *bar_qk = bars, *bar_v = bars + 1, *bar_s = bars + 2, *bar_o = bars + 3;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 4);

  const int qt = blockIdx.x, kc = blockIdx.y, bg = blockIdx.z;   // bg = b * Hkv + g
  const int b = bg / p.n_kv_heads, g = bg % p.n_kv_heads;
  const int kvz = (b * p.n_layers + p.layer) * p.n_kv_heads + g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(bars + i, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)), "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // S occupies columns [0, 128); O = P V reuses columns [0, DH) once every thread has read S
  const uint32_t tS = tmem, tO = tmem;
  pdl_trigger();
  pdl_wait();

  if (threadIdx.x == 0) {
    const uint64_t pol = policy_evict_last();
    mbar_expect_tx(bar_qk, QB + KB);
#pragma unroll
    for (int c = 0; c < NC; ++c) {
      tma_3d(sQ + c * (kQT * 128), &tq, c * 64, qt * kQT, bg, bar_qk, pol);
      tma_3d(sK + c * (kKT * 128), &tk, c * 64, kc * kKT, kvz, bar_qk, pol);
    }
    mbar_expect_tx(bar_v, VB);
#pragma unroll
    for (int u = 0; u < kKT / 64; ++u) tma_3d(sV + u * (DH * 128), &tv, kc * kKT + u * 64, 0, kvz, bar_v, pol);
  } else if (threadIdx.x == 32) {
    if (mbar_wait(bar_qk, 0, p.err, 21)) {
      tc_fence_after();
      const uint32_t q0 = su32(sQ), k0 = su32(sK);
#pragma unroll
      for (int c = 0; c < NC; ++c)
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16(tS, sw128_desc(q0 + c * (kQT * 128) + 32 * k), sw128_desc(k0 + c * (kKT * 128) + 32 * k),
                   idesc_m128(kKT), (c | k) ? 1u : 0u);
    }
    mma_commit(bar_s);
  }
  __syncwarp();

  // ---- softmax over this key chunk: one query row per thread ----
  const bool ok_s = mbar_wait(bar_s, 0, p.err, 22);
  tc_fence_after();
  const int row = warp * 32 + lane;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  const float c2 = p.scale_log2;             // log2(e) / sqrt(dh)
  const int key0 = kc * kKT;
  const int nv = p.n_keys - key0;            // valid keys of the chunk (all of them but in the last)
  float sv[kKT];                             // the chunk's scores of this row, one wait for all
  __syncwarp();
  tmem_ld128(tS + lane_base, sv);
  if (nv < kKT) {   // keys past the end (last chunk): excluded from the maximum, P = 2^-inf = 0
#pragma unroll
    for (int i = 0; i < kKT; ++i)
      if (i >= nv) sv[i] = -INFINITY;
  }
  float mx = -INFINITY;
#pragma unroll
  for (int i = 0; i < kKT; ++i) mx = fmaxf(mx, sv[i]);
  const float ms = mx * c2;
  float l = 0.f;
  const int r8 = row & 7;
#pragma unroll
  for (int cc = 0; cc < kKT / 32; ++cc) {
    uint32_t pk[16];
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      const int k = cc * 32 + i;
      const float e0 = ex2_fast(fmaf(sv[k], c2, -ms)), e1 = ex2_fast(fmaf(sv[k + 1], c2, -ms));
      const __nv_bfloat162 h = __floats2bfloat162_rn(e0, e1);
      const float2 hf = __bfloat1622float2(h);
      l += hf.x + hf.y;   // normalise by what the MMA actually sums
      pk[i / 2] = *reinterpret_cast<const uint32_t*>(&h);
    }
    // 32 keys = four 16-byte granules of row `row` in P block (cc / 2), granules (cc % 2) * 4 + q
    uint8_t* prow = sP + (cc / 2) * (kQT * 128) + row * 128;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int gidx = (cc % 2) * 4 + q;
      *reinterpret_cast<uint4*>(prow + ((gidx ^ r8) * 16)) = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
    }
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  tc_fence_before();
  __syncthreads();

  if (threadIdx.x == 32) {
    tc_fence_after();
    if (ok_s && mbar_wait(bar_v, 0, p.err, 23)) {
      const uint32_t p0 = su32(sP), v0 = su32(sV);
#pragma unroll
      for (int u = 0; u < kKT / 64; ++u)
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16(tO, sw128_desc(p0 + u * (kQT * 128) + 32 * k), sw128_desc(v0 + u * (DH * 128) + 32 * k),
                   idesc_m128(DH), (u | k) ? 1u : 0u);
    }
    mma_commit(bar_o);
  }
  __syncwarp();
  const bool ok_o = mbar_wait(bar_o, 0, p.err, 24);
  tc_fence_after();

  // ---- partial output row (unnormalised) + (max, sum): the row is staged in shared memory (all
  //      operand tiles are free once O is complete; rows padded by 16 bytes against bank
  //      conflicts) and written with one 1-KB bulk copy per row ----
  const int qrow = qt * kQT + row;
  const size_t prow_idx = ((size_t)bg * gridDim.y + kc) * p.r_pad + qrow;
  constexpr uint32_t pitch = DH * 4 + 16;
  uint8_t* srow = smem + (size_t)row * pitch;
  __syncwarp();
#pragma unroll
  for (int cc = 0; cc < DH / 32; ++cc) {
    tmem_ld32(tO + lane_base + cc * 32, sv);
#pragma unroll
    for (int i = 0; i < 32; i += 4)
      *reinterpret_cast<float4*>(srow + (cc * 32 + i) * 4) = make_float4(sv[i], sv[i + 1], sv[i + 2], sv[i + 3]);
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (ok_o && qrow < p.rows) {
    bulk_s2g(p.part_o + prow_idx * DH, srow, DH * 4);
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
    p.part_ml[prow_idx * 2] = mx;
    p.part_ml[prow_idx * 2 + 1] = l;
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

// ---- one-pass attention for many query tiles: no partials, no combine ---------------------
// One CTA per (128-row query tile, robot-group), keys in chunks of 128 (S = Q K^T with MMA
// N = 128). Shared memory: Q and a ring of five operand slots that take, in the order the MMAs
// read them, each chunk's K in head-dim pieces and its Vt in two 64-key halves; a slot is refilled
// as soon as the MMAs that read it are done, so the next chunk's operands load while S and P V of
// this one run. Per chunk: S on tcgen05 (double-buffered in TMEM), then each softmax thread (one
// query row) forms P = exp(S - M) in bf16 against its running maximum M and writes it into tensor
// memory over the S it came from, and O += P V accumulates in TMEM with P as the MMA's A operand
// from tensor memory (P is double-buffered with S). The issuer issues S of chunk c + 1 before
// P V of chunk c, so that it runs while the softmax of chunk c does. M is raised only when the
// chunk's maximum exceeds it by more than 2^8 in the exponent; the O row and the row sum are then
// rescaled in place (after the previous P V has completed). Otherwise the stale M stays: every P
// is at most 2^8, and O and the row sum share the same reference, so O / sum is unchanged. O / l
// is written in bf16.
constexpr int kKC2 = 128;                       // keys per chunk
constexpr uint32_t kTmem2 = 512;                // S buffers at columns [0,128) and [128,256), O at [256, 256 + DV)
constexpr float kRescaleLog2 = 8.f;             // raise M only past this many powers of two
constexpr int kSlots2 = 5;                      // operand ring slots
constexpr int kBars2 = 9 + 2 * kSlots2;         // mbarriers of the kernel
__host__ __device__ constexpr int attn2_kpieces(int dh) { return dh >= 128 ? 2 : 1; }
// ring slot bytes: a K piece (128 keys x dh / pieces) or a Vt half (dh x 64 keys), the larger
__host__ __device__ constexpr uint32_t attn2_slot_bytes(int dh) {
  return (uint32_t)(dh / attn2_kpieces(dh)) * kKC2 * 2 > (uint32_t)dh * 128 ? (uint32_t)(dh / attn2_kpieces(dh)) * kKC2 * 2
                                                                           : (uint32_t)dh * 128;
}

// Warps 0-3: softmax and output (they own the four TMEM lane quadrants); warp 4: TMA producer;
// warp 5: MMA issuer. The producer and issuer wait on the softmax warps' progress, so they must
// not share a warp with them. DV = head dims of O per CTA: DH, or DH / 2 when the query tiles are
// at most half as many as the SMs (two CTAs per tile, blockIdx.z = which half of the head dims;
// each computes S and P in full, and P V and the output for its half only).
template <int DH, int DV>
__global__ void __launch_bounds__(192, 1) attn_tc2_kernel(const __grid_constant__ CUtensorMap tq,
                                                          const __grid_constant__ CUtensorMap tk,
                                                          const __grid_constant__ CUtensorMap tv, AttnTcArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  constexpr int NC = DH / 64;
  constexpr int KP = attn2_kpieces(DH);          // K pieces per chunk
  constexpr int NCP = NC / KP;                   // 64-dim blocks of 128 keys per piece
  constexpr int PPC = KP + 2;                    // ring entries per chunk: K pieces, two Vt halves
  constexpr uint32_t QB = DH * kQT * 2;          // Q: NC blocks of 128 rows x 64
  constexpr uint32_t PB = NCP * kKC2 * 128;      // one K piece
  constexpr uint32_t VBLK = DV * 128;            // one Vt half: DV rows x 64 keys
  constexpr uint32_t SLOT = attn2_slot_bytes(DH);
  uint8_t* sQ = smem;
  uint8_t* sR = sQ + QB;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sR + kSlots2 * SLOT);
  uint64_t* q_full = bars;          // Q landed
  uint64_t* s_full = bars + 1;      // [2] S buffer written
  uint64_t* s_empty = bars + 3;     // [2] S / P buffer free (the P V that read its P is done)
  uint64_t* p_full = bars + 5;      // [2] P of the S buffer written (and O rescaled) by the 4 warps
  uint64_t* p_empty = bars + 7;     // P V done: O complete up to this chunk
  uint64_t* o_done = bars + 8;
  uint64_t* r_full = bars + 9;            // [kSlots2] ring slot loaded
  uint64_t* r_empty = r_full + kSlots2;   // [kSlots2] ring slot free (the MMAs that read it are done)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kBars2);

  const int qt = blockIdx.x, bg = blockIdx.y, d0 = blockIdx.z * DV;
  const int b = bg / p.n_kv_heads, g = bg % p.n_kv_heads;
  const int kvz = (b * p.n_layers + p.layer) * p.n_kv_heads + g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nck = (p.n_keys + kKC2 - 1) / kKC2;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full + i, 1);
      mbar_init(s_empty + i, 1);
      mbar_init(p_full + i, 4);
    }
    for (int i = 0; i < kSlots2; ++i) {
      mbar_init(r_full + i, 1);
      mbar_init(r_empty + i, 1);
    }
    mbar_init(p_empty, 1);
    mbar_init(o_done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)), "r"(kTmem2));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tO = tmem + 2 * kKC2;
  pdl_trigger();
  pdl_wait();

  // Ring entries in the order the MMAs read them: K of chunk 0, then per chunk c the K of chunk
  // c + 1 (S runs a chunk ahead of P V) and the Vt of chunk c.
  const auto k_entry = [&](int c, int j) { return c == 0 ? j : KP + (c - 1) * PPC + j; };
  const auto v_entry = [&](int c, int h) { return KP + c * PPC + (c + 1 < nck ? KP : 0) + h; };

  if (threadIdx.x == 128) {
    // producer: ring entry e into slot e % kSlots2 once entry e - kSlots2 has been read
    const uint64_t pol = policy_evict_last();
    mbar_expect_tx(q_full, QB);
#pragma unroll
    for (int c = 0; c < NC; ++c) tma_3d(sQ + c * (kQT * 128), &tq, c * 64, qt * kQT, bg, q_full, pol);
    int e = 0;
    bool ok = true;
    const auto slot = [&](int& t) {
      t = e % kSlots2;
      const int u = e / kSlots2;
      ++e;
      return u == 0 || mbar_wait(r_empty + t, (u - 1) & 1, p.err, 41);
    };
    const auto load_k = [&](int c) {
      for (int j = 0; j < KP && ok; ++j) {
        int t;
        if (!(ok = slot(t))) break;
        mbar_expect_tx(r_full + t, PB);
#pragma unroll
        for (int cc = 0; cc < NCP; ++cc)
          tma_3d(sR + t * SLOT + cc * (kKC2 * 128), &tk, (j * NCP + cc) * 64, c * kKC2, kvz, r_full + t, pol);
      }
    };
    load_k(0);
    for (int c = 0; c < nck && ok; ++c) {
      if (c + 1 < nck) load_k(c + 1);
      for (int h = 0; h < 2 && ok; ++h) {
        int t;
        if (!(ok = slot(t))) break;
        mbar_expect_tx(r_full + t, VBLK);
        tma_3d(sR + t * SLOT, &tv, c * kKC2 + h * 64, d0, kvz, r_full + t, pol);
      }
    }
  } else if (threadIdx.x == 160) {
    // issuer: S(0); per chunk c: S(c + 1), then P V(c) once the softmax warps have written P(c)
    bool ok = mbar_wait(q_full, 0, p.err, 42);
    const uint32_t q0 = su32(sQ), r0 = su32(sR);
    const auto issue_s = [&](int c) {
      const int sb = c & 1;
      if (c >= 2) ok = mbar_wait(s_empty + sb, ((c >> 1) - 1) & 1, p.err, 44);
      for (int j = 0; j < KP && ok; ++j) {
        const int e = k_entry(c, j), t = e % kSlots2;
        ok = mbar_wait(r_full + t, (e / kSlots2) & 1, p.err, 43);
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int cc = 0; cc < NCP; ++cc)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_bf16(tmem + sb * kKC2, sw128_desc(q0 + (j * NCP + cc) * (kQT * 128) + 32 * k),
                     sw128_desc(r0 + t * SLOT + cc * (kKC2 * 128) + 32 * k), idesc_m128(kKC2), (j | cc | k) ? 1u : 0u);
        mma_commit(r_empty + t);
      }
      if (ok) mma_commit(s_full + sb);
    };
    if (ok) issue_s(0);
    for (int ch = 0; ch < nck && ok; ++ch) {
      const int sb = ch & 1;
      if (ch + 1 < nck) issue_s(ch + 1);
      ok = ok && mbar_wait(p_full + sb, (ch >> 1) & 1, p.err, 45);
      for (int h = 0; h < 2 && ok; ++h) {
        const int e = v_entry(ch, h), t = e % kSlots2;
        ok = mbar_wait(r_full + t, (e / kSlots2) & 1, p.err, 46);
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16_ts(tO, tmem + sb * kKC2 + 8 * (4 * h + k), sw128_desc(r0 + t * SLOT + 32 * k), idesc_m128(DV),
                      (ch | h | k) ? 1u : 0u);
        mma_commit(r_empty + t);
      }
      if (!ok) break;
      mma_commit(p_empty);
      mma_commit(s_empty + sb);
    }
    mma_commit(o_done);
  }
  if (warp >= 4) {
    // producer / issuer warps: done issuing; wait for the output stage before releasing TMEM
    __syncthreads();
    return;
  }

  // ---- softmax warps: one query row per thread ----
  const int row = warp * 32 + lane;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  const float c2s = p.scale_log2;
  float sv[kKC2];                    // the chunk's scores of this row
  float mref = -INFINITY, l = 0.f;   // the row's reference maximum and sum of P
  bool ok = true;
  for (int ch = 0; ch < nck; ++ch) {
    const int sb = ch & 1;
    const int key0 = ch * kKC2;
    const int nv = p.n_keys - key0;   // valid keys of the chunk (all of them but in the last)
    ok = ok && mbar_wait(s_full + sb, (ch >> 1) & 1, p.err, 47);
    tc_fence_after();
    __syncwarp();
    tmem_ld128(tmem + sb * kKC2 + lane_base, sv);
    if (nv < kKC2) {   // keys past the end (last chunk): excluded from the maximum, P = 2^-inf = 0
#pragma unroll
      for (int i = 0; i < kKC2; ++i)
        if (i >= nv) sv[i] = -INFINITY;
    }
    float mx[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) mx[j] = sv[j];
#pragma unroll
    for (int i = 8; i < kKC2; ++i) mx[i & 7] = fmaxf(mx[i & 7], sv[i]);
    const float mc = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
    // raise the reference past 2^8 (and at the first chunk); the previous P V must have completed
    // before O is touched (P goes to this chunk's own buffer, free since S landed in it)
    const bool raise = ch == 0 ? true : (mc - mref) * c2s > kRescaleLog2;
    const float factor = ch == 0 ? 1.f : (raise ? exp2f((mref - mc) * c2s) : 1.f);
    if (__any_sync(0xffffffffu, ch > 0 && raise)) {
      ok = ok && mbar_wait(p_empty, (ch - 1) & 1, p.err, 48);
      tc_fence_after();
      float ov[32];
#pragma unroll 1
      for (int cc = 0; cc < DV / 32; ++cc) {
        tmem_ld32(tO + lane_base + cc * 32, ov);
#pragma unroll
        for (int i = 0; i < 32; ++i) ov[i] *= factor;
        tmem_st32(tO + lane_base + cc * 32, ov);
      }
    }
    if (raise) {
      l *= factor;
      mref = mc;
    }
    const float ms = mref * c2s;
    float la = 0.f, lb = 0.f;
#pragma unroll
    for (int cc = 0; cc < kKC2 / 32; ++cc) {
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        const int k = cc * 32 + i;
        const float e0 = ex2_fast(fmaf(sv[k], c2s, -ms)), e1 = ex2_fast(fmaf(sv[k + 1], c2s, -ms));
        const __nv_bfloat162 h = __floats2bfloat162_rn(e0, e1);
        const float2 hf = __bfloat1622float2(h);
        la += hf.x;   // normalise by what the MMA sums
        lb += hf.y;
        pk[i / 2] = *reinterpret_cast<const uint32_t*>(&h);
      }
      // keys 32 cc .. 32 cc + 31 -> columns 16 cc .. + 15 of the chunk's S buffer (its scores are
      // in registers)
      tmem_st16_nowait(tmem + sb * kKC2 + lane_base + 16 * cc, pk);
    }
    l += la + lb;
    tmem_wait_st();
    // (p_full of this S buffer completes again only after S of chunk ch + 2, which the issuer
    // issues after its wait for this phase)
    tc_fence_before();
    __syncwarp();
    if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(p_full + sb)) : "memory");
  }
  float sv32[32];
  ok = ok && mbar_wait(o_done, 0, p.err, 49);
  tc_fence_after();
  __syncwarp();

  // ---- o = O / l in bf16, row (j, i) of this tile -> o[(b*H + i)][(g*G + j)*dh + d] ----
  const int qrow = qt * kQT + row;
  const float inv = 1.f / l;
  const int jj = qrow / p.H, ii = qrow % p.H;
  __nv_bfloat16* orow = p.out + ((size_t)b * p.H + ii) * p.out_ld + (size_t)(g * p.group + jj) * DH + d0;
#pragma unroll
  for (int cc = 0; cc < DV / 32; ++cc) {
    tmem_ld32(tO + lane_base + cc * 32, sv32);
    if (ok && qrow < p.rows) {
#pragma unroll
      for (int i = 0; i < 32; i += 8) {
        uint4 w;
        w.x = pack_bf16(sv32[i] * inv, sv32[i + 1] * inv);
        w.y = pack_bf16(sv32[i + 2] * inv, sv32[i + 3] * inv);
        w.z = pack_bf16(sv32[i + 4] * inv, sv32[i + 5] * inv);
        w.w = pack_bf16(sv32[i + 6] * inv, sv32[i + 7] * inv);
        *reinterpret_cast<uint4*>(orow + cc * 32 + i) = w;
      }
    }
  }
  tc_fence_before();
  __syncthreads();   // pairs with the producer / issuer warps' final barrier
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmem2));
}

// Merge the key chunks of every query row: o = sum_c w_c O_c / sum_c w_c l_c, w_c = 2^((m_c - M) c2).
// One CTA per (query row, robot-group), one thread per two head dims (dh / 2 threads: the grid
// fits the GPU in one wave, 8-byte loads); every partial is loaded before any arithmetic. Writes
// o [(b*H + i)][(g*G + j)*dh + d] in bf16.
__global__ void attn_combine_kernel(AttnTcArgs p, int n_chunks) {
  constexpr int MAXC = kMaxKeyChunks;
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x, bg = blockIdx.y, d = 2 * threadIdx.x, DH = 2 * blockDim.x;
  const int b = bg / p.n_kv_heads, g = bg % p.n_kv_heads;
  float m[MAXC], l[MAXC];
  float2 o[MAXC];
#pragma unroll
  for (int c = 0; c < MAXC; ++c) {
    if (c < n_chunks) {
      const size_t idx = ((size_t)bg * n_chunks + c) * p.r_pad + r;
      m[c] = p.part_ml[idx * 2];
      l[c] = p.part_ml[idx * 2 + 1];
      o[c] = *reinterpret_cast<const float2*>(p.part_o + idx * DH + d);
    }
  }
  float M = -INFINITY;
#pragma unroll
  for (int c = 0; c < MAXC; ++c)
    if (c < n_chunks) M = fmaxf(M, m[c]);
  float L = 0.f, ax = 0.f, ay = 0.f;
#pragma unroll
  for (int c = 0; c < MAXC; ++c) {
    if (c < n_chunks) {
      const float w = exp2f((m[c] - M) * p.scale_log2);
      L = fmaf(w, l[c], L);
      ax = fmaf(w, o[c].x, ax);
      ay = fmaf(w, o[c].y, ay);
    }
  }
  const int j = r / p.H, i = r % p.H;
  *reinterpret_cast<__nv_bfloat162*>(p.out + ((size_t)b * p.H + i) * p.out_ld + (size_t)(g * p.group + j) * DH + d) =
      __floats2bfloat162_rn(ax / L, ay / L);
}

// Prefix K/V of one robot (fp32 or bf16 source [L][P][Hkv][dh]) into the K and Vt caches.
__global__ void kv_prefix_kernel(const void* k, const void* v, int src_dt, AttnTcArgs p, int robot) {
  const int dh = p.head_dim;
  const long long n = (long long)p.n_layers * p.prefix * p.n_kv_heads * dh;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n; e += (long long)gridDim.x * blockDim.x) {
    const int d = (int)(e % dh);
    const int g = (int)((e / dh) % p.n_kv_heads);
    const int pp = (int)((e / ((long long)dh * p.n_kv_heads)) % p.prefix);
    const int l = (int)(e / ((long long)dh * p.n_kv_heads * p.prefix));
    const float kv = src_dt == BF16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(k)[e]) : static_cast<const float*>(k)[e];
    const float vv = src_dt == BF16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(v)[e]) : static_cast<const float*>(v)[e];
    const size_t z = ((size_t)robot * p.n_layers + l) * p.n_kv_heads + g;
    p.kcache[(z * p.n_keys + pp) * dh + d] = __float2bfloat16_rn(kv);
    p.vtcache[(z * dh + d) * p.nk_pad + pp] = __float2bfloat16_rn(vv);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* q = nullptr;
    cudaDriverEntryPointQueryResult r;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &q, 12000, cudaEnableDefault, &r) ==
            cudaSuccess && r == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(q);
  }
  return fn;
}

int tmap3(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1, uint64_t s2,
          uint32_t b0, uint32_t b1) {
  auto enc = encoder();
  if (!enc) return -1;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {s1, s2};
  const cuuint32_t box[3] = {b0, b1, 1};
  const cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS ? 0 : -2;
}

}  // namespace

size_t attn_tc2_smem_bytes(int dh) {
  return 1024 + (size_t)dh * kQT * 2 + (size_t)kSlots2 * attn2_slot_bytes(dh) + (kBars2 + 1) * 8;
}

bool attn_tc_use_two_pass(const AttnTcArgs& a) {
  const int tiles = (a.rows + kQT - 1) / kQT * a.batch * a.n_kv_heads;
  return tiles >= 64;
}

size_t attn_tc_smem_bytes(int dh) {
  const size_t tiles = 3 * attn_q_bytes(dh) + attn_p_extra(dh);
  const size_t ostage = (size_t)kQT * (dh * 4 + 16);   // O rows staged over the free operand tiles
  return 1024 + (tiles > ostage ? tiles : ostage) + 4 * 8 + 16;
}

int attn_tc_prepare(AttnTcMaps* maps, const AttnTcArgs& a, int batch_max) {
  const int dh = a.head_dim;
  const uint64_t R = a.rows, NK = a.n_keys, NKp = a.nk_pad;
  if (tmap3(&maps->q, a.q, dh, R, (uint64_t)batch_max * a.n_kv_heads, (uint64_t)dh * 2, R * dh * 2, 64, kQT)) return -1;
  if (tmap3(&maps->k, a.kcache, dh, NK, (uint64_t)batch_max * a.n_layers * a.n_kv_heads, (uint64_t)dh * 2,
            NK * dh * 2, 64, kKT)) return -1;
  if (tmap3(&maps->vt, a.vtcache, NK, dh, (uint64_t)batch_max * a.n_layers * a.n_kv_heads, NKp * 2,
            (uint64_t)dh * NKp * 2, 64, (uint32_t)dh)) return -1;
  // 64-key K boxes for the persistent step kernel's attention items; the one-pass kernel loads
  // 128-key K chunks through `k` and Vt in 64-key boxes
  if (tmap3(&maps->k2, a.kcache, dh, NK, (uint64_t)batch_max * a.n_layers * a.n_kv_heads, (uint64_t)dh * 2,
            NK * dh * 2, 64, 64)) return -1;
  // Vt boxes of half the head dims for the one-pass kernel's split form
  if (dh >= 128) {
    if (tmap3(&maps->vt2, a.vtcache, NK, dh, (uint64_t)batch_max * a.n_layers * a.n_kv_heads, NKp * 2,
              (uint64_t)dh * NKp * 2, 64, (uint32_t)dh / 2)) return -1;
  } else {
    maps->vt2 = maps->vt;
  }
  const int smem2 = (int)attn_tc2_smem_bytes(dh);
  if (dh == 64) cudaFuncSetAttribute(attn_tc2_kernel<64, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
  if (dh == 128) {
    cudaFuncSetAttribute(attn_tc2_kernel<128, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
    cudaFuncSetAttribute(attn_tc2_kernel<128, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
  }
  if (dh == 256) {
    cudaFuncSetAttribute(attn_tc2_kernel<256, 256>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
    cudaFuncSetAttribute(attn_tc2_kernel<256, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
  }
  const int smem = (int)attn_tc_smem_bytes(dh);
  if (dh == 64) cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (dh == 128) cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (dh == 256) cudaFuncSetAttribute(attn_tc_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  return 0;
}

int attn_tc_chunks(int n_keys) { return (n_keys + kKT - 1) / kKT; }
int attn_tc_max_keys() { return kMaxKeyChunks * kKT; }
int attn_tc_rpad(int rows) { return (rows + kQT - 1) / kQT * kQT; }

void launch_attn_tc(const AttnTcMaps& maps, const AttnTcArgs& a, cudaStream_t s) {
  if (attn_tc_use_two_pass(a)) {
    const int tiles = (a.rows + kQT - 1) / kQT * a.batch * a.n_kv_heads;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const bool split = a.head_dim >= 128 && 2 * tiles <= sms;
    dim3 grid2((a.rows + kQT - 1) / kQT, a.batch * a.n_kv_heads, split ? 2 : 1);
    const size_t smem2 = attn_tc2_smem_bytes(a.head_dim);
    if (a.head_dim == 64) launch_k(attn_tc2_kernel<64, 64>, grid2, dim3(192), smem2, s, maps.q, maps.k, maps.vt, a);
    if (a.head_dim == 128) {
      if (split) launch_k(attn_tc2_kernel<128, 64>, grid2, dim3(192), smem2, s, maps.q, maps.k, maps.vt2, a);
      else launch_k(attn_tc2_kernel<128, 128>, grid2, dim3(192), smem2, s, maps.q, maps.k, maps.vt, a);
    }
    if (a.head_dim == 256) {
      if (split) launch_k(attn_tc2_kernel<256, 128>, grid2, dim3(192), smem2, s, maps.q, maps.k, maps.vt2, a);
      else launch_k(attn_tc2_kernel<256, 256>, grid2, dim3(192), smem2, s, maps.q, maps.k, maps.vt, a);
    }
    return;
  }
  dim3 grid((a.rows + kQT - 1) / kQT, attn_tc_chunks(a.n_keys), a.batch * a.n_kv_heads);
  const size_t smem = attn_tc_smem_bytes(a.head_dim);
  if (a.head_dim == 64) launch_k(attn_tc_kernel<64>, grid, dim3(128), smem, s, maps.q, maps.k, maps.vt, a);
  if (a.head_dim == 128) launch_k(attn_tc_kernel<128>, grid, dim3(128), smem, s, maps.q, maps.k, maps.vt, a);
  if (a.head_dim == 256) launch_k(attn_tc_kernel<256>, grid, dim3(128), smem, s, maps.q, maps.k, maps.vt, a);
  launch_k(attn_combine_kernel, dim3(a.rows, a.batch * a.n_kv_heads), dim3(a.head_dim / 2), 0, s, a,
           attn_tc_chunks(a.n_keys));
}

void launch_kv_prefix(const void* k, const void* v, int src_dtype, const AttnTcArgs& a, int robot, cudaStream_t s) {
  kv_prefix_kernel<<<1024, 256, 0, s>>>(k, v, src_dtype, a, robot);
}

}  // namespace uad
