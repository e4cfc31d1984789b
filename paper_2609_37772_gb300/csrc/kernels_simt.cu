// CUDA-core kernels: fp32-FFMA GEMM (the fp32 mode and one-time table fills), adaptive
// norms, attention over prefix + chunk, and the Euler / TR / release / GAC step epilogue.
#include "uad_internal.cuh"
#include "euler.cuh"

namespace uad {

bool pdl_enabled() {
  static int on = -1;
  if (on < 0) {
    const char* e = getenv("UAD_PDL");
    on = !(e && e[0] == '0');
  }
  return on != 0;
}

// ------------------------------------------------------------------------------------------
// small helpers
// ------------------------------------------------------------------------------------------
template <int DT>
__device__ __forceinline__ float ldf(const void* p, long long i) {
  if constexpr (DT == BF16) return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
  else return static_cast<const float*>(p)[i];
}
__device__ __forceinline__ float ldf_rt(const void* p, long long i, int dt) {
  return dt == BF16 ? ldf<BF16>(p, i) : ldf<F32>(p, i);
}
__device__ __forceinline__ void stf(void* p, long long i, float v, int dt) {
  if (dt == BF16) static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
  else static_cast<float*>(p)[i] = v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float gelu_tanh(float x) {
  const float k0 = 0.7978845608028654f;  // sqrt(2/pi)
  return 0.5f * x * (1.f + tanhf(k0 * (x + 0.044715f * x * x * x)));
}
__device__ __forceinline__ float silu(float x) { return x / (1.f + expf(-x)); }
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------------------------------------
// GEMM: out[m][n] = epi(sum_k A[m][k] * Wt[n][k]); 64x64 tile, 4x4 outputs per thread, k in
// ascending order (deterministic).
// ------------------------------------------------------------------------------------------
template <int AD, int WD>
__global__ void __launch_bounds__(256) gemm_simt_kernel(GemmArgs p) {
  __shared__ float As[32][68];
  __shared__ float Ws[32][68];
  pdl_trigger();
  pdl_wait();
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < p.K; k0 += 32) {
    for (int e = tid; e < 64 * 32; e += 256) {
      const int r = e >> 5, c = e & 31, k = k0 + c;
      const int m = m0 + r, n = n0 + r;
      As[c][r] = (m < p.M && k < p.K) ? ldf<AD>(p.A, (long long)m * p.lda + k) : 0.f;
      Ws[c][r] = (n < p.N && k < p.K) ? ldf<WD>(p.W, (long long)n * p.K + k) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < 32; ++kk) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) w[j] = Ws[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }

#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= p.M) continue;
    if (p.epi == EPI_GEGLU) {
#pragma unroll
      for (int jp = 0; jp < 2; ++jp) {
        const int n = n0 + tx * 4 + 2 * jp;
        if (n + 1 < p.N)
          stf(p.out, (long long)m * p.ldo + n / 2, gelu_tanh(acc[i][2 * jp]) * acc[i][2 * jp + 1],
              p.out_dtype);
      }
      continue;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= p.N) continue;
      float r = acc[i][j] + (p.bias ? p.bias[n] : 0.f);
      switch (p.epi) {
        case EPI_STORE:
          if (p.add_rows) r += p.add_rows[(long long)(m % p.add_mod) * p.N + n];
          stf(p.out, (long long)m * p.ldo + n, r, p.out_dtype);
          break;
        case EPI_BIAS_SILU: stf(p.out, (long long)m * p.ldo + n, silu(r), p.out_dtype); break;
        case EPI_BIAS_GELU: stf(p.out, (long long)m * p.ldo + n, gelu_tanh(r), p.out_dtype); break;
        case EPI_RESID_GATE: {
          const float gt = p.gate_tab ? p.gate_tab[(long long)p.tau_row[m] * p.gate_stride + n] : 1.f;
          float* dst = p.resid + (long long)m * p.ldr + n;
          *dst = fmaf(gt, r, *dst);
          break;
        }
        default: break;
      }
    }
  }
}

// Projections with a tiny side (action in: K = D; action out: N = D): one CTA per token row m,
// the row staged in shared memory, then one warp per output (long K) or one thread per output
// (short K). out[m][n] = sum_k A[m][k] Wt[n][k] + bias[n] (+ add_rows[m % add_mod][n]), fp32.
template <int AD, int WD>
__global__ void __launch_bounds__(256) gemv_rows_kernel(GemmArgs p) {
  __shared__ float a_s[kGemvMaxK];
  pdl_trigger();
  pdl_wait();
  const int m = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int k = tid; k < p.K; k += 256) a_s[k] = ldf<AD>(p.A, (long long)m * p.lda + k);
  __syncthreads();
  float* out = static_cast<float*>(p.out) + (long long)m * p.ldo;
  const float* add = p.add_rows ? p.add_rows + (long long)(m % p.add_mod) * p.N : nullptr;
  if (p.K <= 64) {
    for (int n = tid; n < p.N; n += 256) {
      float acc = 0.f;
      for (int k = 0; k < p.K; ++k) acc = fmaf(a_s[k], ldf<WD>(p.W, (long long)n * p.K + k), acc);
      out[n] = acc + (p.bias ? p.bias[n] : 0.f) + (add ? add[n] : 0.f);
    }
  } else {
    for (int n = warp; n < p.N; n += 8) {
      float acc = 0.f;
#pragma unroll 8
      for (int k = lane; k < p.K; k += 32) acc = fmaf(a_s[k], ldf<WD>(p.W, (long long)n * p.K + k), acc);
      acc = warp_sum(acc);
      if (lane == 0) out[n] = acc + (p.bias ? p.bias[n] : 0.f) + (add ? add[n] : 0.f);
    }
  }
}

bool gemv_rows_ok(const GemmArgs& a) {
  return a.epi == EPI_STORE && a.out_dtype == F32 && a.K <= kGemvMaxK && (a.N <= 64 || a.K <= 64);
}

void launch_gemv_rows(const GemmArgs& a, cudaStream_t s) {
  if (a.a_dtype == F32 && a.w_dtype == F32) launch_k(gemv_rows_kernel<F32, F32>, dim3(a.M), dim3(256), 0, s, a);
  else if (a.a_dtype == F32 && a.w_dtype == BF16) launch_k(gemv_rows_kernel<F32, BF16>, dim3(a.M), dim3(256), 0, s, a);
  else if (a.a_dtype == BF16 && a.w_dtype == BF16) launch_k(gemv_rows_kernel<BF16, BF16>, dim3(a.M), dim3(256), 0, s, a);
  else launch_k(gemv_rows_kernel<BF16, F32>, dim3(a.M), dim3(256), 0, s, a);
}

void launch_gemm_simt(const GemmArgs& a, cudaStream_t s) {
  dim3 grid((a.N + 63) / 64, (a.M + 63) / 64);
  if (a.a_dtype == F32 && a.w_dtype == F32) launch_k(gemm_simt_kernel<F32, F32>, grid, dim3(256), 0, s, a);
  else if (a.a_dtype == F32 && a.w_dtype == BF16) launch_k(gemm_simt_kernel<F32, BF16>, grid, dim3(256), 0, s, a);
  else if (a.a_dtype == BF16 && a.w_dtype == BF16) launch_k(gemm_simt_kernel<BF16, BF16>, grid, dim3(256), 0, s, a);
  else launch_k(gemm_simt_kernel<BF16, F32>, grid, dim3(256), 0, s, a);
}

// ------------------------------------------------------------------------------------------
// Adaptive norm: y = norm(h) * (1 + scale[tau]) + shift[tau]; one warp per token row.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) norm_kernel(NormArgs p) {
  pdl_trigger();
  pdl_wait();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= p.M) return;
  const float* r = p.h + (long long)row * p.ldh;
  float mean = 0.f;
  if (p.layer_norm) {
    float s = 0.f;
    for (int c = lane; c < p.W; c += 32) s += r[c];
    mean = warp_sum(s) / p.W;
  }
  float ss = 0.f;
  for (int c = lane; c < p.W; c += 32) {
    const float d = r[c] - mean;
    ss = fmaf(d, d, ss);
  }
  const float rstd = 1.f / sqrtf(warp_sum(ss) / p.W + 1e-6f);
  const float* mod = p.tab ? p.tab + (long long)p.tau_row[row] * p.stride : nullptr;
  for (int c = lane; c < p.W; c += 32) {
    float y = (r[c] - mean) * rstd;
    if (mod) y = fmaf(y, 1.f + mod[p.scale_off + c], mod[p.shift_off + c]);
    stf(p.out, (long long)row * p.ldo + c, y, p.out_dtype);
  }
}

// Same computation with the whole row held in registers (W = 128 * NV): every load of the row
// and of its modulation vectors is issued before any arithmetic, so a row costs two memory
// round trips (modulation-row index, then data) instead of one per 32 elements.
template <int NV>
__global__ void __launch_bounds__(256) norm_reg_kernel(NormArgs p) {
  pdl_trigger();
  pdl_wait();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= p.M) return;
  const float4* r4 = reinterpret_cast<const float4*>(p.h + (long long)row * p.ldh);
  const float* mod = p.tab ? p.tab + (long long)p.tau_row[row] * p.stride : nullptr;
  float4 x[NV], sc[NV], sh[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) x[i] = r4[i * 32 + lane];
  if (mod) {
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      sc[i] = __ldg(reinterpret_cast<const float4*>(mod + p.scale_off) + i * 32 + lane);
      sh[i] = __ldg(reinterpret_cast<const float4*>(mod + p.shift_off) + i * 32 + lane);
    }
  }
  float mean = 0.f;
  if (p.layer_norm) {
    float t = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) t += (x[i].x + x[i].y) + (x[i].z + x[i].w);
    mean = warp_sum(t) / p.W;
  }
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const float a = x[i].x - mean, b = x[i].y - mean, c = x[i].z - mean, d = x[i].w - mean;
    ss = fmaf(a, a, fmaf(b, b, fmaf(c, c, fmaf(d, d, ss))));
  }
  const float rstd = 1.f / sqrtf(warp_sum(ss) / p.W + 1e-6f);
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    float4 y = make_float4((x[i].x - mean) * rstd, (x[i].y - mean) * rstd, (x[i].z - mean) * rstd,
                           (x[i].w - mean) * rstd);
    if (mod) {
      y.x = fmaf(y.x, 1.f + sc[i].x, sh[i].x);
      y.y = fmaf(y.y, 1.f + sc[i].y, sh[i].y);
      y.z = fmaf(y.z, 1.f + sc[i].z, sh[i].z);
      y.w = fmaf(y.w, 1.f + sc[i].w, sh[i].w);
    }
    const long long off = (long long)row * p.ldo + (i * 32 + lane) * 4;
    if (p.out_dtype == BF16) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(y.x, y.y), hi = __floats2bfloat162_rn(y.z, y.w);
      uint2 pk;
      pk.x = *reinterpret_cast<uint32_t*>(&lo);
      pk.y = *reinterpret_cast<uint32_t*>(&hi);
      *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.out) + off) = pk;
    } else {
      *reinterpret_cast<float4*>(static_cast<float*>(p.out) + off) = y;
    }
  }
}

// Residual update + adaptive norm, one CTA per token row, 4 columns per thread:
//   h += gate(tau) * (sum_s part[s] + bias);  y = norm(h) * (1 + scale[tau]) + shift[tau].
// The K-split partial planes are summed in plane order (deterministic); all of a thread's
// loads are issued before the arithmetic that needs them.
__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  __syncthreads();                       // red[] may still be read by the previous call
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < nw; ++i) t += red[i];
  return t;
}

__global__ void __launch_bounds__(1024) resid_norm_kernel(NormArgs p) {
  __shared__ float red[32];
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x, c4 = threadIdx.x;
  const bool on = c4 * 4 < p.W;
  const int tr = p.tau_row[row];
  float4 x = make_float4(0.f, 0.f, 0.f, 0.f), sc = x, sh = x, gt = make_float4(1.f, 1.f, 1.f, 1.f), bs = x;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float4* h4 = reinterpret_cast<float4*>(p.h + (long long)row * p.ldh) + c4;
  if (on) {
    x = *h4;
    const float* mod = p.tab ? p.tab + (long long)tr * p.stride : nullptr;
    if (mod) {
      sc = __ldg(reinterpret_cast<const float4*>(mod + p.scale_off) + c4);
      sh = __ldg(reinterpret_cast<const float4*>(mod + p.shift_off) + c4);
    }
    if (p.rgate_tab) gt = __ldg(reinterpret_cast<const float4*>(p.rgate_tab + (long long)tr * p.stride + p.rgate_off) + c4);
    if (p.rbias) bs = __ldg(reinterpret_cast<const float4*>(p.rbias) + c4);
    const long long plane4 = (long long)p.M * p.W / 4;
    const float4* pp = reinterpret_cast<const float4*>(p.part + (long long)row * p.W) + c4;
    int i = 0;
    for (; i + 8 <= p.n_part; i += 8) {
      float4 q[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) q[u] = __ldcg(pp + (i + u) * plane4);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        acc.x += q[u].x; acc.y += q[u].y; acc.z += q[u].z; acc.w += q[u].w;
      }
    }
    for (; i < p.n_part; ++i) {
      const float4 q = __ldcg(pp + i * plane4);
      acc.x += q.x; acc.y += q.y; acc.z += q.z; acc.w += q.w;
    }
    x.x = fmaf(gt.x, acc.x + bs.x, x.x);
    x.y = fmaf(gt.y, acc.y + bs.y, x.y);
    x.z = fmaf(gt.z, acc.z + bs.z, x.z);
    x.w = fmaf(gt.w, acc.w + bs.w, x.w);
    *h4 = x;
  }
  float mean = 0.f;
  if (p.layer_norm) mean = block_sum(on ? (x.x + x.y) + (x.z + x.w) : 0.f, red) / p.W;
  const float a = x.x - mean, b = x.y - mean, c = x.z - mean, d = x.w - mean;
  const float ss = block_sum(on ? fmaf(a, a, fmaf(b, b, fmaf(c, c, d * d))) : 0.f, red);
  const float rstd = 1.f / sqrtf(ss / p.W + 1e-6f);
  if (!on) return;
  float4 y = make_float4(a * rstd, b * rstd, c * rstd, d * rstd);
  if (p.tab) {
    y.x = fmaf(y.x, 1.f + sc.x, sh.x);
    y.y = fmaf(y.y, 1.f + sc.y, sh.y);
    y.z = fmaf(y.z, 1.f + sc.z, sh.z);
    y.w = fmaf(y.w, 1.f + sc.w, sh.w);
  }
  const long long off = (long long)row * p.ldo + c4 * 4;
  if (p.out_dtype == BF16) {
    __nv_bfloat162 lo = __floats2bfloat162_rn(y.x, y.y), hi = __floats2bfloat162_rn(y.z, y.w);
    uint2 pk;
    pk.x = *reinterpret_cast<uint32_t*>(&lo);
    pk.y = *reinterpret_cast<uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.out) + off) = pk;
  } else {
    *reinterpret_cast<float4*>(static_cast<float*>(p.out) + off) = y;
  }
}

// The same with one warp per token row and the whole row in registers (W = 128 * NV): the row's
// h, planes and gate are loaded before the arithmetic that needs them, and its sums are warp
// reductions (no CTA barrier); the scale and shift vectors are loaded after the reduction, so
// that a thread holds three row-sized arrays at most and four-warp CTAs fit three or four to an
// SM (more rows in flight). The planes are summed in plane order as above.
template <int NV>
__global__ void __launch_bounds__(128) resid_norm_reg_kernel(NormArgs p) {
  pdl_trigger();
  pdl_wait();
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= p.M) return;
  const int tr = p.tau_row[row];
  float4* h4 = reinterpret_cast<float4*>(p.h + (long long)row * p.ldh);
  const float4* pp = reinterpret_cast<const float4*>(p.part + (long long)row * p.W);
  const long long plane4 = (long long)p.M * p.W / 4;
  const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f), one = make_float4(1.f, 1.f, 1.f, 1.f);
  float4 x[NV], acc[NV], gt[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    x[i] = h4[i * 32 + lane];
    acc[i] = p.n_part > 0 ? __ldcg(pp + i * 32 + lane) : zero;
  }
  const float* mod = p.tab ? p.tab + (long long)tr * p.stride : nullptr;
  const float4* g4 = p.rgate_tab ? reinterpret_cast<const float4*>(p.rgate_tab + (long long)tr * p.stride + p.rgate_off) : nullptr;
#pragma unroll
  for (int i = 0; i < NV; ++i) gt[i] = g4 ? __ldg(g4 + i * 32 + lane) : one;
  for (int sp = 1; sp < p.n_part; ++sp) {
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      const float4 q = __ldcg(pp + sp * plane4 + i * 32 + lane);
      acc[i].x += q.x;
      acc[i].y += q.y;
      acc[i].z += q.z;
      acc[i].w += q.w;
    }
  }
  float t = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const float4 bs = p.rbias ? __ldg(reinterpret_cast<const float4*>(p.rbias) + i * 32 + lane) : zero;
    x[i].x = fmaf(gt[i].x, acc[i].x + bs.x, x[i].x);
    x[i].y = fmaf(gt[i].y, acc[i].y + bs.y, x[i].y);
    x[i].z = fmaf(gt[i].z, acc[i].z + bs.z, x[i].z);
    x[i].w = fmaf(gt[i].w, acc[i].w + bs.w, x[i].w);
    h4[i * 32 + lane] = x[i];
    t += (x[i].x + x[i].y) + (x[i].z + x[i].w);
  }
  const float mean = p.layer_norm ? warp_sum(t) / p.W : 0.f;
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    const float a = x[i].x - mean, b = x[i].y - mean, c = x[i].z - mean, d = x[i].w - mean;
    ss = fmaf(a, a, fmaf(b, b, fmaf(c, c, fmaf(d, d, ss))));
  }
  const float rstd = 1.f / sqrtf(warp_sum(ss) / p.W + 1e-6f);
  float4 sc[NV], sh[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    sc[i] = mod ? __ldg(reinterpret_cast<const float4*>(mod + p.scale_off) + i * 32 + lane) : zero;
    sh[i] = mod ? __ldg(reinterpret_cast<const float4*>(mod + p.shift_off) + i * 32 + lane) : zero;
  }
#pragma unroll
  for (int i = 0; i < NV; ++i) {
    float4 y = make_float4((x[i].x - mean) * rstd, (x[i].y - mean) * rstd, (x[i].z - mean) * rstd,
                           (x[i].w - mean) * rstd);
    if (mod) {
      y.x = fmaf(y.x, 1.f + sc[i].x, sh[i].x);
      y.y = fmaf(y.y, 1.f + sc[i].y, sh[i].y);
      y.z = fmaf(y.z, 1.f + sc[i].z, sh[i].z);
      y.w = fmaf(y.w, 1.f + sc[i].w, sh[i].w);
    }
    const long long off = (long long)row * p.ldo + (i * 32 + lane) * 4;
    if (p.out_dtype == BF16) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(y.x, y.y), hi = __floats2bfloat162_rn(y.z, y.w);
      uint2 pk;
      pk.x = *reinterpret_cast<uint32_t*>(&lo);
      pk.y = *reinterpret_cast<uint32_t*>(&hi);
      *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.out) + off) = pk;
    } else {
      *reinterpret_cast<float4*>(static_cast<float*>(p.out) + off) = y;
    }
  }
}

void launch_norm(const NormArgs& a, cudaStream_t s) {
  if (a.part) {
    const bool aligned = a.ldh % 4 == 0 && a.ldo % 4 == 0 && a.scale_off % 4 == 0 && a.shift_off % 4 == 0 &&
                         a.rgate_off % 4 == 0 && a.stride % 4 == 0 && a.W % 128 == 0;
    const int blocks = (a.M + 3) / 4;
    // a warp per row pays with enough rows to fill the SMs; with fewer, one CTA per row
    switch (aligned && a.M >= 512 ? a.W / 128 : 0) {
      case 2: launch_k(resid_norm_reg_kernel<2>, dim3(blocks), dim3(128), 0, s, a); return;
      case 4: launch_k(resid_norm_reg_kernel<4>, dim3(blocks), dim3(128), 0, s, a); return;
      case 8: launch_k(resid_norm_reg_kernel<8>, dim3(blocks), dim3(128), 0, s, a); return;
      default: break;
    }
    // the caller guarantees 16-byte rows: W, ldh, ldo, stride and the offsets multiples of 4
    const int threads = ((a.W / 4 + 31) / 32) * 32;
    launch_k(resid_norm_kernel, dim3(a.M), dim3(threads), 0, s, a);
    return;
  }
  const int blocks = (a.M + 7) / 8;
  const bool aligned = a.ldh % 4 == 0 && a.ldo % 4 == 0 && a.scale_off % 4 == 0 && a.shift_off % 4 == 0 &&
                       a.stride % 4 == 0 && a.W % 128 == 0;
  switch (aligned ? a.W / 128 : 0) {
    case 2: launch_k(norm_reg_kernel<2>, dim3(blocks), dim3(256), 0, s, a); break;
    case 3: launch_k(norm_reg_kernel<3>, dim3(blocks), dim3(256), 0, s, a); break;
    case 4: launch_k(norm_reg_kernel<4>, dim3(blocks), dim3(256), 0, s, a); break;
    case 8: launch_k(norm_reg_kernel<8>, dim3(blocks), dim3(256), 0, s, a); break;
    case 12: launch_k(norm_reg_kernel<12>, dim3(blocks), dim3(256), 0, s, a); break;
    default: launch_k(norm_kernel, dim3(blocks), dim3(256), 0, s, a); break;
  }
}

// ------------------------------------------------------------------------------------------
// Attention of chunk queries over [prefix keys ; chunk keys] with grouped KV heads,
// online softmax in fp32. CTA = (16 queries, one query head, one robot); warp = 4 queries;
// lane = one key of a 32-key block for the scores, 32-strided head dims for the output.
// ------------------------------------------------------------------------------------------
constexpr int AQ = 16, AKB = 32;

__device__ __forceinline__ float rope_elem(const void* base, long long off, int d, int half,
                                           const float* cs, int dt) {
  const float x = ldf_rt(base, off + d, dt);
  const int j = d < half ? d : d - half;
  const float c = cs[2 * j], s = cs[2 * j + 1];
  const float o = ldf_rt(base, off + (d < half ? d + half : d - half), dt);
  return d < half ? x * c - o * s : x * c + o * s;
}

template <int DPL>
__global__ void __launch_bounds__(128) attn_kernel(AttnArgs p) {
  extern __shared__ float sm[];
  pdl_trigger();
  pdl_wait();
  const int dh = DPL * 32, half = dh / 2;
  float* qs = sm;                   // [AQ][dh]
  float* ks = qs + AQ * dh;         // [AKB][dh + 1]
  float* vs = ks + AKB * (dh + 1);  // [AKB][dh]
  float* ps = vs + AKB * dh;        // [AQ][AKB]
  const int b = blockIdx.z, hq = blockIdx.y, i0 = blockIdx.x * AQ;
  const int g = hq / (p.n_heads / p.n_kv_heads);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  for (int e = tid; e < AQ * dh; e += 128) {
    const int qi = e / dh, d = e % dh, i = i0 + qi;
    float val = 0.f;
    if (i < p.H) {
      const long long off = (long long)(b * p.H + i) * p.q_ld + hq * dh;
      val = p.rope_cs ? rope_elem(p.q, off, d, half, p.rope_cs + (long long)i * dh, p.dtype)
                      : ldf_rt(p.q, off + d, p.dtype);
    }
    qs[qi * dh + d] = val * p.scale;
  }

  float m_run[4], l_run[4], o[4][DPL];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    m_run[q] = -INFINITY;
    l_run[q] = 0.f;
#pragma unroll
    for (int t = 0; t < DPL; ++t) o[q][t] = 0.f;
  }
  const int n_keys = p.P + (p.kc ? p.H : 0);
  for (int j0 = 0; j0 < n_keys; j0 += AKB) {
    __syncthreads();
    for (int e = tid; e < AKB * dh; e += 128) {
      const int jj = e / dh, d = e % dh, j = j0 + jj;
      float kv = 0.f, vv = 0.f;
      if (j < p.P) {
        const long long off = b * p.kp_bstride + (long long)j * p.kp_ld + g * dh;
        kv = ldf_rt(p.kp, off + d, p.dtype);
        vv = ldf_rt(p.vp, off + d, p.dtype);
      } else if (j < n_keys) {
        const int i = j - p.P;
        const long long off = (long long)(b * p.H + i) * p.kc_ld + g * dh;
        kv = p.rope_cs ? rope_elem(p.kc, off, d, half, p.rope_cs + (long long)i * dh, p.dtype)
                       : ldf_rt(p.kc, off + d, p.dtype);
        vv = ldf_rt(p.vc, off + d, p.dtype);
      }
      ks[jj * (dh + 1) + d] = kv;
      vs[jj * dh + d] = vv;
    }
    __syncthreads();
    const bool valid = j0 + lane < n_keys;
#pragma unroll
    for (int qq = 0; qq < 4; ++qq) {
      const int q = warp * 4 + qq;
      float s = 0.f;
      for (int d = 0; d < dh; ++d) s = fmaf(qs[q * dh + d], ks[lane * (dh + 1) + d], s);
      s = valid ? s : -INFINITY;
      const float m_new = fmaxf(m_run[qq], warp_max(s));
      const float pe = valid ? expf(s - m_new) : 0.f;
      const float alpha = m_run[qq] == -INFINITY ? 0.f : expf(m_run[qq] - m_new);
      l_run[qq] = l_run[qq] * alpha + warp_sum(pe);
      m_run[qq] = m_new;
      ps[q * AKB + lane] = pe;
#pragma unroll
      for (int t = 0; t < DPL; ++t) o[qq][t] *= alpha;
    }
    __syncwarp();
    for (int jj = 0; jj < AKB; ++jj) {
#pragma unroll
      for (int t = 0; t < DPL; ++t) {
        const float vv = vs[jj * dh + lane + 32 * t];
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) o[qq][t] = fmaf(ps[(warp * 4 + qq) * AKB + jj], vv, o[qq][t]);
      }
    }
  }
#pragma unroll
  for (int qq = 0; qq < 4; ++qq) {
    const int i = i0 + warp * 4 + qq;
    if (i >= p.H) continue;
    const float inv = 1.f / l_run[qq];
#pragma unroll
    for (int t = 0; t < DPL; ++t)
      stf(p.out, (long long)(b * p.H + i) * p.out_ld + hq * dh + lane + 32 * t, o[qq][t] * inv, p.dtype);
  }
}

// ------------------------------------------------------------------------------------------
// Attention for few queries (bf16 operands, head dim 64), split over 64-key chunks (split-KV):
// CTA (query block of 16, key chunk, head, robot) computes the chunk's scores with 256 threads over
// (query, 4 keys) pairs, its softmax partials (max, sum) and P V with threads over (query, 4 dims).
// With one chunk the rows are written at once; otherwise each CTA leaves its partial rows in the
// workspace and the last CTA of the (robot, head, query block) merges them by log-sum-exp and
// resets the arrival count for the next launch. Used by the DiT head: self-attention over the
// chunk's tokens and cross-attention over the projected prefix.
constexpr int kFewDh = 64, kFewQ = 16, kFewKC = 64;
constexpr int kFewPart = kFewDh + 4;     // partial row: O, max, sum, padding (16-byte rows)
constexpr int kFewKPitch = kFewDh + 2;   // bf16 per key row: rows 33 words apart, no bank conflicts

__host__ __device__ inline int few_chunks(int n_keys) { return (n_keys + kFewKC - 1) / kFewKC; }

__device__ __forceinline__ uint32_t pack_bf16_pair(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

__global__ void __launch_bounds__(256) attn_few_kernel(AttnArgs p) {
  __shared__ float qs[kFewQ][kFewDh];
  __shared__ float ps[kFewQ][kFewKC];
  __shared__ __align__(16) __nv_bfloat16 ks[kFewKC * kFewKPitch];
  __shared__ __align__(16) __nv_bfloat16 vs[kFewKC * kFewDh];
  __shared__ float ml[kFewQ][2];
  __shared__ int last;
  pdl_trigger();
  pdl_wait();
  constexpr int dh = kFewDh, half = dh / 2;
  const int n_keys = p.P + (p.kc ? p.H : 0);
  const int C = few_chunks(n_keys), qb = blockIdx.x / C, kc = blockIdx.x % C, key0 = kc * kFewKC;
  const int nk = min(kFewKC, n_keys - key0);
  const int b = blockIdx.z, hq = blockIdx.y, i0 = qb * kFewQ;
  const int g = hq / (p.n_heads / p.n_kv_heads);
  const int tid = threadIdx.x;
  // the chunk's keys and values: 16-byte loads, all issued before any use
  for (int e = tid; e < nk * (dh / 8); e += 256) {
    const int j = key0 + e / (dh / 8), c8 = e % (dh / 8);
    uint4 kv, vv;
    if (j < p.P) {
      const long long off = b * p.kp_bstride + (long long)j * p.kp_ld + g * dh + c8 * 8;
      kv = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.kp) + off);
      vv = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.vp) + off);
    } else {
      const long long off = (long long)(b * p.H + j - p.P) * p.kc_ld + g * dh + c8 * 8;
      kv = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.kc) + off);
      vv = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.vc) + off);
    }
    uint32_t* kd = reinterpret_cast<uint32_t*>(ks + (size_t)(j - key0) * kFewKPitch + c8 * 8);
    kd[0] = kv.x;
    kd[1] = kv.y;
    kd[2] = kv.z;
    kd[3] = kv.w;
    *reinterpret_cast<uint4*>(vs + (size_t)(j - key0) * dh + c8 * 8) = vv;
  }
  for (int e = tid; e < kFewQ * dh; e += 256) {
    const int qi = e / dh, d = e % dh, i = i0 + qi;
    float val = 0.f;
    if (i < p.H) {
      const long long off = (long long)(b * p.H + i) * p.q_ld + hq * dh;
      val = p.rope_cs ? rope_elem(p.q, off, d, half, p.rope_cs + (long long)i * dh, BF16)
                      : ldf_rt(p.q, off + d, BF16);
    }
    qs[qi][d] = val * p.scale;
  }
  __syncthreads();
  // chunk keys carry RoPE like the queries (prefix keys come rotated)
  if (p.rope_cs && p.kc) {
    for (int e = tid; e < nk * half; e += 256) {
      const int jj = e / half, d = e % half, j = key0 + jj;
      if (j < p.P) continue;
      __nv_bfloat16* kr = ks + (size_t)jj * kFewKPitch;
      const float* cs = p.rope_cs + (long long)(j - p.P) * dh;
      const float x0 = __bfloat162float(kr[d]), x1 = __bfloat162float(kr[d + half]);
      kr[d] = __float2bfloat16_rn(x0 * cs[2 * d] - x1 * cs[2 * d + 1]);
      kr[d + half] = __float2bfloat16_rn(x1 * cs[2 * d] + x0 * cs[2 * d + 1]);
    }
    __syncthreads();
  }
  // scores: thread (query q, keys 4 kg .. 4 kg + 3); a 16-lane group shares q
  const int q = tid >> 4, kg = tid & 15;
  float sc[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) sc[e] = 0.f;
#pragma unroll 4
  for (int d2 = 0; d2 < dh / 2; ++d2) {
    const float q0 = qs[q][2 * d2], q1 = qs[q][2 * d2 + 1];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 kf = __bfloat1622float2(reinterpret_cast<const __nv_bfloat162*>(ks + (size_t)(4 * kg + e) * kFewKPitch)[d2]);
      sc[e] = fmaf(q0, kf.x, fmaf(q1, kf.y, sc[e]));
    }
  }
  float mx = -INFINITY;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    if (4 * kg + e >= nk) sc[e] = -INFINITY;   // keys past the end
    mx = fmaxf(mx, sc[e]);
  }
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  float sum = 0.f;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float pe = expf(sc[e] - mx);
    ps[q][4 * kg + e] = pe;
    sum += pe;
  }
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  if (kg == 0) {
    ml[q][0] = mx;
    ml[q][1] = sum;
  }
  __syncthreads();
  // O = P V: thread (query q, dims 4 c .. 4 c + 3)
  const int c = tid & 15;
  float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
  for (int j = 0; j < nk; ++j) {
    const float pj = ps[q][j];
    const __nv_bfloat162* v2 = reinterpret_cast<const __nv_bfloat162*>(vs + (size_t)j * dh + 4 * c);
    const float2 v0 = __bfloat1622float2(v2[0]), v1 = __bfloat1622float2(v2[1]);
    o.x = fmaf(pj, v0.x, o.x);
    o.y = fmaf(pj, v0.y, o.y);
    o.z = fmaf(pj, v1.x, o.z);
    o.w = fmaf(pj, v1.y, o.w);
  }
  const int i = i0 + q;
  __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(p.out) + (long long)(b * p.H + i) * p.out_ld + hq * dh + 4 * c;
  if (C == 1) {
    if (i < p.H) {
      const float inv = 1.f / ml[q][1];
      uint2 pk;
      pk.x = pack_bf16_pair(o.x * inv, o.y * inv);
      pk.y = pack_bf16_pair(o.z * inv, o.w * inv);
      *reinterpret_cast<uint2*>(dst) = pk;
    }
    return;
  }
  // partial rows of this chunk: [group][chunk][q][kFewPart] (O, then max and sum)
  const int QB = gridDim.x / C;
  const size_t grp = ((size_t)b * p.n_heads + hq) * QB + qb;
  float* part = p.split_ws + ((grp * C + kc) * kFewQ + q) * kFewPart;
  *reinterpret_cast<float4*>(part + 4 * c) = o;
  if (c == 0) {
    part[dh] = ml[q][0];
    part[dh + 1] = ml[q][1];
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned prev = atomicAdd(p.split_ctr + grp, 1u);
    last = prev == (unsigned)C - 1u;
    if (last) p.split_ctr[grp] = 0u;   // every chunk has arrived: reset for the next launch
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  // merge the chunks by log-sum-exp
  const float* base = p.split_ws + (grp * C * kFewQ + q) * kFewPart;
  float M = -INFINITY;
  for (int k = 0; k < C; ++k) M = fmaxf(M, __ldcg(base + (size_t)k * kFewQ * kFewPart + dh));
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float L = 0.f;
  for (int k = 0; k < C; ++k) {
    const float* r = base + (size_t)k * kFewQ * kFewPart;
    const float w = expf(__ldcg(r + dh) - M);
    L = fmaf(w, __ldcg(r + dh + 1), L);
    const float4 v = __ldcg(reinterpret_cast<const float4*>(r + 4 * c));
    acc.x = fmaf(w, v.x, acc.x);
    acc.y = fmaf(w, v.y, acc.y);
    acc.z = fmaf(w, v.z, acc.z);
    acc.w = fmaf(w, v.w, acc.w);
  }
  if (i < p.H) {
    const float inv = 1.f / L;
    uint2 pk;
    pk.x = pack_bf16_pair(acc.x * inv, acc.y * inv);
    pk.y = pack_bf16_pair(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2*>(dst) = pk;
  }
}

size_t attn_few_ws_floats(int B, int n_heads, int H, int n_keys) {
  return (size_t)B * n_heads * ((H + kFewQ - 1) / kFewQ) * few_chunks(n_keys) * kFewQ * kFewPart;
}
size_t attn_few_ctr_count(int B, int n_heads, int H) { return (size_t)B * n_heads * ((H + kFewQ - 1) / kFewQ); }

bool attn_few_ok(const AttnArgs& a) {
  const int n_keys = a.P + (a.kc ? a.H : 0);
  const bool aligned = a.kp_ld % 8 == 0 && a.kc_ld % 8 == 0 && a.q_ld % 8 == 0 && a.out_ld % 4 == 0;
  return a.dtype == BF16 && a.head_dim == kFewDh && n_keys >= 1 && aligned && (a.kp_bstride % 8) == 0 &&
         (a.n_heads * a.head_dim) % 8 == 0 && (few_chunks(n_keys) == 1 || (a.split_ws && a.split_ctr));
}

__global__ void add_tau_silu_kernel(const float* __restrict__ x, const float* __restrict__ tab, int stride, int off,
                                    const int* __restrict__ tau_row, int M, int N, void* y, int dt) {
  pdl_trigger();
  pdl_wait();
  const long long total = (long long)M * N;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total; e += (long long)gridDim.x * blockDim.x) {
    const int m = (int)(e / N), n = (int)(e % N);
    const float v = x[e] + tab[(size_t)tau_row[m] * stride + off + n];
    stf(y, e, v / (1.f + expf(-v)), dt);
  }
}

void launch_add_tau_silu(const float* x, const float* tab, int stride, int off, const int* tau_row, int M, int N,
                         void* y, int dt, cudaStream_t s) {
  const long long total = (long long)M * N;
  int blocks = (int)((total + 255) / 256);
  if (blocks > 1024) blocks = 1024;
  launch_k(add_tau_silu_kernel, dim3(blocks), dim3(256), 0, s, x, tab, stride, off, tau_row, M, N, y, dt);
}

template <int DPL>
static void launch_attn_dpl(const AttnArgs& a, dim3 grid, size_t smem, cudaStream_t s) {
  launch_k(attn_kernel<DPL>, grid, dim3(128), smem, s, a);
}

size_t attention_smem_bytes(int dh) {
  return sizeof(float) * (AQ * dh + AKB * (dh + 1) + AKB * dh + AQ * AKB);
}

void launch_attention_prepare(int dh) {
  const int smem = (int)attention_smem_bytes(dh);
  const cudaFuncAttribute at = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if (dh == 64) cudaFuncSetAttribute(attn_kernel<2>, at, smem);
  if (dh == 128) cudaFuncSetAttribute(attn_kernel<4>, at, smem);
  if (dh == 256) cudaFuncSetAttribute(attn_kernel<8>, at, smem);
}

void launch_attention(const AttnArgs& a, cudaStream_t s) {
  const int dh = a.head_dim;
  if (attn_few_ok(a)) {
    const int n_keys = a.P + (a.kc ? a.H : 0);
    launch_k(attn_few_kernel, dim3(((a.H + kFewQ - 1) / kFewQ) * few_chunks(n_keys), a.n_heads, a.B), dim3(256), 0, s, a);
    return;
  }
  const size_t smem = attention_smem_bytes(dh);
  dim3 grid((a.H + AQ - 1) / AQ, a.n_heads, a.B);
  switch (dh) {
    case 64: launch_attn_dpl<2>(a, grid, smem, s); break;
    case 128: launch_attn_dpl<4>(a, grid, smem, s); break;
    case 256: launch_attn_dpl<8>(a, grid, smem, s); break;
    default: break;  // rejected at init
  }
}

// ------------------------------------------------------------------------------------------
// Step epilogue, one CTA per robot (the work itself is euler_robot, euler.cuh).
// ------------------------------------------------------------------------------------------
struct CtaSync {
  __device__ void operator()() const { __syncthreads(); }
};
__global__ void __launch_bounds__(256) euler_kernel(EulerArgs p) {
  pdl_trigger();
  pdl_wait();
  __shared__ int s_rel;
  __shared__ float E_s[64];
  __shared__ float Cr[9];   // SO(3) correction of the tail (rotation dimensions)
  extern __shared__ float ediff[];   // [H][D]
  const EulerSmem sm{ediff, E_s, Cr, &s_rel};
  euler_robot(p, blockIdx.x, threadIdx.x, blockDim.x, sm, CtaSync());
}

void launch_euler_prepare() {
  cudaFuncSetAttribute(euler_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 256 * 64 * (int)sizeof(float));
}

void launch_euler(const EulerArgs& a, cudaStream_t s) {
  launch_k(euler_kernel, dim3(a.B), dim3(256), (size_t)a.H * a.D * sizeof(float), s, a);
}

__global__ void begin_kernel(const float* noise, float* x, float* g, float* u, int n, int* nonfinite,
                             int* evals, unsigned long long* stamps) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) {
    *nonfinite = 0;
    *evals = 0;
    stamps[0] = global_ns();
  }
  if (i < n) {
    const float v = noise[i];
    x[i] = v;
    g[i] = v;
    u[i] = v;
  }
}

void launch_begin(const float* noise, float* x, float* g, float* u, int n, int* nonfinite, int* evals,
                  unsigned long long* stamps, cudaStream_t s) {
  launch_k(begin_kernel, dim3((n + 255) / 256), dim3(256), 0, s, noise, x, g, u, n, nonfinite, evals, stamps);
}

// ------------------------------------------------------------------------------------------
// Weight re-layout: dst[(n * mult + off) * K + k] = src[k * N + n] (transpose + convert).
// ------------------------------------------------------------------------------------------
__global__ void relayout_kernel(const float* src, int K, int N, void* dst, int dt, int mult, long long off) {
  __shared__ float t[32][33];
  const int k0 = blockIdx.y * 32, n0 = blockIdx.x * 32;
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int k = k0 + r, n = n0 + threadIdx.x;
    t[r][threadIdx.x] = (k < K && n < N) ? src[(long long)k * N + n] : 0.f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += blockDim.y) {
    const int n = n0 + r, k = k0 + threadIdx.x;
    if (n < N && k < K) stf(dst, ((long long)n * mult + off) * K + k, t[threadIdx.x][r], dt);
  }
}

void launch_relayout(const float* src, int K, int N, void* dst, int dtype, int mult, long long off,
                     cudaStream_t s) {
  dim3 grid((N + 31) / 32, (K + 31) / 32);
  relayout_kernel<<<grid, dim3(32, 8), 0, s>>>(src, K, N, dst, dtype, mult, off);
}

__global__ void convert_kernel(const void* src, int sdt, void* dst, int ddt, long long n) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    stf(dst, i, ldf_rt(src, i, sdt), ddt);
}

// The rotations of Ghost Action Correction on SO(3) on given rotation vectors (testing aid):
// log_exp[i] = log(exp(w_i)), log_comp[i] = log(exp(w_i) exp(w_{i+1 mod n})^T).
__global__ void so3_check_kernel(const float* w, int n, float* log_exp, float* log_comp) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  float A[9], B[9], Bt[9], C[9];
  so3_exp(w + 3 * i, A);
  so3_log(A, log_exp + 3 * i);
  so3_exp(w + 3 * ((i + 1) % n), B);
#pragma unroll
  for (int r = 0; r < 3; ++r)
#pragma unroll
    for (int c = 0; c < 3; ++c) Bt[r * 3 + c] = B[c * 3 + r];
  mat3_mul(A, Bt, C);
  so3_log(C, log_comp + 3 * i);
}

void launch_so3_check(const float* w, int n, float* log_exp, float* log_comp, cudaStream_t s) {
  so3_check_kernel<<<(n + 127) / 128, 128, 0, s>>>(w, n, log_exp, log_comp);
}

void launch_convert(const void* src, int src_dtype, void* dst, int dst_dtype, long long n, cudaStream_t s) {
  const int blocks = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  convert_kernel<<<blocks > 0 ? blocks : 1, 256, 0, s>>>(src, src_dtype, dst, dst_dtype, n);
}

}  // namespace uad
