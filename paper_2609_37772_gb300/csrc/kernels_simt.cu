// CUDA-core kernels: fp32-FFMA GEMM (the fp32 mode and one-time table fills), adaptive
// norms, attention over prefix + chunk, and the Euler / TR / release / GAC step epilogue.
#include "uad_internal.cuh"

namespace uad {

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

void launch_gemm_simt(const GemmArgs& a, cudaStream_t s) {
  dim3 grid((a.N + 63) / 64, (a.M + 63) / 64);
  if (a.a_dtype == F32 && a.w_dtype == F32) gemm_simt_kernel<F32, F32><<<grid, 256, 0, s>>>(a);
  else if (a.a_dtype == F32 && a.w_dtype == BF16) gemm_simt_kernel<F32, BF16><<<grid, 256, 0, s>>>(a);
  else if (a.a_dtype == BF16 && a.w_dtype == BF16) gemm_simt_kernel<BF16, BF16><<<grid, 256, 0, s>>>(a);
  else gemm_simt_kernel<BF16, F32><<<grid, 256, 0, s>>>(a);
}

// ------------------------------------------------------------------------------------------
// Adaptive norm: y = norm(h) * (1 + scale[tau]) + shift[tau]; one warp per token row.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) norm_kernel(NormArgs p) {
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

void launch_norm(const NormArgs& a, cudaStream_t s) {
  norm_kernel<<<(a.M + 7) / 8, 256, 0, s>>>(a);
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

template <int DPL>
static void launch_attn_dpl(const AttnArgs& a, dim3 grid, size_t smem, cudaStream_t s) {
  attn_kernel<DPL><<<grid, 128, smem, s>>>(a);
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
// Step epilogue (one CTA per robot): Euler update with per-action step (Eq. 5), TR running
// sum (Eqs. 6-7), release of early actions (UAER), next model input, and at the robot's
// last step GAC (Eqs. 8-9). Released rows go to mapped pinned memory, then a per-step flag.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) euler_kernel(EulerArgs p) {
  const int b = blockIdx.x, tid = threadIdx.x;
  const int HD = p.H * p.D;
  const float gs = p.gstep[b];
  const bool last = p.k == p.last_step[b];
  __shared__ int s_rel;
  __shared__ float E_s[64];
  if (tid == 0) s_rel = 0;
  __syncthreads();
  for (int e = tid; e < HD; e += blockDim.x) {
    const int i = e / p.D;
    const long long idx = (long long)b * HD + e;
    const PlanTok t = p.plan[b * p.H + i];
    const float v = p.v[idx];
    if (!isfinite(v)) atomicAdd(p.nonfinite, 1);
    float x = p.x[idx], g = p.g[idx];
    if (t.flags & PF_ACTIVE) x = fmaf(t.dx, v, x);
    if (t.flags & PF_EARLY) g = fmaf(gs, v, g);
    p.x[idx] = x;
    p.g[idx] = g;
    float r = 0.f;
    if (t.flags & PF_RELEASE) {
      p.rel[idx] = x;
      p.host_rel[idx] = x;
      s_rel = 1;
    }
    if (t.flags & PF_NEXT_REL) r = p.rel[idx];
    p.u[idx] = (t.flags & PF_NEXT_G) ? g : ((t.flags & PF_NEXT_REL) ? r : x);
  }
  __syncthreads();
  if (last) {
    const int T = p.tail_count[b];
    if (tid < p.D) {
      float E = 0.f;
      for (int i = 0; i < p.H; ++i) {
        if (p.plan[b * p.H + i].flags & PF_EARLY) {
          const long long idx = (long long)b * HD + i * p.D + tid;
          E += p.g[idx] - p.rel[idx];
        }
      }
      E = T > 0 ? E : 0.f;
      E_s[tid] = E;
      p.E_out[b * p.D + tid] = E;
    }
    __syncthreads();
    for (int e = tid; e < HD; e += blockDim.x) {
      const int i = e / p.D, d = e % p.D;
      const long long idx = (long long)b * HD + e;
      const int fl = p.plan[b * p.H + i].flags;
      const bool early = fl & PF_EARLY;
      const float x = p.x[idx];
      float fin = early ? p.rel[idx] : x;
      if (T > 0 && p.tail_flag[b * p.H + i] && p.gac_mask[d]) fin = x + E_s[d] / (float)T;
      p.final_out[idx] = fin;
      // ghost: reconciled end state with TR; without TR, the frozen action fed back
      p.ghost_out[idx] = early ? ((fl & PF_FROZEN) ? p.rel[idx] : p.g[idx]) : x;
      if (!early) p.host_rel[idx] = fin;
    }
  }
  if (s_rel || last) {
    __threadfence_system();
    __syncthreads();
    if (tid == 0) {
      volatile int* f = p.host_flags + b * kFlagStride + p.k;
      *f = *p.epoch;
      __threadfence_system();
    }
  }
  if (b == 0 && tid == 0) {
    atomicAdd(p.evals, 1);  // one velocity field consumed per step
    p.stamps[p.k] = global_ns();
  }
}

void launch_euler(const EulerArgs& a, cudaStream_t s) { euler_kernel<<<a.B, 256, 0, s>>>(a); }

__global__ void begin_kernel(const float* noise, float* x, float* g, float* u, int n, int* nonfinite,
                             int* evals, unsigned long long* stamps) {
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
  begin_kernel<<<(n + 255) / 256, 256, 0, s>>>(noise, x, g, u, n, nonfinite, evals, stamps);
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

void launch_convert(const void* src, int src_dtype, void* dst, int dst_dtype, long long n, cudaStream_t s) {
  const int blocks = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  convert_kernel<<<blocks > 0 ? blocks : 1, 256, 0, s>>>(src, src_dtype, dst, dst_dtype, n);
}

}  // namespace uad
