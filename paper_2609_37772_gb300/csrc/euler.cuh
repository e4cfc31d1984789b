// Step epilogue of one robot: Euler update with per-action step (Sec. 4.2, Eq. 5), TR running
// sum (Sec. 4.3, Eqs. 6-7), release of early actions (UAER, Sec. 4.2), the next model input, and
// at the robot's last step Ghost Action Correction (Sec. 4.4, Eqs. 8-9; rotation dimensions on
// SO(3), App. C.1). Released rows go to mapped pinned memory, then a per-step flag after a system
// fence. Used by the per-operation `euler_kernel` (one CTA per robot) and by the persistent
// evaluation kernel's final phase; `sync()` is a barrier over the `nthr` participating threads.
#pragma once
#include "uad_internal.cuh"

namespace uad {

// ---- rotations for Ghost Action Correction on SO(3) (App. C.1), fp32 -----------------------
// R(w) = I + sin(t)/t [w]x + (1 - cos(t))/t^2 [w]x^2 (Rodrigues), t = |w|; matrices row-major.
__device__ __forceinline__ void so3_exp(const float* w, float* R) {
  const float t2 = w[0] * w[0] + w[1] * w[1] + w[2] * w[2], t = sqrtf(t2);
  float a, b;
  if (t < 1e-4f) {
    a = 1.f - t2 / 6.f;
    b = 0.5f - t2 / 24.f;
  } else {
    float s, c;
    sincosf(t, &s, &c);
    a = s / t;
    b = (1.f - c) / t2;
  }
  const float x = w[0], y = w[1], z = w[2];
  // [w]x^2 = w w^T - t^2 I
  R[0] = 1.f + b * (x * x - t2); R[1] = -a * z + b * x * y;    R[2] = a * y + b * x * z;
  R[3] = a * z + b * x * y;      R[4] = 1.f + b * (y * y - t2); R[5] = -a * x + b * y * z;
  R[6] = -a * y + b * x * z;     R[7] = a * x + b * y * z;      R[8] = 1.f + b * (z * z - t2);
}

// Principal rotation vector of R (angle in [0, pi]): angle from atan2(|axial part|, cos), the
// axis from the symmetric part when the angle is close to pi.
__device__ __forceinline__ void so3_log(const float* R, float* w) {
  const float v0 = 0.5f * (R[7] - R[5]), v1 = 0.5f * (R[2] - R[6]), v2 = 0.5f * (R[3] - R[1]);
  const float c = 0.5f * (R[0] + R[4] + R[8] - 1.f);
  const float s = sqrtf(v0 * v0 + v1 * v1 + v2 * v2);
  const float t = atan2f(s, c);
  if (t < 1e-4f) {
    const float f = 1.f + t * t / 6.f;
    w[0] = v0 * f; w[1] = v1 * f; w[2] = v2 * f;
    return;
  }
  if (3.14159265f - t > 1e-2f) {
    const float f = t / s;
    w[0] = v0 * f; w[1] = v1 * f; w[2] = v2 * f;
    return;
  }
  // near pi: (R + R^T)/2 - cos(t) I = (1 - cos(t)) n n^T
  const float inv = 1.f / (1.f - c);
  const float B[9] = {(R[0] - c) * inv, 0.5f * (R[1] + R[3]) * inv, 0.5f * (R[2] + R[6]) * inv,
                      0.5f * (R[1] + R[3]) * inv, (R[4] - c) * inv, 0.5f * (R[5] + R[7]) * inv,
                      0.5f * (R[2] + R[6]) * inv, 0.5f * (R[5] + R[7]) * inv, (R[8] - c) * inv};
  int k = 0;
  if (B[4] > B[k * 4]) k = 1;
  if (B[8] > B[k * 4]) k = 2;
  const float r = rsqrtf(fmaxf(B[k * 4], 1e-30f));
  float n0 = B[k] * r, n1 = B[3 + k] * r, n2 = B[6 + k] * r;
  if (n0 * v0 + n1 * v1 + n2 * v2 < 0.f) { n0 = -n0; n1 = -n1; n2 = -n2; }
  w[0] = n0 * t; w[1] = n1 * t; w[2] = n2 * t;
}

__device__ __forceinline__ void mat3_mul(const float* A, const float* B, float* C) {
#pragma unroll
  for (int i = 0; i < 3; ++i)
#pragma unroll
    for (int j = 0; j < 3; ++j) C[i * 3 + j] = A[i * 3] * B[j] + A[i * 3 + 1] * B[3 + j] + A[i * 3 + 2] * B[6 + j];
}

__device__ __forceinline__ unsigned long long euler_global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Shared-memory scratch of euler_robot: ediff [H][D] floats, E [64], C [9], one flag.
struct EulerSmem {
  float* ediff;
  float* E_s;
  float* Cr;
  int* s_rel;
};

// Robot b's step epilogue, run by threads tid = 0 .. nthr-1 of one CTA.
template <class Sync>
__device__ __forceinline__ void euler_robot(const EulerArgs& p, int b, int tid, int nthr, const EulerSmem& sm,
                                            Sync sync) {
  const int HD = p.H * p.D;
  const float gs = p.gstep[b];
  const bool last = p.k == p.last_step[b];
  float* ediff = sm.ediff;
  float* E_s = sm.E_s;
  float* Cr = sm.Cr;
  if (tid == 0) *sm.s_rel = 0;
  sync();
  for (int e = tid; e < HD; e += nthr) {
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
      *sm.s_rel = 1;
    }
    if (t.flags & PF_NEXT_REL) r = p.rel[idx];
    p.u[idx] = (t.flags & PF_NEXT_G) ? g : ((t.flags & PF_NEXT_REL) ? r : x);
  }
  sync();
  if (last) {
    const int T = p.tail_count[b];
    // Eq. 8 terms (ghost - released) of early actions, staged in shared memory by all threads,
    // then summed per dimension in token order
    for (int e = tid; e < HD; e += nthr) {
      const int i = e / p.D;
      const long long idx = (long long)b * HD + e;
      ediff[e] = (p.plan[b * p.H + i].flags & PF_EARLY) ? p.g[idx] - p.rel[idx] : 0.f;
    }
    sync();
    const int rd = *p.rot_dim;
    if (tid < p.D) {
      float E = 0.f;
      for (int i = 0; i < p.H; ++i) E += ediff[i * p.D + tid];
      E = T > 0 ? E : 0.f;
      E_s[tid] = E;
      if (rd < 0 || tid < rd || tid >= rd + 3) p.E_out[b * p.D + tid] = E;
    }
    if (rd >= 0 && tid == 32 % nthr) {
      // accumulated rotation error E_R = prod of R(ghost) R(released)^T over early actions in
      // token order (later ones on the left); correction C = exp(log(E_R) / |tail|)
      float E[9] = {1.f, 0.f, 0.f, 0.f, 1.f, 0.f, 0.f, 0.f, 1.f};
      for (int i = 0; i < p.H; ++i) {
        if (!(p.plan[b * p.H + i].flags & PF_EARLY)) continue;
        const long long idx = (long long)b * HD + (long long)i * p.D + rd;
        const float wg[3] = {p.g[idx], p.g[idx + 1], p.g[idx + 2]};
        const float wr[3] = {p.rel[idx], p.rel[idx + 1], p.rel[idx + 2]};
        float Rg[9], Rr[9], Dm[9], En[9];
        so3_exp(wg, Rg);
        so3_exp(wr, Rr);
        const float RrT[9] = {Rr[0], Rr[3], Rr[6], Rr[1], Rr[4], Rr[7], Rr[2], Rr[5], Rr[8]};
        mat3_mul(Rg, RrT, Dm);
        mat3_mul(Dm, E, En);
#pragma unroll
        for (int q = 0; q < 9; ++q) E[q] = En[q];
      }
      float e[3];
      so3_log(E, e);
      const float inv = T > 0 ? 1.f / (float)T : 0.f;
      const float ec[3] = {e[0] * inv, e[1] * inv, e[2] * inv};
      so3_exp(ec, Cr);
      for (int q = 0; q < 3; ++q) p.E_out[b * p.D + rd + q] = T > 0 ? e[q] : 0.f;
    }
    sync();
    for (int e = tid; e < HD; e += nthr) {
      const int i = e / p.D, d = e % p.D;
      const long long idx = (long long)b * HD + e;
      const int fl = p.plan[b * p.H + i].flags;
      const bool early = fl & PF_EARLY;
      const float x = p.x[idx];
      float fin = early ? p.rel[idx] : x;
      const bool rot = rd >= 0 && d >= rd && d < rd + 3;
      if (T > 0 && p.tail_flag[b * p.H + i] && p.gac_mask[d] && !rot) fin = x + E_s[d] / (float)T;
      p.final_out[idx] = fin;
      // ghost: reconciled end state with TR; without TR, the frozen action fed back
      p.ghost_out[idx] = early ? ((fl & PF_FROZEN) ? p.rel[idx] : p.g[idx]) : x;
      if (!early && !(rot && T > 0 && p.tail_flag[b * p.H + i])) p.host_rel[idx] = fin;
    }
    if (rd >= 0 && T > 0) {
      // rotation dimensions of the tail: R(a) <- C R(a), the representative nearest to a
      sync();
      for (int i = tid; i < p.H; i += nthr) {
        if (!p.tail_flag[b * p.H + i]) continue;
        const long long idx = (long long)b * HD + (long long)i * p.D + rd;
        const float w0[3] = {p.x[idx], p.x[idx + 1], p.x[idx + 2]};
        float R0[9], R1[9], w[3];
        so3_exp(w0, R0);
        mat3_mul(Cr, R0, R1);
        so3_log(R1, w);
        const float t = sqrtf(w[0] * w[0] + w[1] * w[1] + w[2] * w[2]);
        if (t > 1e-12f) {
          float best = 3.4e38f, pick[3] = {w[0], w[1], w[2]};
          for (int m = -1; m <= 1; ++m) {
            const float f = 1.f + 6.2831853f * (float)m / t;
            const float c0 = w[0] * f, c1 = w[1] * f, c2 = w[2] * f;
            const float dd = (c0 - w0[0]) * (c0 - w0[0]) + (c1 - w0[1]) * (c1 - w0[1]) + (c2 - w0[2]) * (c2 - w0[2]);
            if (dd < best) { best = dd; pick[0] = c0; pick[1] = c1; pick[2] = c2; }
          }
          w[0] = pick[0]; w[1] = pick[1]; w[2] = pick[2];
        }
        for (int q = 0; q < 3; ++q) {
          p.final_out[idx + q] = w[q];
          p.host_rel[idx + q] = w[q];
        }
      }
    }
  }
  if (*reinterpret_cast<volatile int*>(sm.s_rel) || last) {
    __threadfence_system();
    sync();
    if (tid == 0) {
      volatile int* f = p.host_flags + b * kFlagStride + p.k;
      *f = *p.epoch;
      __threadfence_system();
    }
  }
  if (b == 0 && tid == 0) {
    atomicAdd(p.evals, 1);  // one velocity field consumed per step
    p.stamps[p.k] = euler_global_ns();
  }
  sync();
}

}  // namespace uad
