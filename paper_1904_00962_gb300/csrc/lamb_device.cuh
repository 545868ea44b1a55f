// Device helpers shared by the two-pass and the on-chip kernels: the
// element arithmetic of Algs. 1-4 (explicit round-to-nearest intrinsics,
// so every kernel forms bit-identical values), vector loads and stores,
// warp reductions, and the helpers that close a step.
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "lamb_internal.h"

namespace lamb {
namespace {

// ---------------------------------------------------------------------------
// Element arithmetic.  Every operation is an explicit round-to-nearest
// intrinsic, so the compiler cannot fuse differently in the two passes.
// ---------------------------------------------------------------------------
struct LambConsts {
  float b1, omb1, b2, omb2;   // beta1, 1-beta1, beta2, 1-beta2
  float c1, c2;               // 1/(1-beta1^t), 1/(1-beta2^t)
  float eps;
  float am, ag, bv, bg;       // N-LAMB / NN-LAMB direction coefficients
};

// Alg. 2: m_t = beta1 m + (1-beta1) g ;  v_t = beta2 v + (1-beta2) g^2
__device__ __forceinline__ void lamb_moments(float g, float& m, float& v,
                                             const LambConsts& k) {
  m = __fmaf_rn(k.b1, m, __fmul_rn(k.omb1, g));
  v = __fmaf_rn(k.b2, v, __fmul_rn(k.omb2, __fmul_rn(g, g)));
}

// Alg. 2: u = (m_t c1) / (sqrt(v_t c2) + eps) + lambda_k w
__device__ __forceinline__ float lamb_direction(float m, float v, float w,
                                                float lam,
                                                const LambConsts& k) {
  const float mh = __fmul_rn(m, k.c1);
  const float vh = __fmul_rn(v, k.c2);
  const float den = __fadd_rn(__fsqrt_rn(vh), k.eps);
  return __fmaf_rn(lam, w, __fdiv_rn(mh, den));
}

// Appendix Alg. 3 / 4 (N-LAMB / NN-LAMB):
//   u = (am m_t + ag g) / (sqrt(bv v_t [+ bg g^2]) + eps) + lambda_k w
// with am = mu_{t+1}/(1 - prod_{i<=t+1} mu_i), ag = (1 - mu_t)/(1 - prod_{i<=t}
// mu_i); N-LAMB: bv = 1/(1 - beta2^t); NN-LAMB: bv = beta2/(1 - beta2^(t+1)),
// bg = (1 - beta2)/(1 - beta2^t).
template <int kNest>
__device__ __forceinline__ float nlamb_direction(float m, float v, float g,
                                                 float w, float lam,
                                                 const LambConsts& k) {
  const float mh = __fmaf_rn(k.am, m, __fmul_rn(k.ag, g));
  const float vh = kNest == 2
                       ? __fmaf_rn(k.bv, v, __fmul_rn(k.bg, __fmul_rn(g, g)))
                       : __fmul_rn(v, k.bv);
  const float den = __fadd_rn(__fsqrt_rn(vh), k.eps);
  return __fmaf_rn(lam, w, __fdiv_rn(mh, den));
}

// Alg. 1: m_t = beta1 m + (1-beta1) (g + lambda_k w)
__device__ __forceinline__ float lars_momentum(float g, float m, float w,
                                               float lam, float b1,
                                               float omb1) {
  return __fmaf_rn(b1, m, __fmul_rn(omb1, __fmaf_rn(lam, w, g)));
}

// ---------------------------------------------------------------------------
// Memory helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float4 ld4(const float* p) {
  return *reinterpret_cast<const float4*>(p);
}
__device__ __forceinline__ float4 ld4_last(const float* p) {  // last use
  return __ldcs(reinterpret_cast<const float4*>(p));
}
__device__ __forceinline__ void st4(float* p, float4 x) {
  *reinterpret_cast<float4*>(p) = x;
}
__device__ __forceinline__ void st4_last(float* p, float4 x) {
  __stcs(reinterpret_cast<float4*>(p), x);
}

// Gradients are read exactly once: streaming (evict-first) loads.
__device__ __forceinline__ float4 ld_grad4(const float* p) {
  return __ldcs(reinterpret_cast<const float4*>(p));
}
// bf16 -> f32 widening is exact: the bf16 pattern is the top half of the f32.
__device__ __forceinline__ float4 ld_grad4(const __nv_bfloat16* p) {
  const uint2 u = __ldcs(reinterpret_cast<const uint2*>(p));
  return make_float4(__uint_as_float(u.x << 16),
                     __uint_as_float(u.x & 0xffff0000u),
                     __uint_as_float(u.y << 16),
                     __uint_as_float(u.y & 0xffff0000u));
}
__device__ __forceinline__ float ld_grad1(const float* p) { return __ldcs(p); }
__device__ __forceinline__ float ld_grad1(const __nv_bfloat16* p) {
  const unsigned short h = __ldcs(reinterpret_cast<const unsigned short*>(p));
  return __uint_as_float(uint32_t(h) << 16);
}

__device__ __forceinline__ void st_copy4(void* base, int64_t i, float4 x) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(x.x, x.y);  // RNE
  const __nv_bfloat162 hi = __floats2bfloat162_rn(x.z, x.w);
  uint2 u;
  u.x = *reinterpret_cast<const uint32_t*>(&lo);
  u.y = *reinterpret_cast<const uint32_t*>(&hi);
  __stcs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(base) + i), u);
}
__device__ __forceinline__ void st_copy1(void* base, int64_t i, float x) {
  static_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(x);
}

// ---------------------------------------------------------------------------
// Reductions: fixed trees, so the result depends only on the data layout.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_down_sync(0xffffffffu, x, o);
  return x;
}

// eta_t: read from device memory, or (kFlagLrSchedule) the Section 4
// schedule eta_0 t / T_w during warmup, then eta_0 max(0, 1 - t / T).
__device__ __forceinline__ float step_lr(const StepParams& p, int64_t t) {
  if (!(p.flags & kFlagLrSchedule)) return *p.d_lr;
  double lr;
  if (p.lr_warmup > 0 && t < p.lr_warmup)
    lr = p.lr_base * (double)t / (double)p.lr_warmup;
  else
    lr = p.lr_base * fmax(0.0, 1.0 - (double)t / (double)p.lr_total);
  return (float)lr;
}

// The CTA or warp that closes a step: advance the step counter and report
// the scheduled learning rate.
__device__ __forceinline__ void close_step(const StepParams& p,
                                           const StepScalars& sc) {
  if (p.flags & kFlagNoClose) return;
  if ((p.flags & kFlagLrSchedule) && p.d_lr_out) *p.d_lr_out = sc.lr;
  if ((p.flags & kFlagIncrementStep) && p.d_step) *p.d_step = sc.t + 1;
}

// b^t for an integer step count t from log2(b): exp2 in fp64 (a power of
// the bias correction or of a momentum schedule; exact rounding of the
// exponent product is irrelevant next to the final rounding to float).
__device__ __forceinline__ double pow_from_log2(double log2_b, double t) {
  return exp2(t * log2_b);
}

__device__ __forceinline__ double phi_of(double z, const StepParams& p) {
  if (p.phi == 1) {  // clip; comparisons keep NaN as NaN
    if (z < p.gamma_l) return p.gamma_l;
    if (z > p.gamma_u) return p.gamma_u;
  }
  return z;
}

// Nadam momentum schedule term (appendix Alg. 3 inputs): mu_t =
// beta1 (1 - 0.5 * 0.96^(t psi)).
__device__ __forceinline__ double nadam_mu(const StepParams& p, int64_t t) {
  return p.beta1 * (1.0 - 0.5 * pow_from_log2(p.log2_mu_decay, (double)t));
}

// Per-launch constants of a LAMB / N-LAMB step (Alg. 2 bias correction, the
// appendix Algs. 3/4 momentum schedule).  The fp64 work is spread over the
// lane 0 of warps 0-3 (one power each, with the divisions that need only it)
// while warp 4 draws the first chunk (kDraw: a pass 1 that takes work from
// counters[0]) and warp 5 fetches the N-LAMB product; thread 0 then forms the
// rest.  The results do not depend on the split.  CTA 0 stores them in
// *p.scal; s_t (optional) receives the step count t.
template <int kNest, bool kDraw>
__device__ __forceinline__ void step_constants(const StepParams& p,
                                               uint32_t* s_next, int* s_skip,
                                               LambConsts* s_k,
                                               int64_t* s_t_out) {
  __shared__ double s_x[3];     // mu_t, mu_{t+1}, prod_{i<t} mu_i
  __shared__ float s_c[2];      // c1, c2 (LAMB) or bv, bg (N-LAMB)
  __shared__ int64_t s_t;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool bc = kNest != 0 || (p.flags & kFlagBiasCorrection) != 0;
  if (lane == 0 && warp < 6) {
    const int64_t t = p.d_step ? *p.d_step : int64_t(1);
    const bool skip = bc && t < 1;
    const double td = (double)t;
    if (warp == 0) {
      *s_skip = skip ? 1 : 0;
      s_t = t;
    }
    if (!skip) {
      if (warp == 4) {
        if (kDraw) s_next[0] = atomicAdd(&p.counters[0], 1u);
      } else if (!kNest) {
        if (warp < 2)   // Alg. 2 bias correction: 1/(1 - beta^t)
          s_c[warp] = !bc ? 1.f
                          : (float)(1.0 / (1.0 - pow_from_log2(
                                warp == 0 ? p.log2_beta1 : p.log2_beta2, td)));
      } else if (warp < 2) {           // appendix Alg. 3/4: mu_t, mu_{t+1}
        s_x[warp] = nadam_mu(p, t + warp);
      } else if (warp == 2) {          // v_hat's correction at t
        const double b = pow_from_log2(p.log2_beta2, td);
        if (kNest == 2) s_c[1] = (float)((1.0 - p.beta2) / (1.0 - b));
        else s_c[0] = (float)(1.0 / (1.0 - b));
      } else if (warp == 3) {          // NN-LAMB: beta2 / (1 - beta2^(t+1))
        if (kNest == 2)
          s_c[0] = (float)(p.beta2 /
                           (1.0 - pow_from_log2(p.log2_beta2, td + 1.0)));
      } else if (kNest) {              // warp 5
        s_x[2] = *p.d_mu_product;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const int64_t t = s_t;
    const int skip = *s_skip;
    LambConsts kc{p.b1, p.omb1, p.b2, p.omb2, 1.f, 1.f, p.eps,
                  0.f, 0.f, 0.f, 0.f};
    double mu_prod = 0.0;
    if (!skip) {
      if (!kNest) {
        kc.c1 = s_c[0];
        kc.c2 = s_c[1];
      } else {
        const double mu_t = s_x[0], mu_n = s_x[1];
        mu_prod = s_x[2] * mu_t;
        kc.am = (float)(mu_n / (1.0 - mu_prod * mu_n));
        kc.ag = (float)((1.0 - mu_t) / (1.0 - mu_prod));
        kc.bv = s_c[0];
        kc.bg = kNest == 2 ? s_c[1] : 0.f;
      }
    }
    *s_k = kc;
    if (s_t_out) *s_t_out = t;
    if (blockIdx.x == 0) {
      StepScalars sc{};
      sc.t = t;
      sc.c1 = kc.c1;
      sc.c2 = kc.c2;
      sc.lr = step_lr(p, t);
      sc.skip = skip;
      sc.am = kc.am;
      sc.ag = kc.ag;
      sc.bv = kc.bv;
      sc.bg = kc.bg;
      sc.mu_prod = mu_prod;
      *p.scal = sc;
      if (skip) atomicOr(p.status, kStatusBadStep);
    }
  }
  __syncthreads();
}

}  // namespace
}  // namespace lamb
