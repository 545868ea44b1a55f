// sm_103a kernels of the two-pass LAMB / LARS step.
//
// The step of Algorithm 2 needs, per tensor, ||x|| and ||r + lambda x|| over
// the WHOLE tensor before any element of x may change, so it is split in two
// streaming passes over HBM:
//
//   pass 1  reads g, m, v, w; writes the new m, v (Alg. 2 moment lines);
//           forms u = r + lambda_k w in registers and accumulates sum w^2 and
//           sum u^2 per chunk (fp32 per thread, fixed warp/CTA tree) into the
//           chunk's slot.  The CTA that finishes the last chunk of a tensor
//           (ticket counter) combines that tensor's slots in a fixed order in
//           fp64 and writes ||w||, ||u|| and rho = phi(||w||)/||u|| (Alg. 2
//           last line; rho = 1 on a zero norm).
//   pass 2  reads m, v, w; recomputes u bit-identically (same __device__
//           function, explicit round-to-nearest intrinsics, no contraction)
//           and writes w - eta*rho*u (and its bf16 copy).
//
// LARS (Algorithm 1) has the same shape with u = m_t.
//
// Optional, chosen per step from the flags:
//   gradient check  pass 1 also sums g^2 per chunk and 0*g (0, or NaN once
//                   any element is Inf/NaN); the tensors' finalisers form
//                   ||g_k||, and the last one the global ||g|| and the
//                   step's decision.
//   skip mode       pass 1 leaves m, v untouched; pass 2 reads the decision
//                   first and either writes nothing or forms the moments
//                   from g itself and writes m, v, w (42 instead of 40 bytes
//                   per parameter with bf16 g).
//   decoupled decay lambda_k w leaves u and is applied outside the trust
//                   ratio: w <- w - eta rho u - eta lambda_k w.
//
// Both passes are persistent grids (CTAs = SMs x resident CTAs per SM) that
// draw chunks from a device work counter, so hundreds of tiny tensors and a
// 31M-element embedding share one launch.  The grid never waits on itself:
// tickets and counters only decide WHO does a piece of work, never block.
// The last CTA to draw from a counter resets it (and the last chunk of a
// tensor resets its ticket), so the kernels can be replayed from a CUDA
// graph with no host involvement.

#include <type_traits>

#include "lamb_device.cuh"

namespace lamb {
namespace {

// 4-element packets in flight per thread and array.  Pass 1 keeps 2 so that
// its LAMB kernels fit 80 registers and run 3 CTAs per SM like pass 2: a
// CTA's chunk epilogue (block reduction, slot, ticket, next descriptors)
// then leaves two other CTAs streaming on the SM.  Measured on BERT-large:
// 2 CTAs/SM x 4 packets 1072 us, 3 x 2 1066 us per pass 1 (16,384-element
// chunks; 1131 vs 1080 us at 8,192).
constexpr int kUnroll1 = 2;
constexpr int kUnroll2 = 4;   // pass 2: 80 registers, 3 CTAs per SM
constexpr int kMinBlocks1 = 3;

// Sums of the first N of x[] over the CTA, valid in thread 0 (fixed trees:
// lanes, then warps).  Contains one barrier; red must hold N rows.
template <int N>
__device__ __forceinline__ void cta_sum(float* x, float (*red)[kWarps]) {
#pragma unroll
  for (int i = 0; i < N; ++i) x[i] = warp_sum(x[i]);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < N; ++i) red[i][warp] = x[i];
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int i = 0; i < N; ++i) x[i] = warp_sum(lane < kWarps ? red[i][lane] : 0.f);
  }
}

// The tensor that finishes last in pass 1 (gradient check only): the global
// ||g|| as a fixed-order fp64 sum over the tensors' sum g^2, and the step's
// decision, which pass 2 reads before it writes anything.  Warp-wide.
__device__ __forceinline__ void finalize_grad(const StepParams& p) {
  __threadfence();
  const int lane = threadIdx.x & 31;
  double a = 0.0;
  for (int k = lane; k < p.n_tensors; k += 32) a += __ldcg(&p.gsq[k]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) a += __shfl_down_sync(0xffffffffu, a, o);
  if (lane == 0) {
    const uint32_t bad = atomicExch(&p.gcheck->acc, 0u);
    p.gcheck->norm = sqrt(a);
    p.gcheck->nonfinite = bad;
    if (bad)
      atomicOr(p.status, kStatusGradNonfinite |
                             ((p.flags & kFlagSkipNonfinite) ? kStatusSkipped
                                                             : 0u));
    p.gcheck->done = 0u;
  }
}

// All threads of the CTA that finished tensor k's last chunk: fixed-order
// fp64 combine of the chunk slots -> norms and trust ratio.  Thread t adds
// slots t, t + kThreads, ... in that order; each warp adds its lanes, then
// warp 0 the warps, in fixed trees.  Spreading the slots over the whole CTA
// keeps a tensor of thousands of chunks (BERT's word embedding: 1,908) to a
// few dependent L2 loads per thread.  Resets the ticket.  With the gradient
// check (kGn) it also forms the tensor's sum g^2 and whether any of its
// elements was Inf/NaN, and counts the tensor done.
template <bool kGn>
__device__ __noinline__ void finalize_tensor(const StepParams& p, int k,
                                             int first, int n, double coef) {
  __shared__ double s_fin[4][kWarps];
  __threadfence();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  double aw = 0.0, au = 0.0, ag = 0.0;
  float az = 0.f;
  for (int i = (int)threadIdx.x; i < n; i += kThreads) {
    const float2 s = __ldcg(&p.slots[first + i]);
    aw += (double)s.x;
    au += (double)s.y;
    if (kGn) {
      const float2 q = __ldcg(&p.grad_slots[first + i]);
      ag += (double)q.x;
      az += q.y;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    aw += __shfl_down_sync(0xffffffffu, aw, o);
    au += __shfl_down_sync(0xffffffffu, au, o);
    if (kGn) {
      ag += __shfl_down_sync(0xffffffffu, ag, o);
      az += __shfl_down_sync(0xffffffffu, az, o);
    }
  }
  if (lane == 0) {
    s_fin[0][warp] = aw;
    s_fin[1][warp] = au;
    s_fin[2][warp] = ag;
    s_fin[3][warp] = (double)az;
  }
  __syncthreads();
  if (warp != 0) return;
  aw = lane < kWarps ? s_fin[0][lane] : 0.0;
  au = lane < kWarps ? s_fin[1][lane] : 0.0;
  ag = lane < kWarps ? s_fin[2][lane] : 0.0;
  az = lane < kWarps ? (float)s_fin[3][lane] : 0.f;
#pragma unroll
  for (int o = kWarps / 2; o > 0; o >>= 1) {
    aw += __shfl_down_sync(0xffffffffu, aw, o);
    au += __shfl_down_sync(0xffffffffu, au, o);
    if (kGn) {
      ag += __shfl_down_sync(0xffffffffu, ag, o);
      az += __shfl_down_sync(0xffffffffu, az, o);
    }
  }
  int last_tensor = 0;
  if (lane == 0) {
    const double wn = sqrt(aw), un = sqrt(au);
    double rho = 1.0;                                  // zero-norm rule
    if (!(wn == 0.0 || un == 0.0)) rho = coef * phi_of(wn, p) / un;
    p.ratio[k] = rho;
    p.wnorm[k] = wn;
    p.unorm[k] = un;
    if (!isfinite(aw) || !isfinite(au)) atomicOr(p.status, kStatusNonfinite);
    if (kGn) {
      p.gsq[k] = ag;
      p.gnorm[k] = sqrt(ag);
      if (isnan(az)) atomicOr(&p.gcheck->acc, 1u);
      __threadfence();
      last_tensor =
          atomicAdd(&p.gcheck->done, 1u) + 1u == (uint32_t)p.n_live;
    }
    p.tickets[k] = 0u;
  }
  if (kGn && __shfl_sync(0xffffffffu, last_tensor, 0)) finalize_grad(p);
}

// Chunk epilogue of pass 1: publish the CTA's partial sums (acc[0] = sum w^2,
// acc[1] = sum u^2; with kGn also acc[2] = sum g^2, acc[3] = sum 0*g), take a
// ticket, and let the last chunk of the tensor finalise it.
template <bool kGn>
__device__ __forceinline__ void publish_chunk(const StepParams& p, int c,
                                              const ChunkDesc& ch,
                                              const TensorDesc& td, float* acc,
                                              float (*red)[kWarps],
                                              int* s_last, double coef) {
  cta_sum<kGn ? 4 : 2>(acc, red);
  if (threadIdx.x == 0) {
    p.slots[c] = make_float2(acc[0], acc[1]);
    if (kGn) p.grad_slots[c] = make_float2(acc[2], acc[3]);
    if (p.flags & kFlagNoFinalize) {   // a shard: the sums are exchanged first
      *s_last = 0;
    } else {
      __threadfence();
      const uint32_t prev = atomicAdd(&p.tickets[ch.tensor], 1u);
      *s_last = (prev + 1u == (uint32_t)td.n_chunks);
    }
  }
  __syncthreads();
  if (*s_last)   // the whole CTA
    finalize_tensor<kGn>(p, ch.tensor, td.first_chunk, td.n_chunks, coef);
}

// Work distribution.  Thread 0 draws chunk indices from counters[which];
// indices >= n_chunks mean "done".  Every CTA draws exactly one such index,
// so the CTA that draws n_chunks + gridDim.x - 1 is the last one to draw and
// may reset the counter for the next launch.  Returns true for that CTA.
__device__ __forceinline__ bool retire(const StepParams& p, int which,
                                       uint32_t last_drawn) {
  const bool last = last_drawn == (uint32_t)p.n_chunks + gridDim.x - 1u;
  if (last && threadIdx.x == 0) atomicExch(&p.counters[which], 0u);
  return last;
}


// ---------------------------------------------------------------------------
// LAMB pass 1 (also N-LAMB / NN-LAMB: kNest = 1 / 2)
//
// acc[] accumulates per thread: sum w^2, sum u^2 and, with the gradient check
// (kGn), sum g^2 and sum 0*g -- the last is 0 unless some g is Inf or NaN,
// which makes it NaN whatever the order of the sum.  store = false (the
// skip-on-non-finite mode) leaves m, v untouched: pass 2 forms and writes
// them once the step is known to be applied.
// ---------------------------------------------------------------------------
template <int kNest, bool kGn>
__device__ __forceinline__ void lamb1_elem(float g, float& m, float& v,
                                           float w, float lam,
                                           const LambConsts& k, float* acc) {
  lamb_moments(g, m, v, k);
  const float u = kNest ? nlamb_direction<kNest>(m, v, g, w, lam, k)
                        : lamb_direction(m, v, w, lam, k);
  acc[0] = __fmaf_rn(w, w, acc[0]);
  acc[1] = __fmaf_rn(u, u, acc[1]);
  if (kGn) {
    acc[2] = __fmaf_rn(g, g, acc[2]);
    acc[3] = __fmaf_rn(g, 0.f, acc[3]);
  }
}

template <typename GT, int kNest, bool kGn>
__device__ __forceinline__ void lamb1_chunk(const TensorPtrs& tp,
                                            const ChunkDesc& ch, float lam,
                                            const LambConsts& k, bool store,
                                            float* acc) {
  float* __restrict__ w = tp.w + ch.offset;
  float* __restrict__ m = tp.m + ch.offset;
  float* __restrict__ v = tp.v + ch.offset;
  const GT* __restrict__ g = static_cast<const GT*>(tp.g) + ch.offset;
  const int n = ch.len;
  int scalar_from = 0;
  if (tp.vec_ok) {
    const int nv = n >> 2;
    for (int base = threadIdx.x; base < nv; base += kThreads * kUnroll1) {
      float4 wv[kUnroll1], mv[kUnroll1], vv[kUnroll1], gv[kUnroll1];
#pragma unroll
      for (int u = 0; u < kUnroll1; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          gv[u] = ld_grad4(g + 4 * j);
          mv[u] = ld4(m + 4 * j);
          vv[u] = ld4(v + 4 * j);
          wv[u] = ld4(w + 4 * j);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll1; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          lamb1_elem<kNest, kGn>(gv[u].x, mv[u].x, vv[u].x, wv[u].x, lam, k, acc);
          lamb1_elem<kNest, kGn>(gv[u].y, mv[u].y, vv[u].y, wv[u].y, lam, k, acc);
          lamb1_elem<kNest, kGn>(gv[u].z, mv[u].z, vv[u].z, wv[u].z, lam, k, acc);
          lamb1_elem<kNest, kGn>(gv[u].w, mv[u].w, vv[u].w, wv[u].w, lam, k, acc);
          if (store) {
            st4(m + 4 * j, mv[u]);
            st4(v + 4 * j, vv[u]);
          }
        }
      }
    }
    scalar_from = nv << 2;
  }
  for (int i = scalar_from + threadIdx.x; i < n; i += kThreads) {
    float mi = m[i], vi = v[i];
    lamb1_elem<kNest, kGn>(ld_grad1(g + i), mi, vi, w[i], lam, k, acc);
    if (store) {
      m[i] = mi;
      v[i] = vi;
    }
  }
}

// lambda_k inside the normalised direction u (Alg. 2); 0 with decoupled
// decay, where pass 2 applies lambda_k w outside the trust ratio instead.
__device__ __forceinline__ float lam_in_u(const StepParams& p,
                                          const TensorDesc& td) {
  return (p.flags & kFlagDecoupledDecay) ? 0.f : td.decay * p.wd;
}

template <typename GT, int kNest, bool kGn>
__global__ void __launch_bounds__(kThreads, kMinBlocks1)
    lamb_pass1_kernel(const StepParams p) {
  __shared__ float red[4][kWarps];
  __shared__ uint32_t s_next[2];
  __shared__ int s_last, s_skip;
  __shared__ LambConsts s_k;
  step_constants<kNest, true>(p, s_next, &s_skip, &s_k, nullptr);
  if (s_skip) return;
  const LambConsts k = s_k;
  const bool store = !(kGn && (p.flags & kFlagSkipNonfinite));
  int it = 0;
  uint32_t c = s_next[0];
  while (c < (uint32_t)p.n_chunks) {
    if (threadIdx.x == 0) s_next[(it + 1) & 1] = atomicAdd(&p.counters[0], 1u);
    const ChunkDesc ch = p.chunks[c];
    const TensorDesc td = p.tensors[ch.tensor];
    const TensorPtrs tp = p.ptrs[ch.tensor];
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    lamb1_chunk<GT, kNest, kGn>(tp, ch, lam_in_u(p, td), k, store, acc);
    publish_chunk<kGn>(p, (int)c, ch, td, acc, red, &s_last, 1.0);
    ++it;
    c = s_next[it & 1];
  }
  retire(p, 0, c);
}

// ---------------------------------------------------------------------------
// LAMB pass 2
//
// w <- w - s u with s = eta rho_k, u recomputed bit-identically from the
// pass-1 operands.  kDefer (skip-on-non-finite mode): m, v still hold the
// previous step's values, so the moments are formed here from g and written
// together with w.  Decoupled decay (dd = eta lambda_k != 0): w <- w - s u -
// dd w; with dd == 0 the extra term is skipped, not added as a zero, so the
// plain step keeps w - s u bit for bit (signed zeros, Inf - Inf).
// ---------------------------------------------------------------------------
template <int kNest>
__device__ __forceinline__ float lamb2_dir(float m, float v, float g, float w,
                                           float lam, const LambConsts& k) {
  return kNest ? nlamb_direction<kNest>(m, v, g, w, lam, k)
               : lamb_direction(m, v, w, lam, k);
}

template <int kNest, bool kDefer>
__device__ __forceinline__ float lamb2_elem(float g, float& m, float& v,
                                            float w, float lam, float s,
                                            float dd, const LambConsts& k) {
  if (kDefer) lamb_moments(g, m, v, k);
  float o = __fmaf_rn(-s, lamb2_dir<kNest>(m, v, g, w, lam, k), w);
  if (dd != 0.f) o = __fmaf_rn(-dd, w, o);
  return o;
}

template <bool kCopy, int kNest, typename GT, bool kDefer>
__device__ __forceinline__ void lamb2_chunk(const TensorPtrs& tp,
                                            const ChunkDesc& ch, float lam,
                                            float s, float dd,
                                            const LambConsts& k) {
  constexpr bool kG = kNest != 0 || kDefer;   // reads g
  float* __restrict__ w = tp.w + ch.offset;
  float* __restrict__ m = tp.m + ch.offset;
  float* __restrict__ v = tp.v + ch.offset;
  const GT* __restrict__ g = static_cast<const GT*>(tp.g) + ch.offset;
  const int n = ch.len;
  int scalar_from = 0;
  if (tp.vec_ok) {
    const int nv = n >> 2;
    for (int base = threadIdx.x; base < nv; base += kThreads * kUnroll2) {
      float4 wv[kUnroll2], mv[kUnroll2], vv[kUnroll2], gv[kUnroll2];
#pragma unroll
      for (int u = 0; u < kUnroll2; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          mv[u] = ld4_last(m + 4 * j);
          vv[u] = ld4_last(v + 4 * j);
          wv[u] = ld4_last(w + 4 * j);
          if (kG) gv[u] = ld_grad4(g + 4 * j);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll2; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          float4 o;
          if (!kG) gv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
          o.x = lamb2_elem<kNest, kDefer>(gv[u].x, mv[u].x, vv[u].x, wv[u].x, lam, s, dd, k);
          o.y = lamb2_elem<kNest, kDefer>(gv[u].y, mv[u].y, vv[u].y, wv[u].y, lam, s, dd, k);
          o.z = lamb2_elem<kNest, kDefer>(gv[u].z, mv[u].z, vv[u].z, wv[u].z, lam, s, dd, k);
          o.w = lamb2_elem<kNest, kDefer>(gv[u].w, mv[u].w, vv[u].w, wv[u].w, lam, s, dd, k);
          if (kDefer) {
            st4_last(m + 4 * j, mv[u]);
            st4_last(v + 4 * j, vv[u]);
          }
          st4_last(w + 4 * j, o);
          if (kCopy) st_copy4(tp.copy, ch.offset + 4 * j, o);
        }
      }
    }
    scalar_from = nv << 2;
  }
  for (int i = scalar_from + threadIdx.x; i < n; i += kThreads) {
    float mi = m[i], vi = v[i];
    const float gi = kG ? ld_grad1(g + i) : 0.f;
    const float o = lamb2_elem<kNest, kDefer>(gi, mi, vi, w[i], lam, s,
                                                   dd, k);
    if (kDefer) {
      m[i] = mi;
      v[i] = vi;
    }
    w[i] = o;
    if (kCopy) st_copy1(tp.copy, ch.offset + i, o);
  }
}

template <bool kCopy, int kNest, typename GT, bool kDefer>
__global__ void __launch_bounds__(kThreads)
    lamb_pass2_kernel(const StepParams p) {
  __shared__ uint32_t s_next[2];
  const StepScalars sc = *p.scal;
  if (sc.skip) return;
  // a step whose gradients held an Inf/NaN writes nothing (and does not
  // advance t); no CTA draws, so the work counter stays at 0
  if (kDefer && p.gcheck->nonfinite) return;
  const LambConsts k{p.b1, p.omb1, p.b2, p.omb2, sc.c1, sc.c2, p.eps,
                     sc.am, sc.ag, sc.bv, sc.bg};
  const bool decoupled = (p.flags & kFlagDecoupledDecay) != 0;
  if (threadIdx.x == 0) s_next[0] = atomicAdd(&p.counters[1], 1u);
  __syncthreads();
  int it = 0;
  uint32_t c = s_next[0];
  const int nc = p.n_chunks;
  while (c < (uint32_t)nc) {
    if (threadIdx.x == 0) s_next[(it + 1) & 1] = atomicAdd(&p.counters[1], 1u);
    // reverse order: the chunks pass 1 touched last are still in L2
    const ChunkDesc ch = p.chunks[nc - 1 - (int)c];
    const TensorDesc td = p.tensors[ch.tensor];
    const TensorPtrs tp = p.ptrs[ch.tensor];
    const float lamk = td.decay * p.wd;
    const float s = __double2float_rn((double)sc.lr * p.ratio[ch.tensor]);
    const float dd =
        decoupled ? __double2float_rn((double)sc.lr * (double)lamk) : 0.f;
    lamb2_chunk<kCopy, kNest, GT, kDefer>(tp, ch, decoupled ? 0.f : lamk, s,
                                          dd, k);
    __syncthreads();  // s_next[(it+1)&1] visible; old slot free to reuse
    ++it;
    c = s_next[it & 1];
  }
  if (retire(p, 1, c) && threadIdx.x == 0) {
    if (kNest && p.d_mu_product && !(p.flags & kFlagNoClose))
      *p.d_mu_product = sc.mu_prod;
    close_step(p, sc);
  }
}

// ---------------------------------------------------------------------------
// LARS pass 1 / pass 2 (u = m_t; same gradient check and deferred mode)
// ---------------------------------------------------------------------------
template <bool kGn>
__device__ __forceinline__ void lars1_elem(float g, float m, float w,
                                           float lam, float b1, float omb1,
                                           float* acc, float& o) {
  o = lars_momentum(g, m, w, lam, b1, omb1);
  acc[0] = __fmaf_rn(w, w, acc[0]);
  acc[1] = __fmaf_rn(o, o, acc[1]);
  if (kGn) {
    acc[2] = __fmaf_rn(g, g, acc[2]);
    acc[3] = __fmaf_rn(g, 0.f, acc[3]);
  }
}

template <typename GT, bool kGn>
__device__ __forceinline__ void lars1_chunk(const TensorPtrs& tp,
                                            const ChunkDesc& ch, float lam,
                                            float b1, float omb1, bool store,
                                            float* acc) {
  const float* __restrict__ w = tp.w + ch.offset;
  float* __restrict__ m = tp.m + ch.offset;
  const GT* __restrict__ g = static_cast<const GT*>(tp.g) + ch.offset;
  const int n = ch.len;
  int scalar_from = 0;
  if (tp.vec_ok) {
    const int nv = n >> 2;
    for (int base = threadIdx.x; base < nv; base += kThreads * kUnroll1) {
      float4 wv[kUnroll1], mv[kUnroll1], gv[kUnroll1];
#pragma unroll
      for (int u = 0; u < kUnroll1; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          gv[u] = ld_grad4(g + 4 * j);
          mv[u] = ld4(m + 4 * j);
          wv[u] = ld4(w + 4 * j);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll1; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          float4 o;
          lars1_elem<kGn>(gv[u].x, mv[u].x, wv[u].x, lam, b1, omb1, acc, o.x);
          lars1_elem<kGn>(gv[u].y, mv[u].y, wv[u].y, lam, b1, omb1, acc, o.y);
          lars1_elem<kGn>(gv[u].z, mv[u].z, wv[u].z, lam, b1, omb1, acc, o.z);
          lars1_elem<kGn>(gv[u].w, mv[u].w, wv[u].w, lam, b1, omb1, acc, o.w);
          if (store) st4(m + 4 * j, o);
        }
      }
    }
    scalar_from = nv << 2;
  }
  for (int i = scalar_from + threadIdx.x; i < n; i += kThreads) {
    float o;
    lars1_elem<kGn>(ld_grad1(g + i), m[i], w[i], lam, b1, omb1, acc, o);
    if (store) m[i] = o;
  }
}

template <typename GT, bool kGn>
__global__ void __launch_bounds__(kThreads)
    lars_pass1_kernel(const StepParams p) {
  __shared__ float red[4][kWarps];
  __shared__ uint32_t s_next[2];
  __shared__ int s_last;
  if (threadIdx.x == 0) {
    if (blockIdx.x == 0) {
      StepScalars sc{};
      sc.t = p.d_step ? *p.d_step : int64_t(0);
      sc.c1 = 1.f;
      sc.c2 = 1.f;
      sc.lr = step_lr(p, sc.t);
      sc.skip = 0;
      *p.scal = sc;
    }
    s_next[0] = atomicAdd(&p.counters[0], 1u);
  }
  __syncthreads();
  const bool store = !(kGn && (p.flags & kFlagSkipNonfinite));
  int it = 0;
  uint32_t c = s_next[0];
  while (c < (uint32_t)p.n_chunks) {
    if (threadIdx.x == 0) s_next[(it + 1) & 1] = atomicAdd(&p.counters[0], 1u);
    const ChunkDesc ch = p.chunks[c];
    const TensorDesc td = p.tensors[ch.tensor];
    const TensorPtrs tp = p.ptrs[ch.tensor];
    const float lam = td.decay * p.wd;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    lars1_chunk<GT, kGn>(tp, ch, lam, p.b1, p.omb1, store, acc);
    publish_chunk<kGn>(p, (int)c, ch, td, acc, red, &s_last, p.trust);
    ++it;
    c = s_next[it & 1];
  }
  retire(p, 0, c);
}

// kDefer: m still holds m_{t-1}; form m_t here (Alg. 1) and write it with w.
template <bool kCopy, typename GT, bool kDefer>
__device__ __forceinline__ void lars2_chunk(const TensorPtrs& tp,
                                            const ChunkDesc& ch, float s,
                                            float lam, float b1, float omb1) {
  float* __restrict__ w = tp.w + ch.offset;
  float* __restrict__ m = tp.m + ch.offset;
  const GT* __restrict__ g = static_cast<const GT*>(tp.g) + ch.offset;
  const int n = ch.len;
  int scalar_from = 0;
  if (tp.vec_ok) {
    const int nv = n >> 2;
    for (int base = threadIdx.x; base < nv; base += kThreads * kUnroll2) {
      float4 wv[kUnroll2], mv[kUnroll2], gv[kUnroll2];
#pragma unroll
      for (int u = 0; u < kUnroll2; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          mv[u] = ld4_last(m + 4 * j);
          wv[u] = ld4_last(w + 4 * j);
          if (kDefer) gv[u] = ld_grad4(g + 4 * j);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll2; ++u) {
        const int j = base + u * kThreads;
        if (j < nv) {
          if (kDefer) {
            mv[u].x = lars_momentum(gv[u].x, mv[u].x, wv[u].x, lam, b1, omb1);
            mv[u].y = lars_momentum(gv[u].y, mv[u].y, wv[u].y, lam, b1, omb1);
            mv[u].z = lars_momentum(gv[u].z, mv[u].z, wv[u].z, lam, b1, omb1);
            mv[u].w = lars_momentum(gv[u].w, mv[u].w, wv[u].w, lam, b1, omb1);
            st4_last(m + 4 * j, mv[u]);
          }
          float4 o;
          o.x = __fmaf_rn(-s, mv[u].x, wv[u].x);
          o.y = __fmaf_rn(-s, mv[u].y, wv[u].y);
          o.z = __fmaf_rn(-s, mv[u].z, wv[u].z);
          o.w = __fmaf_rn(-s, mv[u].w, wv[u].w);
          st4_last(w + 4 * j, o);
          if (kCopy) st_copy4(tp.copy, ch.offset + 4 * j, o);
        }
      }
    }
    scalar_from = nv << 2;
  }
  for (int i = scalar_from + threadIdx.x; i < n; i += kThreads) {
    const float wi = w[i];
    float mi = m[i];
    if (kDefer) {
      mi = lars_momentum(ld_grad1(g + i), mi, wi, lam, b1, omb1);
      m[i] = mi;
    }
    const float o = __fmaf_rn(-s, mi, wi);
    w[i] = o;
    if (kCopy) st_copy1(tp.copy, ch.offset + i, o);
  }
}

template <bool kCopy, typename GT, bool kDefer>
__global__ void __launch_bounds__(kThreads)
    lars_pass2_kernel(const StepParams p) {
  __shared__ uint32_t s_next[2];
  const StepScalars sc = *p.scal;
  if (kDefer && p.gcheck->nonfinite) return;   // skipped step: no writes
  if (threadIdx.x == 0) s_next[0] = atomicAdd(&p.counters[1], 1u);
  __syncthreads();
  int it = 0;
  uint32_t c = s_next[0];
  const int nc = p.n_chunks;
  while (c < (uint32_t)nc) {
    if (threadIdx.x == 0) s_next[(it + 1) & 1] = atomicAdd(&p.counters[1], 1u);
    const ChunkDesc ch = p.chunks[nc - 1 - (int)c];
    const TensorPtrs tp = p.ptrs[ch.tensor];
    const float s = __double2float_rn((double)sc.lr * p.ratio[ch.tensor]);
    const float lam = kDefer ? p.tensors[ch.tensor].decay * p.wd : 0.f;
    lars2_chunk<kCopy, GT, kDefer>(tp, ch, s, lam, p.b1, p.omb1);
    __syncthreads();
    ++it;
    c = s_next[it & 1];
  }
  if (retire(p, 1, c) && threadIdx.x == 0) close_step(p, sc);
}

// Every tensor's norms and trust ratio from the complete chunk slots (a
// sharded step, after the slots were exchanged): one CTA per tensor, the
// same fixed-order combine as the finaliser of pass 1, so the results equal
// an unsharded step's bit for bit.
__global__ void __launch_bounds__(kThreads)
    finalize_all_kernel(const StepParams p, double coef) {
  // one CTA per tensor, as when pass 1 finalises it: the same sums
  for (int k = (int)blockIdx.x; k < p.n_tensors; k += (int)gridDim.x) {
    const TensorDesc td = p.tensors[k];
    if (td.n_chunks > 0)
      finalize_tensor<false>(p, k, td.first_chunk, td.n_chunks, coef);
    __syncthreads();   // the finaliser's shared sums are reused
  }
}

template <typename K>
int occupancy_of(K kernel, int* blocks) {
  return (int)cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, kernel,
                                                            kThreads, 0);
}

// Variant selection from the step's flags.
template <typename GT, int kNest>
int lamb_p1(const StepParams& p, int grid, cudaStream_t s) {
  if (p.flags & (kFlagGradNorm | kFlagSkipNonfinite))
    lamb_pass1_kernel<GT, kNest, true><<<grid, kThreads, 0, s>>>(p);
  else
    lamb_pass1_kernel<GT, kNest, false><<<grid, kThreads, 0, s>>>(p);
  return (int)cudaGetLastError();
}

template <bool kCopy, int kNest, typename GT>
int lamb_p2(const StepParams& p, int grid, cudaStream_t s) {
  // plain LAMB's pass 2 does not read g: one instantiation for both types
  using GT2 = typename std::conditional<kNest != 0, GT, float>::type;
  if (p.flags & kFlagSkipNonfinite)
    lamb_pass2_kernel<kCopy, kNest, GT, true><<<grid, kThreads, 0, s>>>(p);
  else
    lamb_pass2_kernel<kCopy, kNest, GT2, false><<<grid, kThreads, 0, s>>>(p);
  return (int)cudaGetLastError();
}

template <typename GT>
int lars_p1(const StepParams& p, int grid, cudaStream_t s) {
  if (p.flags & (kFlagGradNorm | kFlagSkipNonfinite))
    lars_pass1_kernel<GT, true><<<grid, kThreads, 0, s>>>(p);
  else
    lars_pass1_kernel<GT, false><<<grid, kThreads, 0, s>>>(p);
  return (int)cudaGetLastError();
}

template <bool kCopy, typename GT>
int lars_p2(const StepParams& p, int grid, cudaStream_t s) {
  if (p.flags & kFlagSkipNonfinite)
    lars_pass2_kernel<kCopy, GT, true><<<grid, kThreads, 0, s>>>(p);
  else
    lars_pass2_kernel<kCopy, float, false><<<grid, kThreads, 0, s>>>(p);
  return (int)cudaGetLastError();
}

}  // namespace

int launch_lamb_pass1(const StepParams& p, int nest, int grad_bf16, int grid,
                      void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch ((nest == 2 ? 4 : nest == 1 ? 2 : 0) | (grad_bf16 ? 1 : 0)) {
    case 0: return lamb_p1<float, 0>(p, grid, s);
    case 1: return lamb_p1<__nv_bfloat16, 0>(p, grid, s);
    case 2: return lamb_p1<float, 1>(p, grid, s);
    case 3: return lamb_p1<__nv_bfloat16, 1>(p, grid, s);
    case 4: return lamb_p1<float, 2>(p, grid, s);
    default: return lamb_p1<__nv_bfloat16, 2>(p, grid, s);
  }
}

int launch_lamb_pass2(const StepParams& p, int nest, int grad_bf16,
                      int copy_bf16, int grid, void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch ((nest == 2 ? 8 : nest == 1 ? 4 : 0) | (grad_bf16 ? 2 : 0) |
          (copy_bf16 ? 1 : 0)) {
    case 0: return lamb_p2<false, 0, float>(p, grid, s);
    case 1: return lamb_p2<true, 0, float>(p, grid, s);
    case 2: return lamb_p2<false, 0, __nv_bfloat16>(p, grid, s);
    case 3: return lamb_p2<true, 0, __nv_bfloat16>(p, grid, s);
    case 4: return lamb_p2<false, 1, float>(p, grid, s);
    case 5: return lamb_p2<true, 1, float>(p, grid, s);
    case 6: return lamb_p2<false, 1, __nv_bfloat16>(p, grid, s);
    case 7: return lamb_p2<true, 1, __nv_bfloat16>(p, grid, s);
    case 8: return lamb_p2<false, 2, float>(p, grid, s);
    case 9: return lamb_p2<true, 2, float>(p, grid, s);
    case 10: return lamb_p2<false, 2, __nv_bfloat16>(p, grid, s);
    default: return lamb_p2<true, 2, __nv_bfloat16>(p, grid, s);
  }
}

int launch_lars_pass1(const StepParams& p, int grad_bf16, int grid,
                      void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  return grad_bf16 ? lars_p1<__nv_bfloat16>(p, grid, s)
                   : lars_p1<float>(p, grid, s);
}

int launch_lars_pass2(const StepParams& p, int grad_bf16, int copy_bf16,
                      int grid, void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch ((grad_bf16 ? 2 : 0) | (copy_bf16 ? 1 : 0)) {
    case 0: return lars_p2<false, float>(p, grid, s);
    case 1: return lars_p2<true, float>(p, grid, s);
    case 2: return lars_p2<false, __nv_bfloat16>(p, grid, s);
    default: return lars_p2<true, __nv_bfloat16>(p, grid, s);
  }
}

int launch_finalize_all(const StepParams& p, double coef, void* stream) {
  const int grid = p.n_tensors < 4096 ? p.n_tensors : 4096;
  finalize_all_kernel<<<grid < 1 ? 1 : grid, kThreads, 0,
                        static_cast<cudaStream_t>(stream)>>>(p, coef);
  return (int)cudaGetLastError();
}

int occupancy_lamb_pass1(int grad_bf16, int* blocks) {
  return grad_bf16
             ? occupancy_of(lamb_pass1_kernel<__nv_bfloat16, 0, false>, blocks)
             : occupancy_of(lamb_pass1_kernel<float, 0, false>, blocks);
}
int occupancy_lamb_pass2(int copy_bf16, int* blocks) {
  return copy_bf16
             ? occupancy_of(lamb_pass2_kernel<true, 0, float, false>, blocks)
             : occupancy_of(lamb_pass2_kernel<false, 0, float, false>, blocks);
}
int occupancy_lars_pass1(int grad_bf16, int* blocks) {
  return grad_bf16 ? occupancy_of(lars_pass1_kernel<__nv_bfloat16, false>, blocks)
                   : occupancy_of(lars_pass1_kernel<float, false>, blocks);
}
int occupancy_lars_pass2(int copy_bf16, int* blocks) {
  return copy_bf16 ? occupancy_of(lars_pass2_kernel<true, float, false>, blocks)
                   : occupancy_of(lars_pass2_kernel<false, float, false>, blocks);
}

}  // namespace lamb
