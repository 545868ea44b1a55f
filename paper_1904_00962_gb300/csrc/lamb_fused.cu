// sm_103a kernel of the single-touch LAMB / LARS step (one persistent
// launch per step; see the comment at the top of the kernel section).
#include "lamb_device.cuh"

namespace lamb {
namespace {

// ---------------------------------------------------------------------------
// Single-touch fused step (one persistent kernel, warps are the workers)
//
// Items are drawn in schedule order from counters[2].  A pass-1 item runs one
// fused chunk (512 elements) through Alg. 2's moment and ratio lines (Alg. 1
// for LARS), stores the new m, v and publishes the chunk's sums; the warp that
// completes a group of 32 chunks sums them (fp64, fixed order), and the warp
// that completes a tensor's last group computes its norms and trust ratio and
// releases ready[k] = epoch.  A pass-2 item applies the update once ready[k]
// == epoch.  Pass-2 items of a tensor come after all its pass-1 items in the
// schedule and items are drawn in order, so the earliest unfinished item never
// waits on anything unfinished: the kernel cannot deadlock.  A wait still
// gives up after ~0.5 s, sets a status bit and makes every other waiter of
// the same launch give up at once.
//
// Memory pipeline: every warp owns a ring of kStages shared-memory stages and
// prefetches the operands of its next items with cp.async while it computes
// the current one, so many bytes are in flight without holding registers.  A
// pass-2 item is prefetched only if its tensor's norms are already final when
// its stage is filled (its m, v come from other warps' pass-1 stores);
// otherwise, and for tail chunks and unaligned tensors, the item reads global
// memory directly when its turn comes.  The control traffic (draws, item
// descriptors, ready flags, tickets) is pipelined as described at the warp
// worker below.
//
// L2 policy: pass-1 loads/stores of m, v, w of "resident" tensors (those
// whose state fits the L2 budget) are evict_last, so pass 2 -- about one
// wave later -- finds them in L2; gradients and all pass-2 traffic are
// evict_first.
// ---------------------------------------------------------------------------
constexpr int kFusedThreads = 256;                     // 8 warps per CTA
constexpr int kFusedWarps = kFusedThreads / 32;
constexpr int kStages = 3;                             // prefetch depth per warp
constexpr int kPktsPerLane = kFusedChunk / 4 / 32;     // 4-element packets
static_assert(kPktsPerLane * 4 * 32 == kFusedChunk, "fused chunk shape");
constexpr uint32_t kSpinLimit = 1u << 21;              // x <= 256 ns ~ 0.5 s

// stage layout: m | v (LAMB only) | w | g
template <bool kLars, typename GT>
__host__ __device__ constexpr int stage_bytes() {
  return kFusedChunk * (4 * (kLars ? 2 : 3) + (int)sizeof(GT));
}
template <bool kLars, typename GT>
__host__ __device__ constexpr int fused_smem_bytes() {
  return kFusedWarps * kStages * stage_bytes<kLars, GT>();
}
constexpr int kOffM = 0;
constexpr int kOffV = 4 * kFusedChunk;
template <bool kLars> __host__ __device__ constexpr int off_w() {
  return 4 * kFusedChunk * (kLars ? 1 : 2);
}
template <bool kLars> __host__ __device__ constexpr int off_g() {
  return 4 * kFusedChunk * (kLars ? 2 : 3);
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ float4 ldp4(const float* p, uint64_t pol) {
  float4 r;
  asm volatile(
      "ld.global.L1::no_allocate.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %5;"
      : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
      : "l"(p), "l"(pol));
  return r;
}
__device__ __forceinline__ void stp4(float* p, float4 v, uint64_t pol) {
  asm volatile(
      "st.global.L1::no_allocate.L2::cache_hint.v4.f32 [%0], {%1,%2,%3,%4}, %5;"
      ::"l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "l"(pol)
      : "memory");
}
__device__ __forceinline__ float4 ldp_grad4(const float* p, uint64_t pol) {
  return ldp4(p, pol);
}
__device__ __forceinline__ float4 unpack_bf16x4(uint32_t a, uint32_t b) {
  return make_float4(__uint_as_float(a << 16), __uint_as_float(a & 0xffff0000u),
                     __uint_as_float(b << 16), __uint_as_float(b & 0xffff0000u));
}
__device__ __forceinline__ float4 ldp_grad4(const __nv_bfloat16* p,
                                            uint64_t pol) {
  uint32_t a, b;
  asm volatile(
      "ld.global.L1::no_allocate.L2::cache_hint.v2.u32 {%0,%1}, [%2], %3;"
      : "=r"(a), "=r"(b)
      : "l"(p), "l"(pol));
  return unpack_bf16x4(a, b);
}
// gradient packet j of a stage
__device__ __forceinline__ float4 lds_grad4(const char* gbase, int j,
                                            const float*) {
  return *reinterpret_cast<const float4*>(gbase + 16 * j);
}
__device__ __forceinline__ float4 lds_grad4(const char* gbase, int j,
                                            const __nv_bfloat16*) {
  const uint2 u = *reinterpret_cast<const uint2*>(gbase + 8 * j);
  return unpack_bf16x4(u.x, u.y);
}
__device__ __forceinline__ void stp_copy4(void* base, int64_t i, float4 x,
                                          uint64_t pol) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(x.x, x.y);
  const __nv_bfloat162 hi = __floats2bfloat162_rn(x.z, x.w);
  const uint32_t a = *reinterpret_cast<const uint32_t*>(&lo);
  const uint32_t b = *reinterpret_cast<const uint32_t*>(&hi);
  asm volatile(
      "st.global.L1::no_allocate.L2::cache_hint.v2.u32 [%0], {%1,%2}, %3;"
      ::"l"(static_cast<__nv_bfloat16*>(base) + i), "r"(a), "r"(b), "l"(pol)
      : "memory");
}
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async16(uint32_t saddr, const void* g,
                                           uint64_t pol) {
  asm volatile(
      "cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2;"
      ::"r"(saddr), "l"(g), "l"(pol)
      : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p)
               : "memory");
  return v;
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v)
               : "memory");
}
__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;"
               : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_down_sync(0xffffffffu, x, o);
  return x;
}

// Element of the fused pass 1: LAMB (Alg. 2) or LARS (Alg. 1) moment update,
// then the direction u whose norm the trust ratio needs.
template <bool kLars>
__device__ __forceinline__ void fused1_elem(float g, float& m, float& v,
                                            float w, float lam,
                                            const LambConsts& k, float& sw,
                                            float& su) {
  float u;
  if (kLars) {
    m = lars_momentum(g, m, w, lam, k.b1, k.omb1);
    u = m;
  } else {
    lamb_moments(g, m, v, k);
    u = lamb_direction(m, v, w, lam, k);
  }
  sw = __fmaf_rn(w, w, sw);
  su = __fmaf_rn(u, u, su);
}

template <bool kLars>
__device__ __forceinline__ float fused2_dir(float m, float v, float w,
                                            float lam, const LambConsts& k) {
  return kLars ? m : lamb_direction(m, v, w, lam, k);
}

template <bool kLars>
__device__ __forceinline__ void fused1_pkt(float4 gv, float4& mv, float4& vv,
                                           float4 wv, float lam,
                                           const LambConsts& k, float& sw,
                                           float& su) {
  fused1_elem<kLars>(gv.x, mv.x, vv.x, wv.x, lam, k, sw, su);
  fused1_elem<kLars>(gv.y, mv.y, vv.y, wv.y, lam, k, sw, su);
  fused1_elem<kLars>(gv.z, mv.z, vv.z, wv.z, lam, k, sw, su);
  fused1_elem<kLars>(gv.w, mv.w, vv.w, wv.w, lam, k, sw, su);
}

template <bool kLars>
__device__ __forceinline__ float4 fused2_pkt(float4 mv, float4 vv, float4 wv,
                                             float s, float lam,
                                             const LambConsts& k) {
  float4 o;
  o.x = __fmaf_rn(-s, fused2_dir<kLars>(mv.x, vv.x, wv.x, lam, k), wv.x);
  o.y = __fmaf_rn(-s, fused2_dir<kLars>(mv.y, vv.y, wv.y, lam, k), wv.y);
  o.z = __fmaf_rn(-s, fused2_dir<kLars>(mv.z, vv.z, wv.z, lam, k), wv.z);
  o.w = __fmaf_rn(-s, fused2_dir<kLars>(mv.w, vv.w, wv.w, lam, k), wv.w);
  return o;
}

__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p)
               : "memory");
  return v;
}
__device__ __forceinline__ void fence_acq_rel() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
}

// Issue the cp.async copies of one full, aligned chunk into `stage`: m, v
// (LAMB), w, and for pass 1 the gradient.
template <bool kLars, typename GT>
__device__ __forceinline__ void fused_prefetch_ops(
    const TensorPtrs& tp, int64_t off, bool pass2, bool resident, char* stage,
    uint64_t pol_first, uint64_t pol_last, int lane) {
  const uint64_t pol = (!pass2 && resident) ? pol_last : pol_first;
  const uint32_t s = smem_u32(stage);
#pragma unroll
  for (int u = 0; u < kPktsPerLane; ++u) {
    const int j = lane + 32 * u;                    // 16-byte piece index
    cp_async16(s + kOffM + 16 * j, tp.m + off + 4 * j, pol);
    if (!kLars) cp_async16(s + kOffV + 16 * j, tp.v + off + 4 * j, pol);
    cp_async16(s + off_w<kLars>() + 16 * j, tp.w + off + 4 * j, pol);
  }
  if (!pass2) {
    const char* g = reinterpret_cast<const char*>(
        static_cast<const GT*>(tp.g) + off);
    constexpr int kGPieces = kFusedChunk * (int)sizeof(GT) / 16;
#pragma unroll
    for (int u = 0; u < kGPieces / 32; ++u) {
      const int j = lane + 32 * u;
      cp_async16(s + off_g<kLars>() + 16 * j, g + 16 * j, pol_first);
    }
  }
}

// Pass 1 of a staged chunk: new m, v into registers, sums of w^2 and u^2.
template <bool kLars, typename GT>
__device__ __forceinline__ void fused1_from_stage(const char* stage,
                                                  float lam,
                                                  const LambConsts& k,
                                                  float4* mo, float4* vo,
                                                  float& sw, float& su,
                                                  int lane) {
  const GT* tag = nullptr;
#pragma unroll
  for (int u = 0; u < kPktsPerLane; ++u) {
    const int j = lane + 32 * u;
    mo[u] = *reinterpret_cast<const float4*>(stage + kOffM + 16 * j);
    vo[u] = kLars ? make_float4(0.f, 0.f, 0.f, 0.f)
                  : *reinterpret_cast<const float4*>(stage + kOffV + 16 * j);
    const float4 wv =
        *reinterpret_cast<const float4*>(stage + off_w<kLars>() + 16 * j);
    const float4 gv = lds_grad4(stage + off_g<kLars>(), j, tag);
    fused1_pkt<kLars>(gv, mo[u], vo[u], wv, lam, k, sw, su);
  }
}

template <bool kLars>
__device__ __forceinline__ void fused1_store(const TensorPtrs& tp,
                                             int64_t off, const float4* mo,
                                             const float4* vo,
                                             uint64_t pol_keep, int lane) {
#pragma unroll
  for (int u = 0; u < kPktsPerLane; ++u) {
    const int j = lane + 32 * u;
    stp4(tp.m + off + 4 * j, mo[u], pol_keep);
    if (!kLars) stp4(tp.v + off + 4 * j, vo[u], pol_keep);
  }
}

// Pass 1 straight from global memory (tail chunks, unaligned tensors).
template <bool kLars, typename GT>
__device__ __forceinline__ void fused1_direct(const TensorPtrs& tp,
                                              int64_t off, int len, float lam,
                                              const LambConsts& k, float& sw,
                                              float& su, uint64_t pol_first,
                                              uint64_t pol_keep, int lane) {
  float* __restrict__ m = tp.m + off;
  float* __restrict__ v = kLars ? nullptr : tp.v + off;
  const float* __restrict__ w = tp.w + off;
  const GT* __restrict__ g = static_cast<const GT*>(tp.g) + off;
  int scalar_from = 0;
  if (tp.vec_ok) {
    const int nv = len >> 2;
#pragma unroll 1
    for (int base = lane; base < nv; base += 64) {
      float4 wv[2], mv[2], vv[2], gv[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int j = base + 32 * u;
        if (j < nv) {
          gv[u] = ldp_grad4(g + 4 * j, pol_first);
          mv[u] = ldp4(m + 4 * j, pol_keep);
          if (!kLars) vv[u] = ldp4(v + 4 * j, pol_keep);
          wv[u] = ldp4(w + 4 * j, pol_keep);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int j = base + 32 * u;
        if (j < nv) {
          fused1_pkt<kLars>(gv[u], mv[u], vv[u], wv[u], lam, k, sw, su);
          stp4(m + 4 * j, mv[u], pol_keep);
          if (!kLars) stp4(v + 4 * j, vv[u], pol_keep);
        }
      }
    }
    scalar_from = nv << 2;
  }
  for (int i = scalar_from + lane; i < len; i += 32) {
    float mi = m[i];
    float vi = kLars ? 0.f : v[i];
    fused1_elem<kLars>(ld_grad1(g + i), mi, vi, w[i], lam, k, sw, su);
    m[i] = mi;
    if (!kLars) v[i] = vi;
  }
}

// Pass 2 of a staged chunk: new w into registers.
template <bool kLars>
__device__ __forceinline__ void fused2_from_stage(const char* stage, float s,
                                                  float lam,
                                                  const LambConsts& k,
                                                  float4* wo, int lane) {
#pragma unroll
  for (int u = 0; u < kPktsPerLane; ++u) {
    const int j = lane + 32 * u;
    const float4 mv = *reinterpret_cast<const float4*>(stage + kOffM + 16 * j);
    const float4 vv = kLars ? make_float4(0.f, 0.f, 0.f, 0.f)
                            : *reinterpret_cast<const float4*>(stage + kOffV + 16 * j);
    const float4 wv =
        *reinterpret_cast<const float4*>(stage + off_w<kLars>() + 16 * j);
    wo[u] = fused2_pkt<kLars>(mv, vv, wv, s, lam, k);
  }
}

template <bool kCopy>
__device__ __forceinline__ void fused2_store(const TensorPtrs& tp,
                                             int64_t off, const float4* wo,
                                             uint64_t pol_first, int lane) {
#pragma unroll
  for (int u = 0; u < kPktsPerLane; ++u) {
    const int j = lane + 32 * u;
    stp4(tp.w + off + 4 * j, wo[u], pol_first);
    if (kCopy) stp_copy4(tp.copy, off + 4 * j, wo[u], pol_first);
  }
}

// Pass 2 straight from global memory.
template <bool kLars, bool kCopy>
__device__ __forceinline__ void fused2_direct(const TensorPtrs& tp,
                                              int64_t off, int len, float s,
                                              float lam, const LambConsts& k,
                                              uint64_t pol_first, int lane) {
  float* __restrict__ w = tp.w + off;
  const float* __restrict__ m = tp.m + off;
  const float* __restrict__ v = kLars ? nullptr : tp.v + off;
  int scalar_from = 0;
  if (tp.vec_ok) {
    const int nv = len >> 2;
#pragma unroll 1
    for (int base = lane; base < nv; base += 64) {
      float4 wv[2], mv[2], vv[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int j = base + 32 * u;
        if (j < nv) {
          mv[u] = ldp4(m + 4 * j, pol_first);
          if (!kLars) vv[u] = ldp4(v + 4 * j, pol_first);
          wv[u] = ldp4(w + 4 * j, pol_first);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int j = base + 32 * u;
        if (j < nv) {
          const float4 o = fused2_pkt<kLars>(mv[u], vv[u], wv[u], s, lam, k);
          stp4(w + 4 * j, o, pol_first);
          if (kCopy) stp_copy4(tp.copy, off + 4 * j, o, pol_first);
        }
      }
    }
    scalar_from = nv << 2;
  }
  for (int i = scalar_from + lane; i < len; i += 32) {
    const float wi = w[i];
    const float o = __fmaf_rn(
        -s, fused2_dir<kLars>(m[i], kLars ? 0.f : v[i], wi, lam, k), wi);
    w[i] = o;
    if (kCopy) st_copy1(tp.copy, off + i, o);
  }
}

// The warp whose ticket completed group `gl` of tensor `tensor`: fixed-order
// fp64 sum of the group's chunk sums; the warp that completes the tensor's
// last group computes its norms and trust ratio and releases ready[tensor].
template <bool kLars>
__device__ __forceinline__ void fused_group_combine(const StepParams& p,
                                                 const FusedParams& f,
                                                 const FusedTensor& ft,
                                                 int tensor, int gl, int gsize,
                                                 uint32_t epoch, int lane) {
  __syncwarp();
  const int group = ft.first_group + gl;
  double aw = 0.0, au = 0.0;
  if (lane < gsize) {
    const float2 s = __ldcg(&f.fslots[ft.first_chunk + gl * kGroup + lane]);
    aw = (double)s.x;
    au = (double)s.y;
  }
  aw = warp_sum_d(aw);
  au = warp_sum_d(au);
  uint32_t last = 0;
  if (lane == 0) {
    f.gslots[group] = make_double2(aw, au);
    f.gtickets[group] = 0u;
    last = atom_add_acq_rel(&f.tickets[tensor], 1u) + 1u ==
           (uint32_t)ft.n_groups;
  }
  if (!__shfl_sync(0xffffffffu, last, 0)) return;
  __syncwarp();
  double tw = 0.0, tu = 0.0;
  for (int i = lane; i < ft.n_groups; i += 32) {
    const double2 s = __ldcg(&f.gslots[ft.first_group + i]);
    tw += s.x;
    tu += s.y;
  }
  tw = warp_sum_d(tw);
  tu = warp_sum_d(tu);
  if (lane == 0) {
    const double wn = sqrt(tw), un = sqrt(tu);
    double rho = 1.0;
    if (!(wn == 0.0 || un == 0.0))
      rho = (kLars ? p.trust : 1.0) * phi_of(wn, p) / un;
    p.ratio[tensor] = rho;
    p.wnorm[tensor] = wn;
    p.unorm[tensor] = un;
    if (!isfinite(tw) || !isfinite(tu)) atomicOr(p.status, kStatusNonfinite);
    f.tickets[tensor] = 0u;
    st_release(&f.ready[tensor], epoch);
  }
}

// Bounded wait of a pass-2 item for its tensor's norms (all lanes).
__device__ __forceinline__ bool fused_wait(const StepParams& p,
                                           const FusedParams& f, int tensor,
                                           uint32_t epoch, int lane) {
  uint32_t ok = 1;
  if (lane == 0) {
    uint32_t spins = 0, ns = 32;
    while (ld_acquire(&f.ready[tensor]) != epoch) {
      // give up after ~0.5 s, or at once if another warp of this launch
      // already gave up (counters[4] holds the epoch of an aborted launch)
      if (++spins > kSpinLimit ||
          *reinterpret_cast<volatile uint32_t*>(&p.counters[4]) == epoch) {
        ok = 0;
        atomicOr(p.status, kStatusWaitTimeout);
        atomicExch(&p.counters[4], epoch);
        break;
      }
      __nanosleep(ns);
      if (ns < 256) ns <<= 1;
    }
  }
  if (!__shfl_sync(0xffffffffu, ok, 0)) return false;
  __syncwarp();
  (void)ld_acquire(&f.ready[tensor]);               // per-lane acquire
  return true;
}

// ---------------------------------------------------------------------------
// The warp worker.  Per warp:
//   * a data ring of kStages shared-memory stages; the item in a stage had
//     its operands prefetched with cp.async kStages items earlier;
//   * a control pipeline one item deep per step: the draw atomic, the item
//     descriptor load and (pass 2) a relaxed load of the tensor's ready flag
//     are each issued one item before their results are used;
//   * a deferred publish: a pass-1 item's ticket is taken one item later (its
//     stores are long complete, so the release costs little), and the
//     ticket's answer is looked at one item after that.
// Before any wait the warp flushes its deferred publishes, so it never waits
// for work it holds itself.
// ---------------------------------------------------------------------------
struct PubState {
  uint32_t tensor, index;   // pass-1 chunk whose sums are held (publish)
  float sw, su;             // its sums, valid in lane 0
  uint32_t chk_tensor, chk_index;   // chunk whose ticket awaits its check
  uint32_t ticket;          // that ticket's answer (lane 0)
  bool pub, chk;            // a publish is pending / a check is pending
};

__device__ __forceinline__ uint2 invalid_desc() {
  return make_uint2(0xffffffffu, 0u);
}

template <bool kLars>
__device__ __forceinline__ void fused_check(const StepParams& p,
                                            const FusedParams& f,
                                            PubState& ps, uint32_t epoch,
                                            int lane) {
  if (!ps.chk) return;
  const FusedTensor ft = f.ftensors[ps.chk_tensor];
  const int gl = (int)ps.chk_index / kGroup;
  const int gsize = min(kGroup, ft.n_chunks - gl * kGroup);
  const uint32_t last =
      __shfl_sync(0xffffffffu, ps.ticket + 1u == (uint32_t)gsize, 0);
  ps.chk = false;
  if (last) fused_group_combine<kLars>(p, f, ft, (int)ps.chk_tensor, gl,
                                       gsize, epoch, lane);
}

__device__ __forceinline__ void fused_publish_now(const FusedParams& f,
                                                  PubState& ps, int lane) {
  if (!ps.pub) return;
  if (lane == 0) {
    const FusedTensor ft = f.ftensors[ps.tensor];
    f.fslots[ft.first_chunk + ps.index] = make_float2(ps.sw, ps.su);
    // release: this warp's stores of the chunk's m, v and the slot
    ps.ticket = atom_add_acq_rel(
        &f.gtickets[ft.first_group + (int)ps.index / kGroup], 1u);
  }
  ps.chk_tensor = ps.tensor;
  ps.chk_index = ps.index;
  ps.pub = false;
  ps.chk = true;
}

template <bool kLars>
__device__ __forceinline__ void fused_publish_step(const StepParams& p,
                                                   const FusedParams& f,
                                                   PubState& ps,
                                                   uint32_t epoch, int lane) {
  fused_check<kLars>(p, f, ps, epoch, lane);
  fused_publish_now(f, ps, lane);
}

template <bool kLars>
__device__ __forceinline__ void fused_flush(const StepParams& p,
                                            const FusedParams& f,
                                            PubState& ps, uint32_t epoch,
                                            int lane) {
  fused_publish_step<kLars>(p, f, ps, epoch, lane);
  fused_check<kLars>(p, f, ps, epoch, lane);
}

template <bool kLars, typename GT, bool kCopy>
__global__ void __launch_bounds__(kFusedThreads, 1)
    fused_step_kernel(const StepParams p, const FusedParams f) {
  extern __shared__ __align__(128) char fused_smem[];
  __shared__ LambConsts s_k;
  __shared__ float s_lr;
  __shared__ int s_skip;
  __shared__ uint32_t s_epoch;
  __shared__ int64_t s_t;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  __shared__ float s_c2;
  const bool bc = !kLars && (p.flags & kFlagBiasCorrection) != 0;
  if (threadIdx.x == 32) {  // Alg. 2 bias correction of v, beside c1
    const int64_t t = p.d_step ? *p.d_step : int64_t(1);
    s_c2 = (bc && t >= 1) ? (float)(1.0 / (1.0 - pow_from_log2(
                                p.log2_beta2, (double)t)))
                          : 1.f;
  }
  float c1 = 1.f;
  int64_t t = 1;
  int skip = 0;
  if (threadIdx.x == 0) {
    t = p.d_step ? *p.d_step : int64_t(1);
    skip = (bc && t < 1) ? 1 : 0;
    if (bc && !skip)
      c1 = (float)(1.0 / (1.0 - pow_from_log2(p.log2_beta1, (double)t)));
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const float c2 = s_c2;
    s_k = LambConsts{p.b1, p.omb1, p.b2, p.omb2, c1, c2, p.eps};
    s_lr = step_lr(p, t);
    s_skip = skip;
    s_t = t;
    s_epoch = *reinterpret_cast<volatile uint32_t*>(&p.counters[3]);
    if (blockIdx.x == 0) {
      StepScalars sc{};
      sc.t = t;
      sc.c1 = c1;
      sc.c2 = c2;
      sc.lr = s_lr;
      sc.skip = skip;
      *p.scal = sc;
      if (skip) atomicOr(p.status, kStatusBadStep);
    }
  }
  __syncthreads();
  if (s_skip) return;
  const LambConsts k = s_k;
  const float lr = s_lr;
  const uint32_t epoch = s_epoch;
  const uint64_t pol_first = policy_evict_first();
  const uint64_t pol_last = policy_evict_last();
  const uint32_t n_items = (uint32_t)f.n_items;
  constexpr int kSB = stage_bytes<kLars, GT>();
  char* ring = fused_smem + warp * kStages * kSB;

  // ---- control pipeline --------------------------------------------------
  // Each warp draws indices until it gets one >= n_items, then stops, so it
  // draws exactly one such index.
  uint32_t last_drawn = 0;
  bool drawing = true;
  auto draw = [&]() -> uint32_t {
    if (!drawing) return n_items;
    uint32_t v = 0;
    if (lane == 0) v = atomicAdd(&p.counters[2], 1u);
    v = __shfl_sync(0xffffffffu, v, 0);
    if (v >= n_items) {
      drawing = false;
      last_drawn = v;
    }
    return v;
  };
  auto load_desc = [&](uint32_t i) -> uint2 {
    return i < n_items ? __ldg(&f.items[i]) : invalid_desc();
  };
  auto ready_load = [&](uint2 d) -> uint32_t {
    if (d.x == 0xffffffffu || (d.x & 1u) == 0u) return 0u;
    return ld_relaxed(&f.ready[d.x >> 1]);
  };
  uint32_t idx_a = draw();
  uint2 desc_b = load_desc(idx_a);
  idx_a = draw();
  uint2 desc_c = desc_b;
  uint32_t rdy_c = ready_load(desc_c);
  desc_b = load_desc(idx_a);
  idx_a = draw();
  uint32_t synced = 0xffffffffu;   // tensor whose norms this warp acquired

  uint2 sd[kStages];
  bool staged[kStages];
  // fill stage s with desc_c, then advance the control pipeline
  auto fill_advance = [&](int s) {
    sd[s] = desc_c;
    staged[s] = false;
    if (desc_c.x != 0xffffffffu) {
      const bool p2 = (desc_c.x & 1u) != 0u;
      const uint32_t tensor = desc_c.x >> 1;
      const FusedTensor ft = f.ftensors[tensor];
      const TensorPtrs tp = p.ptrs[tensor];
      const int64_t off = (int64_t)desc_c.y * kFusedChunk;
      bool go = tp.vec_ok && ft.numel - off >= kFusedChunk;
      if (go && p2) {
        go = __shfl_sync(0xffffffffu, rdy_c == epoch, 0) != 0;
        if (go && tensor != synced) {
          fence_acq_rel();           // acquire: the relaxed load saw the release
          synced = tensor;
        }
      }
      if (go) {
        fused_prefetch_ops<kLars, GT>(tp, off, p2, ft.resident != 0u,
                                      ring + s * kSB, pol_first, pol_last,
                                      lane);
        staged[s] = true;
      }
    }
    cp_async_commit();
    desc_c = desc_b;
    rdy_c = ready_load(desc_c);
    desc_b = load_desc(idx_a);
    idx_a = draw();
  };
#pragma unroll
  for (int s = 0; s < kStages; ++s) fill_advance(s);

  // pass-2 item of this warp whose tensor was not final when its turn came
  uint2 parked = invalid_desc();
  // run a pass-2 item from global memory once its tensor is known final
  auto run_direct_p2 = [&](uint2 d) {
    const uint32_t tensor = d.x >> 1;
    if (tensor != synced) {
      fence_acq_rel();                 // acquire: the relaxed load saw it
      synced = tensor;
    }
    const FusedTensor ft = f.ftensors[tensor];
    const TensorPtrs tp = p.ptrs[tensor];
    const int64_t off = (int64_t)d.y * kFusedChunk;
    const int64_t rem = ft.numel - off;
    const int len = (int)(rem < kFusedChunk ? rem : kFusedChunk);
    const float s2 = __double2float_rn((double)lr * __ldcg(&p.ratio[tensor]));
    fused2_direct<kLars, kCopy>(tp, off, len, s2, ft.decay * p.wd, k,
                                pol_first, lane);
  };
  // the same after a bounded wait (callers flush their publishes first)
  auto wait_direct_p2 = [&](uint2 d) {
    const uint32_t tensor = d.x >> 1;
    if (fused_wait(p, f, (int)tensor, epoch, lane)) {
      synced = tensor;
      run_direct_p2(d);
    }
  };

  PubState ps;
  ps.pub = ps.chk = false;
  ps.tensor = ps.index = ps.chk_tensor = ps.chk_index = 0u;
  ps.sw = ps.su = 0.f;
  ps.ticket = 0u;

  bool done = false;
  while (!done) {
#pragma unroll
    for (int s = 0; s < kStages; ++s) {
      const uint2 d = sd[s];
      if (d.x == 0xffffffffu) {
        done = true;
        break;
      }
      char* stage = ring + s * kSB;
      cp_async_wait<kStages - 1>();   // this stage's copies have landed
      __syncwarp();
      const bool p2 = (d.x & 1u) != 0u;
      const uint32_t tensor = d.x >> 1;
      const FusedTensor ft = f.ftensors[tensor];
      const TensorPtrs tp = p.ptrs[tensor];
      const int64_t off = (int64_t)d.y * kFusedChunk;
      const int64_t rem = ft.numel - off;
      const int len = (int)(rem < kFusedChunk ? rem : kFusedChunk);
      const float lam = ft.decay * p.wd;
      if (!p2) {
        const uint64_t pol_keep = ft.resident ? pol_last : pol_first;
        float sw = 0.f, su = 0.f;
        if (staged[s]) {
          float4 mo[kPktsPerLane], vo[kPktsPerLane];
          fused1_from_stage<kLars, GT>(stage, lam, k, mo, vo, sw, su, lane);
          __syncwarp();               // every lane is done with the stage
          fill_advance(s);
          fused_publish_step<kLars>(p, f, ps, epoch, lane);
          fused1_store<kLars>(tp, off, mo, vo, pol_keep, lane);
        } else {
          __syncwarp();
          fill_advance(s);
          fused_publish_step<kLars>(p, f, ps, epoch, lane);
          fused1_direct<kLars, GT>(tp, off, len, lam, k, sw, su, pol_first,
                                   pol_keep, lane);
        }
        ps.sw = warp_sum(sw);
        ps.su = warp_sum(su);
        ps.tensor = tensor;
        ps.index = d.y;
        ps.pub = true;
      } else {
        const float s_upd =
            staged[s] ? __double2float_rn((double)lr * __ldcg(&p.ratio[tensor]))
                      : 0.f;
        if (staged[s]) {
          float4 wo[kPktsPerLane];
          fused2_from_stage<kLars>(stage, s_upd, lam, k, wo, lane);
          __syncwarp();
          fill_advance(s);
          fused_publish_step<kLars>(p, f, ps, epoch, lane);
          fused2_store<kCopy>(tp, off, wo, pol_first, lane);
        } else {
          __syncwarp();
          fill_advance(s);
          fused_publish_step<kLars>(p, f, ps, epoch, lane);
          // every lane loads the flag itself (one broadcast access) before
          // its acquire fence; lane 0's value makes the decision uniform
          const uint32_t r = __shfl_sync(0xffffffffu,
                                         ld_relaxed(&f.ready[tensor]), 0);
          if (r == epoch) {               // became final since the fill
            run_direct_p2(d);
          } else {
            // Not final yet: park it instead of waiting, so this warp keeps
            // working (and publishing) its later pass-1 items.  With the
            // parking slot taken, finish the parked item first.
            if (parked.x != 0xffffffffu) {
              fused_flush<kLars>(p, f, ps, epoch, lane);
              wait_direct_p2(parked);
            }
            parked = d;
          }
        }
      }
      // a parked item whose tensor has become final in the meantime
      if (parked.x != 0xffffffffu) {
        const uint32_t r = __shfl_sync(
            0xffffffffu, ld_relaxed(&f.ready[parked.x >> 1]), 0);
        if (r == epoch) {
          run_direct_p2(parked);
          parked = invalid_desc();
        }
      }
    }
  }
  fused_flush<kLars>(p, f, ps, epoch, lane);
  if (parked.x != 0xffffffffu) wait_direct_p2(parked);
  cp_async_wait<0>();
  // The warp that drew the last index >= n_items closes the launch.
  const uint32_t warps = gridDim.x * kFusedWarps;
  if (lane == 0 && last_drawn == n_items + warps - 1u) {
    atomicExch(&p.counters[2], 0u);
    const uint32_t ne = epoch + 1u == 0u ? 1u : epoch + 1u;
    atomicExch(&p.counters[3], ne);
    StepScalars sc{};
    sc.t = s_t;
    sc.lr = s_lr;
    close_step(p, sc);
  }
}

}  // namespace

template <bool kLars, typename GT, bool kCopy>
int launch_fused_t(const StepParams& p, const FusedParams& f, int grid,
                   cudaStream_t s) {
  fused_step_kernel<kLars, GT, kCopy>
      <<<grid, kFusedThreads, fused_smem_bytes<kLars, GT>(), s>>>(p, f);
  return (int)cudaGetLastError();
}

template <bool kLars, typename GT, bool kCopy>
int occupancy_fused_t(int* blocks) {
  // opt in to the dynamic shared memory of the stage rings (a property of
  // the function, set once; not a device setting)
  cudaError_t e = cudaFuncSetAttribute(
      fused_step_kernel<kLars, GT, kCopy>,
      cudaFuncAttributeMaxDynamicSharedMemorySize,
      fused_smem_bytes<kLars, GT>());
  if (e != cudaSuccess) return (int)e;
  return (int)cudaOccupancyMaxActiveBlocksPerMultiprocessor(
      blocks, fused_step_kernel<kLars, GT, kCopy>, kFusedThreads,
      fused_smem_bytes<kLars, GT>());
}

int launch_fused(const StepParams& p, const FusedParams& f, int lars,
                 int grad_bf16, int copy_bf16, int grid, void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch ((lars ? 4 : 0) | (grad_bf16 ? 2 : 0) | (copy_bf16 ? 1 : 0)) {
    case 0: return launch_fused_t<false, float, false>(p, f, grid, s);
    case 1: return launch_fused_t<false, float, true>(p, f, grid, s);
    case 2: return launch_fused_t<false, __nv_bfloat16, false>(p, f, grid, s);
    case 3: return launch_fused_t<false, __nv_bfloat16, true>(p, f, grid, s);
    case 4: return launch_fused_t<true, float, false>(p, f, grid, s);
    case 5: return launch_fused_t<true, float, true>(p, f, grid, s);
    case 6: return launch_fused_t<true, __nv_bfloat16, false>(p, f, grid, s);
    default: return launch_fused_t<true, __nv_bfloat16, true>(p, f, grid, s);
  }
}

int occupancy_fused(int lars, int grad_bf16, int copy_bf16, int* blocks) {
  switch ((lars ? 4 : 0) | (grad_bf16 ? 2 : 0) | (copy_bf16 ? 1 : 0)) {
    case 0: return occupancy_fused_t<false, float, false>(blocks);
    case 1: return occupancy_fused_t<false, float, true>(blocks);
    case 2: return occupancy_fused_t<false, __nv_bfloat16, false>(blocks);
    case 3: return occupancy_fused_t<false, __nv_bfloat16, true>(blocks);
    case 4: return occupancy_fused_t<true, float, false>(blocks);
    case 5: return occupancy_fused_t<true, float, true>(blocks);
    case 6: return occupancy_fused_t<true, __nv_bfloat16, false>(blocks);
    default: return occupancy_fused_t<true, __nv_bfloat16, true>(blocks);
  }
}

}  // namespace lamb
