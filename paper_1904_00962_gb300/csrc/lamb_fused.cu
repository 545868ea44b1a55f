// sm_103a kernel of the single-touch LAMB / LARS step: one persistent launch
// per step, in which the pass 2 of a tensor follows its pass 1 closely enough
// to read m, v, w back from L2 (28 instead of 40 bytes of HBM traffic per
// parameter for BERT-large's bf16 gradients and bf16 copy).
//
// Work items are fused chunks of kFusedChunk elements, pass 1 or pass 2,
// drawn in the order of a host-built schedule (planner.cpp, plan_fused): the
// pass-1 items tensor by tensor; the pass-2 block of a tensor whose state fits
// the L2 budget placed `lag` items after its last pass-1 item; the pass-2
// blocks of larger tensors at the end.
//
// One CTA per SM, warp-specialised:
//   producer   (warp 16, one lane) draws items in schedule order, keeps the
//              draws and descriptors of the next items in flight, waits for
//              a pass-2 item's tensor to be final, and stages each item's
//              operands in a ring of up to 8 shared-memory stages with TMA
//              bulk copies (cp.async.bulk) that complete on the stage's
//              mbarrier;
//   consumers  (warps 0-15, each walking the stage ring on its own) apply
//              Alg. 2 (Alg. 1 for LARS) to a staged item and store the
//              results; for a pass-1 item the last warp to finish it adds
//              the warps' sums of w^2 and u^2 in warp order and hands the
//              pair to
//   publisher  (warp 17), which stores the chunk's sums, takes the tensor's
//              ticket and, for the tensor's last chunk, combines the chunk
//              sums in a fixed order in fp64, writes rho_k and releases
//              ready[k] = epoch.
// The consumers never wait on a global atomic, and the producer never waits
// on the consumers' arithmetic except through a free stage.
//
// Deadlock freedom: every pass-2 item follows all pass-1 items of its tensor
// in the schedule, and each CTA takes its items in the order it drew them.
// The unfinished item with the smallest index therefore sits at the head of
// its CTA's pipeline with everything it depends on finished, so it always
// completes; no co-residency of the CTAs is needed.  Every wait is still
// bounded (~0.5 s): on a timeout the CTA sets LAMB_STATUS_WAIT_TIMEOUT and an
// abort word that makes every other waiter of the launch give up, waits (also
// bounded) for its own copies in flight, and returns.
//
// Memory ordering: a consumer's m, v stores -> block-scope fence and
// counter -> the last warp's mbarrier arrive (CTA scope) -> the publisher's
// acq_rel ticket (GPU scope) -> the
// finaliser's release of ready[k] -> a producer's acquire of ready[k] ->
// fence.proxy.async.global -> its TMA reads of m, v (async proxy).
//
// Identical arithmetic to the two-pass kernels (lamb_device.cuh); per-chunk
// fp32 sums and the per-tensor fp64 combine in chunk order make the result
// independent of which CTA ran which item.
#include "lamb_device.cuh"

namespace lamb {
namespace {

constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;           // 512 threads
constexpr int kProducerWarp = kConsumerWarps;             // warp 16
constexpr int kPublisherWarp = kConsumerWarps + 1;        // warp 17
constexpr int kFusedThreads = (kConsumerWarps + 2) * 32;  // 576
constexpr int kMaxStages = 8;                             // operand ring
constexpr int kStageBudget = 220 * 1024;                  // dynamic smem
constexpr int kPubSlots = 16;                             // sums ring
constexpr int kRedRing = 2 * kMaxStages;                  // partial-sum ring
constexpr int kPkts = kFusedChunk / 4 / kConsumers;       // float4 per array
static_assert(kPkts * 4 * kConsumers == kFusedChunk, "fused chunk shape");
static_assert(kPubSlots <= 32, "the publisher takes up to a warp of entries");
constexpr uint32_t kSpinLimit = 1u << 21;                 // polls, <= ~0.5 s

// stage layout: m | v (LAMB) | w | g, each kFusedChunk elements
template <bool kLars, typename GT>
__host__ __device__ constexpr int stage_bytes() {
  return kFusedChunk * (4 * (kLars ? 2 : 3) + (int)sizeof(GT));
}
// as many stages as fit the budget (7 for LAMB with bf16 g, 6 with fp32 g):
// the ring must cover the TMA latency of the items behind the one in use
template <bool kLars, typename GT>
__host__ __device__ constexpr int n_stages() {
  return kStageBudget / stage_bytes<kLars, GT>() < kMaxStages
             ? kStageBudget / stage_bytes<kLars, GT>()
             : kMaxStages;
}
template <bool kLars, typename GT>
__host__ __device__ constexpr int fused_smem_bytes() {
  return n_stages<kLars, GT>() * stage_bytes<kLars, GT>();
}
constexpr int kOffM = 0;
constexpr int kOffV = 4 * kFusedChunk;
template <bool kLars> __host__ __device__ constexpr int off_w() {
  return 4 * kFusedChunk * (kLars ? 1 : 2);
}
template <bool kLars> __host__ __device__ constexpr int off_g() {
  return 4 * kFusedChunk * (kLars ? 2 : 3);
}

// item flags in a stage descriptor
enum : uint32_t { kItemP2 = 1u, kItemDirect = 2u, kItemEnd = 4u,
                  kItemSkip = 8u, kItemResident = 16u };

struct StageDesc {      // written by the producer, read by the consumers
  TensorPtrs tp;        // the tensor's arrays (the consumers load nothing
                        // but the stage and this descriptor)
  int32_t tensor;
  int32_t index;        // fused chunk index inside the tensor
  int32_t len;          // elements in the chunk
  uint32_t flags;
  float s;              // pass 2: eta * rho_k
  float lam;            // lambda_k
  int32_t first_chunk;  // slot base and chunk count of the tensor
  int32_t n_chunks;
};

struct PubEntry {       // a pass-1 chunk's sums, consumers -> publisher
  int32_t tensor;       // -1: end of the stream
  int32_t first_chunk;  // the tensor's first fused chunk in the plan
  int32_t index;        // the chunk's index inside the tensor
  int32_t n_chunks;
  float sw, su;
};

// ---------------------------------------------------------------------------
// PTX helpers: cache policies, stores with hints, mbarriers, TMA bulk
// copies, scoped atomics
// ---------------------------------------------------------------------------
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
__device__ __forceinline__ void stp4(float* p, float4 v, uint64_t pol) {
  asm volatile(
      "st.global.L1::no_allocate.L2::cache_hint.v4.f32 [%0], {%1,%2,%3,%4}, %5;"
      ::"l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "l"(pol)
      : "memory");
}
__device__ __forceinline__ float4 unpack_bf16x4(uint32_t a, uint32_t b) {
  return make_float4(__uint_as_float(a << 16), __uint_as_float(a & 0xffff0000u),
                     __uint_as_float(b << 16), __uint_as_float(b & 0xffff0000u));
}
// gradient packet j (4 elements) of a stage
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
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p)
               : "memory");
  return v;
}
__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p)
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
// after acquiring another SM's generic-proxy stores: make them visible to
// this thread's later TMA (async-proxy) reads
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;"
               ::"r"(smem_u32(b)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
  asm volatile("{\n\t.reg .b64 st;\n\t"
               "mbarrier.arrive.shared::cta.b64 st, [%0];\n\t}"
               ::"r"(smem_u32(b)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("{\n\t.reg .b64 st;\n\t"
               "mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}"
               ::"r"(smem_u32(b)), "r"(bytes) : "memory");
}
// true once the phase of the given parity has completed (non-blocking)
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(smem_u32(b)), "r"(parity) : "memory");
  return ok != 0;
}
// TMA bulk copy global -> shared; completion counted in bytes on `bar`
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src,
                                         uint32_t bytes, uint64_t* bar,
                                         uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1], %2, [%3], %4;"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}
// A wait that ran out: report it and make every other waiter of this launch
// (abort word counters[4] == epoch) give up too.
__device__ __forceinline__ void give_up(uint32_t* status, uint32_t* counters,
                                        uint32_t epoch) {
  atomicOr(status, kStatusWaitTimeout);
  atomicExch(&counters[4], epoch);
}

// Poll an mbarrier phase with a bounded number of tries; gives up early if
// another CTA of this launch has aborted.  Returns false on give-up.
__device__ __noinline__ bool wait_phase(uint64_t* b, uint32_t parity,
                                        uint32_t* status, uint32_t* counters,
                                        uint32_t epoch) {
  for (uint32_t i = 0; i < kSpinLimit; ++i) {
    if (mbar_test(b, parity)) return true;
    if ((i & 255) == 255 && ld_relaxed(&counters[4]) == epoch) return false;
    if (i >= 64) __nanosleep(i >= 4096 ? 256 : 32);
  }
  give_up(status, counters, epoch);
  return false;
}

// ---------------------------------------------------------------------------
// Element arithmetic (same functions as the two-pass kernels)
// ---------------------------------------------------------------------------
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
__device__ __forceinline__ float fused2_elem(float m, float v, float w,
                                             float s, float lam,
                                             const LambConsts& k) {
  const float u = kLars ? m : lamb_direction(m, v, w, lam, k);
  return __fmaf_rn(-s, u, w);
}

// ---------------------------------------------------------------------------
// Consumer work on one item
// ---------------------------------------------------------------------------
// Pass 1 from a stage (chunk length a multiple of 8): each consumer thread
// takes packets tid, tid + kConsumers, ...
template <bool kLars, typename GT>
__device__ __forceinline__ void c_pass1_staged(const char* st,
                                               const TensorPtrs& tp,
                                               int64_t off, int len,
                                               float lam, const LambConsts& k,
                                               uint64_t pol_keep, float& sw,
                                               float& su, int tid) {
  const GT* tag = nullptr;
  const int np = len >> 2;
#pragma unroll
  for (int q = 0; q < kPkts; ++q) {
    const int j = tid + q * kConsumers;
    if (j < np) {
      float4 mv = *reinterpret_cast<const float4*>(st + kOffM + 16 * j);
      float4 vv = kLars ? make_float4(0.f, 0.f, 0.f, 0.f)
                        : *reinterpret_cast<const float4*>(st + kOffV + 16 * j);
      const float4 wv =
          *reinterpret_cast<const float4*>(st + off_w<kLars>() + 16 * j);
      const float4 gv = lds_grad4(st + off_g<kLars>(), j, tag);
      fused1_elem<kLars>(gv.x, mv.x, vv.x, wv.x, lam, k, sw, su);
      fused1_elem<kLars>(gv.y, mv.y, vv.y, wv.y, lam, k, sw, su);
      fused1_elem<kLars>(gv.z, mv.z, vv.z, wv.z, lam, k, sw, su);
      fused1_elem<kLars>(gv.w, mv.w, vv.w, wv.w, lam, k, sw, su);
      stp4(tp.m + off + 4 * j, mv, pol_keep);
      if (!kLars) stp4(tp.v + off + 4 * j, vv, pol_keep);
    }
  }
}

// Pass 1 straight from global memory (tail chunks, unaligned tensors)
template <bool kLars, typename GT>
__device__ __forceinline__ void c_pass1_direct(const TensorPtrs& tp,
                                               int64_t off, int len,
                                               float lam, const LambConsts& k,
                                               float& sw, float& su, int tid) {
  float* __restrict__ m = tp.m + off;
  float* __restrict__ v = kLars ? nullptr : tp.v + off;
  const float* __restrict__ w = tp.w + off;
  const GT* __restrict__ g = static_cast<const GT*>(tp.g) + off;
  for (int i = tid; i < len; i += kConsumers) {
    float mi = m[i];
    float vi = kLars ? 0.f : v[i];
    fused1_elem<kLars>(ld_grad1(g + i), mi, vi, w[i], lam, k, sw, su);
    m[i] = mi;
    if (!kLars) v[i] = vi;
  }
}

template <bool kLars, bool kCopy>
__device__ __forceinline__ void c_pass2_staged(const char* st,
                                               const TensorPtrs& tp,
                                               int64_t off, int len, float s,
                                               float lam, const LambConsts& k,
                                               uint64_t pol_first, int tid) {
  const int np = len >> 2;
#pragma unroll
  for (int q = 0; q < kPkts; ++q) {
    const int j = tid + q * kConsumers;
    if (j < np) {
      const float4 mv = *reinterpret_cast<const float4*>(st + kOffM + 16 * j);
      const float4 vv =
          kLars ? make_float4(0.f, 0.f, 0.f, 0.f)
                : *reinterpret_cast<const float4*>(st + kOffV + 16 * j);
      const float4 wv =
          *reinterpret_cast<const float4*>(st + off_w<kLars>() + 16 * j);
      float4 o;
      o.x = fused2_elem<kLars>(mv.x, vv.x, wv.x, s, lam, k);
      o.y = fused2_elem<kLars>(mv.y, vv.y, wv.y, s, lam, k);
      o.z = fused2_elem<kLars>(mv.z, vv.z, wv.z, s, lam, k);
      o.w = fused2_elem<kLars>(mv.w, vv.w, wv.w, s, lam, k);
      stp4(tp.w + off + 4 * j, o, pol_first);
      if (kCopy) stp_copy4(tp.copy, off + 4 * j, o, pol_first);
    }
  }
}

template <bool kLars, bool kCopy>
__device__ __forceinline__ void c_pass2_direct(const TensorPtrs& tp,
                                               int64_t off, int len, float s,
                                               float lam, const LambConsts& k,
                                               int tid) {
  float* __restrict__ w = tp.w + off;
  const float* __restrict__ m = tp.m + off;
  const float* __restrict__ v = kLars ? nullptr : tp.v + off;
  // m, v come from other SMs' pass 1 of this launch: read them from L2
  for (int i = tid; i < len; i += kConsumers) {
    const float o = fused2_elem<kLars>(__ldcg(m + i), kLars ? 0.f : __ldcg(v + i),
                                       w[i], s, lam, k);
    w[i] = o;
    if (kCopy) st_copy1(tp.copy, off + i, o);
  }
}

// ---------------------------------------------------------------------------
// Publisher: a tensor's last chunk -> norms, trust ratio, ready flag
// ---------------------------------------------------------------------------
template <bool kLars>
__device__ __forceinline__ void finalize_fused(const StepParams& p,
                                               const FusedParams& f, int k,
                                               int first, int n,
                                               uint32_t epoch, int lane) {
  __threadfence();
  double aw = 0.0, au = 0.0;
  for (int i = lane; i < n; i += 32) {
    const float2 s = __ldcg(&f.fslots[first + i]);
    aw += (double)s.x;
    au += (double)s.y;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    aw += __shfl_down_sync(0xffffffffu, aw, o);
    au += __shfl_down_sync(0xffffffffu, au, o);
  }
  if (lane == 0) {
    const double wn = sqrt(aw), un = sqrt(au);
    double rho = 1.0;                                  // zero-norm rule
    if (!(wn == 0.0 || un == 0.0))
      rho = (kLars ? p.trust : 1.0) * phi_of(wn, p) / un;
    p.ratio[k] = rho;
    p.wnorm[k] = wn;
    p.unorm[k] = un;
    if (!isfinite(aw) || !isfinite(au)) atomicOr(p.status, kStatusNonfinite);
    f.tickets[k] = 0u;
    st_release(&f.ready[k], epoch);
  }
  __syncwarp();
}

// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------
template <bool kLars, typename GT, bool kCopy>
__global__ void __launch_bounds__(kFusedThreads, 1)
    fused_step_kernel(const StepParams p, const FusedParams f) {
  extern __shared__ __align__(128) char fused_smem[];
  constexpr int kStages = n_stages<kLars, GT>();
  __shared__ __align__(8) uint64_t s_full[kStages], s_empty[kStages];
  __shared__ __align__(8) uint64_t s_pfull[kPubSlots], s_pempty[kPubSlots];
  __shared__ StageDesc s_desc[kStages];
  __shared__ PubEntry s_pub[kPubSlots];
  __shared__ uint32_t s_uses[kStages];   // phases armed on each full barrier
  __shared__ float s_red[kRedRing][2][kConsumerWarps];
  __shared__ uint32_t s_redcnt[kRedRing];
  __shared__ uint32_t s_stopped;
  __shared__ LambConsts s_k;
  __shared__ float s_lr, s_c1, s_c2;
  __shared__ int s_skip;
  __shared__ uint32_t s_epoch;
  __shared__ int64_t s_t;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;

  // ---- per-launch constants (c2 beside c1, in another warp) -------------
  const bool bc = !kLars && (p.flags & kFlagBiasCorrection) != 0;
  if (threadIdx.x == 32) {
    const int64_t t = p.d_step ? *p.d_step : int64_t(1);
    s_c2 = (bc && t >= 1) ? (float)(1.0 / (1.0 - pow_from_log2(
                                p.log2_beta2, (double)t)))
                          : 1.f;
  }
  if (threadIdx.x == 0) {
    const int64_t t = p.d_step ? *p.d_step : int64_t(1);
    const int skip = (bc && t < 1) ? 1 : 0;
    s_t = t;
    s_skip = skip;
    s_c1 = (bc && !skip)
               ? (float)(1.0 / (1.0 - pow_from_log2(p.log2_beta1, (double)t)))
               : 1.f;
    s_lr = step_lr(p, t);
    s_epoch = *reinterpret_cast<volatile uint32_t*>(&p.counters[3]);
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], kConsumerWarps);
      s_uses[i] = 0u;
    }
    for (int i = 0; i < kPubSlots; ++i) {
      mbar_init(&s_pfull[i], 1);
      mbar_init(&s_pempty[i], 1);
    }
    for (int i = 0; i < kRedRing; ++i) s_redcnt[i] = 0u;
    s_stopped = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const float c1 = s_c1, c2 = s_c2;
    s_k = LambConsts{p.b1, p.omb1, p.b2, p.omb2, c1, c2, p.eps,
                     0.f, 0.f, 0.f, 0.f};
    if (blockIdx.x == 0) {
      StepScalars sc{};
      sc.t = s_t;
      sc.c1 = c1;
      sc.c2 = c2;
      sc.lr = s_lr;
      sc.skip = s_skip;
      *p.scal = sc;
      if (s_skip) atomicOr(p.status, kStatusBadStep);
    }
  }
  __syncthreads();
  if (s_skip) return;
  const LambConsts k = s_k;
  const uint32_t epoch = s_epoch;
  const uint32_t* abort_word = &p.counters[4];
  constexpr int kSB = stage_bytes<kLars, GT>();

  if (warp == kProducerWarp) {
    // ======================= producer =====================================
    if (lane == 0) {
      const uint32_t n_items = (uint32_t)f.n_items;
      const uint64_t pol_first = policy_evict_first();
      const uint64_t pol_last = policy_evict_last();
      const float lr = s_lr;
      // Items are drawn in batches of kDrawBatch consecutive schedule items
      // (one atomic per batch).  Software pipeline, per batch n: the draw of
      // batch n+3 and the records of batch n+2 are issued, and the tensor
      // descriptor of batch n+1's first item; each is used one batch later,
      // so the producer never waits for an atomic or a load it just issued.
      auto draw = [&]() -> uint32_t {
        return atomicAdd(&p.counters[2], (uint32_t)kDrawBatch);
      };
      // the device item list is padded to a multiple of kDrawBatch
      auto load_recs = [&](uint32_t b, uint4& ra, uint4& rb) {
        if (b < n_items) {
          const uint4* p4 = reinterpret_cast<const uint4*>(f.items + b);
          ra = p4[0];
          rb = p4[1];
        }
      };
      uint32_t b0 = draw();
      uint4 a0 = make_uint4(0u, 0u, 0u, 0u), c0 = a0;
      load_recs(b0, a0, c0);
      uint32_t b1 = draw();
      uint4 a1 = make_uint4(0u, 0u, 0u, 0u), c1 = a1;
      load_recs(b1, a1, c1);
      uint32_t b2 = draw();
      int kcur = -1, knext = -1;
      FusedTensor tcur{}, tnext{};
      TensorPtrs qcur{}, qnext{};
      int ready_k = -1;          // tensor whose final norms were acquired
      float ready_s = 0.f;
      bool aborted = false, done = false;
      uint32_t it = 0;
      while (!done) {
        // ---- issue the loads used by the next batches ---------------------
        uint4 a2 = make_uint4(0u, 0u, 0u, 0u), c2 = a2;
        load_recs(b2, a2, c2);
        // (b2 was drawn a batch ago; past the end, stop drawing)
        const uint32_t b3 = b2 < n_items ? draw() : n_items;
        knext = -1;
        if (b1 < n_items) {
          const int kn = (int)(a1.x >> 1);
          if (kn != kcur) {
            tnext = f.ftensors[kn];
            qnext = p.ptrs[kn];
            knext = kn;
          }
        }
        // ---- the items of batch b0 ---------------------------------------
#pragma unroll 1
        for (int j = 0; j < kDrawBatch; ++j, ++it) {
          const int s = (int)(it % kStages);
          const uint32_t use = it / kStages;
          if (!wait_phase(&s_empty[s], (use & 1u) ^ 1u, p.status, p.counters,
                          epoch)) {
            aborted = done = true;
            break;
          }
          s_uses[s] = use + 1u;
          StageDesc d{};
          if (b0 + j >= n_items) {
            d.flags = kItemEnd;
            s_desc[s] = d;
            mbar_arrive(&s_full[s]);
            done = true;
            break;
          }
          const uint4& rr = j < 2 ? a0 : c0;
          const uint2 r = (j & 1) ? make_uint2(rr.z, rr.w)
                                  : make_uint2(rr.x, rr.y);
          const int kt = (int)(r.x >> 1);
          if (kt != kcur) {
            if (kt == knext) {
              tcur = tnext;
              qcur = qnext;
            } else {
              tcur = f.ftensors[kt];
              qcur = p.ptrs[kt];
            }
            kcur = kt;
          }
          const bool p2 = (r.x & 1u) != 0;
          const int64_t off = (int64_t)r.y * kFusedChunk;
          const int64_t rem = tcur.numel - off;
          d.tp = qcur;
          d.tensor = kt;
          d.index = (int)r.y;
          d.len = (int)(rem < kFusedChunk ? rem : kFusedChunk);
          d.lam = tcur.decay * p.wd;
          d.first_chunk = tcur.first_chunk;
          d.n_chunks = tcur.n_chunks;
          const bool resident = tcur.resident != 0;
          d.flags = (p2 ? kItemP2 : 0u) | (resident ? kItemResident : 0u);
          // bulk copies need 16-byte aligned addresses and sizes
          const uintptr_t amask =
              (uintptr_t)qcur.w | (uintptr_t)qcur.m | (uintptr_t)qcur.g |
              (kLars ? (uintptr_t)0 : (uintptr_t)qcur.v);
          const bool direct = (amask & 15u) != 0 || (d.len & 7) != 0;
          if (direct) d.flags |= kItemDirect;
          if (p2) {
            if (kt != ready_k) {
              bool ok = false;
              for (uint32_t i = 0; i < kSpinLimit; ++i) {
                if (ld_acquire(&f.ready[kt]) == epoch) {
                  ok = true;
                  break;
                }
                if ((i & 255) == 255 && ld_relaxed(abort_word) == epoch) break;
                __nanosleep(i >= 4096 ? 256 : 32);
              }
              if (!ok) {
                if (ld_relaxed(abort_word) != epoch)
                  give_up(p.status, p.counters, epoch);
                d.flags |= kItemSkip;
                aborted = done = true;
              } else {
                fence_proxy_async_global();
                ready_k = kt;
                ready_s =
                    __double2float_rn((double)lr * __ldcg(&p.ratio[kt]));
              }
            }
            d.s = ready_s;
          }
          s_desc[s] = d;
          if (direct || (d.flags & kItemSkip)) {
            mbar_arrive(&s_full[s]);
          } else {
            char* st = fused_smem + s * kSB;
            const uint32_t nb = (uint32_t)d.len * 4u;
            const uint32_t gb = p2 ? 0u : (uint32_t)(d.len * (int)sizeof(GT));
            mbar_arrive_tx(&s_full[s], nb * (kLars ? 2u : 3u) + gb);
            const uint64_t pol = (!p2 && resident) ? pol_last : pol_first;
            bulk_g2s(st + kOffM, qcur.m + off, nb, &s_full[s], pol);
            if (!kLars)
              bulk_g2s(st + kOffV, qcur.v + off, nb, &s_full[s], pol);
            bulk_g2s(st + off_w<kLars>(), qcur.w + off, nb, &s_full[s], pol);
            if (!p2)
              bulk_g2s(st + off_g<kLars>(),
                       static_cast<const GT*>(qcur.g) + off, gb, &s_full[s],
                       pol_first);
          }
          if (aborted) break;
        }
        b0 = b1;
        a0 = a1;
        c0 = c1;
        b1 = b2;
        a1 = a2;
        c1 = c2;
        b2 = b3;
      }
      // The producer that finishes drawing last closes the launch
      // (counters[5] counts finished producers): the work counter returns to
      // 0 and the epoch advances -- the other CTAs cached the epoch and t, so
      // they are unaffected -- and t advances only if the launch completed.
      __threadfence();
      if (atomicAdd(&p.counters[5], 1u) + 1u == gridDim.x) {
        __threadfence();
        atomicExch(&p.counters[2], 0u);
        atomicExch(&p.counters[5], 0u);
        const uint32_t ne = epoch + 1u == 0u ? 1u : epoch + 1u;
        atomicExch(&p.counters[3], ne);
        if (ld_relaxed(abort_word) != epoch) {
          StepScalars sc{};
          sc.t = s_t;
          sc.lr = lr;
          close_step(p, sc);
        }
      }
    }
  } else if (warp == kPublisherWarp) {
    // ======================= publisher ====================================
    // Lane 0 waits for the next entry; then every entry already pushed
    // behind it (up to kPubSlots) is taken at once, lane j handling the j-th,
    // so the ticket atomics of several chunks are in flight together.
    bool live = true;
    for (uint32_t q = 0; live;) {
      int ok = 1;
      if (lane == 0)
        ok = wait_phase(&s_pfull[q % kPubSlots], (q / kPubSlots) & 1u,
                        p.status, p.counters, epoch) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      const uint32_t qj = q + (uint32_t)lane;
      const int slot = (int)(qj % kPubSlots);
      const bool full = lane == 0 ||
                        (lane < kPubSlots &&
                         mbar_test(&s_pfull[slot], (qj / kPubSlots) & 1u));
      // entries are taken in order: stop at the first one not yet pushed
      const uint32_t not_full = __ballot_sync(0xffffffffu, !full);
      const int cnt = __ffs(not_full) - 1;           // lanes 0 .. cnt-1
      PubEntry e{};
      if (lane < cnt) e = s_pub[slot];
      const uint32_t ends = __ballot_sync(0xffffffffu, lane < cnt && e.tensor < 0);
      const int take = ends ? __ffs(ends) - 1 : cnt; // entries before the end
      if (ends) live = false;
      uint32_t last = 0;
      if (lane < take) {
        f.fslots[e.first_chunk + e.index] = make_float2(e.sw, e.su);
        const uint32_t prev = atom_add_acq_rel(&f.tickets[e.tensor], 1u);
        last = (prev + 1u == (uint32_t)e.n_chunks) ? 1u : 0u;
      }
      if (lane < cnt) mbar_arrive(&s_pempty[slot]);
      uint32_t lasts = __ballot_sync(0xffffffffu, last != 0u);
      while (lasts) {                                // tensors completed here
        const int j = __ffs(lasts) - 1;
        lasts &= lasts - 1u;
        const int kt = __shfl_sync(0xffffffffu, e.tensor, j);
        const int fc = __shfl_sync(0xffffffffu, e.first_chunk, j);
        const int nc = __shfl_sync(0xffffffffu, e.n_chunks, j);
        finalize_fused<kLars>(p, f, kt, fc, nc, epoch, lane);
      }
      q += (uint32_t)cnt;
    }
  } else {
    // ======================= consumers ====================================
    // The consumer warps walk the stage ring independently (no barrier among
    // them).  For a pass-1 item each warp leaves its partial sums in s_red;
    // the last warp to finish the item (shared-memory counter) adds the 16
    // partials in warp order and hands them to the publisher, so sums are
    // pushed in item order.  A warp can run at most kStages items ahead of
    // the slowest, hence the 2 x kStages rings.
    const int tid = threadIdx.x;                     // 0 .. kConsumers-1
    const uint64_t pol_first = policy_evict_first();
    const uint64_t pol_last = policy_evict_last();
    uint32_t q = 0;                                  // pass-1 items seen
    for (uint32_t it = 0;; ++it) {
      const int s = (int)(it % kStages);
      const uint32_t use = it / kStages;
      int ok = 1;
      if (lane == 0)
        ok = wait_phase(&s_full[s], use & 1u, p.status, p.counters, epoch) ? 1
                                                                           : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      __syncwarp();                                  // lane 0 acquired it
      const StageDesc d = s_desc[s];
      if (d.flags & kItemEnd) break;
      if (!(d.flags & kItemSkip)) {
        const TensorPtrs& tp = d.tp;
        const int64_t off = (int64_t)d.index * kFusedChunk;
        const char* st = fused_smem + s * kSB;
        if (!(d.flags & kItemP2)) {
          float sw = 0.f, su = 0.f;
          const uint64_t pol_keep =
              (d.flags & kItemResident) ? pol_last : pol_first;
          if (d.flags & kItemDirect)
            c_pass1_direct<kLars, GT>(tp, off, d.len, d.lam, k, sw, su, tid);
          else
            c_pass1_staged<kLars, GT>(st, tp, off, d.len, d.lam, k, pol_keep,
                                      sw, su, tid);
          sw = warp_sum(sw);
          su = warp_sum(su);
          const int r = (int)(q % kRedRing);
          if (lane == 0) {
            s_red[r][0][warp] = sw;
            s_red[r][1][warp] = su;
            __threadfence_block();
            const uint32_t c = atomicAdd(&s_redcnt[r], 1u);
            if (c + 1u == (uint32_t)kConsumerWarps) {  // last warp of item
              __threadfence_block();
              float tw = 0.f, tu = 0.f;
#pragma unroll
              for (int i = 0; i < kConsumerWarps; ++i) {
                tw += s_red[r][0][i];
                tu += s_red[r][1][i];
              }
              s_redcnt[r] = 0u;
              const int ps = (int)(q % kPubSlots);
              const uint32_t pph = ((q / kPubSlots) & 1u) ^ 1u;
              if (wait_phase(&s_pempty[ps], pph, p.status, p.counters,
                             epoch)) {
                s_pub[ps] = PubEntry{d.tensor, d.first_chunk, d.index,
                                     d.n_chunks, tw, tu};
                mbar_arrive(&s_pfull[ps]);
              }
            }
          }
          ++q;
        } else if (d.flags & kItemDirect) {
          c_pass2_direct<kLars, kCopy>(tp, off, d.len, d.s, d.lam, k, tid);
        } else {
          c_pass2_staged<kLars, kCopy>(st, tp, off, d.len, d.s, d.lam, k,
                                       pol_first, tid);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[s]);
    }
    // the last consumer warp to stop ends the sums stream (every push of a
    // pass-1 item precedes its pusher's stop)
    if (lane == 0) {
      __threadfence_block();
      if (atomicAdd(&s_stopped, 1u) + 1u == (uint32_t)kConsumerWarps) {
        const int ps = (int)(q % kPubSlots);
        const uint32_t pph = ((q / kPubSlots) & 1u) ^ 1u;
        if (wait_phase(&s_pempty[ps], pph, p.status, p.counters, epoch)) {
          s_pub[ps] = PubEntry{-1, 0, 0, 0, 0.f, 0.f};
          mbar_arrive(&s_pfull[ps]);
        }
      }
    }
  }

  // ---- no bulk copy may still be writing this CTA's shared memory --------
  // (after a give-up only: in a completed launch the consumers have taken
  // every armed phase).  Each armed phase was arrived on by the producer, so
  // only the bytes of its copies can be outstanding.
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      const uint32_t u = s_uses[i];
      if (u == 0u) continue;               // stage never used
      for (uint32_t n = 0; n < kSpinLimit; ++n) {
        if (mbar_test(&s_full[i], (u - 1u) & 1u)) break;
        __nanosleep(64);
      }
    }
  }
}

template <bool kLars, typename GT, bool kCopy>
int launch_fused_t(const StepParams& p, const FusedParams& f, int grid,
                   cudaStream_t s) {
  fused_step_kernel<kLars, GT, kCopy>
      <<<grid, kFusedThreads, fused_smem_bytes<kLars, GT>(), s>>>(p, f);
  return (int)cudaGetLastError();
}

template <bool kLars, typename GT, bool kCopy>
int occupancy_fused_t(int* blocks) {
  // opt in to the dynamic shared memory of the stage ring (a property of
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

}  // namespace

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
