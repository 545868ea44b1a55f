// sm_103a kernel of the on-chip single-touch LAMB / LARS step.
//
// Algorithm 2 needs ||w_k|| and ||u_k|| (u = r + lambda_k w) of a WHOLE tensor
// before any of its elements may change.  The two-pass kernels therefore read
// m, v, w twice from HBM (40 B per parameter with bf16 g and a bf16 copy).
// This kernel reads and writes every operand once (28 B per parameter) by
// keeping, between the two halves of the step, each element's w and u in the
// shared memory of the SM that formed them.
//
// One cooperative launch per step: one CTA per SM (all resident at once),
// 768 threads (24 warps), ~221 KB of dynamic shared memory holding up to 224
// rows of 128 elements (w and u in fp32, 1 KB per row; 216 on a GB300).  The
// host planner (planner.cpp, plan_onchip) cuts the tensors into ROUNDS of
// consecutive whole tensors whose rows fit the grid (~4.2M parameters on 152
// SMs).  Each CTA owns a fixed slice of a round's rows, in pieces (a piece =
// the rows of one tensor in one CTA, at most 16 per CTA); warp w takes rows
// w, w + 24, ...  When a round's tables are loaded, every row gets a 32-bit
// record (its row inside the tensor, its count, its piece, its flags), which
// is all the per-row work reads.  Per round r:
//
//   pass 1   each warp keeps two rows in flight: w and m of a row are copied
//            (cp.async) straight into the row's shared-memory slot, g and v
//            into registers.  For each arrived row: the new m, v (Alg. 2
//            moment lines; Alg. 1 momentum for LARS) go back to HBM, u
//            replaces m in the slot, and each lane adds its elements' w^2 and
//            u^2 to per-piece two-float sums (a fixed warp tree when the
//            warp leaves the piece); per piece, the warps' sums are added in
//            warp order into the piece's slot, tagged with the launch.
//   exchange the CTA loads round r + 1's tables; then, for each of its
//            tensors, it reloads the tensor's slots (written by every CTA
//            that holds a piece of it) until all carry this launch's tag.
//            No grid-wide barrier is needed: nothing else passes between
//            CTAs.
//   ratio    the slots in slot order (two-float) give rho_k =
//            phi(||w||)/||u|| in fp32 (1 on a zero norm; LARS: kappa
//            phi(||w||)/||m||); the CTA holding the tensor's first piece
//            exports rho_k and the norms.
//   pass 2   w <- w - eta rho_k u from shared memory (+ the bf16 copy): no HBM
//            reads at all.  It runs inside pass 1 of round r + 1: a row's
//            slot is written back just before round r + 1's copy into it is
//            issued, so the stores of one round overlap the loads of the
//            next.
//
// The reductions avoid fp64: GB300 issues fp64 at a small fraction of its
// fp32 rate, and the compensated two-float sums keep ~44 bits.
//
// A tensor with more rows than the grid holds (BERT's 30522 x 1024 word
// embedding) is not the kernel's: the two-pass kernels update it, over a chunk
// table of such tensors only, before this launch.
//
// The partial sums have a fixed shape given by the plan, so the result does
// not depend on timing: every run is bitwise identical.  The element
// arithmetic is the two-pass kernels' (lamb_device.cuh), so m, v and u are
// bit-identical to theirs; only the summation of the norms differs.
//
// The prologue's independent loads (the abort and epoch words, eta, round 0's
// pieces, the step count) run in separate warps and meet at one CTA barrier.
//
// The tags come from a launch epoch that the last CTA of a launch advances,
// so the step can be replayed from a CUDA graph.  The wait for a tensor's
// slots is bounded: a CTA that waits longer than the plan's limit (1 s by
// default) sets LAMB_STATUS_WAIT_TIMEOUT and an abort word; every other
// waiter then gives up too and the launch returns.  A launch that finds the
// abort word set does nothing; the plan must be destroyed.  The last CTA to
// finish also closes the step (t + 1, the scheduled eta, the N-LAMB product).
#include "lamb_device.cuh"
#include "lamb_onchip.h"

namespace lamb {
namespace {

constexpr int kOptLars = 3;

// ---------------------------------------------------------------------------
// PTX helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];"
               : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];"
               : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_relaxed_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;"
               :: "l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], %2;"
               : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ void st_relaxed_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.relaxed.gpu.global.u32 [%0], %1;"
               :: "l"(p), "r"(v) : "memory");
}

// 16-byte asynchronous copy global -> shared (L2 only), in this thread's
// current group
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;"
               :: "r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory");
}

// ---------------------------------------------------------------------------
// Two-float sums (a value is hi + lo): TwoSum of the high parts, the error
// and the low parts folded in, then renormalised.  All inputs here are
// non-negative sums of squares, for which this keeps ~44 significant bits.
// ---------------------------------------------------------------------------
struct F2 {
  float hi, lo;
};

__device__ __forceinline__ F2 ff_add(F2 a, F2 b) {
  const float s = __fadd_rn(a.hi, b.hi);
  const float bb = __fsub_rn(s, a.hi);
  const float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, bb)),
                            __fsub_rn(b.hi, bb));
  const float t = __fadd_rn(e, __fadd_rn(a.lo, b.lo));
  const float hi = __fadd_rn(s, t);
  return F2{hi, __fsub_rn(t, __fsub_rn(hi, s))};
}

__device__ __forceinline__ F2 warp_sum_ff(F2 x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    F2 y;
    y.hi = __shfl_down_sync(0xffffffffu, x.hi, o);
    y.lo = __shfl_down_sync(0xffffffffu, x.lo, o);
    x = ff_add(x, y);
  }
  return x;
}

// A row of a round's slice, formed once when the round's tables are loaded so
// that the per-row work does not walk the piece table; packed in 32 bits to
// leave the shared memory to the rows themselves: bits 0-15 the row's index
// inside its tensor (a resident tensor has fewer than 2^16 rows), 16-23 its
// element count (1..kOcRow), 24-27 its piece, 28 whether the piece's arrays
// take 16-byte accesses, 29 whether it is its warp's last row of its piece.
struct OcRow {
  uint32_t bits;
  __device__ int64_t x() const { return (int64_t)(bits & 0xFFFFu) * kOcRow; }
  __device__ int cnt() const { return (int)((bits >> 16) & 0xFFu); }
  __device__ int piece() const { return (int)((bits >> 24) & 0xFu); }
  __device__ bool vec() const { return (bits >> 28) & 1u; }
  __device__ bool last() const { return (bits >> 29) & 1u; }
};
static_assert(kOcRow <= 255 && kOcMaxPieces <= 16, "OcRow fields");

// The tables of one round (double-buffered: one round's pass 2 runs inside
// the next round's pass 1).
struct OcTables {
  OcPiece piece[kOcMaxPieces];
  float s[kOcMaxPieces];           // eta rho_k of each piece's tensor
  float dd[kOcMaxPieces];          // eta lambda_k (decoupled decay) or 0
  OcRow row[kOcMaxRows];           // per row of the slice
  int np, nr;                      // pieces and rows of this CTA's slice
};

struct OcShared {
  OcTables tab[2];
  float4 red[kOcMaxPieces][kOcWarps];  // per piece and warp: two-float
                                       // sums of w^2 (x, y) and u^2 (z, w)
  LambConsts k;
  int64_t t;
  float lr;
  int skip;
  int ok;
  uint32_t unused_draw;
  uint32_t epoch;        // the plan's launch epoch when this launch started
  uint32_t abort;        // the plan's abort word when this launch started
};

// Exchange of the piece sums between CTAs, without a grid barrier.  A
// piece's slot is two 64-bit words, (sum w^2) and (sum u^2), each holding a
// two-float value: hi in the low half, lo in the high half with its four
// lowest bits replaced by a tag (lo is at most half an ulp of hi, so the
// truncation changes the sum by less than 2^-44 of it).  Every launch writes
// every slot once, with the tag (epoch + 1) mod 16 of its own launch; a CTA
// that needs a tensor's sums reloads its slots until every word carries that
// tag.  The words are written and read with single-copy-atomic relaxed 64-bit
// accesses, so a word with the right tag holds the right value, and no other
// data passes between CTAs: no fence is needed.  Slots keep the previous
// launch's tag until overwritten, and the plan zeroes them (tag 0) while the
// first launch uses tag 1.  The epoch advances when the last CTA of a launch
// finishes (a ticket), so the next launch, which starts after this one ends,
// reads the new value.  Nothing is reset by the host: the step can be
// replayed from a CUDA graph.
__device__ __forceinline__ uint64_t slot_word(F2 x, uint32_t tag) {
  return (uint64_t)__float_as_uint(x.hi) |
         ((uint64_t)((__float_as_uint(x.lo) & ~0xFu) | tag) << 32);
}
__device__ __forceinline__ F2 slot_value(uint64_t x) {
  return F2{__uint_as_float((uint32_t)x),
            __uint_as_float((uint32_t)(x >> 32) & ~0xFu)};
}
__device__ __forceinline__ bool slot_tagged(uint64_t x, uint32_t tag) {
  return ((uint32_t)(x >> 32) & 0xFu) == tag;
}
// Tag of this launch's slots; test plans wait for a tag nobody writes.
__device__ __forceinline__ uint32_t write_tag(uint32_t epoch) {
  return (epoch + 1u) & 0xFu;
}
__device__ __forceinline__ uint32_t wait_tag(const OcParams& q,
                                             uint32_t epoch) {
  return (epoch + 1u + (uint32_t)q.extra_arrivals) & 0xFu;
}

// ---------------------------------------------------------------------------
// Gradient registers: kept as loaded (bf16 pairs stay packed) until the row
// is computed, so nothing waits on the load before then.
// ---------------------------------------------------------------------------
template <typename GT> struct GradRaw;

template <> struct GradRaw<float> {
  using T = float4;
  __device__ static T load4(const float* p) {
    return __ldcs(reinterpret_cast<const float4*>(p));
  }
  __device__ static T load_n(const float* p, int c) {
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c > 0) x.x = __ldcs(p);
    if (c > 1) x.y = __ldcs(p + 1);
    if (c > 2) x.z = __ldcs(p + 2);
    if (c > 3) x.w = __ldcs(p + 3);
    return x;
  }
  __device__ static float4 widen(const T& x) { return x; }
};

template <> struct GradRaw<__nv_bfloat16> {
  using T = uint2;
  __device__ static T load4(const __nv_bfloat16* p) {
    return __ldcs(reinterpret_cast<const uint2*>(p));
  }
  __device__ static T load_n(const __nv_bfloat16* p, int c) {
    const unsigned short* h = reinterpret_cast<const unsigned short*>(p);
    uint32_t b[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (j < c) b[j] = __ldcs(h + j);
    return make_uint2(b[0] | (b[1] << 16), b[2] | (b[3] << 16));
  }
  // bf16 -> f32 is exact: the pattern is the top half of the f32
  __device__ static float4 widen(const T& u) {
    return make_float4(__uint_as_float(u.x << 16),
                       __uint_as_float(u.x & 0xffff0000u),
                       __uint_as_float(u.y << 16),
                       __uint_as_float(u.y & 0xffff0000u));
  }
};

// Stores elements i..i+c-1 of x into `dst` (evict-first).
__device__ __forceinline__ void store4(float* dst, int64_t i, int c, bool vec,
                                       const float4& x) {
  if (c == 4 && vec) {
    st4_last(dst + i, x);
    return;
  }
  const float y[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (j < c) dst[i + j] = y[j];
}

__device__ __forceinline__ void store_copy4(void* dst, int64_t i, int c,
                                            bool vec, const float4& x) {
  if (c == 4 && vec) {
    st_copy4(dst, i, x);
    return;
  }
  const float y[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (j < c) st_copy1(dst, i + j, y[j]);
}

// Pass 1 of one element: the new moments (Alg. 2) or momentum (Alg. 1), and
// the direction u whose norm the trust ratio needs.
template <int kOpt>
__device__ __forceinline__ float elem1(float g, float& m, float& v, float w,
                                       float lam, const LambConsts& k) {
  if (kOpt == kOptLars) {
    m = lars_momentum(g, m, w, lam, k.b1, k.omb1);
    return m;
  }
  lamb_moments(g, m, v, k);
  return kOpt ? nlamb_direction<kOpt>(m, v, g, w, lam, k)
              : lamb_direction(m, v, w, lam, k);
}

// Four elements of pass 1: moments in m, v; u in u; valid elements (j < c)
// add w^2 and u^2 to sw, su; invalid ones give u = 0.
template <int kOpt>
__device__ __forceinline__ void row1(const float4& g, float4& m, float4& v,
                                     const float4& w, float4& u, int c,
                                     float lam, const LambConsts& k, float& sw,
                                     float& su) {
  float gg[4] = {g.x, g.y, g.z, g.w}, mm[4] = {m.x, m.y, m.z, m.w},
        vv[4] = {v.x, v.y, v.z, v.w}, ww[4] = {w.x, w.y, w.z, w.w}, uu[4];
  if (c == 4) {   // a full row: the same operations, without the guards
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      uu[j] = elem1<kOpt>(gg[j], mm[j], vv[j], ww[j], lam, k);
      sw = __fmaf_rn(ww[j], ww[j], sw);
      su = __fmaf_rn(uu[j], uu[j], su);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (j < c) {
        uu[j] = elem1<kOpt>(gg[j], mm[j], vv[j], ww[j], lam, k);
        sw = __fmaf_rn(ww[j], ww[j], sw);
        su = __fmaf_rn(uu[j], uu[j], su);
      } else {
        uu[j] = 0.f;
      }
    }
  }
  m = make_float4(mm[0], mm[1], mm[2], mm[3]);
  v = make_float4(vv[0], vv[1], vv[2], vv[3]);
  u = make_float4(uu[0], uu[1], uu[2], uu[3]);
}

__device__ __forceinline__ float4 update4(const float4& w, const float4& u,
                                          float s, float dd) {
  float4 o;
  o.x = __fmaf_rn(-s, u.x, w.x);
  o.y = __fmaf_rn(-s, u.y, w.y);
  o.z = __fmaf_rn(-s, u.z, w.z);
  o.w = __fmaf_rn(-s, u.w, w.w);
  if (dd != 0.f) {   // decoupled decay; skipped, not added as 0 (signed 0)
    o.x = __fmaf_rn(-dd, w.x, o.x);
    o.y = __fmaf_rn(-dd, w.y, o.y);
    o.z = __fmaf_rn(-dd, w.z, o.z);
    o.w = __fmaf_rn(-dd, w.w, o.w);
  }
  return o;
}

// ---------------------------------------------------------------------------
// Pass 1.  Row slot layout: float4 index row * 64 + lane holds lane's w,
// row * 64 + 32 + lane its m until the row is computed, then its u.  Warp w
// owns rows w, w + kOcWarps, ... of every round; i counts a warp's rows.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int warp_rows(int n_rows) {
  const int warp = threadIdx.x >> 5;
  return n_rows > warp ? (n_rows - warp + kOcWarps - 1) / kOcWarps : 0;
}

template <int kOpt, typename GT>
__device__ __forceinline__ void ring_issue(const OcTables& T, float4* rows,
                                           int i, int nw,
                                           typename GradRaw<GT>::T& g,
                                           float4& v, OcRow& R) {
  constexpr bool kV = kOpt != kOptLars;
  R.bits = 0u;   // no row: no elements
  if (i < nw) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row = warp + i * kOcWarps;
    R = T.row[row];
    const OcPiece& P = T.piece[R.piece()];
    const int cnt = min(max(R.cnt() - lane * 4, 0), 4);
    const int64_t x = R.x() + lane * 4;
    const GT* gp = static_cast<const GT*>(P.g) + x;
    float4* slot_w = rows + row * 64 + lane;
    float4* slot_m = slot_w + 32;
    if (cnt == 4 && R.vec()) {
      cp_async16(slot_w, P.w + x);
      cp_async16(slot_m, P.m + x);
      g = GradRaw<GT>::load4(gp);
      if (kV) v = ld4_last(P.v + x);
    } else {   // ragged tail or unaligned tensor: element-wise, zeros past cnt
      float4 w4 = make_float4(0.f, 0.f, 0.f, 0.f), m4 = w4, v4 = w4;
      float* wa = &w4.x;
      float* ma = &m4.x;
      float* va = &v4.x;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (j < cnt) {
          wa[j] = P.w[x + j];
          ma[j] = P.m[x + j];
          if (kV) va[j] = P.v[x + j];
        }
      }
      *slot_w = w4;
      *slot_m = m4;
      g = GradRaw<GT>::load_n(gp, cnt);
      v = v4;
    }
  }
}

// One arrived row (its record R as ring_issue read it): the new m, v to HBM,
// u over m in the slot; the lane's sums of its (up to) four w^2 and u^2 in
// sw, su.
template <int kOpt, typename GT>
__device__ __forceinline__ void ring_consume(const OcTables& T, float4* rows,
                                             int i,
                                             const typename GradRaw<GT>::T& g,
                                             const float4& v, OcRow R,
                                             const LambConsts& k, float wd,
                                             bool decoupled, float& sw,
                                             float& su) {
  constexpr bool kV = kOpt != kOptLars;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = warp + i * kOcWarps;
  const int cnt = min(max(R.cnt() - lane * 4, 0), 4);
  const OcPiece& P = T.piece[R.piece()];
  const float lam = decoupled ? 0.f : P.decay * wd;
  float4* slot_w = rows + row * 64 + lane;
  float4* slot_m = slot_w + 32;
  const float4 w4 = *slot_w;
  float4 m4 = *slot_m, v4 = v, u4;
  sw = 0.f;
  su = 0.f;
  row1<kOpt>(GradRaw<GT>::widen(g), m4, v4, w4, u4, cnt, lam, k, sw, su);
  if (cnt > 0) {
    const int64_t x = R.x() + lane * 4;
    store4(P.m, x, cnt, R.vec(), m4);
    if (kV) store4(P.v, x, cnt, R.vec(), v4);
  }
  *slot_m = u4;
}

// Per-lane two-float sums of w^2 and u^2 over a warp's rows of one piece;
// flushed (warp tree, then red[piece][warp]) when the next row belongs to
// another piece.  Every (piece, warp) entry starts at zero each round.
struct PieceAcc {
  F2 w, u;
  __device__ void add(float sw, float su) {
    w = ff_add(w, F2{sw, 0.f});
    u = ff_add(u, F2{su, 0.f});
  }
  __device__ void flush(OcShared& sh, int piece) {
    const F2 a = warp_sum_ff(w), b = warp_sum_ff(u);
    if ((threadIdx.x & 31) == 0)
      sh.red[piece][threadIdx.x >> 5] = make_float4(a.hi, a.lo, b.hi, b.lo);
    w = u = F2{0.f, 0.f};
  }
};

// Adds a row's sums; flushes if the row (record R) is its warp's last row of
// its piece.
__device__ __forceinline__ void acc_row(OcShared& sh, PieceAcc& acc, OcRow R,
                                        float sw, float su) {
  acc.add(sw, su);
  if (R.last()) acc.flush(sh, R.piece());
}

// Pass 2 of row i of a round whose ratios are known: w <- w - eta rho_k u
// (+ decoupled decay, + the bf16 copy), from the row's slot.
template <bool kCopy>
__device__ __forceinline__ void pass2_row(const OcTables& T,
                                          const float4* rows, int i) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = warp + i * kOcWarps;
  const OcRow R = T.row[row];
  const int j = R.piece();
  const int c = min(max(R.cnt() - lane * 4, 0), 4);
  if (c > 0) {
    const float4 o = update4(rows[row * 64 + lane],
                             rows[row * 64 + 32 + lane], T.s[j], T.dd[j]);
    const int64_t x = R.x() + lane * 4;
    store4(T.piece[j].w, x, c, R.vec(), o);
    if (kCopy) store_copy4(T.piece[j].copy, x, c, R.vec(), o);
  }
}

// Pass 1 of the round with tables `cur` (if any), with pass 2 of the previous
// round (tables `prev`, if any) folded in: a slot's previous row is written
// back just before the next round's copy into it is issued, so the stores of
// one round overlap the loads of the next.  Each warp keeps one pair of rows
// in flight.
template <int kOpt, typename GT, bool kCopy>
__device__ __forceinline__ void fused_pass(OcShared& sh, float4* rows,
                                           const OcTables* prev,
                                           const OcTables* cur,
                                           const LambConsts& k, float wd,
                                           bool decoupled) {
  const int nwp = prev ? warp_rows(prev->nr) : 0;
  const int nwc = cur ? warp_rows(cur->nr) : 0;
  int done2 = 0;   // rows of the previous round written back
  typename GradRaw<GT>::T g0, g1;
  float4 v0, v1;
  OcRow r0{0u}, r1{0u};
  PieceAcc acc{F2{0.f, 0.f}, F2{0.f, 0.f}};
  for (; done2 < min(2, nwp); ++done2) pass2_row<kCopy>(*prev, rows, done2);
  if (nwc > 0) {
    ring_issue<kOpt, GT>(*cur, rows, 0, nwc, g0, v0, r0);
    ring_issue<kOpt, GT>(*cur, rows, 1, nwc, g1, v1, r1);
  }
  cp_async_commit();
  for (int i = 0; i < nwc; i += 2) {
    cp_async_wait<0>();   // rows i, i + 1 have landed
    float sw0, su0, sw1 = 0.f, su1 = 0.f;
    ring_consume<kOpt, GT>(*cur, rows, i, g0, v0, r0, k, wd, decoupled, sw0,
                           su0);
    if (i + 1 < nwc)
      ring_consume<kOpt, GT>(*cur, rows, i + 1, g1, v1, r1, k, wd, decoupled,
                             sw1, su1);
    acc_row(sh, acc, r0, sw0, su0);
    if (i + 1 < nwc) acc_row(sh, acc, r1, sw1, su1);
    for (; done2 < min(i + 4, nwp); ++done2)
      pass2_row<kCopy>(*prev, rows, done2);
    ring_issue<kOpt, GT>(*cur, rows, i + 2, nwc, g0, v0, r0);
    ring_issue<kOpt, GT>(*cur, rows, i + 3, nwc, g1, v1, r1);
    cp_async_commit();
  }
  cp_async_wait<0>();
  for (; done2 < nwp; ++done2) pass2_row<kCopy>(*prev, rows, done2);
}

// ---------------------------------------------------------------------------
// Tables, norms and trust ratio
// ---------------------------------------------------------------------------
// Loads round r's slice of this CTA into T (two CTA barriers inside).
// Round r's pieces of this CTA into T, by the calling threads with index
// i = 0..kOcMaxPieces - 1 (the row map follows after a CTA barrier).
__device__ __forceinline__ void load_pieces(OcTables& T, const OcParams& q,
                                            int r, int i) {
  const OcSlice sl = q.slices[r * (int)gridDim.x + (int)blockIdx.x];
  if (i < sl.n_pieces) T.piece[i] = q.pieces[sl.piece_begin + i];
  if (i == 0) {
    T.np = sl.n_pieces;
    T.nr = sl.n_rows;
  }
}

// The row records of T's slice: each row's piece, first element and count.
__device__ __forceinline__ int piece_of_row(const OcTables& T, int row) {
  int j = 0;
  for (int i = 1; i < T.np; ++i)
    if (T.piece[i].first_row <= row) j = i;
  return j;
}

__device__ __forceinline__ void piece_rows(OcTables& T) {
  const int row = (int)threadIdx.x;
  if (row < T.nr) {
    const int j = piece_of_row(T, row);
    // the warp that takes this row next takes row + kOcWarps
    const bool last = row + kOcWarps >= T.nr ||
                      piece_of_row(T, row + kOcWarps) != j;
    const OcPiece& P = T.piece[j];
    const int r_in = row - P.first_row;   // row inside the piece
    const uint32_t t_row = (uint32_t)(P.offset / kOcRow) + (uint32_t)r_in;
    const uint32_t cnt = (uint32_t)min(P.len - r_in * kOcRow, kOcRow);
    T.row[row].bits = (t_row & 0xFFFFu) | (cnt << 16) | ((uint32_t)j << 24) |
                      ((P.flags & kOcVec) ? (1u << 28) : 0u) |
                      (last ? (1u << 29) : 0u);
  }
}

__device__ __forceinline__ void load_tables(OcTables& T, const OcParams& q,
                                            int r) {
  load_pieces(T, q, r, (int)threadIdx.x);
  __syncthreads();
  piece_rows(T);
  __syncthreads();
}

__device__ __forceinline__ void zero_red(OcShared& sh) {
  if ((int)threadIdx.x < kOcMaxPieces * kOcWarps)
    (&sh.red[0][0])[threadIdx.x] = make_float4(0.f, 0.f, 0.f, 0.f);
}

// Per piece (one warp each): the warps' sums in warp order -> its slot,
// tagged with this launch's tag.
__device__ __forceinline__ void piece_sums(const OcShared& sh,
                                           const OcTables& T,
                                           const OcParams& q, uint32_t tag) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int j = warp; j < T.np; j += kOcWarps) {
    const float4 x = lane < kOcWarps ? sh.red[j][lane]
                                     : make_float4(0.f, 0.f, 0.f, 0.f);
    const F2 a = warp_sum_ff(F2{x.x, x.y}), b = warp_sum_ff(F2{x.z, x.w});
    if (lane == 0) {
      uint64_t* w = q.slots + 2 * (size_t)T.piece[j].slot;
      st_relaxed_u64(w, slot_word(a, tag));
      st_relaxed_u64(w + 1, slot_word(b, tag));
    }
  }
}

__device__ __forceinline__ float phi_f(float z, const StepParams& p) {
  if (p.phi == 1) {  // clip; comparisons keep NaN as NaN
    const float gl = (float)p.gamma_l, gu = (float)p.gamma_u;
    if (z < gl) return gl;
    if (z > gu) return gu;
  }
  return z;
}

// Slots a lane keeps in flight when forming a ratio: a tensor has at most
// one slot per CTA, so 8 x 32 covers a 152-SM grid in one round trip.
constexpr int kRatioLoads = 8;

// Warp-wide, per piece: the tensor's slots in slot order (lane-strided,
// kRatioLoads slots in flight, reloaded until every word carries this
// launch's tag, then a fixed tree) -> ||w||, ||u||, rho_k (Alg. 2 last line
// with the zero-norm rule; LARS: times kappa), eta rho_k and eta lambda_k
// for pass 2; exports where this CTA holds the tensor's first piece.  Returns
// false if the wait gave up (see the file header).
__device__ __forceinline__ bool piece_ratio(const StepParams& p,
                                         const OcParams& q, const OcPiece& P,
                                         float coef, float lr, bool decoupled,
                                         uint32_t tag, float* s_out,
                                         float* dd_out) {
  const int lane = threadIdx.x & 31;
  const uint64_t* slots = q.slots + 2 * (size_t)P.t_slot;
  const uint64_t zero = slot_word(F2{0.f, 0.f}, tag);
  F2 a{0.f, 0.f}, b{0.f, 0.f};
  for (int base = 0; base < P.t_nslots; base += kRatioLoads * 32) {
    uint64_t x[kRatioLoads][2];
#pragma unroll
    for (int j = 0; j < kRatioLoads; ++j) {
      const int k = base + lane + 32 * j;
      x[j][0] = k < P.t_nslots ? ld_relaxed_u64(slots + 2 * k) : zero;
      x[j][1] = k < P.t_nslots ? ld_relaxed_u64(slots + 2 * k + 1) : zero;
    }
    uint64_t t0 = 0;
    for (uint32_t polls = 0;; ++polls) {
      bool ready = true;
#pragma unroll
      for (int j = 0; j < kRatioLoads; ++j)
        ready = ready && slot_tagged(x[j][0], tag) && slot_tagged(x[j][1], tag);
      if (__all_sync(0xffffffffu, ready)) break;
      if (polls == 0) t0 = global_ns();
      if ((polls & 15u) == 15u) {   // warp-uniform: every lane counts alike
        int stop = 0;
        if (lane == 0) {
          if (ld_acquire_u32(q.bar + kBarAbort)) {
            stop = 1;
          } else if (global_ns() - t0 > (uint64_t)q.wait_limit_ns) {
            atomicOr(p.status, kStatusWaitTimeout);
            atomicExch(q.bar + kBarAbort, 1u);
            stop = 1;
          }
        }
        if (__shfl_sync(0xffffffffu, stop, 0)) return false;
      }
#pragma unroll
      for (int j = 0; j < kRatioLoads; ++j) {
        const int k = base + lane + 32 * j;
        if (k < P.t_nslots) {
          if (!slot_tagged(x[j][0], tag)) x[j][0] = ld_relaxed_u64(slots + 2 * k);
          if (!slot_tagged(x[j][1], tag))
            x[j][1] = ld_relaxed_u64(slots + 2 * k + 1);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < kRatioLoads; ++j) {
      a = ff_add(a, slot_value(x[j][0]));
      b = ff_add(b, slot_value(x[j][1]));
    }
  }
  a = warp_sum_ff(a);
  b = warp_sum_ff(b);
  if (lane == 0) {
    const float aw = __fadd_rn(a.hi, a.lo), au = __fadd_rn(b.hi, b.lo);
    const float wn = __fsqrt_rn(aw), un = __fsqrt_rn(au);
    float rho = 1.f;                                   // zero-norm rule
    if (!(wn == 0.f || un == 0.f))
      rho = __fdiv_rn(__fmul_rn(coef, phi_f(wn, p)), un);
    *s_out = __fmul_rn(lr, rho);
    *dd_out = decoupled ? __fmul_rn(lr, __fmul_rn(P.decay, p.wd)) : 0.f;
    if (P.flags & kOcExport) {
      p.ratio[P.tensor] = (double)rho;
      p.wnorm[P.tensor] = (double)wn;
      p.unorm[P.tensor] = (double)un;
      if (!isfinite(a.hi) || !isfinite(b.hi))
        atomicOr(p.status, kStatusNonfinite);
    }
  }
  return true;
}

// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------
template <int kOpt, typename GT, bool kCopy>
__global__ void __launch_bounds__(kOcThreads, 1)
    onchip_step_kernel(const StepParams p, const OcParams q) {
  extern __shared__ float4 s_rows[];   // rows x (w[128] | m, then u[128])
  __shared__ OcShared sh;
  constexpr bool kLars = kOpt == kOptLars;
  constexpr int kNest = kLars ? 0 : kOpt;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // ---- prologue: the launch's independent loads run in separate warps and
  // meet at the first CTA barrier -- the abort and epoch words (the last
  // warp), eta (the warp before it), round 0's pieces (warp 8), and the step
  // count with the constants formed from it (warps 0-5)
  if (warp == kOcWarps - 1 && lane == 0) {
    sh.abort = ld_acquire_u32(q.bar + kBarAbort);
    sh.epoch = ld_acquire_u32(q.bar + kBarEpoch);
  }
  if (warp == kOcWarps - 2 && lane == 0)
    sh.lr = (p.flags & kFlagLrSchedule) ? 0.f : *p.d_lr;
  if (warp == 8 && q.n_rounds > 0) load_pieces(sh.tab[0], q, 0, lane);
  if (!kLars) {
    step_constants<kNest, false>(p, &sh.unused_draw, &sh.skip, &sh.k, &sh.t);
  } else if (threadIdx.x == 0) {
    const int64_t t = p.d_step ? *p.d_step : int64_t(0);
    sh.t = t;
    sh.skip = 0;
    sh.k = LambConsts{p.b1, p.omb1, p.b2, p.omb2, 1.f, 1.f, p.eps,
                      0.f, 0.f, 0.f, 0.f};
    if (blockIdx.x == 0) {
      StepScalars sc{};
      sc.t = t;
      sc.c1 = 1.f;
      sc.c2 = 1.f;
      sc.lr = step_lr(p, t);
      *p.scal = sc;
    }
  }
  zero_red(sh);
  __syncthreads();
  // a launch after one that gave up does nothing more; a step count < 1 is
  // skipped (status set by CTA 0)
  if (sh.abort || sh.skip) return;
  if (threadIdx.x == 0 && (p.flags & kFlagLrSchedule))
    sh.lr = step_lr(p, sh.t);
  if (q.n_rounds > 0) piece_rows(sh.tab[0]);
  __syncthreads();
  const LambConsts k = sh.k;
  const float lr = sh.lr;
  const bool decoupled = !kLars && (p.flags & kFlagDecoupledDecay) != 0;
  const float wd = p.wd;
  const float coef = kLars ? (float)p.trust : 1.f;

  if (q.n_rounds > 0) {
    fused_pass<kOpt, GT, kCopy>(sh, s_rows, nullptr, &sh.tab[0], k, wd,
                                decoupled);
    __syncthreads();
  }
  for (int r = 0; r < q.n_rounds; ++r) {
    OcTables& T = sh.tab[r & 1];
    OcTables* next = r + 1 < q.n_rounds ? &sh.tab[(r + 1) & 1] : nullptr;
    piece_sums(sh, T, q, write_tag(sh.epoch));
    if (threadIdx.x == 0) sh.ok = 1;
    if (next)
      load_tables(*next, q, r + 1);   // while the other CTAs finish
    else
      __syncthreads();
    zero_red(sh);
    for (int j = warp; j < T.np; j += kOcWarps)
      if (!piece_ratio(p, q, T.piece[j], coef, lr, decoupled,
                       wait_tag(q, sh.epoch), &T.s[j], &T.dd[j]))
        sh.ok = 0;
    __syncthreads();
    if (!sh.ok) return;   // the launch gave up
    fused_pass<kOpt, GT, kCopy>(sh, s_rows, &T, next, k, wd, decoupled);
    __syncthreads();   // T's buffer is reloaded for round r + 2
  }
  // The last CTA to finish advances the epoch and closes the step: every
  // CTA read t (and the N-LAMB product) before its ticket, which releases
  // it; CTA 0 stored the step scalars before its own.
  __syncthreads();
  if (threadIdx.x == 0 &&
      atom_add_acq_rel(q.bar + kBarTicket, 1u) == gridDim.x - 1u) {
    st_relaxed_u32(q.bar + kBarTicket, 0u);
    st_relaxed_u32(q.bar + kBarEpoch, sh.epoch + 1u);
    const StepScalars sc = *p.scal;
    if (kNest && p.d_mu_product) *p.d_mu_product = sc.mu_prod;
    close_step(p, sc);
  }
}

template <int kOpt, typename GT, bool kCopy>
int launch_one(const StepParams& p, const OcParams& q, int grid, int rows,
               cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kOcThreads);
  cfg.dynamicSmemBytes = (size_t)rows * kOcRowBytes;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return (int)cudaLaunchKernelEx(&cfg, onchip_step_kernel<kOpt, GT, kCopy>, p,
                                 q);
}

template <int kOpt, typename GT>
int launch_copy(const StepParams& p, const OcParams& q, int copy, int grid,
                int rows, cudaStream_t s) {
  return copy ? launch_one<kOpt, GT, true>(p, q, grid, rows, s)
              : launch_one<kOpt, GT, false>(p, q, grid, rows, s);
}

template <int kOpt>
int launch_opt(const StepParams& p, const OcParams& q, int g_bf16, int copy,
               int grid, int rows, cudaStream_t s) {
  return g_bf16 ? launch_copy<kOpt, __nv_bfloat16>(p, q, copy, grid, rows, s)
                : launch_copy<kOpt, float>(p, q, copy, grid, rows, s);
}

// Static shared memory of the largest instantiation, and the dynamic limit
// raised on every instantiation.
template <int kOpt, typename GT, bool kCopy>
int prepare_one(int dyn_bytes, int* static_bytes) {
  auto* f = onchip_step_kernel<kOpt, GT, kCopy>;
  if (dyn_bytes < 0) {
    cudaFuncAttributes a;
    const cudaError_t e = cudaFuncGetAttributes(&a, f);
    if (e != cudaSuccess) return (int)e;
    if ((int)a.sharedSizeBytes > *static_bytes)
      *static_bytes = (int)a.sharedSizeBytes;
    return 0;
  }
  return (int)cudaFuncSetAttribute(
      f, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn_bytes);
}

template <int kOpt>
int prepare_opt(int dyn_bytes, int* static_bytes) {
  int rc = prepare_one<kOpt, float, false>(dyn_bytes, static_bytes);
  if (!rc) rc = prepare_one<kOpt, float, true>(dyn_bytes, static_bytes);
  if (!rc) rc = prepare_one<kOpt, __nv_bfloat16, false>(dyn_bytes, static_bytes);
  if (!rc) rc = prepare_one<kOpt, __nv_bfloat16, true>(dyn_bytes, static_bytes);
  return rc;
}

int prepare_all(int dyn_bytes, int* static_bytes) {
  int rc = prepare_opt<0>(dyn_bytes, static_bytes);
  if (!rc) rc = prepare_opt<1>(dyn_bytes, static_bytes);
  if (!rc) rc = prepare_opt<2>(dyn_bytes, static_bytes);
  if (!rc) rc = prepare_opt<3>(dyn_bytes, static_bytes);
  return rc;
}

}  // namespace

int onchip_prepare(int device, int* rows_per_cta) {
  int optin = 0;
  cudaError_t e = cudaDeviceGetAttribute(
      &optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, device);
  if (e != cudaSuccess) return (int)e;
  int static_bytes = 0;
  int rc = prepare_all(-1, &static_bytes);
  if (rc) return rc;
  int rows = (optin - static_bytes) / kOcRowBytes;
  if (rows > kOcMaxRows) rows = kOcMaxRows;
  if (rows < 1) return (int)cudaErrorInvalidConfiguration;
  rc = prepare_all(rows * kOcRowBytes, &static_bytes);
  if (rc) return rc;
  // the launch needs one resident CTA per SM
  int blocks = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
      &blocks, onchip_step_kernel<0, __nv_bfloat16, true>, kOcThreads,
      (size_t)rows * kOcRowBytes);
  if (e != cudaSuccess) return (int)e;
  if (blocks < 1) return (int)cudaErrorInvalidConfiguration;
  *rows_per_cta = rows;
  return 0;
}

int launch_onchip(const StepParams& p, const OcParams& q, int opt,
                  int grad_bf16, int copy_bf16, int grid, int rows_per_cta,
                  void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (opt) {
    case 0: return launch_opt<0>(p, q, grad_bf16, copy_bf16, grid, rows_per_cta, s);
    case 1: return launch_opt<1>(p, q, grad_bf16, copy_bf16, grid, rows_per_cta, s);
    case 2: return launch_opt<2>(p, q, grad_bf16, copy_bf16, grid, rows_per_cta, s);
    default: return launch_opt<3>(p, q, grad_bf16, copy_bf16, grid, rows_per_cta, s);
  }
}

}  // namespace lamb
