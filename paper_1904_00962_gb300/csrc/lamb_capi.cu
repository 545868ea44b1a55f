// C ABI of the library (declared in include/lamb.h): plan lifecycle, binding,
// the LAMB / LARS step entry points, and queries.  Host code only; the
// kernels live in lamb_kernels.cu.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "lamb.h"
#include "lamb_internal.h"
#include "lamb_onchip.h"

using namespace lamb;

namespace {

thread_local char g_err[512] = "";

lamb_status_t fail(lamb_status_t st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return st;
}

lamb_status_t cuda_fail(cudaError_t e, const char* what) {
  if (e == cudaErrorMemoryAllocation)
    return fail(LAMB_ERR_OOM, "%s: %s", what, cudaGetErrorString(e));
  return fail(LAMB_ERR_CUDA, "%s: %s (%d)", what, cudaGetErrorString(e),
              (int)e);
}

}  // namespace

void lamb::set_last_error(const char* msg) {
  snprintf(g_err, sizeof(g_err), "%s", msg);
}

namespace {

constexpr int kMaxTimedSteps = 4096;
constexpr int kKernelsPerStep = 3;

// Restores the caller's current device on scope exit.
struct DeviceGuard {
  int prev = -1;
  cudaError_t err = cudaSuccess;
  explicit DeviceGuard(int dev) {
    err = cudaGetDevice(&prev);
    if (err == cudaSuccess && prev != dev) err = cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev)
      cudaSetDevice(prev);
  }
};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

// LAMB_ALGO_AUTO takes the on-chip step up to this many rounds (measured:
// ResNet-50, 7 rounds, 5.7% faster on-chip; the ragged layout, 623 rounds,
// 4.5% slower).
constexpr int kAutoMaxRounds = 32;

struct lamb_plan {
  int device = 0;
  int n_tensors = 0;
  int64_t n_chunks = 0;
  int64_t n_params = 0;
  int chunk_elems = kDefaultChunk;
  int64_t tail_elems = 0;       // elements at each end in short chunks
  int shard_world = 1, shard_rank = 0;
  int64_t shard_cb = 0, shard_ce = 0;   // this shard's chunk range
  int grad_bf16 = 0;
  int copy_bf16 = 0;
  int num_sms = 0;
  int blocks_per_sm_opt = 0;
  int grid[4] = {0, 0, 0, 0};  // lamb p1, lamb p2, lars p1, lars p2
  int algorithm = LAMB_ALGO_TWO_PASS;
  bool auto_algo = false;       // chosen by LAMB_ALGO_AUTO
  bool bound = false;
  bool has_v = false;
  int n_vec = 0;
  std::vector<TensorDesc> h_tensors;

  void* arena = nullptr;
  size_t arena_bytes = 0;
  ChunkDesc* chunks = nullptr;
  TensorDesc* tensors = nullptr;
  TensorPtrs* ptrs = nullptr;
  float2* slots = nullptr;
  uint32_t* tickets = nullptr;
  double* ratio = nullptr;
  double* wnorm = nullptr;
  double* unorm = nullptr;
  StepScalars* scal = nullptr;
  uint32_t* status = nullptr;
  uint32_t* counters = nullptr;
  // gradient check
  float2* grad_slots = nullptr;
  double* grad_sq = nullptr;
  double* grad_norm = nullptr;
  GradCheck* grad_check = nullptr;
  int n_live = 0;               // tensors with at least one chunk
  // on-chip single-touch tables
  int oc_grid = 0;
  int oc_rows = 0;              // rows of shared memory per CTA
  int oc_n_rounds = 0;
  int oc_n_streamed = 0;
  int64_t oc_n_slots = 0;
  int64_t oc_wait_ns = 0;
  int oc_extra = 0;
  std::vector<OcPiece> h_oc_pieces;   // without pointers (filled by bind)
  OcSlice* oc_slices = nullptr;
  OcPiece* oc_pieces = nullptr;
  uint64_t* oc_slots = nullptr;
  uint32_t* oc_bar = nullptr;
  // the streamed tensors' chunk table for the two-pass kernels
  int64_t oc_n_chunks = 0;
  int oc_sub_grid[4] = {0, 0, 0, 0};
  ChunkDesc* oc_chunks = nullptr;
  TensorDesc* oc_tensors = nullptr;

  bool timing = false;
  int timed_steps = 0;
  std::vector<cudaEvent_t> events;  // kMaxTimedSteps * (kKernelsPerStep + 1)
  std::vector<uint8_t> timed_kernels;  // kernels each timed step launched
};

void lamb::fill_hyper(const lamb_hyper_t& h, StepParams* sp) {
  // (1 - beta) formed in double and rounded once
  sp->b1 = (float)h.beta1;
  sp->omb1 = (float)(1.0 - h.beta1);
  sp->b2 = (float)h.beta2;
  sp->omb2 = (float)(1.0 - h.beta2);
  sp->eps = (float)h.eps;
  sp->wd = (float)h.weight_decay;
  sp->beta1 = h.beta1;
  sp->beta2 = h.beta2;
  sp->log2_beta1 = std::log2(h.beta1);   // -inf for beta = 0: beta^t = 0
  sp->log2_beta2 = std::log2(h.beta2);
  sp->gamma_l = h.gamma_l;
  sp->gamma_u = h.gamma_u;
  sp->trust = h.trust_coef;
  sp->phi = h.phi;
  sp->flags = h.flags;
}

extern "C" {

const char* lamb_last_error(void) { return g_err; }

int32_t lamb_abi_version(void) { return LAMB_ABI_VERSION; }

lamb_status_t lamb_layout_chunks(const int64_t* sizes, int32_t n_tensors,
                                 int32_t chunk_elems, int64_t tail_elems,
                                 int32_t* chunk_tensor, int64_t* chunk_offset,
                                 int32_t* chunk_len, int32_t capacity,
                                 int32_t* n_chunks) {
  if (n_chunks == nullptr) return fail(LAMB_ERR_INVALID_ARG, "n_chunks is NULL");
  if (capacity < 0) return fail(LAMB_ERR_INVALID_ARG, "capacity < 0");
  if (capacity > 0 && (!chunk_tensor || !chunk_offset || !chunk_len))
    return fail(LAMB_ERR_INVALID_ARG, "output arrays are NULL");
  if (chunk_elems == 0) chunk_elems = kDefaultChunk;
  std::vector<ChunkDesc> rows;
  try {
    rows.resize((size_t)capacity);
  } catch (const std::bad_alloc&) {
    return fail(LAMB_ERR_OOM, "host allocation failed");
  }
  int64_t count = 0;
  char err[256] = "";
  if (tail_elems < 0) return fail(LAMB_ERR_INVALID_ARG, "tail_elems < 0");
  const int rc = plan_chunks(sizes, n_tensors, chunk_elems,
                             capacity ? rows.data() : nullptr, capacity,
                             &count, nullptr, nullptr, err, sizeof(err),
                             tail_elems, kTailChunk);
  *n_chunks = (int32_t)(count > INT32_MAX ? INT32_MAX : count);
  if (rc) return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  if (count > capacity && capacity > 0)
    return fail(LAMB_ERR_INVALID_ARG, "capacity %d < %lld chunks", capacity,
                (long long)count);
  for (int64_t i = 0; i < count && i < capacity; ++i) {
    chunk_tensor[i] = rows[i].tensor;
    chunk_offset[i] = rows[i].offset;
    chunk_len[i] = rows[i].len;
  }
  return LAMB_OK;
}

lamb_status_t lamb_layout_shard(const int64_t* sizes, int32_t n_tensors,
                                int32_t chunk_elems, int64_t tail_elems,
                                int32_t world, int32_t rank,
                                int64_t* chunk_begin, int64_t* chunk_end) {
  if (!chunk_begin || !chunk_end)
    return fail(LAMB_ERR_INVALID_ARG, "chunk_begin and chunk_end are required");
  if (world < 1 || rank < 0 || rank >= world)
    return fail(LAMB_ERR_INVALID_ARG, "need 0 <= rank < world");
  if (tail_elems < 0) return fail(LAMB_ERR_INVALID_ARG, "tail_elems < 0");
  if (chunk_elems == 0) chunk_elems = kDefaultChunk;
  char err[256] = "";
  int64_t count = 0;
  if (plan_chunks(sizes, n_tensors, chunk_elems, nullptr, 0, &count, nullptr,
                  nullptr, err, sizeof(err), tail_elems, kTailChunk))
    return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  std::vector<ChunkDesc> rows;
  try {
    rows.resize((size_t)count);
  } catch (const std::bad_alloc&) {
    return fail(LAMB_ERR_OOM, "host allocation failed");
  }
  if (plan_chunks(sizes, n_tensors, chunk_elems, rows.data(), count, &count,
                  nullptr, nullptr, err, sizeof(err), tail_elems, kTailChunk))
    return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  shard_range(rows.data(), count, world, rank, chunk_begin, chunk_end);
  return LAMB_OK;
}

lamb_status_t lamb_layout_rounds(const int64_t* sizes, int32_t n_tensors,
                                 int32_t grid, int32_t rows_per_cta,
                                 int32_t* piece_round, int32_t* piece_cta,
                                 int32_t* piece_tensor, int64_t* piece_offset,
                                 int64_t* piece_len, int32_t* piece_first_row,
                                 int32_t* piece_rows, int64_t capacity,
                                 int64_t* n_pieces, int32_t* n_rounds) {
  if (!n_pieces || !n_rounds)
    return fail(LAMB_ERR_INVALID_ARG, "n_pieces and n_rounds are required");
  if (n_tensors < 1 || !sizes)
    return fail(LAMB_ERR_INVALID_ARG, "need n_tensors >= 1 and sizes");
  if (capacity < 0 ||
      (capacity > 0 && (!piece_round || !piece_cta || !piece_tensor ||
                        !piece_offset || !piece_len || !piece_first_row ||
                        !piece_rows)))
    return fail(LAMB_ERR_INVALID_ARG, "bad capacity or output arrays");
  int64_t total = 0;
  for (int32_t k = 0; k < n_tensors; ++k) {
    if (sizes[k] < 0)
      return fail(LAMB_ERR_INVALID_ARG, "sizes[%d] is negative", k);
    if (sizes[k] > (int64_t(1) << 62) - total)
      return fail(LAMB_ERR_INVALID_ARG, "total element count exceeds 2^62");
    total += sizes[k];
  }
  std::vector<OcSlice> slices;
  std::vector<OcPiece> pieces;
  std::vector<int32_t> streamed;
  int64_t n_slots = 0;
  int32_t rounds = 0;
  char err[256] = "";
  try {
    if (plan_onchip(sizes, n_tensors, nullptr, grid, rows_per_cta, &rounds,
                    &slices, &pieces, &streamed, &n_slots, err, sizeof(err)))
      return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  } catch (const std::bad_alloc&) {
    return fail(LAMB_ERR_OOM, "host allocation failed");
  }
  const int64_t total_pieces = (int64_t)(pieces.size() + streamed.size());
  *n_pieces = total_pieces;
  *n_rounds = rounds;
  if (total_pieces > capacity)
    return capacity == 0 ? LAMB_OK
                         : fail(LAMB_ERR_INVALID_ARG, "capacity too small");
  int64_t i = 0;
  for (int32_t r = 0; r < rounds; ++r) {
    for (int32_t c = 0; c < grid; ++c) {
      const OcSlice& sl = slices[(size_t)r * (size_t)grid + (size_t)c];
      for (int j = 0; j < sl.n_pieces; ++j) {
        const OcPiece& pc = pieces[(size_t)sl.piece_begin + (size_t)j];
        piece_round[i] = r;
        piece_cta[i] = c;
        piece_tensor[i] = pc.tensor;
        piece_offset[i] = pc.offset;
        piece_len[i] = pc.len;
        piece_first_row[i] = pc.first_row;
        piece_rows[i] = pc.n_rows;
        ++i;
      }
    }
  }
  for (int32_t k : streamed) {
    piece_round[i] = -1;
    piece_cta[i] = -1;
    piece_tensor[i] = k;
    piece_offset[i] = 0;
    piece_len[i] = sizes[k];
    piece_first_row[i] = 0;
    piece_rows[i] = 0;
    ++i;
  }
  return LAMB_OK;
}

static lamb_status_t plan_create(const int64_t* sizes, int32_t n_tensors,
                                 const uint8_t* decay_mask, int32_t grad_dtype,
                                 int32_t copy_dtype, int32_t device,
                                 const lamb_plan_options_t* opts,
                                 lamb_plan_t* out) {
  if (out == nullptr) return fail(LAMB_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (grad_dtype != LAMB_F32 && grad_dtype != LAMB_BF16)
    return fail(LAMB_ERR_UNSUPPORTED_DTYPE, "grad_dtype %d unsupported",
                grad_dtype);
  if (copy_dtype != LAMB_DTYPE_NONE && copy_dtype != LAMB_BF16)
    return fail(LAMB_ERR_UNSUPPORTED_DTYPE,
                "copy_dtype %d unsupported (NONE or BF16)", copy_dtype);
  int chunk = kDefaultChunk, bps = 0, algo = LAMB_ALGO_AUTO;
  int64_t wait_ms = 1000;
  int unmet_wait = 0, oc_max_ctas = 0, oc_rows_opt = 0;
  int64_t tail_opt = 0;
  int sh_world = 1, sh_rank = 0;
  if (opts) {
    if (opts->chunk_elems) chunk = opts->chunk_elems;
    if (opts->blocks_per_sm < 0)
      return fail(LAMB_ERR_INVALID_ARG, "blocks_per_sm < 0");
    bps = opts->blocks_per_sm;
    algo = opts->algorithm;
    if (algo != LAMB_ALGO_AUTO && algo != LAMB_ALGO_TWO_PASS &&
        algo != LAMB_ALGO_ON_CHIP)
      return fail(LAMB_ERR_INVALID_ARG, "unknown algorithm %d", algo);
    if (opts->wait_limit_ms < 0)
      return fail(LAMB_ERR_INVALID_ARG, "wait_limit_ms >= 0");
    if (opts->wait_limit_ms) wait_ms = opts->wait_limit_ms;
    unmet_wait = opts->test_unmet_wait != 0;
    if (opts->onchip_max_ctas < 0 || opts->onchip_rows < 0)
      return fail(LAMB_ERR_INVALID_ARG, "onchip_max_ctas, onchip_rows >= 0");
    oc_max_ctas = opts->onchip_max_ctas;
    oc_rows_opt = opts->onchip_rows;
    if (opts->tail_elems < 0)
      return fail(LAMB_ERR_INVALID_ARG, "tail_elems must be >= 0");
    tail_opt = opts->tail_elems;
    if (opts->shard_world < 0 || opts->shard_rank < 0 ||
        (opts->shard_world > 0 && opts->shard_rank >= opts->shard_world) ||
        (opts->shard_world == 0 && opts->shard_rank != 0))
      return fail(LAMB_ERR_INVALID_ARG,
                  "need 0 <= shard_rank < shard_world (or both 0)");
    if (opts->shard_world > 0) {
      sh_world = opts->shard_world;
      sh_rank = opts->shard_rank;
    }
  }
  const bool auto_algo = algo == LAMB_ALGO_AUTO;
  if (device < 0) return fail(LAMB_ERR_INVALID_ARG, "device < 0");

  lamb_plan* p = new (std::nothrow) lamb_plan();
  if (!p) return fail(LAMB_ERR_OOM, "host allocation failed");
  // Frees the plan (and its device arena, on its own device) on every path
  // that does not hand it to the caller, a thrown host allocation included.
  struct Owner {
    lamb_plan* p;
    ~Owner() {
      if (!p) return;
      if (p->arena) {
        int cur = -1;
        const bool got = cudaGetDevice(&cur) == cudaSuccess;
        if (cudaSetDevice(p->device) == cudaSuccess) cudaFree(p->arena);
        if (got) cudaSetDevice(cur);
      }
      delete p;
    }
  } owner{p};
  p->device = device;
  p->n_tensors = n_tensors;
  p->chunk_elems = chunk;
  p->grad_bf16 = grad_dtype == LAMB_BF16;
  p->copy_bf16 = copy_dtype == LAMB_BF16;
  p->blocks_per_sm_opt = bps;
  p->algorithm = algo;

  // ---- host planning ----------------------------------------------------
  char err[256] = "";
  int64_t nch = 0;
  if (n_tensors < 1 || sizes == nullptr) {
    return fail(LAMB_ERR_INVALID_ARG, n_tensors < 1
                                          ? "n_tensors must be >= 1"
                                          : "sizes is NULL");
  }
  p->h_tensors.resize((size_t)n_tensors);
  // validates the sizes, the chunk size and the tail before the device is
  // touched
  if (plan_chunks(sizes, n_tensors, chunk, nullptr, 0, &nch,
                  p->h_tensors.data(), decay_mask, err, sizeof(err),
                  tail_opt, kTailChunk)) {
    return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  }
  for (int k = 0; k < n_tensors; ++k) p->n_params += sizes[k];

  // ---- device ------------------------------------------------------------
  DeviceGuard guard(device);
  if (guard.err != cudaSuccess) {
    return cuda_fail(guard.err, "cudaSetDevice");
  }
  cudaError_t e = cudaDeviceGetAttribute(&p->num_sms,
                                         cudaDevAttrMultiProcessorCount, device);
  if (e != cudaSuccess) {
    return cuda_fail(e, "cudaDeviceGetAttribute");
  }
  // the chunk table, optionally with short chunks at both ends of the layout
  // (the last chunks each pass draws)
  p->tail_elems = tail_opt;
  if (plan_chunks(sizes, n_tensors, chunk, nullptr, 0, &nch,
                  p->h_tensors.data(), decay_mask, err, sizeof(err),
                  p->tail_elems, kTailChunk)) {
    return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  }
  std::vector<ChunkDesc> h_chunks((size_t)nch);
  if (plan_chunks(sizes, n_tensors, chunk, h_chunks.data(), nch, &nch,
                  p->h_tensors.data(), decay_mask, err, sizeof(err),
                  p->tail_elems, kTailChunk)) {
    return fail(LAMB_ERR_INVALID_ARG, "%s", err);
  }
  p->n_chunks = nch;
  for (int k = 0; k < n_tensors; ++k)
    p->n_live += p->h_tensors[(size_t)k].n_chunks > 0 ? 1 : 0;
  p->shard_world = sh_world;
  p->shard_rank = sh_rank;
  shard_range(h_chunks.data(), nch, sh_world, sh_rank, &p->shard_cb,
              &p->shard_ce);
  int occ[4] = {0, 0, 0, 0};
  int rc = occupancy_lamb_pass1(p->grad_bf16, &occ[0]);
  if (!rc) rc = occupancy_lamb_pass2(p->copy_bf16, &occ[1]);
  if (!rc) rc = occupancy_lars_pass1(p->grad_bf16, &occ[2]);
  if (!rc) rc = occupancy_lars_pass2(p->copy_bf16, &occ[3]);
  if (rc) {
    return cuda_fail((cudaError_t)rc, "occupancy query");
  }
  for (int i = 0; i < 4; ++i) {
    int b = occ[i] < 1 ? 1 : occ[i];
    if (bps > 0 && bps < b) b = bps;
    int64_t g = (int64_t)p->num_sms * b;
    if (g > nch) g = nch;      // never more CTAs than chunks
    if (g < 1) g = 1;
    p->grid[i] = (int)g;
  }
  // on-chip rounds
  std::vector<OcSlice> h_slices;
  std::vector<ChunkDesc> h_sub_chunks;
  std::vector<TensorDesc> h_sub_tensors;
  if (algo == LAMB_ALGO_ON_CHIP || auto_algo) {
    rc = onchip_prepare(device, &p->oc_rows);
    if (rc) {
      return cuda_fail((cudaError_t)rc, "on-chip kernel set-up");
    }
    if (oc_rows_opt > 0) {
      if (oc_rows_opt > p->oc_rows)
        return fail(LAMB_ERR_INVALID_ARG,
                    "onchip_rows %d exceeds the %d rows a CTA holds",
                    oc_rows_opt, p->oc_rows);
      p->oc_rows = oc_rows_opt;
    }
    int64_t total_rows = 0;
    for (int k = 0; k < n_tensors; ++k)
      total_rows += (sizes[k] + kOcRow - 1) / kOcRow;
    int ctas = p->num_sms;
    if (oc_max_ctas > 0 && oc_max_ctas < ctas) ctas = oc_max_ctas;
    p->oc_grid = onchip_grid(total_rows, ctas);
    std::vector<int32_t> streamed;
    if (plan_onchip(sizes, n_tensors, decay_mask, p->oc_grid, p->oc_rows,
                    &p->oc_n_rounds, &h_slices, &p->h_oc_pieces, &streamed,
                    &p->oc_n_slots, err, sizeof(err))) {
      return fail(LAMB_ERR_INVALID_ARG, "%s", err);
    }
    p->oc_n_streamed = (int)streamed.size();
    if (p->oc_n_rounds == 0) p->oc_grid = 1;   // nothing to do but close
    // AUTO: the on-chip step when no tensor is larger than a round and the
    // layout takes at most kAutoMaxRounds rounds.  With a streamed tensor
    // (BERT's word embedding), or with hundreds of rounds (the 10,000-tensor
    // ragged layout: 623), the two-pass step is as fast or faster; LARS steps
    // on several rounds also run two-pass (onchip_takes).
    if (auto_algo) {
      const bool fits = streamed.empty() && p->oc_n_rounds <= kAutoMaxRounds;
      algo = fits ? LAMB_ALGO_ON_CHIP : LAMB_ALGO_TWO_PASS;
      p->algorithm = algo;
      p->auto_algo = true;
      if (!fits) {
        h_slices.clear();
        p->h_oc_pieces.clear();
        streamed.clear();
        p->oc_n_rounds = 0;
        p->oc_n_streamed = 0;
        p->oc_n_slots = 0;
      }
    }
    if (!streamed.empty()) {
      // chunk table of the streamed tensors only (the others count as empty)
      std::vector<int64_t> sub((size_t)n_tensors, 0);
      for (int32_t k : streamed) sub[(size_t)k] = sizes[k];
      h_sub_tensors.resize((size_t)n_tensors);
      const int64_t sub_tail = tail_opt;
      if (plan_chunks(sub.data(), n_tensors, chunk, nullptr, 0,
                      &p->oc_n_chunks, h_sub_tensors.data(), decay_mask, err,
                      sizeof(err), sub_tail, kTailChunk)) {
        return fail(LAMB_ERR_INVALID_ARG, "%s", err);
      }
      h_sub_chunks.resize((size_t)p->oc_n_chunks);
      if (plan_chunks(sub.data(), n_tensors, chunk, h_sub_chunks.data(),
                      p->oc_n_chunks, &p->oc_n_chunks, h_sub_tensors.data(),
                      decay_mask, err, sizeof(err), sub_tail, kTailChunk)) {
        return fail(LAMB_ERR_INVALID_ARG, "%s", err);
      }
      for (int i = 0; i < 4; ++i)
        p->oc_sub_grid[i] = (int)(p->oc_n_chunks < p->grid[i]
                                      ? p->oc_n_chunks : p->grid[i]);
    }
    p->oc_wait_ns = wait_ms * 1000000;
    p->oc_extra = unmet_wait;
  }

  const size_t n = (size_t)n_tensors, c = (size_t)nch;
  size_t off = 0;
  auto carve = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + (bytes ? bytes : 1), 256);
    return at;
  };
  const size_t o_chunks = carve(c * sizeof(ChunkDesc));
  const size_t o_tensors = carve(n * sizeof(TensorDesc));
  const size_t o_ptrs = carve(n * sizeof(TensorPtrs));
  const size_t o_slots = carve(c * sizeof(float2));
  const size_t o_tickets = carve(n * sizeof(uint32_t));
  const size_t o_ratio = carve(n * sizeof(double));
  const size_t o_wnorm = carve(n * sizeof(double));
  const size_t o_unorm = carve(n * sizeof(double));
  const size_t o_scal = carve(sizeof(StepScalars));
  const size_t o_status = carve(sizeof(uint32_t));
  const size_t o_counters = carve(8 * sizeof(uint32_t));
  const size_t o_grad_slots = carve(c * sizeof(float2));
  const size_t o_grad_sq = carve(n * sizeof(double));
  const size_t o_grad_norm = carve(n * sizeof(double));
  const size_t o_grad_check = carve(sizeof(GradCheck));
  const size_t o_oc_chunks = carve(h_sub_chunks.size() * sizeof(ChunkDesc));
  const size_t o_oc_tensors = carve(h_sub_tensors.size() * sizeof(TensorDesc));
  const size_t o_oc_slices = carve(h_slices.size() * sizeof(OcSlice));
  const size_t o_oc_pieces = carve(p->h_oc_pieces.size() * sizeof(OcPiece));
  const size_t o_oc_slots = carve((size_t)p->oc_n_slots * 2 * sizeof(uint64_t));
  const size_t o_oc_bar = carve(kBarWords * sizeof(uint32_t));
  p->arena_bytes = off;
  e = cudaMalloc(&p->arena, p->arena_bytes);
  if (e != cudaSuccess) {
    return cuda_fail(e, "cudaMalloc(plan)");
  }
  char* base = static_cast<char*>(p->arena);
  p->chunks = reinterpret_cast<ChunkDesc*>(base + o_chunks);
  p->tensors = reinterpret_cast<TensorDesc*>(base + o_tensors);
  p->ptrs = reinterpret_cast<TensorPtrs*>(base + o_ptrs);
  p->slots = reinterpret_cast<float2*>(base + o_slots);
  p->tickets = reinterpret_cast<uint32_t*>(base + o_tickets);
  p->ratio = reinterpret_cast<double*>(base + o_ratio);
  p->wnorm = reinterpret_cast<double*>(base + o_wnorm);
  p->unorm = reinterpret_cast<double*>(base + o_unorm);
  p->scal = reinterpret_cast<StepScalars*>(base + o_scal);
  p->status = reinterpret_cast<uint32_t*>(base + o_status);
  p->counters = reinterpret_cast<uint32_t*>(base + o_counters);
  p->grad_slots = reinterpret_cast<float2*>(base + o_grad_slots);
  p->grad_sq = reinterpret_cast<double*>(base + o_grad_sq);
  p->grad_norm = reinterpret_cast<double*>(base + o_grad_norm);
  p->grad_check = reinterpret_cast<GradCheck*>(base + o_grad_check);
  p->oc_chunks = reinterpret_cast<ChunkDesc*>(base + o_oc_chunks);
  p->oc_tensors = reinterpret_cast<TensorDesc*>(base + o_oc_tensors);
  p->oc_slices = reinterpret_cast<OcSlice*>(base + o_oc_slices);
  p->oc_pieces = reinterpret_cast<OcPiece*>(base + o_oc_pieces);
  p->oc_slots = reinterpret_cast<uint64_t*>(base + o_oc_slots);
  p->oc_bar = reinterpret_cast<uint32_t*>(base + o_oc_bar);

  // zero everything (tickets, counters, status, results, pointer table)
  e = cudaMemset(p->arena, 0, p->arena_bytes);
  if (e == cudaSuccess && c)
    e = cudaMemcpy(p->chunks, h_chunks.data(), c * sizeof(ChunkDesc),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(p->tensors, p->h_tensors.data(), n * sizeof(TensorDesc),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !h_sub_chunks.empty())
    e = cudaMemcpy(p->oc_chunks, h_sub_chunks.data(),
                   h_sub_chunks.size() * sizeof(ChunkDesc),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !h_sub_tensors.empty())
    e = cudaMemcpy(p->oc_tensors, h_sub_tensors.data(),
                   h_sub_tensors.size() * sizeof(TensorDesc),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !h_slices.empty())
    e = cudaMemcpy(p->oc_slices, h_slices.data(),
                   h_slices.size() * sizeof(OcSlice), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) {
    // trust ratio 1 for every tensor until a step computes it; a 0-element
    // tensor keeps it (its norms are 0, and a zero norm gives ratio 1)
    std::vector<double> ones(n, 1.0);
    e = cudaMemcpy(p->ratio, ones.data(), n * sizeof(double),
                   cudaMemcpyHostToDevice);
  }
  if (e != cudaSuccess) {
    return cuda_fail(e, "plan upload");
  }
  owner.p = nullptr;
  *out = p;
  return LAMB_OK;
}

lamb_status_t lamb_plan_create(const int64_t* sizes, int32_t n_tensors,
                               const uint8_t* decay_mask, int32_t grad_dtype,
                               int32_t copy_dtype, int32_t device,
                               const lamb_plan_options_t* opts,
                               lamb_plan_t* out) {
  try {
    return plan_create(sizes, n_tensors, decay_mask, grad_dtype, copy_dtype,
                       device, opts, out);
  } catch (const std::bad_alloc&) {
    return fail(LAMB_ERR_OOM, "host allocation failed");
  }
}

lamb_status_t lamb_plan_bind(lamb_plan_t plan, void* const* w,
                             const void* const* g, void* const* m,
                             void* const* v, void* const* w_copy,
                             cudaStream_t stream) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  if (!w || !g || !m)
    return fail(LAMB_ERR_INVALID_ARG, "w, g and m pointer arrays are required");
  if (plan->copy_bf16 && !w_copy)
    return fail(LAMB_ERR_INVALID_ARG,
                "plan writes a bf16 copy: w_copy pointer array is required");
  const int n = plan->n_tensors;
  std::vector<TensorPtrs> h;
  try {
    h.resize((size_t)n);
  } catch (const std::bad_alloc&) {
    return fail(LAMB_ERR_OOM, "host allocation failed");
  }
  int n_vec = 0;
  const uintptr_t ga = plan->grad_bf16 ? 8 : 16;
  for (int k = 0; k < n; ++k) {
    TensorPtrs& t = h[(size_t)k];
    std::memset(&t, 0, sizeof(t));
    t.w = static_cast<float*>(w[k]);
    t.g = g[k];
    t.m = static_cast<float*>(m[k]);
    t.v = v ? static_cast<float*>(v[k]) : nullptr;
    t.copy = plan->copy_bf16 ? w_copy[k] : nullptr;
    if (plan->h_tensors[(size_t)k].numel > 0) {
      if (!t.w || !t.g || !t.m)
        return fail(LAMB_ERR_INVALID_ARG, "tensor %d: NULL w/g/m pointer", k);
      if (v && !t.v)
        return fail(LAMB_ERR_INVALID_ARG, "tensor %d: NULL v pointer", k);
      if (plan->copy_bf16 && !t.copy)
        return fail(LAMB_ERR_INVALID_ARG, "tensor %d: NULL w_copy pointer", k);
      if ((uintptr_t)t.w % 4 || (uintptr_t)t.m % 4 ||
          (t.v && (uintptr_t)t.v % 4) ||
          (uintptr_t)t.g % (plan->grad_bf16 ? 2 : 4) ||
          (t.copy && (uintptr_t)t.copy % 2))
        return fail(LAMB_ERR_INVALID_ARG,
                    "tensor %d: pointer not aligned to its element size", k);
    }
    bool ok = (uintptr_t)t.w % 16 == 0 && (uintptr_t)t.m % 16 == 0 &&
              (!t.v || (uintptr_t)t.v % 16 == 0) &&
              (uintptr_t)t.g % ga == 0 && (!t.copy || (uintptr_t)t.copy % 8 == 0);
    t.vec_ok = ok ? 1u : 0u;
    n_vec += ok;
  }
  // on-chip pieces carry their tensor's pointers
  std::vector<OcPiece> oc;
  try {
    oc = plan->h_oc_pieces;
  } catch (const std::bad_alloc&) {
    return fail(LAMB_ERR_OOM, "host allocation failed");
  }
  for (OcPiece& pc : oc) {
    const TensorPtrs& t = h[(size_t)pc.tensor];
    pc.w = t.w;
    pc.g = t.g;
    pc.m = t.m;
    pc.v = t.v;
    pc.copy = t.copy;
    pc.flags = (pc.flags & ~kOcVec) | (t.vec_ok ? kOcVec : 0u);
  }
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  cudaError_t e = cudaMemcpyAsync(plan->ptrs, h.data(),
                                  (size_t)n * sizeof(TensorPtrs),
                                  cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess && !oc.empty())
    e = cudaMemcpyAsync(plan->oc_pieces, oc.data(), oc.size() * sizeof(OcPiece),
                        cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "pointer table upload");
  plan->bound = true;
  plan->has_v = v != nullptr;
  plan->n_vec = n_vec;
  return LAMB_OK;
}

static lamb_status_t check_hyper(const lamb_hyper_t* h, bool lamb) {
  if (!h) return fail(LAMB_ERR_INVALID_ARG, "hyper is NULL");
  if (!(h->beta1 >= 0.0 && h->beta1 < 1.0))
    return fail(LAMB_ERR_INVALID_ARG, "beta1 must be in [0, 1)");
  if (lamb && !(h->beta2 >= 0.0 && h->beta2 < 1.0))
    return fail(LAMB_ERR_INVALID_ARG, "beta2 must be in [0, 1)");
  if (lamb && !(h->eps >= 0.0 && std::isfinite(h->eps)))
    return fail(LAMB_ERR_INVALID_ARG, "eps must be finite and >= 0");
  if (!std::isfinite(h->weight_decay))
    return fail(LAMB_ERR_INVALID_ARG, "weight_decay must be finite");
  if (h->phi != LAMB_PHI_IDENTITY && h->phi != LAMB_PHI_CLIP)
    return fail(LAMB_ERR_INVALID_ARG, "phi must be IDENTITY or CLIP");
  if (h->phi == LAMB_PHI_CLIP && !(h->gamma_l <= h->gamma_u))
    return fail(LAMB_ERR_INVALID_ARG, "clip bounds need gamma_l <= gamma_u");
  if (!lamb && !std::isfinite(h->trust_coef))
    return fail(LAMB_ERR_INVALID_ARG, "trust_coef must be finite");
  if (h->flags & ~(uint32_t)(LAMB_FLAG_BIAS_CORRECTION |
                             LAMB_FLAG_INCREMENT_STEP | LAMB_FLAG_LR_SCHEDULE |
                             LAMB_FLAG_GRAD_NORM | LAMB_FLAG_SKIP_NONFINITE |
                             LAMB_FLAG_DECOUPLED_DECAY))
    return fail(LAMB_ERR_INVALID_ARG, "unknown flag bits 0x%x", h->flags);
  if (!lamb && (h->flags & LAMB_FLAG_DECOUPLED_DECAY))
    return fail(LAMB_ERR_INVALID_ARG,
                "LAMB_FLAG_DECOUPLED_DECAY applies to lamb_step and "
                "nlamb_step only");
  if ((h->flags & LAMB_FLAG_LR_SCHEDULE) &&
      !(h->lr_base >= 0.0 && std::isfinite(h->lr_base) &&
        h->lr_warmup_steps >= 0 && h->lr_total_steps >= 1))
    return fail(LAMB_ERR_INVALID_ARG,
                "lr schedule needs lr_base >= 0, warmup >= 0, total >= 1");
  return LAMB_OK;
}

static void fill_params(lamb_plan* p, const lamb_hyper_t* h, int64_t* d_step,
                        const float* d_lr, StepParams* sp) {
  std::memset(sp, 0, sizeof(*sp));
  fill_hyper(*h, sp);
  sp->chunks = p->chunks;
  sp->tensors = p->tensors;
  sp->ptrs = p->ptrs;
  sp->slots = p->slots;
  sp->tickets = p->tickets;
  sp->counters = p->counters;
  sp->ratio = p->ratio;
  sp->wnorm = p->wnorm;
  sp->unorm = p->unorm;
  sp->scal = p->scal;
  sp->status = p->status;
  sp->d_step = d_step;
  sp->d_lr = d_lr;
  sp->n_chunks = (int32_t)p->n_chunks;
  sp->grad_slots = p->grad_slots;
  sp->gsq = p->grad_sq;
  sp->gnorm = p->grad_norm;
  sp->gcheck = p->grad_check;
  sp->n_tensors = p->n_tensors;
  sp->n_live = p->n_live;
  if (h->flags & LAMB_FLAG_LR_SCHEDULE) {
    sp->lr_base = h->lr_base;
    sp->lr_warmup = h->lr_warmup_steps;
    sp->lr_total = h->lr_total_steps;
    sp->d_lr_out = const_cast<float*>(d_lr);
  }
}

// The on-chip kernel runs every step but those with the gradient check or the
// skip mode (their decision needs all of g before anything is written), and,
// on a plan that AUTO made on-chip, LARS steps over several rounds: LARS's
// two-pass step moves only 8 B/parameter more, less than the per-round cost
// of the on-chip exchange (ResNet-50: 0.111 against 0.120 ms).
static bool onchip_takes(const lamb_plan* p, uint32_t flags, bool lars) {
  return p->algorithm == LAMB_ALGO_ON_CHIP &&
         !(flags & (LAMB_FLAG_GRAD_NORM | LAMB_FLAG_SKIP_NONFINITE)) &&
         !(lars && p->auto_algo && p->oc_n_rounds > 1);
}

// An on-chip step: the streamed tensors (if any) through the two-pass kernels
// over their own chunk table, with the closing writes (t + 1, the scheduled
// eta, the N-LAMB product) left to the on-chip kernel, which runs last.
// Records an event after each kernel when ev is not NULL; returns the number
// of kernels launched, or a negated CUDA error.
static int launch_onchip_step(const lamb_plan* p, const StepParams& sp,
                              int opt, cudaStream_t stream, cudaEvent_t* ev) {
  int n = 0, rc = 0;
  if (p->oc_n_chunks > 0) {
    StepParams sub = sp;
    sub.chunks = p->oc_chunks;
    sub.tensors = p->oc_tensors;
    sub.n_chunks = (int32_t)p->oc_n_chunks;
    sub.flags |= kFlagNoClose;
    const bool lars = opt == 3;
    rc = lars ? launch_lars_pass1(sub, p->grad_bf16, p->oc_sub_grid[2], stream)
              : launch_lamb_pass1(sub, opt, p->grad_bf16, p->oc_sub_grid[0],
                                  stream);
    if (!rc && ev) rc = (int)cudaEventRecord(ev[++n], stream);
    else if (!rc) ++n;
    if (!rc)
      rc = lars ? launch_lars_pass2(sub, p->grad_bf16, p->copy_bf16,
                                    p->oc_sub_grid[3], stream)
                : launch_lamb_pass2(sub, opt, p->grad_bf16, p->copy_bf16,
                                    p->oc_sub_grid[1], stream);
    if (!rc && ev) rc = (int)cudaEventRecord(ev[++n], stream);
    else if (!rc) ++n;
    if (rc) return -rc;
  }
  OcParams q;
  q.slices = p->oc_slices;
  q.pieces = p->oc_pieces;
  q.slots = p->oc_slots;
  q.bar = p->oc_bar;
  q.n_rounds = p->oc_n_rounds;
  q.extra_arrivals = p->oc_extra;
  q.wait_limit_ns = p->oc_wait_ns;
  rc = launch_onchip(sp, q, opt, p->grad_bf16, p->copy_bf16, p->oc_grid,
                     p->oc_rows, stream);
  if (!rc && ev) rc = (int)cudaEventRecord(ev[++n], stream);
  else if (!rc) ++n;
  return rc ? -rc : n;
}

static lamb_status_t run_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                              int64_t* d_step, const float* d_lr,
                              cudaStream_t stream, bool lamb) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  lamb_status_t st = check_hyper(hyper, lamb);
  if (st != LAMB_OK) return st;
  if (plan->shard_world > 1)
    return fail(LAMB_ERR_INVALID_ARG,
                "a sharded plan steps with lamb_shard_pass1/lamb_shard_pass2");
  if (!plan->bound) return fail(LAMB_ERR_NOT_BOUND, "plan is not bound");
  if (lamb && !plan->has_v)
    return fail(LAMB_ERR_NOT_BOUND, "lamb_step needs v: bind v pointers");
  const bool sched = (hyper->flags & LAMB_FLAG_LR_SCHEDULE) != 0;
  if (!d_lr && !sched) return fail(LAMB_ERR_INVALID_ARG, "d_lr is NULL");
  const bool needs_step =
      (hyper->flags & LAMB_FLAG_INCREMENT_STEP) || sched ||
      (lamb && (hyper->flags & LAMB_FLAG_BIAS_CORRECTION));
  if (needs_step && !d_step)
    return fail(LAMB_ERR_INVALID_ARG, "d_step is NULL but the flags need it");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  StepParams sp;
  fill_params(plan, hyper, d_step, d_lr, &sp);

  const bool timed = plan->timing && plan->timed_steps < kMaxTimedSteps;
  cudaEvent_t* ev = timed ? &plan->events[(size_t)plan->timed_steps *
                                          (kKernelsPerStep + 1)]
                          : nullptr;
  cudaError_t e = cudaSuccess;
  if (timed) e = cudaEventRecord(ev[0], stream);
  int rc = (int)e;
  if (onchip_takes(plan, hyper->flags, !lamb)) {
    const int n = rc ? -rc : launch_onchip_step(plan, sp, lamb ? 0 : 3, stream,
                                                 ev);
    if (n < 0) return cuda_fail((cudaError_t)-n, lamb ? "lamb_step" : "lars_step");
    if (timed) plan->timed_kernels[(size_t)plan->timed_steps++] = (uint8_t)n;
    return LAMB_OK;
  }
  // two-pass plans, and on-chip plans with the gradient check or the skip
  // mode
  if (!rc)
    rc = lamb ? launch_lamb_pass1(sp, 0, plan->grad_bf16, plan->grid[0], stream)
              : launch_lars_pass1(sp, plan->grad_bf16, plan->grid[2], stream);
  if (!rc && timed) rc = (int)cudaEventRecord(ev[1], stream);
  if (!rc)
    rc = lamb ? launch_lamb_pass2(sp, 0, plan->grad_bf16, plan->copy_bf16,
                                  plan->grid[1], stream)
              : launch_lars_pass2(sp, plan->grad_bf16, plan->copy_bf16,
                                  plan->grid[3], stream);
  if (!rc && timed) rc = (int)cudaEventRecord(ev[2], stream);
  if (rc) return cuda_fail((cudaError_t)rc, lamb ? "lamb_step" : "lars_step");
  if (timed) plan->timed_kernels[(size_t)plan->timed_steps++] = 2;
  return LAMB_OK;
}

lamb_status_t lamb_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                        int64_t* d_step, const float* d_lr,
                        cudaStream_t stream) {
  return run_step(plan, hyper, d_step, d_lr, stream, true);
}

lamb_status_t lars_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                        int64_t* d_step, const float* d_lr,
                        cudaStream_t stream) {
  return run_step(plan, hyper, d_step, d_lr, stream, false);
}

lamb_status_t nlamb_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                         double momentum_decay, int32_t nesterov_second_moment,
                         int64_t* d_step, const float* d_lr,
                         double* d_mu_product, cudaStream_t stream) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  lamb_status_t st = check_hyper(hyper, true);
  if (st != LAMB_OK) return st;
  if (!(momentum_decay >= 0.0 && std::isfinite(momentum_decay)))
    return fail(LAMB_ERR_INVALID_ARG, "momentum_decay must be finite, >= 0");
  if (nesterov_second_moment != 0 && nesterov_second_moment != 1)
    return fail(LAMB_ERR_INVALID_ARG, "nesterov_second_moment must be 0 or 1");
  if (plan->shard_world > 1)
    return fail(LAMB_ERR_INVALID_ARG,
                "a sharded plan steps with lamb_shard_pass1/lamb_shard_pass2");
  if (!plan->bound) return fail(LAMB_ERR_NOT_BOUND, "plan is not bound");
  if (!plan->has_v)
    return fail(LAMB_ERR_NOT_BOUND, "nlamb_step needs v: bind v pointers");
  if (!d_step || !d_mu_product ||
      (!d_lr && !(hyper->flags & LAMB_FLAG_LR_SCHEDULE)))
    return fail(LAMB_ERR_INVALID_ARG,
                "d_step, d_mu_product and d_lr (or a schedule) are required");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  StepParams sp;
  fill_params(plan, hyper, d_step, d_lr, &sp);
  sp.psi = momentum_decay;
  sp.log2_mu_decay = momentum_decay * std::log2(0.96);
  sp.d_mu_product = d_mu_product;
  const int nest = nesterov_second_moment ? 2 : 1;
  const bool timed = plan->timing && plan->timed_steps < kMaxTimedSteps;
  cudaEvent_t* ev = timed ? &plan->events[(size_t)plan->timed_steps *
                                          (kKernelsPerStep + 1)]
                          : nullptr;
  int rc = timed ? (int)cudaEventRecord(ev[0], stream) : 0;
  if (onchip_takes(plan, hyper->flags, false)) {
    const int n = rc ? -rc : launch_onchip_step(plan, sp, nest, stream, ev);
    if (n < 0) return cuda_fail((cudaError_t)-n, "nlamb_step");
    if (timed) plan->timed_kernels[(size_t)plan->timed_steps++] = (uint8_t)n;
    return LAMB_OK;
  }
  if (!rc)
    rc = launch_lamb_pass1(sp, nest, plan->grad_bf16, plan->grid[0], stream);
  if (!rc && timed) rc = (int)cudaEventRecord(ev[1], stream);
  if (!rc)
    rc = launch_lamb_pass2(sp, nest, plan->grad_bf16, plan->copy_bf16,
                           plan->grid[1], stream);
  if (!rc && timed) rc = (int)cudaEventRecord(ev[2], stream);
  if (rc) return cuda_fail((cudaError_t)rc, "nlamb_step");
  if (timed) plan->timed_kernels[(size_t)plan->timed_steps++] = 2;
  return LAMB_OK;
}

// Shared checks and parameters of the two halves of a sharded step.
static lamb_status_t shard_params(lamb_plan_t plan, const lamb_hyper_t* hyper,
                                  int32_t optimizer, double momentum_decay,
                                  int64_t* d_step, const float* d_lr,
                                  double* d_mu_product, StepParams* sp) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  if (optimizer < LAMB_OPT_LAMB || optimizer > LAMB_OPT_NNLAMB)
    return fail(LAMB_ERR_INVALID_ARG, "unknown optimizer %d", optimizer);
  const bool lars = optimizer == LAMB_OPT_LARS;
  const bool nest = optimizer >= LAMB_OPT_NLAMB;
  lamb_status_t st = check_hyper(hyper, !lars);
  if (st != LAMB_OK) return st;
  if (hyper->flags & (LAMB_FLAG_GRAD_NORM | LAMB_FLAG_SKIP_NONFINITE))
    return fail(LAMB_ERR_INVALID_ARG,
                "a sharded step takes neither GRAD_NORM nor SKIP_NONFINITE");
  if (!plan->bound) return fail(LAMB_ERR_NOT_BOUND, "plan is not bound");
  if (!lars && !plan->has_v)
    return fail(LAMB_ERR_NOT_BOUND, "this optimizer needs v: bind v pointers");
  const bool sched = (hyper->flags & LAMB_FLAG_LR_SCHEDULE) != 0;
  if (!d_lr && !sched) return fail(LAMB_ERR_INVALID_ARG, "d_lr is NULL");
  const bool needs_step =
      (hyper->flags & LAMB_FLAG_INCREMENT_STEP) || sched || nest ||
      (!lars && (hyper->flags & LAMB_FLAG_BIAS_CORRECTION));
  if (needs_step && !d_step)
    return fail(LAMB_ERR_INVALID_ARG, "d_step is NULL but the step needs it");
  if (nest && !(momentum_decay >= 0.0 && std::isfinite(momentum_decay)))
    return fail(LAMB_ERR_INVALID_ARG, "momentum_decay must be finite, >= 0");
  if (nest && !d_mu_product)
    return fail(LAMB_ERR_INVALID_ARG, "N-LAMB needs d_mu_product");
  fill_params(plan, hyper, d_step, d_lr, sp);
  if (nest) {
    sp->psi = momentum_decay;
    sp->log2_mu_decay = momentum_decay * std::log2(0.96);
    sp->d_mu_product = d_mu_product;
  }
  // this shard's chunks; the slots keep their global chunk index
  sp->chunks = plan->chunks + plan->shard_cb;
  sp->slots = plan->slots + plan->shard_cb;
  sp->n_chunks = (int32_t)(plan->shard_ce - plan->shard_cb);
  return LAMB_OK;
}

static int shard_grid(const lamb_plan* p, int which) {
  const int64_t n = p->shard_ce - p->shard_cb;
  const int g = p->grid[which];
  return n < 1 ? 1 : (n < g ? (int)n : g);
}

lamb_status_t lamb_shard_pass1(lamb_plan_t plan, const lamb_hyper_t* hyper,
                               int32_t optimizer, double momentum_decay,
                               int64_t* d_step, const float* d_lr,
                               double* d_mu_product, cudaStream_t stream) {
  StepParams sp;
  lamb_status_t st = shard_params(plan, hyper, optimizer, momentum_decay,
                                  d_step, d_lr, d_mu_product, &sp);
  if (st != LAMB_OK) return st;
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  sp.flags |= kFlagNoFinalize;
  // every slot starts at zero, so that a sum over the ranks' arrays is exact
  cudaError_t e = cudaMemsetAsync(plan->slots, 0,
                                  (size_t)plan->n_chunks * sizeof(float2),
                                  stream);
  int rc = (int)e;
  if (!rc)
    rc = optimizer == LAMB_OPT_LARS
             ? launch_lars_pass1(sp, plan->grad_bf16, shard_grid(plan, 2),
                                 stream)
             : launch_lamb_pass1(sp, optimizer - (optimizer >= 2 ? 1 : 0),
                                 plan->grad_bf16, shard_grid(plan, 0), stream);
  if (rc) return cuda_fail((cudaError_t)rc, "lamb_shard_pass1");
  return LAMB_OK;
}

lamb_status_t lamb_shard_pass2(lamb_plan_t plan, const lamb_hyper_t* hyper,
                               int32_t optimizer, double momentum_decay,
                               int64_t* d_step, const float* d_lr,
                               double* d_mu_product, cudaStream_t stream) {
  StepParams sp;
  lamb_status_t st = shard_params(plan, hyper, optimizer, momentum_decay,
                                  d_step, d_lr, d_mu_product, &sp);
  if (st != LAMB_OK) return st;
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  const bool lars = optimizer == LAMB_OPT_LARS;
  StepParams all = sp;   // the finaliser reads every tensor's slots
  all.chunks = plan->chunks;
  all.slots = plan->slots;
  all.n_chunks = (int32_t)plan->n_chunks;
  int rc = launch_finalize_all(all, lars ? hyper->trust_coef : 1.0, stream);
  if (!rc)
    rc = lars ? launch_lars_pass2(sp, plan->grad_bf16, plan->copy_bf16,
                                  shard_grid(plan, 3), stream)
              : launch_lamb_pass2(sp, optimizer - (optimizer >= 2 ? 1 : 0),
                                  plan->grad_bf16, plan->copy_bf16,
                                  shard_grid(plan, 1), stream);
  if (rc) return cuda_fail((cudaError_t)rc, "lamb_shard_pass2");
  return LAMB_OK;
}

lamb_status_t lamb_plan_partials(lamb_plan_t plan, float** d_partials,
                                 int64_t* n_floats) {
  if (!plan || !d_partials || !n_floats)
    return fail(LAMB_ERR_INVALID_ARG, "NULL argument");
  *d_partials = reinterpret_cast<float*>(plan->slots);
  *n_floats = 2 * plan->n_chunks;
  return LAMB_OK;
}

lamb_status_t lamb_plan_copy_partials(lamb_plan_t plan, float* buf,
                                      int32_t to_plan, cudaStream_t stream) {
  if (!plan || !buf) return fail(LAMB_ERR_INVALID_ARG, "NULL argument");
  if (to_plan != 0 && to_plan != 1)
    return fail(LAMB_ERR_INVALID_ARG, "to_plan must be 0 or 1");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  const size_t bytes = (size_t)plan->n_chunks * sizeof(float2);
  const cudaError_t e =
      to_plan ? cudaMemcpyAsync(plan->slots, buf, bytes, cudaMemcpyDefault,
                                stream)
              : cudaMemcpyAsync(buf, plan->slots, bytes, cudaMemcpyDefault,
                                stream);
  if (e != cudaSuccess) return cuda_fail(e, "partials copy");
  return LAMB_OK;
}

lamb_status_t lamb_plan_trust_ratios(lamb_plan_t plan, const double** d_ratio,
                                     const double** d_wnorm,
                                     const double** d_unorm) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  if (d_ratio) *d_ratio = plan->ratio;
  if (d_wnorm) *d_wnorm = plan->wnorm;
  if (d_unorm) *d_unorm = plan->unorm;
  return LAMB_OK;
}

lamb_status_t lamb_plan_grad_norms(lamb_plan_t plan, const double** d_gnorm,
                                   const double** d_gnorm_global,
                                   const uint32_t** d_nonfinite) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  if (d_gnorm) *d_gnorm = plan->grad_norm;
  if (d_gnorm_global) *d_gnorm_global = &plan->grad_check->norm;
  if (d_nonfinite) *d_nonfinite = &plan->grad_check->nonfinite;
  return LAMB_OK;
}

lamb_status_t lamb_plan_copy_grad_norms(lamb_plan_t plan, double* gnorm,
                                        double* gnorm_global,
                                        uint32_t* nonfinite,
                                        cudaStream_t stream) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  cudaError_t e = cudaSuccess;
  if (gnorm)
    e = cudaMemcpyAsync(gnorm, plan->grad_norm,
                        (size_t)plan->n_tensors * sizeof(double),
                        cudaMemcpyDefault, stream);
  if (e == cudaSuccess && gnorm_global)
    e = cudaMemcpyAsync(gnorm_global, &plan->grad_check->norm, sizeof(double),
                        cudaMemcpyDefault, stream);
  if (e == cudaSuccess && nonfinite)
    e = cudaMemcpyAsync(nonfinite, &plan->grad_check->nonfinite,
                        sizeof(uint32_t), cudaMemcpyDefault, stream);
  if (e != cudaSuccess) return cuda_fail(e, "grad norm copy");
  return LAMB_OK;
}

lamb_status_t lamb_plan_copy_trust_ratios(lamb_plan_t plan, double* ratio,
                                          double* wnorm, double* unorm,
                                          cudaStream_t stream) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  const size_t bytes = (size_t)plan->n_tensors * sizeof(double);
  const double* src[3] = {plan->ratio, plan->wnorm, plan->unorm};
  double* dst[3] = {ratio, wnorm, unorm};
  for (int i = 0; i < 3; ++i) {
    if (!dst[i]) continue;
    cudaError_t e = cudaMemcpyAsync(dst[i], src[i], bytes, cudaMemcpyDefault,
                                    stream);
    if (e != cudaSuccess) return cuda_fail(e, "trust ratio copy");
  }
  return LAMB_OK;
}

lamb_status_t lamb_plan_query(lamb_plan_t plan, uint32_t* status_bits,
                              int32_t clear, cudaStream_t stream) {
  if (!plan || !status_bits)
    return fail(LAMB_ERR_INVALID_ARG, "plan or status_bits is NULL");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  uint32_t h = 0;
  cudaError_t e = cudaMemcpyAsync(&h, plan->status, sizeof(h),
                                  cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess && clear)
    e = cudaMemsetAsync(plan->status, 0, sizeof(uint32_t), stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "status query");
  *status_bits = h;
  return LAMB_OK;
}

lamb_status_t lamb_plan_get_info(lamb_plan_t plan, lamb_plan_info_t* info) {
  if (!plan || !info) return fail(LAMB_ERR_INVALID_ARG, "NULL argument");
  std::memset(info, 0, sizeof(*info));
  info->n_tensors = plan->n_tensors;
  info->n_chunks = (int32_t)plan->n_chunks;
  info->n_params = plan->n_params;
  info->chunk_elems = plan->chunk_elems;
  info->grid_blocks = plan->grid[0];
  info->threads_per_block = kThreads;
  info->num_sms = plan->num_sms;
  info->device = plan->device;
  info->grad_dtype = plan->grad_bf16 ? LAMB_BF16 : LAMB_F32;
  info->copy_dtype = plan->copy_bf16 ? LAMB_BF16 : LAMB_DTYPE_NONE;
  info->bound = plan->bound ? 1 : 0;
  info->n_vector_tensors = plan->n_vec;
  info->device_bytes = (int64_t)plan->arena_bytes;
  info->algorithm = plan->algorithm;
  if (plan->algorithm == LAMB_ALGO_ON_CHIP) {
    info->grid_blocks = plan->oc_grid;
    info->threads_per_block = kOcThreads;
  }
  info->n_rounds = plan->oc_n_rounds;
  info->n_streamed_tensors = plan->oc_n_streamed;
  info->rows_per_cta = plan->oc_rows;
  info->tail_elems = plan->tail_elems;
  info->shard_world = plan->shard_world;
  info->shard_rank = plan->shard_rank;
  info->shard_chunk_begin = plan->shard_cb;
  info->shard_chunk_end = plan->shard_ce;
  info->row_elems = kOcRow;
  return LAMB_OK;
}

lamb_status_t lamb_plan_set_timing(lamb_plan_t plan, int32_t enable) {
  if (!plan) return fail(LAMB_ERR_INVALID_ARG, "plan is NULL");
  const size_t n_events = (size_t)kMaxTimedSteps * (kKernelsPerStep + 1);
  if (enable && plan->events.size() < n_events) {
    DeviceGuard guard(plan->device);
    if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
    try {
      plan->timed_kernels.assign((size_t)kMaxTimedSteps, 0);
      plan->events.reserve(n_events);
    } catch (const std::bad_alloc&) {
      return fail(LAMB_ERR_OOM, "host allocation failed");
    }
    // only created events are kept (destroy releases exactly those); a
    // failed call leaves timing off and the next one carries on
    while (plan->events.size() < n_events) {
      cudaEvent_t ev;
      cudaError_t e = cudaEventCreate(&ev);
      if (e != cudaSuccess) return cuda_fail(e, "cudaEventCreate");
      plan->events.push_back(ev);
    }
  }
  plan->timing = enable != 0;
  plan->timed_steps = 0;
  return LAMB_OK;
}

lamb_status_t lamb_plan_read_timing(lamb_plan_t plan, int32_t* n_steps,
                                    double* ms_per_kernel, int32_t n_kernels) {
  if (!plan || !n_steps || (n_kernels > 0 && !ms_per_kernel))
    return fail(LAMB_ERR_INVALID_ARG, "NULL argument");
  DeviceGuard guard(plan->device);
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  for (int j = 0; j < n_kernels; ++j) ms_per_kernel[j] = 0.0;
  for (int s = 0; s < plan->timed_steps; ++s) {
    const int per_step = plan->timed_kernels[(size_t)s];
    cudaEvent_t* ev = &plan->events[(size_t)s * (kKernelsPerStep + 1)];
    cudaError_t e = cudaEventSynchronize(ev[per_step]);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
    for (int j = 0; j < per_step && j < n_kernels; ++j) {
      float ms = 0.f;
      e = cudaEventElapsedTime(&ms, ev[j], ev[j + 1]);
      if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
      ms_per_kernel[j] += ms;
    }
  }
  *n_steps = plan->timed_steps;
  plan->timed_steps = 0;
  return LAMB_OK;
}

lamb_status_t lamb_plan_destroy(lamb_plan_t plan) {
  if (!plan) return LAMB_OK;
  DeviceGuard guard(plan->device);
  cudaError_t e = cudaSuccess;
  if (guard.err == cudaSuccess) {
    e = cudaDeviceSynchronize();
    for (auto& ev : plan->events) cudaEventDestroy(ev);
    if (plan->arena) {
      cudaError_t e2 = cudaFree(plan->arena);
      if (e == cudaSuccess) e = e2;
    }
  }
  delete plan;
  if (guard.err != cudaSuccess) return cuda_fail(guard.err, "cudaSetDevice");
  if (e != cudaSuccess) return cuda_fail(e, "lamb_plan_destroy");
  return LAMB_OK;
}

}  // extern "C"
