// lamb_step_noalloc: one LAMB step that never allocates device memory.
//
// Who needs this: callers that must not call cudaMalloc -- code running
// under an allocator that owns all device memory (a framework caching
// allocator, a memory pool sized up front), code that must not hit the
// implicit device synchronisation a cudaMalloc/cudaFree can cause, or
// plugins that are handed a stream and buffers but no right to allocate.
// The plan API (lamb_plan_create) allocates its tables once with cudaMalloc;
// this entry point instead keeps every table, partial sum and counter in one
// fixed, file-scope device array that exists in every process that loads
// the library, on every GPU it runs on, until the process exits.
//
// The array is shared by all calls: calls that overlap on the GPU (different
// streams, or different host threads without ordering) race on it.  Each
// call rebuilds the tables and clears its counters, so it does not depend on
// what an earlier call left there.
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "lamb.h"
#include "lamb_internal.h"

namespace lamb {
namespace {

// ---- limits and layout of the scratch array --------------------------------
constexpr int kNaMaxTensors = 4096;
constexpr int kNaMaxChunks = 131072;          // 2^31 elements at 16384/chunk
constexpr int kNaChunk = kDefaultChunk;       // same chunking as the plan API

constexpr size_t na_align(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t kOffSizes = 0;
constexpr size_t kOffMask = na_align(kOffSizes + 8ull * kNaMaxTensors);
constexpr size_t kOffRaw = na_align(kOffMask + 1ull * kNaMaxTensors);  // 5 arrays
constexpr size_t kOffTensors = na_align(kOffRaw + 5ull * 8 * kNaMaxTensors);
constexpr size_t kOffPtrs = na_align(kOffTensors + sizeof(TensorDesc) * kNaMaxTensors);
constexpr size_t kOffChunks = na_align(kOffPtrs + sizeof(TensorPtrs) * kNaMaxTensors);
constexpr size_t kOffSlots = na_align(kOffChunks + sizeof(ChunkDesc) * (size_t)kNaMaxChunks);
constexpr size_t kOffTickets = na_align(kOffSlots + 8ull * kNaMaxChunks);
constexpr size_t kOffRatio = na_align(kOffTickets + 4ull * kNaMaxTensors);
constexpr size_t kOffWnorm = na_align(kOffRatio + 8ull * kNaMaxTensors);
constexpr size_t kOffUnorm = na_align(kOffWnorm + 8ull * kNaMaxTensors);
constexpr size_t kOffScal = na_align(kOffUnorm + 8ull * kNaMaxTensors);
constexpr size_t kOffStatus = na_align(kOffScal + sizeof(StepScalars));
constexpr size_t kOffCounters = na_align(kOffStatus + 4);
constexpr size_t kNaScratchBytes = na_align(kOffCounters + 16);
static_assert(kNaScratchBytes <= (4u << 20), "scratch layout exceeds 4 MiB");

// The scratch itself: 4 MiB per GPU, for the life of the process.
static __device__ __align__(256) unsigned char g_noalloc_scratch[4u << 20];

// Failures are reported through lamb_last_error() like every other call.
lamb_status_t na_fail(lamb_status_t st, const char* fmt, ...) {
  char msg[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(msg, sizeof(msg), fmt, ap);
  va_end(ap);
  set_last_error(msg);
  return st;
}

// ---- per-device set-up (symbol address, SM count, grid sizes) --------------
constexpr int kNaMaxDevices = 64;
struct NaDevice {
  unsigned char* scratch = nullptr;   // device address of g_noalloc_scratch
  int num_sms = 0;
  int occ[4] = {0, 0, 0, 0};          // pass1 f32/bf16 g, pass2 no copy/copy
};
NaDevice g_na_dev[kNaMaxDevices];
std::atomic<int> g_na_ready[kNaMaxDevices];
std::mutex g_na_mutex;

// Runs once per device, with that device current.
cudaError_t na_setup(int dev, NaDevice** out) {
  if (g_na_ready[dev].load(std::memory_order_acquire)) {
    *out = &g_na_dev[dev];
    return cudaSuccess;
  }
  std::lock_guard<std::mutex> lock(g_na_mutex);
  if (!g_na_ready[dev].load(std::memory_order_relaxed)) {
    NaDevice d;
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    d.scratch = static_cast<unsigned char*>(ptr);
    e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    int rc = occupancy_lamb_pass1(0, &d.occ[0]);
    if (!rc) rc = occupancy_lamb_pass1(1, &d.occ[1]);
    if (!rc) rc = occupancy_lamb_pass2(0, &d.occ[2]);
    if (!rc) rc = occupancy_lamb_pass2(1, &d.occ[3]);
    if (rc) return (cudaError_t)rc;
    g_na_dev[dev] = d;
    g_na_ready[dev].store(1, std::memory_order_release);
  }
  *out = &g_na_dev[dev];
  return cudaSuccess;
}

// ---- set-up kernel: builds the tables inside the scratch array -------------
// One CTA of 1024 threads.  Reads the per-tensor sizes, mask and pointer
// arrays the host copied into the scratch, and writes the tensor table,
// pointer table (with the 128-bit alignment flag), tickets, default results
// (ratio 1, norms 0), status and work counters; then every thread writes
// every 1024th chunk of the chunk table, finding its tensor by a binary
// search over the tensors' first chunks, kept in shared memory with the
// length of each tensor's last chunk.
constexpr int kSetupThreads = 1024;
constexpr int kPerThread = kNaMaxTensors / kSetupThreads;   // 4

__global__ void __launch_bounds__(kSetupThreads)
    noalloc_setup_kernel(int n, int has_mask, int grad_bf16, int has_v,
                         int copy_bf16) {
  unsigned char* s = g_noalloc_scratch;
  const int64_t* sizes = reinterpret_cast<const int64_t*>(s + kOffSizes);
  const uint8_t* mask = s + kOffMask;
  void* const* raw = reinterpret_cast<void* const*>(s + kOffRaw);
  TensorDesc* tens = reinterpret_cast<TensorDesc*>(s + kOffTensors);
  TensorPtrs* ptrs = reinterpret_cast<TensorPtrs*>(s + kOffPtrs);
  ChunkDesc* chunks = reinterpret_cast<ChunkDesc*>(s + kOffChunks);
  uint32_t* tickets = reinterpret_cast<uint32_t*>(s + kOffTickets);
  double* ratio = reinterpret_cast<double*>(s + kOffRatio);
  double* wnorm = reinterpret_cast<double*>(s + kOffWnorm);
  double* unorm = reinterpret_cast<double*>(s + kOffUnorm);
  uint32_t* status = reinterpret_cast<uint32_t*>(s + kOffStatus);
  uint32_t* counters = reinterpret_cast<uint32_t*>(s + kOffCounters);

  __shared__ int64_t part[kSetupThreads];
  __shared__ int32_t s_first[kNaMaxTensors];     // first chunk of tensor k
  __shared__ int32_t s_lastlen[kNaMaxTensors];   // length of its last chunk
  const int t = threadIdx.x;
  // chunk counts of this thread's tensors, then an exclusive scan
  int64_t local[kPerThread];
  int64_t sum = 0;
  for (int i = 0; i < kPerThread; ++i) {
    const int k = t * kPerThread + i;
    const int64_t d = k < n ? sizes[k] : 0;
    local[i] = (d + kNaChunk - 1) / kNaChunk;
    sum += local[i];
  }
  part[t] = sum;
  __syncthreads();
  for (int off = 1; off < kSetupThreads; off <<= 1) {   // Hillis-Steele
    const int64_t x = t >= off ? part[t - off] : 0;
    __syncthreads();
    part[t] += x;
    __syncthreads();
  }
  int64_t first = part[t] - sum;
  for (int i = 0; i < kPerThread; ++i) {
    const int k = t * kPerThread + i;
    if (k >= n) break;
    const int64_t d = sizes[k];
    TensorDesc td{};
    td.numel = d;
    td.first_chunk = (int32_t)first;
    td.n_chunks = (int32_t)local[i];
    td.decay = (!has_mask || mask[k]) ? 1.0f : 0.0f;
    tens[k] = td;
    s_first[k] = (int32_t)first;
    s_lastlen[k] = (int32_t)(d - (local[i] - 1) * kNaChunk);
    TensorPtrs tp{};
    tp.w = static_cast<float*>(raw[0 * kNaMaxTensors + k]);
    tp.g = raw[1 * kNaMaxTensors + k];
    tp.m = static_cast<float*>(raw[2 * kNaMaxTensors + k]);
    tp.v = has_v ? static_cast<float*>(raw[3 * kNaMaxTensors + k]) : nullptr;
    tp.copy = copy_bf16 ? raw[4 * kNaMaxTensors + k] : nullptr;
    const uintptr_t ga = grad_bf16 ? 8 : 16;
    const bool ok = (uintptr_t)tp.w % 16 == 0 && (uintptr_t)tp.m % 16 == 0 &&
                    (!tp.v || (uintptr_t)tp.v % 16 == 0) &&
                    (uintptr_t)tp.g % ga == 0 &&
                    (!tp.copy || (uintptr_t)tp.copy % 8 == 0);
    tp.vec_ok = ok ? 1u : 0u;
    ptrs[k] = tp;
    first += local[i];
    tickets[k] = 0u;
    ratio[k] = 1.0;
    wnorm[k] = 0.0;
    unorm[k] = 0.0;
  }
  if (t == 0) {
    *status = 0u;
    counters[0] = counters[1] = counters[2] = counters[3] = 0u;
  }
  __syncthreads();   // the tensor table is complete
  const int32_t n_chunks = (int32_t)part[kSetupThreads - 1];
  for (int32_t c = t; c < n_chunks; c += kSetupThreads) {
    // the last tensor whose first chunk is <= c (a 0-chunk tensor shares its
    // first chunk with the next one, which comes later and wins)
    int lo = 0, hi = n - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) / 2;
      if (s_first[mid] <= c) lo = mid;
      else hi = mid - 1;
    }
    // tensor lo holds chunk c; its chunks end where the next tensor's begin
    const int32_t end = lo + 1 < n ? s_first[lo + 1] : n_chunks;
    ChunkDesc cd;
    cd.offset = (int64_t)(c - s_first[lo]) * kNaChunk;
    cd.tensor = lo;
    cd.len = c + 1 == end ? s_lastlen[lo] : kNaChunk;
    chunks[c] = cd;
  }
}

}  // namespace
}  // namespace lamb

using namespace lamb;

extern "C" LAMB_API lamb_status_t lamb_step_noalloc(
    const int64_t* sizes, int32_t n_tensors, const uint8_t* decay_mask,
    int32_t grad_dtype, int32_t copy_dtype, void* const* w,
    const void* const* g, void* const* m, void* const* v,
    void* const* w_copy, const lamb_hyper_t* hyper, int64_t* d_step,
    const float* d_lr, double* d_ratio, cudaStream_t stream) {
  // ---- host-side checks (no device work yet) -----------------------------
  if (n_tensors < 1 || n_tensors > kNaMaxTensors)
    return na_fail(LAMB_ERR_INVALID_ARG,
                   "lamb_step_noalloc: n_tensors must be in [1, %d] (got %d)",
                   kNaMaxTensors, n_tensors);
  if (!sizes || !w || !g || !m || !v || !hyper || !d_lr)
    return na_fail(LAMB_ERR_INVALID_ARG,
                   "lamb_step_noalloc: sizes, w, g, m, v, hyper and d_lr are "
                   "required");
  if (grad_dtype != LAMB_F32 && grad_dtype != LAMB_BF16)
    return na_fail(LAMB_ERR_UNSUPPORTED_DTYPE,
                   "lamb_step_noalloc: grad_dtype %d unsupported", grad_dtype);
  if (copy_dtype != LAMB_DTYPE_NONE && copy_dtype != LAMB_BF16)
    return na_fail(LAMB_ERR_UNSUPPORTED_DTYPE,
                   "lamb_step_noalloc: copy_dtype %d unsupported", copy_dtype);
  const bool copy = copy_dtype == LAMB_BF16;
  if (copy && !w_copy)
    return na_fail(LAMB_ERR_INVALID_ARG,
                   "lamb_step_noalloc: w_copy is required with a bf16 copy");
  const lamb_hyper_t& h = *hyper;
  if (!(h.beta1 >= 0.0 && h.beta1 < 1.0) || !(h.beta2 >= 0.0 && h.beta2 < 1.0) ||
      !(h.eps >= 0.0 && std::isfinite(h.eps)) || !std::isfinite(h.weight_decay) ||
      (h.phi != LAMB_PHI_IDENTITY && h.phi != LAMB_PHI_CLIP) ||
      (h.phi == LAMB_PHI_CLIP && !(h.gamma_l <= h.gamma_u)) ||
      (h.flags & ~(uint32_t)(LAMB_FLAG_BIAS_CORRECTION | LAMB_FLAG_INCREMENT_STEP)))
    return na_fail(LAMB_ERR_INVALID_ARG, "lamb_step_noalloc: bad hyper");
  if (!d_step && (h.flags & (LAMB_FLAG_BIAS_CORRECTION | LAMB_FLAG_INCREMENT_STEP)))
    return na_fail(LAMB_ERR_INVALID_ARG,
                   "lamb_step_noalloc: d_step is NULL but the flags need it");
  int64_t n_chunks = 0;
  for (int k = 0; k < n_tensors; ++k) {
    const int64_t d = sizes[k];
    if (d < 0)
      return na_fail(LAMB_ERR_INVALID_ARG,
                     "lamb_step_noalloc: sizes[%d] is negative", k);
    if (d > (int64_t)kNaMaxChunks * kNaChunk)   // before any rounding sum
      return na_fail(LAMB_ERR_INVALID_ARG,
                     "lamb_step_noalloc: sizes[%d] = %lld exceeds the %lld "
                     "parameters the scratch holds", k, (long long)d,
                     (long long)kNaMaxChunks * kNaChunk);
    n_chunks += (d + kNaChunk - 1) / kNaChunk;
    if (n_chunks > kNaMaxChunks)
      return na_fail(LAMB_ERR_INVALID_ARG,
                     "lamb_step_noalloc: more than %d chunks of %d elements "
                     "(at most %lld parameters in total)",
                     kNaMaxChunks, kNaChunk,
                     (long long)kNaMaxChunks * kNaChunk);
    if (d > 0) {
      if (!w[k] || !g[k] || !m[k] || !v[k] || (copy && !w_copy[k]))
        return na_fail(LAMB_ERR_INVALID_ARG,
                       "lamb_step_noalloc: tensor %d has a NULL pointer", k);
      if ((uintptr_t)w[k] % 4 || (uintptr_t)m[k] % 4 || (uintptr_t)v[k] % 4 ||
          (uintptr_t)g[k] % (grad_dtype == LAMB_BF16 ? 2 : 4) ||
          (copy && (uintptr_t)w_copy[k] % 2))
        return na_fail(LAMB_ERR_INVALID_ARG,
                       "lamb_step_noalloc: tensor %d pointer not aligned to "
                       "its element size", k);
    }
  }

  // ---- per-device set-up (first call on a device) --------------------------
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kNaMaxDevices)
    return na_fail(LAMB_ERR_CUDA, "lamb_step_noalloc: cudaGetDevice: %s",
                   cudaGetErrorString(e));
  NaDevice* nd = nullptr;
  e = na_setup(dev, &nd);
  if (e != cudaSuccess)
    return na_fail(LAMB_ERR_CUDA, "lamb_step_noalloc: set-up: %s",
                   cudaGetErrorString(e));
  unsigned char* s = nd->scratch;

  // ---- stage the caller's host arrays into the scratch ---------------------
  const size_t nb = (size_t)n_tensors * 8;
  e = cudaMemcpyAsync(s + kOffSizes, sizes, nb, cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess && decay_mask)
    e = cudaMemcpyAsync(s + kOffMask, decay_mask, (size_t)n_tensors,
                        cudaMemcpyHostToDevice, stream);
  const void* const* arrays[5] = {w, g, m, v, copy ? w_copy : nullptr};
  for (int i = 0; i < 5 && e == cudaSuccess; ++i)
    if (arrays[i])
      e = cudaMemcpyAsync(s + kOffRaw + (size_t)i * 8 * kNaMaxTensors,
                          arrays[i], nb, cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess)
    return na_fail(LAMB_ERR_CUDA, "lamb_step_noalloc: staging copy: %s",
                   cudaGetErrorString(e));
  noalloc_setup_kernel<<<1, kSetupThreads, 0, stream>>>(
      n_tensors, decay_mask ? 1 : 0, grad_dtype == LAMB_BF16 ? 1 : 0, 1,
      copy ? 1 : 0);
  e = cudaGetLastError();
  if (e != cudaSuccess)
    return na_fail(LAMB_ERR_CUDA, "lamb_step_noalloc: set-up launch: %s",
                   cudaGetErrorString(e));

  // ---- the two LAMB passes on tables inside the scratch --------------------
  // The flags check above admits BIAS_CORRECTION and INCREMENT_STEP only:
  // the fields of the schedule, the gradient check and the N-LAMB product
  // stay zero / NULL here, which is what those two flags need.
  StepParams sp;
  std::memset(&sp, 0, sizeof(sp));
  fill_hyper(h, &sp);
  sp.chunks = reinterpret_cast<const ChunkDesc*>(s + kOffChunks);
  sp.tensors = reinterpret_cast<const TensorDesc*>(s + kOffTensors);
  sp.ptrs = reinterpret_cast<const TensorPtrs*>(s + kOffPtrs);
  sp.slots = reinterpret_cast<float2*>(s + kOffSlots);
  sp.tickets = reinterpret_cast<uint32_t*>(s + kOffTickets);
  sp.counters = reinterpret_cast<uint32_t*>(s + kOffCounters);
  sp.ratio = reinterpret_cast<double*>(s + kOffRatio);
  sp.wnorm = reinterpret_cast<double*>(s + kOffWnorm);
  sp.unorm = reinterpret_cast<double*>(s + kOffUnorm);
  sp.scal = reinterpret_cast<StepScalars*>(s + kOffScal);
  sp.status = reinterpret_cast<uint32_t*>(s + kOffStatus);
  sp.d_step = d_step;
  sp.d_lr = d_lr;
  sp.n_chunks = (int32_t)n_chunks;
  const int gbf = grad_dtype == LAMB_BF16 ? 1 : 0;
  auto grid_of = [&](int occ) {
    int64_t gsz = (int64_t)nd->num_sms * (occ < 1 ? 1 : occ);
    if (gsz > n_chunks) gsz = n_chunks;
    return (int)(gsz < 1 ? 1 : gsz);
  };
  int rc = launch_lamb_pass1(sp, 0, gbf, grid_of(nd->occ[gbf]), stream);
  if (!rc)
    rc = launch_lamb_pass2(sp, 0, gbf, copy ? 1 : 0,
                           grid_of(nd->occ[2 + (copy ? 1 : 0)]), stream);
  if (!rc && d_ratio)
    rc = (int)cudaMemcpyAsync(d_ratio, s + kOffRatio, nb,
                              cudaMemcpyDeviceToDevice, stream);
  if (rc)
    return na_fail(LAMB_ERR_CUDA, "lamb_step_noalloc: %s",
                   cudaGetErrorString((cudaError_t)rc));
  return LAMB_OK;
}
