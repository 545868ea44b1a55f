// Internal layout of a plan and the kernel parameter block.
//
// HBM layout of a plan (one cudaMalloc, carved in this order, each piece
// 256-byte aligned):
//   ChunkDesc  chunks[n_chunks]   16 B  read-only after create
//   TensorDesc tensors[n_tensors] 32 B  read-only after create
//   TensorPtrs ptrs[n_tensors]    48 B  written by bind
//   float2     slots[n_chunks]     8 B  per-chunk (sum w^2, sum u^2), pass 1
//   uint32     tickets[n_tensors]  4 B  chunks of tensor k finished in pass 1;
//                                       reset to 0 by the last one
//   double     ratio/wnorm/unorm[n_tensors]  per-tensor results
//   StepScalars, status word, work counters
//   float2     grad_slots[n_chunks] 8 B  per-chunk (sum g^2, sum 0*g), pass 1
//                                       with the gradient check
//   double     gsq/gnorm[n_tensors]     per-tensor sum g^2 and ||g_k||
//   GradCheck                           global ||g|| and the step's decision
#pragma once
#include <stdint.h>

#include <vector>

#include "lamb.h"

namespace lamb {

constexpr int kDefaultChunk = 16384;
constexpr int kThreads = 256;          // threads per CTA, all kernels
constexpr int kWarps = kThreads / 32;
constexpr int kMaxChunks = 1 << 30;

struct __align__(16) ChunkDesc {
  int64_t offset;   // first element of the chunk inside its tensor
  int32_t tensor;   // tensor index k
  int32_t len;      // elements in the chunk (1 .. chunk_elems)
};

struct __align__(16) TensorDesc {
  int64_t numel;
  int32_t first_chunk;
  int32_t n_chunks;
  float decay;      // 1.0f: weight decay applies, 0.0f: masked
  uint32_t pad[3];
};

struct __align__(16) TensorPtrs {
  float* w;
  const void* g;    // float or bf16
  float* m;
  float* v;         // may be null (LARS-only binding)
  void* copy;       // bf16 copy of w, or null
  uint32_t vec_ok;  // every array aligned for 4-element vector access
  uint32_t pad;
};

// Written by pass 1 (CTA 0) and read by pass 2, so both passes use the very
// same float constants.
struct __align__(16) StepScalars {
  int64_t t;
  float c1;         // 1/(1-beta1^t) (1 without bias correction)
  float c2;         // 1/(1-beta2^t)
  float lr;
  int32_t skip;     // 1: bad step count, nothing is written
  // N-LAMB / NN-LAMB: m_hat = am*m + ag*g, v_hat = bv*v + bg*g^2
  float am, ag, bv, bg;
  double mu_prod;   // prod_{i<=t} mu_i, stored back when the step completes
};

enum : uint32_t { kStatusNonfinite = 1u, kStatusBadStep = 2u,
                  kStatusWaitTimeout = 4u, kStatusGradNonfinite = 8u,
                  kStatusSkipped = 16u };
enum : uint32_t { kFlagBiasCorrection = 1u, kFlagIncrementStep = 2u,
                  kFlagLrSchedule = 4u, kFlagGradNorm = 8u,
                  kFlagSkipNonfinite = 16u, kFlagDecoupledDecay = 32u,
                  // internal: a launch that is not the step's last leaves
                  // t, the scheduled eta and the N-LAMB product alone
                  kFlagNoClose = 1u << 30,
                  // internal: pass 1 of a shard stores its chunk sums and
                  // finalises nothing (the sums are exchanged first)
                  kFlagNoFinalize = 1u << 29 };

// Gradient check of one step (kFlagGradNorm / kFlagSkipNonfinite).  Pass 1
// forms it; pass 2 reads the decision before it writes anything.
struct __align__(16) GradCheck {
  double norm;          // sqrt(sum over all tensors of sum g^2)
  uint32_t nonfinite;   // 1: some element of g was Inf or NaN
  uint32_t acc;         // OR of the tensors' flags while pass 1 runs
  uint32_t done;        // tensors finalised by the running pass 1 (ticket)
  uint32_t pad;
};

struct StepParams {
  const ChunkDesc* chunks;
  const TensorDesc* tensors;
  const TensorPtrs* ptrs;
  float2* slots;
  uint32_t* tickets;
  uint32_t* counters;     // [0] pass-1, [1] pass-2 work counter
  double* ratio;
  double* wnorm;
  double* unorm;
  StepScalars* scal;
  uint32_t* status;
  int64_t* d_step;
  const float* d_lr;
  // per-step constants, rounded once from double on the host
  float b1, omb1, b2, omb2, eps, wd;
  double beta1, beta2;
  // log2 of the bases of the step-count powers, formed on the host in fp64:
  // the device takes beta^t as exp2(t * log2(beta)) (fp64 pow is ~4.7x
  // slower than exp2 on sm_103a, and every CTA needs the values first)
  double log2_beta1, log2_beta2;
  double log2_mu_decay;   // psi * log2(0.96): 0.96^(t psi) of the Nadam
                          // momentum schedule
  double gamma_l, gamma_u, trust;
  int32_t phi;            // 0 identity, 1 clip
  uint32_t flags;
  int32_t n_chunks;
  // N-LAMB / NN-LAMB only
  double psi;             // momentum-schedule decay (Nadam's psi)
  double* d_mu_product;   // prod_{i<t} mu_i on entry, prod_{i<=t} on exit
  // learning-rate schedule (kFlagLrSchedule)
  double lr_base;
  int64_t lr_warmup, lr_total;
  float* d_lr_out;        // where the applied eta_t is written (may be null)
  // gradient check (kFlagGradNorm / kFlagSkipNonfinite)
  float2* grad_slots;     // per chunk (sum g^2, sum 0*g); the second is 0,
                          // or NaN if some element is Inf/NaN
  double* gsq;            // per tensor sum g^2
  double* gnorm;          // per tensor ||g_k||
  GradCheck* gcheck;
  int32_t n_tensors;
  int32_t n_live;         // tensors with at least one chunk
};

// Launchers (lamb_kernels.cu).  grid = number of CTAs of the persistent grid.
// Return cudaError_t as int to keep this header free of CUDA includes.
// nest: 0 LAMB, 1 N-LAMB, 2 NN-LAMB.  The gradient-check and deferred-moment
// variants are chosen from p.flags.
int launch_lamb_pass1(const StepParams& p, int nest, int grad_bf16, int grid,
                      void* stream);
int launch_lamb_pass2(const StepParams& p, int nest, int grad_bf16,
                      int copy_bf16, int grid, void* stream);
int launch_lars_pass1(const StepParams& p, int grad_bf16, int grid,
                      void* stream);
int launch_lars_pass2(const StepParams& p, int grad_bf16, int copy_bf16,
                      int grid, void* stream);
// Every tensor's rho_k and norms from the complete chunk slots (coef: 1 for
// LAMB, kappa for LARS).
int launch_finalize_all(const StepParams& p, double coef, void* stream);
// Chunk range [*begin, *end) of shard `rank` of `world`: contiguous ranges
// of the chunk table with about equal elements, cut at chunk boundaries
// (planner.cpp).
void shard_range(const ChunkDesc* chunks, int64_t n_chunks, int32_t world,
                 int32_t rank, int64_t* begin, int64_t* end);
// Resident CTAs per SM of each kernel instantiation (occupancy calculator).
int occupancy_lamb_pass1(int grad_bf16, int* blocks);
int occupancy_lamb_pass2(int copy_bf16, int* blocks);
int occupancy_lars_pass1(int grad_bf16, int* blocks);
int occupancy_lars_pass2(int copy_bf16, int* blocks);

// The hyperparameter-derived fields of a StepParams (lamb_capi.cu): betas,
// their complements and log2s, eps, lambda, phi and its bounds, kappa, flags.
void fill_hyper(const lamb_hyper_t& h, StepParams* sp);

// Sets the thread-local message returned by lamb_last_error() (lamb_capi.cu).
void set_last_error(const char* msg);

// Host planner (planner.cpp).  Returns 0 on success, else writes a message.
// Within tail_elems of either end of the layout the chunks hold tail_chunk
// elements (0: no tail).
int plan_chunks(const int64_t* sizes, int32_t n, int32_t chunk_elems,
                ChunkDesc* chunks, int64_t capacity, int64_t* n_chunks,
                TensorDesc* tensors, const uint8_t* decay_mask, char* err,
                int errlen, int64_t tail_elems = 0, int32_t tail_chunk = 0);
constexpr int kTailChunk = 2048;   // elements per chunk near the layout's ends

}  // namespace lamb
