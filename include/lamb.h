/*
 * lamb.h -- C ABI of the GB300 (sm_103a) layerwise-adaptive optimizer step.
 *
 * The library applies one step of LAMB (You et al., "Large Batch
 * Optimization for Deep Learning: Training BERT in 76 minutes", ICLR 2020,
 * Algorithm 2) or LARS (Algorithm 1 of the same paper) to every parameter
 * tensor of a model in one call.  A "block" x^(i) of Section 2 is one
 * parameter tensor here; norms, trust ratios and weight decay are per tensor.
 *
 * Per tensor k, with step count t >= 1, lambda_k = lambda * mask_k:
 *   LAMB (Algorithm 2):
 *     m <- beta1 m + (1-beta1) g,          v <- beta2 v + (1-beta2) g^2
 *     r  = (m / (1-beta1^t)) / (sqrt(v / (1-beta2^t)) + eps) + lambda_k w
 *     rho_k = phi(||w_k||) / ||r_k||       (1 if either norm is 0)
 *     w <- w - eta * rho_k * r
 *   LARS (Algorithm 1, with a trust coefficient kappa):
 *     m <- beta1 m + (1-beta1) (g + lambda_k w)
 *     rho_k = kappa * phi(||w_k||) / ||m_k|| (1 if either norm is 0)
 *     w <- w - eta * rho_k * m
 *   phi (Section 3) is the identity or min(max(z, gamma_l), gamma_u).
 * m and v are stored without bias correction; the correction is applied only
 * where r is formed.  eps is added outside the square root.
 *
 * Types and layout: w, m, v are contiguous float32 arrays (one per tensor);
 * g is float32 or bfloat16; an optional bfloat16 copy of the new w is written
 * with round-to-nearest-even.  All tensor pointers are DEVICE pointers on the
 * plan's device.  Pointers aligned to 16 bytes (8 bytes for bfloat16 arrays)
 * take the vectorised path; others are handled element by element.
 *
 * Ownership: the caller owns w, g, m, v, the bf16 copy, the step counter,
 * the learning rate and the streams.  The plan owns its chunk table, pointer
 * table, partial sums, norms, trust ratios and counters, and frees them in
 * lamb_plan_destroy.  Bound pointers must stay valid until the last step
 * that uses them has completed.
 *
 * Errors: every call returns a lamb_status_t; nothing throws across the ABI.
 * Argument errors are detected on the host before any launch; a
 * thread-local message is available from lamb_last_error().  CUDA launch
 * errors are reported without synchronising.  Conditions only visible on
 * the device (a step count < 1, non-finite norms) set bits in the plan's
 * device status word, read with lamb_plan_query().
 *
 * Threading: a plan may be used from one host thread at a time.
 */
#ifndef LAMB_GB300_H
#define LAMB_GB300_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LAMB_ABI_VERSION 3

/* Only the entry points below are exported from liblamb.so. */
#if defined(__GNUC__)
#define LAMB_API __attribute__((visibility("default")))
#else
#define LAMB_API
#endif

typedef enum {
  LAMB_OK = 0,
  LAMB_ERR_INVALID_ARG = 1,        /* bad size, count, pointer or value   */
  LAMB_ERR_UNSUPPORTED_DTYPE = 2,  /* dtype code not supported here       */
  LAMB_ERR_CUDA = 3,               /* a CUDA runtime call or launch failed */
  LAMB_ERR_OOM = 4,                /* device or host allocation failed    */
  LAMB_ERR_NOT_BOUND = 5           /* step before lamb_plan_bind, or the
                                      array the step needs was not bound  */
} lamb_status_t;

typedef enum {
  LAMB_DTYPE_NONE = -1,            /* "no bf16 copy"                      */
  LAMB_F32 = 0,
  LAMB_BF16 = 1
} lamb_dtype_t;

/* phi of Section 3 */
typedef enum { LAMB_PHI_IDENTITY = 0, LAMB_PHI_CLIP = 1 } lamb_phi_t;

/* lamb_hyper_t.flags */
#define LAMB_FLAG_BIAS_CORRECTION 0x1u  /* divide by (1-beta^t), Alg. 2 and
                                           the appendix on adam-correction */
#define LAMB_FLAG_INCREMENT_STEP  0x2u  /* the step writes *d_step = t + 1
                                           on the device when it completes */
#define LAMB_FLAG_LR_SCHEDULE     0x4u  /* eta_t from t on the device
                                           (Section 4): eta_0 t / T_w for
                                           t < T_w, else eta_0 max(0, 1 -
                                           t / T); d_lr may be NULL, else
                                           the step writes the eta_t it
                                           applied there                   */
#define LAMB_FLAG_GRAD_NORM       0x8u  /* pass 1 also forms ||g_k|| of every
                                           tensor and the global ||g|| =
                                           sqrt(sum_k ||g_k||^2), and checks
                                           every gradient element for Inf /
                                           NaN (lamb_plan_grad_norms).  The
                                           sums are fp32 per chunk, fp64
                                           across chunks: a chunk whose sum
                                           of g^2 exceeds FLT_MAX reports an
                                           infinite norm without counting as
                                           non-finite                       */
#define LAMB_FLAG_SKIP_NONFINITE  0x10u /* implies GRAD_NORM.  If any element
                                           of g is Inf or NaN the step writes
                                           nothing: w, m, v, the bf16 copy,
                                           *d_step, the scheduled *d_lr and
                                           the N-LAMB product keep their
                                           values, and LAMB_STATUS_SKIPPED is
                                           set.  Pass 2 then forms and writes
                                           m, v instead of pass 1: one more
                                           read of g per step              */
#define LAMB_FLAG_DECOUPLED_DECAY 0x20u /* lamb_step / nlamb_step only: the
                                           decay term leaves the normalised
                                           direction, u = r, rho = phi(||w||)
                                           / ||r||, w <- w - eta rho r - eta
                                           lambda_k w (an ablation of Alg. 2's
                                           r + lambda w; not in the paper)  */

/* bits of the device status word (lamb_plan_query) */
#define LAMB_STATUS_NONFINITE 0x1u      /* a tensor's sum of w^2 or of r^2
                                           (LARS: m^2) was Inf/NaN         */
#define LAMB_STATUS_BAD_STEP  0x2u      /* *d_step < 1 with bias correction:
                                           the step was skipped, nothing was
                                           written                          */
#define LAMB_STATUS_WAIT_TIMEOUT 0x4u   /* on-chip: a wait for the other
                                           CTAs' partial sums inside the
                                           kernel (wait_limit_ms) gave up
                                           and the rest of the launch gave up
                                           with it, so the step is
                                           incomplete and the plan must be
                                           destroyed (its later steps do
                                           nothing); never expected         */
#define LAMB_STATUS_GRAD_NONFINITE 0x8u /* GRAD_NORM: a gradient element was
                                           Inf or NaN                       */
#define LAMB_STATUS_SKIPPED   0x10u     /* SKIP_NONFINITE: a step was skipped
                                           for that reason                  */

/* Hyperparameters.  Doubles on purpose: (1 - beta) is formed in double and
 * rounded once to float, so e.g. beta2 = 0.999 gives 1-beta2 = 0.001 to
 * float precision.  eta and t are read from device memory instead (any
 * schedule stays on the device; the step is CUDA-graph capturable). */
typedef struct {
  double beta1;          /* Alg. 1/2 beta1 (LARS momentum)                  */
  double beta2;          /* Alg. 2 beta2 (ignored by lars_step)             */
  double eps;            /* Alg. 2 epsilon (ignored by lars_step)           */
  double weight_decay;   /* lambda; applied to tensors whose mask is 1      */
  double gamma_l;        /* phi clip bounds, used when phi == LAMB_PHI_CLIP */
  double gamma_u;
  double trust_coef;     /* LARS kappa (ignored by lamb_step)               */
  int32_t phi;           /* lamb_phi_t                                      */
  uint32_t flags;        /* LAMB_FLAG_*                                     */
  /* LAMB_FLAG_LR_SCHEDULE only */
  double lr_base;            /* eta_0 >= 0                                  */
  int64_t lr_warmup_steps;   /* T_w >= 0 (0: no warmup)                     */
  int64_t lr_total_steps;    /* T >= 1                                      */
} lamb_hyper_t;

/* lamb_plan_options_t.algorithm */
#define LAMB_ALGO_AUTO 0          /* the library's default: on-chip when no
                                     tensor is larger than an on-chip round
                                     (~4.2M parameters on a GB300) and the
                                     layout takes at most 32 rounds, else
                                     two-pass; on such an on-chip plan,
                                     lars_step over more than one round runs
                                     the two-pass kernels
                                     (lamb_plan_get_info reports the choice) */
#define LAMB_ALGO_TWO_PASS 1      /* two streaming kernels per step: 40 B of
                                     HBM traffic per parameter (bf16 g/copy) */
/* 2 is not assigned (plan creation rejects it)                           */
#define LAMB_ALGO_ON_CHIP 3       /* one cooperative kernel per step (one CTA
                                     per SM).  Consecutive tensors are taken in
                                     rounds that fit the grid's shared memory
                                     (rows of LAMB_ONCHIP_ROW_ELEMS elements,
                                     216 rows per SM: ~4.2M parameters on
                                     152 SMs): pass 1 reads g, m, v, w once and
                                     keeps w and the direction on chip while
                                     the CTAs exchange their partial sums,
                                     pass 2 writes w from there -- 28
                                     B/parameter (bf16 g/copy).  A
                                     tensor larger than a round ("streamed")
                                     goes through the two-pass kernels first
                                     (40 B/parameter; 3 launches per step
                                     then).  LAMB, LARS, N-LAMB, NN-LAMB,
                                     decoupled decay and the schedule; the
                                     gradient check and the skip mode run
                                     two-pass on such a plan               */
#define LAMB_ONCHIP_ROW_ELEMS 128
#define LAMB_TAIL_CHUNK_ELEMS 2048

/* Optional plan-creation knobs (pass NULL for defaults). */
typedef struct {
  int32_t chunk_elems;   /* two-pass: elements per chunk, multiple of 1024 in
                            [1024, 1<<24]; 0 = default (16384)             */
  int32_t blocks_per_sm; /* resident CTAs per SM for the persistent grid;
                            0 = as many as the occupancy calculator allows */
  int32_t algorithm;     /* LAMB_ALGO_*                                     */
  int32_t wait_limit_ms; /* on-chip: a CTA's wait for the other CTAs'
                            partial sums gives up after this long
                            (LAMB_STATUS_WAIT_TIMEOUT); 0 = 1000           */
  int32_t test_unmet_wait; /* on-chip, for tests of the give-up path only:
                            nonzero makes every CTA wait for partial sums
                            tagged for a launch that never comes, so the
                            first wait runs out after wait_limit_ms and the
                            launch returns with LAMB_STATUS_WAIT_TIMEOUT.  0
                            for every real use                             */
  int32_t onchip_max_ctas; /* on-chip: at most this many CTAs (one per SM);
                            0 = the SM count                               */
  int32_t onchip_rows;   /* on-chip: rows of shared memory per CTA, at most
                            what the device holds; 0 = that maximum.  Fewer
                            rows make smaller rounds                       */
  int64_t tail_elems;    /* two-pass: elements at each end of the layout
                            (the tensors laid end to end) cut into chunks
                            of LAMB_TAIL_CHUNK_ELEMS, so that the last
                            chunks a pass draws are short; 0 = none (the
                            default: measured slower on every layout here,
                            the short chunks' per-chunk cost outweighs the
                            shorter tail).  A tail needs chunk_elems >=
                            LAMB_TAIL_CHUNK_ELEMS                          */
  int32_t shard_world;   /* data-parallel shards of the step (0 or 1: the
                            plan covers every chunk).  With shard_world = W
                            the plan owns chunk range shard_rank of W
                            (lamb_layout_shard) and is driven by
                            lamb_shard_pass1 / lamb_shard_pass2; every rank
                            must build its plan from the same sizes,
                            chunk_elems and tail_elems                     */
  int32_t shard_rank;    /* 0 <= shard_rank < shard_world                  */
} lamb_plan_options_t;

typedef struct {
  int32_t n_tensors;
  int32_t n_chunks;
  int64_t n_params;
  int32_t chunk_elems;
  int32_t grid_blocks;       /* CTAs per launch (persistent grid)           */
  int32_t threads_per_block;
  int32_t num_sms;
  int32_t device;
  int32_t grad_dtype;
  int32_t copy_dtype;
  int32_t bound;             /* 1 after a successful lamb_plan_bind         */
  int32_t n_vector_tensors;  /* tensors on the vectorised path (after bind) */
  int64_t device_bytes;      /* device memory owned by the plan             */
  int32_t algorithm;         /* LAMB_ALGO_TWO_PASS or LAMB_ALGO_ON_CHIP     */
  int32_t n_rounds;          /* on-chip: rounds per step                    */
  int32_t n_streamed_tensors;/* on-chip: tensors too large for a round,
                                updated by the two-pass kernels            */
  int32_t rows_per_cta;      /* on-chip: rows of shared memory per CTA      */
  int32_t row_elems;         /* on-chip: elements per row                   */
  int64_t tail_elems;        /* two-pass: elements at each end of the layout
                                in LAMB_TAIL_CHUNK_ELEMS chunks             */
  int32_t shard_world;       /* 1 if the plan is not sharded                */
  int32_t shard_rank;
  int64_t shard_chunk_begin; /* this shard's chunks [begin, end)            */
  int64_t shard_chunk_end;
} lamb_plan_info_t;

typedef struct lamb_plan* lamb_plan_t;

/* Build a plan for n_tensors tensors of the given element counts.
 *   sizes       host array [n_tensors], each >= 0 (0-element tensors are
 *               allowed: they get trust ratio 1 and norms 0).
 *   decay_mask  host array [n_tensors]; 1 = weight decay applies (lambda_k =
 *               lambda), 0 = masked (lambda_k = 0).  NULL = all 1.
 *   grad_dtype  LAMB_F32 or LAMB_BF16.
 *   copy_dtype  LAMB_DTYPE_NONE or LAMB_BF16 (bf16 copy of the new w).
 *   device      CUDA device ordinal; the plan's memory lives there.
 *   opts        NULL or tuning knobs.
 * Cuts every tensor into chunks of chunk_elems elements and uploads the chunk
 * table (tensor id, offset, length) once.  Synchronous; not capturable.
 * Errors: INVALID_ARG (n_tensors < 1, a negative size, total > 2^62 elements,
 * more than 2^30 chunks, bad opts), UNSUPPORTED_DTYPE, CUDA, OOM. */
LAMB_API lamb_status_t lamb_plan_create(const int64_t* sizes, int32_t n_tensors,
                               const uint8_t* decay_mask, int32_t grad_dtype,
                               int32_t copy_dtype, int32_t device,
                               const lamb_plan_options_t* opts,
                               lamb_plan_t* out);

/* Bind the tensors' device pointers (host arrays of n_tensors pointers).
 * w, g, m are required; v is required by lamb_step only (NULL for a
 * LARS-only plan); w_copy is required iff the plan has a bf16 copy.  A
 * pointer may be NULL only for a 0-element tensor.  Records per tensor
 * whether every array is aligned for 128-bit access.  Uploads the pointer
 * table on `stream` and synchronises it; not capturable.  Re-binding is
 * allowed between steps. */
LAMB_API lamb_status_t lamb_plan_bind(lamb_plan_t plan, void* const* w,
                             const void* const* g, void* const* m,
                             void* const* v, void* const* w_copy,
                             cudaStream_t stream);

/* One LAMB step (Algorithm 2) over every tensor, enqueued on `stream`.
 *   d_step  DEVICE int64: t (>= 1 when bias correction is on).  Needed when
 *           LAMB_FLAG_BIAS_CORRECTION, LAMB_FLAG_INCREMENT_STEP or
 *           LAMB_FLAG_LR_SCHEDULE is set, else may be NULL (INVALID_ARG
 *           when it is NULL but needed).
 *   d_lr    DEVICE float: eta_t for this step (with LAMB_FLAG_LR_SCHEDULE:
 *           NULL, or where the step writes the eta_t it computed).
 * Updates w, m, v in place (and the bf16 copy); g is read only.  Writes the
 * per-tensor norms and trust ratios (lamb_plan_trust_ratios).  No host
 * synchronisation, allocation or pageable copy: capturable in a CUDA graph,
 * and replays of the graph read the current *d_step and *d_lr.
 * On an on-chip plan the step is one cooperative launch that holds every SM
 * and whose CTAs wait for each other's partial sums: do not run on-chip
 * steps of two plans at the same time on different streams (a wait that
 * cannot be met gives up after wait_limit_ms with LAMB_STATUS_WAIT_TIMEOUT
 * and leaves the plan unusable).  Steps of one plan, like all steps, must
 * not overlap either. */
LAMB_API lamb_status_t lamb_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                        int64_t* d_step, const float* d_lr,
                        cudaStream_t stream);

/* One LARS step (Algorithm 1 with trust coefficient kappa) over every
 * tensor.  Uses w, g, m (v is not touched).  beta1 is the momentum; the
 * momentum is damped by (1-beta1) as in Algorithm 1.  d_step is read only for
 * LAMB_FLAG_INCREMENT_STEP and LAMB_FLAG_LR_SCHEDULE (may be NULL otherwise).
 * Same capture and ownership rules as lamb_step. */
LAMB_API lamb_status_t lars_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                        int64_t* d_step, const float* d_lr,
                        cudaStream_t stream);

/* One N-LAMB step (appendix Algorithm 3: Nesterov momentum in the first
 * moment) or, with nesterov_second_moment = 1, one NN-LAMB step (Algorithm
 * 4: also in the second moment), over every tensor.  Uses w, g, m, v and
 * the two-pass kernels, or the on-chip kernel on an on-chip plan.
 *   hyper          beta1, beta2, eps, weight_decay, phi as for lamb_step;
 *                  the bias-correction flag is ignored (the Nesterov forms
 *                  carry their own corrections); INCREMENT_STEP honoured
 *   momentum_decay psi of the momentum schedule read from Algorithm 3's
 *                  inputs: mu_t = beta1 * (1 - 0.5 * 0.96^(t psi)) (Dozat's
 *                  Nadam schedule; psi = 0.004 is its usual value)
 *   d_step         DEVICE int64 t >= 1 (required)
 *   d_lr           DEVICE float eta_t
 *   d_mu_product   DEVICE double: prod_{i<t} mu_i on entry (1.0 before the
 *                  first step), replaced by prod_{i<=t} mu_i when the step
 *                  completes -- optimizer state, like m and v
 * With u = (mu_{t+1} m_t / (1 - prod_{i<=t+1} mu_i) + (1 - mu_t) g /
 * (1 - prod_{i<=t} mu_i)) / (sqrt(v_hat) + eps) + lambda_k w, v_hat =
 * v_t / (1 - beta2^t) (N-LAMB) or beta2 v_t / (1 - beta2^(t+1)) + (1 -
 * beta2) g^2 / (1 - beta2^t) (NN-LAMB), the update is w <- w - eta
 * phi(||w||)/||u|| u as in lamb_step.  Capturable like lamb_step. */
LAMB_API lamb_status_t nlamb_step(lamb_plan_t plan, const lamb_hyper_t* hyper,
                                  double momentum_decay,
                                  int32_t nesterov_second_moment,
                                  int64_t* d_step, const float* d_lr,
                                  double* d_mu_product, cudaStream_t stream);

/* DEVICE arrays [n_tensors] of the last step's trust ratio rho_k, ||w_k||
 * and ||r_k|| (LARS: ||m_k||), in double.  Owned by the plan; valid until
 * destroy; overwritten by the next step.  Any out pointer may be NULL. */
LAMB_API lamb_status_t lamb_plan_trust_ratios(lamb_plan_t plan, const double** d_ratio,
                                     const double** d_wnorm,
                                     const double** d_unorm);

/* DEVICE results of the last step's gradient check (LAMB_FLAG_GRAD_NORM or
 * LAMB_FLAG_SKIP_NONFINITE; the arrays keep their values across steps
 * without those flags):
 *   d_gnorm         [n_tensors] ||g_k|| in double (0 for 0-element tensors)
 *   d_gnorm_global  [1] sqrt(sum_k ||g_k||^2)
 *   d_nonfinite     [1] 1 if some element of g was Inf or NaN, else 0 (with
 *                   SKIP_NONFINITE: the step was skipped)
 * Owned by the plan, valid until destroy.  Any out pointer may be NULL.
 * A CUDA graph can read them on the device, e.g. to adapt a loss scale. */
LAMB_API lamb_status_t lamb_plan_grad_norms(lamb_plan_t plan,
                                            const double** d_gnorm,
                                            const double** d_gnorm_global,
                                            const uint32_t** d_nonfinite);

/* Copy the gradient-check results (as lamb_plan_grad_norms) into
 * caller-owned memory -- device or host, any pointer may be NULL: gnorm
 * [n_tensors] doubles, gnorm_global [1] double, nonfinite [1] uint32 --
 * with cudaMemcpyAsync on `stream`.  Does not synchronise. */
LAMB_API lamb_status_t lamb_plan_copy_grad_norms(lamb_plan_t plan,
                                                 double* gnorm,
                                                 double* gnorm_global,
                                                 uint32_t* nonfinite,
                                                 cudaStream_t stream);

/* Copy the last step's per-tensor results (as lamb_plan_trust_ratios) into
 * caller-owned arrays of n_tensors doubles -- device or host memory, any of
 * the three may be NULL -- with cudaMemcpyAsync on `stream` (kind inferred
 * from the addresses).  Does not synchronise; with device destinations it is
 * capturable. */
LAMB_API lamb_status_t lamb_plan_copy_trust_ratios(lamb_plan_t plan, double* ratio,
                                          double* wnorm, double* unorm,
                                          cudaStream_t stream);

/* Read (and optionally clear) the device status word (LAMB_STATUS_* bits).
 * Synchronises `stream`; not capturable. */
LAMB_API lamb_status_t lamb_plan_query(lamb_plan_t plan, uint32_t* status_bits,
                              int32_t clear, cudaStream_t stream);

LAMB_API lamb_status_t lamb_plan_get_info(lamb_plan_t plan, lamb_plan_info_t* info);

/* Instrumentation: when enabled, each step records CUDA events on its
 * stream around every kernel it launches (up to 4096 steps are kept).
 * lamb_plan_read_timing waits for those events, returns the number of steps
 * recorded and the summed device time of each kernel in milliseconds
 * (ms_per_kernel[0..n_kernels-1]; a two-pass step launches 2 kernels, an
 * on-chip step 1, or 3 when it streams tensors through the two-pass kernels
 * first; entries past the step's kernels are 0), and clears
 * the record. */
LAMB_API lamb_status_t lamb_plan_set_timing(lamb_plan_t plan, int32_t enable);
LAMB_API lamb_status_t lamb_plan_read_timing(lamb_plan_t plan, int32_t* n_steps,
                                    double* ms_per_kernel, int32_t n_kernels);

/* Frees everything the plan owns (synchronises the plan's device). */
LAMB_API lamb_status_t lamb_plan_destroy(lamb_plan_t plan);

/* Host-only planner, no device needed: the chunk table lamb_plan_create
 * would build.  Chunks hold chunk_elems elements (0 = 16384), except within
 * tail_elems of either end of the layout (the tensors laid end to end), where
 * they hold LAMB_TAIL_CHUNK_ELEMS; a chunk never spans two tensors.  A plan
 * uses the tail reported by lamb_plan_get_info.  Writes up to `capacity`
 * rows into the three host arrays (any may be NULL when capacity is 0) and
 * the total row count into *n_chunks.  capacity 0 only counts: LAMB_OK with
 * *n_chunks written.  INVALID_ARG on bad sizes, chunk_elems or tail_elems
 * (< 0, or > 0 with chunk_elems < LAMB_TAIL_CHUNK_ELEMS), or a capacity
 * above 0 that is too small (n_chunks is still written). */
LAMB_API lamb_status_t lamb_layout_chunks(const int64_t* sizes, int32_t n_tensors,
                                 int32_t chunk_elems, int64_t tail_elems,
                                 int32_t* chunk_tensor, int64_t* chunk_offset,
                                 int32_t* chunk_len, int32_t capacity,
                                 int32_t* n_chunks);

/* One LAMB step (the same two kernels, chunking and numerics as lamb_step on
 * a two-pass plan with the default 16384-element chunks and no tail: the
 * results are bitwise equal) for callers that may not allocate device
 * memory: code that runs under an allocator owning all GPU memory (a
 * framework's caching allocator or a fixed pool), code that must not pay the
 * device-wide synchronisation cudaMalloc/cudaFree can cause, or a plug-in
 * that is handed a stream and buffers but no right to allocate.  It needs no
 * plan: every table, partial sum and counter lives in one fixed 4 MiB device
 * array built into the library, which each GPU that uses it holds until the
 * process exits.  (The paper has no counterpart of this entry point; it is a
 * deployment convenience.)
 *
 *   sizes, decay_mask   host arrays [n_tensors] as in lamb_plan_create
 *                       (decay_mask may be NULL = all decayed)
 *   w, g, m, v, w_copy  host arrays [n_tensors] of DEVICE pointers as in
 *                       lamb_plan_bind; v is required; w_copy iff copy_dtype
 *                       is LAMB_BF16
 *   hyper, d_step, d_lr as in lamb_step (flags: BIAS_CORRECTION and
 *                       INCREMENT_STEP only)
 *   d_ratio             NULL or a DEVICE array [n_tensors] of doubles that
 *                       receives the trust ratios of this step
 * Limits: n_tensors <= 4096, no tensor above 2^31 elements and at most
 * 131072 chunks of 16384 elements in total (2^31 parameters); larger inputs
 * are rejected with LAMB_ERR_INVALID_ARG before any device work.  Calls no
 * cudaMalloc, cudaFree or other allocating routine.
 * The caller's host arrays (sizes, decay_mask and the five pointer arrays)
 * are copied into the device array with cudaMemcpyAsync on `stream`.  From
 * pageable memory those copies have read them when the call returns, so
 * they may be reused at once; from page-locked (pinned) memory a copy may
 * still be reading them after the call returns, so keep them unchanged until
 * `stream` has passed the call (e.g. synchronise it).  Under stream capture
 * the copies become graph nodes that read the same host arrays at every
 * replay, which must then stay valid and unchanged for the graph's life.
 * The first call on each device (the current device) looks up the array's
 * device address; with CUDA's lazy module loading (the default) that first
 * use also loads the library's kernels and reserves the 4 MiB there, so make
 * the first call before any stream capture and before a memory pool claims
 * all device memory (or load eagerly with CUDA_MODULE_LOADING=EAGER).  All
 * calls share the one array: calls that may overlap on the GPU (other
 * streams, other host threads) race and must be ordered by the caller.
 * Each call rebuilds the tables and clears the counters it needs, so it does
 * not depend on what the previous call left there.  Device-side conditions
 * (a step count < 1: the step is skipped; non-finite norms: NaN/Inf
 * propagate) behave as in lamb_step; there is no status query for this
 * entry point. */
LAMB_API lamb_status_t lamb_step_noalloc(
    const int64_t* sizes, int32_t n_tensors, const uint8_t* decay_mask,
    int32_t grad_dtype, int32_t copy_dtype, void* const* w,
    const void* const* g, void* const* m, void* const* v,
    void* const* w_copy, const lamb_hyper_t* hyper, int64_t* d_step,
    const float* d_lr, double* d_ratio, cudaStream_t stream);

/* Host-only planner, no device needed: the rounds of an on-chip plan
 * (LAMB_ALGO_ON_CHIP) with `grid` CTAs of rows_per_cta rows (1..224) each.
 * One output row per piece, in round order, then CTA order: its round, its
 * CTA, tensor, first element inside the tensor, element count, first row
 * inside the CTA's slice and row count; then one row per tensor too large
 * for a round (updated by the two-pass kernels), with round and CTA -1, the
 * whole tensor as its elements and 0 rows.
 * Writes up to `capacity` pieces (the output arrays may be NULL when
 * capacity is 0), the total into *n_pieces and the round count into
 * *n_rounds.  capacity 0 only counts: LAMB_OK with the counts written.
 * INVALID_ARG on bad input or a capacity above 0 that is too small (the
 * counts are still written).  lamb_plan_create uses the same planner with
 * the device's SM count (at most; at least 32 rows per CTA) and
 * shared-memory rows (lamb_plan_get_info reports both). */
LAMB_API lamb_status_t lamb_layout_rounds(
    const int64_t* sizes, int32_t n_tensors, int32_t grid,
    int32_t rows_per_cta, int32_t* piece_round, int32_t* piece_cta,
    int32_t* piece_tensor, int64_t* piece_offset, int64_t* piece_len,
    int32_t* piece_first_row, int32_t* piece_rows, int64_t capacity,
    int64_t* n_pieces, int32_t* n_rounds);

/* ---------------------------------------------------------------------------
 * Data-parallel (sharded) step.
 *
 * The step shards over chunk ranges: rank r of W updates only the chunks of
 * its range (lamb_layout_shard), with one exchange per step -- the per-chunk
 * sums of w^2 and u^2 (u = r + lambda_k w; LARS: m), 2 floats per chunk (165
 * KB for BERT-large), which every rank needs to form the trust ratios of
 * the tensors its range touches.  Per step, on each rank:
 *   lamb_shard_pass1   zeroes the plan's sums array, then reads g, m, v, w
 *                      of the rank's chunks, writes m, v and the chunks'
 *                      sums (Alg. 2 moment lines; Alg. 1 for LARS);
 *   (caller)           all-reduce (sum) of the float array lamb_plan_partials
 *                      returns, in place, across the ranks -- every entry
 *                      has one non-zero contributor, so the sum is exact and
 *                      every rank ends with the same array;
 *   lamb_shard_pass2   forms every tensor's norms and rho_k from the array
 *                      with the fixed-order combine of an unsharded step,
 *                      then updates w (and the bf16 copy) of the rank's
 *                      chunks; closes the step (INCREMENT_STEP, schedule,
 *                      N-LAMB product) like lamb_step.
 * The results on each rank's range, and the trust ratios, are bitwise equal
 * to one unsharded step of the same layout and tail.  The gradients of the
 * rank's range must be reduced (e.g. reduce-scattered) before pass 1, and
 * the new w gathered after pass 2, by the caller.  The kernels touch only
 * the rank's elements of w, g, m, v and the copy.  Not taken: GRAD_NORM,
 * SKIP_NONFINITE (INVALID_ARG).  Both halves are capturable; no timing
 * events are recorded for them.
 *   optimizer       LAMB_OPT_*; LARS uses trust_coef, the N-LAMB forms
 *                   momentum_decay and d_mu_product as in nlamb_step (both
 *                   halves take the same arguments)
 *   d_step, d_lr    as in lamb_step (N-LAMB: d_step required)
 * ------------------------------------------------------------------------- */
#define LAMB_OPT_LAMB 0
#define LAMB_OPT_LARS 1
#define LAMB_OPT_NLAMB 2
#define LAMB_OPT_NNLAMB 3

LAMB_API lamb_status_t lamb_shard_pass1(lamb_plan_t plan,
                                        const lamb_hyper_t* hyper,
                                        int32_t optimizer,
                                        double momentum_decay,
                                        int64_t* d_step, const float* d_lr,
                                        double* d_mu_product,
                                        cudaStream_t stream);
LAMB_API lamb_status_t lamb_shard_pass2(lamb_plan_t plan,
                                        const lamb_hyper_t* hyper,
                                        int32_t optimizer,
                                        double momentum_decay,
                                        int64_t* d_step, const float* d_lr,
                                        double* d_mu_product,
                                        cudaStream_t stream);

/* DEVICE float array of 2 x n_chunks values (per chunk: sum of w^2, sum of
 * u^2) that lamb_shard_pass1 writes and lamb_shard_pass2 reads; owned by the
 * plan, valid until destroy.  *n_floats receives 2 x n_chunks. */
LAMB_API lamb_status_t lamb_plan_partials(lamb_plan_t plan, float** d_partials,
                                          int64_t* n_floats);

/* Copies the sums array (2 x n_chunks floats, as lamb_plan_partials) out of
 * the plan into buf (to_plan = 0) or from buf into the plan (to_plan = 1),
 * with cudaMemcpyAsync on `stream`; buf is device or host memory.  For a
 * caller whose all-reduce wants its own buffer (e.g. a framework tensor):
 * copy out, all-reduce, copy back.  Capturable with a device buffer. */
LAMB_API lamb_status_t lamb_plan_copy_partials(lamb_plan_t plan, float* buf,
                                               int32_t to_plan,
                                               cudaStream_t stream);

/* Host-only: the chunk range [*chunk_begin, *chunk_end) of shard `rank` of
 * `world` for the chunk table lamb_layout_chunks(sizes, chunk_elems,
 * tail_elems) gives: the chunks whose first element, counted over the layout
 * (tensors laid end to end), lies in [floor(total rank / world),
 * floor(total (rank + 1) / world)), total being the layout's element count.
 * The ranges of ranks 0..world-1 are contiguous and cover every chunk once;
 * a range may be empty.  INVALID_ARG on bad input. */
LAMB_API lamb_status_t lamb_layout_shard(const int64_t* sizes,
                                         int32_t n_tensors,
                                         int32_t chunk_elems,
                                         int64_t tail_elems, int32_t world,
                                         int32_t rank, int64_t* chunk_begin,
                                         int64_t* chunk_end);

/* Message of the last failed call on this host thread ("" if none). */
LAMB_API const char* lamb_last_error(void);

/* LAMB_ABI_VERSION of the built library. */
LAMB_API int32_t lamb_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* LAMB_GB300_H */
