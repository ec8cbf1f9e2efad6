/*
 * isoloco.h -- C ABI of the GB300-native IsoLoCo / DiLoCo outer step.
 *
 * Method: "Can Model Merging Improve Aggregation in DiLoCo?" (arXiv 2607.03011).
 *   Alg. 1 (DiLoCo):  Delta = (1/R) sum_i (theta^{t-1} - theta_i^{t}); OuterOpt = SGD
 *                     with Nesterov momentum.
 *   Alg. 2 (IsoLoCo): mean pseudo-gradient; every 2-D tensor is replaced by its Iso-C
 *                     correction sigma_bar * U V^T (U S V^T = SVD(Delta),
 *                     sigma_bar = mean of the singular values); then
 *                     B <- mu B + Delta, P <- Delta + mu B, theta <- theta - eta_out P.
 *   Sec. 2.2, Eq. 1:  task-arithmetic merging theta_0 + lambda sum_t tau_t; Iso-C sums
 *                     the task matrices and flattens their spectrum.
 *
 * The polar factor U V^T is computed without an SVD: a batched Newton-Schulz-type
 * iteration X <- X (a I + b X^T X + c (X^T X)^2) on tcgen05 tensor cores (Sec. 4.3
 * uses Newton-Schulz for the same purpose), and sigma_bar = tr(Q^T Delta) / min(m, n),
 * which equals the mean singular value exactly when Q is the polar factor.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All tensors live in ONE flat fp32 buffer per role (theta, momentum, output),
 *   described by a parameter table; parameter p occupies elements
 *   [offset, offset + rows * max(cols, 1)).  cols == 0 marks a 1-D tensor of
 *   `rows` elements; every other entry is a row-major rows x cols matrix.
 * - Worker replicas are K more flat buffers of the same layout, fp32 or bf16,
 *   passed as a HOST array of K DEVICE pointers.  They are only read.
 * - Pointers are device pointers, 16-byte aligned, unless the name says host.
 *   The caller owns them; the library never frees or keeps them past a call.
 * - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls enqueue work
 *   and return without waiting, unless opts->sync is set.  A plan's workspace is
 *   used by one call at a time: calls on the same plan from different streams
 *   must be ordered by the caller.
 * - Return values are isoloco_status_t codes.  No C++ exception crosses the ABI.
 *   isoloco_last_error() gives a thread-local message for the last failure.
 * - Sign convention (Alg. 1/2): Delta_k = theta - theta_k, and theta moves by
 *   -eta_out * P.  iso_c_merge uses task vectors tau_k = theta_k - theta_base.
 */
#ifndef ISOLOCO_H_
#define ISOLOCO_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct isoloco_plan* isoloco_plan_t;

/* One tensor of the parameter table (see conventions above). */
typedef struct {
    int64_t offset;
    int32_t rows;
    int32_t cols;
} isoloco_param_t;

/* Element type of the worker replicas (bf16 is upcast exactly to fp32). */
typedef enum { ISOLOCO_F32 = 0, ISOLOCO_BF16 = 1 } isoloco_dtype_t;

typedef enum {
    ISOLOCO_OK = 0,
    ISOLOCO_ERR_INVALID = -1,       /* bad argument, table or plan; nothing launched */
    ISOLOCO_ERR_ALIGN = -2,         /* a pointer is not 16-byte aligned; nothing launched */
    ISOLOCO_ERR_NONFINITE = -3,     /* NaN/Inf in the pseudo-gradient: theta, B untouched */
    ISOLOCO_ERR_NOT_CONVERGED = -4, /* a polar iteration hit max_iter (update still applied) */
    ISOLOCO_ERR_CUDA = -5,          /* a CUDA runtime call failed */
    ISOLOCO_ERR_OOM = -6,           /* workspace allocation failed */
    ISOLOCO_ERR_TIMEOUT = -7,       /* a device-side wait gave up (kernel returned early) */
    ISOLOCO_ERR_GUARD = -8          /* isoloco_check_guards: a workspace guard byte was overwritten */
} isoloco_status_t;

/* Options of one outer step (Alg. 2's hyperparameters plus solver controls). */
typedef struct {
    float alpha;      /* Iso-C scale (Eq. 1's lambda); multiplies the 2-D output only. */
    float outer_lr;   /* eta_out of Alg. 2. */
    float momentum;   /* mu of Alg. 2 (0 = plain SGD outer step, Eq. 2). */
    int reduce_mean;  /* 1: Delta is the mean over workers (Alg. 1/2); 0: the sum. */
    int max_iter;     /* cap on quintic polar steps per matrix; <= 0 selects 28. */
    float tol;        /* convergence test ||X^T X - I||_F / sqrt(n) < tol; <= 0 selects 4e-3. */
    int sync;         /* 1: synchronize `stream` and return the step's device status. */
    int fast_steps;   /* 0: exact Iso-C (polar factor to convergence, sigma_bar = tr(Q^T Delta) / r).
                       * k in 1..64: the fast variant of Sec. 4.3 -- exactly k quintic steps of
                       * the standard schedule from X_0 = Delta / ||Delta^T Delta||_F^(1/2) (steps
                       * after its seventh repeat the seventh), no convergence test and no
                       * polish, and sigma_bar = ||Delta||_F / sqrt(r) (the RMS of the singular
                       * values); the paper runs 5. */
    /* The ablations of Sec. 4.5 and App. B (all 0 by default = Alg. 2): */
    int orth_target;   /* 0: Iso-C of Delta.  1: of the momentum update instead: B <- mu B + Delta,
                        * P <- Delta + mu B (or P <- B with standard momentum), then
                        * theta <- theta - eta * Iso(P) for 2-D tensors and theta - eta * P for
                        * 1-D ones (sigma_bar = tr(Q^T P) / r). */
    int momentum_kind; /* 0: Nesterov (Alg. 2).  1: standard momentum, B <- mu B + U and
                        * theta <- theta - eta B. */
    int scale_kind;    /* 0: the Iso-C scale sigma_bar.  1: Muon's spectral scale, U = alpha *
                        * sqrt(rows / cols) * Q for a rows x cols tensor (App. B; sigma_bar is
                        * then not computed). */
    /* The merging aggregators of Sec. 3.2, used by diloco_outer_step in place of the mean
     * of the Delta_k (the outer optimiser stays Nesterov; momentum = 0 is the paper's SGD): */
    int aggregator;    /* 0: mean (Alg. 1).
                        * 1: TIES -- trim: each worker keeps its n_keep = N - floor(sparsity * N)
                        *    largest |Delta_k| over all N entries (entries equal to the
                        *    n_keep-th largest are kept too); elect: sign of P + N, P and N the
                        *    fp32 sums, in worker order, of an entry's kept positive and kept
                        *    negative values; merge: U = the mean of the kept values of the
                        *    elected sign (0 when P + N = 0).
                        * 2: DARE -- drop each entry of each Delta_k with probability
                        *    `sparsity`, rescale the rest by 1 / (1 - sparsity), and average
                        *    (or sum, reduce_mean = 0). */
    float sparsity;    /* in [0, 1) */
    unsigned int seed; /* DARE's drops: entry i (flat index) of worker k is dropped when
                        * u < sparsity, u = top 24 bits of SplitMix64 output number
                        * k * n_total + i + 1 from state `seed` (Steele, Lea and Flood 2014),
                        * times 2^-24. */
    int spectrum_kind; /* isoloco_outer_step's spectrum map (Sec. 4.5): 0: Iso-C, every
                        * singular value set to sigma_bar (Alg. 2).  1: clip_high, only the
                        * singular values above sigma_bar set to it, U = alpha * U_D
                        * diag(min(s_i, sigma_bar)) V_D^T.  2: clip_low, only those below,
                        * max(s_i, sigma_bar).  1 and 2 need fast_steps = 0 and scale_kind = 0;
                        * their first call allocates an auxiliary plan (the n x n matrices
                        * H - sigma_bar I, H = Q^T Delta) and its buffers.  3: Iso-C from the
                        * singular values (Alg. 2's SVD form): every sigma_i of every matrix is
                        * computed, as the eigenvalues of H = Q^T Delta (Delta Q^T when wide;
                        * Householder tridiagonalization in fp32 and bisection), sigma_bar is
                        * their mean, and U = alpha sigma_bar Q as for 0 (the polar iteration
                        * then runs three passes at every step, as for 1 and 2, so that Q's
                        * singular values are 1 to ~1e-6); the sigma_i are read
                        * with isoloco_read_singular_values.  Its first call allocates the
                        * n x n fp32 H of every matrix; the reduction is BLAS-2 bound (about
                        * n^3 / 3 fp32 elements read and written per matrix). */
    int full_precision; /* 0: the polar steps after the first keep one GEMM operand at 11 bits
                         * (two 16-bit passes; its rounding only perturbs the spectrum of a
                         * full-rank iterate, which later steps correct).  1: every step splits
                         * both operands (three passes, ~22 bits each; ~1.5x the GEMM work).
                         * For an exactly rank-deficient Delta (Iso-C's partial isometry
                         * U_rho V_rho^T) whose zero directions are not whole rows of a wide or
                         * whole columns of a tall matrix (e.g. many zero rows of a tall or
                         * square one), the 11-bit operand turns the iterate's row space toward
                         * the zero directions by ~2^-11 per step; 1 keeps the result within
                         * the Iso-C tolerance there. */
    long long precision_schedule; /* which quintic polar steps run a single 16-bit pass instead of
                         * two (full_precision = 0 only).  0: the library's default schedule;
                         * -1: none.  Otherwise eight 5-bit step indices, field i at bits
                         * 5i .. 5i + 4: [f0, f1) the steps whose Gram and polynomial GEMMs and
                         * [f2, f3) those whose update runs one pass, for the standard schedule
                         * (rectangular matrices); f4 .. f7 the same for the deep schedule
                         * (near-square ones).  Step k is the matrix's k-th quintic step
                         * (0-based); the polish and iteration 0's GEMMs keep their passes. */
} isoloco_opts_t;

/* Fills *opts with alpha = 1, outer_lr = 0.7, momentum = 0.9 (the paper's DiLoCo
 * optimum at R = 8, App. A Table 6), reduce_mean = 1, default solver controls. */
int isoloco_opts_default(isoloco_opts_t* opts);

/* Creates a plan for a parameter table.
 *   table[n_params]: copied; tensors must lie inside [0, n_total) and not overlap.
 *   K: number of worker replicas (1..64).  replica_dtype: their element type.
 * Allocates the device workspace (Delta, polar iterates, Gram and polynomial
 * buffers, per-matrix state) on the current device, and builds the TMA
 * descriptors.  Returns OK, INVALID, OOM or CUDA; *plan is NULL on failure. */
int isoloco_plan_create(isoloco_plan_t* plan, const isoloco_param_t* table, int n_params,
                        int64_t n_total, int K, isoloco_dtype_t replica_dtype);

/* Frees the plan and its workspace (synchronizes the device first). */
void isoloco_plan_destroy(isoloco_plan_t plan);

/* Device bytes held by the plan's workspace. */
int64_t isoloco_plan_workspace_bytes(isoloco_plan_t plan);

/* IsoLoCo outer step, Alg. 2.
 *   theta[n_total], momentum[n_total]: fp32, read and overwritten in place.
 *   replicas: host array of K device pointers (the plan's dtype), read only.
 *   update_out: nullable fp32 [n_total]; if given, receives the update direction
 *     U (alpha * sigma_bar * Q for 2-D tensors, the mean Delta for 1-D ones).
 * On a non-finite pseudo-gradient nothing is written and the step's status is
 * NONFINITE.  Asynchronous unless opts->sync. */
int isoloco_outer_step(isoloco_plan_t plan, float* theta, float* momentum,
                       const void* const* replicas, const isoloco_opts_t* opts, void* stream,
                       float* update_out);

/* Same step with every buffer in HOST memory: the result lands in theta_host and
 * momentum_host, and the call synchronizes `stream` before returning the step's status.
 * When theta, momentum and every replica are page-locked memory registered with CUDA
 * (cudaHostAlloc, cudaHostRegister, torch's pin_memory; 16-byte aligned), the reduce pass
 * reads them in place over the host link and theta / momentum are copied to plan-owned
 * device buffers on a plan-owned side stream while the polar iteration runs; otherwise all
 * of them are first copied to plan-owned device buffers on `stream`.  Either way theta and
 * momentum are copied back at the end.  The first call allocates the device buffers (and
 * the side stream). */
int isoloco_outer_step_host(isoloco_plan_t plan, float* theta_host, float* momentum_host,
                            const void* const* replicas_host, const isoloco_opts_t* opts,
                            void* stream);

/* DiLoCo outer step, Alg. 1 with Nesterov SGD: one streaming pass over every
 * parameter (no Iso-C).  Elementwise, so a non-finite input only affects its own
 * element; the step's status reports it.  opts->aggregator selects the merging rule of
 * Sec. 3.2 that replaces the mean (TIES: one extra read pass over the replicas for the
 * trim, four if the sampled bracket of its threshold misses, then one pass; DARE: one
 * pass); TIES's first call allocates its trim buffers (~K x 4 MB of samples and candidate
 * segments sized from n_total).  The table is not used: every entry of
 * [0, n_total) is updated.  Errors: INVALID for a bad aggregator or sparsity. */
int diloco_outer_step(isoloco_plan_t plan, float* theta, float* momentum,
                      const void* const* replicas, const isoloco_opts_t* opts, void* stream);

/* Iso-C model merging (Sec. 2.2, Eq. 1 form): tau_k = experts_k - theta_base,
 * T = sum_k tau_k;  out = theta_base + alpha * IsoC(T) for 2-D tensors and
 * out = theta_base + alpha * T for 1-D tensors.  out[n_total] fp32 may alias
 * nothing else.  The plan's K is the number of experts. */
int iso_c_merge(isoloco_plan_t plan, const float* theta_base, const void* const* experts,
                float alpha, float* out, void* stream);

/* Synchronizes `stream` and returns the device status of the plan's last call. */
int isoloco_last_status(isoloco_plan_t plan, void* stream);

/* Per-matrix diagnostics of the last call, in table order over the 2-D tensors
 * only (n_matrices entries each; any pointer may be NULL).  Synchronizes `stream`.
 *   sigma_bar: tr(Q^T Delta) / min(m, n);  iters: polar iterations used;
 *   status: 0 or NOT_CONVERGED;  residual: last ||X^T X - I||_F / sqrt(n). */
/* Bounds check of the plan's device workspace (no counterpart in the paper; it stands in
 * for a memory checker).  Every workspace region the plan (and its auxiliary plan) owns
 * sits between 256 guard bytes before it and its padding plus 256 guard bytes after it,
 * filled with 0xA5 when allocated; this synchronizes `stream` and compares them.  Returns OK,
 * GUARD (the message names the region, the side and the distance) or CUDA. */
int isoloco_check_guards(isoloco_plan_t plan, void* stream);

/* Test support for isoloco_check_guards: sets the guard byte right before (after = 0) or
 * right after (after = 1) workspace region `region` of the plan to a value other than the
 * fill, with cudaMemset inside the region's own allocation.  Returns OK or INVALID. */
int isoloco_debug_touch_guard(isoloco_plan_t plan, int region, int after);

/* Singular values of 2-D tensor `matrix` (table order over the 2-D tensors) from the
 * plan's last call with spectrum_kind = 3 (Alg. 2: Delta = U S V^T; here sigma_i of the
 * reduced pseudo-gradient), in descending order, copied to host memory out[0 .. r-1],
 * r = min(rows, cols) <= capacity.  Synchronizes `stream`.  Returns r, or INVALID (no such
 * call yet, bad index, buffer too small) or CUDA.  A zero pseudo-gradient gives zeros. */
int isoloco_read_singular_values(isoloco_plan_t plan, void* stream, int matrix, float* out_host,
                                 int capacity);

int isoloco_read_diag(isoloco_plan_t plan, void* stream, float* sigma_bar_host,
                      int32_t* iters_host, int32_t* status_host, float* residual_host);

/* Number of 2-D tensors in the plan's table. */
int isoloco_plan_num_matrices(isoloco_plan_t plan);

/* Batched split-precision GEMM of the polar iteration, exposed for testing:
 *   D[b] = op(A[b]) op(B[b]) with fp32 inputs rounded to 16-bit hi + lo planes and
 *   tcgen05 passes accumulated in fp32 in tensor memory.
 *   precision 0: bf16 planes, A and B split (hi*hi + hi*lo + lo*hi, 3 passes);
 *             1: fp16 planes, A split, B single (hi*hi + lo*hi, 2 passes);
 *             2: fp16 planes, A single, B split (2 passes);
 *             3: fp16 planes, both split (3 passes).
 *   a_mn_major = 0: A[b] is row-major M x K;  1: A[b] is row-major K x M.
 *   b_mn_major = 0: B[b] is row-major N x K;  1: B[b] is row-major K x N.
 *   D[b] is row-major M x N fp32:  D[b][i][j] = sum_k A(i,k) B(j,k).
 * All pointers are device fp32, contiguous per batch.  Allocates scratch with
 * cudaMalloc and synchronizes `stream` before returning. */
int isoloco_debug_gemm(int a_mn_major, int b_mn_major, int precision, int batch, int M, int N,
                       int K, const float* A, const float* B, float* D, void* stream);

/* The same GEMM as isoloco_debug_gemm (same arguments, same kernels, bitwise the
 * same D), for callers that must not allocate device memory.  The paper has no
 * counterpart: this is a library service, not part of the method.
 *
 * Who needs it: a caller whose process has handed the device's free memory to
 * another allocator (a training framework's caching pool that reserved the HBM
 * up front), so that a cudaMalloc here would fail or force that pool to give
 * memory back; and a caller in the middle of an overlapped step, where the
 * implicit device-wide synchronization of cudaMalloc / cudaFree would stall the
 * work queued on its other streams.  This entry point calls neither, nor any
 * other allocating routine: its scratch (the hi/lo operand planes, the four
 * tensor maps, an error word and a tile counter) lives in one static device
 * array of the library, 16 MiB per device, held by every GPU that loads the
 * library until the process exits.
 *
 * Set-up: the first call on a device (with that device current) looks up the
 * array's device address with cudaGetSymbolAddress and keeps it for later
 * calls; a failure there returns ISOLOCO_ERR_CUDA.  Make that first call on each
 * device before any stream capture begins.
 *
 * Limit: 1024 + 2 * R(2 * batch * a_rows * round8(a_cols))
 *             + 2 * R(2 * batch * b_rows * round8(b_cols)) <= 16 MiB,
 * with (a_rows, a_cols) = (K, M) if a_mn_major else (M, K), likewise B with N,
 * and R() rounding up to 256 bytes.  E.g. batch 1, M = N = K = 1024 fits;
 * M = N = K = 2048 does not.  Larger operands return ISOLOCO_ERR_INVALID with a
 * message giving the bytes needed, before anything is launched.
 *
 * Every call on a device shares that one array.  The call zeroes the error word
 * and the tile counter on `stream` before its kernels and synchronizes `stream`
 * before returning, so calls made one after another are safe.  Calls whose GPU
 * work can overlap (from several host threads, or on streams that are not
 * ordered with one another) race on the shared scratch and give wrong results;
 * such callers must serialize them. */
int isoloco_debug_gemm_noalloc(int a_mn_major, int b_mn_major, int precision, int batch, int M,
                               int N, int K, const float* A, const float* B, float* D,
                               void* stream);

/* Test of the timeout path of the pipelined kernels (no counterpart in the paper): one
 * thread waits, with the bounded mbarrier wait every pipeline stage of the GEMM uses, on a
 * barrier that nothing arrives on, and gives up after limit_ns nanoseconds of the GPU's
 * global timer, as a kernel whose wait runs out does (it raises the TIMEOUT flag and
 * returns; the context stays usable).  limit_ns must lie in 1e6 .. 1e9 (1 ms .. 1 s), else
 * ISOLOCO_ERR_INVALID before any launch.  Returns ISOLOCO_ERR_TIMEOUT when the wait gave up
 * (the expected outcome), ISOLOCO_OK if the barrier completed.  elapsed_ns (may be NULL)
 * receives how long the wait took.  Allocates 12 bytes of scratch and synchronizes `stream`. */
int isoloco_debug_wait_timeout(int64_t limit_ns, int64_t* elapsed_ns, void* stream);

/* Phases of the launch sequence, for isoloco_profile_read. */
enum {
    ISOLOCO_PHASE_REDUCE = 0,   /* pseudo-gradient reduction (HBM stream) */
    ISOLOCO_PHASE_GRAM = 1,     /* X^T X (or X X^T) split-precision tcgen05 GEMMs */
    ISOLOCO_PHASE_FINALIZE = 2, /* split-K sum of the Gram, convergence partials */
    ISOLOCO_PHASE_CONTROL = 3,  /* per-matrix schedule / convergence decisions */
    ISOLOCO_PHASE_POLY = 4,     /* G^2 GEMMs with the P = a I + b G + c G^2 epilogue */
    ISOLOCO_PHASE_UPDATE = 5,   /* X P (or P X) GEMMs */
    ISOLOCO_PHASE_TRACE = 6,    /* sigma_bar = tr(Q^T Delta) / n */
    ISOLOCO_PHASE_APPLY = 7,    /* Nesterov update / merge output (HBM stream) */
    ISOLOCO_PHASE_DILOCO = 8,   /* fused DiLoCo pass (mean, DARE, or TIES's merge pass) */
    ISOLOCO_PHASE_OTHER = 9,
    ISOLOCO_PHASE_TRIM = 10,    /* TIES trim: per-worker radix select of the threshold */
    ISOLOCO_PHASE_CLIP = 11,    /* clip_high / clip_low: H, sign(H / sigma_bar - I), P A' P, Q S' */
    ISOLOCO_NUM_PHASES = 12
};

/* Per-phase timing.  enable != 0 makes every later call record a CUDA event pair
 * around each phase's launches on the call's stream (a few microseconds of
 * overhead per launch); enabling or disabling resets the accumulators and
 * synchronizes the device.  Launch counts accumulate whether or not timing is on. */
int isoloco_profile_enable(isoloco_plan_t plan, int enable);

/* Synchronizes `stream`, then writes the accumulated milliseconds and launch
 * counts of the first `nphases` phases (either array may be NULL). */
int isoloco_profile_read(isoloco_plan_t plan, void* stream, double* ms_host, int64_t* launches_host,
                         int nphases);

/* Kernels launched by the plan since its creation. */
int64_t isoloco_plan_launches(isoloco_plan_t plan);

/* Thread-local message describing the last error returned on this thread. */
const char* isoloco_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* ISOLOCO_H_ */
