/*
 * slorr.h -- C ABI of libslorr, the GB300 (sm_103a) implementation of the SLORR
 * regularizer hot path (SLORR: Simple and Efficient In-Training Low-Rank
 * Regularization, arXiv 2607.08754).
 *
 * For every regularized weight matrix W_i (row-major m_i x n_i; conv kernels in
 * the (C_out, C_in*k*k) view of App. D.1) one call computes, on the caller's
 * stream, the SVD-free forward value and weight gradient of
 *
 *   SLORR-Hoyer  L = sum_i ||W_i||_*^2 / ||W_i||_F^2      (Sec. 3, Eq. 1)
 *   SLORR-Nuc    L = sum_i ||W_i||_*                      (Sec. 3, Eq. 1)
 *
 * with U V^T replaced by the Polar Express approximation P_hat (Sec. 3
 * "Computing the polar factor"): X_0 = W / (||W||_F + eps) on the Gram side
 * (X = W^T when m > n), then T steps of A = X X^T, B = b_t A + c_t A^2,
 * X <- a_t X + B X; n_hat = sum(W * P_hat) (Sec. 3 "Computing the nuclear and
 * Frobenius norms"); value and gradient as in Listing 1:
 *   frob = ||W||_F + eps, reg = n_hat / frob,
 *   Hoyer: L_i = reg^2,  G_i = 2 reg (P_hat / frob - n_hat / frob^3 W)
 *   Nuc:   L_i = n_hat,  G_i = P_hat
 * and the memory-efficient accumulation of Alg. 2 (App. C.3):
 *   W_i.grad += lambda * grad_scale * G_i,   loss = lambda * sum_i L_i.
 *
 * Memory: the caller owns every device buffer (weights, grads, outputs and one
 * workspace); the library allocates no device memory.  The handle owns only
 * host memory (the plan and the coefficient table).
 *
 * Errors: host-detectable problems (bad arguments, misalignment, a workspace
 * that is too small) return a non-zero status before anything is launched.
 * Problems found on the device (a non-finite norm or estimate, an internal
 * wait that ran out of time) are recorded in a status word inside the
 * workspace; slorr_get_status() reads it.  A matrix whose norm or estimate is
 * not finite leaves its gradient untouched.
 */
#ifndef SLORR_H
#define SLORR_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SLORR_API __attribute__((visibility("default")))
#else
#define SLORR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum slorr_status {
    SLORR_OK = 0,
    SLORR_ERR_INVALID_ARG = 1,   /* null / misaligned pointer, bad shape or option   */
    SLORR_ERR_UNSUPPORTED = 2,   /* valid request this build or device cannot serve */
    SLORR_ERR_CUDA = 3,          /* a CUDA runtime call failed                        */
    SLORR_ERR_WORKSPACE = 4,     /* workspace missing or smaller than required        */
    SLORR_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up (status word)  */
    SLORR_ERR_NONFINITE = 6      /* non-finite norm or nuclear estimate (status word) */
} slorr_status;

typedef enum slorr_variant {
    SLORR_HOYER = 0,             /* squared l1/l2 ratio of singular values (Sec. 3)  */
    SLORR_NUCLEAR = 1            /* nuclear norm (Sec. 3)                            */
} slorr_variant;

typedef enum slorr_dtype {       /* storage type of the weights and of their grads   */
    SLORR_F32 = 0,
    SLORR_BF16 = 1
} slorr_dtype;

typedef enum slorr_compute {     /* operand type of the Polar Express matrix products */
    SLORR_COMPUTE_FP16 = 0,      /* fp16 operands, fp32 accumulation (tensor cores)  */
    SLORR_COMPUTE_BF16 = 1,      /* bf16 operands, fp32 accumulation (tensor cores)  */
    SLORR_COMPUTE_FP32 = 2,      /* fp32 operands: three tf32 tensor-core products per
                                    product, short-K fp32 accumulations added with
                                    compensated sums (CUDA cores, compensated dot
                                    products, with SLORR_FLAG_SIMT_GEMM)              */
    SLORR_COMPUTE_BF16_SPLIT = 3 /* bf16 operands (App. C.1) with every product
                                    operand -- the iterate X_t (X_0 included), A
                                    and M -- carried as a bf16 pair hi = bf16(v),
                                    lo = bf16(v - hi), and every product as three
                                    bf16 tensor-core products (hi hi + lo hi +
                                    hi lo, fp32 accumulation); the Poly's b A term
                                    takes hi + lo; X_T is stored in fp16 for the
                                    n_hat and gradient passes.  Three times the
                                    tensor-core work of SLORR_COMPUTE_BF16, at the
                                    bf16 rate; gradient errors of about 1e-3 against
                                    the fp64 approximation, where plain bf16
                                    operands lose up to 4e-2 on the Hoyer gradient.
                                    Tensor cores only, per-phase launches:
                                    SLORR_FLAG_SIMT_GEMM, SLORR_FLAG_SEPARATE_NORM
                                    and SLORR_FLAG_DATAFLOW are rejected              */
} slorr_compute;

typedef struct slorr_shape {
    int64_t m;                   /* rows    (C_out for a conv kernel)                */
    int64_t n;                   /* columns (C_in*k_h*k_w for a conv kernel)          */
} slorr_shape;

typedef struct slorr_options {
    int32_t variant;             /* slorr_variant                        (HOYER)     */
    int32_t compute;             /* slorr_compute                        (FP16)      */
    int32_t dtype;               /* slorr_dtype of weights and grads     (F32)       */
    int32_t iters;               /* T, Polar Express steps, 1..16        (6)         */
    double  ell;                 /* lower singular-value bound ell, (0,1) (1e-3)     */
    double  cushion;             /* cushion ratio; < 0: derived default, 0: off (-1) */
    double  safety;              /* safety factor s >= 1; 1: off          (1.01)     */
    float   lambda;              /* regularization strength lambda       (1)         */
    float   eps;                 /* eps added to ||W||_F, >= 0            (1e-7)      */
    float   grad_scale;          /* extra factor on the gradient only    (1)         */
    int32_t flags;               /* SLORR_FLAG_* bits                     (0)         */
    double  timeout_s;           /* budget of each bounded device wait, s (2.0)      */
} slorr_options;

/* Flags.  slorr_create rejects any other bit with SLORR_ERR_INVALID_ARG. */
#define SLORR_FLAG_SIMT_GEMM    1   /* run the products on CUDA cores (a checker)      */
#define SLORR_FLAG_TEST_STALL  16   /* test only: every tensor-core CTA first waits on a
                                       barrier nothing arrives on, so its bounded wait
                                       runs out after timeout_s and the call reports
                                       SLORR_ERR_TIMEOUT (failure-detection test)     */
#define SLORR_FLAG_WRITE_GRAD  32   /* grads[i] = lambda * grad_scale * G_i instead of +=:
                                       the pre-update gradient of the decoupled variant
                                       (Alg. 1, App. C.2), applied by the caller as
                                       W -= lr * grads[i] after its optimizer step      */
#define SLORR_FLAG_NO_PDL      512  /* launch every kernel after the previous one completes.
                                       By default the memory passes and the CTA-pair
                                       kernel are programmatic dependents of the kernel
                                       before them, so each one's launch and prologue
                                       overlap the previous one's tail (tuning)          */
#define SLORR_FLAG_SEPARATE_NORM 1024 /* 16-bit iterates: take ||W||_F and write X_0 in two
                                       passes over W.  By default one pass does both:
                                       it stores W rounded to 16 bits and the first
                                       Gram and Update epilogues apply 1/(||W||_F+eps)
                                       (a matrix with max |w| > 2^15, or ||W||_F < 1 in
                                       fp16, is re-cast with the scale); tuning          */
#define SLORR_FLAG_NO_SPLIT_K  2048  /* never split the K range of a Gram tile across CTA
                                       pairs.  By default a set whose few Gram tiles have
                                       a long K (Q >> P, e.g. ResNet-18's 512 x 4608
                                       layers) splits each such tile into up to 2 parts
                                       whose fp32 partials are added, in part order, by
                                       the last part's epilogue (tuning)                */
#define SLORR_FLAG_GRAPH       4096  /* capture the launches of a forward/backward or
                                       descent call into a CUDA graph once and replay it
                                       while the workspace, loss_out, per_matrix_out, T
                                       and eta are unchanged (the weight and grad
                                       pointers may change: they are read from the
                                       workspace).  Ignored while timing is on; a stream
                                       that is being captured gets the launches.  Saves
                                       the launch gaps of small sets                    */
#define SLORR_FLAG_PHASE_LAUNCHES 16384 /* tensor-core GEMMs as 3 T launches, one per phase
                                       and step, each waiting for the previous one     */
#define SLORR_FLAG_DATAFLOW    32768 /* tensor-core GEMMs as one dataflow launch: every
                                       phase of every step, a matrix's Poly tiles
                                       starting as soon as that matrix's Gram tiles are
                                       stored, and so on, with no grid-wide barrier, so
                                       the phases of different matrices overlap.
                                       Without either flag the plan takes the dataflow
                                       launch for sets with enough independent work to
                                       overlap (no matrix's chain of phases longer than
                                       3/4 of the work per pair) whose per-phase
                                       launches would be short (fewer than 7 Gram tiles
                                       per CTA pair): measured faster there (fewer
                                       launch tails); per-phase launches otherwise
                                       (measured faster: lighter epilogues).
                                       Both give the same results bit for bit; the two
                                       flags exclude each other                         */

/* Fill *opt with the defaults listed beside each field above (App. C.1: T = 6,
 * ell = 1e-3, degree 5; eps, lambda and grad_scale as in Listing 1 / Alg. 2). */
SLORR_API void slorr_default_options(slorr_options* opt);

typedef struct slorr_handle slorr_handle;

/* Plan one weight set (Sec. 3; Alg. 2).  shapes: host array of `count` shapes,
 * copied.  opt: host struct, copied (NULL = defaults).  Builds the Polar Express
 * coefficient table (Sec. 3, App. C.1) and the tile schedule on the host; makes
 * no CUDA call.  Returns INVALID_ARG for count < 1, a non-positive dimension, a
 * dimension above 65536, or an option outside its range. */
SLORR_API slorr_status slorr_create(slorr_handle** out, const slorr_shape* shapes, int32_t count,
                          const slorr_options* opt);

/* Bytes of device workspace a call needs (host-only; no CUDA call). */
SLORR_API slorr_status slorr_workspace_size(const slorr_handle* h, size_t* bytes);

/* One regularizer forward + backward over the whole weight set (Listing 1,
 * Alg. 2), enqueued on `stream` (a cudaStream_t; NULL = legacy default stream).
 *   weights[i]      device pointer to W_i, row-major m_i x n_i, 16-byte aligned
 *   grads[i]        device pointer to W_i.grad, same layout; ACCUMULATED (+=)
 *   loss_out        device pointer to 1 float, written with lambda * sum_i L_i
 *   per_matrix_out  device pointer to `count` floats (unweighted L_i), or NULL
 *   workspace       device buffer of at least slorr_workspace_size() bytes,
 *                   256-byte aligned; it keeps a plan written on its first use,
 *                   so do not modify it between calls (pass another buffer, or
 *                   call slorr_reset_workspace(), to re-plan)
 * weights/grads are host arrays of `count` device pointers.  The call is
 * asynchronous; the grads must not alias the weights. */
SLORR_API slorr_status slorr_reg_forward_backward(slorr_handle* h, const void* const* weights,
                                        void* const* grads, float* loss_out,
                                        float* per_matrix_out, void* workspace,
                                        size_t workspace_bytes, void* stream);

/* One regularizer-only gradient descent step, in place, over the whole weight
 * set:  W_i <- W_i - eta * lambda * grad_scale * G_i(W_i),  with G_i the same
 * Polar Express gradient slorr_reg_forward_backward produces (Eq. 1).  It is the
 * last line of Alg. 1 (App. C.2, decoupled SLORR: W -= eta lambda G_pre) with
 * no task update in between, i.e. the "regularizer-only gradient step" of
 * Props. 2 and 3 (Sec. 3.1).  The gradient pass reads each W_i once and writes
 * it back; no grad buffer is involved, and SLORR_FLAG_WRITE_GRAD is ignored.
 *   weights[i]      device pointer to W_i, row-major m_i x n_i, 16-byte
 *                   aligned; READ AND OVERWRITTEN
 *   eta             step size (finite; eta * lambda * grad_scale must be finite)
 *   loss_out        device pointer to 1 float: lambda * sum_i L_i at the
 *                   weights BEFORE the step
 *   per_matrix_out, workspace, workspace_bytes, stream: as for
 *                   slorr_reg_forward_backward
 * A matrix whose norm or estimate is non-finite is left unchanged and the
 * status word records SLORR_ERR_NONFINITE.  Asynchronous. */
SLORR_API slorr_status slorr_reg_descent_step(slorr_handle* h, void* const* weights, float eta,
                                    float* loss_out, float* per_matrix_out, void* workspace,
                                    size_t workspace_bytes, void* stream);

/* Forget which workspace holds the plan; the next call re-writes it. */
SLORR_API slorr_status slorr_reset_workspace(slorr_handle* h);

/* Synchronize `stream`, read the device status word of `workspace`, clear it,
 * and return OK, TIMEOUT or NONFINITE (TIMEOUT wins if both were recorded). */
SLORR_API slorr_status slorr_get_status(slorr_handle* h, const void* workspace, void* stream);

/* Run only the Frobenius norm, the normalisation and the first `steps` Polar
 * Express steps (0 <= steps <= T) on `stream`, leaving the iterate X_steps in the
 * workspace (introspection for tests; Sec. 3 "Computing the polar factor"). */
SLORR_API slorr_status slorr_run_steps(slorr_handle* h, const void* const* weights, void* workspace,
                             size_t workspace_bytes, int32_t steps, void* stream);

/* Where matrix i's iterate after `after_steps` steps lives inside `workspace`:
 * an array in W's orientation -- rows x cols = m x n, row-major with leading
 * dimension ld >= n -- of element type elem (0 fp32, 1 fp16, 2 bf16).  The
 * Polar Express iterate X (P x Q, P = min(m,n)) is this array when m <= n and
 * its transpose when m > n (transposed = 1).  With SLORR_COMPUTE_BF16_SPLIT the
 * array holds the hi parts (bf16) before step T and X_T in fp16 after it.  Also
 * returns device pointers to ||W_i||_F^2 (double) and n_hat_i (double). */
typedef struct slorr_matrix_view {
    const void*   x;
    int64_t       rows, cols, ld;
    int32_t       elem;
    int32_t       transposed;
    const double* frob_sq;
    const double* n_hat;
    const float*  x0_scale;  /* X_0 = *x0_scale times the array at after_steps = 0
                                (16-bit iterates store W unscaled; else 1)    */
} slorr_matrix_view;
SLORR_API slorr_status slorr_iterate_view(const slorr_handle* h, const void* workspace, int32_t i,
                                int32_t after_steps, slorr_matrix_view* out);

/* The handle's (a_t, b_t, c_t) table, t = 1..T, as 3*T doubles (App. C.1). */
SLORR_API slorr_status slorr_get_coefficients(const slorr_handle* h, double* abc, int32_t capacity);

/* Polar Express schedule without a handle (host-only): greedy minimax odd
 * quintics on [l_t, u_t], l_{t+1} = p_t(l_t), u_{t+1} = 2 - l_{t+1}, with the
 * cushion and safety-factor options of slorr_options (Sec. 3, App. C.1).
 * Writes 3*iters doubles. */
SLORR_API slorr_status slorr_pe_coefficients(int32_t iters, double ell, double cushion, double safety,
                                   double* abc);

/* The derived cushion ratio kappa (minimax error 9/11 on [kappa, 1]). */
SLORR_API double slorr_cushion_ratio(void);

/* Algorithmic FLOPs of one call: T * sum_i (4 P_i^2 Q_i + 2 P_i^3) (Sec. 3
 * "Computational cost"). */
SLORR_API int64_t slorr_flops(const slorr_shape* shapes, int32_t count, int32_t iters);

/* Layer partition for data-parallel training (App. F: each rank regularizes a
 * subset of the layers; set grad_scale = world so the existing gradient
 * average restores lambda).  Longest-processing-time split of the matrices by
 * FLOPs; writes the indices owned by `rank` (ascending) to out_indices
 * (capacity >= count) and their number to *out_count.  Host-only. */
SLORR_API slorr_status slorr_partition(const slorr_shape* shapes, int32_t count, int32_t world,
                             int32_t rank, int32_t* out_indices, int32_t* out_count);

/* FLOPs the matrix products of one call execute on the path the handle's
 * options select (host-only): 2 x rows x columns x K over every tile of every
 * Gram, Poly and Update launch, counting the zero padding (P to a multiple of
 * 128, Q to a multiple of 128) and the 256-row CTA-pair MMAs, and skipping
 * the strictly-lower tiles of the symmetric products.  slorr_flops gives the
 * paper's algorithmic count (Sec. 3 "Computational cost") instead. */
SLORR_API slorr_status slorr_executed_flops(const slorr_handle* h, double* out);

/* Work items of one GEMM launch of the plan (host-only): phase 0 Gram, 1 Poly,
 * 2 Update.  For the tensor-core kernel an item is a 256 x 256 output tile or,
 * for Gram tiles whose K range is split (the default for sets with few long-K
 * tiles, unless SLORR_FLAG_NO_SPLIT_K is set), one K part of such a tile; for
 * the CUDA-core kernel it is a 32 x 32 tile. */
SLORR_API slorr_status slorr_gemm_items(const slorr_handle* h, int32_t phase, int32_t* items);

/* The work items of one GEMM launch of the plan (host-only), in the order the
 * launch hands them out (tensor cores: item i to CTA pair i mod npairs):
 * 7 int32 per item, (mat, tm, tn, msz, nsz, part, parts): matrix index, row
 * and column tile index, rows and columns of the tile, and for a Gram tile
 * whose K range is split, which of `parts` equal K ranges this item
 * accumulates (part 0 of 1 otherwise).  `out` holds `capacity` int32, at
 * least 7 * slorr_gemm_items().  Errors: SLORR_ERR_INVALID_ARG for a NULL
 * pointer, a phase outside 0..2 or a capacity that is too small. */
SLORR_API slorr_status slorr_gemm_item_list(const slorr_handle* h, int32_t phase, int32_t* out, int32_t capacity);

/* The dataflow plan of the tensor-core GEMMs (host-only): every Gram, Poly and
 * Update item of the T steps in one launch.  CTA pair q runs its items in
 * order; an item may start once its matrix's completion count (each epilogue
 * warp of both CTAs adds 1 per item it finishes: 16 per item) reaches the
 * item's threshold, i.e. once every item of the matrix's earlier (step, phase)
 * groups is stored.  *npairs receives the pairs the plan is made for (76 for
 * GB300's 152 SMs until a call re-plans for the current device) and *count
 * the items.  Unless `out` is NULL, it receives 10 int32 per item, pair by
 * pair: (pair, seq, step, phase, mat, tm, tn, part, parts, wait), where seq
 * is the item's rank when all items are ordered by their planned start
 * (every item comes after every item it waits for), step is 0-based, phase 0
 * Gram, 1 Poly, 2 Update, and part/parts as for slorr_gemm_item_list.
 * `capacity` counts int32.  *makespan_k (if not NULL) receives the planned
 * duration in K blocks of a 256 x 256 tile.  Errors: SLORR_ERR_INVALID_ARG
 * for a NULL handle or count, a capacity below 10 x items, or a handle that
 * runs per-phase launches (SLORR_FLAG_PHASE_LAUNCHES, a set above the size
 * for which the dataflow launch is chosen, fp32 or CUDA-core). */
SLORR_API slorr_status slorr_dataflow_items(const slorr_handle* h, int32_t* out, int32_t capacity, int32_t* npairs,
                                            int32_t* count, double* makespan_k);

/* Balance of one tensor-core GEMM launch (host-only): the launch hands item i
 * to CTA pair i mod npairs.  *max_k is the largest total K (the K
 * range of each item, summed over one pair's items) and *total_k the sum over
 * all items, so total_k / npairs is the ideal.  The CTA-pair plan is ordered
 * to balance npairs = 76 (152 SMs).  Errors: SLORR_ERR_INVALID_ARG for a NULL
 * pointer, a phase outside 0..2 or npairs < 1. */
SLORR_API slorr_status slorr_gemm_pair_load(const slorr_handle* h, int32_t phase, int32_t npairs, int64_t* max_k,
                                            int64_t* total_k);

/* Per-kernel timing (tracing).  While enabled, every kernel this handle
 * launches is bracketed by a pair of CUDA events recorded on the caller's
 * stream (events are created on the host; no device memory is allocated).
 * slorr_read_timing() waits for the recorded events, adds the elapsed
 * milliseconds and kernel launch counts per kind into ms[k] / launches[k]
 * (k < kinds, kinds <= SLORR_NUM_KERNEL_KINDS; kinds are sumsq, cast, gram,
 * poly, update, dot, combine, normcast: the 16-bit iterates' single pass
 * for the norm and X_0, which replaces sumsq and cast; gemm: the dataflow
 * launch of every Gram, Poly and Update of a call, which replaces the gram,
 * poly and update launches; sumsq, normcast and dot each include their
 * finalize kernel) and forgets them. */
#define SLORR_NUM_KERNEL_KINDS 9
SLORR_API slorr_status slorr_set_timing(slorr_handle* h, int32_t enable);
SLORR_API slorr_status slorr_read_timing(slorr_handle* h, double* ms, int64_t* launches, int32_t kinds);

/* ||W||_F^2 of one matrix (the squared Frobenius norm of Listing 1 and Sec. 3
 * "Computing the nuclear and Frobenius norms") without any device allocation.
 * The allocation-free form has no counterpart in the paper: it exists for
 * callers that cannot provide a workspace, e.g. code running while a stream
 * is captured, or under a framework that owns all device memory.
 *   weight       device pointer, row-major m x n, of slorr_dtype `dtype`
 *   out_frob_sq  device pointer to one double, written with sum_ij W_ij^2
 * Enqueued on `stream`; deterministic (fixed-order partial sums).  Scratch is
 * a fixed 256 KB array inside the library, present on every GPU that loads
 * it until the process exits; m * n may not exceed 536870912 (INVALID_ARG
 * otherwise).  All calls share that array: calls that overlap on the GPU
 * (other streams or host threads) race and must be serialised by the caller.
 * The first call on each device looks up the array's device address
 * (cudaGetSymbolAddress); make that first call before any stream capture.
 * Calls no cudaMalloc, cudaFree or other allocating routine. */
SLORR_API slorr_status slorr_frob_sq_noalloc(const void* weight, int64_t m, int64_t n, int32_t dtype,
                                             double* out_frob_sq, void* stream);

SLORR_API void        slorr_destroy(slorr_handle* h);
SLORR_API const char* slorr_status_string(slorr_status s);

/* ---- Host-resident weights and grads: a copy/compute pipeline ---------------
 * The same forward + backward as slorr_reg_forward_backward (Listing 1,
 * Alg. 2) for a weight set whose weights and grads live in host memory.  The
 * set is split into `groups` runs of consecutive matrices of about equal size
 * (the regularizer is a sum of independent per-matrix terms, Sec. 3), each
 * with its own plan; while group g is regularized on the caller's stream, the
 * weights and grads of the next groups are copied in on a second stream and
 * the updated grads of the previous ones are copied out on a third, so that
 * the host<->device copies in both directions overlap each other and the
 * kernels.  The results equal those of slorr_reg_forward_backward on the same
 * data (per-matrix values and grads bit for bit; the loss adds the groups'
 * partial losses in group order).
 *
 * slorr_pipeline_create: shapes / opt as for slorr_create; groups >= 1 (more
 * than `count` is clamped).  Host-only: no CUDA call until the first run,
 * which creates the two copy streams and the events on the current device;
 * every later run must use that device. */
typedef struct slorr_pipeline slorr_pipeline;
SLORR_API slorr_status slorr_pipeline_create(slorr_pipeline** out, const slorr_shape* shapes, int32_t count,
                                   const slorr_options* opt, int32_t groups);

/* Device workspace bytes a run needs (the groups' workspaces, the partial
 * losses and the per-matrix values); host-only. */
SLORR_API slorr_status slorr_pipeline_workspace_size(const slorr_pipeline* p, size_t* bytes);

/* One pipelined forward + backward, enqueued on `stream`:
 *   host_weights[i]  W_i in host memory, row-major m_i x n_i (page-locked,
 *                    e.g. cudaHostAlloc, for the copies to overlap)
 *   host_grads[i]    W_i.grad in host memory, same layout; ACCUMULATED (+=):
 *                    copied in, accumulated on the device, copied back
 *   host_loss        page-locked host float, written with lambda * sum_i L_i
 *   host_per_matrix  page-locked host array of `count` floats, or NULL
 *   dev_weights[i], dev_grads[i]
 *                    device staging buffers of W_i's size (16-byte aligned),
 *                    owned by the caller; overwritten
 *   workspace        >= slorr_pipeline_workspace_size() bytes, 256-byte aligned
 * When `stream` reaches the end of the call's work, every copy back to the
 * host has completed.  Host buffers must not be touched until then. */
SLORR_API slorr_status slorr_pipeline_forward_backward(slorr_pipeline* p, const void* const* host_weights,
                                             void* const* host_grads, float* host_loss, float* host_per_matrix,
                                             void* const* dev_weights, void* const* dev_grads, void* workspace,
                                             size_t workspace_bytes, void* stream);

/* As slorr_get_status, over every group of the pipeline. */
SLORR_API slorr_status slorr_pipeline_get_status(slorr_pipeline* p, const void* workspace, void* stream);

SLORR_API void slorr_pipeline_destroy(slorr_pipeline* p);

/* Human-readable reason for the last non-OK status returned on this thread. */
SLORR_API const char* slorr_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SLORR_H */
