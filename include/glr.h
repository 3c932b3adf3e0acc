/*
 * glr.h -- C ABI of the GB300 GreedyLore compression library (libglr.so).
 *
 * One handle holds the compressor state of ONE layer matrix X in R^{m x n}
 * trained by N data-parallel nodes (the problem statement of Sec. 1, Eq.
 * formulation), all simulated on one GPU.  glr_step runs one iteration of
 * Algorithm 3 (GreedyLore) for that matrix:
 *
 *   M_i   = G_i + E_i                          error-compensated gradient
 *   J, P  = Approx-Top-r(M_1..M_N, U, r)       Algorithm 2, Eq. semi-lazy-svd-3
 *   R_i   = P^T M_i,  Rbar = mean_i R_i        Eq. 8zhb2we09 (the All-Reduce is a
 *                                               fixed-order sum in device memory)
 *   Ghat  = P Rbar                             decompression
 *   X     = Optimizer(X, Ghat)                 Eq. msgd / Eq. adam
 *   E_i   = M_i - P R_i                        error feedback, Eq. ef2
 *
 * and, when (t - compress_start) mod tau == 0, the Semi-Lazy SVD refresh of
 * Eq. SVD-P1: U <- left singular basis of mean_i M_i; under Algorithm 3 that
 * step uses the uncompressed mean and resets E_i = 0.  Matrices with m > n are
 * handled on their transpose (Algorithm 4 orientation rule, Appendix D), so the
 * basis is min(m, n)^2.  Notation below: m' = min(m, n), n' = max(m, n).
 *
 * Conventions for every entry point
 *   - Return value: GLR_OK (0) or a negative GLR_E* code; nothing throws.  The
 *     message of the last failure on a handle is glr_last_error(handle); a
 *     failure of glr_create is reported by glr_last_error(NULL).
 *   - "device pointer": memory of the CUDA device that was current when the
 *     handle was created; "host pointer": ordinary or pinned host memory.
 *   - All GPU work is enqueued on the caller's stream (cudaStream_t passed as
 *     void*; NULL = legacy default stream) and is stream-ordered.  Functions
 *     that return host data synchronise that stream first.
 *   - A handle is not thread-safe; distinct handles may be used concurrently.
 *   - The library owns every buffer it allocates; the caller owns G, X and all
 *     output buffers it passes in.
 */
#ifndef GLR_H
#define GLR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------------------------- */
#define GLR_OK          0
#define GLR_EINVAL     -1   /* bad argument (sizes, null pointer, unknown enum value)      */
#define GLR_ENOMEM     -2   /* a device or host allocation failed                          */
#define GLR_ECUDA      -3   /* a CUDA runtime call or kernel launch failed                 */
#define GLR_ENUMERIC   -4   /* the refresh could not orthonormalise its basis (glr_get_stats) */
#define GLR_ENONFINITE -5   /* a NaN or Inf reached the node-mean gradient (glr_get_stats)  */
#define GLR_ETIMEOUT   -6   /* a bounded device-side wait gave up (reported by glr_get_stats) */

/* ---- enumerations -------------------------------------------------------------------- */
#define GLR_ALG3 0   /* refresh step: uncompressed mean, E reset to 0 (Algorithm 3)          */
#define GLR_ALG4 1   /* refresh step still compressed with P = U[:, :r], no E reset (Alg. 4) */

#define GLR_MSGD 0   /* Eq. msgd:  M = b1 M + (1 - b1) G;  X -= lr M                          */
#define GLR_ADAM 1   /* Eq. adam:  M, V EMAs; X -= lr M / (sqrt(V) + eps); no bias correction */
#define GLR_AMSGRAD 2   /* the analysis' AMSGrad-type Adam (App. A): M, V EMAs as GLR_ADAM,   *
                         * Vt = max(Vt, max_e V), X -= lr M / sqrt(Vt + eps) (one scalar)    */
#define GLR_ADAMW 3     /* bias-corrected AdamW: M, V EMAs, X -= lr (Mh / (sqrt(Vh) + eps) +   *
                         * weight_decay X), Mh = M / (1 - b1^s), Vh = V / (1 - b2^s), s = the  *
                         * optimizer step (1, 2, ...: every step, refresh and warm-up included)*/
#define GLR_GALORE_ADAM 4  /* Algorithm 5 (distributed Adam-type GaLore, App. E): Adam state on *
                            * the projected mean, M, V r x n' (EMAs as GLR_ADAM of Rbar), zeroed *
                            * at every refresh; X -= lr P (M / (sqrt(V) + eps)), transposed back *
                            * when m > n.  Needs refresh_mode GLR_ALG4, selection GLR_SEL_FIXED, *
                            * no_error_feedback 1 and compress_start 0                          */

#define GLR_SEL_APPROX 0   /* Algorithm 2 (Approx-Top-r) picks J at every compressed step    */
#define GLR_SEL_FIXED  1   /* P = U[:, :r] for the whole refresh period: the Lazy-SVD of       *
                            * Algorithm 1 (with no_error_feedback = 1 it is Algorithm 1)       */

#define GLR_F32  0   /* gradients G_i are float32                                            */
#define GLR_BF16 1   /* gradients G_i are bfloat16                                           */

#define GLR_MAX_NODES 64

/* Compressor and optimizer settings (Algorithm 3 inputs: tau, r; Sec. 2 optimizers).
 *   tau            refresh period (>= 1)
 *   refresh_mode   GLR_ALG3 | GLR_ALG4
 *   optimizer      GLR_MSGD | GLR_ADAM | GLR_AMSGRAD | GLR_ADAMW | GLR_GALORE_ADAM; lr = gamma;
 *                  beta1 = beta (MSGD) or beta_1 (Adam types); beta2, eps used by the Adam
 *                  types only
 *   seed           64-bit key of the shared random vectors v_j (Eq. random-v): all nodes
 *                  of one matrix draw the same v_j; give every matrix its own seed
 *   basis_rank     k.  0 (or m') keeps the full m' x m' singular basis U of Eq. SVD-P1
 *                  (paper-exact): any m' <= 1024; above that m' a multiple of 128 up to 4096
 *                  with n' a multiple of 8, bf16 gradients, MSGD or Adam, 16 <= r <= 128 (a
 *                  multiple of 4) and N <= 8 (the tcgen05 path; its refresh is a blocked
 *                  Jacobi eigen-solve of Mbar Mbar^T, GLR_ENUMERIC from glr_get_stats when it
 *                  has not converged in 30 sweeps).  r <= k < m', k <= 512, keeps the top-k
 *                  singular vectors and completes them to an orthogonal U with Householder
 *                  reflectors; the refresh then uses power_iters block power iterations
 *   power_iters    q >= 1 (truncated basis only)
 *   grad_dtype     GLR_F32 | GLR_BF16
 *   compress_start the first compress_start steps are uncompressed (plain node mean, no
 *                  error feedback); step compress_start is the first refresh
 *   no_error_feedback  1 drops error feedback (E_i stays 0, M_i = G_i): the comparison of
 *                  Sec. 4 / Fig. 2 and, with selection = GLR_SEL_FIXED, Algorithm 1
 *   selection      GLR_SEL_APPROX (default) | GLR_SEL_FIXED
 *   weight_decay   GLR_ADAMW's decoupled weight decay (ignored by the other optimizers)
 * A zero-initialised schedule with tau set is GreedyLore (Algorithm 3) with MSGD.        */
typedef struct glr_schedule {
    int32_t  tau;
    int32_t  refresh_mode;
    int32_t  optimizer;
    float    lr;
    float    beta1;
    float    beta2;
    float    eps;
    uint64_t seed;
    int32_t  basis_rank;
    int32_t  power_iters;
    int32_t  grad_dtype;
    int32_t  compress_start;
    int32_t  no_error_feedback;
    int32_t  selection;
    float    weight_decay;
} glr_schedule;

typedef struct glr_handle glr_handle;

/* Counters of one handle.  comm_floats_* are the floats the paper's nodes would exchange
 * (Table 2: n r + m per compressed step, m n at a refresh), counted per node.           */
typedef struct glr_stats {
    int64_t t;                      /* steps taken                                           */
    int64_t refreshes;              /* refresh steps taken                                   */
    int64_t comm_floats_total;      /* sum over steps of the per-node exchanged floats       */
    int64_t state_bytes;            /* device bytes owned by the handle                      */
    int32_t m_prime, n_prime, r, k; /* oriented sizes, rank, basis rank                      */
    int32_t transposed;             /* 1 when m > n (the handle works on G^T)                */
    int32_t last_refresh_sweeps;    /* eigen-solver sweeps used by the last refresh          */
    int64_t launches;               /* kernels launched by this handle so far                */
    int32_t path;                   /* kernel family that runs the step: GLR_PATH_*          */
    int32_t nonfinite;              /* warps of the compose pass that found a NaN or Inf in  *
                                     * the node-mean gradient since creation (0: all finite) */
    int32_t numeric_failures;       /* refresh factorisations that could not be completed    */
    int32_t reserved;
} glr_stats;

/* Kernel families (glr_stats.path), chosen by glr_create from the shape and schedule.       */
#define GLR_PATH_STRIP   0   /* fused strip kernels, products on the FP32 pipes (m' <= 4096)  */
#define GLR_PATH_MMA     1   /* fused strip kernels, 3xTF32 mma.sync compose (small m', r)    */
#define GLR_PATH_TCGEN05 2   /* tcgen05 tensor-core path: TF32 products, TMA-staged epilogues *
                              * (truncated basis, bf16 gradients, MSGD / Adam, 16 <= r <= 128) */
#define GLR_PATH_LIBRARY 3   /* unfused passes with cuBLAS products (large fp32 matrices)     */
#define GLR_PATH_PLAIN   4   /* unfused passes with the library's own FFMA GEMM               */

/* Phases of a step, for glr_profile_read.                                                 */
#define GLR_PH_PREV_PROJECT 0   /* R_i = P_{t-1}^T B_i for the deferred error                 */
#define GLR_PH_COMPOSE      1   /* K1: M_i = G_i + E_i, B_i <- M_i, Mbar                      */
#define GLR_PH_LAMBDA       2   /* Algorithm 2 bilinear forms (and W = Y^T Mbar, truncated)   */
#define GLR_PH_SELECT       3   /* arg-top-r and P = U[:, J]                                  */
#define GLR_PH_PROJECT      4   /* Rbar = P^T Mbar                                            */
#define GLR_PH_UPDATE       5   /* K3: Ghat = P Rbar (or Mbar) + optimizer                    */
#define GLR_PH_REFRESH      6   /* Semi-Lazy SVD refresh of the basis                         */
#define GLR_PHASES          7

/* Device time per phase, accumulated over the steps taken while profiling was enabled.   */
typedef struct glr_profile {
    double  ms[GLR_PHASES];         /* CUDA-event milliseconds on the step's stream          */
    int64_t launches[GLR_PHASES];   /* kernel launches                                        */
    int64_t count[GLR_PHASES];      /* number of timed occurrences                            */
} glr_profile;

/* ---- lifetime ------------------------------------------------------------------------ */

/* Create the state for one m x n layer matrix and N nodes (Sec. 1, Eq. formulation;
 * Algorithm 3 inputs).  Requires m, n >= 1, 1 <= r <= min(m, n), 1 <= N <= GLR_MAX_NODES,
 * tau >= 1 and a valid schedule (see glr_schedule).  Allocates all state on the current
 * CUDA device: E_i (N x m' x n' fp32), the basis, optimizer moments (m x n fp32, two for
 * the Adam types; r x n' for GLR_GALORE_ADAM) and workspace.  E starts at 0 and U at I
 * (Algorithm 3 input); t = 0.  On success *out receives the handle.
 * Errors: GLR_EINVAL, GLR_ENOMEM, GLR_ECUDA.                                             */
int glr_create(int64_t m, int64_t n, int32_t r, int32_t N, const glr_schedule* schedule,
               glr_handle** out);

/* Free every device and host buffer of the handle (after synchronising the device).
 * NULL is accepted.                                                                      */
int glr_destroy(glr_handle* h);

/* ---- the step --------------------------------------------------------------------------- */

/* One iteration of Algorithm 3 (Algorithm 4 orientation) for this matrix.
 *   G       host array of N device pointers; G[i] is node i's gradient, row-major m x n
 *           of the schedule's grad_dtype, 16-byte aligned.  Read only; must stay valid
 *           until the stream has passed the step.
 *   X       device pointer, row-major m x n float32 weights, updated in place.
 *   stream  cudaStream_t (as void*).
 * No host/device synchronisation.  Errors: GLR_EINVAL (null or misaligned pointer),
 * GLR_ECUDA (launch failure).                                                            */
int glr_step(glr_handle* h, const void* const* G, float* X, void* stream);

/* One step of several handles at once (typically every layer matrix of a model), with the
 * streaming passes of all of them batched into shared kernel launches.  handles[j] gets the
 * gradient pointer array G[j] (N_j device pointers, as in glr_step) and the weights X[j].
 * Equivalent to calling glr_step on each handle in turn (same results); handles must be
 * distinct and on the current device.  Failures are reported by glr_last_error of the
 * offending handle, or glr_last_error(NULL) for malformed arrays.                        */
int glr_step_group(glr_handle* const* handles, int32_t count, const void* const* const* G, float* const* X,
                   void* stream);

/* The same step with host gradients: G_host[i] are host pointers (pinned memory gives
 * asynchronous copies) that are copied into library-owned device staging on the stream
 * before the step.  X is the device weight matrix (updated in place); when X_host_out is
 * not NULL the updated X is copied back to it and the stream is synchronised.          */
int glr_step_host(glr_handle* h, const void* const* G_host, float* X, float* X_host_out,
                  void* stream);

/* glr_step_group with host gradients, for a training loop that produces them on the host:
 * G_host[j][i] is node i's gradient of handles[j] (host memory, m x n of the gradient dtype;
 * pinned memory makes the copies asynchronous).  They are copied on one library copy stream
 * (the first handle's) into one of two library-owned device staging buffers per handle
 * (alternating per call, so the copies of one call overlap the compute of the previous one) and
 * the step waits for them on `stream`.  X[j] is the device weight matrix (updated in place);
 * when X_host_out is not NULL and X_host_out[j] is not NULL the updated X[j] is copied back to
 * it after the step on a second library stream (the first handle's read-back stream, so the
 * next call's gradient copies and compute run beside it; only that call's update, which
 * rewrites X, waits for it).  The call only enqueues work: X_host_out holds the
 * result after cudaDeviceSynchronize, or once `stream` has passed the next call on the same
 * handles; the gradient host buffers must stay valid until `stream` has passed this step.
 * Errors as glr_step_group.                                                                 */
int glr_step_group_host(glr_handle* const* handles, int32_t count, const void* const* const* G_host,
                        float* const* X, float* const* X_host_out, void* stream);

/* Data-parallel steps across processes: Algorithm 3's All-Reduce lines (Sec. 4.3; the per-step
 * traffic of Table 2) made explicit for nodes that live in different processes.  Each rank
 * creates a handle for its own shard of the N nodes of the data-parallel group (the same shard
 * size, m, n, r, schedule and seed on every rank) and runs every step in three calls; between them
 * the caller averages each buffer a call exposes over the ranks (an all-reduce of the sum divided
 * by the number of ranks, in place, in device memory, ordered after `stream`):
 *
 *   glr_dp_begin   M_i = G_i + E_i for the local nodes (Eq. ef1).  Exposes the shard's
 *                  Approx-Top-r scores lambda-bar (m' floats; Algorithm 2, Eq. lambda-bar: linear
 *                  in the node mean, so the average over shards is the group's), or on a refresh
 *                  or warm-up step the shard's node mean Mbar (m' x n' floats).
 *   glr_dp_select  With the averaged buffers: the refresh of the averaged Mbar (Eq. SVD-P1) or the
 *                  arg-top-r of the averaged lambda-bar, P = U[:, J], and the shard's projected
 *                  mean Rbar = P^T Mbar (exposed as Rbar^T, n' x rpad floats, rpad = r rounded up to
 *                  32; Eq. 8zhb2we09).  Nothing is exposed when the step is uncompressed.
 *   glr_dp_finish  With the averaged Rbar: Ghat = P Rbar (Mbar when uncompressed), the optimizer on
 *                  X (Eq. msgd / adam), and the error feedback E_i = M_i - P R_i of the local nodes
 *                  (deferred to the next step's compose pass, as in glr_step).
 *
 * The floats exchanged per step are Table 2's: m' + r n' on a compressed step (plus the padding
 * columns of Rbar^T when r is not a multiple of 32), m' n' on an Algorithm 3 refresh;
 * glr_stats.comm_floats_* count them.  G's pointers must stay valid until glr_dp_finish.  Only
 * handles on the tcgen05 path (glr_stats.path == GLR_PATH_TCGEN05) take these calls; others,
 * out-of-order calls (a begin before the last finish, a select without a begin, a finish without
 * a select), null or misaligned pointers return GLR_EINVAL.  `out` receives device pointers into
 * the handle's state (valid until the next call on the handle) and their sizes; count is 0..1. */
typedef struct {
    int32_t count;          /* buffers to average */
    int32_t pad_;
    float* ptr[2];          /* device pointers into the handle's state */
    int64_t floats[2];      /* floats in each */
} glr_dp_exchange;
int glr_dp_begin(glr_handle* h, const void* const* G, void* stream, glr_dp_exchange* out);
int glr_dp_select(glr_handle* h, void* stream, glr_dp_exchange* out);
int glr_dp_finish(glr_handle* h, float* X, void* stream);

/* Checkpoints.  glr_state_size gives the bytes of a checkpoint of h now; glr_save copies the
 * handle's whole state into host memory host_buf (at least that many bytes): the schedule
 * position (t, the refresh period, a pending forced selection), the basis, P, the error state
 * B, the optimizer moments and every other buffer glr_create allocated.  It runs on `stream`
 * after the work already queued there and synchronises it.  glr_load restores such a checkpoint
 * into a handle created with the same m, n, r, N, basis rank, gradient dtype, optimizer,
 * refresh mode and seed (GLR_EINVAL otherwise, or when the buffer is not a checkpoint, is
 * truncated, or its header names buffers or a pending selection this handle cannot hold),
 * also synchronising `stream`; stepping the restored handle continues exactly as the saved one
 * would have (same results bit for bit).  The format is this library's own (host byte order).  */
int glr_state_size(const glr_handle* h, int64_t* bytes);
int glr_save(glr_handle* h, void* host_buf, int64_t bytes, void* stream);
int glr_load(glr_handle* h, const void* host_buf, int64_t bytes, void* stream);

/* Make the next glr_step a refresh step (Semi-Lazy SVD, Eq. SVD-P1) and restart the tau
 * period there.                                                                          */
int glr_refresh(glr_handle* h);

/* ---- introspection (tests, debugging) ------------------------------------------------- */

/* Counters (see glr_stats).  Reads the handle's device flags with a blocking copy, so it
 * waits for work already queued on the device.  Returns GLR_ETIMEOUT (with out filled) when a
 * bounded wait inside a kernel of this handle's launches has given up since creation (the
 * results of those steps are not valid), else GLR_ENUMERIC when a refresh met a Gram matrix it
 * could not factor (a rank-deficient or zero node mean, e.g. all-zero gradients: the basis of
 * that refresh is not orthonormal), else GLR_ENONFINITE when a compose pass found a NaN or Inf
 * in the node-mean gradient (a node sent a non-finite gradient, or the error state overflowed),
 * else GLR_OK.                                                                             */
int glr_get_stats(const glr_handle* h, glr_stats* out);

/* Message of the last failure on h (or of the last failed glr_create when h is NULL);
 * "" when there was none.  The string stays valid until the next call on h.             */
const char* glr_last_error(const glr_handle* h);

/* E_i after the last step (Eq. ef2), oriented m' x n' row-major fp32, written to the
 * device buffer E_out.  0 <= i < N.                                                      */
int glr_get_error(glr_handle* h, int32_t i, float* E_out, void* stream);

/* The last step's selection: J (r int32, ascending, to host J_host), and when not NULL
 * the device buffers P_out (m' x r fp32), Rbar_out (r x n' fp32), lambda_out (m' fp32,
 * the node-mean lambda-bar of Algorithm 2) and Mbar_out (m' x n', mean_i M_i).  After a
 * refresh step under Algorithm 3 J is all -1 (no selection).  Synchronises the stream. */
int glr_get_selection(glr_handle* h, int32_t* J_host, float* P_out, float* Rbar_out,
                      float* lambda_out, float* Mbar_out, void* stream);

/* The current orthogonal basis U (m' x m' fp32, row-major) to the device buffer U_out.
 * With a truncated basis the Householder complement is materialised.                     */
int glr_get_basis(glr_handle* h, float* U_out, void* stream);

/* Replace the basis: Q (device, m' x k row-major fp32, orthonormal columns; k = the basis
 * rank, m' for the full basis) becomes U[:, :k]; a truncated basis is completed with
 * Householder reflectors on the device.  For tests that start both sides from one U.   */
int glr_set_basis(glr_handle* h, const float* Q, void* stream);

/* Turn per-phase timing on (1) or off (0).  While on, every phase of glr_step records a
 * pair of CUDA events on the step's stream (a few microseconds of overhead per phase).   */
int glr_profile_enable(glr_handle* h, int32_t enable);

/* Accumulated per-phase times since the last reset (synchronises the device); reset != 0
 * clears the accumulators afterwards.                                                    */
int glr_profile_read(glr_handle* h, glr_profile* out, int32_t reset);

/* Override the selection of the next compressed step with J_host (r distinct indices in
 * [0, m')), instead of Algorithm 2.  One-shot.                                           */
int glr_force_selection(glr_handle* h, const int32_t* J_host);

/* Test aid for the bounded device waits: one kernel on `stream` waits, with the same bounded
 * polling loop as the pipeline kernels, on an mbarrier that nothing arrives on; after `polls`
 * polls (1 <= polls <= 2^24) the wait gives up and counts the event in the handle's flags, and
 * the kernel returns normally (the device stays usable).  glr_get_stats then reports
 * GLR_ETIMEOUT, as it does after a real stuck wait.  Errors: GLR_EINVAL, GLR_ECUDA.       */
int glr_test_expire_wait(glr_handle* h, int32_t polls, void* stream);

/* ---- selection without device allocation ------------------------------------------------ */

/* The Approx-Top-r selection (the lambda-bar and J that glr_step computes for a full basis)
 * for callers that cannot let a library allocate device memory: frameworks that own the GPU
 * through their own caching allocator and forbid raw cudaMalloc from other libraries,
 * services that reserve all memory at start-up and allow no allocation on the hot path, and
 * code that must not risk the device synchronisation cudaMalloc/cudaFree can cause.  The
 * paper has no counterpart: this is a deployment variant, not a step of the method.
 *   U           device, m' x m' row-major fp32 orthogonal basis (columns u_j)
 *   Mbar        device, m' x n' row-major fp32 node-mean gradient
 *   seed, t     key and step of the shared random vectors v_j (same stream as glr_step)
 *   lambda_out  device, m' fp32: lambda-bar_j = u_j^T Mbar v_j
 *   J_out       device, r int32: the r largest lambda-bar^2 (ties to the lower index),
 *               ascending
 * Allocates nothing: the per-tile partial sums live in a fixed 4 MiB array inside the
 * library (2^20 floats; every GPU that loads the library holds it until the process exits).
 * Sizes with m' * ceil(n'/64) > 2^20 are rejected with GLR_EINVAL and a message in
 * glr_last_error(NULL).  The first call on each device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current; make that first call before any stream
 * capture.  Every call shares the one array and overwrites the partial sums it uses, so
 * calls that overlap on the GPU (other streams, other threads) race: serialise them.
 * Asynchronous on `stream`.  Errors: GLR_EINVAL, GLR_ECUDA.                              */
int glr_select_noalloc(int32_t m_prime, int32_t n_prime, int32_t r, const float* U, const float* Mbar,
                       uint64_t seed, int64_t t, float* lambda_out, int32_t* J_out, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* GLR_H */
