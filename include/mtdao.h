/*
 * mtdao.h -- C ABI of the GB300 MT-DAO hot path (libmtdao.so).
 *
 * MT-DAO (Multi-timescale Distributed Adaptive Optimizers, arXiv 2510.05361)
 * runs M data-parallel workers that each take local optimizer steps with N
 * first-momentum EMAs at different beta timescales (section 2.3, Algorithm 1
 * for Adam, Algorithm 2 for ADOPT, Algorithm 3 for SGDM) and periodically
 * average their parameters x, each momentum u^j and the second moment v over
 * the workers, every state on its own period K_x, K_j, K_v.  This library
 * keeps the M workers as M replicas resident in one GPU's memory: the local
 * step is one fused elementwise pass over HBM and the averaging is an
 * in-memory reduction across replicas.
 *
 * Conventions shared by every call
 *   - Status: every call returns an mtdao_status (0 = success, negative =
 *     error) unless stated otherwise; nothing is thrown across the ABI.  The
 *     message of the last failure is kept per handle (mtdao_last_error).
 *   - Streams: all device work is enqueued on the handle's CUDA stream and is
 *     asynchronous unless a call says it synchronises.  Pointers marked
 *     "device" must be device-accessible on the handle's device.
 *   - Ownership: the library owns the state arena (x, u^1..u^N, v for all
 *     replicas) and its workspaces; the caller owns gradients, output buffers
 *     and the stream.
 *   - Threads: a handle must not be used from two threads at once.
 *   - Layout: the caller's list of tensors (numel_k, k = 0..n_tensors-1) is
 *     flattened into one per-replica vector of n_padded fp32 elements.
 *     Tensor k starts at offset_k, a multiple of 8 elements; padding between
 *     tensors and at the end is zero and stays zero when the gradient's
 *     padding is zero.  n_padded is a multiple of 256 elements.  State s of
 *     replica m occupies arena[(s*M + m)*n_padded .. +n_padded).
 *   - States: index 0 = x, 1..N = u^1..u^N, N+1 = v (Adam and ADOPT only).
 *     A sync mask has bit s set for state s.
 *   - Numerics: states are fp32; every update is computed in fp32 with
 *     IEEE-rounded division and square root (no fast-math).  Per-step
 *     scalars (bias corrections, clip bounds) are computed in double on the
 *     host and rounded once.
 */
#ifndef MTDAO_H
#define MTDAO_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MTDAO_VERSION 2
#define MTDAO_MAX_MOM 4          /* largest N supported */
#define MTDAO_MAX_REPLICAS 1024  /* largest M supported */

typedef enum {
    MTDAO_OK = 0,
    MTDAO_ERR_INVALID = -1,      /* bad argument or configuration */
    MTDAO_ERR_OOM = -2,          /* device or pinned-host allocation failed */
    MTDAO_ERR_CUDA = -3,         /* a CUDA runtime call or launch failed */
    MTDAO_ERR_ALIGN = -4,        /* a pointer is not aligned as the call requires (16 bytes
                                    for vectors, 8 bytes for double outputs) */
    MTDAO_ERR_STATE = -5         /* call not allowed in the handle's state */
} mtdao_status;

typedef enum {
    MTDAO_BASE_ADAM = 0,         /* Algorithm 1 */
    MTDAO_BASE_ADOPT = 1,        /* Algorithm 2 */
    MTDAO_BASE_SGDM = 2          /* Algorithm 3 */
} mtdao_base;

typedef enum {
    MTDAO_CLIP_NONE = 0,
    /* Adam/SGDM clip(g, rho): each replica's whole flattened gradient is
     * scaled by min(1, rho / (||g||_2 + 1e-6)); v keeps the raw gradient. */
    MTDAO_CLIP_GLOBAL_NORM = 1,
    /* ADOPT clip(g-hat, c_t): elementwise clamp to +-c_t, c_t = (t+1)^(1/4)
     * (t the 0-based step; see adopt_prev_v for the other ordering). */
    MTDAO_CLIP_ELEMENTWISE = 2
} mtdao_clip;

typedef enum { MTDAO_F32 = 0, MTDAO_BF16 = 1 } mtdao_dtype;

typedef enum {
    /* Algorithm 1: a state whose period K divides the completed local-step
     * count c = t+1 is averaged at the end of step t. */
    MTDAO_PHASE_ALG1 = 0,
    /* Algorithm 2 as printed: u^j and v are averaged at the end of step t
     * when t mod K == 0, x when (t+1) mod K_x == 0. */
    MTDAO_PHASE_ALG2_LITERAL = 1
} mtdao_phase;

/*
 * Hyper-parameters of Algorithms 1-3 (their "Require" lists).  Decay rates
 * and weights are doubles so that 1 - beta keeps its precision.
 */
typedef struct {
    int32_t base;                       /* mtdao_base */
    int32_t n_mom;                      /* N, 1..MTDAO_MAX_MOM */
    double beta1[MTDAO_MAX_MOM];        /* beta_{1,j} in [0, 1) */
    double omega[MTDAO_MAX_MOM];        /* omega_j in [0, 1], sum <= 1 */
    double beta2;                       /* beta_2 in [0, 1) (Adam, ADOPT) */
    double eps;                         /* epsilon > 0 (Adam, ADOPT) */
    int32_t bias_correction;            /* Adam: 1 = divide u^j by 1-beta_{1,j}^(t+1)
                                           and v by 1-beta_2^(t+1); 0 = Algorithm 1
                                           as printed.  Must be 0 otherwise. */
    int32_t clip_mode;                  /* mtdao_clip */
    double clip_rho;                    /* rho > 0 for MTDAO_CLIP_GLOBAL_NORM */
    int32_t sync_phase;                 /* mtdao_phase */
    int64_t period_x;                   /* K_x; 0 = never averaged */
    int64_t period_u[MTDAO_MAX_MOM];    /* K_j; 0 = never */
    int64_t period_v;                   /* K_v; 0 = never (ignored for SGDM) */
    int32_t adopt_prev_v;               /* ADOPT only.  0 = Algorithm 2 order: normalise
                                           with the freshly updated v.  1 = the original
                                           ADOPT order: step 0 only sets v = g_0^2, later
                                           steps normalise with the previous v, then update
                                           it.  The clamp bound is c = k^(1/4) for the k-th
                                           parameter update (1-based) in both orders. */
} mtdao_config;

typedef struct mtdao_ctx *mtdao_handle;

/* ------------------------------------------------------------------ host-only */

/* MTDAO_VERSION of the loaded library. */
int32_t mtdao_version(void);

/*
 * Fill *cfg with defaults for a base and N: beta_1 = (0.9, 0.999, 0.5, 0.99)
 * prefix, omega_j = 0.95/N, beta_2 = 0.999 (0.9999 for ADOPT, section 4.1),
 * eps = 1e-8, bias correction on for Adam, no clipping, Algorithm 1 phase,
 * all periods 32 (section 4.1 default K).  No device access.
 */
int mtdao_config_default(mtdao_config *cfg, int32_t base, int32_t n_mom);

/*
 * Check a configuration for M replicas against the ranges of Algorithms
 * 1-3 (beta in [0,1), omega_j in [0,1], sum omega <= 1 + 1e-6, periods >= 0,
 * clip mode matching the base).  MTDAO_OK or MTDAO_ERR_INVALID; the reason
 * is available from mtdao_last_error(NULL).  No device access.
 */
int mtdao_config_validate(const mtdao_config *cfg, int32_t M);

/* Number of state vectors per replica: 1 + N (+1 for v unless SGDM). */
int32_t mtdao_num_states(const mtdao_config *cfg);

/*
 * Flattened layout of a tensor list: offsets_out[k] (n_tensors entries,
 * caller-owned) and *n_padded_out as described under "Layout" above.
 * Zero-size tensors take no space (their offset is that of the next one).
 * MTDAO_ERR_INVALID for a negative numel, n_tensors < 1 or a list with no
 * element at all.  No device access.
 */
int mtdao_plan_layout(const int64_t *tensor_numel, int32_t n_tensors,
                      int64_t *offsets_out, int64_t *n_padded_out);

/*
 * Sync schedule (Algorithms 1 and 2, the "sync every K steps" rows): the
 * mask of states to average at the end of local step `step` (0-based)
 * under cfg->sync_phase.  No device access.
 */
int mtdao_due_mask(const mtdao_config *cfg, int64_t step, uint32_t *mask_out);

/*
 * Half-life of an EMA with decay rate beta (section 2.1):
 * tau_0.5(beta) = ln 0.5 / ln beta, the number of steps after which a
 * value's weight in u = beta u + (1 - beta) g has halved.  *tau_out gets
 * tau for 0 < beta < 1 and 0 for beta = 0.  MTDAO_ERR_INVALID for beta
 * outside [0, 1) or a NULL output.  No device access.
 */
int mtdao_half_life(double beta, double *tau_out);

/*
 * Half-life sync strategy (appendix on the wall-clock model, table of the
 * modelled configurations): the parameters keep period_x and every state
 * with a decay rate is averaged once per half-life of that rate, rounded to
 * the nearest integer, but never more often than the parameters:
 *   K_x = period_x,  K_j = max(K_x, round(tau_0.5(beta_{1,j}))),
 *   K_v = max(K_x, round(tau_0.5(beta_2)))    (K_v untouched for SGDM).
 * The table's caption speaks of the closest power of two, but its entries
 * (69, 693 and 6931 for beta = 0.99, 0.999 and 0.9999; K_x = 32 for
 * beta = 0.95, whose half-life is 13.5) are these rounded half-lives; the
 * entries are what is implemented.  Only the period fields of *cfg change.
 * MTDAO_ERR_INVALID for a NULL cfg, period_x < 0, or a decay rate outside
 * [0, 1).  No device access.
 */
int mtdao_config_half_life_periods(mtdao_config *cfg, int64_t period_x);

/*
 * Communication of a configuration relative to DDP, which averages one
 * d-element vector (the gradient) every step (section 2.3, the reduction
 * factor stated after the algorithm's description): each state s is
 * averaged once every K_s steps, so
 *   *factor_out = (1/K_x + sum_j 1/K_j + 1/K_v)^-1
 * (no v term for SGDM; a period of 0, never averaged, adds nothing;
 * +infinity when nothing is ever averaged).  MTDAO_ERR_INVALID for a NULL
 * argument or a negative period.  No device access.
 */
int mtdao_comm_reduction(const mtdao_config *cfg, double *factor_out);

/* ------------------------------------------------------------------ lifecycle */

/*
 * Create a handle on the current CUDA device for M replicas of the tensor
 * list tensor_numel[0..n_tensors-1] (host array).  This takes the inputs of
 * the "Require" lists of Algorithms 1-3: the number of workers M, the
 * hyper-parameters in *cfg (decay rates beta_j and beta_2, weights omega_j,
 * epsilon, the sync periods K_x, K_j, K_v, the clipping rule) and the shape
 * of the parameters x (the learning rates eta_t arrive per step, the
 * initial x_0 through mtdao_set_params).  Allocates the state
 * arena (num_states * M * n_padded fp32) and workspaces, zeroes every state
 * and sets the step counter t to 0.  cuda_stream is a cudaStream_t (NULL =
 * legacy default stream).  On failure *out is NULL and the reason is
 * available from mtdao_last_error(NULL).  Synchronises the stream once.
 */
int mtdao_create(const mtdao_config *cfg, int32_t M, const int64_t *tensor_numel,
                 int32_t n_tensors, void *cuda_stream, mtdao_handle *out);

/* Release everything the handle owns.  NULL-safe.  Synchronises its streams. */
void mtdao_destroy(mtdao_handle h);

/* Switch the stream later calls enqueue on (the caller orders the change). */
int mtdao_set_stream(mtdao_handle h, void *cuda_stream);

/*
 * Initial state (Algorithm 1 "for each worker: initialize"): copy x0
 * (device, [n_padded] fp32, padding zero) into x of every replica, zero all
 * u^j and v, set t = 0.  All workers start from the same x_0 (appendix,
 * x_{-1} = x_0 shared).
 */
int mtdao_set_params(mtdao_handle h, const float *x0_dev);

/* ------------------------------------------------------------------ hot path */

/*
 * One local step t (= the handle's counter, then t+1) of Algorithm 1, 2 or 3
 * on every replica, as one pass over HBM:
 *   Adam  : g-hat = clip(g); u^j = beta_j u^j + (1-beta_j) g-hat;
 *           v = beta_2 v + (1-beta_2) g^2;
 *           Delta = [(1-sum w) g-hat + sum w_j u^j/b_j] / (sqrt(v/b_v) + eps);
 *           x = x - lr * Delta        (b = 1 - beta^(t+1), or 1 if no correction)
 *   ADOPT : v = beta_2 v + (1-beta_2) g^2; g-tilde = clip(g/(sqrt(v)+eps), c_t);
 *           u^j = beta_j u^j + (1-beta_j) g-tilde;
 *           Delta = (1-sum w) g-tilde + sum w_j u^j;  x = x - lr * Delta
 *   SGDM  : as Adam without v and without the denominator.
 * grads_dev: device, [M][n_padded] of grad_dtype (mtdao_dtype), 16-byte
 *   aligned, padding zero; read only.
 * lr: eta_t for this step.
 * sync_mask: states to average over the replicas at the end of this same
 *   step (E_m[.] of Algorithm 1); usually the value of mtdao_sync_due.  The
 *   average is fused into the step's pass: it costs no extra HBM traffic for
 *   2 <= M <= 64 (a block stages a span of all replicas in shared memory
 *   from M = 9); larger M fall back to a separate averaging pass.
 * With MTDAO_CLIP_GLOBAL_NORM a reduction pass over grads precedes the step.
 * With adopt_prev_v (the original ADOPT order) step 0 runs a separate pass
 * that writes v = g_0^2 and reads or writes nothing else, so u and x keep
 * their initial values even where g_0 is not finite.
 * Errors: MTDAO_ERR_INVALID (dtype, mask bits beyond the states),
 * MTDAO_ERR_ALIGN, MTDAO_ERR_CUDA.  On error t is unchanged.
 */
int mtdao_step(mtdao_handle h, const void *grads_dev, int32_t grad_dtype, double lr,
               uint32_t sync_mask);

/*
 * count consecutive local steps in one call, each with the averages its end
 * brings under the handle's schedule (mtdao_due_mask at the handle's t):
 * the same work as count pairs of mtdao_sync_due + mtdao_step, without a
 * round trip to the caller per step (for small models, whose steps take
 * tens of microseconds).  Step k reads its gradients at
 * grads_dev + k * grads_stride_bytes (stride 0: the same buffer for every
 * step; otherwise a multiple of 16) and uses lrs[k] (host array of count
 * doubles).  Stops at the first failing step (t counts the steps done).
 */
int mtdao_run(mtdao_handle h, const void *grads_dev, int64_t grads_stride_bytes, int32_t grad_dtype,
              const double *lrs, int32_t count);

/*
 * mtdao_step with the gradients in host memory ([M][n_padded], 16-byte
 * aligned).  Pinned memory (cudaHostAlloc / cudaHostRegister) is read by the
 * step kernel directly over the host link, with no copy and no staging
 * memory.  Other (pageable) memory is first copied into a library-owned
 * device staging buffer (two buffers, allocated on first use, so that a
 * copy can overlap the previous step).  grads_host must stay unchanged until
 * the call's work on the stream has completed.
 */
int mtdao_step_host(mtdao_handle h, const void *grads_host, int32_t grad_dtype, double lr,
                    uint32_t sync_mask);

/*
 * Outer synchronisation (Algorithms 1-3, E_m[.] with OuterOpt = averaging):
 * every state in mask is replaced, on every replica, by the equal-weight
 * mean over the M replicas.  Computed in fp32 as s_0 + (A + B) / M, A and
 * B the Kahan-compensated sums of (s_m - s_0) over replicas 1..h-1 and
 * h..M-1 (h = floor(M/2)), each in replica order; this returns s_0 bit for
 * bit when the replicas agree, and otherwise stays within a few roundings
 * of the largest replica value for any M (relative to the mean itself only
 * when the replicas do not cancel).  Where that is NaN (the compensation
 * meets an infinite value) the mean is the plain sum of the M values over
 * M: +-Inf when they hold infinities of one sign, NaN otherwise.  The
 * fused average in mtdao_step and mtdao_sync_stats use the same routine
 * (identical bits).  mask 0 is a no-op.
 */
int mtdao_sync(mtdao_handle h, uint32_t mask);

/*
 * mtdao_sync plus the paper's cross-worker diagnostics (section 4.1, "Other
 * Metrics"), formed in the same pass over the replicas at no extra state
 * traffic.  For every state s in mask, in increasing state order, stats_dev
 * (device, caller-owned, 8-byte aligned, popcount(mask) * (2 + 2M) doubles)
 * receives, from
 * the replicas before they are averaged and their fp32 mean s_bar:
 *   [0]              (1/M) sum_m ||s_m - s_bar||^2   cross-worker variance
 *   [1]              ||s_bar||^2
 *   [2 + m]          ||s_m||^2                        m = 0..M-1
 *   [2 + M + m]      <s_m, s_bar>                     (cosine = [2+M+m] /
 *                                                      sqrt([2+m] * [1]))
 * The averaged states are bit-identical to mtdao_sync's.  Sums are
 * fixed-order (bit-reproducible).  With M = 1 the states are left as they
 * are and only the diagnostics are written.  For M <= 64 the sums are
 * formed in the averaging pass itself (the sync's traffic, 8 M bytes per
 * element and state; from M = 9 a block stages a span of all replicas in
 * shared memory); for larger M each state takes two passes through a
 * library-owned [n_padded] fp32 scratch that holds the mean (about twice
 * the traffic).  Every path forms (s_m - s_bar) against the fp32 mean it
 * stores, sums a thread's elements in fp32 with Kahan compensation and
 * adds the partial sums in fp64.  Workspaces are allocated on the first call.
 */
int mtdao_sync_stats(mtdao_handle h, uint32_t mask, double *stats_dev);

/*
 * Anchors for the diagnostics of change over a round (section 4.1 "Other
 * Metrics": relative change ||s_{t+K} - s_t|| / ||s_t||; section 5.4: the
 * pseudo-gradient Delta^m = x^m_{t+K} - x^m_t, the worker update over a
 * round, and its mean).  Bit s of state_mask keeps an anchor for state s:
 * one [n_padded] fp32 vector, set to replica 0's value now and, from then
 * on, after every step, sync or sync_stats that averages state s (one
 * device-to-device copy of n_padded floats per average), so it holds the
 * state at the start of the current round.  Anchors whose bit is clear are
 * freed (synchronises the stream); state_mask 0 frees all.
 */
int mtdao_track_anchor(mtdao_handle h, uint32_t state_mask);

/*
 * Change diagnostics of one state against its anchor a, read-only (no state
 * changes), fixed-order sums.  With s_bar the replica mean an average would
 * store now, out_dev (device, 8-byte aligned, 2M + 2 doubles) gets
 *   [m]        ||s_m - a||^2                 m = 0..M-1  (local change, for x
 *                                                          the pseudo-gradient)
 *   [M + m]    <s_m - a, s_bar - a>
 *   [2M]       ||s_bar - a||^2                           (global change)
 *   [2M + 1]   ||a||^2
 * so cos(local, global) = [M+m] / sqrt([m] [2M]) and the relative change of
 * the averaged state over the round = sqrt([2M] / [2M+1]).  Call it before
 * the round's average of that state.  MTDAO_ERR_STATE if the state has no
 * anchor.  For M > 64 it takes two read-only passes through the scratch of
 * mtdao_sync_stats.
 */
int mtdao_pseudo_grad_stats(mtdao_handle h, int32_t state, double *out_dev);

/* Mask of states due at the end of the next step (mtdao_due_mask at t). */
int mtdao_sync_due(mtdao_handle h, uint32_t *mask_out);

/*
 * Squared L2 norm of each replica's flattened gradient (the quantity that
 * clip(g, rho) of Algorithms 1 and 3 is based on): out_dev (device, M
 * doubles, caller-owned, 8-byte aligned) receives sum_i g[m][i]^2.
 * Deterministic: fixed grid and fixed reduction order.  Squares are summed
 * in fp32 with compensation where they stay within fp32's range; groups of
 * four f32 or eight bf16 values (one 16-byte load) whose squares overflow or
 * underflow fp32 (|g| above ~1e19 or below ~1e-19) are summed in fp64, so
 * every finite gradient gives a finite, accurate sum.  Uses a handle-owned
 * workspace of partial sums.
 * Errors: MTDAO_ERR_INVALID, MTDAO_ERR_ALIGN, MTDAO_ERR_CUDA.
 */
int mtdao_grad_sqnorm(mtdao_handle h, const void *grads_dev, int32_t grad_dtype,
                      double *out_dev);

/*
 * Gradient health check (the paper has no counterpart; NaN and Inf
 * gradients otherwise propagate into every state of the replica, as the
 * algorithms written out would propagate them): out_dev (device, M doubles,
 * caller-owned, 8-byte aligned) receives the number of NaN or +-Inf values in replica m's
 * gradient, exact.  A caller can skip a step whose count is nonzero (e.g.
 * an overflow of bf16 gradients).  Same grid, workspace and
 * determinism as mtdao_grad_sqnorm; reads the gradient once (g_b bytes per
 * element).  Errors as mtdao_grad_sqnorm.
 */
int mtdao_grad_nonfinite(mtdao_handle h, const void *grads_dev, int32_t grad_dtype,
                         double *out_dev);

/*
 * mtdao_grad_sqnorm_static -- the per-replica sum of squares of
 * mtdao_grad_sqnorm for callers that cannot allocate device memory.
 * The paper has no counterpart; this is a library convenience.
 *
 * Who needs it: a process whose device memory is reserved up front by
 * another allocator (so a cudaMalloc from this library would fail), a
 * latency-critical loop in which cudaMalloc/cudaFree would synchronise the
 * device, or a hook that sees only a gradient buffer and holds no handle
 * (mtdao_create allocates).  This call allocates nothing: neither
 * cudaMalloc/cudaFree nor any allocating library routine.
 *
 * Scratch: its per-block partial sums live in one file-scope device array
 * of MTDAO_STATIC_SCRATCH_DOUBLES doubles (32 KiB), which every device that
 * loads the library holds until the process exits.  A call needs
 * M * blocks_per_replica slots (blocks_per_replica = max(1, 4 * SMs / M),
 * the grid of mtdao_grad_sqnorm, so both return the same bits); a call that
 * would need more fails with MTDAO_ERR_INVALID and a message.  On a 152-SM
 * GB300 a call needs at most max(M, 608) <= 1024 slots, so every valid M
 * fits; the limit binds only on devices with more than 1024 SMs.  Every slot a
 * call reads is written earlier in the same call, so nothing has to be
 * cleared between calls; the array keeps the last call's partial sums.
 * All calls on a device share the array: calls whose GPU work overlaps (on
 * different streams or from different threads) race and return garbage.
 *
 * Set-up: the first call on a device (with that device current) looks up
 * the array's device address with cudaGetSymbolAddress and caches it, keyed
 * by the device and the unique id of its current context; the first call
 * after the context changed (after a cudaDeviceReset, say) looks it up
 * again.  Make the first call on a device before any stream capture begins.
 *
 * grads_dev: device, [M][n_padded] of grad_dtype, 16-byte aligned;
 * n_padded a positive multiple of 256; 1 <= M <= MTDAO_MAX_REPLICAS.
 * out_dev: device, M doubles (caller-owned, 8-byte aligned), receives
 *   sum_i g[m][i]^2 (computed as by mtdao_grad_sqnorm).
 * cuda_stream: cudaStream_t the work is enqueued on (asynchronous).
 * Errors: MTDAO_ERR_INVALID, MTDAO_ERR_ALIGN, MTDAO_ERR_CUDA; the message is
 * available from mtdao_last_error(NULL) in the calling thread.
 */
#define MTDAO_STATIC_SCRATCH_DOUBLES 4096
int mtdao_grad_sqnorm_static(const void *grads_dev, int32_t grad_dtype, int32_t M,
                             int64_t n_padded, double *out_dev, void *cuda_stream);

/* ------------------------------------------------------------------ state access */

/*
 * Device pointer to state `state` of replica `replica` ([n_padded] fp32,
 * owned by the handle, valid until destroy): the outputs of Algorithms 1-3
 * ("Ensure x_T, {u^j}, v") are read here, x = state 0 of any replica after
 * an average of x, u^j = state j, v = state N+1.  Errors: MTDAO_ERR_INVALID
 * for a state or replica out of range or a NULL dev_ptr.
 */
int mtdao_get_state_ptr(mtdao_handle h, int32_t state, int32_t replica, float **dev_ptr);

/* Copy one state vector to host memory ([n_padded] floats); synchronises. */
int mtdao_copy_state_to_host(mtdao_handle h, int32_t state, int32_t replica, float *host_out);

/* Copy one state vector from host memory ([n_padded] floats); synchronises. */
int mtdao_copy_state_from_host(mtdao_handle h, int32_t state, int32_t replica,
                               const float *host_in);

/*
 * Layout of the handle: *n_padded, *n_tensors, *M, *n_states and a pointer
 * to the handle-owned offsets array (valid until destroy).  Any output
 * pointer may be NULL.  This maps the flattened state vectors back to the
 * caller's tensors, the shape in which Algorithms 1-3 hand back their
 * outputs x_T, {u^j}, v ("Ensure"): tensor k of state s, replica m starts at
 * state pointer + offset_k.  Host-only, no device access.
 */
int mtdao_layout(mtdao_handle h, int64_t *n_padded, int32_t *n_tensors, int32_t *M,
                 int32_t *n_states, const int64_t **tensor_offsets);

/* Step counter t (local steps taken); -1 for a NULL handle. */
int64_t mtdao_get_step(mtdao_handle h);

/* Set t, e.g. when resuming from a checkpoint of the states; t >= 0. */
int mtdao_set_step(mtdao_handle h, int64_t step);

/*
 * Message of the handle's last failure ("" if none).  With h == NULL: the
 * last failure of a call without a handle (mtdao_create,
 * mtdao_config_validate, mtdao_grad_sqnorm_static, ...) in this thread.
 */
const char *mtdao_last_error(mtdao_handle h);

#ifdef __cplusplus
}
#endif

#endif /* MTDAO_H */
