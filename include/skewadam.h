/*
 * libskewadam -- the SkewAdam optimizer step (tiered optimizer state for MoE
 * training) on one NVIDIA GB300 (sm_103a).
 *
 * The step follows "Where Should Optimizer State Live? Tiered State Allocation
 * for Memory-Efficient MoE Training":
 *   - tiers (Sec. 3 "The tiers", Fig. 1): backbone tensors keep fp32 momentum
 *     and a factored second moment; expert tensors keep only the factored
 *     second moment; the router keeps the exact (unfactored) second moment and
 *     no weight decay; any vector (1-D tensor) keeps the exact second moment
 *     (Algorithm 1);
 *   - factored second moment (Eq. 1): per matrix W (n x m) an fp32 row vector
 *     R (n) and column vector C (m) of exponential moving averages of the row
 *     and column means of G*G; Vhat = R C^T / mean(R);
 *   - update (Algorithm 1): D = sqrt(max(Vhat, eps)); backbone
 *     U = sqrt(1-beta2^t)/(1-beta1^t) * M / D with M = beta1 M + (1-beta1) G;
 *     other tiers U = sqrt(1-beta2^t) * G / D;
 *   - update clipping (Sec. 3 "Update clipping and low-precision updates"):
 *     U <- U / max(1, RMS(U)/d), RMS over the whole tensor;
 *   - decoupled weight decay fused into the fp32 update ahead of the cast
 *     (Sec. 3 footnote, Sec. 5): x = w (1 - lr*lambda) - lr * U;
 *   - dithered bf16 write-back (Sec. 3, Algorithm 1 last line): the fp32 value
 *     x is rounded to bf16 by adding a uniform 16-bit integer r to its bit
 *     pattern and truncating (unbiased stochastic rounding with the exact bf16
 *     ulp of x); r is a Philox-4x32-10 draw keyed by (seed) and counted by
 *     (element index / 8, tensor id, step), so a step is bit-reproducible;
 *   - state size (Sec. 3 "Memory model", Eq. 2, App. B Table 5): 4 bytes per
 *     momentum element, per exact-second-moment element and per R / C entry.
 *
 * Conventions for every entry point:
 *   - Return SKEW_OK (0) or a negative SKEW_E* code; nothing aborts or throws.
 *     skew_last_error() gives a one-line reason for the last failure on a
 *     handle (skew_create failures: pass NULL).
 *   - Device memory (weights, gradients, state, workspace) is owned by the
 *     caller; the library owns only host-side metadata in the handle.
 *   - Pointers passed as `void *stream` are cudaStream_t values (0 = legacy
 *     default stream). Work is enqueued asynchronously on that stream; one
 *     stream per handle at a time.
 *   - Element counts are 64-bit; a tensor may exceed 2^31 elements.
 */
#ifndef SKEWADAM_H_
#define SKEWADAM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes -------------------------------------------------------- */
#define SKEW_OK 0
#define SKEW_EINVAL (-1)   /* invalid argument (null, shape, tier, hyper-parameter, step, size) */
#define SKEW_ENOMEM (-2)   /* host allocation failed                                        */
#define SKEW_ECUDA (-3)    /* a CUDA runtime call failed                                   */
#define SKEW_ETIMEOUT (-4) /* a bounded device-side wait gave up (see skew_sync_status)    */
#define SKEW_ESTATE (-5)   /* call out of order (e.g. skew_step before skew_bind)          */
#define SKEW_ETOOBIG (-6)  /* tensor needs more scratch than skew_step_tensor_noalloc has */

/* ---- tiers (Sec. 3 "The tiers") -------------------------------------------- */
#define SKEW_TIER_BACKBONE 0 /* embeddings, positions, attention, dense FFN, norms */
#define SKEW_TIER_EXPERT 1   /* expert matrices                                     */
#define SKEW_TIER_ROUTER 2   /* the gate                                            */

/* ---- allocation policies: the paper's policy and the Table 3 variants ------ */
#define SKEW_POLICY_TIERED 0          /* SkewAdam as published                         */
#define SKEW_POLICY_EXPERT_MOMENTUM 1 /* "+ momentum on experts"                        */
#define SKEW_POLICY_FACTORED_ROUTER 2 /* "factored router"                              */
#define SKEW_POLICY_UNIFORM 3         /* "uniform (momentum + factored)" on every tier  */
/* The Adafactor comparator (Sec. 5, Table 4 and its footnote, App. A; Shazeer &
 * Stern 2018): every matrix factored (the router too), vectors exact, no momentum, the
 * second-moment decay annealed as beta2_t = 1 - t^-0.8 (beta1 and beta2 are then
 * unused) and no bias correction; the same clipping, decay and write-back. */
#define SKEW_POLICY_ADAFACTOR 4

/* ---- per-tensor flags ------------------------------------------------------ */
#define SKEW_F_NO_DECAY 1u /* exempt this tensor from weight decay (the router always is) */
/* Weights and gradient are fp32 (4-byte aligned), as the paper keeps the norms and
 * the router (App. A): the new weight is the fp32 update itself, with no dithered
 * cast. Such a tensor takes the scalar tile path (it is small). */
#define SKEW_F_FP32 2u

/* ---- second-moment kinds reported by skew_tensor_info ----------------------- */
#define SKEW_KIND_FULL 0     /* exact second moment v (router, vectors)  */
#define SKEW_KIND_FACTORED 1 /* row / column factors R, C (Eq. 1)        */

typedef struct skew_handle skew_handle_t; /* opaque */

/*
 * One parameter tensor. The tensor id used by the dither is its index in the
 * array passed to skew_create.
 *   weight : device pointer to the bf16 weights (fp32 with SKEW_F_FP32),
 *            contiguous row-major, updated in place by skew_step; 2-byte
 *            aligned, 4-byte for fp32 (16-byte alignment enables the
 *            vectorised bf16 path). Borrowed: must stay valid while the handle
 *            is bound.
 *   grad   : device pointer to the gradient, the weights' type, shape and
 *            layout; read only. Borrowed like `weight`.
 *   shape  : shape[0] = rows n (>= 1); shape[1] = columns m (>= 1) when
 *            ndim >= 2, ignored when ndim == 1.
 *   ndim   : 1 (vector), 2 (matrix) or 3 (a stack of `stack` matrices of
 *            n x m, contiguous: matrix e starts at element e*n*m).
 *   tier   : SKEW_TIER_*.
 *   flags  : SKEW_F_* bits.
 *   stack  : the number of matrices when ndim == 3 (>= 1); 0 otherwise.
 *
 * A stacked tensor (experts kept as one (E, n, m) array) is stepped as E
 * matrices, each with its own second-moment factors, RMS and clip factor
 * (Algorithm 1 is stated per matrix; the paper counts 128 x 3 expert
 * matrices); its dither uses the descriptor's index as tensor id and the flat
 * index e*n*m + i*m + j over the whole stack.
 */
typedef struct {
    void *weight;
    const void *grad;
    int64_t shape[2];
    int32_t ndim;
    int32_t tier;
    uint32_t flags;
    uint32_t stack;
} skew_param_desc_t;

/*
 * Hyper-parameters (Algorithm 1, App. A Table 9). The paper's defaults are
 * beta1 = 0.9, beta2 = 0.999, eps = 1e-8, clip_d = 1, weight_decay = 0.05.
 *   0 <= beta1 < 1, 0 <= beta2 < 1, eps > 0 (finite), clip_d > 0 (finite),
 *   weight_decay >= 0 (finite), policy = SKEW_POLICY_*.
 */
typedef struct {
    float beta1;
    float beta2;
    float eps;
    float clip_d;
    float weight_decay;
    int32_t policy;
} skew_hparams_t;

/*
 * Where one tensor's state lives inside the caller's state buffer (offsets in
 * fp32 elements from its start; -1 when the tensor has no such array).
 *   m_offset: momentum M (numel floats, row-major)
 *   v_offset: exact second moment v (numel floats)
 *   r_offset: R (rows floats), c_offset: C (cols floats)
 */
typedef struct {
    int32_t kind;       /* SKEW_KIND_*                                         */
    int32_t momentum;   /* 1 if the tensor keeps fp32 momentum                 */
    int32_t decay;      /* 1 if weight decay applies                           */
    int32_t vectorized; /* 1 if the 16-byte vector path serves it (after bind) */
    int64_t rows, cols, numel;
    int64_t m_offset, v_offset, r_offset, c_offset;
    int32_t rowpath;    /* 1 if phase A runs on whole rows and sum(U^2) needs no  */
                        /* second pass over G unless a clamp may bind (bilinear) */
    int32_t stack;      /* matrices of a stacked tensor (ndim 3), else 0; then   */
                        /* rows / cols are one matrix's, numel the whole stack's, */
                        /* and each state array holds the E matrices' in order   */
} skew_tensor_info_t;

/*
 * Plans the step for `n_params` tensors (n_params >= 0; 0 gives a handle whose
 * step does nothing). Validates every descriptor and the hyper-parameters,
 * resolves each tensor's tier policy (kind / momentum / decay), lays out the
 * optimizer state and the workspace. Host only: no CUDA call, no device
 * memory touched. On success *out receives a new handle (free with
 * skew_destroy). Errors: SKEW_EINVAL (reason in skew_last_error(NULL)),
 * SKEW_ENOMEM.
 */
int skew_create(const skew_param_desc_t *params, int32_t n_params, const skew_hparams_t *hp,
                skew_handle_t **out);

/* Frees the handle's host metadata (not the caller's device memory). NULL is a no-op. */
int skew_destroy(skew_handle_t *h);

/*
 * Exact optimizer-state size in bytes: 4 * (sum over momentum tensors of numel
 * + sum over factored tensors of (rows + cols) + sum over exact-second-moment
 * tensors of numel) -- Eq. 2 with the vectors' full v of Table 5. The caller
 * allocates exactly this many bytes of device memory for the state. 0 for NULL.
 */
size_t skew_state_bytes(const skew_handle_t *h);

/*
 * Scratch the step needs besides the state (per-tensor partial sums, scalars,
 * descriptor and tile tables). Not optimizer state. 0 for NULL.
 */
size_t skew_workspace_bytes(const skew_handle_t *h);

/*
 * Binds caller-owned device buffers to the handle: `state` (exactly
 * skew_state_bytes bytes) and `workspace` (exactly skew_workspace_bytes bytes),
 * both 256-byte aligned device pointers (NULL allowed when the size is 0).
 * Uploads the descriptor and tile tables into the workspace and zero-fills the
 * state (the paper's initial M = v = R = C = 0), enqueued on `stream`.
 * May be called again to re-bind (the state is zeroed again).
 * Errors: SKEW_EINVAL (size / alignment), SKEW_ECUDA.
 */
int skew_bind(skew_handle_t *h, void *state, size_t state_bytes, void *workspace, size_t workspace_bytes,
              void *stream);

/*
 * Enqueues one SkewAdam step over every tensor on `stream`: reads each
 * gradient, updates the state and writes the bf16 weights in place.
 *   step : global 1-based step t (bias corrections beta^t; the dither counter
 *          uses its low 32 bits). All tensors advance together.
 *   lr   : the scheduled learning rate eta_t (finite, >= 0); the caller owns
 *          the schedule.
 *   seed : 64-bit dither seed.
 * Asynchronous: device-side problems are reported by skew_sync_status.
 * Errors: SKEW_ESTATE (not bound), SKEW_EINVAL (step < 1, lr not finite or
 * negative), SKEW_ECUDA (launch failure).
 */
int skew_step(skew_handle_t *h, int64_t step, float lr, uint64_t seed, void *stream);

/*
 * skew_step with the trainer's global gradient-norm clip applied inside the step.
 * The paper's training setup (Sec. 4) and App. A Table 9 clip the global gradient
 * norm at 1.0 before the optimizer step: G <- gamma * G with gamma = min(1, c /
 * ||G||). Here the step sees gamma * G without a separate pass over the gradients:
 * gamma enters only the moving-average increments ((1 - beta1) gamma on g,
 * (1 - beta2) gamma^2 on g^2) and the update coefficient of momentum-free tensors,
 * so the step reads and writes exactly the bytes of skew_step. (Scaling the learning
 * rate instead is not the same step: the second moments are moving averages of the
 * scaled gradient.)
 *   grad_scale : device pointer to one fp32 gamma (finite), computed by the caller
 *                on `stream` before this call (e.g. from its norm reduction); read
 *                by the kernels, never by the host; 4-byte aligned. NULL means
 *                gamma = 1, and then the call is skew_step, bit for bit; so is a
 *                pointer to 1.0f.
 * Other arguments, asynchrony and errors as skew_step (SKEW_EINVAL also for a
 * misaligned grad_scale).
 */
int skew_step_scaled(skew_handle_t *h, int64_t step, float lr, uint64_t seed, const float *grad_scale, void *stream);

/*
 * Synchronises `stream` and reports the device-side status word of the last
 * steps: SKEW_OK, or SKEW_ETIMEOUT if a bounded device wait gave up (the word
 * is cleared by this call). Errors: SKEW_ESTATE, SKEW_ECUDA.
 */
int skew_sync_status(skew_handle_t *h, void *stream);

/*
 * Self-test of the failure path of the bounded device waits: enqueues on
 * `stream` one thread that waits, exactly as the whole-row kernels wait for a
 * copied chunk, on an mbarrier phase that nothing completes. The wait gives up
 * after its poll limit (about two seconds at most) and records the timeout in
 * the handle's status word, so the next skew_sync_status returns SKEW_ETIMEOUT
 * and clears it; the context stays usable and later steps are unaffected.
 * Asynchronous. Errors: SKEW_EINVAL (null), SKEW_ESTATE (not bound),
 * SKEW_ECUDA (launch failure).
 */
int skew_selftest_wait_timeout(skew_handle_t *h, void *stream);

/*
 * Per-tensor scalars of the last completed step, for inspection and tests:
 * out[0] = mean(R) (factored tensors, else 0), out[1] = sum of U^2 over the
 * tensor, out[2] = RMS(U), out[3] = clip factor 1/max(1, RMS/d). Synchronises
 * `stream`. Errors: SKEW_EINVAL (tid), SKEW_ESTATE, SKEW_ECUDA.
 */
int skew_tensor_scalars(skew_handle_t *h, int32_t tid, double out[4], void *stream);

/* As skew_tensor_scalars, for matrix `e` of stacked tensor `tid` (e = 0 for any
 * other tensor). Errors: SKEW_EINVAL (tid, e), SKEW_ESTATE, SKEW_ECUDA. */
int skew_matrix_scalars(skew_handle_t *h, int32_t tid, int32_t e, double out[4], void *stream);

/* Resolved policy and state offsets of tensor `tid`. Errors: SKEW_EINVAL. */
int skew_tensor_info(const skew_handle_t *h, int32_t tid, skew_tensor_info_t *out);

/*
 * Benchmark support: launch timing. After skew_profile_begin(h, n), each of the
 * next n calls of skew_step records a CUDA event before and after each timed
 * launch it makes on the step's stream (seven grouped launches, named by
 * skew_kernel_name; a phase with no work times ~0; no extra
 * synchronisation). skew_profile_end(h, ms, cap, &steps, &launches)
 * synchronises, writes the durations in milliseconds row-major into
 * ms[steps][launches] (up to cap values), releases the events and stops
 * recording. skew_kernel_name(k) names timed launch k of a step.
 * Errors: SKEW_EINVAL, SKEW_ECUDA.
 */
int skew_profile_begin(skew_handle_t *h, int32_t max_steps);
int skew_profile_end(skew_handle_t *h, double *ms, int64_t cap, int32_t *n_steps, int32_t *n_kernels);
const char *skew_kernel_name(int32_t k);

/*
 * A step over ONE tensor that allocates nothing -- no cudaMalloc / cudaFree, no
 * allocating library routine, no host heap. The paper has no counterpart; this
 * is a deployment convenience.
 *
 * Who needs it: callers that cannot allocate device memory when they step the
 * optimizer, e.g. code running while a framework's caching allocator holds all
 * free memory, plugins that are only handed pre-sized buffers, or runtimes that
 * forbid allocation after start-up. skew_bind needs a caller-allocated
 * workspace; this entry point instead uses a fixed scratch array compiled into
 * the library: SKEW_NOALLOC_SCRATCH_BYTES of device memory on every GPU that
 * loads the library, held until the process exits. That is enough for one
 * 4,096-wide matrix of up to about 65,000 rows with momentum (the paper's
 * 50,304 x 4,096 embedding fits; the whole-row partials take 256 bytes per row)
 * and about twice that without (128 bytes per row on its 256-row tiles); larger
 * tensors are rejected with SKEW_ETOOBIG before any work is enqueued.
 *
 * Arguments: weight / grad as in skew_param_desc_t (device, bf16 or with
 * SKEW_F_FP32 fp32, row-major);
 * ndim, rows, cols, tier, flags as in skew_param_desc_t; hp as for
 * skew_create; state: this tensor's fp32 state, exactly state_bytes =
 * 4 * ((momentum ? numel : 0) + (full second moment ? numel : rows + cols))
 * bytes, laid out [M][v] or [M][R][C] (absent arrays take no room), 4-byte
 * aligned, zero-filled by the caller before the first step; tensor_id: the id
 * fed to the dither (use the tensor's index in a skew_create list to get the
 * same bits as skew_step); step, lr, seed as for skew_step; stream: a
 * cudaStream_t. Updates weight and state in place, asynchronously on stream,
 * with the same kernels and results as skew_step on a one-tensor handle.
 *
 * Every call looks up the array's device address on the current device with
 * cudaGetSymbolAddress. The first such lookup on a device may load the
 * library's device code there: make the first call on each device before any
 * stream capture. All calls on a device share the one array: calls whose
 * work overlaps on the GPU (different streams, or other host threads) race
 * and corrupt each other's results -- serialise them. The array keeps the
 * last call's contents; everything a step needs zeroed is cleared by the step.
 *
 * Device-side failures: the whole-row kernels' bounded waits (as for
 * skew_step) record a copy that did not land in a status word at the start of
 * the array. No call clears it; skew_noalloc_sync_status reads it. A step
 * whose wait gave up has left some tiles of that tensor unwritten.
 * Errors: SKEW_EINVAL (argument or state size), SKEW_ETOOBIG, SKEW_ECUDA.
 */
#define SKEW_NOALLOC_SCRATCH_BYTES (16u * 1024u * 1024u)
int skew_step_tensor_noalloc(void *weight, const void *grad, int32_t ndim, int64_t rows, int64_t cols, int32_t tier,
                             uint32_t flags, const skew_hparams_t *hp, void *state, size_t state_bytes,
                             uint32_t tensor_id, int64_t step, float lr, uint64_t seed, void *stream);

/*
 * Synchronises `stream` and reports the no-alloc status word of the current
 * device: SKEW_OK, or SKEW_ETIMEOUT if a bounded device wait of a
 * skew_step_tensor_noalloc call gave up since the word was last read (the word
 * is then cleared, with a memset enqueued on `stream` and waited for). Uses no
 * allocation (a 4-byte device-to-host copy). Errors: SKEW_ECUDA.
 */
int skew_noalloc_sync_status(void *stream);

/*
 * Self-test of that failure path: enqueues on `stream` one thread that waits,
 * exactly as the whole-row kernels wait for a copied chunk, on an mbarrier
 * phase that nothing completes; after its poll limit (about two seconds) the
 * wait gives up and sets the no-alloc status word, so the next
 * skew_noalloc_sync_status returns SKEW_ETIMEOUT. Nothing else is touched and
 * the context stays usable. Asynchronous. Errors: SKEW_ECUDA.
 */
int skew_noalloc_selftest_wait_timeout(void *stream);

/*
 * Kernel launches one skew_step performs (its grouped launches over item
 * tables; 0 for NULL or an empty handle).
 */
int64_t skew_launches_per_step(const skew_handle_t *h);

/* Number of tensors the handle plans for (0 for NULL). */
int32_t skew_num_tensors(const skew_handle_t *h);

/* One-line reason for the last failure on `h` (or of skew_create when h is NULL). */
const char *skew_last_error(const skew_handle_t *h);

#ifdef __cplusplus
}
#endif

#endif /* SKEWADAM_H_ */
