/*
 * dpo.h -- one-step-delayed AdamW step with Error Feedback, C ABI.
 *
 * The per-parameter optimizer step of arXiv 2606.30634 ("One-Step Gradient
 * Delay is Not a Barrier for Large-Scale Asynchronous Pipeline Parallel LLM
 * Pretraining"), for one GPU (sm_103a):
 *
 *   Alg. 1 (Sec. 2), Delayed Gradient Update. Iteration t updates the
 *   optimizer statistics with the stale gradient g_{t-1}, forms the update
 *   u_{t-1}(g_{t-1}) and applies
 *       x_{t+1} = x_t - u_{t-1}                          standard, or t <= 1
 *       x_{t+1} = x_t - u_{t-1} - lambda (u_{t-1} - u_{t-2})   Error Feedback
 *   (Eq. (1), Sec. 3.2 for lambda = 1; App. A.4 for general lambda).
 *   u is AdamW (Sec. 2.1: beta = (0.9, 0.95); Sec. 2.2: EMA moments) with
 *   decoupled weight decay on the current iterate x_t (Alg. 2) and optional
 *   global gradient-norm clipping (App. E.1):
 *       g^ = s g,  s = min(1, max_norm / (||g||_2 + 1e-6))  (1 without clipping)
 *       m  = beta1 m + (1 - beta1) g^,   v = beta2 v + (1 - beta2) g^2
 *       u  = lr ( (m / (1 - beta1^k)) / (sqrt(v / (1 - beta2^k)) + eps) + wd x_t )
 *   k counts the gradients consumed (the k-th dpo_step is iteration t = k;
 *   iteration t = 0 only sets x_1 = x_0 since u_{-1} = 0).
 *
 *   Weight-version stash (Sec. 2, PipeDream-2BW keeps one extra weight
 *   version): after each step the stash holds x_t, the weights before the
 *   update, and the latest copy holds x_{t+1}. The next forward/backward reads
 *   the stash (dpo_read_weights(DPO_STALE)), so the gradient the next
 *   dpo_step consumes was evaluated one version behind the weights it updates.
 *
 * Layout and ownership. The caller owns and allocates every buffer named in
 * a dpo_tensor (32-byte aligned, not overlapping one another), keeps them
 * alive until dpo_destroy, and may not move them. The optimizer state
 * (master, m, v, stash, EF buffer) is device memory of the current device.
 * grad and param may be device memory too, or host memory the GPU addresses
 * directly: pinned memory mapped at the same address (cudaHostAlloc), or
 * pageable memory on a device with pageable-memory access (NVLink-C2C
 * systems). The fused kernel then reads the gradients from and writes the new
 * weights to host memory itself, over the host link, with no staging copy;
 * the step is then bound by that link (2 B per parameter each way for bf16).
 * The host must not touch those buffers while a step is in flight. The
 * library owns only its context: a device copy of the tensor table and a few
 * hundred bytes of device scratch per SM for the gradient norm. All launches
 * go to the stream passed in (a cudaStream_t, NULL for the legacy default
 * stream); dpo_step never synchronizes the host.
 *
 * Errors. Every call returns DPO_OK (0) or a negative DPO_E* code; nothing
 * aborts. dpo_last_error gives a message for the last failing call on a
 * context (or, with NULL, for the last dpo_init failure of this thread).
 */
#ifndef DPO_H
#define DPO_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DPO_ABI_VERSION 1

/* Status codes. */
#define DPO_OK 0
#define DPO_EINVAL (-1)  /* bad argument: NULL or overlapping buffers, bad size or value */
#define DPO_EALIGN (-2)  /* a buffer is not 32-byte aligned */
#define DPO_EDTYPE (-3)  /* unsupported dtype or dtype combination */
#define DPO_ECUDA (-4)   /* a CUDA runtime call or launch failed */
#define DPO_ESTATE (-5)  /* the context is not in a state that allows the call */
#define DPO_ENOMEM (-6)  /* the library's own small device allocation failed */

typedef enum { DPO_F32 = 0, DPO_BF16 = 1 } dpo_dtype;

/* dpo_tensor.flags */
#define DPO_WD_ON 1u     /* apply weight decay to this tensor */
#define DPO_SYNC 2u      /* train this tensor synchronously even while the run is
                          * delayed: its gradient is evaluated at the latest
                          * weights, no stash is written and no correction runs
                          * (WPipe's second half, App. B.2; the synchronous LM
                          * head of App. A.9) */

/* dpo_read_weights(which) */
#define DPO_STALE 0      /* what the next forward/backward reads (the stash) */
#define DPO_LATEST 1     /* the newest weights x_{t+1} */

/* dpo_init(init_mode) */
#define DPO_INIT_FRESH 0   /* m = v = 0, EF buffer = 0, stash and param := master */
#define DPO_INIT_RESUME 1  /* keep every buffer as given (restore with dpo_set_step) */

/* dpo_get_flags() bits */
#define DPO_FLAG_NONFINITE 1u  /* a clipped step saw a non-finite gradient norm */

/* dpo_hparams.correction: the staleness correction run when the table has
 * update-history (EF) buffers and delay == 1.
 *   DPO_CORR_EF              Eq. (1) / App. A.4: x_{t+1} = x_t - u - lambda (u - u_prev);
 *                            the stash receives x_t.
 *   DPO_CORR_SAPIPE_SAME     App. B.1, SAPipe-WP weight prediction with the same
 *                            optimizer state: the weights take the standard rule
 *                            x_{t+1} = x_t - u, and the stash (what the next
 *                            forward/backward reads) receives the prediction made
 *                            at the previous step, x_t - u_prev; the buffer then
 *                            holds u.
 *   DPO_CORR_SAPIPE_UPDATED  App. B.1 with the updated state: as above, but the
 *                            buffer holds the prediction update: the rule's step
 *                            at the next time index on the same gradient, from
 *                            the state the real update left (for AdamW the
 *                            moments blended with g once more, bias corrections
 *                            at k + 1, decay on x_{t+1}; NAdam also takes its
 *                            momentum schedule at k + 1, Lion the sign of the
 *                            beta1 blend of its updated momentum, Adan a zero
 *                            gradient difference), not kept in the statistics.
 *                            Every rule. */
#define DPO_CORR_EF 0
#define DPO_CORR_SAPIPE_SAME 1
#define DPO_CORR_SAPIPE_UPDATED 2

/* dpo_hparams.optimizer: the update rule u. AdamW is the hot path's; the
 * others are the elementwise optimizers the paper also benchmarks under
 * one-step delay (Sec. 2.2, Tab. main_results), in their published forms with
 * decoupled weight decay on x_t:
 *   DPO_OPT_ADAMW  as above.
 *   DPO_OPT_NADAM  Dozat 2016 (as torch.optim.NAdam, decoupled decay):
 *                  mu_k = beta1 (1 - 0.5 * 0.96^(k momentum_decay)),
 *                  u = lr ((1-mu_k)/(1-prod_{i<=k} mu_i) g/d
 *                      + mu_{k+1}/(1-prod_{i<=k+1} mu_i) m/d + wd x_t),
 *                  d = sqrt(v / (1 - beta2^k)) + eps.
 *   DPO_OPT_LION   Chen et al. 2023: u = lr (sign(beta1 m + (1-beta1) g) + wd x_t),
 *                  m = beta2 m + (1 - beta2) g; v is not used (may be NULL).
 *   DPO_OPT_ADAN   Xie et al. 2022 (its authors' distributed form): diff = g - g_prev
 *                  (0 at the first gradient), m = beta1 m + (1-beta1) g,
 *                  v = beta2 v + (1-beta2) diff, n = beta3 n + (1-beta3)(g + beta2 diff)^2,
 *                  u = lr ((m/(1-beta1^k) + beta2 v/(1-beta2^k)) / (sqrt(n/(1-beta3^k)) + eps)
 *                      + wd x_t); needs the n and grad_prev buffers.
 * Every rule takes every correction (DPO_CORR_*). */
/* dpo_hparams.stash_mode. PipeDream-2BW keeps two weight versions (Sec. 2):
 *   DPO_STASH_COPY      the step writes x_t into the stash buffer and
 *                       x_{t+1} into the param buffer (every layout).
 *   DPO_STASH_PINGPONG  with bf16 param and stash buffers, the stale version
 *                       x_t is bitwise the bf16 weights the previous call
 *                       wrote, so the two buffers of a delayed tensor swap
 *                       roles instead: call k writes x_{k+1} into the buffer
 *                       that held x_{k-1}, and no stash is written (2 bytes per
 *                       parameter less). After call k the param buffer holds
 *                       the latest weights when k is even and the stash buffer
 *                       when k is odd; dpo_read_weights resolves the roles.
 *                       Needs param_dtype = stash_dtype = DPO_BF16, device
 *                       param buffers, and the standard rule or EF (the SAPipe
 *                       corrections stash a prediction, not a previous version).
 *                       Synchronously trained tensors (DPO_SYNC) keep their
 *                       weights in the param buffer. */
#define DPO_STASH_COPY 0
#define DPO_STASH_PINGPONG 1

#define DPO_OPT_ADAMW 0
#define DPO_OPT_NADAM 1
#define DPO_OPT_LION 2
#define DPO_OPT_ADAN 3

typedef struct {
    float beta1;          /* first-moment EMA coefficient, [0, 1) */
    float beta2;          /* second-moment EMA coefficient, [0, 1) */
    float eps;            /* added to sqrt(v_hat), >= 0 */
    float weight_decay;   /* decoupled decay (tensors with DPO_WD_ON), >= 0 */
    float ef_lambda;      /* lambda of the EF correction (tables with EF buffers) */
    float max_grad_norm;  /* > 0: global-norm clipping threshold; <= 0: off */
    int delay;            /* 1: one-step-delayed with stash; 0: synchronous */
    int correction;       /* DPO_CORR_* (tables with EF buffers, delay == 1) */
    int optimizer;        /* DPO_OPT_* */
    float beta3;          /* DPO_OPT_ADAN: EMA coefficient of n, [0, 1) */
    float momentum_decay; /* DPO_OPT_NADAM: psi of the momentum schedule, >= 0 */
    /* DC-ASGD (Sec. 3.1): when != 0, delayed tensors' gradients are first
     * compensated, g~ = g + dc_lambda g^2 (x_t - stash), the stash holding the
     * weights the gradient was evaluated at (after clipping). */
    float dc_lambda;
    int stash_mode;       /* DPO_STASH_* */
} dpo_hparams;

typedef struct {
    /* Latest weights x_{t+1} in the param dtype. With DPO_BF16 params this is
     * written every step (round to nearest even from master). With DPO_F32
     * params it must be NULL: the fp32 master is then the latest copy. */
    void *param;
    float *master;     /* fp32 master weights, read and written */
    float *m;          /* Adam first moment, fp32, read and written */
    float *v;          /* second moment, fp32, read and written (Adan: the averaged
                        * gradient difference; Lion: unused, may be NULL) */
    /* Stale weights in the stash dtype: x_t after each step (the SAPipe
     * prediction point under those corrections). Required for tensors without
     * DPO_SYNC when delay == 1; with delay == 0 it may be NULL, and giving it
     * lets dpo_set_delay switch the run to delayed training later. */
    void *stash;
    /* Update-history (EF) buffer (fp32): u_{t-2} on entry, u_{t-1} on return
     * (the prediction update under DPO_CORR_SAPIPE_UPDATED). NULL on every
     * tensor: standard delayed rule. Non-NULL on every tensor: the correction
     * hparams.correction (EF with lambda = 0 gives the standard result). */
    float *ef;
    /* The gradient the step consumes, in the grad dtype, evaluated at the
     * stash (delay == 1) or at the latest weights (delay == 0). Read only. */
    const void *grad;
    float *n;          /* DPO_OPT_ADAN: third moment (fp32), else NULL */
    float *grad_prev;  /* DPO_OPT_ADAN: previous corrected gradient (fp32), else NULL */
    int64_t numel;     /* elements, >= 0; 0 is allowed and skipped */
    uint32_t flags;    /* DPO_WD_ON or 0 */
} dpo_tensor;

typedef struct dpo_ctx dpo_ctx;

/*
 * Create a context over n_tensors tensors (table is copied; the buffers it
 * points to are not). Validates every pointer (NULL, 32-byte alignment,
 * overlap, residency as above), dtype and hyperparameter. With DPO_INIT_FRESH
 * it then enqueues, on cuda_stream, the Alg. 1 start state: m = v = 0, EF
 * buffer = 0 (u_{-1} = 0), stash := x_0 and param := x_0 from master, and
 * sets k = 0. Supported dtypes: param F32|BF16, stash F32|BF16, grad
 * F32|BF16. Returns DPO_OK and *out, or an error and *out = NULL.
 */
int dpo_init(dpo_ctx **out, const dpo_tensor *table, int n_tensors,
             dpo_dtype param_dtype, dpo_dtype stash_dtype, dpo_dtype grad_dtype,
             const dpo_hparams *hp, int init_mode, void *cuda_stream);

/*
 * stash := the current master weights (rounded to the stash dtype), and the
 * bf16 param copy := master. Used at start-up and when delayed training is
 * (re)entered after synchronous steps. Enqueued on cuda_stream.
 */
int dpo_stash(dpo_ctx *ctx, void *cuda_stream);

/*
 * One delayed step (Alg. 1 iteration t = k + 1) with learning rate lr:
 * consumes every tensor's grad, updates master, m, v (and the EF buffer),
 * writes stash := x_t (delay == 1) and param := x_{t+1}, then k += 1.
 * With clipping, first computes the global gradient norm over all tensors
 * (deterministic, fixed reduction order), or takes it from the clip source
 * set by dpo_set_clip_source. Asynchronous on cuda_stream, no
 * host synchronization, no allocation. lr must be finite and >= 0.
 */
int dpo_step(dpo_ctx *ctx, float lr, void *cuda_stream);

/*
 * Capturable mode, for CUDA graphs. A dpo_step captured into a graph and
 * replayed must not reuse the scalars of the call it was captured at (the
 * bias corrections and NAdam/Adan factors depend on k, EF's lambda on
 * t = k - k0, the ping-pong roles on the parity of t). With on != 0 the
 * counters (k, the phase start, NAdam's running product) move to device
 * memory and every dpo_step enqueues a one-thread kernel that forms that
 * call's scalars from them, in the same double arithmetic as the host path,
 * and advances them; the fused kernel reads the scalars from there. The
 * learning rate is read from lr_source (a device float, 4-byte aligned, kept
 * alive while set; write it between replays for a schedule) or, when
 * lr_source is NULL, is dpo_step's lr argument (fixed in a captured graph).
 * dpo_step then enqueues launches only and can be captured; the calls that
 * report or change the counters (dpo_get_step, dpo_set_step, dpo_get/
 * set_phase_start, dpo_set_delay, dpo_read_weights with the ping-pong stash)
 * synchronize the device first, so they do not belong inside a capture.
 * on = 0 brings the counters back to the host (synchronizing). The hyper-
 * parameters and the delay mode are fixed in a captured graph: change them
 * outside it and capture again. Returns DPO_OK, DPO_EINVAL or DPO_ECUDA.
 */
int dpo_set_capturable(dpo_ctx *ctx, int on, const float *lr_source, void *cuda_stream);

/*
 * One global gradient norm across contexts and ranks. Clipping scales every
 * gradient by one coefficient from the norm over all parameters (App. E.1);
 * when those parameters are split over several contexts (an AdamW context
 * for the vectors and embeddings beside a dpo_muon context for the
 * matrices, or one shard per rank of a partitioned set), each context adds
 * its share and all of them clip from the total:
 *
 *   dpo_grad_sqnorm: enqueue on cuda_stream  *d_sumsq += sum of g^2  over
 *     this context's gradients (fp64; the same fixed-order reduction as
 *     dpo_step's own norm pass, whatever max_grad_norm is). d_sumsq is
 *     caller-owned device memory, 8-byte aligned; contributions to it must
 *     be ordered (one stream, or events), and the caller zeroes it before
 *     the first. A context with no elements adds nothing.
 *   dpo_set_clip_source: with d_sumsq != NULL, every later dpo_step clips
 *     from sqrt(*d_sumsq) (read on the device when the step runs) instead of
 *     computing its own norm: coefficient min(1, max_grad_norm /
 *     (sqrt(*d_sumsq) + 1e-6)). NULL goes back to the context's own norm.
 *     Needs max_grad_norm > 0 (DPO_ESTATE otherwise). The pointer must stay
 *     valid while it is set.
 *
 * Summing the per-rank values of *d_sumsq (an all-reduce) between the two
 * calls is the one exchange a partitioned step needs. Both return DPO_OK,
 * DPO_EINVAL, DPO_ESTATE or DPO_ECUDA.
 */
int dpo_grad_sqnorm(dpo_ctx *ctx, double *d_sumsq, void *cuda_stream);
int dpo_set_clip_source(dpo_ctx *ctx, const double *d_sumsq);

/*
 * Switch the run between synchronous (delay = 0) and one-step-delayed
 * (delay = 1) training: synchronous start and synchronous cooldown (Sec. 3.1,
 * App. A.10). Entering delayed training enqueues stash := master for every
 * delayed tensor and zeroes the update-history buffers, so Alg. 1 restarts at
 * the next dpo_step: the gradient it consumes is evaluated at the stash (the
 * current weights), its update uses the standard rule, and EF applies from the
 * following call. Needs stash buffers for every tensor without DPO_SYNC
 * (DPO_ESTATE otherwise). Leaving it takes effect at the next dpo_step, whose
 * gradient must then be evaluated at the latest weights. No host
 * synchronization.
 */
int dpo_set_delay(dpo_ctx *ctx, int delay, void *cuda_stream);

/*
 * Pointer and dtype of tensor `tensor`'s stale (DPO_STALE) or latest
 * (DPO_LATEST) weights. Under delay == 0, and for DPO_SYNC tensors, both name
 * the latest weights. The pointer is one of the caller's own buffers; no copy
 * is made.
 */
int dpo_read_weights(const dpo_ctx *ctx, int which, int tensor,
                     const void **ptr, dpo_dtype *dtype);

/* Step counter k (gradients consumed so far); set it when resuming. */
int dpo_get_step(const dpo_ctx *ctx, int64_t *k);
int dpo_set_step(dpo_ctx *ctx, int64_t k);

/*
 * The value of k at which the current delayed phase began (0 for a run that
 * is delayed from the start; dpo_set_delay(1) sets it to the current k).
 * Alg. 1's iteration index is t = k - k0: it decides where EF starts (t >= 2)
 * and, with the ping-pong stash, which buffer holds which weights (the parity
 * of t). A checkpoint saves it with k and the delay mode, and a resumed
 * context restores it after dpo_set_step; 0 <= k0 <= k. Returns DPO_OK or
 * DPO_EINVAL.
 */
int dpo_get_phase_start(const dpo_ctx *ctx, int64_t *k0);
int dpo_set_phase_start(dpo_ctx *ctx, int64_t k0);

/*
 * Diagnostics of the last clipped step: the DPO_FLAG_* bits raised since the
 * previous dpo_get_flags (reading clears them), the global gradient norm and
 * the clip coefficient used. Synchronizes cuda_stream (not for the hot
 * loop). Any output pointer may be NULL.
 */
int dpo_get_flags(dpo_ctx *ctx, uint32_t *flags, double *grad_norm,
                  float *clip_scale, void *cuda_stream);

/*
 * Bytes one dpo_step must move through memory by the layout of the context
 * (algorithmic, not measured): *step_bytes for the fused step over all
 * tensors, *norm_bytes for the gradient-norm pass (0 without clipping, or
 * with a clip source: dpo_grad_sqnorm then reads the gradients once more).
 */
int dpo_algorithmic_bytes(const dpo_ctx *ctx, int64_t *step_bytes,
                          int64_t *norm_bytes);

/* Launch geometry chosen at init: CTAs of the fused step and of the norm
 * pass (both persistent: a multiple of the SM count for sets large enough to
 * fill the GPU) and threads per CTA of the fused step. */
int dpo_launch_config(const dpo_ctx *ctx, int *step_ctas, int *norm_ctas,
                      int *threads);

/*
 * Per-kernel timing, for measurement. With timing on, every dpo_step that
 * launches work records three CUDA events on its stream: before the
 * gradient-norm pass (or the clip-coefficient kernel of a clip source), before
 * the fused step, and after it. dpo_get_timing waits for the recorded events,
 * returns the summed milliseconds of the norm interval (*norm_ms, 0 without
 * clipping) and of the fused-step interval (*step_ms) over the *calls timed
 * calls since the last read, and starts a new count. The events' host
 * bookkeeping is not repeated by a CUDA-graph replay: leave timing off while
 * capturing. Returns DPO_OK, DPO_EINVAL or DPO_ECUDA.
 */
int dpo_set_timing(dpo_ctx *ctx, int on);
int dpo_get_timing(dpo_ctx *ctx, double *norm_ms, double *step_ms, int64_t *calls);

/*
 * Gradient norm without device allocation.
 *
 * The paper has no counterpart to this entry point; it serves callers that
 * cannot call cudaMalloc. A training framework whose caching allocator has
 * already reserved the GPU's memory cannot let a library take more behind
 * its back, and a latency-critical loop cannot take the device-wide
 * synchronization cudaMalloc and cudaFree may imply; dpo_init allocates a
 * small device block, so such callers use this instead. It computes what
 * the clipped dpo_step computes before its update, for one contiguous
 * gradient buffer: the global L2 norm (deterministic for a given numel:
 * fixed chunking and summation order) and the clip coefficient
 * min(1, max_grad_norm / (norm + 1e-6)): 1 when max_grad_norm <= 0, 1 for
 * numel == 0 (norm 0), NaN when the norm is NaN (as the clipped dpo_step).
 *
 *   grad          device buffer of numel gradients (grad_dtype F32 or BF16),
 *                 32-byte aligned; 0 <= numel <= DPO_NOALLOC_MAX_NUMEL.
 *   max_grad_norm finite (dpo_init's rule for its hyperparameters); a
 *                 non-finite value gives DPO_EINVAL.
 *   norm_out      device pointer, receives the norm (double, 8-byte aligned).
 *   clip_out      device pointer, receives the coefficient (float).
 *
 * Its scratch is a fixed file-scope device array of
 * DPO_NOALLOC_MAX_CHUNKS partial sums (128 KiB), one per chunk of at most
 * DPO_NOALLOC_CHUNK_ELEMS elements (smaller chunks for smaller buffers, so
 * they still spread over the SMs); every GPU that loads the library holds
 * it until the process exits. Larger inputs are rejected with DPO_EINVAL.
 * The call allocates nothing: it enqueues one small memset (clearing the
 * scratch's counter, which must start at zero) and one kernel on
 * cuda_stream. The first call on each device looks up the scratch array's
 * device address (cudaGetSymbolAddress) with that device current and keeps
 * it until the process exits, which assumes the device's primary context
 * lives that long (no cudaDeviceReset in between); make that first call
 * before any stream capture. All calls share the scratch array, which keeps
 * the last call's contents, so calls whose kernels overlap on the GPU
 * (different streams or host threads on one device) race on it.
 * Returns DPO_OK, DPO_EINVAL, DPO_EALIGN, DPO_EDTYPE or DPO_ECUDA.
 */
#define DPO_NOALLOC_CHUNK_ELEMS (1 << 20)
#define DPO_NOALLOC_MAX_CHUNKS 16384
#define DPO_NOALLOC_MAX_NUMEL ((int64_t)DPO_NOALLOC_MAX_CHUNKS * DPO_NOALLOC_CHUNK_ELEMS)

int dpo_grad_norm_noalloc(const void *grad, int64_t numel, dpo_dtype grad_dtype,
                          float max_grad_norm, double *norm_out, float *clip_out,
                          void *cuda_stream);

/*
 * Test hook for the allocation-failure paths, process-wide: of the library's
 * next device allocations (dpo_init makes one, dpo_muon_init one or two: its
 * table, then its workspace), let `after` succeed and make the following
 * `count` fail as if the device were out of memory (the call then returns
 * DPO_ENOMEM and frees what it had allocated). count = 0 turns the hook off.
 * Returns DPO_OK or DPO_EINVAL (a negative argument).
 */
int dpo_test_fail_allocs(int after, int count);

/* Message of the last failing call on ctx (NULL ctx: last dpo_init failure of
 * the calling thread). Never NULL; owned by the library. */
const char *dpo_last_error(const dpo_ctx *ctx);

/* Free the context and its device scratch (after the work enqueued on it has
 * finished or been synchronized by the caller). NULL is ignored. */
void dpo_destroy(dpo_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* DPO_H */
