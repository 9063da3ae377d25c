/*
 * dpo_muon.h -- one-step-delayed Muon with Error Feedback, C ABI.
 *
 * Alg. 2 (Sec. 4) of arXiv 2606.30634, for the 2-D weight matrices of a
 * model on one GPU (sm_103a). Per call, for each matrix X (rows x cols) and
 * its stale gradient G_{t-1} (evaluated at the stashed weights):
 *
 *   G^ = s G,  s = min(1, max_norm / (||G||_2 + 1e-6))   global clipping over
 *        all matrices of the context, or over every parameter through a
 *        shared clip source (App. E.1), 1 when max_grad_norm <= 0
 *   M  = mu M + (1 - mu) G^          momentum as an exponential moving average
 *        (Sec. 2.2's convention for the momentum decay mu; Alg. 2 prints the
 *        two weights the other way round)
 *   O  = NewtonSchulz(M)             the quintic iteration of Muon (Jordan et
 *        al. 2024): X_0 = M / (||M||_F + eps), on the transpose when
 *        rows > cols; ns_steps times A = X X^T, B = b A + c A A,
 *        X <- a X + B X. Every iterate is held in bf16 and every product
 *        accumulates in fp32 on the tensor cores.
 *   U  = lr (r O + wd X_t),  r = rms_scale sqrt(max(rows, cols)) when
 *        rms_scale > 0 (update RMS 0.2, Sec. 2.1, with the scaling of Liu et
 *        al. 2025), else r = 1 (Alg. 2 as printed); wd = 0 for matrices
 *        without DPO_WD_ON
 *   X_{t+1} = X_t - U                           standard delayed rule, t <= 1
 *   X_{t+1} = X_t - U - lambda (U - U_prev)     Error Feedback (Eq. (1);
 *        Alg. 2 is lambda = 1: X_t - 2 U_{t-1} + U_{t-2})
 *   stash := X_t,  U_prev := U,  param := bf16(X_{t+1})
 *   With correction DPO_CORR_SAPIPE_SAME (SAPipe-WP, App. B.1) the weights take
 *   the standard rule and the stash receives the predicted point X_t - U_prev.
 *   With DPO_CORR_SAPIPE_UPDATED (App. B.1, updated state) the same, but
 *   U_prev := U', the step taken once more on the same gradient from the
 *   updated momentum: M' = mu M + (1 - mu) G^ (not kept in M),
 *   O' = NewtonSchulz(M'), U' = lr (r O' + wd X_{t+1}). M' is formed in the
 *   history buffer, so the prediction needs no extra memory; it doubles the
 *   step's tensor-core work.
 *
 * The k-th dpo_muon_step is Alg. 1's iteration t = k (t = 0 only sets
 * X_1 = X_0). With delay = 0 the same update runs on gradients of the latest
 * weights, without stash or correction.
 *
 * Layout and ownership. The caller owns every buffer of a dpo_matrix: device
 * memory of the current device, row-major, 32-byte aligned, no overlaps, kept
 * alive and in place until dpo_muon_destroy. The library allocates, in
 * dpo_muon_init, the Newton-Schulz workspace (bf16, for every matrix: two
 * copies of the iterate, its transpose and two Gram-sized matrices, each
 * dimension padded to a multiple of 256) plus a small table; no other call
 * allocates or synchronizes the host. All launches go to the stream passed in.
 *
 * Errors. Every call returns DPO_OK (0) or a negative DPO_E* code from
 * dpo.h. dpo_muon_last_error gives the message of the last failing call on a
 * context (NULL context: the last dpo_muon_init failure of this thread).
 */
#ifndef DPO_MUON_H
#define DPO_MUON_H

#include <stdint.h>

#include "dpo.h"

#ifdef __cplusplus
extern "C" {
#endif

/* One weight matrix. */
typedef struct {
    void *param;        /* bf16 latest weights X_{t+1} (rows x cols), or NULL */
    float *master;      /* fp32 master weights */
    float *mom;         /* fp32 momentum M */
    void *stash;        /* stash (stash dtype) = X_t, what the next forward reads; NULL only
                           for delay 0 */
    float *ef;          /* fp32 U_prev (Error Feedback history), or NULL (standard rule) */
    const void *grad;   /* gradient (grad dtype) */
    int64_t rows, cols; /* >= 0; a matrix with no elements is skipped */
    uint32_t flags;     /* DPO_WD_ON; DPO_SYNC: trained synchronously even while the run
                           is delayed (no stash, no correction; its gradient comes from
                           the latest weights, as for dpo_tensor) */
} dpo_matrix;

typedef struct {
    float momentum;       /* mu in [0, 1) (Sec. 2.1: 0.95) */
    float weight_decay;   /* decay on X_t (Alg. 2) */
    float ef_lambda;      /* lambda of the EF correction; used when ef buffers are given */
    float max_grad_norm;  /* > 0: global clipping threshold; <= 0: off */
    float ns_a, ns_b, ns_c; /* quintic coefficients (3.4445, -4.7750, 2.0315) */
    float ns_eps;         /* added to ||M||_F (1e-7) */
    float rms_scale;      /* 0.2: match the update RMS; 0: no scaling */
    int ns_steps;         /* iterations, 0..16 (5) */
    int delay;            /* 1: one-step-delayed (Alg. 1 / 2); 0: synchronous */
    int correction;       /* with ef buffers: DPO_CORR_EF (lambda-scaled Error Feedback),
                             DPO_CORR_SAPIPE_SAME (SAPipe-WP with the same state, App. B.1:
                             the weights take the standard rule, the stash receives the
                             prediction point X_t - U_prev, the history U) or
                             DPO_CORR_SAPIPE_UPDATED (the same with the history U', the
                             updated-state prediction above) */
} dpo_muon_hparams;

typedef struct dpo_muon_ctx dpo_muon_ctx;

/*
 * Validate the matrices and settings, allocate the workspace and (init_mode
 * DPO_INIT_FRESH) enqueue the start state: mom = 0, ef = 0, stash and param
 * := master. Every matrix needs master, mom and grad; a stash when delay = 1
 * (unless DPO_SYNC); ef for all matrices or none. param_dtype is DPO_BF16; stash_dtype and
 * grad_dtype are DPO_F32 or DPO_BF16. Returns DPO_OK and *out, or DPO_EINVAL,
 * DPO_EALIGN, DPO_EDTYPE, DPO_ENOMEM or DPO_ECUDA and *out = NULL.
 */
int dpo_muon_init(dpo_muon_ctx **out, const dpo_matrix *mats, int n, dpo_dtype stash_dtype,
                  dpo_dtype grad_dtype, const dpo_muon_hparams *hp, int init_mode,
                  void *cuda_stream);

/*
 * One iteration with learning rate lr (> 0) for every matrix, enqueued on
 * stream: the norm pass when clipping, the momentum pass, the
 * normalisation pass, 3 ns_steps GEMM launches per matrix shape (or, when
 * some shape's launches are short, per set of up to four shapes sharing each
 * launch) and the update pass. Returns DPO_OK, DPO_EINVAL or DPO_ECUDA.
 */
int dpo_muon_step(dpo_muon_ctx *ctx, float lr, void *cuda_stream);

/*
 * Switch between synchronous (0) and one-step-delayed (1) training
 * (synchronous start and cooldown, Sec. 3.1, App. A.10), as dpo_set_delay does
 * for the elementwise path: entering delayed training stashes the current
 * weights of every matrix without DPO_SYNC and zeroes the update history, so
 * Alg. 1 restarts (its first delayed call takes the standard rule). Needs a
 * stash for every such matrix (DPO_ESTATE otherwise). Returns DPO_OK,
 * DPO_EINVAL, DPO_ESTATE or DPO_ECUDA.
 */
int dpo_muon_set_delay(dpo_muon_ctx *ctx, int delay, void *cuda_stream);

/*
 * Newton-Schulz output O of the last step for matrix i, as a strided bf16
 * view into the workspace (valid until the next dpo_muon_step): element
 * (r, c) of O (rows x cols) is at (*ptr)[r * *ld + c]. With the SAPipe-WP
 * updated state in delayed training it is the prediction's output O'.
 */
int dpo_muon_last_update(const dpo_muon_ctx *ctx, int i, const void **ptr, int64_t *ld);

/*
 * Copy that output for matrix i into dst (device, bf16, rows x cols
 * row-major), enqueued on cuda_stream. Returns DPO_OK, DPO_EINVAL or
 * DPO_ECUDA.
 */
int dpo_muon_copy_update(const dpo_muon_ctx *ctx, int i, void *dst, void *cuda_stream);

/*
 * Error bits of the tensor-core pipeline since init (a wait inside a GEMM
 * that gave up after one second; 0 when healthy). Synchronizes with the
 * context's last work. Returns DPO_OK or DPO_ECUDA.
 */
int dpo_muon_get_status(dpo_muon_ctx *ctx, uint32_t *bits);

/*
 * The global gradient norm shared with other contexts (see dpo_grad_sqnorm
 * and dpo_set_clip_source in dpo.h, which these follow): add this context's
 * sum of G^2 over all its matrices to *d_sumsq, and clip later steps from
 * the total. Returns DPO_OK, DPO_EINVAL, DPO_ESTATE or DPO_ECUDA.
 */
int dpo_muon_grad_sqnorm(dpo_muon_ctx *ctx, double *d_sumsq, void *cuda_stream);
int dpo_muon_set_clip_source(dpo_muon_ctx *ctx, const double *d_sumsq);

/*
 * Clear the error bits that dpo_muon_get_status reports (enqueued on
 * cuda_stream). Returns DPO_OK, DPO_EINVAL or DPO_ECUDA.
 */
int dpo_muon_clear_status(dpo_muon_ctx *ctx, void *cuda_stream);

/*
 * Test hook for the failure path: in each of the next `launches` Newton-Schulz
 * GEMM launches, the MMA lane's first accumulator wait targets a phase that
 * no arrival completes. The wait gives up after its one-second limit, every
 * role of the kernel leaves through its own bounded wait, and the launch ends
 * with error bits set (its output is not computed); later launches run
 * normally. Returns DPO_OK or DPO_EINVAL (launches < 0).
 */
int dpo_muon_test_stall(dpo_muon_ctx *ctx, int launches);

/*
 * Capturable mode for CUDA graphs, as dpo_set_capturable (dpo.h): the step
 * counters move to device memory, and each dpo_muon_step forms its update's
 * lr, lr wd and EF start (t >= 2) on the device, so a step captured in a
 * graph replays correctly; lr from lr_source (a device float) when set, else
 * dpo_muon_step's argument. The counter calls and dpo_muon_set_delay
 * synchronize the device and do not belong inside a capture; with
 * dpo_muon_set_timing on, the step records events whose host bookkeeping a
 * replay does not repeat, so leave timing off while capturing. Returns
 * DPO_OK, DPO_EINVAL or DPO_ECUDA.
 */
int dpo_muon_set_capturable(dpo_muon_ctx *ctx, int on, const float *lr_source,
                            void *cuda_stream);

/* Calls consumed so far (k), and restore after loading a checkpoint. */
int dpo_muon_get_step(const dpo_muon_ctx *ctx, int64_t *k);
int dpo_muon_set_step(dpo_muon_ctx *ctx, int64_t k);

/*
 * k at the start of the current delayed phase, as dpo_get_phase_start /
 * dpo_set_phase_start (dpo.h): Alg. 1's t = k - k0 decides where EF starts.
 * Save it with k; restore it after dpo_muon_set_step. Returns DPO_OK or
 * DPO_EINVAL.
 */
int dpo_muon_get_phase_start(const dpo_muon_ctx *ctx, int64_t *k0);
int dpo_muon_set_phase_start(dpo_muon_ctx *ctx, int64_t k0);

/*
 * Tensor-core work of one step, summed over the matrices (r x w the
 * orientation with r <= w, unpadded), two flops per multiply-add:
 * ns_steps (r (r + 1) w + r (r + 1) r + 2 r^2 w), the first two terms being
 * the unique entries of the symmetric products X X^T and A A; twice that
 * with the SAPipe-WP updated state in delayed training.
 */
int dpo_muon_flops(const dpo_muon_ctx *ctx, double *flops);

/*
 * Measurement of the tensor-core work: with on != 0, each later dpo_muon_step
 * brackets its Newton-Schulz GEMM launches (every shape's chain) with a pair
 * of CUDA events recorded on its stream. dpo_muon_get_gemm_time waits
 * for those events, returns the summed milliseconds and the number of GEMM
 * launches since the previous read, and starts a new count. Returns DPO_OK,
 * DPO_EINVAL or DPO_ECUDA.
 */
int dpo_muon_set_timing(dpo_muon_ctx *ctx, int on);
int dpo_muon_get_gemm_time(dpo_muon_ctx *ctx, double *ms, int64_t *launches);

/* Bytes of the Newton-Schulz workspace the context allocated. */
int dpo_muon_workspace_bytes(const dpo_muon_ctx *ctx, int64_t *bytes);

const char *dpo_muon_last_error(const dpo_muon_ctx *ctx);
/* Free the context and its workspace (after the work on its stream is done). */
void dpo_muon_destroy(dpo_muon_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* DPO_MUON_H */
