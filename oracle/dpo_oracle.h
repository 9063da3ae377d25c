/*
 * dpo_oracle.h -- plain CPU oracle of the one-step-delayed optimizer step.
 *
 * TEST INFRASTRUCTURE. Only the tests, the package smoke check and the CPU
 * baseline leg of the benchmark load this library. The product library
 * (libdpo) never links, loads or calls it, and the two share no code.
 *
 * Method (arXiv 2606.30634, "One-Step Gradient Delay is Not a Barrier for
 * Large-Scale Asynchronous Pipeline Parallel LLM Pretraining"):
 *   Alg. 1 (Delayed Gradient Update), Sec. 2: at iteration t the optimizer
 *     statistics are updated with the stale gradient g_{t-1}, the step
 *     u_{t-1}(g_{t-1}) is formed, and
 *        x_{t+1} = x_t - u_{t-1}                       (standard, or t <= 1)
 *        x_{t+1} = x_t - 2 u_{t-1} + u_{t-2}           (Error Feedback)
 *   Eq. (1), Sec. 3.2: the Error-Feedback update above.
 *   App. A.4 (Error Feedback Coefficient Ablation): the lambda-scaled form
 *        x_{t+1} = x_t - u_{t-1} - lambda (u_{t-1} - u_{t-2}),
 *     lambda = 0 standard delayed training, lambda = 1 Eq. (1).
 *   u is AdamW with beta = (0.9, 0.95) (Sec. 2.1), EMA convention
 *     m_t = beta m_{t-1} + (1 - beta) g_t (Sec. 2.2), decoupled weight decay
 *     on the current iterate x_t (Alg. 2: U_{t-1} = eta (O_{t-1} + lambda X_t)),
 *     and global gradient-norm clipping at 1.0 (Sec. 2, App. E.1).
 *
 * Every arithmetic operation is done in double. After each step every state
 * buffer is rounded to its storage format (double: no rounding; fp32; bf16
 * round-to-nearest-even from the fp32 master), exactly as a GPU holding the
 * same buffers in those formats would store them.
 */
#ifndef DPO_ORACLE_H
#define DPO_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Storage formats of the state buffers. */
enum { ORACLE_F64 = 0, ORACLE_F32 = 1, ORACLE_BF16 = 2 };

/* Update rules u. ADAMW is the optimizer of the hot path. SGD (u = lr g)
 * exists only so that tests can check the delay/EF driver of Alg. 1 apart
 * from Adam. NADAM, LION and ADAN are the other elementwise optimizers the
 * paper benchmarks under one-step delay (Sec. 2.2, Tab. main_results); the
 * paper cites them without restating them, so each follows its published
 * form, with decoupled weight decay on the current iterate as for AdamW:
 *   NADAM  Dozat 2016, as torch.optim.NAdam with decoupled_weight_decay:
 *          momentum schedule mu_k = beta1 (1 - 0.5 * 0.96^(k psi)),
 *          u = lr ( (1 - mu_k) / (1 - prod_{i<=k} mu_i) g / d
 *               + mu_{k+1} / (1 - prod_{i<=k+1} mu_i) m / d + wd x ),
 *          d = sqrt(v / (1 - beta2^k)) + eps.
 *   LION   Chen et al. 2023: c = beta1 m + (1 - beta1) g,
 *          u = lr (sign(c) + wd x), then m = beta2 m + (1 - beta2) g
 *          (v unused).
 *   ADAN   Xie et al. 2022, in its authors' distributed form: with
 *          diff = g - g_prev (0 at the first gradient),
 *          m = beta1 m + (1 - beta1) g, v = beta2 v + (1 - beta2) diff,
 *          n = beta3 n + (1 - beta3) (g + beta2 diff)^2,
 *          u = lr ( (m / (1 - beta1^k) + beta2 v / (1 - beta2^k))
 *                   / (sqrt(n / (1 - beta3^k)) + eps) + wd x ), g_prev = g. */
enum {
    ORACLE_RULE_ADAMW = 0,
    ORACLE_RULE_SGD = 1,
    ORACLE_RULE_NADAM = 2,
    ORACLE_RULE_LION = 3,
    ORACLE_RULE_ADAN = 4
};

/* Staleness correction applied when an update-history buffer is given
 * (u_prev != NULL) under delay == 1:
 *   EF             Eq. (1) / App. A.4: x_{t+1} = x_t - u - lambda (u - u_prev);
 *                  the stash receives x_t.
 *   SAPIPE_SAME    App. B.1, SAPipe-WP with the same optimizer state: the
 *                  weights follow the standard rule x_{t+1} = x_t - u, and the
 *                  next forward/backward reads the prediction made at the
 *                  previous step, x~_t = x_t - u_{t-2} (the stash). u_prev
 *                  then holds u.
 *   SAPIPE_UPDATED App. B.1, SAPipe-WP with the updated state: as SAPIPE_SAME,
 *                  but the prediction update is the rule's step at the next
 *                  time index on the same gradient, from the state after the
 *                  real update (for AdamW a temporary second blend of g into m
 *                  and v, bias corrections at k + 1, decay on x_{t+1}; NAdam
 *                  also takes its momentum schedule at k + 1; Lion the sign of
 *                  the beta1 blend of its updated momentum; Adan a zero
 *                  gradient difference, its previous gradient being g itself);
 *                  u_prev holds that prediction update. */
enum { ORACLE_CORR_EF = 0, ORACLE_CORR_SAPIPE_SAME = 1, ORACLE_CORR_SAPIPE_UPDATED = 2 };

typedef struct {
    double lr;            /* learning rate eta of the call */
    double beta1, beta2;  /* EMA coefficients of m and v */
    double eps;           /* added to sqrt(v_hat) */
    double weight_decay;  /* decoupled decay coefficient */
    double ef_lambda;     /* lambda of the EF correction; 0 = standard */
    double beta3;         /* ADAN: EMA coefficient of n */
    double momentum_decay;/* NADAM: psi of the momentum schedule */
    double dc_lambda;     /* DC-ASGD compensation strength (Sec. 3.1); 0 = off */
    int delay;            /* 1 = one-step-delayed (Alg. 1), 0 = synchronous */
    int rule;             /* ORACLE_RULE_* */
    int correction;       /* ORACLE_CORR_*, used when u_prev != NULL and delay == 1 */
    int x_store;          /* storage of master x, m, v and u_prev (F64 or F32) */
    int stash_store;      /* storage of the stash (F64, F32 or BF16) */
    int param_store;      /* storage of the latest-weights copy (F64, F32, BF16) */
} oracle_hparams;

/*
 * One call of the delayed step over n elements (one flat tensor or the
 * concatenation of several; the step is elementwise).
 *
 *   k          number of gradients consumed including this one (>= 1): the
 *              index of Adam's bias corrections.
 *   t          Alg. 1 iteration of this call within the current delayed
 *              phase (>= 1): t = k when training is delayed from the start;
 *              after a switch from synchronous to delayed training Alg. 1
 *              restarts, its first delayed call being t = 1 (t = 0 only sets
 *              x_1 = x_0, u_{-1} = 0). The EF correction applies from t = 2.
 *   g          the gradient evaluated at the stash (the stale weights), as
 *              doubles holding values of the gradient storage format.
 *              With dc_lambda != 0 and delay == 1 it is first corrected by
 *              DC-ASGD's Taylor term (Zheng et al. 2017; Sec. 3.1):
 *              g~ = g + dc_lambda g^2 (x_t - stash), the stash holding the
 *              weights the gradient was evaluated at (after clipping).
 *   clip_scale multiplier applied to g (1 when clipping is off), from
 *              oracle_clip_coef().
 *   wd_on      per-element 0/1 mask for weight decay, or NULL (decay on all).
 *   delay_on   per-element 0/1 mask under delay == 1: 0 marks elements of a
 *              tensor trained synchronously (its gradient evaluated at the
 *              latest weights: no stash, no correction, history untouched), as
 *              in WPipe (App. B.2) or a synchronous LM head (App. A.9); NULL
 *              means every element is delayed.
 *   x, m, v    master weights and Adam moments, updated in place.
 *   u_prev     update-history buffer: u_{t-2} on entry and u_{t-1} on return
 *              (SAPIPE_UPDATED: the prediction updates). NULL selects the
 *              standard delayed rule; with a buffer and delay == 1 the
 *              correction hp->correction runs (EF with lambda = 0 gives the
 *              standard result).
 *   stash      receives the weights the next gradient is evaluated at: x_t,
 *              or the SAPipe prediction point; may be NULL when delay == 0
 *              (the latest weights are read).
 *   param      receives the new latest weights x_{t+1}, or NULL.
 *   n, g_prev  ADAN's third moment and previous (corrected) gradient; NULL
 *              for the other rules.
 *
 * Returns 0, or -1 on an invalid argument.
 */
int oracle_step(int64_t n, int64_t k, int64_t t, const oracle_hparams *hp,
                const double *g, double clip_scale, const uint8_t *wd_on,
                const uint8_t *delay_on, double *x, double *m, double *v,
                double *u_prev, double *stash, double *param, double *n3,
                double *g_prev);

/* Sum of g_i^2 in double over n elements (fixed order: blocks of 65536
 * elements summed left to right, block sums added left to right). */
double oracle_sqnorm(int64_t n, const double *g);

/* Same, with the gradient given as bf16 bit patterns or as fp32 values. */
double oracle_sqnorm_bf16(int64_t n, const uint16_t *g_bits);
double oracle_sqnorm_f32(int64_t n, const float *g);

/* Clip coefficient min(1, max_norm / (sqrt(sqnorm) + 1e-6)); 1 when
 * max_norm <= 0 (clipping off). */
double oracle_clip_coef(double sqnorm, double max_norm);

/* Number of threads the element loops use (OpenMP), 1 without OpenMP. */
int oracle_num_threads(void);
/* Set it (n > 0; no effect without OpenMP). Results do not depend on it:
 * the element loops are independent and the sums run in fixed blocks. */
void oracle_set_num_threads(int n);

/* Round a value to a storage format (ORACLE_F64 / F32 / BF16). */
double oracle_round(double x, int store);
/* out[i] = oracle_round(in[i], store) for i < n (in and out may alias). */
void oracle_round_n(int64_t n, const double *in, double *out, int store);

/* Quadratic workload f(w) = 1/2 sum a_i (w_i - w*_i)^2 (the noisy diagonal
 * quadratic used to emulate delayed training):
 *   grad_i = a_i (w_i - wstar_i) + noise_i, rounded to `store`;
 *   returns the loss 1/2 sum a_i (w_i - wstar_i)^2 at w. */
double oracle_quadratic(int64_t n, const double *a, const double *wstar,
                        const double *w, const double *noise, int store,
                        double *grad_out);

/*
 * Delayed Muon (Alg. 2, Sec. 4), one weight matrix at a time.
 *
 * Per call, with G the (clipped) stale gradient of a rows x cols matrix:
 *   M <- mu M + (1 - mu) G                 momentum as an EMA (Sec. 2.2's
 *                                          convention for the momentum decay
 *                                          mu; Alg. 2 prints the two weights
 *                                          the other way round)
 *   O  = NewtonSchulz(M)                   oracle_newton_schulz below
 *   U  = lr (s O + wd X_t),  s = rms_scale sqrt(max(rows, cols)) when
 *        rms_scale > 0 (update RMS 0.2, Sec. 2.1, as Liu et al. 2025 scale
 *        it), else s = 1 (Alg. 2 as printed)
 *   X_{t+1} = X_t - U - lambda_eff (U - U_prev)   (Alg. 2 with EF is
 *        lambda = 1: X_t - 2 U_{t-1} + U_{t-2}; lambda_eff = 0 at t = 1)
 * The stash receives X_t and the history buffer U, exactly as oracle_step
 * does for the elementwise rules.
 */
typedef struct {
    double lr;             /* eta of the call */
    double momentum;       /* mu */
    double weight_decay;   /* decay on X_t (Alg. 2) */
    double ef_lambda;      /* lambda of the EF correction; 0 = standard */
    double ns_a, ns_b, ns_c;  /* coefficients of the quintic iteration */
    int ns_steps;          /* iterations */
    double ns_eps;         /* added to ||M||_F before normalising */
    double rms_scale;      /* see above; 0 = no scaling */
    int ns_store;          /* storage of every Newton-Schulz matrix: F64 or BF16 */
    int delay;             /* 1 = one-step-delayed, 0 = synchronous */
    int correction;        /* ORACLE_CORR_EF, ORACLE_CORR_SAPIPE_SAME (App. B.1: the
                              weights take the standard rule, the stash receives the
                              prediction point X_t - U_prev, the history U) or
                              ORACLE_CORR_SAPIPE_UPDATED (the same, but the history
                              receives the prediction update: Alg. 2's step once more
                              on G_{t-1} from the updated momentum, with a second
                              Newton-Schulz and decay on X_{t+1}) */
    int x_store;           /* storage of X, M and U_prev (F64 or F32) */
    int stash_store;       /* storage of the stash */
    int param_store;       /* storage of the latest-weights copy */
} oracle_muon_hparams;

/*
 * Newton-Schulz orthogonalisation of a rows x cols matrix M (row-major), the
 * quintic iteration of Jordan et al. 2024 that Muon uses:
 *   X_0 = M / (||M||_F + eps), taken as its transpose when rows > cols so
 *         that the Gram matrix is the smaller one;
 *   A   = X X^T,  B = b A + c A A,  X <- a X + B X     (`steps` times);
 *   O   = X (transposed back when rows > cols).
 * store = ORACLE_BF16 rounds X_0 and every A, B and X to bf16 when it is
 * formed (each from exact products of its rounded inputs), which is how the
 * iteration runs in bf16 on tensor cores; ORACLE_F64 keeps them exact.
 * Writes O (rows x cols). Returns 0, or -1 on bad arguments or no memory.
 */
int oracle_newton_schulz(int64_t rows, int64_t cols, const double *M, double eps, double a,
                         double b, double c, int steps, int store, double *O);

/*
 * One call of delayed Muon on one matrix (see above). t is the Alg. 1
 * iteration within the current delayed phase (>= 1). x, mom are updated in
 * place; u_prev (history, or NULL for the standard rule), stash (needed when
 * delay == 1) and param (or NULL) as in oracle_step. o_out, when not NULL,
 * receives the Newton-Schulz output O of the real step. Returns 0, or -1 on
 * bad arguments or no memory.
 */
int oracle_muon_step(int64_t rows, int64_t cols, int64_t t, const oracle_muon_hparams *hp,
                     const double *g, double clip_scale, double *x, double *mom,
                     double *u_prev, double *stash, double *param, double *o_out);

#ifdef __cplusplus
}
#endif
#endif /* DPO_ORACLE_H */
