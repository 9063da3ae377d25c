/*
 * dpo_oracle.c -- plain CPU oracle of the one-step-delayed AdamW step with
 * update-level Error Feedback (arXiv 2606.30634).
 *
 * TEST INFRASTRUCTURE. Loaded only by the tests, the package smoke check and
 * the benchmark's CPU-baseline leg; the product library never uses it.
 *
 * The code follows the paper's statement step by step, one element at a
 * time, in double precision, with no fusion or reordering: see the header
 * for the passages each step comes from. The element loop may run on several
 * OpenMP threads; every element is independent, so the result does not depend
 * on the thread count. Sums run in a fixed order.
 */
#include "dpo_oracle.h"

#include <math.h>
#include <stddef.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_num_threads(int n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* bf16: 8 significant bits, the exponent range of fp32. Round half to even
 * on the value's own ulp; below 2^-126 the ulp is fixed at 2^-133. */
static double round_bf16(double x)
{
    if (isnan(x) || isinf(x) || x == 0.0)
        return x;
    int e;
    (void)frexp(fabs(x), &e);          /* |x| = f * 2^e, f in [0.5, 1) */
    if (e < -125)
        e = -125;                      /* subnormal range: ulp 2^-133 */
    double q = ldexp(fabs(x), 8 - e);  /* |x| in units of one bf16 ulp */
    q = nearbyint(q);                  /* default mode: ties to even */
    double r = ldexp(q, e - 8);
    if (r >= 0x1p128)
        r = INFINITY;
    return copysign(r, x);
}

double oracle_round(double x, int store)
{
    switch (store) {
    case ORACLE_F32:
        return (double)(float)x;
    case ORACLE_BF16:
        return round_bf16(x);
    default:
        return x;
    }
}

void oracle_round_n(int64_t n, const double *in, double *out, int store)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = oracle_round(in[i], store);
}

int oracle_step(int64_t n, int64_t k, int64_t t, const oracle_hparams *hp,
                const double *g, double clip_scale, const uint8_t *wd_on,
                const uint8_t *delay_on, double *x, double *m, double *v,
                double *u_prev, double *stash, double *param, double *n3,
                double *g_prev)
{
    if (n < 0 || k < 1 || t < 1 || hp == NULL || (n > 0 && (g == NULL || x == NULL)))
        return -1;
    const int rule = hp->rule;
    if (rule < ORACLE_RULE_ADAMW || rule > ORACLE_RULE_ADAN)
        return -1;
    if (rule != ORACLE_RULE_SGD && n > 0 && m == NULL)
        return -1;
    if ((rule == ORACLE_RULE_ADAMW || rule == ORACLE_RULE_NADAM || rule == ORACLE_RULE_ADAN) &&
        n > 0 && v == NULL)
        return -1;
    if (rule == ORACLE_RULE_ADAN && n > 0 && (n3 == NULL || g_prev == NULL))
        return -1;
    if (hp->delay == 1 && n > 0 && stash == NULL)
        return -1;

    /* A staleness correction is active for delayed training with an
     * update-history buffer; the lambda-scaled EF form reduces to the
     * standard rule at lambda = 0. */
    const int use_ef = (hp->delay == 1 && u_prev != NULL);
    const int corr = use_ef ? hp->correction : ORACLE_CORR_EF;
    if (corr != ORACLE_CORR_EF && corr != ORACLE_CORR_SAPIPE_SAME &&
        corr != ORACLE_CORR_SAPIPE_UPDATED)
        return -1;
    /* Alg. 1: the standard rule is used for t <= 1 even under EF. */
    const int ef_now = use_ef && corr == ORACLE_CORR_EF && t >= 2;
    const double lam = hp->ef_lambda;

    /* Bias corrections of Adam at the k-th gradient, and at the (k+1)-th for
     * the SAPipe updated-state prediction. */
    const double bc1 = 1.0 - pow(hp->beta1, (double)k);
    const double bc2 = 1.0 - pow(hp->beta2, (double)k);
    const double bc1_next = 1.0 - pow(hp->beta1, (double)(k + 1));
    const double bc2_next = 1.0 - pow(hp->beta2, (double)(k + 1));
    const double bc3 = 1.0 - pow(hp->beta3, (double)k);
    const double bc3_next = 1.0 - pow(hp->beta3, (double)(k + 1));

    /* NAdam's momentum schedule mu_i = beta1 (1 - 0.5 * 0.96^(i psi)) and its
     * running products up to k and k + 1. */
    double mu_prod = 1.0;
    for (int64_t i = 1; i <= k; ++i)
        mu_prod *= hp->beta1 * (1.0 - 0.5 * pow(0.96, (double)i * hp->momentum_decay));
    const double mu_k = hp->beta1 * (1.0 - 0.5 * pow(0.96, (double)k * hp->momentum_decay));
    const double mu_next =
        hp->beta1 * (1.0 - 0.5 * pow(0.96, (double)(k + 1) * hp->momentum_decay));
    const double mu_prod_next = mu_prod * mu_next;
    /* ... and one index further, for the SAPipe updated-state prediction
     * (NAdam's step at index k + 1 uses mu_{k+1}, mu_{k+2} and the products
     * up to them). */
    const double mu_next2 =
        hp->beta1 * (1.0 - 0.5 * pow(0.96, (double)(k + 2) * hp->momentum_decay));
    const double mu_prod_next2 = mu_prod_next * mu_next2;

#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        const double wd = (wd_on == NULL || wd_on[i]) ? hp->weight_decay : 0.0;
        const double xt = x[i];
        /* An element of a synchronously trained tensor: no stash, no
         * correction, its history untouched. */
        const int delayed = hp->delay == 1 && (delay_on == NULL || delay_on[i]);
        const int hist_i = use_ef && delayed;
        double gi = clip_scale * g[i];
        /* DC-ASGD: first-order Taylor compensation of the stale gradient,
         * with the stash still holding the weights it was evaluated at. */
        if (hp->dc_lambda != 0.0 && delayed)
            gi = gi + hp->dc_lambda * gi * gi * (xt - stash[i]);

        /* Update the optimizer statistics with g_{t-1} and form u_{t-1}. */
        double u, mi = 0.0, vi = 0.0;
        if (rule == ORACLE_RULE_ADAMW) {
            mi = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;
            const double m_hat = mi / bc1;
            const double v_hat = vi / bc2;
            u = hp->lr * (m_hat / (sqrt(v_hat) + hp->eps) + wd * xt);
            m[i] = oracle_round(mi, hp->x_store);
            v[i] = oracle_round(vi, hp->x_store);
        } else if (rule == ORACLE_RULE_NADAM) {
            mi = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;
            const double d = sqrt(vi / bc2) + hp->eps;
            u = hp->lr * ((1.0 - mu_k) / (1.0 - mu_prod) * gi / d +
                          mu_next / (1.0 - mu_prod_next) * mi / d + wd * xt);
            m[i] = oracle_round(mi, hp->x_store);
            v[i] = oracle_round(vi, hp->x_store);
        } else if (rule == ORACLE_RULE_LION) {
            const double c = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
            const double sgn = c > 0.0 ? 1.0 : (c < 0.0 ? -1.0 : 0.0);
            u = hp->lr * (sgn + wd * xt);
            m[i] = oracle_round(hp->beta2 * m[i] + (1.0 - hp->beta2) * gi, hp->x_store);
        } else if (rule == ORACLE_RULE_ADAN) {
            const double diff = k == 1 ? 0.0 : gi - g_prev[i];
            mi = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * diff;
            const double w = gi + hp->beta2 * diff;
            const double ni = hp->beta3 * n3[i] + (1.0 - hp->beta3) * w * w;
            const double d = sqrt(ni / bc3) + hp->eps;
            u = hp->lr * ((mi / bc1 + hp->beta2 * vi / bc2) / d + wd * xt);
            m[i] = oracle_round(mi, hp->x_store);
            v[i] = oracle_round(vi, hp->x_store);
            n3[i] = oracle_round(ni, hp->x_store);
            g_prev[i] = oracle_round(gi, hp->x_store);
        } else {
            u = hp->lr * (gi + wd * xt);
        }

        /* Apply it: standard delayed rule, or the EF correction. */
        double xn;
        if (!(ef_now && delayed))
            xn = xt - u;
        else
            xn = xt - u - lam * (u - u_prev[i]);

        /* The stash: the weights the next gradient is evaluated at. Under
         * EF (and the standard rule) that is the pre-update x_t, one step
         * behind the latest; under SAPipe-WP it is the prediction made at the
         * previous step, x_t - u_prev, a weight in the master's format
         * rounded to the stash format. */
        if (delayed) {
            if (corr == ORACLE_CORR_EF)
                stash[i] = oracle_round(xt, hp->stash_store);
            else
                stash[i] = oracle_round(oracle_round(xt - u_prev[i], hp->x_store),
                                        hp->stash_store);
        }
        if (hist_i) {
            double hist = u;
            if (corr == ORACLE_CORR_SAPIPE_UPDATED && rule == ORACLE_RULE_ADAMW) {
                /* The optimizer step once more on g_{t-1}, from the state the
                 * real update left (the statistics as stored), at the next
                 * time index, decaying x_{t+1}. */
                const double m2 = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
                const double v2 = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;
                hist = hp->lr * ((m2 / bc1_next) / (sqrt(v2 / bc2_next) + hp->eps) +
                                 wd * oracle_round(xn, hp->x_store));
            } else if (corr == ORACLE_CORR_SAPIPE_UPDATED) {
                /* The same for the other rules: each rule's own step at index
                 * k + 1 on g_{t-1}, from the statistics this call stored, with
                 * decay on x_{t+1}. */
                const double x_next = oracle_round(xn, hp->x_store);
                if (rule == ORACLE_RULE_NADAM) {
                    const double nm = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
                    const double nv = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;
                    const double d2 = sqrt(nv / bc2_next) + hp->eps;
                    hist = hp->lr * ((1.0 - mu_next) / (1.0 - mu_prod_next) * gi / d2 +
                                     mu_next2 / (1.0 - mu_prod_next2) * nm / d2 + wd * x_next);
                } else if (rule == ORACLE_RULE_LION) {
                    /* the sign of the beta1 blend of the updated momentum */
                    const double c2 = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
                    const double s2 = c2 > 0.0 ? 1.0 : (c2 < 0.0 ? -1.0 : 0.0);
                    hist = hp->lr * (s2 + wd * x_next);
                } else if (rule == ORACLE_RULE_ADAN) {
                    /* the stored previous gradient is now g_{t-1} itself, so
                     * the next step's gradient difference is zero (up to that
                     * store's rounding) */
                    const double ad = gi - g_prev[i];
                    const double am = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;
                    const double av = hp->beta2 * v[i] + (1.0 - hp->beta2) * ad;
                    const double aw = gi + hp->beta2 * ad;
                    const double an = hp->beta3 * n3[i] + (1.0 - hp->beta3) * aw * aw;
                    const double d2 = sqrt(an / bc3_next) + hp->eps;
                    hist = hp->lr * ((am / bc1_next + hp->beta2 * av / bc2_next) / d2 +
                                     wd * x_next);
                } else {   /* SGD: no statistics */
                    hist = hp->lr * (gi + wd * x_next);
                }
            }
            u_prev[i] = oracle_round(hist, hp->x_store);
        }
        x[i] = oracle_round(xn, hp->x_store);
        if (param != NULL)
            param[i] = oracle_round(x[i], hp->param_store);
    }
    return 0;
}

#define ORACLE_SUM_BLOCK 65536

/* Fixed-order sum of squares: per-block sums (blocks may run on different
 * threads), then the block sums added left to right. */
#define DEFINE_SQNORM(NAME, T, WIDEN)                                       \
    double NAME(int64_t n, const T *g)                                      \
    {                                                                       \
        if (n <= 0)                                                         \
            return 0.0;                                                     \
        const int64_t nb = (n + ORACLE_SUM_BLOCK - 1) / ORACLE_SUM_BLOCK;   \
        double total = 0.0;                                                 \
        double *part = (double *)malloc(sizeof(double) * (size_t)nb);       \
        if (part == NULL)                                                   \
            return NAN;                                                     \
        _Pragma("omp parallel for schedule(static)")                        \
        for (int64_t b = 0; b < nb; ++b) {                                  \
            const int64_t lo = b * ORACLE_SUM_BLOCK;                        \
            const int64_t hi = lo + ORACLE_SUM_BLOCK < n ? lo + ORACLE_SUM_BLOCK : n; \
            double s = 0.0;                                                 \
            for (int64_t i = lo; i < hi; ++i) {                             \
                const double gi = WIDEN(g[i]);                              \
                s += gi * gi;                                               \
            }                                                               \
            part[b] = s;                                                    \
        }                                                                   \
        for (int64_t b = 0; b < nb; ++b)                                    \
            total += part[b];                                               \
        free(part);                                                         \
        return total;                                                       \
    }

static double widen_f64(double g) { return g; }
static double widen_f32(float g) { return (double)g; }
/* A bf16 bit pattern is the upper half of the fp32 with the same value. */
static double widen_bf16(uint16_t bits)
{
    uint32_t w = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

DEFINE_SQNORM(oracle_sqnorm, double, widen_f64)
DEFINE_SQNORM(oracle_sqnorm_f32, float, widen_f32)
DEFINE_SQNORM(oracle_sqnorm_bf16, uint16_t, widen_bf16)

/* Global-norm clipping (App. E.1 uses a threshold of 1.0): the coefficient
 * is clamped at 1 and 1e-6 is added to the norm. A NaN norm is not clamped,
 * so NaN reaches every element, as torch.nn.utils.clip_grad_norm_ does. */
double oracle_clip_coef(double sqnorm, double max_norm)
{
    if (!(max_norm > 0.0))
        return 1.0;
    const double coef = max_norm / (sqrt(sqnorm) + 1e-6);
    return coef > 1.0 ? 1.0 : coef;   /* a NaN norm gives a NaN coefficient */
}

double oracle_quadratic(int64_t n, const double *a, const double *wstar,
                        const double *w, const double *noise, int store,
                        double *grad_out)
{
    if (n <= 0)
        return 0.0;
    const int64_t nb = (n + ORACLE_SUM_BLOCK - 1) / ORACLE_SUM_BLOCK;
    double *part = (double *)malloc(sizeof(double) * (size_t)nb);
    if (part == NULL)
        return NAN;
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        const int64_t lo = b * ORACLE_SUM_BLOCK;
        const int64_t hi = lo + ORACLE_SUM_BLOCK < n ? lo + ORACLE_SUM_BLOCK : n;
        double s = 0.0;
        for (int64_t i = lo; i < hi; ++i) {
            const double d = w[i] - wstar[i];
            if (grad_out != NULL)
                grad_out[i] = oracle_round(a[i] * d + (noise ? noise[i] : 0.0), store);
            s += a[i] * d * d;
        }
        part[b] = s;
    }
    double total = 0.0;
    for (int64_t b = 0; b < nb; ++b)
        total += part[b];
    free(part);
    return 0.5 * total;
}

/* ------------------------------------------------------------- Muon ---- */

/* C (r x q) = P (r x s) Q (s x q), all row-major, exact products summed in
 * double, k in increasing order. */
static void matmul(int64_t r, int64_t s, int64_t q, const double *P, const double *Q, double *C)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < r; ++i) {
        for (int64_t j = 0; j < q; ++j)
            C[i * q + j] = 0.0;
        for (int64_t l = 0; l < s; ++l) {
            const double p = P[i * s + l];
            for (int64_t j = 0; j < q; ++j)
                C[i * q + j] += p * Q[l * q + j];
        }
    }
}

int oracle_newton_schulz(int64_t rows, int64_t cols, const double *M, double eps, double a,
                         double b, double c, int steps, int store, double *O)
{
    if (rows < 0 || cols < 0 || steps < 0 || (rows * cols > 0 && (M == NULL || O == NULL)))
        return -1;
    if (rows == 0 || cols == 0)
        return 0;
    /* Work on the orientation with the smaller Gram matrix: X is r x w. */
    const int tall = rows > cols;
    const int64_t r = tall ? cols : rows, w = tall ? rows : cols;
    double *X = (double *)malloc(sizeof(double) * (size_t)(r * w));
    double *Xt = (double *)malloc(sizeof(double) * (size_t)(w * r));
    double *A = (double *)malloc(sizeof(double) * (size_t)(r * r));
    double *AA = (double *)malloc(sizeof(double) * (size_t)(r * r));
    double *BX = (double *)malloc(sizeof(double) * (size_t)(r * w));
    if (!X || !Xt || !A || !AA || !BX) {
        free(X); free(Xt); free(A); free(AA); free(BX);
        return -1;
    }
    for (int64_t i = 0; i < r; ++i)
        for (int64_t j = 0; j < w; ++j)
            X[i * w + j] = tall ? M[j * cols + i] : M[i * cols + j];
    double ss = 0.0;
    for (int64_t i = 0; i < r * w; ++i)
        ss += X[i] * X[i];
    const double scale = 1.0 / (sqrt(ss) + eps);
    for (int64_t i = 0; i < r * w; ++i)
        X[i] = oracle_round(X[i] * scale, store);

    for (int s = 0; s < steps; ++s) {
        /* A = X X^T */
        for (int64_t i = 0; i < r; ++i)
            for (int64_t j = 0; j < w; ++j)
                Xt[j * r + i] = X[i * w + j];
        matmul(r, w, r, X, Xt, A);
        oracle_round_n(r * r, A, A, store);
        /* B = b A + c A A (B kept in AA) */
        matmul(r, r, r, A, A, AA);
        for (int64_t i = 0; i < r * r; ++i)
            AA[i] = oracle_round(b * A[i] + c * AA[i], store);
        /* X <- a X + B X */
        matmul(r, r, w, AA, X, BX);
        for (int64_t i = 0; i < r * w; ++i)
            X[i] = oracle_round(a * X[i] + BX[i], store);
    }
    for (int64_t i = 0; i < r; ++i)
        for (int64_t j = 0; j < w; ++j) {
            if (tall)
                O[j * cols + i] = X[i * w + j];
            else
                O[i * cols + j] = X[i * w + j];
        }
    free(X); free(Xt); free(A); free(AA); free(BX);
    return 0;
}

int oracle_muon_step(int64_t rows, int64_t cols, int64_t t, const oracle_muon_hparams *hp,
                     const double *g, double clip_scale, double *x, double *mom,
                     double *u_prev, double *stash, double *param, double *o_out)
{
    const int64_t n = rows * cols;
    if (rows < 0 || cols < 0 || t < 1 || hp == NULL ||
        (n > 0 && (g == NULL || x == NULL || mom == NULL)))
        return -1;
    if (hp->delay == 1 && n > 0 && stash == NULL)
        return -1;
    if (n == 0)
        return 0;
    double *O = (double *)malloc(sizeof(double) * (size_t)n);
    if (O == NULL)
        return -1;

    /* Momentum of the stale gradient G_{t-1}. */
    for (int64_t i = 0; i < n; ++i)
        mom[i] = oracle_round(hp->momentum * mom[i] + (1.0 - hp->momentum) * (clip_scale * g[i]),
                              hp->x_store);
    if (oracle_newton_schulz(rows, cols, mom, hp->ns_eps, hp->ns_a, hp->ns_b, hp->ns_c,
                             hp->ns_steps, hp->ns_store, O) != 0) {
        free(O);
        return -1;
    }
    const double s = hp->rms_scale > 0.0
                         ? hp->rms_scale * sqrt((double)(rows > cols ? rows : cols))
                         : 1.0;
    if (hp->correction != ORACLE_CORR_EF && hp->correction != ORACLE_CORR_SAPIPE_SAME &&
        hp->correction != ORACLE_CORR_SAPIPE_UPDATED) {
        free(O);
        return -1;
    }
    const int use_ef = hp->delay == 1 && u_prev != NULL;
    const int updated = use_ef && hp->correction == ORACLE_CORR_SAPIPE_UPDATED;
    const int sapipe = use_ef && (hp->correction == ORACLE_CORR_SAPIPE_SAME || updated);
    /* Alg. 1 / Alg. 2: the standard rule at t <= 1, EF from t = 2. */
    const int ef_now = use_ef && !sapipe && t >= 2;
    for (int64_t i = 0; i < n; ++i) {
        const double xt = x[i];
        const double u = hp->lr * (s * O[i] + hp->weight_decay * xt);
        const double xn = ef_now ? xt - u - hp->ef_lambda * (u - u_prev[i]) : xt - u;
        if (sapipe)   /* SAPipe-WP: the next gradient is taken at x_t - U_prev */
            stash[i] = oracle_round(oracle_round(x[i] - u_prev[i], hp->x_store), hp->stash_store);
        else if (hp->delay == 1)   /* the weights the next gradient is evaluated at */
            stash[i] = oracle_round(x[i], hp->stash_store);
        if (use_ef && !updated)
            u_prev[i] = oracle_round(u, hp->x_store);
        x[i] = oracle_round(xn, hp->x_store);
        if (param != NULL)
            param[i] = oracle_round(x[i], hp->param_store);
    }
    if (o_out != NULL)
        memcpy(o_out, O, sizeof(double) * (size_t)n);
    if (updated) {
        /* SAPipe-WP with the updated state (App. B.1): Alg. 2's step once
         * more on G_{t-1} from the momentum the real step left, that momentum
         * formed as the real step forms it (in its storage format), through
         * a second Newton-Schulz, with decay on X_{t+1}. The history holds
         * this prediction update; the momentum keeps the real step's. */
        double *M2 = (double *)malloc(sizeof(double) * (size_t)n);
        if (M2 == NULL) {
            free(O);
            return -1;
        }
        for (int64_t i = 0; i < n; ++i)
            M2[i] = oracle_round(hp->momentum * mom[i] + (1.0 - hp->momentum) *
                                 (clip_scale * g[i]), hp->x_store);
        if (oracle_newton_schulz(rows, cols, M2, hp->ns_eps, hp->ns_a, hp->ns_b, hp->ns_c,
                                 hp->ns_steps, hp->ns_store, O) != 0) {
            free(M2);
            free(O);
            return -1;
        }
        for (int64_t i = 0; i < n; ++i)
            u_prev[i] = oracle_round(hp->lr * (s * O[i] + hp->weight_decay * x[i]), hp->x_store);
        free(M2);
    }
    free(O);
    return 0;
}
