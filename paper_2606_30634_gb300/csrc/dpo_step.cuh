// dpo_step.cuh -- the fused delayed step, templated on layout, staleness
// correction and update rule; instantiated by dpo_step_<rule>.cu.
//
// One pass over HBM per step (Alg. 1 of arXiv 2606.30634): per element the
// (clipped, optionally DC-ASGD-compensated) stale gradient updates the
// optimizer statistics, the update u is formed, and the weights move by the
// standard rule or a staleness correction (lambda-scaled Error Feedback,
// Eq. (1) / App. A.4; SAPipe-WP weight prediction, App. B.1). The stash
// receives the weights the next gradient is evaluated at, the bf16 param the
// new weights. Tensors flagged DPO_SYNC take the standard update with no
// stash and no correction.
#pragma once

#include "dpo_device.cuh"

namespace dpo {
namespace {

struct Scalars {
    float beta1, omb1, beta2, omb2, step_size, inv_sqrt_bc2, eps, lam;
    float step_size_next, inv_sqrt_bc2_next;
    float lr, nadam_cg, nadam_cm;
    float beta3, omb3, inv_sqrt_bc3, adan_c2;
    float nadam_cg_next, nadam_cm_next, inv_sqrt_bc3_next, adan_c2_next;
    bool first;
};

// beta m + (1 - beta) g with the product (1 - beta) g carried exactly (its
// rounding error recovered with an fma): where beta m and the product nearly
// cancel the result keeps full relative accuracy.
__device__ __forceinline__ float ema_exact(float beta, float omb, float m, float g)
{
    const float p = omb * g;
    const float p_err = fmaf(omb, g, -p);
    return fmaf(beta, m, p) + p_err;
}

// The update u of each rule from the (corrected) stale gradient g, updating
// the rule's statistics in place. Decoupled decay acts on the current x_t.
//   AdamW  u = lr (m_hat / (sqrt(v_hat) + eps) + wd x)
//   NAdam  u = cg g / d + cm m / d + lr wd x,  d = sqrt(v_hat) + eps
//   Lion   u = lr (sign(beta1 m + (1 - beta1) g) + wd x), m <- beta2 EMA
//   Adan   u = (lr/bc1 m + lr beta2/bc2 v) / (sqrt(n_hat) + eps) + lr wd x
//          with v the averaged gradient difference and n the EMA of
//          (g + beta2 diff)^2; g_prev <- g
// with lr / (1 - beta1^k), 1 / sqrt(1 - beta2^k) etc. folded on the host.
template <int OPT>
__device__ __forceinline__ float rule_update(const Scalars &s, float g, float x, float wd_lr,
                                             float &m, float &v, float &n, float &gp)
{
    if (OPT == kOptAdamW) {
        m = ema_exact(s.beta1, s.omb1, m, g);
        v = fmaf(s.beta2, v, (s.omb2 * g) * g);
        const float denom = fmaf(sqrtf(v), s.inv_sqrt_bc2, s.eps);
        return fmaf(s.step_size, m / denom, wd_lr * x);
    } else if (OPT == kOptNAdam) {
        m = ema_exact(s.beta1, s.omb1, m, g);
        v = fmaf(s.beta2, v, (s.omb2 * g) * g);
        const float denom = fmaf(sqrtf(v), s.inv_sqrt_bc2, s.eps);
        return fmaf(s.nadam_cg, g, s.nadam_cm * m) / denom + wd_lr * x;
    } else if (OPT == kOptLion) {
        const float c = ema_exact(s.beta1, s.omb1, m, g);
        const float sgn = c > 0.0f ? 1.0f : (c < 0.0f ? -1.0f : 0.0f);
        m = ema_exact(s.beta2, s.omb2, m, g);
        return fmaf(s.lr, sgn, wd_lr * x);
    } else {   // Adan
        const float diff = s.first ? 0.0f : g - gp;
        m = ema_exact(s.beta1, s.omb1, m, g);
        v = ema_exact(s.beta2, s.omb2, v, diff);
        const float w = fmaf(s.beta2, diff, g);
        n = fmaf(s.beta3, n, (s.omb3 * w) * w);
        gp = g;
        const float denom = fmaf(sqrtf(n), s.inv_sqrt_bc3, s.eps);
        return fmaf(s.step_size, m, s.adan_c2 * v) / denom + wd_lr * x;
    }
}

// SAPipe-WP with the updated state (App. B.1): the rule's update at the next
// time index k + 1 on the same gradient g, from the statistics m, v, n, gp
// the real update left (blended with g once more into temporaries), decaying
// x_{t+1}. Adan's stored previous gradient is g itself, so its difference is
// zero.
template <int OPT>
__device__ __forceinline__ float rule_prediction(const Scalars &s, float g, float x_next,
                                                 float wd_lr, float m, float v, float n,
                                                 float gp)
{
    if (OPT == kOptAdamW) {
        const float m2 = ema_exact(s.beta1, s.omb1, m, g);
        const float v2 = fmaf(s.beta2, v, (s.omb2 * g) * g);
        const float denom = fmaf(sqrtf(v2), s.inv_sqrt_bc2_next, s.eps);
        return fmaf(s.step_size_next, m2 / denom, wd_lr * x_next);
    } else if (OPT == kOptNAdam) {
        const float m2 = ema_exact(s.beta1, s.omb1, m, g);
        const float v2 = fmaf(s.beta2, v, (s.omb2 * g) * g);
        const float denom = fmaf(sqrtf(v2), s.inv_sqrt_bc2_next, s.eps);
        return fmaf(s.nadam_cg_next, g, s.nadam_cm_next * m2) / denom + wd_lr * x_next;
    } else if (OPT == kOptLion) {
        const float c = ema_exact(s.beta1, s.omb1, m, g);
        const float sgn = c > 0.0f ? 1.0f : (c < 0.0f ? -1.0f : 0.0f);
        return fmaf(s.lr, sgn, wd_lr * x_next);
    } else {   // Adan
        const float diff = g - gp;
        const float m2 = ema_exact(s.beta1, s.omb1, m, g);
        const float v2 = ema_exact(s.beta2, s.omb2, v, diff);
        const float w = fmaf(s.beta2, diff, g);
        const float n2 = fmaf(s.beta3, n, (s.omb3 * w) * w);
        const float denom = fmaf(sqrtf(n2), s.inv_sqrt_bc3_next, s.eps);
        return fmaf(s.step_size_next, m2, s.adan_c2_next * v2) / denom + wd_lr * x_next;
    }
}

// Displacement of the lambda-scaled EF rule, x_{t+1} = x_t - (u + lambda (u - u_prev)):
// the small terms are summed first so the weight is rounded once, at its own
// magnitude (subtracting u and then the correction would round x twice).
__device__ __forceinline__ float ef_displacement(float lam, float u, float u_prev)
{
    return fmaf(lam, u - u_prev, u);
}

// DC-ASGD (Sec. 3.1): g~ = g + lambda g^2 (x_t - x_stale), x_stale the stash
// the gradient was evaluated at.
__device__ __forceinline__ float dc_compensate(float lambda, float g, float x, float x_stale)
{
    return fmaf(lambda * g * g, x - x_stale, g);
}

// CORR is a Correction: kCorrNone (standard rule, no history buffer),
// kCorrEF (lambda-scaled EF; the buffer is read only when lambda != 0),
// kCorrSapipeSame / kCorrSapipeUpdated (the stash receives the prediction
// point x_t - u_prev; the weights take the standard rule). OPT is the rule.
// DC selects the DC-ASGD compensation of delayed tensors (instances with a
// stash only); without it the kernel holds no registers for the stash read.
// PP selects the ping-pong stash (bf16 param and stash, standard rule or EF):
// the buffers of delayed tensors swap roles instead of the stash being stored.
template <int PB, int SK, int GB, int CORR, int OPT, int DC, int PP>
__global__ void __launch_bounds__(kStepThreads) fused_step_kernel(const StepArgs a)
{
    using GT = typename Elem<GB != 0>::T;
    using ST = typename StashT<SK>::T;
    constexpr bool kHist = CORR != kCorrNone;
    constexpr bool kSapipe = CORR == kCorrSapipeSame || CORR == kCorrSapipeUpdated;
    constexpr bool kV = OPT != kOptLion;
    constexpr bool kAdan = OPT == kOptAdan;

    const int64_t stride = (int64_t)gridDim.x * kStepThreads;
    int64_t p = (int64_t)blockIdx.x * kStepThreads + threadIdx.x;
    if (p >= a.total_pkts)
        return;

    // The per-call scalars: kernel parameters, or (capturable context) the
    // values step_scalars_kernel left in device memory for this call.
    StepScalars sc{a.step_size, a.inv_sqrt_bc2, a.lr_wd, a.lam, a.step_size_next,
                   a.inv_sqrt_bc2_next, a.lr, a.nadam_cg, a.nadam_cm, a.inv_sqrt_bc3, a.adan_c2,
                   a.nadam_cg_next, a.nadam_cm_next, a.inv_sqrt_bc3_next, a.adan_c2_next,
                   a.first, a.swap};
    if (a.dev != nullptr)
        sc = *a.dev;
    const Scalars s{a.beta1, a.omb1, a.beta2, a.omb2, sc.step_size, sc.inv_sqrt_bc2, a.eps, sc.lam,
                    sc.step_size_next, sc.inv_sqrt_bc2_next, sc.lr, sc.nadam_cg, sc.nadam_cm,
                    a.beta3, a.omb3, sc.inv_sqrt_bc3, sc.adan_c2, sc.nadam_cg_next,
                    sc.nadam_cm_next, sc.inv_sqrt_bc3_next, sc.adan_c2_next, sc.first != 0};
    const float clip = a.clip != nullptr ? __ldg(a.clip) : 1.0f;
    const bool use_prev = kSapipe || (CORR == kCorrEF && sc.lam != 0.0f);
    const bool ef_now = CORR == kCorrEF && sc.lam != 0.0f;
    const float dc = a.dc_lambda;

    Cursor c;
    c.seek(a.pkt_begin, a.n_tensors, p);
    DevTensor d = a.table[c.t];
    for (; p < a.total_pkts; p += stride) {
        if (c.advance(a.pkt_begin, p))
            d = a.table[c.t];
        float *__restrict__ master = d.master;
        float *__restrict__ mm = d.m;
        float *__restrict__ vv = d.v;
        float *__restrict__ nn = d.n;
        float *__restrict__ gpv = d.grad_prev;
        float *__restrict__ ef = d.ef;
        const GT *__restrict__ grad = static_cast<const GT *>(d.grad);
        const float wd_lr = (d.flags & kFlagWd) ? sc.lr_wd : 0.0f;
        // A DPO_SYNC tensor takes the standard update with no stash and no
        // correction even while the run is delayed.
        const bool dly = SK != kStashNone && !(d.flags & kFlagSync);
        // Ping-pong stash (bf16 param and stash): the new weights go into the
        // buffer holding the stale version, which is then the one DC-ASGD
        // reads, and no stash is stored.
        const bool pp = PP && dly;
        __nv_bfloat16 *param = static_cast<__nv_bfloat16 *>(pp && sc.swap ? d.stash : d.param);
        ST *stash = pp ? reinterpret_cast<ST *>(param) : static_cast<ST *>(d.stash);   // may alias param
        const bool prev_t = dly && use_prev;
        const bool efn_t = dly && ef_now;
        const bool dc_t = DC && dly;
        const int64_t e = (p - c.tb) * kPacket;

        if (e + kPacket <= d.numel) {
            float x[8], m[8], v[8], n[8], gp[8], g[8], up[8], sw[8];
            ld8(master + e, x);
            ld8(mm + e, m);
            if (kV)
                ld8(vv + e, v);
            if (kAdan) {
                ld8(nn + e, n);
                ld8(gpv + e, gp);
            }
            ld8(grad + e, g);
            if (prev_t)
                ld8(ef + e, up);
            if (dc_t)
                ld8(stash + e, sw);   // the weights the gradient was evaluated at
            if (dly && !pp) {
                if (kSapipe) {   // stash := the prediction point x_t - u_prev
                    float xp[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        xp[j] = x[j] - up[j];
                    st8(stash + e, xp);
                } else {
                    st8(stash + e, x);   // stash := x_t, before the update
                }
            }
            float u[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                float gc = g[j] * clip;
                if (dc_t)
                    gc = dc_compensate(dc, gc, x[j], sw[j]);
                u[j] = rule_update<OPT>(s, gc, x[j], wd_lr, m[j], v[j], n[j], gp[j]);
                x[j] -= efn_t ? ef_displacement(s.lam, u[j], up[j]) : u[j];
                if (CORR == kCorrSapipeUpdated)
                    u[j] = rule_prediction<OPT>(s, gc, x[j], wd_lr, m[j], v[j], n[j], gp[j]);
            }
            st8(master + e, x);
            st8(mm + e, m);
            if (kV)
                st8(vv + e, v);
            if (kAdan) {
                st8(nn + e, n);
                st8(gpv + e, gp);
            }
            if (kHist && dly)
                st8(ef + e, u);
            if (PB)
                st8(param + e, x);
        } else {
            // the tensor's last, partial packet
            for (int64_t i = e; i < d.numel; ++i) {
                float x = master[i], m = mm[i];
                float v = kV ? vv[i] : 0.0f;
                float n = kAdan ? nn[i] : 0.0f, gp = kAdan ? gpv[i] : 0.0f;
                float g = ld1(grad + i) * clip;
                const float up = prev_t ? ef[i] : 0.0f;
                if (dc_t)
                    g = dc_compensate(dc, g, x, ld1(stash + i));
                if (dly && !pp)
                    st1(stash + i, kSapipe ? x - up : x);
                float u = rule_update<OPT>(s, g, x, wd_lr, m, v, n, gp);
                x -= efn_t ? ef_displacement(s.lam, u, up) : u;
                if (CORR == kCorrSapipeUpdated)
                    u = rule_prediction<OPT>(s, g, x, wd_lr, m, v, n, gp);
                master[i] = x;
                mm[i] = m;
                if (kV)
                    vv[i] = v;
                if (kAdan) {
                    nn[i] = n;
                    gpv[i] = gp;
                }
                if (kHist && dly)
                    ef[i] = u;
                if (PB)
                    st1(param + i, x);
            }
        }
    }
}

// ------------------------------------------------------------ dispatch ----

template <int PB, int SK, int GB, int OPT, int DC>
StepFn pick_step_corr(Correction corr, bool pp)
{
    // the ping-pong stash: bf16 param and stash, standard rule or EF
    constexpr bool kPP = PB == 1 && SK == kStashBF16;
    switch (corr) {
    case kCorrNone:
        if (pp)
            return kPP ? fused_step_kernel<PB, SK, GB, kCorrNone, OPT, DC, kPP ? 1 : 0> : nullptr;
        return fused_step_kernel<PB, SK, GB, kCorrNone, OPT, DC, 0>;
    case kCorrEF:
        if (pp)
            return kPP ? fused_step_kernel<PB, SK, GB, kCorrEF, OPT, DC, kPP ? 1 : 0> : nullptr;
        return fused_step_kernel<PB, SK, GB, kCorrEF, OPT, DC, 0>;
    case kCorrSapipeSame:
        return pp ? nullptr : fused_step_kernel<PB, SK, GB, kCorrSapipeSame, OPT, DC, 0>;
    case kCorrSapipeUpdated:
        return pp ? nullptr : fused_step_kernel<PB, SK, GB, kCorrSapipeUpdated, OPT, DC, 0>;
    }
    return nullptr;
}

template <int PB, int GB, int OPT>
StepFn pick_step_sk(StashKind sk, Correction corr, bool dc, bool pp)
{
    switch (sk) {
    case kStashF32:
        return dc ? pick_step_corr<PB, kStashF32, GB, OPT, 1>(corr, pp)
                  : pick_step_corr<PB, kStashF32, GB, OPT, 0>(corr, pp);
    case kStashBF16:
        return dc ? pick_step_corr<PB, kStashBF16, GB, OPT, 1>(corr, pp)
                  : pick_step_corr<PB, kStashBF16, GB, OPT, 0>(corr, pp);
    default:   // synchronous: no stash, no correction, no compensation
        return corr == kCorrNone && !dc && !pp
                   ? fused_step_kernel<PB, kStashNone, GB, kCorrNone, OPT, 0, 0>
                   : nullptr;
    }
}

template <int OPT>
StepFn pick_step(bool pb, StashKind sk, bool gb, Correction corr, bool dc, bool pp)
{
    if (pb)
        return gb ? pick_step_sk<1, 1, OPT>(sk, corr, dc, pp)
                  : pick_step_sk<1, 0, OPT>(sk, corr, dc, pp);
    return gb ? pick_step_sk<0, 1, OPT>(sk, corr, dc, pp) : pick_step_sk<0, 0, OPT>(sk, corr, dc, pp);
}

}  // namespace
}  // namespace dpo
