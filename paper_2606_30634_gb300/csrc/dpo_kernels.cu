// dpo_kernels.cu -- sm_103a kernels of the one-step-delayed step, and the
// launchers of all of them.
//
//   fused_step_kernel   (dpo_step.cuh, instantiated per update rule in
//                       dpo_step_<rule>.cu) the whole per-element step of
//                       Alg. 1 with a staleness correction in one pass over
//                       HBM.
//   grad_sqnorm_kernel  global ||g||^2 over the whole table for clipping
//                       (App. E.1), deterministic: fixed per-thread order,
//                       fixed block tree, fixed-order sum of the per-CTA
//                       partials by the last CTA to finish (no spin-wait).
//   stash_kernel        stash := master (tensors without DPO_SYNC), param :=
//                       master (Alg. 1 start, switches into delayed training),
//                       optionally zeroing m, v and / or the EF buffer.
//
// All three are persistent (a fixed number of CTAs per SM) and walk the
// 8-element packets of the virtual concatenation of the tensors grid-stride
// (see dpo_internal.h). fp32 packets move as single 256-bit accesses, bf16
// packets as 128-bit ones, all with streaming (evict-first) cache hints: no
// element is touched twice in a step. The step is elementwise and HBM-bound;
// there is no tensor-core work in it.
#include "dpo_reduce.cuh"

namespace dpo {
namespace {

// ------------------------------------------------------ gradient norm ----

// Norm and clip coefficient min(1, max_norm / (norm + 1e-6)) from a sum of
// squares; a NaN norm stays NaN and reaches every element.
__device__ void finish_clip(double total, double max_norm, NormScalars *out)
{
    const double norm = sqrt(total);
    double coef = max_norm / (norm + 1e-6);
    coef = coef > 1.0 ? 1.0 : coef;
    if (!isfinite(total))
        out->flags |= 1u;
    out->clip = (float)coef;
    out->norm = norm;
}

__global__ void clip_from_sumsq_kernel(const double *sumsq, double max_norm, NormScalars *out)
{
    finish_clip(*sumsq, max_norm, out);
}

template <int GB>
__global__ void __launch_bounds__(kNormThreads) grad_sqnorm_kernel(const NormArgs a)
{
    using GT = typename Elem<GB != 0>::T;
    constexpr int U = NormUnroll<GT>::value;
    __shared__ double red[kNormThreads / 32];
    __shared__ bool last;

    // Each thread takes U packets per round, kNormThreads apart, and issues
    // the loads of all of them before it sums any; rounds are grid-stride.
    // The packets of a round and of the rounds after it have growing
    // indices, so one forward-moving tensor cursor serves them all, and a
    // tensor's gradient pointer and length are read only when the cursor
    // enters it.
    const int64_t round = (int64_t)gridDim.x * kNormThreads * U;
    const int64_t first = (int64_t)blockIdx.x * kNormThreads * U + threadIdx.x;
    float sum = 0.0f, comp = 0.0f;
    if (first < a.total_pkts) {
        Cursor c;
        c.seek(a.pkt_begin, a.n_tensors, first);
        const GT *grad = static_cast<const GT *>(a.table[c.t].grad);
        int64_t numel = a.table[c.t].numel;
        for (int64_t base = first; base < a.total_pkts; base += round) {
            const GT *ptr[U];
            int cnt[U];   // elements of the packet: 8, 1..7 (a tensor's last), 0 (none)
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t p = base + (int64_t)u * kNormThreads;
                ptr[u] = grad;
                cnt[u] = 0;
                if (p < a.total_pkts) {
                    if (c.advance(a.pkt_begin, p)) {
                        grad = static_cast<const GT *>(a.table[c.t].grad);
                        numel = a.table[c.t].numel;
                    }
                    const int64_t e = (p - c.tb) * kPacket;
                    ptr[u] = grad + e;
                    cnt[u] = numel - e < kPacket ? (int)(numel - e) : kPacket;
                }
            }
            RawPacket<GT> raw[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (cnt[u] == kPacket)
                    raw[u].load(ptr[u]);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                float s = 0.0f;
                if (cnt[u] == kPacket) {
                    s = raw[u].sqsum();
                } else {
                    for (int i = 0; i < cnt[u]; ++i) {
                        const float x = ld1(ptr[u] + i);
                        s += x * x;
                    }
                }
                kahan_add(sum, comp, s);
            }
        }
    }
    const double cta = block_sum<kNormThreads>((double)sum - (double)comp, red);

    // Publish this CTA's partial; the last CTA to arrive finishes the sum in
    // CTA order, so the result does not depend on arrival order.
    if (threadIdx.x == 0) {
        a.partials[blockIdx.x] = cta;
        __threadfence();
        const unsigned int prev = atomicAdd(&a.out->ticket, 1u);
        last = (prev == gridDim.x - 1);
    }
    __syncthreads();
    if (!last)
        return;
    __threadfence();
    double acc = 0.0;
    for (int b = threadIdx.x; b < (int)gridDim.x; b += kNormThreads)
        acc += __ldcg(a.partials + b);
    const double total = block_sum<kNormThreads>(acc, red);
    if (threadIdx.x == 0) {
        if (a.accum != nullptr) {   // one share of a norm over several contexts
            if (!isfinite(total))
                a.out->flags |= 1u;
            *a.accum += total;
        } else {
            finish_clip(total, a.max_norm, a.out);
        }
        a.out->ticket = 0u;   // ready for the next launch
    }
}

// -------------------------------------------------------------- stash ----

template <int PB, int SK>
__global__ void __launch_bounds__(kStepThreads) stash_kernel(const StashArgs a)
{
    using ST = typename StashT<SK>::T;
    const int64_t stride = (int64_t)gridDim.x * kStepThreads;
    int64_t p = (int64_t)blockIdx.x * kStepThreads + threadIdx.x;
    if (p >= a.total_pkts)
        return;
    Cursor c;
    c.seek(a.pkt_begin, a.n_tensors, p);
    DevTensor d = a.table[c.t];
    for (; p < a.total_pkts; p += stride) {
        if (c.advance(a.pkt_begin, p))
            d = a.table[c.t];
        ST *stash = static_cast<ST *>(d.stash);
        __nv_bfloat16 *param = static_cast<__nv_bfloat16 *>(d.param);
        const bool do_stash = SK != kStashNone && stash != nullptr && !(d.flags & kFlagSync);
        const bool zero_ef = d.ef != nullptr && (a.zero_state || a.zero_hist);
        const int64_t e = (p - c.tb) * kPacket;
        if (e + kPacket <= d.numel) {
            float x[8];
            const float z[8] = {0, 0, 0, 0, 0, 0, 0, 0};
            ld8(d.master + e, x);
            if (do_stash)
                st8(stash + e, x);
            if (PB)
                st8(param + e, x);
            if (a.zero_state) {
                st8(d.m + e, z);
                if (d.v != nullptr)
                    st8(d.v + e, z);
                if (d.n != nullptr) {
                    st8(d.n + e, z);
                    st8(d.grad_prev + e, z);
                }
            }
            if (zero_ef)
                st8(d.ef + e, z);
        } else {
            for (int64_t i = e; i < d.numel; ++i) {
                const float x = d.master[i];
                if (do_stash)
                    st1(stash + i, x);
                if (PB)
                    st1(param + i, x);
                if (a.zero_state) {
                    d.m[i] = 0.0f;
                    if (d.v != nullptr)
                        d.v[i] = 0.0f;
                    if (d.n != nullptr) {
                        d.n[i] = 0.0f;
                        d.grad_prev[i] = 0.0f;
                    }
                }
                if (zero_ef)
                    d.ef[i] = 0.0f;
            }
        }
    }
}

// ------------------------------------------------------------ dispatch ----

using StashFn = void (*)(StashArgs);

template <int PB>
StashFn pick_stash_sk(StashKind sk)
{
    switch (sk) {
    case kStashF32:
        return stash_kernel<PB, kStashF32>;
    case kStashBF16:
        return stash_kernel<PB, kStashBF16>;
    default:
        return stash_kernel<PB, kStashNone>;
    }
}

}  // namespace

static StepFn pick_step_for(Optimizer opt, bool pb, StashKind sk, bool gb, Correction corr,
                            bool dc, bool pp)
{
    switch (opt) {
    case kOptAdamW:
        return pick_step_adamw(pb, sk, gb, corr, dc, pp);
    case kOptNAdam:
        return pick_step_nadam(pb, sk, gb, corr, dc, pp);
    case kOptLion:
        return pick_step_lion(pb, sk, gb, corr, dc, pp);
    case kOptAdan:
        return pick_step_adan(pb, sk, gb, corr, dc, pp);
    }
    return nullptr;
}

cudaError_t launch_step(Optimizer opt, bool pb, StashKind sk, bool gb, Correction corr, bool dc,
                        bool pp, int grid, const StepArgs &a, cudaStream_t s)
{
    StepFn f = pick_step_for(opt, pb, sk, gb, corr, dc, pp);
    if (f == nullptr)
        return cudaErrorInvalidValue;
    f<<<grid, kStepThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_norm(bool gb, int grid, const NormArgs &a, cudaStream_t s)
{
    if (gb)
        grad_sqnorm_kernel<1><<<grid, kNormThreads, 0, s>>>(a);
    else
        grad_sqnorm_kernel<0><<<grid, kNormThreads, 0, s>>>(a);
    return cudaGetLastError();
}

// NAdam's momentum schedule mu_i = beta1 (1 - 0.5 * 0.96^(i psi)).
__device__ double nadam_mu_dev(const ScalarConsts &k, int64_t i)
{
    return k.beta1 * (1.0 - 0.5 * pow(0.96, (double)i * k.momentum_decay));
}

// The host's per-call arithmetic of dpo_step, on the device counters.
__global__ void step_scalars_kernel(StepCounters *cnt, const float *lr_src, float lr_host,
                                    const ScalarConsts k, StepScalars *out)
{
    const int64_t kk = cnt->k + 1;            // this call consumes the kk-th gradient
    const int64_t t = kk - cnt->phase_k0;     // Alg. 1 iteration within the delayed phase
    const float lr = lr_src != nullptr ? *lr_src : lr_host;
    const double lrd = lr;
    const double bc1 = 1.0 - pow(k.beta1, (double)kk);
    const double bc2 = 1.0 - pow(k.beta2, (double)kk);
    StepScalars sc;
    sc.step_size = (float)(lrd / bc1);
    sc.inv_sqrt_bc2 = (float)(1.0 / sqrt(bc2));
    sc.lr_wd = (float)(lrd * k.weight_decay);
    sc.lam = (k.ef_corr && t >= 2) ? k.ef_lambda : 0.0f;   // Alg. 1: standard rule at t <= 1
    sc.step_size_next = (float)(lrd / (1.0 - pow(k.beta1, (double)(kk + 1))));
    sc.inv_sqrt_bc2_next = (float)(1.0 / sqrt(1.0 - pow(k.beta2, (double)(kk + 1))));
    sc.lr = lr;
    const double mu_k = nadam_mu_dev(k, kk), mu_next = nadam_mu_dev(k, kk + 1);
    const double mu_prod = cnt->mu_prod * mu_k;
    sc.nadam_cg = (float)(lrd * (1.0 - mu_k) / (1.0 - mu_prod));
    sc.nadam_cm = (float)(lrd * mu_next / (1.0 - mu_prod * mu_next));
    sc.inv_sqrt_bc3 = (float)(1.0 / sqrt(1.0 - pow(k.beta3, (double)kk)));
    sc.adan_c2 = (float)(lrd * k.beta2 / bc2);
    const double mu_next2 = nadam_mu_dev(k, kk + 2);
    sc.nadam_cg_next = (float)(lrd * (1.0 - mu_next) / (1.0 - mu_prod * mu_next));
    sc.nadam_cm_next = (float)(lrd * mu_next2 / (1.0 - mu_prod * mu_next * mu_next2));
    sc.inv_sqrt_bc3_next = (float)(1.0 / sqrt(1.0 - pow(k.beta3, (double)(kk + 1))));
    sc.adan_c2_next = (float)(lrd * k.beta2 / (1.0 - pow(k.beta2, (double)(kk + 1))));
    sc.first = kk == 1;
    sc.swap = k.pingpong && (t & 1) != 0;
    *out = sc;
    cnt->k = kk;
    cnt->mu_prod = mu_prod;
}

cudaError_t launch_step_scalars(StepCounters *cnt, const float *lr_src, float lr,
                                const ScalarConsts &k, StepScalars *out, cudaStream_t s)
{
    step_scalars_kernel<<<1, 1, 0, s>>>(cnt, lr_src, lr, k, out);
    return cudaGetLastError();
}

cudaError_t launch_clip_from_sumsq(const double *sumsq, double max_norm, NormScalars *out,
                                   cudaStream_t s)
{
    clip_from_sumsq_kernel<<<1, 1, 0, s>>>(sumsq, max_norm, out);
    return cudaGetLastError();
}

cudaError_t launch_stash(bool pb, StashKind sk, int grid, const StashArgs &a, cudaStream_t s)
{
    StashFn f = pb ? pick_stash_sk<1>(sk) : pick_stash_sk<0>(sk);
    f<<<grid, kStepThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t step_ctas_per_sm(Optimizer opt, bool pb, StashKind sk, bool gb, Correction corr,
                             bool dc, bool pp, int *n)
{
    StepFn f = pick_step_for(opt, pb, sk, gb, corr, dc, pp);
    if (f == nullptr)
        return cudaErrorInvalidValue;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, f, kStepThreads, 0);
}

cudaError_t norm_ctas_per_sm(bool gb, int *n)
{
    return gb ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, grad_sqnorm_kernel<1>, kNormThreads, 0)
              : cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, grad_sqnorm_kernel<0>, kNormThreads, 0);
}

}  // namespace dpo
