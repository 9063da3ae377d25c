// dpo_kernels.cu -- sm_103a kernels of the one-step-delayed AdamW step.
//
//   fused_step_kernel   the whole per-element step of Alg. 1 with AdamW and a
//                       staleness correction (lambda-scaled Error Feedback,
//                       Eq. (1) / App. A.4, or SAPipe-WP weight prediction,
//                       App. B.1) in one pass over HBM: read master, m, v,
//                       grad (and the update-history buffer); write master,
//                       m, v, stash, the bf16 latest copy (and the buffer).
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
#include "dpo_internal.h"

#include <cuda_bf16.h>
#include <math.h>

namespace dpo {
namespace {

// ---------------------------------------------------------------- I/O ----
// fp32 packet: one 32-byte (256-bit) load or store per thread.

__device__ __forceinline__ void ld8(const float *p, float (&r)[8])
{
    asm volatile("ld.global.cs.v8.f32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=f"(r[0]), "=f"(r[1]), "=f"(r[2]), "=f"(r[3]), "=f"(r[4]), "=f"(r[5]),
                   "=f"(r[6]), "=f"(r[7])
                 : "l"(p));
}

__device__ __forceinline__ void st8(float *p, const float (&r)[8])
{
    asm volatile("st.global.cs.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};"
                 :: "l"(p), "f"(r[0]), "f"(r[1]), "f"(r[2]), "f"(r[3]), "f"(r[4]), "f"(r[5]),
                    "f"(r[6]), "f"(r[7])
                 : "memory");
}

// bf16 packet: one 16-byte load or store; values widen exactly to fp32.
__device__ __forceinline__ void ld8(const __nv_bfloat16 *p, float (&r)[8])
{
    const uint4 q = __ldcs(reinterpret_cast<const uint4 *>(p));
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        r[2 * j] = __uint_as_float(w[j] << 16);
        r[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);   // round to nearest even
    return *reinterpret_cast<const uint32_t *>(&h);
}

__device__ __forceinline__ void st8(__nv_bfloat16 *p, const float (&r)[8])
{
    const uint4 q = make_uint4(pack_bf16x2(r[0], r[1]), pack_bf16x2(r[2], r[3]),
                               pack_bf16x2(r[4], r[5]), pack_bf16x2(r[6], r[7]));
    __stcs(reinterpret_cast<uint4 *>(p), q);
}

__device__ __forceinline__ float ld1(const float *p) { return __ldcs(p); }
__device__ __forceinline__ float ld1(const __nv_bfloat16 *p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st1(float *p, float x) { __stcs(p, x); }
__device__ __forceinline__ void st1(__nv_bfloat16 *p, float x) { *p = __float2bfloat16_rn(x); }

template <bool BF16> struct Elem { using T = float; };
template <> struct Elem<true> { using T = __nv_bfloat16; };

template <int SK> struct StashT { using T = float; };
template <> struct StashT<kStashBF16> { using T = __nv_bfloat16; };

// ------------------------------------------------------------- cursor ----

// Last tensor whose first packet is <= p (pkt_begin sorted, pkt_begin[0] = 0,
// pkt_begin[n] = total): for p < total, the tensor holding packet p.
__device__ __forceinline__ int find_tensor(const int64_t *pkt_begin, int n, int64_t p)
{
    int lo = 0, hi = n;   // answer in [lo, hi)
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(pkt_begin + mid) <= p)
            lo = mid;
        else
            hi = mid;
    }
    return lo;
}

// The tensor holding a thread's current packet. Packet indices only grow, so
// the cursor moves forward, skipping whole tensors (empty ones included).
struct Cursor {
    int t;
    int64_t tb, te;   // packet range [tb, te) of tensor t

    __device__ __forceinline__ void seek(const int64_t *pkt_begin, int n, int64_t p)
    {
        t = find_tensor(pkt_begin, n, p);
        tb = __ldg(pkt_begin + t);
        te = __ldg(pkt_begin + t + 1);
    }
    // true when the packet moved to another tensor (p < total)
    __device__ __forceinline__ bool advance(const int64_t *pkt_begin, int64_t p)
    {
        if (p < te)
            return false;
        do {
            ++t;
            tb = te;
            te = __ldg(pkt_begin + t + 1);
        } while (p >= te);
        return true;
    }
};

// ------------------------------------------------------- the fused step ----

struct Scalars {
    float beta1, omb1, beta2, omb2, step_size, inv_sqrt_bc2, eps, lam;
    float step_size_next, inv_sqrt_bc2_next;
};

// Moments with the (clipped) stale gradient, then the AdamW update
//   u = lr (m_hat / (sqrt(v_hat) + eps) + wd x_t)
// with lr / (1 - beta1^k) and 1 / sqrt(1 - beta2^k) folded on the host.
// The first moment's product (1 - beta1) g is carried exactly (its rounding
// error recovered with an fma), so where beta1 m and that product nearly
// cancel the new m keeps full relative accuracy; v has no cancellation.
__device__ __forceinline__ float adamw_update(const Scalars &s, float g, float x, float wd_lr,
                                              float &m, float &v)
{
    const float p = s.omb1 * g;
    const float p_err = fmaf(s.omb1, g, -p);
    m = fmaf(s.beta1, m, p) + p_err;
    v = fmaf(s.beta2, v, (s.omb2 * g) * g);
    const float denom = fmaf(sqrtf(v), s.inv_sqrt_bc2, s.eps);
    return fmaf(s.step_size, m / denom, wd_lr * x);
}

// SAPipe-WP with the updated state (App. B.1): the AdamW update at the next
// time index on the same gradient g, from the moments m, v the real update
// left (blended with g once more into temporaries), decaying x_{t+1}.
__device__ __forceinline__ float adamw_prediction(const Scalars &s, float g, float x_next,
                                                  float wd_lr, float m, float v)
{
    const float p = s.omb1 * g;
    const float p_err = fmaf(s.omb1, g, -p);
    const float m2 = fmaf(s.beta1, m, p) + p_err;
    const float v2 = fmaf(s.beta2, v, (s.omb2 * g) * g);
    const float denom = fmaf(sqrtf(v2), s.inv_sqrt_bc2_next, s.eps);
    return fmaf(s.step_size_next, m2 / denom, wd_lr * x_next);
}

// Displacement of the lambda-scaled EF rule, x_{t+1} = x_t - (u + lambda (u - u_prev)):
// the small terms are summed first so the weight is rounded once, at its own
// magnitude (subtracting u and then the correction would round x twice).
__device__ __forceinline__ float ef_displacement(float lam, float u, float u_prev)
{
    return fmaf(lam, u - u_prev, u);
}

// CORR is a Correction: kCorrNone (standard rule, no history buffer),
// kCorrEF (lambda-scaled EF; the buffer is read only when lambda != 0),
// kCorrSapipeSame / kCorrSapipeUpdated (the stash receives the prediction
// point x_t - u_prev; the weights take the standard rule).
template <int PB, int SK, int GB, int CORR>
__global__ void __launch_bounds__(kStepThreads) fused_step_kernel(const StepArgs a)
{
    using GT = typename Elem<GB != 0>::T;
    using ST = typename StashT<SK>::T;
    constexpr bool kHist = CORR != kCorrNone;
    constexpr bool kSapipe = CORR == kCorrSapipeSame || CORR == kCorrSapipeUpdated;

    const int64_t stride = (int64_t)gridDim.x * kStepThreads;
    int64_t p = (int64_t)blockIdx.x * kStepThreads + threadIdx.x;
    if (p >= a.total_pkts)
        return;

    const Scalars s{a.beta1, a.omb1, a.beta2, a.omb2, a.step_size, a.inv_sqrt_bc2, a.eps, a.lam,
                    a.step_size_next, a.inv_sqrt_bc2_next};
    const float clip = a.clip != nullptr ? __ldg(a.clip) : 1.0f;
    const bool use_prev = kSapipe || (CORR == kCorrEF && a.lam != 0.0f);
    const bool ef_now = CORR == kCorrEF && a.lam != 0.0f;

    Cursor c;
    c.seek(a.pkt_begin, a.n_tensors, p);
    DevTensor d = a.table[c.t];
    for (; p < a.total_pkts; p += stride) {
        if (c.advance(a.pkt_begin, p))
            d = a.table[c.t];
        float *__restrict__ master = d.master;
        float *__restrict__ mm = d.m;
        float *__restrict__ vv = d.v;
        float *__restrict__ ef = d.ef;
        const GT *__restrict__ grad = static_cast<const GT *>(d.grad);
        ST *__restrict__ stash = static_cast<ST *>(d.stash);
        __nv_bfloat16 *__restrict__ param = static_cast<__nv_bfloat16 *>(d.param);
        const float wd_lr = (d.flags & kFlagWd) ? a.lr_wd : 0.0f;
        // A DPO_SYNC tensor takes the standard update with no stash and no
        // correction even while the run is delayed.
        const bool dly = SK != kStashNone && !(d.flags & kFlagSync);
        const bool prev_t = dly && use_prev;
        const bool efn_t = dly && ef_now;
        const int64_t e = (p - c.tb) * kPacket;

        if (e + kPacket <= d.numel) {
            float x[8], m[8], v[8], g[8], up[8];
            ld8(master + e, x);
            ld8(mm + e, m);
            ld8(vv + e, v);
            ld8(grad + e, g);
            if (prev_t)
                ld8(ef + e, up);
            if (dly) {
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
                const float gc = g[j] * clip;
                u[j] = adamw_update(s, gc, x[j], wd_lr, m[j], v[j]);
                x[j] -= efn_t ? ef_displacement(s.lam, u[j], up[j]) : u[j];
                if (CORR == kCorrSapipeUpdated)
                    u[j] = adamw_prediction(s, gc, x[j], wd_lr, m[j], v[j]);
            }
            st8(master + e, x);
            st8(mm + e, m);
            st8(vv + e, v);
            if (kHist && dly)
                st8(ef + e, u);
            if (PB)
                st8(param + e, x);
        } else {
            // the tensor's last, partial packet
            for (int64_t i = e; i < d.numel; ++i) {
                float x = master[i], m = mm[i], v = vv[i];
                const float g = ld1(grad + i) * clip;
                const float up = prev_t ? ef[i] : 0.0f;
                if (dly)
                    st1(stash + i, kSapipe ? x - up : x);
                float u = adamw_update(s, g, x, wd_lr, m, v);
                x -= efn_t ? ef_displacement(s.lam, u, up) : u;
                if (CORR == kCorrSapipeUpdated)
                    u = adamw_prediction(s, g, x, wd_lr, m, v);
                master[i] = x;
                mm[i] = m;
                vv[i] = v;
                if (kHist && dly)
                    ef[i] = u;
                if (PB)
                    st1(param + i, x);
            }
        }
    }
}

// ------------------------------------------------------ gradient norm ----

template <int NT>
__device__ __forceinline__ double block_sum(double x, double *red)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
        x += __shfl_down_sync(0xFFFFFFFFu, x, off);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0)
        red[warp] = x;
    __syncthreads();
    double r = 0.0;
    if (warp == 0) {
        r = lane < NT / 32 ? red[lane] : 0.0;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
            r += __shfl_down_sync(0xFFFFFFFFu, r, off);
    }
    __syncthreads();
    return r;   // valid in thread 0
}

// Kahan-compensated fp32 accumulation of per-packet sums of squares (the
// compensation keeps the per-thread error near one rounding however many
// packets a thread visits), fp64 from the block reduction on.
__device__ __forceinline__ void kahan_add(float &sum, float &c, float x)
{
    const float y = x - c;
    const float t = sum + y;
    c = (t - sum) - y;
    sum = t;
}

template <class GT>
__device__ __forceinline__ float packet_sqsum(const GT *grad, int64_t e, int64_t numel)
{
    if (e + kPacket <= numel) {
        float g[8];
        ld8(grad + e, g);
        return ((g[0] * g[0] + g[1] * g[1]) + (g[2] * g[2] + g[3] * g[3])) +
               ((g[4] * g[4] + g[5] * g[5]) + (g[6] * g[6] + g[7] * g[7]));
    }
    float s = 0.0f;
    for (int64_t i = e; i < numel; ++i) {
        const float g = ld1(grad + i);
        s += g * g;
    }
    return s;
}

template <int GB>
__global__ void __launch_bounds__(kNormThreads) grad_sqnorm_kernel(const NormArgs a)
{
    using GT = typename Elem<GB != 0>::T;
    __shared__ double red[kNormThreads / 32];
    __shared__ bool last;

    // Each thread takes kNormUnroll packets per round, kNormThreads apart, so
    // their loads are in flight together; rounds are grid-stride, and each of
    // the kNormUnroll packet streams keeps its own tensor cursor.
    const int64_t round = (int64_t)gridDim.x * kNormThreads * kNormUnroll;
    const int64_t first = (int64_t)blockIdx.x * kNormThreads * kNormUnroll + threadIdx.x;
    float sum = 0.0f, comp = 0.0f;
    if (first < a.total_pkts) {
        Cursor c[kNormUnroll];
#pragma unroll
        for (int u = 0; u < kNormUnroll; ++u) {
            const int64_t p = first + (int64_t)u * kNormThreads;
            c[u].seek(a.pkt_begin, a.n_tensors, p < a.total_pkts ? p : a.total_pkts - 1);
        }
        for (int64_t base = first; base < a.total_pkts; base += round) {
            float part[kNormUnroll];
#pragma unroll
            for (int u = 0; u < kNormUnroll; ++u) {
                const int64_t p = base + (int64_t)u * kNormThreads;
                part[u] = 0.0f;
                if (p < a.total_pkts) {
                    c[u].advance(a.pkt_begin, p);
                    const DevTensor &d = a.table[c[u].t];
                    part[u] = packet_sqsum(static_cast<const GT *>(d.grad),
                                           (p - c[u].tb) * kPacket, d.numel);
                }
            }
#pragma unroll
            for (int u = 0; u < kNormUnroll; ++u)
                kahan_add(sum, comp, part[u]);
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
        const double norm = sqrt(total);
        double coef = a.max_norm / (norm + 1e-6);
        coef = coef > 1.0 ? 1.0 : coef;   // a NaN norm stays NaN and reaches every element
        if (!isfinite(total))
            a.out->flags |= 1u;
        a.out->clip = (float)coef;
        a.out->norm = norm;
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
                st8(d.v + e, z);
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
                    d.v[i] = 0.0f;
                }
                if (zero_ef)
                    d.ef[i] = 0.0f;
            }
        }
    }
}

// ------------------------------------------------------------ dispatch ----

using StepFn = void (*)(StepArgs);

template <int PB, int SK, int GB>
StepFn pick_step_corr(Correction corr)
{
    switch (corr) {
    case kCorrNone:
        return fused_step_kernel<PB, SK, GB, kCorrNone>;
    case kCorrEF:
        return fused_step_kernel<PB, SK, GB, kCorrEF>;
    case kCorrSapipeSame:
        return fused_step_kernel<PB, SK, GB, kCorrSapipeSame>;
    case kCorrSapipeUpdated:
        return fused_step_kernel<PB, SK, GB, kCorrSapipeUpdated>;
    }
    return nullptr;
}

template <int PB, int GB>
StepFn pick_step_sk(StashKind sk, Correction corr)
{
    switch (sk) {
    case kStashF32:
        return pick_step_corr<PB, kStashF32, GB>(corr);
    case kStashBF16:
        return pick_step_corr<PB, kStashBF16, GB>(corr);
    default:   // synchronous: no stash, no correction
        return corr == kCorrNone ? fused_step_kernel<PB, kStashNone, GB, kCorrNone> : nullptr;
    }
}

StepFn pick_step(bool pb, StashKind sk, bool gb, Correction corr)
{
    if (pb)
        return gb ? pick_step_sk<1, 1>(sk, corr) : pick_step_sk<1, 0>(sk, corr);
    return gb ? pick_step_sk<0, 1>(sk, corr) : pick_step_sk<0, 0>(sk, corr);
}

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

cudaError_t launch_step(bool pb, StashKind sk, bool gb, Correction corr, int grid,
                        const StepArgs &a, cudaStream_t s)
{
    StepFn f = pick_step(pb, sk, gb, corr);
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

cudaError_t launch_stash(bool pb, StashKind sk, int grid, const StashArgs &a, cudaStream_t s)
{
    StashFn f = pb ? pick_stash_sk<1>(sk) : pick_stash_sk<0>(sk);
    f<<<grid, kStepThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t step_ctas_per_sm(bool pb, StashKind sk, bool gb, Correction corr, int *n)
{
    StepFn f = pick_step(pb, sk, gb, corr);
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
