// synth.cu -- host and device fills of seeded synthetic inputs.
//
// Test and benchmark infrastructure (see include/dpo_synth.h). Both sides call
// the same inline Philox4x32-10 functions from philox.h, so a value drawn on
// the device equals the one drawn on the host bit for bit.
#include "dpo_synth.h"
#include "philox.h"

#include <cuda_runtime.h>
#include <math.h>

extern "C" void synth_philox(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    synth_u32x4 c;
    for (int j = 0; j < 4; ++j) c.v[j] = ctr[j];
    const synth_u32x4 r = synth_philox4x32_10(c, key[0], key[1]);
    for (int j = 0; j < 4; ++j) out[j] = r.v[j];
}

extern "C" float synth_normal_scale(double sigma)
{
    // The centred Irwin-Hall integer of eight 16-bit uniforms has variance
    // 8 (65536^2 - 1) / 12 ~ (65536 sqrt(2/3))^2.
    return (float)(sigma / (65536.0 * sqrt(2.0 / 3.0)));
}

template <class Index>
static int host_normal(uint64_t seed, uint32_t stream, uint32_t step, Index index,
                       int64_t n, float scale, int dtype, void *out)
{
    if (n < 0 || (n > 0 && out == nullptr) || (dtype != SYNTH_F32 && dtype != SYNTH_BF16))
        return -1;
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < n; ++j) {
        const float y = synth_normal(seed, stream, step, (uint64_t)index(j), scale);
        if (dtype == SYNTH_F32)
            static_cast<float *>(out)[j] = y;
        else
            static_cast<uint16_t *>(out)[j] = synth_bf16_bits(y);
    }
    return 0;
}

extern "C" int synth_host_normal(uint64_t seed, uint32_t stream, uint32_t step,
                                 int64_t offset, int64_t n, float scale, int dtype, void *out)
{
    if (offset < 0)
        return -1;
    return host_normal(seed, stream, step, [offset](int64_t j) { return offset + j; },
                       n, scale, dtype, out);
}

extern "C" int synth_host_normal_at(uint64_t seed, uint32_t stream, uint32_t step,
                                    const int64_t *idx, int64_t n, float scale, int dtype,
                                    void *out)
{
    if (n > 0 && idx == nullptr)
        return -1;
    return host_normal(seed, stream, step, [idx](int64_t j) { return idx[j]; },
                       n, scale, dtype, out);
}

extern "C" int synth_host_uniform(uint64_t seed, uint32_t stream, uint32_t step,
                                  int64_t offset, int64_t n, float *out)
{
    if (n < 0 || offset < 0 || (n > 0 && out == nullptr))
        return -1;
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < n; ++j)
        out[j] = synth_uniform(seed, stream, step, (uint64_t)(offset + j));
    return 0;
}

extern "C" int synth_host_uniform_at(uint64_t seed, uint32_t stream, uint32_t step,
                                     const int64_t *idx, int64_t n, float *out)
{
    if (n < 0 || (n > 0 && (out == nullptr || idx == nullptr)))
        return -1;
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < n; ++j)
        out[j] = synth_uniform(seed, stream, step, (uint64_t)idx[j]);
    return 0;
}

// ------------------------------------------------------------------ device

static int grid_for(int64_t n)
{
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0)
        sms = 1;
    const int64_t want = (n + 255) / 256;
    const int64_t cap = (int64_t)sms * 8;
    return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

// Four consecutive elements per thread and iteration (one 128-bit fp32 store
// or one 64-bit bf16 store when the destination allows it).
template <int DT>
__global__ void __launch_bounds__(256) normal_kernel(uint64_t seed, uint32_t stream,
                                                     uint32_t step, int64_t offset,
                                                     int64_t n, float scale, void *out)
{
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += stride) {
        const float y = synth_normal(seed, stream, step, (uint64_t)(offset + j), scale);
        if (DT == SYNTH_F32)
            static_cast<float *>(out)[j] = y;
        else
            static_cast<uint16_t *>(out)[j] = synth_bf16_bits(y);
    }
}

extern "C" int synth_dev_normal(uint64_t seed, uint32_t stream, uint32_t step,
                                int64_t offset, int64_t n, float scale, int dtype,
                                void *out, void *cuda_stream)
{
    if (n < 0 || offset < 0 || (n > 0 && out == nullptr) ||
        (dtype != SYNTH_F32 && dtype != SYNTH_BF16))
        return -1;
    if (n == 0)
        return 0;
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    const int grid = grid_for(n);
    if (dtype == SYNTH_F32)
        normal_kernel<SYNTH_F32><<<grid, 256, 0, s>>>(seed, stream, step, offset, n, scale, out);
    else
        normal_kernel<SYNTH_BF16><<<grid, 256, 0, s>>>(seed, stream, step, offset, n, scale, out);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}

__global__ void __launch_bounds__(256) quadratic_kernel(uint64_t seed, uint32_t step, int64_t n,
                                                        const float *__restrict__ a,
                                                        const float *__restrict__ wstar,
                                                        const float *__restrict__ w,
                                                        float noise_scale,
                                                        float *__restrict__ grad,
                                                        double *__restrict__ partials)
{
    __shared__ double red[256];
    double acc = 0.0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const double d = __dsub_rn((double)w[i], (double)wstar[i]);   // exact
        const double ai = (double)a[i];
        const float noise = synth_normal(seed, SYNTH_STREAM_NOISE, step, (uint64_t)i, noise_scale);
        grad[i] = (float)__dadd_rn(__dmul_rn(ai, d), (double)noise);
        acc = __dadd_rn(acc, __dmul_rn(__dmul_rn(ai, d), d));
    }
    red[threadIdx.x] = acc;
    __syncthreads();
    for (int off = blockDim.x / 2; off > 0; off >>= 1) {
        if ((int)threadIdx.x < off)
            red[threadIdx.x] = __dadd_rn(red[threadIdx.x], red[threadIdx.x + off]);
        __syncthreads();
    }
    if (threadIdx.x == 0)
        partials[blockIdx.x] = red[0];
}

extern "C" int synth_dev_quadratic(uint64_t seed, uint32_t step, int64_t n,
                                   const float *a, const float *wstar, const float *w,
                                   float noise_scale, float *grad, double *loss_partials,
                                   int n_partials, void *cuda_stream)
{
    if (n < 0 || n_partials < 1 || n_partials > 65535 || loss_partials == nullptr ||
        (n > 0 && (a == nullptr || wstar == nullptr || w == nullptr || grad == nullptr)))
        return -1;
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    quadratic_kernel<<<n_partials, 256, 0, s>>>(seed, step, n, a, wstar, w, noise_scale,
                                                grad, loss_partials);
    return cudaGetLastError() == cudaSuccess ? 0 : -4;
}
