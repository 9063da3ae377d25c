/*
 * dpo_synth.h -- seeded synthetic inputs for the delayed optimizer step.
 *
 * Test and benchmark infrastructure, a module of its own: it holds none of
 * the optimizer's arithmetic. The tests and the benchmark use it to fill
 * parameter sets shaped like the models the paper trains (arXiv 2606.30634,
 * App. E.2: SmolLM2-style dense models and MoE models; here GPT-2 small,
 * Llama-1B and Llama-7B shapes) with seeded values, on the device (large
 * sets) and on the host (the oracle's side), bit-identically.
 *
 * Draws follow Philox4x32-10 (Salmon et al., SC'11); see
 * paper_2606_30634_gb300/synth/philox.h for the exact mapping from
 * (seed, stream, step, element index) to a value.
 *
 * Conventions for every call below:
 *   - Element indices are global: a value depends only on (seed, stream, step,
 *     index), so a tensor placed at offset o of a larger set draws elements
 *     o .. o + n - 1, and any subset can be regenerated on its own.
 *   - dtype is SYNTH_F32 (float) or SYNTH_BF16 (bf16 bit patterns, rounded
 *     to nearest even from the fp32 draw).
 *   - scale comes from synth_normal_scale(sigma).
 *   - Host buffers are caller-owned host memory; device buffers are
 *     caller-owned device memory on the current device, 4-byte aligned.
 *   - Return 0 on success, -1 on an invalid argument, -4 on a CUDA error.
 *     Device calls are asynchronous on cuda_stream (a cudaStream_t, NULL for
 *     the legacy default stream).
 */
#ifndef DPO_SYNTH_H
#define DPO_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SYNTH_F32 0
#define SYNTH_BF16 1

/* Stream ids used by the workloads. */
#define SYNTH_STREAM_INIT 0   /* initial weights x_0 */
#define SYNTH_STREAM_GRAD 1   /* per-step gradients */
#define SYNTH_STREAM_NOISE 2  /* per-step gradient noise of the quadratic */
#define SYNTH_STREAM_CURV 3   /* curvature a of the quadratic */
#define SYNTH_STREAM_TARGET 4 /* minimiser w* of the quadratic */

/* One Philox4x32-10 block: out = philox(ctr, key). For known-answer tests. */
void synth_philox(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);

/* fp32 multiplier turning the centred Irwin-Hall integer into N(0, sigma^2). */
float synth_normal_scale(double sigma);

/* Host: normal draws for indices offset .. offset + n - 1. */
int synth_host_normal(uint64_t seed, uint32_t stream, uint32_t step,
                      int64_t offset, int64_t n, float scale, int dtype,
                      void *out);

/* Host: normal draws for the n listed indices idx[0..n-1]. */
int synth_host_normal_at(uint64_t seed, uint32_t stream, uint32_t step,
                         const int64_t *idx, int64_t n, float scale, int dtype,
                         void *out);

/* Host: uniform draws in [0, 1) (fp32), indices offset .. offset + n - 1. */
int synth_host_uniform(uint64_t seed, uint32_t stream, uint32_t step,
                       int64_t offset, int64_t n, float *out);

/* Host: uniform draws for the n listed indices. */
int synth_host_uniform_at(uint64_t seed, uint32_t stream, uint32_t step,
                          const int64_t *idx, int64_t n, float *out);

/* Device: normal draws for indices offset .. offset + n - 1 into out. */
int synth_dev_normal(uint64_t seed, uint32_t stream, uint32_t step,
                     int64_t offset, int64_t n, float scale, int dtype,
                     void *out, void *cuda_stream);

/* Device: the noisy diagonal quadratic 1/2 sum a (w - w*)^2 at w:
 *   grad[i] = fp32( a[i] (w[i] - wstar[i]) + noise_i ), evaluated in double
 *   (separately rounded multiply and add), noise_i the normal draw of stream
 *   SYNTH_STREAM_NOISE at (seed, step, i);
 *   loss_partials[b] = sum over the elements block b handles of
 *   a (w - w*)^2 in double (block b handles i = b, b + n_partials, ...);
 *   the loss is 1/2 of the sum of the partials.
 * n_partials in 1 .. 65535. */
int synth_dev_quadratic(uint64_t seed, uint32_t step, int64_t n,
                        const float *a, const float *wstar, const float *w,
                        float noise_scale, float *grad, double *loss_partials,
                        int n_partials, void *cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* DPO_SYNTH_H */
