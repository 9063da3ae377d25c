/*
 * A plain C user of the dpo C ABI (include/dpo.h): no Python and no PyTorch.
 *
 * It owns every buffer (allocated with the CUDA runtime), fills the fp32
 * start weights and each step's bf16 gradients from an input file, and runs
 * one-step-delayed AdamW with Error Feedback and global-norm clipping
 * (Alg. 1, Eq. (1), App. E.1) through dpo_init, dpo_step, dpo_read_weights,
 * dpo_get_flags and dpo_get_step. The results go to an output file, which a
 * test compares with the CPU oracle.
 *
 *   consumer <in> <out>
 *   in:  int32 n_tensors, int32 steps, int64 numel[n_tensors], float lr,
 *        float max_grad_norm, float x0[N], uint16 grad[steps][N] (bf16 bits),
 *        N = sum of numel (tensors laid out one after another)
 *   out: float master[N], uint16 latest[N], uint16 stale[N] (bf16 bits),
 *        double grad_norm, float clip_coef, uint32 flags, int64 k
 *
 * Exit status 0 on success; otherwise a message on stderr and status 1.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "dpo.h"

#define MAX_TENSORS 64

static void die(const char *what, const char *detail)
{
    fprintf(stderr, "consumer: %s: %s\n", what, detail ? detail : "");
    exit(1);
}

static void check_cuda(cudaError_t e, const char *what)
{
    if (e != cudaSuccess)
        die(what, cudaGetErrorString(e));
}

static void check_dpo(int rc, const dpo_ctx *ctx, const char *what)
{
    if (rc != DPO_OK)
        die(what, dpo_last_error(ctx));
}

static void read_exact(FILE *f, void *p, size_t bytes)
{
    if (bytes > 0 && fread(p, 1, bytes, f) != bytes)
        die("input", "short read");
}

static void *dev_alloc(size_t bytes)
{
    void *p = NULL;
    check_cuda(cudaMalloc(&p, bytes), "cudaMalloc");
    return p;
}

int main(int argc, char **argv)
{
    if (argc != 3)
        die("usage", "consumer <in> <out>");
    FILE *in = fopen(argv[1], "rb");
    if (in == NULL)
        die("input", argv[1]);
    int32_t n = 0, steps = 0;
    read_exact(in, &n, sizeof n);
    read_exact(in, &steps, sizeof steps);
    if (n < 1 || n > MAX_TENSORS || steps < 1)
        die("input", "bad tensor or step count");
    int64_t numel[MAX_TENSORS], total = 0;
    read_exact(in, numel, sizeof(int64_t) * (size_t)n);
    for (int t = 0; t < n; ++t) {
        if (numel[t] < 1)
            die("input", "every tensor needs elements");
        total += numel[t];
    }
    float lr = 0.0f, max_norm = 0.0f;
    read_exact(in, &lr, sizeof lr);
    read_exact(in, &max_norm, sizeof max_norm);
    float *x0 = (float *)malloc(sizeof(float) * (size_t)total);
    uint16_t *grads = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)total * (size_t)steps);
    if (x0 == NULL || grads == NULL)
        die("host allocation", NULL);
    read_exact(in, x0, sizeof(float) * (size_t)total);
    read_exact(in, grads, sizeof(uint16_t) * (size_t)total * (size_t)steps);
    fclose(in);

    check_cuda(cudaSetDevice(0), "cudaSetDevice");
    /* One allocation per buffer: cudaMalloc returns 256-byte aligned,
     * non-overlapping memory, as dpo_init requires. */
    dpo_tensor table[MAX_TENSORS];
    memset(table, 0, sizeof table);
    int64_t off = 0;
    for (int t = 0; t < n; ++t) {
        const size_t ne = (size_t)numel[t];
        dpo_tensor *d = &table[t];
        d->param = dev_alloc(2 * ne);
        d->master = (float *)dev_alloc(4 * ne);
        d->m = (float *)dev_alloc(4 * ne);
        d->v = (float *)dev_alloc(4 * ne);
        d->stash = dev_alloc(2 * ne);
        d->ef = (float *)dev_alloc(4 * ne);
        d->grad = dev_alloc(2 * ne);
        d->numel = numel[t];
        d->flags = DPO_WD_ON;
        check_cuda(cudaMemcpy(d->master, x0 + off, 4 * ne, cudaMemcpyHostToDevice),
                   "copy x0");
        off += numel[t];
    }
    dpo_hparams hp;
    memset(&hp, 0, sizeof hp);
    hp.beta1 = 0.9f;
    hp.beta2 = 0.95f;
    hp.eps = 1e-8f;
    hp.weight_decay = 0.1f;
    hp.ef_lambda = 1.0f;
    hp.max_grad_norm = max_norm;
    hp.delay = 1;
    hp.correction = DPO_CORR_EF;
    hp.optimizer = DPO_OPT_ADAMW;
    hp.stash_mode = DPO_STASH_COPY;

    dpo_ctx *ctx = NULL;
    check_dpo(dpo_init(&ctx, table, n, DPO_BF16, DPO_BF16, DPO_BF16, &hp, DPO_INIT_FRESH, NULL),
              NULL, "dpo_init");
    for (int k = 0; k < steps; ++k) {
        /* the gradient of step k + 1, evaluated at the stale weights */
        off = 0;
        for (int t = 0; t < n; ++t) {
            const uint16_t *g = grads + (size_t)k * (size_t)total + (size_t)off;
            check_cuda(cudaMemcpy((void *)table[t].grad, g, 2 * (size_t)numel[t],
                                  cudaMemcpyHostToDevice),
                       "copy gradient");
            off += numel[t];
        }
        check_dpo(dpo_step(ctx, lr, NULL), ctx, "dpo_step");
    }
    check_cuda(cudaDeviceSynchronize(), "synchronize");

    uint32_t flags = 0;
    double norm = 0.0;
    float clip = 0.0f;
    int64_t k_done = 0;
    check_dpo(dpo_get_flags(ctx, &flags, &norm, &clip, NULL), ctx, "dpo_get_flags");
    check_dpo(dpo_get_step(ctx, &k_done), ctx, "dpo_get_step");

    float *master = (float *)malloc(sizeof(float) * (size_t)total);
    uint16_t *latest = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)total);
    uint16_t *stale = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)total);
    if (master == NULL || latest == NULL || stale == NULL)
        die("host allocation", NULL);
    off = 0;
    for (int t = 0; t < n; ++t) {
        const size_t ne = (size_t)numel[t];
        const void *p = NULL;
        dpo_dtype dt;
        check_cuda(cudaMemcpy(master + off, table[t].master, 4 * ne, cudaMemcpyDeviceToHost),
                   "copy master");
        check_dpo(dpo_read_weights(ctx, DPO_LATEST, t, &p, &dt), ctx, "dpo_read_weights");
        if (dt != DPO_BF16)
            die("dpo_read_weights", "latest weights are not bf16");
        check_cuda(cudaMemcpy(latest + off, p, 2 * ne, cudaMemcpyDeviceToHost), "copy latest");
        check_dpo(dpo_read_weights(ctx, DPO_STALE, t, &p, &dt), ctx, "dpo_read_weights");
        check_cuda(cudaMemcpy(stale + off, p, 2 * ne, cudaMemcpyDeviceToHost), "copy stale");
        off += numel[t];
    }
    dpo_destroy(ctx);
    for (int t = 0; t < n; ++t) {
        cudaFree(table[t].param);
        cudaFree(table[t].master);
        cudaFree(table[t].m);
        cudaFree(table[t].v);
        cudaFree(table[t].stash);
        cudaFree(table[t].ef);
        cudaFree((void *)table[t].grad);
    }

    FILE *out = fopen(argv[2], "wb");
    if (out == NULL)
        die("output", argv[2]);
    if (fwrite(master, sizeof(float), (size_t)total, out) != (size_t)total ||
        fwrite(latest, sizeof(uint16_t), (size_t)total, out) != (size_t)total ||
        fwrite(stale, sizeof(uint16_t), (size_t)total, out) != (size_t)total ||
        fwrite(&norm, sizeof norm, 1, out) != 1 || fwrite(&clip, sizeof clip, 1, out) != 1 ||
        fwrite(&flags, sizeof flags, 1, out) != 1 || fwrite(&k_done, sizeof k_done, 1, out) != 1)
        die("output", "short write");
    fclose(out);
    free(x0);
    free(grads);
    free(master);
    free(latest);
    free(stale);
    return 0;
}
