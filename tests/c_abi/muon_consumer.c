/*
 * A plain C user of the delayed-Muon C ABI (include/dpo_muon.h): no Python
 * and no PyTorch.
 *
 * It owns every buffer of its matrices (allocated with the CUDA runtime),
 * fills the fp32 start weights and each step's bf16 gradients from an input
 * file, and runs delayed Muon with Error Feedback (Alg. 2: momentum,
 * Newton-Schulz on the tensor cores, the EF update, stash and bf16 weights)
 * through dpo_muon_init, dpo_muon_step, dpo_muon_get_status and
 * dpo_muon_get_step. The results go to an output file, which a test compares
 * with the CPU oracle.
 *
 *   muon_consumer <in> <out>
 *   in:  int32 n_matrices, int32 steps, int32 ns_steps, int64 rows[n],
 *        int64 cols[n], float lr, float x0[N], uint16 grad[steps][N] (bf16
 *        bits), N = sum of rows * cols (row-major matrices one after another)
 *   out: float master[N], float mom[N], uint16 param[N], uint16 stash[N]
 *        (bf16 bits), uint32 status, int64 k
 *
 * Exit status 0 on success; otherwise a message on stderr and status 1.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "dpo_muon.h"

#define MAX_MATS 64

static void die(const char *what, const char *detail)
{
    fprintf(stderr, "muon_consumer: %s: %s\n", what, detail ? detail : "");
    exit(1);
}

static void check_cuda(cudaError_t e, const char *what)
{
    if (e != cudaSuccess)
        die(what, cudaGetErrorString(e));
}

static void check_dpo(int rc, const dpo_muon_ctx *ctx, const char *what)
{
    if (rc != DPO_OK)
        die(what, dpo_muon_last_error(ctx));
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

static void copy_out(void *dst, const void *src, size_t bytes, const char *what)
{
    check_cuda(cudaMemcpy(dst, src, bytes, cudaMemcpyDeviceToHost), what);
}

int main(int argc, char **argv)
{
    if (argc != 3)
        die("usage", "muon_consumer <in> <out>");
    FILE *in = fopen(argv[1], "rb");
    if (in == NULL)
        die("input", argv[1]);
    int32_t n = 0, steps = 0, ns_steps = 0;
    read_exact(in, &n, sizeof n);
    read_exact(in, &steps, sizeof steps);
    read_exact(in, &ns_steps, sizeof ns_steps);
    if (n < 1 || n > MAX_MATS || steps < 1 || ns_steps < 0)
        die("input", "bad matrix, step or Newton-Schulz step count");
    int64_t rows[MAX_MATS], cols[MAX_MATS], total = 0;
    read_exact(in, rows, sizeof(int64_t) * (size_t)n);
    read_exact(in, cols, sizeof(int64_t) * (size_t)n);
    for (int i = 0; i < n; ++i) {
        if (rows[i] < 1 || cols[i] < 1)
            die("input", "every matrix needs elements");
        total += rows[i] * cols[i];
    }
    float lr = 0.0f;
    read_exact(in, &lr, sizeof lr);
    float *x0 = (float *)malloc(sizeof(float) * (size_t)total);
    uint16_t *grads = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)total * (size_t)steps);
    if (x0 == NULL || grads == NULL)
        die("host allocation", NULL);
    read_exact(in, x0, sizeof(float) * (size_t)total);
    read_exact(in, grads, sizeof(uint16_t) * (size_t)total * (size_t)steps);
    fclose(in);

    check_cuda(cudaSetDevice(0), "cudaSetDevice");
    dpo_matrix mats[MAX_MATS];
    memset(mats, 0, sizeof mats);
    int64_t off = 0;
    for (int i = 0; i < n; ++i) {
        const size_t ne = (size_t)(rows[i] * cols[i]);
        dpo_matrix *d = &mats[i];
        d->param = dev_alloc(2 * ne);
        d->master = (float *)dev_alloc(4 * ne);
        d->mom = (float *)dev_alloc(4 * ne);
        d->stash = dev_alloc(2 * ne);
        d->ef = (float *)dev_alloc(4 * ne);
        d->grad = dev_alloc(2 * ne);
        d->rows = rows[i];
        d->cols = cols[i];
        d->flags = DPO_WD_ON;
        check_cuda(cudaMemcpy(d->master, x0 + off, 4 * ne, cudaMemcpyHostToDevice), "copy x0");
        off += (int64_t)ne;
    }
    dpo_muon_hparams hp;
    memset(&hp, 0, sizeof hp);
    hp.momentum = 0.95f;
    hp.weight_decay = 0.1f;
    hp.ef_lambda = 1.0f;
    hp.max_grad_norm = 0.0f;
    hp.ns_a = 3.4445f;
    hp.ns_b = -4.7750f;
    hp.ns_c = 2.0315f;
    hp.ns_eps = 1e-7f;
    hp.rms_scale = 0.2f;
    hp.ns_steps = ns_steps;
    hp.delay = 1;
    hp.correction = DPO_CORR_EF;

    dpo_muon_ctx *ctx = NULL;
    check_dpo(dpo_muon_init(&ctx, mats, n, DPO_BF16, DPO_BF16, &hp, DPO_INIT_FRESH, NULL), NULL,
              "dpo_muon_init");
    for (int k = 0; k < steps; ++k) {
        off = 0;
        for (int i = 0; i < n; ++i) {
            const size_t ne = (size_t)(rows[i] * cols[i]);
            const uint16_t *g = grads + (size_t)k * (size_t)total + (size_t)off;
            check_cuda(cudaMemcpy((void *)mats[i].grad, g, 2 * ne, cudaMemcpyHostToDevice),
                       "copy gradient");
            off += (int64_t)ne;
        }
        check_dpo(dpo_muon_step(ctx, lr, NULL), ctx, "dpo_muon_step");
    }
    check_cuda(cudaDeviceSynchronize(), "synchronize");
    uint32_t status = 0;
    int64_t k_done = 0;
    check_dpo(dpo_muon_get_status(ctx, &status), ctx, "dpo_muon_get_status");
    check_dpo(dpo_muon_get_step(ctx, &k_done), ctx, "dpo_muon_get_step");

    float *master = (float *)malloc(sizeof(float) * (size_t)total);
    float *mom = (float *)malloc(sizeof(float) * (size_t)total);
    uint16_t *param = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)total);
    uint16_t *stash = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)total);
    if (master == NULL || mom == NULL || param == NULL || stash == NULL)
        die("host allocation", NULL);
    off = 0;
    for (int i = 0; i < n; ++i) {
        const size_t ne = (size_t)(rows[i] * cols[i]);
        copy_out(master + off, mats[i].master, 4 * ne, "copy master");
        copy_out(mom + off, mats[i].mom, 4 * ne, "copy momentum");
        copy_out(param + off, mats[i].param, 2 * ne, "copy weights");
        copy_out(stash + off, mats[i].stash, 2 * ne, "copy stash");
        off += (int64_t)ne;
    }
    dpo_muon_destroy(ctx);
    for (int i = 0; i < n; ++i) {
        cudaFree(mats[i].param);
        cudaFree(mats[i].master);
        cudaFree(mats[i].mom);
        cudaFree(mats[i].stash);
        cudaFree(mats[i].ef);
        cudaFree((void *)mats[i].grad);
    }

    FILE *out = fopen(argv[2], "wb");
    if (out == NULL)
        die("output", argv[2]);
    if (fwrite(master, sizeof(float), (size_t)total, out) != (size_t)total ||
        fwrite(mom, sizeof(float), (size_t)total, out) != (size_t)total ||
        fwrite(param, sizeof(uint16_t), (size_t)total, out) != (size_t)total ||
        fwrite(stash, sizeof(uint16_t), (size_t)total, out) != (size_t)total ||
        fwrite(&status, sizeof status, 1, out) != 1 ||
        fwrite(&k_done, sizeof k_done, 1, out) != 1)
        die("output", "short write");
    fclose(out);
    free(x0);
    free(grads);
    free(master);
    free(mom);
    free(param);
    free(stash);
    return 0;
}
