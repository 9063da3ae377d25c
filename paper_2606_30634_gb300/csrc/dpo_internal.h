// dpo_internal.h -- shared definitions of the C-ABI layer and the kernels.
//
// The tensor table is a virtual concatenation: tensor t owns packets
// [pkt_begin[t], pkt_begin[t+1]) of 8 elements each (its last packet may be
// partial). Every kernel walks the packets grid-stride: thread i of the grid
// takes packets i, i + T, i + 2T, ... (T threads in the grid), so at any time
// all CTAs work in one narrow window of every array (DRAM row locality), and
// each thread keeps a cursor on the tensor holding its packet, advanced
// monotonically as its packet index grows.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dpo {

constexpr int kPacket = 8;      // elements per packet: 16 B of bf16, 32 B of fp32
constexpr uint32_t kFlagWd = 1u;    // DPO_WD_ON
constexpr uint32_t kFlagSync = 2u;  // DPO_SYNC
constexpr int kAlign = 32;      // buffer alignment: fp32 packets move as 256-bit accesses

// Fused step and stash kernels: 128-thread CTAs, 3 or 4 resident per SM
// (the measured table in set_step_grid, dpo_abi.cpp): enough loads in flight
// to keep HBM3e busy, not so many that DRAM efficiency drops.
constexpr int kStepThreads = 128;

// Gradient-norm kernel: one read stream, so each thread keeps up to
// kNormUnroll packets (bf16; half as many fp32 ones) in flight per round.
constexpr int kNormThreads = 256;
constexpr int kNormUnroll = 8;

// Device copy of one table entry.
struct DevTensor {
    void *param;        // bf16 latest copy or nullptr
    float *master;
    float *m;
    float *v;           // second moment (Adan: the averaged gradient difference)
    void *stash;        // stash dtype, or nullptr when not written
    float *ef;          // update-history buffer or nullptr
    const void *grad;
    float *n;           // Adan: third moment, else nullptr
    float *grad_prev;   // Adan: previous (corrected) gradient, else nullptr
    int64_t numel;
    uint32_t flags;
    uint32_t pad_;
};

// Kernel template selectors.
enum StashKind { kStashNone = 0, kStashF32 = 1, kStashBF16 = 2 };
// Staleness correction of a delayed step (the DPO_CORR_* of include/dpo.h, or
// none when the table has no update-history buffers).
enum Correction { kCorrNone = 0, kCorrEF = 1, kCorrSapipeSame = 2, kCorrSapipeUpdated = 3 };
// Update rule (the DPO_OPT_* of include/dpo.h).
enum Optimizer { kOptAdamW = 0, kOptNAdam = 1, kOptLion = 2, kOptAdan = 3 };

// The scalars of one fused step that change from call to call, formed in
// double and rounded once to fp32: on the host (the fields of StepArgs) or,
// for a capturable context, on the device by step_scalars_kernel.
struct StepScalars {
    float step_size, inv_sqrt_bc2, lr_wd, lam, step_size_next, inv_sqrt_bc2_next, lr;
    float nadam_cg, nadam_cm, inv_sqrt_bc3, adan_c2;
    float nadam_cg_next, nadam_cm_next, inv_sqrt_bc3_next, adan_c2_next;
    int first, swap;
};

// Device-resident step counters of a capturable context.
struct StepCounters {
    int64_t k;          // gradients consumed so far
    int64_t phase_k0;   // k at the start of the current delayed phase
    double mu_prod;     // NAdam: prod_{i<=k} mu_i
};

// The step's constants, for step_scalars_kernel.
struct ScalarConsts {
    double beta1, beta2, beta3, weight_decay, momentum_decay;
    float ef_lambda;
    int ef_corr;        // the correction is EF (lambda applies from t = 2)
    int pingpong;       // ping-pong stash in delayed training
};

// Scalars of one fused step, precomputed on the host in double and rounded
// once to fp32 (the per-call ones come from `dev` instead when it is set).
struct StepArgs {
    const DevTensor *table;
    const int64_t *pkt_begin;   // n_tensors + 1 prefix offsets
    int n_tensors;
    int64_t total_pkts;
    float beta1, omb1;          // beta1, 1 - beta1
    float beta2, omb2;          // beta2, 1 - beta2
    float step_size;            // lr / (1 - beta1^k)
    float inv_sqrt_bc2;         // 1 / sqrt(1 - beta2^k)
    float eps;
    float lr_wd;                // lr * weight_decay
    float lam;                  // lambda of this call (0 at k = 1, Alg. 1)
    float step_size_next;       // lr / (1 - beta1^(k+1))       (SAPipe updated state)
    float inv_sqrt_bc2_next;    // 1 / sqrt(1 - beta2^(k+1))    (SAPipe updated state)
    float lr;                   // Lion: size of the sign step
    float nadam_cg, nadam_cm;   // NAdam: lr (1-mu_k)/(1-prod mu), lr mu_{k+1}/(1-prod' mu)
    float beta3, omb3;          // Adan: beta3, 1 - beta3
    float inv_sqrt_bc3;         // Adan: 1 / sqrt(1 - beta3^k)
    float adan_c2;              // Adan: lr beta2 / (1 - beta2^k)
    // the same at the next index k + 1 (SAPipe updated state)
    float nadam_cg_next, nadam_cm_next;   // lr (1-mu_{k+1})/(1-prod_{k+1}), lr mu_{k+2}/(1-prod_{k+2})
    float inv_sqrt_bc3_next;    // Adan: 1 / sqrt(1 - beta3^(k+1))
    float adan_c2_next;         // Adan: lr beta2 / (1 - beta2^(k+1))
    int first;                  // Adan: k == 1 (the gradient difference is 0)
    float dc_lambda;            // DC-ASGD strength (0: off)
    int swap;                   // ping-pong stash: write delayed tensors' weights into
                                // their stash buffer (else their param buffer)
    const float *clip;          // device clip coefficient, or nullptr
    const StepScalars *dev;     // capturable context: the per-call scalars, or nullptr
};

// Device scalars written by the norm pass (one per context).
struct NormScalars {
    double norm;          // global gradient norm of the last clipped step
    float clip;           // clip coefficient used by that step
    unsigned int ticket;  // CTA arrival counter, 0 between launches
    unsigned int flags;   // DPO_FLAG_* bits, sticky until dpo_get_flags reads them
    unsigned int pad_;
};

struct NormArgs {
    const DevTensor *table;
    const int64_t *pkt_begin;
    int n_tensors;
    int64_t total_pkts;
    double max_norm;            // clip threshold (> 0)
    double *partials;           // one per CTA (scratch)
    NormScalars *out;           // norm, clip coefficient, ticket, flags
    double *accum;              // non-null: add ||g||^2 to *accum, form no coefficient
};

struct StashArgs {
    const DevTensor *table;
    const int64_t *pkt_begin;
    int n_tensors;
    int64_t total_pkts;
    int zero_state;             // also zero m, v and the EF buffer (fresh start)
    int zero_hist;              // also zero the EF buffer (delayed training restarts)
};

// The fused-step kernel instance for a layout, correction, rule and DC-ASGD
// setting (one translation unit per rule, dpo_step_<rule>.cu); nullptr when
// that combination is not provided.
using StepFn = void (*)(StepArgs);
StepFn pick_step_adamw(bool param_bf16, StashKind stash, bool grad_bf16, Correction corr,
                       bool dc, bool pp);
StepFn pick_step_nadam(bool param_bf16, StashKind stash, bool grad_bf16, Correction corr,
                       bool dc, bool pp);
StepFn pick_step_lion(bool param_bf16, StashKind stash, bool grad_bf16, Correction corr,
                      bool dc, bool pp);
StepFn pick_step_adan(bool param_bf16, StashKind stash, bool grad_bf16, Correction corr,
                      bool dc, bool pp);

// Device allocation of the library's own blocks (dpo_init, dpo_muon_init),
// through the hook of dpo_test_fail_allocs (dpo_abi.cpp).
cudaError_t device_alloc(void **p, size_t bytes);

// Launchers (dpo_kernels.cu). Each returns the launch's cudaError_t.
cudaError_t launch_step(Optimizer opt, bool param_bf16, StashKind stash, bool grad_bf16,
                        Correction corr, bool dc, bool pp, int grid, const StepArgs &a,
                        cudaStream_t s);
cudaError_t launch_norm(bool grad_bf16, int grid, const NormArgs &a, cudaStream_t s);
// The per-call scalars of the next step from the device counters, which it
// advances (one thread; lr from *lr_src when set, else lr).
cudaError_t launch_step_scalars(StepCounters *cnt, const float *lr_src, float lr,
                                const ScalarConsts &k, StepScalars *out, cudaStream_t s);
// Clip coefficient and norm from an external sum of squares (one thread).
cudaError_t launch_clip_from_sumsq(const double *sumsq, double max_norm, NormScalars *out,
                                   cudaStream_t s);
cudaError_t launch_stash(bool param_bf16, StashKind stash, int grid, const StashArgs &a,
                         cudaStream_t s);

// Resident CTAs per SM of each kernel at its block size (occupancy query).
cudaError_t step_ctas_per_sm(Optimizer opt, bool param_bf16, StashKind stash, bool grad_bf16,
                             Correction corr, bool dc, bool pp, int *n);
cudaError_t norm_ctas_per_sm(bool grad_bf16, int *n);

}  // namespace dpo
