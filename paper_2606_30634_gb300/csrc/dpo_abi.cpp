// dpo_abi.cpp -- the C ABI of include/dpo.h: validation, context, launches.
//
// Host side of the one-step-delayed AdamW step (arXiv 2606.30634, Alg. 1 with
// the Error-Feedback correction of Eq. (1) / App. A.4). The per-call scalars
// (bias corrections, the Alg. 1 "standard rule for t <= 1" switch) are formed
// here in double and handed to the kernels by value; every per-element
// operation runs in dpo_kernels.cu.
#include "dpo.h"
#include "dpo_internal.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <mutex>
#include <new>
#include <string>
#include <vector>

using dpo::DevTensor;
using dpo::StashKind;

struct dpo_ctx {
    int device = 0;
    int n = 0;
    dpo_dtype param_dt = DPO_F32, stash_dt = DPO_F32, grad_dt = DPO_F32;
    dpo_hparams hp{};
    bool ef = false;
    bool clip = false;
    bool host_io = false;   // grad or param in host memory
    bool has_stash = false; // some tensor has a stash buffer
    bool can_delay = false; // every tensor without DPO_SYNC has one
    // step counters; a capturable context keeps the authoritative copy on
    // the device (d_cnt) and refreshes these from it when the host needs them
    mutable int64_t k = 0;
    mutable int64_t phase_k0 = 0;   // k when the current delayed phase began
    mutable double mu_prod = 1.0;   // NAdam: prod_{i<=k} mu_i
    bool capturable = false;        // dpo_set_capturable
    const float *lr_src = nullptr;  // capturable: device learning rate, or nullptr
    int64_t total_pkts = 0;
    int64_t total_elems = 0;
    std::vector<dpo_tensor> table;
    int sms = 0;
    int step_grid = 0, norm_grid = 0, stash_grid = 0;
    // one device allocation: table | pkt_begin | partials | scalars
    void *dev_block = nullptr;
    DevTensor *d_table = nullptr;
    int64_t *d_pkt_begin = nullptr;
    double *d_partials = nullptr;
    dpo::NormScalars *d_scalars = nullptr;
    dpo::StepCounters *d_cnt = nullptr;   // capturable mode's counters
    dpo::StepScalars *d_sc = nullptr;     // capturable mode's per-call scalars
    const double *clip_src = nullptr;   // external sum of squares (dpo_set_clip_source)
    // dpo_set_timing: three events per timed call (before the norm pass,
    // before the fused step, after it), recorded since the last read
    bool timing = false;
    std::vector<cudaEvent_t> ev_pool;
    size_t ev_used = 0;
    std::string err;
};

namespace {

thread_local std::string g_init_err;

// dpo_test_fail_allocs: allocations to let through, then allocations to fail.
std::mutex g_alloc_mu;
int g_alloc_after = 0, g_alloc_fail = 0;

int fail(dpo_ctx *c, int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c != nullptr)
        c->err = buf;
    else
        g_init_err = buf;
    return code;
}

int cuda_fail(dpo_ctx *c, cudaError_t e, const char *what)
{
    return fail(c, DPO_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool valid_dtype(int d) { return d == DPO_F32 || d == DPO_BF16; }
int64_t dt_size(dpo_dtype d) { return d == DPO_BF16 ? 2 : 4; }

// NAdam's momentum schedule mu_i = beta1 (1 - 0.5 * 0.96^(i psi)).
double nadam_mu(const dpo_hparams &hp, int64_t i)
{
    return (double)hp.beta1 * (1.0 - 0.5 * std::pow(0.96, (double)i * (double)hp.momentum_decay));
}

// fp32 state streams of a rule besides master: m, v (not Lion), n and
// grad_prev (Adan).
int rule_state_streams(int opt)
{
    switch (opt) {
    case DPO_OPT_LION:
        return 1;
    case DPO_OPT_ADAN:
        return 4;
    default:
        return 2;
    }
}
bool aligned(const void *p) { return (reinterpret_cast<uintptr_t>(p) % dpo::kAlign) == 0; }
// Stash kind of the fused step: none while the run is synchronous.
StashKind stash_kind(const dpo_ctx *c)
{
    if (c->hp.delay == 0)
        return dpo::kStashNone;
    return c->stash_dt == DPO_BF16 ? dpo::kStashBF16 : dpo::kStashF32;
}

// Ping-pong stash in use (delayed training).
bool pingpong_on(const dpo_ctx *c)
{
    return c->hp.stash_mode == DPO_STASH_PINGPONG && c->hp.delay == 1;
}

// Ping-pong stash: the latest weights of delayed tensors sit in the stash
// buffer after an odd number of calls of the current delayed phase.
// A capturable context's counters live on the device: refresh the host copy
// (after all work on the device so far), or write the host copy back.
int pull_counters(const dpo_ctx *c)
{
    if (!c->capturable)
        return DPO_OK;
    dpo::StepCounters h{};
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess)
        e = cudaMemcpy(&h, c->d_cnt, sizeof h, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return DPO_ECUDA;
    c->k = h.k;
    c->phase_k0 = h.phase_k0;
    c->mu_prod = h.mu_prod;
    return DPO_OK;
}

int push_counters(const dpo_ctx *c, cudaStream_t s)
{
    const dpo::StepCounters h{c->k, c->phase_k0, c->mu_prod};
    // pageable source: the call returns once the bytes are staged
    const cudaError_t e = cudaMemcpyAsync(c->d_cnt, &h, sizeof h, cudaMemcpyHostToDevice, s);
    return e == cudaSuccess ? DPO_OK : DPO_ECUDA;
}

bool latest_in_stash(const dpo_ctx *c)
{
    return pingpong_on(c) && ((c->k - c->phase_k0) & 1) != 0;
}

// Stash kind of the stash kernel: the buffers' dtype whenever they exist.
StashKind stash_buffer_kind(const dpo_ctx *c)
{
    if (!c->has_stash)
        return dpo::kStashNone;
    return c->stash_dt == DPO_BF16 ? dpo::kStashBF16 : dpo::kStashF32;
}

dpo::Correction correction_kind(bool ef, const dpo_hparams &hp)
{
    if (!ef || hp.delay != 1)
        return dpo::kCorrNone;
    switch (hp.correction) {
    case DPO_CORR_SAPIPE_SAME:
        return dpo::kCorrSapipeSame;
    case DPO_CORR_SAPIPE_UPDATED:
        return dpo::kCorrSapipeUpdated;
    default:
        return dpo::kCorrEF;
    }
}

struct Span {
    uintptr_t lo, hi;
    int tensor;
    const char *name;
    bool host_ok;   // grad and param may live in host memory the GPU can address
};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int grid_of(const dpo_ctx *c, int per_sm, int64_t pkts_per_cta)
{
    const int64_t groups = std::max<int64_t>(1, (c->total_pkts + pkts_per_cta - 1) / pkts_per_cta);
    return static_cast<int>(
        std::min<int64_t>(groups, (int64_t)std::max(1, c->sms) * std::max(1, per_sm)));
}

// Whether the fused step compensates gradients with DC-ASGD in the current
// mode (delayed training with a stash and a non-zero strength).
bool dc_on(const dpo_ctx *c)
{
    return stash_kind(c) != dpo::kStashNone && c->hp.dc_lambda != 0.0f;
}

// Grid of the fused step for the context's current mode: 128-thread CTAs,
// a measured number of them per SM. On the 7B-shaped bf16 set (GB300, 20
// timed steps per point, 2 to 8 CTAs per SM tried) the best were:
//                      standard rule   with an update history (EF, SAPipe)
//   AdamW, NAdam, Lion       4                     3
//   Adan                     3                     3
//   SAPipe updated state     -                     4 (Lion, Adan: 3)
//   Lion, ping-pong stash    4                     5
// the same with the copying and the ping-pong stash, except Lion with an
// update history: without the stash store its packets carry too few bytes
// for three CTAs to fill the memory system (ping-pong: 3 CTAs 85.2%, 4 95.0%,
// 5 99.0%, 6 96.6% of the copy peak; copying stash: 3 CTAs 98.0%).
// Three CTAs where packets also carry the history buffer keep about 55 KiB
// of loads in flight per SM; the standard rule loads less per packet and
// wants a fourth; Adan's two extra state streams make three enough; the
// SAPipe prediction's second Adam evaluation spaces the loads out and wants
// four (AdamW: 4 CTAs 98.1%, 3 88.1%; NAdam: 4 97.5%, 3 89.9%), but not
// Lion's, whose prediction is a sign, nor Adan's, whose packets already
// carry the two extra streams (on one box, 3 CTAs against 4: Lion 98.3%
// against 95.3%, Adan 97.6% against 94.0%). A table whose tensors mostly skip the history (DPO_SYNC, as WPipe's
// synchronous half) takes the standard rule's figure (measured: 4 CTAs 96.2%,
// 3 CTAs 93.7% of the copy peak with half the tensors synchronous).
int set_step_grid(dpo_ctx *c)
{
    const dpo::Correction corr = correction_kind(c->ef, c->hp);
    int per_sm = 0;
    const cudaError_t e = dpo::step_ctas_per_sm(
        static_cast<dpo::Optimizer>(c->hp.optimizer), c->param_dt == DPO_BF16, stash_kind(c),
        c->grad_dt == DPO_BF16, corr, dc_on(c), pingpong_on(c), &per_sm);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "occupancy query");
    int64_t hist_elems = 0;
    if (corr != dpo::kCorrNone)
        for (const dpo_tensor &t : c->table)
            if (!(t.flags & DPO_SYNC))
                hist_elems += t.numel;
    const bool mostly_hist = 4 * hist_elems >= 3 * c->total_elems && hist_elems > 0;
    int want;
    if (corr == dpo::kCorrSapipeUpdated)
        want = c->hp.optimizer == DPO_OPT_LION || c->hp.optimizer == DPO_OPT_ADAN ? 3 : 4;
    else if (c->hp.optimizer == DPO_OPT_ADAN)
        want = 3;
    else if (c->hp.optimizer == DPO_OPT_LION && pingpong_on(c) && mostly_hist)
        want = 5;
    else
        want = mostly_hist ? 3 : 4;
    c->step_grid = grid_of(c, std::min(per_sm, want), dpo::kStepThreads);
    return DPO_OK;
}

}  // namespace

extern "C" const char *dpo_last_error(const dpo_ctx *ctx)
{
    if (ctx == nullptr)
        return g_init_err.c_str();
    return ctx->err.c_str();
}

extern "C" int dpo_init(dpo_ctx **out, const dpo_tensor *table, int n_tensors,
                        dpo_dtype param_dtype, dpo_dtype stash_dtype, dpo_dtype grad_dtype,
                        const dpo_hparams *hp, int init_mode, void *cuda_stream)
{
    if (out == nullptr)
        return fail(nullptr, DPO_EINVAL, "out is NULL");
    *out = nullptr;
    if (hp == nullptr)
        return fail(nullptr, DPO_EINVAL, "hparams is NULL");
    if (n_tensors < 1 || table == nullptr)
        return fail(nullptr, DPO_EINVAL, "need a table of at least one tensor");
    if (!valid_dtype(param_dtype) || !valid_dtype(stash_dtype) || !valid_dtype(grad_dtype))
        return fail(nullptr, DPO_EDTYPE, "dtype must be DPO_F32 or DPO_BF16");
    if (init_mode != DPO_INIT_FRESH && init_mode != DPO_INIT_RESUME)
        return fail(nullptr, DPO_EINVAL, "init_mode must be DPO_INIT_FRESH or DPO_INIT_RESUME");
    if (hp->delay != 0 && hp->delay != 1)
        return fail(nullptr, DPO_EINVAL, "delay must be 0 or 1");
    const float reals[] = {hp->beta1, hp->beta2, hp->eps, hp->weight_decay, hp->ef_lambda,
                           hp->max_grad_norm};
    for (float r : reals)
        if (!std::isfinite(r))
            return fail(nullptr, DPO_EINVAL, "hyperparameters must be finite");
    if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f && hp->beta2 >= 0.0f && hp->beta2 < 1.0f))
        return fail(nullptr, DPO_EINVAL, "beta1 and beta2 must lie in [0, 1)");
    if (hp->eps < 0.0f || hp->weight_decay < 0.0f)
        return fail(nullptr, DPO_EINVAL, "eps and weight_decay must be >= 0");
    if (hp->correction != DPO_CORR_EF && hp->correction != DPO_CORR_SAPIPE_SAME &&
        hp->correction != DPO_CORR_SAPIPE_UPDATED)
        return fail(nullptr, DPO_EINVAL, "correction must be one of DPO_CORR_*");
    if (hp->optimizer < DPO_OPT_ADAMW || hp->optimizer > DPO_OPT_ADAN)
        return fail(nullptr, DPO_EINVAL, "optimizer must be one of DPO_OPT_*");
    if (!std::isfinite(hp->beta3) || !std::isfinite(hp->momentum_decay) ||
        !std::isfinite(hp->dc_lambda))
        return fail(nullptr, DPO_EINVAL, "hyperparameters must be finite");
    if (hp->optimizer == DPO_OPT_ADAN && !(hp->beta3 >= 0.0f && hp->beta3 < 1.0f))
        return fail(nullptr, DPO_EINVAL, "beta3 must lie in [0, 1)");
    if (hp->optimizer == DPO_OPT_NADAM && hp->momentum_decay < 0.0f)
        return fail(nullptr, DPO_EINVAL, "momentum_decay must be >= 0");
    if (hp->stash_mode != DPO_STASH_COPY && hp->stash_mode != DPO_STASH_PINGPONG)
        return fail(nullptr, DPO_EINVAL, "stash_mode must be one of DPO_STASH_*");
    if (hp->stash_mode == DPO_STASH_PINGPONG) {
        if (param_dtype != DPO_BF16 || stash_dtype != DPO_BF16)
            return fail(nullptr, DPO_EDTYPE, "the ping-pong stash needs bf16 param and stash buffers");
        if (hp->correction != DPO_CORR_EF)
            return fail(nullptr, DPO_EINVAL,
                        "the ping-pong stash needs the standard rule or EF (the SAPipe "
                        "corrections stash a prediction)");
    }

    // Table: NULL pointers, EF consistency, alignment, overlaps.
    const bool ef = table[0].ef != nullptr;
    bool has_stash = false, can_delay = true;
    std::vector<Span> spans;
    int64_t total_pkts = 0, total_elems = 0;
    for (int t = 0; t < n_tensors; ++t) {
        const dpo_tensor &d = table[t];
        if (d.numel < 0)
            return fail(nullptr, DPO_EINVAL, "tensor %d: numel < 0", t);
        if ((d.ef != nullptr) != ef)
            return fail(nullptr, DPO_EINVAL,
                        "tensor %d: EF buffers must be given for all tensors or for none", t);
        if ((d.flags & ~(DPO_WD_ON | DPO_SYNC)) != 0)
            return fail(nullptr, DPO_EINVAL, "tensor %d: unknown flags 0x%x", t, d.flags);
        if (d.numel == 0)
            continue;
        if (d.master == nullptr || d.m == nullptr || d.grad == nullptr ||
            (d.v == nullptr && hp->optimizer != DPO_OPT_LION))
            return fail(nullptr, DPO_EINVAL, "tensor %d: master, m, v and grad are required", t);
        if (hp->optimizer == DPO_OPT_ADAN && (d.n == nullptr || d.grad_prev == nullptr))
            return fail(nullptr, DPO_EINVAL, "tensor %d: Adan needs the n and grad_prev buffers", t);
        if (hp->delay == 1 && d.stash == nullptr && !(d.flags & DPO_SYNC))
            return fail(nullptr, DPO_EINVAL, "tensor %d: delay = 1 needs a stash buffer", t);
        if (d.stash != nullptr)
            has_stash = true;
        else if (!(d.flags & DPO_SYNC))
            can_delay = false;
        if (param_dtype == DPO_BF16 && d.param == nullptr)
            return fail(nullptr, DPO_EINVAL, "tensor %d: bf16 params need a param buffer", t);
        if (param_dtype == DPO_F32 && d.param != nullptr)
            return fail(nullptr, DPO_EINVAL,
                        "tensor %d: with fp32 params the master is the latest copy; param must be NULL",
                        t);
        const struct {
            const void *p;
            int64_t bytes;
            const char *name;
            bool host_ok;
        } bufs[] = {
            {d.master, 4 * d.numel, "master", false},
            {d.m, 4 * d.numel, "m", false},
            {hp->optimizer == DPO_OPT_LION ? nullptr : d.v, 4 * d.numel, "v", false},
            {hp->optimizer == DPO_OPT_ADAN ? d.n : nullptr, 4 * d.numel, "n", false},
            {hp->optimizer == DPO_OPT_ADAN ? d.grad_prev : nullptr, 4 * d.numel, "grad_prev",
             false},
            {d.grad, dt_size(grad_dtype) * d.numel, "grad", true},
            {d.param, dt_size(param_dtype) * d.numel, "param", true},
            {d.stash, dt_size(stash_dtype) * d.numel, "stash", false},
            {d.ef, 4 * d.numel, "ef", false},
        };
        for (const auto &b : bufs) {
            if (b.p == nullptr)
                continue;
            if (!aligned(b.p))
                return fail(nullptr, DPO_EALIGN, "tensor %d: %s is not %d-byte aligned", t,
                            b.name, dpo::kAlign);
            const uintptr_t lo = reinterpret_cast<uintptr_t>(b.p);
            spans.push_back({lo, lo + static_cast<uintptr_t>(b.bytes), t, b.name, b.host_ok});
        }
        total_pkts += (d.numel + dpo::kPacket - 1) / dpo::kPacket;
        total_elems += d.numel;
    }
    if (hp->ef_lambda != 0.0f && !ef)
        return fail(nullptr, DPO_EINVAL, "ef_lambda != 0 needs EF buffers");
    std::sort(spans.begin(), spans.end(),
              [](const Span &a, const Span &b) { return a.lo < b.lo; });
    for (size_t i = 1; i < spans.size(); ++i)
        if (spans[i].lo < spans[i - 1].hi)
            return fail(nullptr, DPO_EINVAL, "buffers overlap: tensor %d %s and tensor %d %s",
                        spans[i - 1].tensor, spans[i - 1].name, spans[i].tensor, spans[i].name);

    // Residency: the optimizer state must be device memory of the current
    // device. grad and param may instead be host memory the GPU addresses
    // directly (pinned and mapped at the same address, or pageable memory on
    // a device with pageable-memory access, e.g. over NVLink-C2C); the fused
    // kernel then reads the gradients and writes the new weights across the
    // host link itself.
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess)
        return cuda_fail(nullptr, e, "cudaGetDevice");
    int pageable_ok = 0;
    cudaDeviceGetAttribute(&pageable_ok, cudaDevAttrPageableMemoryAccess, device);
    bool host_io = false, host_param = false;
    for (const Span &s : spans) {
        cudaPointerAttributes attr{};
        const void *ptr = reinterpret_cast<const void *>(s.lo);
        e = cudaPointerGetAttributes(&attr, ptr);
        if (e != cudaSuccess)
            return cuda_fail(nullptr, e, "cudaPointerGetAttributes");
        const bool on_device = (attr.type == cudaMemoryTypeDevice ||
                                attr.type == cudaMemoryTypeManaged) && attr.device == device;
        const bool host_mapped = attr.type == cudaMemoryTypeHost && attr.devicePointer == ptr;
        const bool host_pageable = attr.type == cudaMemoryTypeUnregistered && pageable_ok;
        if (on_device)
            continue;
        if (s.host_ok && (host_mapped || host_pageable)) {
            host_io = true;
            host_param = host_param || std::strcmp(s.name, "param") == 0;
            continue;
        }
        return fail(nullptr, DPO_EINVAL,
                    s.host_ok ? "tensor %d: %s is neither device memory of the current device "
                                "nor host memory this device can address"
                              : "tensor %d: %s is not device memory of the current device",
                    s.tensor, s.name);
    }

    if (hp->stash_mode == DPO_STASH_PINGPONG && host_param)
        return fail(nullptr, DPO_EINVAL, "the ping-pong stash needs device param buffers");

    dpo_ctx *c = new (std::nothrow) dpo_ctx;
    if (c == nullptr)
        return fail(nullptr, DPO_ENOMEM, "out of host memory");
    c->device = device;
    c->n = n_tensors;
    c->param_dt = param_dtype;
    c->stash_dt = stash_dtype;
    c->grad_dt = grad_dtype;
    c->hp = *hp;
    c->ef = ef;
    c->clip = hp->max_grad_norm > 0.0f;
    c->total_pkts = total_pkts;
    c->total_elems = total_elems;
    c->host_io = host_io;
    c->has_stash = has_stash;
    c->can_delay = can_delay && has_stash;
    c->table.assign(table, table + n_tensors);

    // Launch geometry: persistent grids, a fixed number of resident CTAs per
    // SM, never more CTAs than there are CTA-widths of packets (set_step_grid
    // for the fused step).
    int per_sm_norm = 0;
    cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, device);
    e = dpo::norm_ctas_per_sm(grad_dtype == DPO_BF16, &per_sm_norm);
    if (e != cudaSuccess) {
        int rc = cuda_fail(nullptr, e, "occupancy query");
        delete c;
        return rc;
    }
    if (set_step_grid(c) != DPO_OK) {
        g_init_err = c->err;
        delete c;
        return DPO_ECUDA;
    }
    c->norm_grid = grid_of(c, per_sm_norm, (int64_t)dpo::kNormThreads * dpo::kNormUnroll);
    c->stash_grid = c->step_grid;

    // Device block: table, packet prefix, norm scratch.
    const size_t off_table = 0;
    const size_t off_pkt = align_up(off_table + sizeof(DevTensor) * n_tensors, 256);
    const size_t off_part = align_up(off_pkt + sizeof(int64_t) * (n_tensors + 1), 256);
    const size_t off_scal = align_up(off_part + sizeof(double) * c->norm_grid, 256);
    const size_t off_cnt = align_up(off_scal + sizeof(dpo::NormScalars), 256);
    const size_t off_sc = align_up(off_cnt + sizeof(dpo::StepCounters), 256);
    const size_t bytes = off_sc + sizeof(dpo::StepScalars);
    e = dpo::device_alloc(&c->dev_block, bytes);
    if (e != cudaSuccess) {
        cudaGetLastError();
        fail(nullptr, DPO_ENOMEM, "cudaMalloc of %zu bytes: %s", bytes, cudaGetErrorString(e));
        delete c;
        return DPO_ENOMEM;
    }
    char *base = static_cast<char *>(c->dev_block);
    c->d_table = reinterpret_cast<DevTensor *>(base + off_table);
    c->d_pkt_begin = reinterpret_cast<int64_t *>(base + off_pkt);
    c->d_partials = reinterpret_cast<double *>(base + off_part);
    c->d_scalars = reinterpret_cast<dpo::NormScalars *>(base + off_scal);
    c->d_cnt = reinterpret_cast<dpo::StepCounters *>(base + off_cnt);
    c->d_sc = reinterpret_cast<dpo::StepScalars *>(base + off_sc);

    std::vector<DevTensor> dt(n_tensors);
    std::vector<int64_t> pkt(n_tensors + 1, 0);
    for (int t = 0; t < n_tensors; ++t) {
        const dpo_tensor &d = table[t];
        DevTensor &x = dt[t];
        x.param = d.param;
        x.master = d.master;
        x.m = d.m;
        x.v = d.v;
        x.stash = d.stash;
        x.ef = d.ef;
        x.grad = d.grad;
        x.v = hp->optimizer == DPO_OPT_LION ? nullptr : d.v;
        x.n = hp->optimizer == DPO_OPT_ADAN ? d.n : nullptr;
        x.grad_prev = hp->optimizer == DPO_OPT_ADAN ? d.grad_prev : nullptr;
        x.numel = d.numel;
        x.flags = d.flags;
        x.pad_ = 0;
        pkt[t + 1] = pkt[t] + (d.numel + dpo::kPacket - 1) / dpo::kPacket;
    }
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    e = cudaMemcpyAsync(c->d_table, dt.data(), sizeof(DevTensor) * n_tensors,
                        cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(c->d_pkt_begin, pkt.data(), sizeof(int64_t) * (n_tensors + 1),
                            cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(base + off_part, 0, bytes - off_part, s);
    // The pageable host copies above are staged before cudaMemcpyAsync
    // returns, so dt and pkt may go out of scope afterwards.
    if (e != cudaSuccess) {
        int rc = cuda_fail(nullptr, e, "uploading the tensor table");
        cudaFree(c->dev_block);
        delete c;
        return rc;
    }
    if (init_mode == DPO_INIT_FRESH && total_pkts > 0) {
        dpo::StashArgs a{c->d_table, c->d_pkt_begin, n_tensors, total_pkts, 1, 1};
        e = dpo::launch_stash(param_dtype == DPO_BF16, stash_buffer_kind(c), c->stash_grid, a,
                              s);
        if (e != cudaSuccess) {
            int rc = cuda_fail(nullptr, e, "launching the initial stash");
            cudaFree(c->dev_block);
            delete c;
            return rc;
        }
    }
    *out = c;
    return DPO_OK;
}

extern "C" int dpo_stash(dpo_ctx *c, void *cuda_stream)
{
    if (c == nullptr)
        return fail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (c->total_pkts == 0)
        return DPO_OK;
    dpo::StashArgs a{c->d_table, c->d_pkt_begin, c->n, c->total_pkts, 0, 0};
    const cudaError_t e = dpo::launch_stash(c->param_dt == DPO_BF16, stash_buffer_kind(c),
                                            c->stash_grid, a,
                                            static_cast<cudaStream_t>(cuda_stream));
    return e == cudaSuccess ? DPO_OK : cuda_fail(c, e, "stash launch");
}

extern "C" int dpo_set_delay(dpo_ctx *c, int delay, void *cuda_stream)
{
    if (c == nullptr)
        return fail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (delay != 0 && delay != 1)
        return fail(c, DPO_EINVAL, "delay must be 0 or 1");
    if (delay == c->hp.delay)
        return DPO_OK;
    if (pull_counters(c) != DPO_OK)
        return fail(c, DPO_ECUDA, "reading the device step counters failed");
    if (delay == 1) {
        if (!c->can_delay)
            return fail(c, DPO_ESTATE,
                        "delayed training needs a stash buffer for every tensor without DPO_SYNC");
        if (c->total_pkts > 0) {
            // stash := the current weights, update history := 0: Alg. 1 restarts
            dpo::StashArgs a{c->d_table, c->d_pkt_begin, c->n, c->total_pkts, 0, 1};
            const cudaError_t e =
                dpo::launch_stash(c->param_dt == DPO_BF16, stash_buffer_kind(c), c->stash_grid, a,
                                  static_cast<cudaStream_t>(cuda_stream));
            if (e != cudaSuccess)
                return cuda_fail(c, e, "stash launch");
        }
        c->phase_k0 = c->k;
        if (c->capturable && push_counters(c, static_cast<cudaStream_t>(cuda_stream)) != DPO_OK)
            return fail(c, DPO_ECUDA, "writing the device step counters failed");
    } else if (latest_in_stash(c) && c->total_pkts > 0) {
        // Ping-pong: the latest weights sit in the stash buffer; synchronous
        // training keeps them in the param buffer (param := bf16(master)).
        dpo::StashArgs a{c->d_table, c->d_pkt_begin, c->n, c->total_pkts, 0, 0};
        const cudaError_t e = dpo::launch_stash(true, stash_buffer_kind(c), c->stash_grid, a,
                                                static_cast<cudaStream_t>(cuda_stream));
        if (e != cudaSuccess)
            return cuda_fail(c, e, "stash launch");
    }
    c->hp.delay = delay;
    const int rc = set_step_grid(c);
    return rc;
}

extern "C" int dpo_step(dpo_ctx *c, float lr, void *cuda_stream)
{
    if (c == nullptr)
        return fail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (!std::isfinite(lr) || lr < 0.0f)
        return fail(c, DPO_EINVAL, "lr must be finite and >= 0");
    const int64_t k = c->k + 1;        // this call consumes the k-th gradient
    const int64_t t = k - c->phase_k0; // Alg. 1 iteration within the delayed phase
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    cudaEvent_t ev_mid = nullptr, ev_end = nullptr;
    if (c->timing && c->total_pkts > 0) {
        while (c->ev_used + 3 > c->ev_pool.size()) {
            cudaEvent_t ev;
            const cudaError_t e = cudaEventCreate(&ev);
            if (e != cudaSuccess)
                return cuda_fail(c, e, "timing event");
            c->ev_pool.push_back(ev);
        }
        const cudaError_t e = cudaEventRecord(c->ev_pool[c->ev_used], s);
        if (e != cudaSuccess)
            return cuda_fail(c, e, "timing event record");
        ev_mid = c->ev_pool[c->ev_used + 1];
        ev_end = c->ev_pool[c->ev_used + 2];
        c->ev_used += 3;
    }
    if (c->total_pkts > 0) {
        if (c->clip && c->clip_src != nullptr) {
            const cudaError_t e = dpo::launch_clip_from_sumsq(
                c->clip_src, (double)c->hp.max_grad_norm, c->d_scalars, s);
            if (e != cudaSuccess)
                return cuda_fail(c, e, "clip-coefficient launch");
        } else if (c->clip) {
            dpo::NormArgs na{c->d_table, c->d_pkt_begin, c->n, c->total_pkts,
                             (double)c->hp.max_grad_norm, c->d_partials, c->d_scalars,
                             nullptr};
            const cudaError_t e = dpo::launch_norm(c->grad_dt == DPO_BF16, c->norm_grid, na, s);
            if (e != cudaSuccess)
                return cuda_fail(c, e, "gradient-norm launch");
        }
        const double b1 = c->hp.beta1, b2 = c->hp.beta2, b3 = c->hp.beta3, lrd = lr;
        const double bc1 = 1.0 - std::pow(b1, (double)k);
        const double bc2 = 1.0 - std::pow(b2, (double)k);
        const dpo::Correction corr = correction_kind(c->ef, c->hp);
        dpo::StepArgs a{};
        a.table = c->d_table;
        a.pkt_begin = c->d_pkt_begin;
        a.n_tensors = c->n;
        a.total_pkts = c->total_pkts;
        a.beta1 = c->hp.beta1;
        a.omb1 = (float)(1.0 - b1);
        a.beta2 = c->hp.beta2;
        a.omb2 = (float)(1.0 - b2);
        a.step_size = (float)(lrd / bc1);
        a.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(bc2));
        a.eps = c->hp.eps;
        a.lr_wd = (float)(lrd * (double)c->hp.weight_decay);
        // Alg. 1: the standard rule for t <= 1, i.e. at the first update.
        a.lam = (corr == dpo::kCorrEF && t >= 2) ? c->hp.ef_lambda : 0.0f;
        a.step_size_next = (float)(lrd / (1.0 - std::pow(b1, (double)(k + 1))));
        a.inv_sqrt_bc2_next = (float)(1.0 / std::sqrt(1.0 - std::pow(b2, (double)(k + 1))));
        a.lr = lr;
        const double mu_k = nadam_mu(c->hp, k), mu_next = nadam_mu(c->hp, k + 1);
        const double mu_prod = c->mu_prod * mu_k;
        a.nadam_cg = (float)(lrd * (1.0 - mu_k) / (1.0 - mu_prod));
        a.nadam_cm = (float)(lrd * mu_next / (1.0 - mu_prod * mu_next));
        a.beta3 = c->hp.beta3;
        a.omb3 = (float)(1.0 - b3);
        a.inv_sqrt_bc3 = (float)(1.0 / std::sqrt(1.0 - std::pow(b3, (double)k)));
        a.adan_c2 = (float)(lrd * b2 / bc2);
        // the same at the next index, for the SAPipe updated-state prediction
        const double mu_next2 = nadam_mu(c->hp, k + 2);
        a.nadam_cg_next = (float)(lrd * (1.0 - mu_next) / (1.0 - mu_prod * mu_next));
        a.nadam_cm_next = (float)(lrd * mu_next2 / (1.0 - mu_prod * mu_next * mu_next2));
        a.inv_sqrt_bc3_next = (float)(1.0 / std::sqrt(1.0 - std::pow(b3, (double)(k + 1))));
        a.adan_c2_next = (float)(lrd * b2 / (1.0 - std::pow(b2, (double)(k + 1))));
        a.first = k == 1;
        a.dc_lambda = c->hp.delay == 1 ? c->hp.dc_lambda : 0.0f;
        // Ping-pong: call t of the delayed phase writes the new weights of
        // delayed tensors into the buffer holding x_{t-1}: the stash buffer
        // when t is odd, the param buffer when t is even.
        a.swap = pingpong_on(c) && (t & 1) != 0;
        a.clip = c->clip ? &c->d_scalars->clip : nullptr;
        if (c->capturable) {   // the per-call scalars come from the device counters
            const dpo::ScalarConsts kc{c->hp.beta1, c->hp.beta2, c->hp.beta3, c->hp.weight_decay,
                                       c->hp.momentum_decay, c->hp.ef_lambda,
                                       corr == dpo::kCorrEF ? 1 : 0, pingpong_on(c) ? 1 : 0};
            const cudaError_t es = dpo::launch_step_scalars(c->d_cnt, c->lr_src, lr, kc, c->d_sc, s);
            if (es != cudaSuccess)
                return cuda_fail(c, es, "step-scalars launch");
            a.dev = c->d_sc;
        }
        if (ev_mid != nullptr) {
            const cudaError_t et = cudaEventRecord(ev_mid, s);
            if (et != cudaSuccess)
                return cuda_fail(c, et, "timing event record");
        }
        const cudaError_t e = dpo::launch_step(static_cast<dpo::Optimizer>(c->hp.optimizer),
                                               c->param_dt == DPO_BF16, stash_kind(c),
                                               c->grad_dt == DPO_BF16, corr, dc_on(c),
                                               pingpong_on(c), c->step_grid, a, s);
        if (e != cudaSuccess)
            return cuda_fail(c, e, "fused step launch");
        if (ev_end != nullptr) {
            const cudaError_t et = cudaEventRecord(ev_end, s);
            if (et != cudaSuccess)
                return cuda_fail(c, et, "timing event record");
        }
    }
    if (c->capturable) {
        if (c->total_pkts == 0) {   // nothing launched: keep the device counter in step
            const dpo::ScalarConsts kc{c->hp.beta1, c->hp.beta2, c->hp.beta3, c->hp.weight_decay,
                                       c->hp.momentum_decay, c->hp.ef_lambda, 0, 0};
            const cudaError_t es = dpo::launch_step_scalars(c->d_cnt, c->lr_src, lr, kc, c->d_sc, s);
            if (es != cudaSuccess)
                return cuda_fail(c, es, "step-scalars launch");
        }
        return DPO_OK;   // the device counters advanced
    }
    c->mu_prod *= nadam_mu(c->hp, k);
    c->k = k;
    return DPO_OK;
}

extern "C" int dpo_set_capturable(dpo_ctx *c, int on, const float *lr_source, void *cuda_stream)
{
    if (c == nullptr)
        return fail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (lr_source != nullptr && reinterpret_cast<uintptr_t>(lr_source) % alignof(float) != 0)
        return fail(c, DPO_EINVAL, "lr_source must be 4-byte aligned");
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    if (on) {
        if (!c->capturable && push_counters(c, s) != DPO_OK)
            return fail(c, DPO_ECUDA, "writing the device step counters failed");
        c->capturable = true;
        c->lr_src = lr_source;
    } else {
        if (c->capturable && pull_counters(c) != DPO_OK)
            return fail(c, DPO_ECUDA, "reading the device step counters failed");
        c->capturable = false;
        c->lr_src = nullptr;
    }
    return DPO_OK;
}

cudaError_t dpo::device_alloc(void **p, size_t bytes)
{
    {
        std::lock_guard<std::mutex> lock(g_alloc_mu);
        if (g_alloc_fail > 0) {
            if (g_alloc_after > 0) {
                --g_alloc_after;
            } else {
                --g_alloc_fail;
                *p = nullptr;
                return cudaErrorMemoryAllocation;
            }
        }
    }
    return cudaMalloc(p, bytes);
}

extern "C" int dpo_test_fail_allocs(int after, int count)
{
    if (after < 0 || count < 0)
        return DPO_EINVAL;
    std::lock_guard<std::mutex> lock(g_alloc_mu);
    g_alloc_after = after;
    g_alloc_fail = count;
    return DPO_OK;
}

extern "C" int dpo_grad_sqnorm(dpo_ctx *c, double *d_sumsq, void *cuda_stream)
{
    if (c == nullptr)
        return fail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (d_sumsq == nullptr || reinterpret_cast<uintptr_t>(d_sumsq) % alignof(double) != 0)
        return fail(c, DPO_EINVAL, "d_sumsq must be an 8-byte aligned device pointer");
    if (c->total_pkts == 0)
        return DPO_OK;
    dpo::NormArgs na{c->d_table, c->d_pkt_begin, c->n, c->total_pkts, 0.0, c->d_partials,
                     c->d_scalars, d_sumsq};
    const cudaError_t e = dpo::launch_norm(c->grad_dt == DPO_BF16, c->norm_grid, na,
                                           static_cast<cudaStream_t>(cuda_stream));
    if (e != cudaSuccess)
        return cuda_fail(c, e, "gradient-norm launch");
    return DPO_OK;
}

extern "C" int dpo_set_clip_source(dpo_ctx *c, const double *d_sumsq)
{
    if (c == nullptr)
        return fail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (d_sumsq != nullptr && reinterpret_cast<uintptr_t>(d_sumsq) % alignof(double) != 0)
        return fail(c, DPO_EINVAL, "d_sumsq must be 8-byte aligned");
    if (d_sumsq != nullptr && !c->clip)
        return fail(c, DPO_ESTATE, "a clip source needs max_grad_norm > 0");
    c->clip_src = d_sumsq;
    return DPO_OK;
}

extern "C" int dpo_read_weights(const dpo_ctx *c, int which, int tensor, const void **ptr,
                                dpo_dtype *dtype)
{
    if (c == nullptr || ptr == nullptr)
        return DPO_EINVAL;
    if (tensor < 0 || tensor >= c->n || (which != DPO_STALE && which != DPO_LATEST))
        return DPO_EINVAL;
    const dpo_tensor &d = c->table[tensor];
    if (pingpong_on(c) && pull_counters(c) != DPO_OK)
        return DPO_ECUDA;
    // Ping-pong: after an odd number of delayed calls the two buffers of a
    // delayed tensor hold each other's role.
    const bool swapped = latest_in_stash(c) && !(d.flags & DPO_SYNC);
    if (which == DPO_STALE && c->hp.delay == 1 && !(d.flags & DPO_SYNC)) {
        *ptr = swapped ? d.param : d.stash;
        if (dtype)
            *dtype = c->stash_dt;
    } else if (c->param_dt == DPO_BF16) {
        *ptr = swapped ? d.stash : d.param;
        if (dtype)
            *dtype = DPO_BF16;
    } else {
        *ptr = d.master;
        if (dtype)
            *dtype = DPO_F32;
    }
    return DPO_OK;
}

extern "C" int dpo_get_step(const dpo_ctx *c, int64_t *k)
{
    if (c == nullptr || k == nullptr)
        return DPO_EINVAL;
    if (pull_counters(c) != DPO_OK)
        return DPO_ECUDA;
    *k = c->k;
    return DPO_OK;
}

extern "C" int dpo_set_step(dpo_ctx *c, int64_t k)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (k < 0)
        return fail(c, DPO_EINVAL, "step counter must be >= 0");
    if (pull_counters(c) != DPO_OK)   // the phase start stays as it is
        return fail(c, DPO_ECUDA, "reading the device step counters failed");
    c->k = k;
    c->mu_prod = 1.0;   // NAdam's running product, rebuilt for the restored counter
    for (int64_t i = 1; i <= k; ++i)
        c->mu_prod *= nadam_mu(c->hp, i);
    if (c->phase_k0 > k)
        c->phase_k0 = k;
    if (c->capturable && (push_counters(c, nullptr) != DPO_OK ||
                          cudaDeviceSynchronize() != cudaSuccess))
        return fail(c, DPO_ECUDA, "writing the device step counters failed");
    return DPO_OK;
}

extern "C" int dpo_get_phase_start(const dpo_ctx *c, int64_t *k0)
{
    if (c == nullptr || k0 == nullptr)
        return DPO_EINVAL;
    if (pull_counters(c) != DPO_OK)
        return DPO_ECUDA;
    *k0 = c->phase_k0;
    return DPO_OK;
}

extern "C" int dpo_set_phase_start(dpo_ctx *c, int64_t k0)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (pull_counters(c) != DPO_OK)
        return fail(c, DPO_ECUDA, "reading the device step counters failed");
    if (k0 < 0 || k0 > c->k)
        return fail(c, DPO_EINVAL, "phase start must lie in [0, k]");
    c->phase_k0 = k0;
    if (c->capturable && (push_counters(c, nullptr) != DPO_OK ||
                          cudaDeviceSynchronize() != cudaSuccess))
        return fail(c, DPO_ECUDA, "writing the device step counters failed");
    return DPO_OK;
}

extern "C" int dpo_get_flags(dpo_ctx *c, uint32_t *flags, double *grad_norm, float *clip_scale,
                             void *cuda_stream)
{
    if (c == nullptr)
        return DPO_EINVAL;
    dpo::NormScalars h{};
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    cudaError_t e = cudaMemcpyAsync(&h, c->d_scalars, sizeof h, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(&c->d_scalars->flags, 0, sizeof(unsigned int), s);   // read clears
    if (e == cudaSuccess)
        e = cudaStreamSynchronize(s);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "reading diagnostics");
    if (flags)
        *flags = h.flags;
    if (grad_norm)
        *grad_norm = h.norm;
    if (clip_scale)
        *clip_scale = c->clip ? h.clip : 1.0f;
    return DPO_OK;
}

extern "C" int dpo_algorithmic_bytes(const dpo_ctx *c, int64_t *step_bytes, int64_t *norm_bytes)
{
    if (c == nullptr)
        return DPO_EINVAL;
    // Per element: read master, m, v (fp32) and grad; write master, m, v and
    // the bf16 param; a delayed tensor also writes its stash, and under a
    // correction reads and writes its update-history buffer.
    const int64_t base = 8 * (1 + rule_state_streams(c->hp.optimizer)) + dt_size(c->grad_dt) +
                         (c->param_dt == DPO_BF16 ? 2 : 0);
    // (the ping-pong stash writes no stash; DC-ASGD reads it)
    const int stash_writes = c->hp.stash_mode == DPO_STASH_PINGPONG ? 0 : 1;
    const int64_t delayed_extra =
        c->hp.delay == 1
            ? dt_size(c->stash_dt) * (stash_writes + (c->hp.dc_lambda != 0.0f ? 1 : 0)) +
                  (c->ef ? 8 : 0)
            : 0;
    int64_t total = 0;
    for (const dpo_tensor &d : c->table)
        total += d.numel * (base + ((d.flags & DPO_SYNC) ? 0 : delayed_extra));
    if (step_bytes)
        *step_bytes = total;
    if (norm_bytes)
        *norm_bytes = c->clip && c->clip_src == nullptr ? dt_size(c->grad_dt) * c->total_elems
                                                        : 0;
    return DPO_OK;
}

extern "C" int dpo_launch_config(const dpo_ctx *c, int *step_ctas, int *norm_ctas, int *threads)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (step_ctas)
        *step_ctas = c->step_grid;
    if (norm_ctas)
        *norm_ctas = c->norm_grid;
    if (threads)
        *threads = dpo::kStepThreads;
    return DPO_OK;
}

extern "C" int dpo_set_timing(dpo_ctx *c, int on)
{
    if (c == nullptr)
        return DPO_EINVAL;
    c->timing = on != 0;
    return DPO_OK;
}

extern "C" int dpo_get_timing(dpo_ctx *c, double *norm_ms, double *step_ms, int64_t *calls)
{
    if (c == nullptr || norm_ms == nullptr || step_ms == nullptr || calls == nullptr)
        return DPO_EINVAL;
    double tn = 0.0, ts = 0.0;
    for (size_t q = 0; q + 3 <= c->ev_used; q += 3) {
        float a = 0.0f, b = 0.0f;
        cudaError_t e = cudaEventSynchronize(c->ev_pool[q + 2]);
        if (e == cudaSuccess)
            e = cudaEventElapsedTime(&a, c->ev_pool[q], c->ev_pool[q + 1]);
        if (e == cudaSuccess)
            e = cudaEventElapsedTime(&b, c->ev_pool[q + 1], c->ev_pool[q + 2]);
        if (e != cudaSuccess)
            return cuda_fail(c, e, "timing event read");
        tn += a;
        ts += b;
    }
    *norm_ms = tn;
    *step_ms = ts;
    *calls = (int64_t)(c->ev_used / 3);
    c->ev_used = 0;
    return DPO_OK;
}

extern "C" void dpo_destroy(dpo_ctx *c)
{
    if (c == nullptr)
        return;
    for (cudaEvent_t e : c->ev_pool)
        cudaEventDestroy(e);
    if (c->dev_block != nullptr)
        cudaFree(c->dev_block);
    delete c;
}
