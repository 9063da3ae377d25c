// dpo_muon.cu -- one-step-delayed Muon (Alg. 2 of arXiv 2606.30634) on the
// sm_103a tensor cores: kernels, Newton-Schulz driver and the C ABI of
// dpo_muon.h.
//
// Per step, in stream order:
//   grad_sqnorm_kernel      global ||G||^2 for clipping (shared with the
//                           elementwise path), when clipping is on
//   muon_momentum_kernel    M <- mu M + (1 - mu) G^, and per-chunk partial
//                           sums of M^2 (fixed chunks: deterministic)
//   muon_norm_kernel        ||M||_F per matrix from its partials, in order
//   muon_normalize_kernel   X_0 = bf16(M / (||M||_F + eps)) into the padded
//                           workspace, in the wide orientation (64 x 64 tiles
//                           through shared memory)
//   ns_gemm_kernel x 3 per Newton-Schulz step and matrix shape, batched over
//                           every matrix of that shape (dpo_gemm.cuh):
//                             A = X X^T;  B = c A A + b A;  X <- B X + a X
//                           (the third reads X MN-major; at the last step it
//                           also writes X^T, the output of tall matrices)
//   muon_apply_kernel       U = lr (r O + wd X_t) and the delayed or EF
//                           update, stash, history and bf16 weights
// With the SAPipe-WP updated-state prediction (App. B.1) the step then runs
// the pipeline once more for the prediction update: the momentum kernel
// forms M' = mu M + (1 - mu) G^ into the history buffer, M' is normalised and
// put through a second Newton-Schulz chain, and muon_predict_kernel writes
// U' = lr (r O' + wd X_{t+1}) into the history.
#include "dpo_muon.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "dpo_device.cuh"
#include "dpo_gemm.cuh"

namespace dpo {
namespace muon {

constexpr int kThreads = 256;
constexpr int64_t kChunk = (int64_t)kThreads * kPacket * 16;  // elements per momentum CTA
constexpr int kPad = 256;                                       // workspace padding

struct DevMat {
    void *param;
    float *master, *mom;
    void *stash;
    float *ef;
    const void *grad;
    int64_t rows, cols;
    const __nv_bfloat16 *o;   // Newton-Schulz output (workspace), row-major, pitch o_ld
    int64_t o_ld;
    float wd_lr_scale;        // 1 with DPO_WD_ON, else 0
    float r_scale;            // rms_scale sqrt(max(rows, cols)), or 1
    int sync;                 // DPO_SYNC: trained synchronously (no stash, no history)
};

struct MomArgs {
    const DevMat *mats;
    const float *clip;        // device clip coefficient, or nullptr
    float mu, omm;
    double *partials;         // [n_mats][chunks]
    int chunks;
    int predict;              // M' = mu M + (1 - mu) G^ into the history buffer of each
                              // delayed matrix; M keeps its value
};

template <class GT>
__global__ void __launch_bounds__(kThreads) muon_momentum_kernel(const MomArgs a)
{
    __shared__ double red[kThreads / 32];
    const DevMat &d = a.mats[blockIdx.y];
    // the prediction pass leaves a synchronous matrix (and its history) alone
    const bool skip = a.predict && (d.sync || d.ef == nullptr);
    const int64_t n = skip ? 0 : d.rows * d.cols;
    float *out = a.predict ? d.ef : d.mom;
    const int64_t lo = (int64_t)blockIdx.x * kChunk;
    float sum = 0.0f, comp = 0.0f;
    if (lo < n) {
        const float clip = a.clip != nullptr ? __ldg(a.clip) : 1.0f;
        const int64_t hi = lo + kChunk < n ? lo + kChunk : n;
        const GT *grad = static_cast<const GT *>(d.grad);
        for (int64_t e = lo + (int64_t)threadIdx.x * kPacket; e < hi; e += (int64_t)kThreads * kPacket) {
            if (e + kPacket <= hi) {
                float m[8], g[8];
                ld8(d.mom + e, m);
                ld8(grad + e, g);
                float s = 0.0f;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float gc = g[j] * clip;
                    const float p = a.omm * gc;
                    m[j] = fmaf(a.mu, m[j], p) + fmaf(a.omm, gc, -p);
                    s = fmaf(m[j], m[j], s);
                }
                st8(out + e, m);
                const float y = s - comp, t = sum + y;   // Kahan
                comp = (t - sum) - y;
                sum = t;
            } else {
                for (int64_t i = e; i < hi; ++i) {
                    const float gc = ld1(grad + i) * clip;
                    const float p = a.omm * gc;
                    const float m = fmaf(a.mu, d.mom[i], p) + fmaf(a.omm, gc, -p);
                    out[i] = m;
                    const float y = m * m - comp, t = sum + y;
                    comp = (t - sum) - y;
                    sum = t;
                }
            }
        }
    }
    double x = (double)sum - (double)comp;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
        x += __shfl_down_sync(0xFFFFFFFFu, x, off);
    if ((threadIdx.x & 31) == 0)
        red[threadIdx.x >> 5] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
        double s = 0.0;
        for (int w = 0; w < kThreads / 32; ++w)
            s += red[w];
        a.partials[(int64_t)blockIdx.y * a.chunks + blockIdx.x] = s;
    }
}

// 1 / (||M||_F + eps) per matrix: one warp per matrix sums its partials in a
// fixed order (lane-strided, then a fixed shuffle tree).
__global__ void muon_norm_kernel(const double *partials, int chunks, int n_mats, float eps,
                                 float *inv_norm)
{
    const int mat = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (mat >= n_mats)
        return;
    double s = 0.0;
    for (int c = lane; c < chunks; c += 32)
        s += partials[(int64_t)mat * chunks + c];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
        s += __shfl_down_sync(0xFFFFFFFFu, s, off);
    if (lane == 0)
        inv_norm[mat] = (float)(1.0 / (sqrt(s) + (double)eps));
}

struct NormArgsM {
    const DevMat *mats;
    const int *group_mats;    // global matrix index of each batch entry
    const float *inv_norm;
    __nv_bfloat16 *x, *xt;    // X (R x W) and X^T (W x R, or nullptr) of batch entry 0
    int64_t R, W;
    int64_t r, w;
    int predict;              // read M' from the history buffer (zeros for a
                              // synchronous matrix) instead of M
};

// One 64 x 64 tile of X (rows i over r, columns j over w) per CTA; padding
// outside r x w is written as zero. M is read along its own rows (32-byte
// fp32 vectors where the row pitch allows) and X written along its rows
// (16-byte bf16 vectors), through a shared-memory tile that transposes the
// tall matrices.
__global__ void __launch_bounds__(kThreads) muon_normalize_kernel(const NormArgsM a)
{
    __shared__ float tile[64][65];
    const int bz = blockIdx.z;
    const int gm = a.group_mats[bz];
    const DevMat &d = a.mats[gm];
    const bool tall = d.rows > d.cols;
    const float s = a.inv_norm[gm];
    const float *src = a.predict ? (d.sync ? nullptr : d.ef) : d.mom;
    const int64_t i0 = (int64_t)blockIdx.y * 64, j0 = (int64_t)blockIdx.x * 64;
    // tile origin in M: (mr0, mc0), 64 x 64, clipped to rows x cols
    const int64_t mr0 = tall ? j0 : i0, mc0 = tall ? i0 : j0;
    const bool vec = (d.cols % kPacket) == 0 && mr0 + 64 <= d.rows && mc0 + 64 <= d.cols;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int v = (int)threadIdx.x + h * kThreads;   // 512 vectors of 8
        const int row = v >> 3, c8 = (v & 7) * 8;         // within the tile, in M's layout
        float x[8];
        if (src == nullptr) {
#pragma unroll
            for (int e = 0; e < 8; ++e)
                x[e] = 0.0f;
        } else if (vec) {
            ld8(src + (mr0 + row) * d.cols + mc0 + c8, x);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int64_t mr = mr0 + row, mc = mc0 + c8 + e;
                x[e] = (mr < d.rows && mc < d.cols) ? src[mr * d.cols + mc] : 0.0f;
            }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (tall)
                tile[c8 + e][row] = x[e] * s;   // X row = M column
            else
                tile[row][c8 + e] = x[e] * s;
        }
    }
    __syncthreads();
    __nv_bfloat16 *xb = a.x + (int64_t)bz * a.R * a.W;
    __nv_bfloat16 *xt = a.xt != nullptr ? a.xt + (int64_t)bz * a.W * a.R : nullptr;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int v = (int)threadIdx.x + h * kThreads;
        const int row = v >> 3, c8 = (v & 7) * 8;   // within the tile, in X's layout
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e)
            o[e] = tile[row][c8 + e];
        st8(xb + (i0 + row) * a.W + j0 + c8, o);
        if (xt != nullptr) {   // X_0^T: the output of tall matrices when there are no steps
#pragma unroll
            for (int e = 0; e < 8; ++e)
                o[e] = tile[c8 + e][row];
            st8(xt + (j0 + row) * a.R + i0 + c8, o);
        }
    }
}

// The update's per-call scalars (host-formed, or device-formed for a
// capturable context by muon_scalars_kernel).
struct ApplyScalars {
    float lr, lr_wd;
    int ef_now;
};

// Device-resident counters of a capturable context.
struct MuonCounters {
    int64_t k, phase_k0;
};

struct ApplyArgs {
    const DevMat *mats;
    int chunks;
    float lr, lr_wd, lam;
    int ef_now, hist, delayed;
    int sapipe;               // SAPipe-WP: stash := x_t - U_prev, standard rule
    int keep_hist;            // SAPipe-WP updated state: the history receives the
                              // prediction update later (muon_predict_kernel)
    const ApplyScalars *dev;  // capturable context: lr, lr_wd, ef_now of this call
};

// One thread: the next call's lr (from *lr_src when set), lr wd and whether
// EF applies (Alg. 1: from t = 2 of the delayed phase); advances k.
__global__ void muon_scalars_kernel(MuonCounters *cnt, const float *lr_src, float lr_host,
                                    double weight_decay, int ef_possible, ApplyScalars *out)
{
    const int64_t k = cnt->k + 1;
    const int64_t t = k - cnt->phase_k0;
    const float lr = lr_src != nullptr ? *lr_src : lr_host;
    ApplyScalars sc;
    sc.lr = lr;
    sc.lr_wd = (float)((double)lr * weight_decay);
    sc.ef_now = ef_possible && t >= 2;
    *out = sc;
    cnt->k = k;
}

template <int SK>
__global__ void __launch_bounds__(kThreads) muon_apply_kernel(const ApplyArgs a)
{
    using ST = typename StashT<SK>::T;
    const DevMat &d = a.mats[blockIdx.y];
    const int64_t n = d.rows * d.cols;
    const int64_t lo = (int64_t)blockIdx.x * kChunk;
    if (lo >= n)
        return;
    const int64_t hi = lo + kChunk < n ? lo + kChunk : n;
    const ApplyScalars sc = a.dev != nullptr ? *a.dev : ApplyScalars{a.lr, a.lr_wd, a.ef_now};
    const float lr_r = sc.lr * d.r_scale, lr_wd = sc.lr_wd * d.wd_lr_scale;
    ST *stash = static_cast<ST *>(d.stash);
    __nv_bfloat16 *param = static_cast<__nv_bfloat16 *>(d.param);
    const bool vec_o = (d.cols % kPacket) == 0;
    // a DPO_SYNC matrix takes the standard update with no stash and no history
    const bool dly = a.delayed && !d.sync;
    const bool hist = a.hist && dly, ef_now = sc.ef_now && dly;
    const bool sapipe = a.sapipe && hist;
    const bool write_hist = hist && !a.keep_hist;
    for (int64_t e = lo + (int64_t)threadIdx.x * kPacket; e < hi; e += (int64_t)kThreads * kPacket) {
        if (e + kPacket <= hi && vec_o) {
            const int64_t i = e / d.cols, j = e - i * d.cols;
            float x[8], o[8], up[8], u[8];
            ld8(d.master + e, x);
            ld8(d.o + i * d.o_ld + j, o);
            if (ef_now || sapipe)
                ld8(d.ef + e, up);
            if (SK != kStashNone && dly) {
                if (sapipe) {   // the prediction point x_t - U_prev
                    float xp[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k)
                        xp[k] = x[k] - up[k];
                    st8(stash + e, xp);
                } else {
                    st8(stash + e, x);
                }
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                u[k] = fmaf(lr_r, o[k], lr_wd * x[k]);
                x[k] -= ef_now ? fmaf(a.lam, u[k] - up[k], u[k]) : u[k];
            }
            st8(d.master + e, x);
            if (write_hist)
                st8(d.ef + e, u);
            if (param != nullptr)
                st8(param + e, x);
        } else {
            const int64_t top = e + kPacket < hi ? e + kPacket : hi;
            for (int64_t q = e; q < top; ++q) {
                const int64_t i = q / d.cols, j = q - i * d.cols;
                float x = d.master[q];
                const float o = __bfloat162float(d.o[i * d.o_ld + j]);
                if (SK != kStashNone && dly)
                    st1(stash + q, sapipe ? x - d.ef[q] : x);
                const float u = fmaf(lr_r, o, lr_wd * x);
                x -= ef_now ? fmaf(a.lam, u - d.ef[q], u) : u;
                d.master[q] = x;
                if (write_hist)
                    d.ef[q] = u;
                if (param != nullptr)
                    st1(param + q, x);
            }
        }
    }
}

// SAPipe-WP updated state (App. B.1): the prediction update
// U' = lr (r O' + wd X_{t+1}) of each delayed matrix into its history, O' the
// Newton-Schulz output of M' and X_{t+1} the master the real update left.
__global__ void __launch_bounds__(kThreads) muon_predict_kernel(const ApplyArgs a)
{
    const DevMat &d = a.mats[blockIdx.y];
    if (d.sync || d.ef == nullptr)
        return;
    const int64_t n = d.rows * d.cols;
    const int64_t lo = (int64_t)blockIdx.x * kChunk;
    if (lo >= n)
        return;
    const int64_t hi = lo + kChunk < n ? lo + kChunk : n;
    const ApplyScalars sc = a.dev != nullptr ? *a.dev : ApplyScalars{a.lr, a.lr_wd, a.ef_now};
    const float lr_r = sc.lr * d.r_scale, lr_wd = sc.lr_wd * d.wd_lr_scale;
    const bool vec_o = (d.cols % kPacket) == 0;
    for (int64_t e = lo + (int64_t)threadIdx.x * kPacket; e < hi; e += (int64_t)kThreads * kPacket) {
        if (e + kPacket <= hi && vec_o) {
            const int64_t i = e / d.cols, j = e - i * d.cols;
            float x[8], o[8], u[8];
            ld8(d.master + e, x);
            ld8(d.o + i * d.o_ld + j, o);
#pragma unroll
            for (int k = 0; k < 8; ++k)
                u[k] = fmaf(lr_r, o[k], lr_wd * x[k]);
            st8(d.ef + e, u);
        } else {
            const int64_t top = e + kPacket < hi ? e + kPacket : hi;
            for (int64_t q = e; q < top; ++q) {
                const int64_t i = q / d.cols, j = q - i * d.cols;
                d.ef[q] = fmaf(lr_r, __bfloat162float(d.o[i * d.o_ld + j]), lr_wd * d.master[q]);
            }
        }
    }
}

// Start state (zero_mom, zero_ef: mom = 0, ef = 0) or the restart of Alg. 1
// on entering delayed training (zero_ef only): stash := master for matrices
// trained delayed, param := master.
template <int SK>
__global__ void __launch_bounds__(kThreads) muon_init_kernel(const DevMat *mats, int zero_mom,
                                                             int zero_ef)
{
    using ST = typename StashT<SK>::T;
    const DevMat &d = mats[blockIdx.y];
    const int64_t n = d.rows * d.cols;
    ST *stash = static_cast<ST *>(d.stash);
    __nv_bfloat16 *param = static_cast<__nv_bfloat16 *>(d.param);
    for (int64_t q = (int64_t)blockIdx.x * kThreads + threadIdx.x; q < n;
         q += (int64_t)gridDim.x * kThreads) {
        const float x = d.master[q];
        if (zero_mom)
            d.mom[q] = 0.0f;
        if (zero_ef && d.ef != nullptr)
            d.ef[q] = 0.0f;
        if (SK != kStashNone && stash != nullptr && !d.sync)
            st1(stash + q, x);
        if (param != nullptr)
            st1(param + q, x);
    }
}

}  // namespace muon
}  // namespace dpo

// ------------------------------------------------------------------ host ----

namespace {

using dpo::muon::DevMat;
using dpo::muon::kPad;
using dpo::muon::kThreads;
using dpo::muon::kChunk;

thread_local std::string g_muon_init_err;

using EncodeTiled = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                 const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                 const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                 CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encode_fn()
{
    static EncodeTiled fn = nullptr;
    if (fn == nullptr) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(p);
    }
    return fn;
}

// 3-D map over nb row-major bf16 matrices of rows x cols (pitch cols),
// consecutive in memory: boxes of 64 columns x box_rows rows, 128-byte swizzle.
bool make_map(CUtensorMap *m, void *base, int64_t rows, int64_t cols, int64_t nb, int box_rows)
{
    EncodeTiled enc = encode_fn();
    if (enc == nullptr)
        return false;
    const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)nb};
    const cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)(rows * cols) * 2};
    const cuuint32_t box[3] = {(cuuint32_t)dpo::gemm::kBoxK, (cuuint32_t)box_rows, 1};
    const cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same over rows x cols with 32 x 32 boxes and the 64-byte swizzle: the
// epilogue's TMA stores.
bool make_store_map(CUtensorMap *m, void *base, int64_t rows, int64_t cols, int64_t nb)
{
    EncodeTiled enc = encode_fn();
    if (enc == nullptr)
        return false;
    const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)nb};
    const cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)(rows * cols) * 2};
    const cuuint32_t box[3] = {32, 32, 1};
    const cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
               CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int64_t pad_up(int64_t v) { return (v + kPad - 1) / kPad * kPad; }

struct Group {
    int64_t r, w, R, W;
    std::vector<int> mats;
    int *d_mats = nullptr;          // into the context's device block
    bool has_tall = false;
    // X ping-pongs between x[0] and x[1]: every tile of X <- B X + a X reads
    // all of the old X, so the new one goes to the other buffer.
    __nv_bfloat16 *x[2] = {nullptr, nullptr}, *xt = nullptr, *a = nullptr, *b = nullptr;
    CUtensorMap x128[2], a128, b128;   // 128-row K-major boxes: one CTA's half of a pair tile
    CUtensorMap x_mn[2];               // 64 x 64 boxes of X read MN-major (B of B X)
    CUtensorMap st_x[2], st_xt, st_a, st_b;   // 32 x 32 store boxes of X, X^T, A, B
};

}  // namespace

struct dpo_muon_ctx {
    int device = 0;
    int n = 0;
    dpo_dtype stash_dt = DPO_F32, grad_dt = DPO_F32;
    dpo_muon_hparams hp{};
    bool ef = false;
    bool has_stash = false;   // some matrix has a stash buffer
    bool can_delay = true;    // every matrix without DPO_SYNC has one
    // step counters; a capturable context keeps the authoritative copy on
    // the device (d_cnt) and refreshes these from it when the host needs them
    mutable int64_t k = 0;
    mutable int64_t phase_k0 = 0;     // k when the current delayed phase began
    bool capturable = false;          // dpo_muon_set_capturable
    const float *lr_src = nullptr;    // capturable: device learning rate, or nullptr
    dpo::muon::MuonCounters *d_cnt = nullptr;
    dpo::muon::ApplyScalars *d_asc = nullptr;
    int sms = 0;
    int gemm_pairs = 0;   // clusters of 2 the GEMM kernel keeps resident at once
    int stall_launches = 0;   // dpo_muon_test_stall: GEMM launches left to stall
    std::vector<dpo_matrix> mats;
    std::vector<DevMat> host_mats;
    std::vector<Group> groups;
    int chunks = 0;
    int64_t total_elems = 0;
    int64_t ws_bytes = 0;
    double flops = 0.0;
    // device memory: one block for tables and scratch, one for the workspace
    void *dev_block = nullptr;
    void *ws = nullptr;
    DevMat *d_mats = nullptr;
    double *d_partials = nullptr;
    float *d_inv_norm = nullptr;
    unsigned int *d_err = nullptr;
    // gradient norm for clipping (the elementwise path's kernel and table)
    dpo::DevTensor *d_norm_table = nullptr;
    int64_t *d_pkt_begin = nullptr;
    double *d_norm_partials = nullptr;
    dpo::NormScalars *d_norm_scalars = nullptr;
    const double *clip_src = nullptr;   // external sum of squares (dpo_muon_set_clip_source)
    int64_t total_pkts = 0;
    int norm_grid = 0;
    // GEMM timing (dpo_muon_set_timing): event pairs recorded since the last read
    bool timing = false;
    std::vector<cudaEvent_t> ev_pool;
    size_t ev_used = 0;
    // short GEMM launches: one launch per product covers every shape group
    bool grouped = false;
    int64_t gemm_launches = 0;
    std::string err;
};

namespace {

int mfail(dpo_muon_ctx *c, int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c != nullptr)
        c->err = buf;
    else
        g_muon_init_err = buf;
    return code;
}

int mcuda(dpo_muon_ctx *c, cudaError_t e, const char *what)
{
    return mfail(c, DPO_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned32(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 31u) == 0; }

void free_ctx(dpo_muon_ctx *c)
{
    if (c == nullptr)
        return;
    for (cudaEvent_t e : c->ev_pool)
        cudaEventDestroy(e);
    if (c->ws != nullptr)
        cudaFree(c->ws);
    if (c->dev_block != nullptr)
        cudaFree(c->dev_block);
    delete c;
}

int launch_init(dpo_muon_ctx *c, cudaStream_t s, int zero_mom, int zero_ef)
{
    int64_t max_n = 0;
    for (const dpo_matrix &m : c->mats)
        max_n = std::max<int64_t>(max_n, m.rows * m.cols);
    if (max_n == 0 || c->n == 0)
        return DPO_OK;
    const dim3 grid((unsigned)std::min<int64_t>((max_n + kThreads - 1) / kThreads, 4096),
                    (unsigned)c->n);
    const DevMat *m = c->d_mats;
    if (!c->has_stash)
        dpo::muon::muon_init_kernel<dpo::kStashNone><<<grid, kThreads, 0, s>>>(m, zero_mom, zero_ef);
    else if (c->stash_dt == DPO_BF16)
        dpo::muon::muon_init_kernel<dpo::kStashBF16><<<grid, kThreads, 0, s>>>(m, zero_mom, zero_ef);
    else
        dpo::muon::muon_init_kernel<dpo::kStashF32><<<grid, kThreads, 0, s>>>(m, zero_mom, zero_ef);
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? DPO_OK : mcuda(c, e, "muon init launch");
}

}  // namespace

extern "C" const char *dpo_muon_last_error(const dpo_muon_ctx *c)
{
    if (c == nullptr)
        return g_muon_init_err.c_str();
    return c->err.c_str();
}

extern "C" int dpo_muon_init(dpo_muon_ctx **out, const dpo_matrix *mats, int n,
                             dpo_dtype stash_dtype, dpo_dtype grad_dtype,
                             const dpo_muon_hparams *hp, int init_mode, void *stream)
{
    if (out == nullptr)
        return mfail(nullptr, DPO_EINVAL, "out is NULL");
    *out = nullptr;
    if (hp == nullptr || n < 0 || (n > 0 && mats == nullptr))
        return mfail(nullptr, DPO_EINVAL, "NULL arguments or negative count");
    if ((stash_dtype != DPO_F32 && stash_dtype != DPO_BF16) ||
        (grad_dtype != DPO_F32 && grad_dtype != DPO_BF16))
        return mfail(nullptr, DPO_EDTYPE, "stash and grad dtypes must be F32 or BF16");
    if (!(hp->momentum >= 0.0f && hp->momentum < 1.0f) || !(hp->weight_decay >= 0.0f) ||
        !std::isfinite(hp->ef_lambda) || hp->ns_steps < 0 || hp->ns_steps > 16 ||
        !(hp->ns_eps >= 0.0f) || !(hp->rms_scale >= 0.0f) || (hp->delay != 0 && hp->delay != 1) ||
        !std::isfinite(hp->ns_a) || !std::isfinite(hp->ns_b) || !std::isfinite(hp->ns_c))
        return mfail(nullptr, DPO_EINVAL, "hyperparameter out of range");
    if (hp->correction != DPO_CORR_EF && hp->correction != DPO_CORR_SAPIPE_SAME &&
        hp->correction != DPO_CORR_SAPIPE_UPDATED)
        return mfail(nullptr, DPO_EINVAL, "correction must be one of DPO_CORR_*");
    if (init_mode != DPO_INIT_FRESH && init_mode != DPO_INIT_RESUME)
        return mfail(nullptr, DPO_EINVAL, "bad init_mode");
    const bool ef = n > 0 && mats[0].ef != nullptr;
    for (int i = 0; i < n; ++i) {
        const dpo_matrix &m = mats[i];
        if (m.rows < 0 || m.cols < 0)
            return mfail(nullptr, DPO_EINVAL, "matrix %d: negative shape", i);
        if (m.rows * m.cols == 0)
            continue;
        if (m.master == nullptr || m.mom == nullptr || m.grad == nullptr)
            return mfail(nullptr, DPO_EINVAL, "matrix %d: master, mom and grad are required", i);
        if ((m.flags & ~(DPO_WD_ON | DPO_SYNC)) != 0)
            return mfail(nullptr, DPO_EINVAL, "matrix %d: unknown flags", i);
        if (hp->delay == 1 && m.stash == nullptr && !(m.flags & DPO_SYNC))
            return mfail(nullptr, DPO_EINVAL, "matrix %d: delay 1 needs a stash", i);
        if ((m.ef != nullptr) != ef)
            return mfail(nullptr, DPO_EINVAL, "ef buffers must be given for all matrices or none");
        const void *ps[6] = {m.param, m.master, m.mom, m.stash, m.ef, m.grad};
        for (const void *p : ps)
            if (p != nullptr && !aligned32(p))
                return mfail(nullptr, DPO_EALIGN, "matrix %d: buffer not 32-byte aligned", i);
    }

    dpo_muon_ctx *c = new dpo_muon_ctx();
    c->n = n;
    c->stash_dt = stash_dtype;
    c->grad_dt = grad_dtype;
    c->hp = *hp;
    c->ef = ef;
    c->mats.assign(mats, mats + n);
    for (int i = 0; i < n; ++i) {
        if (mats[i].rows * mats[i].cols == 0)
            continue;
        c->has_stash = c->has_stash || mats[i].stash != nullptr;
        c->can_delay = c->can_delay && (mats[i].stash != nullptr || (mats[i].flags & DPO_SYNC));
    }
    cudaGetDevice(&c->device);
    cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, c->device);
    cudaStream_t s = static_cast<cudaStream_t>(stream);

    // Group the matrices by their wide orientation r x w (r <= w).
    std::map<std::pair<int64_t, int64_t>, int> gidx;
    int64_t max_n = 0;
    for (int i = 0; i < n; ++i) {
        const dpo_matrix &m = mats[i];
        const int64_t ne = m.rows * m.cols;
        c->total_elems += ne;
        max_n = std::max(max_n, ne);
        if (ne == 0)
            continue;
        const int64_t r = std::min(m.rows, m.cols), w = std::max(m.rows, m.cols);
        auto key = std::make_pair(r, w);
        if (!gidx.count(key)) {
            gidx[key] = (int)c->groups.size();
            Group g;
            g.r = r;
            g.w = w;
            g.R = pad_up(r);
            g.W = pad_up(w);
            c->groups.push_back(g);
        }
        c->groups[gidx[key]].mats.push_back(i);
        // unique entries of the symmetric products X X^T (r (r + 1) / 2, each
        // w multiply-adds) and A A (r (r + 1) / 2, r each), all of B X
        c->flops += (double)hp->ns_steps * ((double)r * (r + 1) * w + (double)r * (r + 1) * r +
                                            2.0 * (double)r * r * w);
    }
    c->chunks = (int)std::max<int64_t>(1, (max_n + kChunk - 1) / kChunk);

    // Workspace: per group X twice, X^T (the output of tall matrices), A, B (bf16).
    int64_t ws = 0;
    for (Group &g : c->groups) {
        const int64_t nb = (int64_t)g.mats.size();
        ws += nb * (g.R * g.W * 3 + g.R * g.R * 2) * 2;
        for (int mi : g.mats)
            g.has_tall = g.has_tall || mats[mi].rows > mats[mi].cols;
    }
    c->ws_bytes = ws;
    // Norm-pass table (the elementwise path's gradient-norm kernel).
    int64_t total_pkts = 0;
    std::vector<int64_t> pkt_begin(n + 1, 0);
    for (int i = 0; i < n; ++i) {
        pkt_begin[i] = total_pkts;
        total_pkts += (mats[i].rows * mats[i].cols + dpo::kPacket - 1) / dpo::kPacket;
    }
    pkt_begin[n] = total_pkts;
    c->total_pkts = total_pkts;
    int per_sm_norm = 0;
    dpo::norm_ctas_per_sm(grad_dtype == DPO_BF16, &per_sm_norm);
    const int64_t norm_groups =
        (total_pkts + (int64_t)dpo::kNormThreads * dpo::kNormUnroll - 1) /
        ((int64_t)dpo::kNormThreads * dpo::kNormUnroll);
    c->norm_grid = (int)std::max<int64_t>(
        1, std::min<int64_t>(norm_groups, (int64_t)std::max(1, c->sms) * std::max(1, per_sm_norm)));

    // Device block: mats | group index arrays | partials | inv_norm | err |
    // norm table | pkt_begin | norm partials | norm scalars.
    auto al = [](int64_t v) { return (v + 255) / 256 * 256; };
    int64_t off = 0;
    const int64_t o_mats = off;
    off += al((int64_t)sizeof(DevMat) * std::max(1, n));
    std::vector<int64_t> o_groups;
    for (Group &g : c->groups) {
        o_groups.push_back(off);
        off += al((int64_t)sizeof(int) * (int64_t)g.mats.size());
    }
    const int64_t o_part = off;
    off += al((int64_t)sizeof(double) * std::max(1, n) * c->chunks);
    const int64_t o_inv = off;
    off += al((int64_t)sizeof(float) * std::max(1, n));
    const int64_t o_err = off;
    off += al(sizeof(unsigned int));
    const int64_t o_ntab = off;
    off += al((int64_t)sizeof(dpo::DevTensor) * std::max(1, n));
    const int64_t o_pkt = off;
    off += al((int64_t)sizeof(int64_t) * (n + 1));
    const int64_t o_npart = off;
    off += al((int64_t)sizeof(double) * c->norm_grid);
    const int64_t o_nsc = off;
    off += al(sizeof(dpo::NormScalars));
    const int64_t o_cnt = off;
    off += al(sizeof(dpo::muon::MuonCounters));
    const int64_t o_asc = off;
    off += al(sizeof(dpo::muon::ApplyScalars));

    cudaError_t e = dpo::device_alloc(&c->dev_block, (size_t)off);
    if (e != cudaSuccess) {
        free_ctx(c);
        return mfail(nullptr, DPO_ENOMEM, "device table allocation failed");
    }
    if (ws > 0) {
        e = dpo::device_alloc(&c->ws, (size_t)ws);
        if (e != cudaSuccess) {
            free_ctx(c);
            return mfail(nullptr, DPO_ENOMEM, "Newton-Schulz workspace (%lld bytes) allocation failed",
                         (long long)ws);
        }
    }
    char *blk = static_cast<char *>(c->dev_block);
    c->d_mats = reinterpret_cast<DevMat *>(blk + o_mats);
    c->d_partials = reinterpret_cast<double *>(blk + o_part);
    c->d_inv_norm = reinterpret_cast<float *>(blk + o_inv);
    c->d_err = reinterpret_cast<unsigned int *>(blk + o_err);
    c->d_norm_table = reinterpret_cast<dpo::DevTensor *>(blk + o_ntab);
    c->d_pkt_begin = reinterpret_cast<int64_t *>(blk + o_pkt);
    c->d_norm_partials = reinterpret_cast<double *>(blk + o_npart);
    c->d_norm_scalars = reinterpret_cast<dpo::NormScalars *>(blk + o_nsc);
    c->d_cnt = reinterpret_cast<dpo::muon::MuonCounters *>(blk + o_cnt);
    c->d_asc = reinterpret_cast<dpo::muon::ApplyScalars *>(blk + o_asc);

    // Carve the workspace and build the tensor maps.
    char *wp = static_cast<char *>(c->ws);
    c->host_mats.resize(n);
    for (int i = 0; i < n; ++i) {
        const dpo_matrix &m = mats[i];
        DevMat &d = c->host_mats[i];
        d.param = m.param;
        d.master = m.master;
        d.mom = m.mom;
        d.stash = m.stash;
        d.ef = m.ef;
        d.grad = m.grad;
        d.rows = m.rows;
        d.cols = m.cols;
        d.o = nullptr;
        d.o_ld = 0;
        d.wd_lr_scale = (m.flags & DPO_WD_ON) ? 1.0f : 0.0f;
        d.r_scale = hp->rms_scale > 0.0f
                        ? (float)(hp->rms_scale * std::sqrt((double)std::max(m.rows, m.cols)))
                        : 1.0f;
        d.sync = (m.flags & DPO_SYNC) ? 1 : 0;
    }
    for (size_t gi = 0; gi < c->groups.size(); ++gi) {
        Group &g = c->groups[gi];
        const int64_t nb = (int64_t)g.mats.size();
        for (int q = 0; q < 2; ++q) {
            g.x[q] = reinterpret_cast<__nv_bfloat16 *>(wp);
            wp += nb * g.R * g.W * 2;
        }
        g.xt = reinterpret_cast<__nv_bfloat16 *>(wp);
        wp += nb * g.W * g.R * 2;
        g.a = reinterpret_cast<__nv_bfloat16 *>(wp);
        wp += nb * g.R * g.R * 2;
        g.b = reinterpret_cast<__nv_bfloat16 *>(wp);
        wp += nb * g.R * g.R * 2;
        g.d_mats = reinterpret_cast<int *>(blk + o_groups[gi]);
        const bool ok = make_map(&g.x128[0], g.x[0], g.R, g.W, nb, dpo::gemm::BM) &&
                        make_map(&g.x128[1], g.x[1], g.R, g.W, nb, dpo::gemm::BM) &&
                        make_map(&g.a128, g.a, g.R, g.R, nb, dpo::gemm::BM) &&
                        make_map(&g.b128, g.b, g.R, g.R, nb, dpo::gemm::BM) &&
                        make_map(&g.x_mn[0], g.x[0], g.R, g.W, nb, 64) &&
                        make_map(&g.x_mn[1], g.x[1], g.R, g.W, nb, 64) &&
                        make_store_map(&g.st_x[0], g.x[0], g.R, g.W, nb) &&
                        make_store_map(&g.st_x[1], g.x[1], g.R, g.W, nb) &&
                        make_store_map(&g.st_xt, g.xt, g.W, g.R, nb) &&
                        make_store_map(&g.st_a, g.a, g.R, g.R, nb) &&
                        make_store_map(&g.st_b, g.b, g.R, g.R, nb);
        if (!ok) {
            free_ctx(c);
            return mfail(nullptr, DPO_ECUDA, "tensor map encoding failed");
        }
        // Newton-Schulz output: X (wide matrices) or X^T (tall ones, whose
        // rows are the original matrix's rows; written by the normalisation
        // when there are no steps, else by the last step).
        for (size_t bi = 0; bi < g.mats.size(); ++bi) {
            DevMat &d = c->host_mats[g.mats[bi]];
            if (d.rows > d.cols) {
                d.o = g.xt + (int64_t)bi * g.W * g.R;
                d.o_ld = g.R;
            } else {   // the buffer the last step wrote
                d.o = g.x[hp->ns_steps % 2] + (int64_t)bi * g.R * g.W;
                d.o_ld = g.W;
            }
        }
    }
    std::vector<dpo::DevTensor> ntab(n);
    for (int i = 0; i < n; ++i) {
        dpo::DevTensor t{};
        t.grad = mats[i].grad;
        t.numel = mats[i].rows * mats[i].cols;
        ntab[i] = t;
    }

#define MUON_COPY(dst, src, bytes)                                                      \
    do {                                                                                \
        if ((bytes) > 0) {                                                              \
            e = cudaMemcpyAsync((dst), (src), (size_t)(bytes), cudaMemcpyHostToDevice, s); \
            if (e != cudaSuccess) {                                                     \
                free_ctx(c);                                                            \
                return mcuda(nullptr, e, "table upload");                               \
            }                                                                           \
        }                                                                               \
    } while (0)
    MUON_COPY(c->d_mats, c->host_mats.data(), sizeof(DevMat) * n);
    for (Group &g : c->groups)
        MUON_COPY(g.d_mats, g.mats.data(), sizeof(int) * g.mats.size());
    MUON_COPY(c->d_norm_table, ntab.data(), sizeof(dpo::DevTensor) * n);
    MUON_COPY(c->d_pkt_begin, pkt_begin.data(), sizeof(int64_t) * (n + 1));
#undef MUON_COPY
    e = cudaMemsetAsync(c->d_err, 0, sizeof(unsigned int), s);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(c->d_norm_scalars, 0, sizeof(dpo::NormScalars), s);
    if (e == cudaSuccess && ws > 0)
        e = cudaMemsetAsync(c->ws, 0, (size_t)ws, s);   // zero padding stays zero
    if (e != cudaSuccess) {
        free_ctx(c);
        return mcuda(nullptr, e, "workspace clear");
    }
    c->gemm_pairs = 1 << 30;
    for (const void *fn : {(const void *)dpo::gemm::ns_gemm_kernel<false>,
                           (const void *)dpo::gemm::ns_gemm_kernel<true>}) {
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 dpo::gemm::kSmemBytes);
        int pairs = 0;
        if (e == cudaSuccess) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(2 * std::max(1, c->sms / 2));
            cfg.blockDim = dim3(dpo::gemm::kThreads);
            cfg.dynamicSmemBytes = dpo::gemm::kSmemBytes;
            e = cudaOccupancyMaxActiveClusters(&pairs, fn, &cfg);
        }
        if (e != cudaSuccess)
            break;
        c->gemm_pairs = std::min(c->gemm_pairs, pairs);
    }
    if (e != cudaSuccess || c->gemm_pairs < 1) {
        free_ctx(c);
        return e != cudaSuccess ? mcuda(nullptr, e, "GEMM launch configuration")
                                : mfail(nullptr, DPO_ECUDA, "GEMM kernel cannot be resident");
    }
    // When some shape group's launches are short (at most 16 rounds of tiles
    // over the CTA pairs), each product of a Newton-Schulz step covers all
    // shape groups in one launch: one group's tiles fill the pairs another
    // leaves idle, and a step takes 3 launches instead of 3 per group (GPT-2:
    // every group short; the Llama-1B set's 512 x 2048 group: 20.08 -> 19.80
    // ms of GEMMs per step on GB300). Sets whose groups are all long keep one
    // group per launch and run the groups' chains one after another (7B set:
    // 0.3% slower grouped; two chains at once on two streams mixed their
    // operands in L2, 336 -> 410 ms per step).
    int64_t min_tiles = INT64_MAX;
    for (const Group &g : c->groups)
        min_tiles = std::min<int64_t>(min_tiles, (int64_t)g.mats.size() *
                                                     (g.R / dpo::gemm::TM) * (g.W / dpo::gemm::TN));
    c->grouped = c->groups.size() > 1 && min_tiles <= 16 * (int64_t)std::max(1, c->gemm_pairs);
    if (init_mode == DPO_INIT_FRESH) {
        const int rc = launch_init(c, s, 1, 1);
        if (rc != DPO_OK) {
            g_muon_init_err = c->err;
            free_ctx(c);
            return rc;
        }
    }
    *out = c;
    return DPO_OK;
}

namespace {

// One product of a Newton-Schulz step for one shape group.
struct GemmJob {
    const CUtensorMap *ta, *tb, *td, *tdt;
    dpo::gemm::Params p;
    int64_t M, N, nb;
};

// One launch over up to kMaxGroups jobs of the same product (all read B
// K-major, or all MN-major), the jobs with more K blocks first: the pairs
// take tiles round-robin, so the longest tiles go out first and the short
// ones fill the last round.
int launch_gemm(dpo_muon_ctx *c, const GemmJob *jobs, int n_jobs, bool b_mn, cudaStream_t s)
{
    if (n_jobs < 1 || n_jobs > dpo::gemm::kMaxGroups)
        return mfail(c, DPO_EINVAL, "GEMM launch of %d groups", n_jobs);
    int order[dpo::gemm::kMaxGroups];
    for (int j = 0; j < n_jobs; ++j)
        order[j] = j;
    std::stable_sort(order, order + n_jobs, [&](int x, int y) {
        return jobs[x].p.k_blocks > jobs[y].p.k_blocks;
    });
    dpo::gemm::GemmLaunch L;
    std::memset(&L, 0, sizeof L);
    int64_t tiles = 0;
    for (int q = 0; q < n_jobs; ++q) {
        const GemmJob &j = jobs[order[q]];
        dpo::gemm::TileGrid tg{(int)(j.M / dpo::gemm::TM), (int)(j.N / dpo::gemm::TN), (int)j.nb,
                               j.p.sym};
        if (j.p.sym && j.M != j.N)
            return mfail(c, DPO_EINVAL, "symmetric product of a non-square shape");
        dpo::gemm::GemmGroup &G = L.g[q];
        G.a = *j.ta;
        G.b = *j.tb;
        G.d = *j.td;
        G.dt = *j.tdt;
        G.p = j.p;
        G.tg = tg;
        G.tile0 = (int)tiles;
        tiles += tg.count();
    }
    L.n_groups = n_jobs;
    L.n_tiles = (int)tiles;
    // one CTA pair per co-resident cluster slot (the tile walk assumes every
    // pair runs at once)
    const int grid = 2 * (int)std::min<int64_t>(tiles, std::max(1, c->gemm_pairs));
    if (b_mn)
        dpo::gemm::ns_gemm_kernel<true><<<grid, dpo::gemm::kThreads, dpo::gemm::kSmemBytes, s>>>(L);
    else
        dpo::gemm::ns_gemm_kernel<false><<<grid, dpo::gemm::kThreads, dpo::gemm::kSmemBytes, s>>>(L);
    if (c->timing)
        ++c->gemm_launches;
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? DPO_OK : mcuda(c, e, "Newton-Schulz GEMM launch");
}

}  // namespace

namespace {

// Momentum (M <- mu M + (1 - mu) G^, or with `predict` M' into the history
// buffers), its Frobenius norms, the normalisation into the workspace and the
// Newton-Schulz chains of every shape group: the Newton-Schulz output of each
// matrix is then in the workspace (DevMat::o).
int orthogonalize(dpo_muon_ctx *c, cudaStream_t s, bool predict)
{
    // momentum and its Frobenius norms
    dpo::muon::MomArgs ma{};
    ma.mats = c->d_mats;
    ma.clip = c->hp.max_grad_norm > 0.0f ? &c->d_norm_scalars->clip : nullptr;
    ma.mu = c->hp.momentum;
    ma.omm = (float)(1.0 - (double)c->hp.momentum);
    ma.partials = c->d_partials;
    ma.chunks = c->chunks;
    ma.predict = predict ? 1 : 0;
    const dim3 mgrid((unsigned)c->chunks, (unsigned)c->n);
    if (c->grad_dt == DPO_BF16)
        dpo::muon::muon_momentum_kernel<__nv_bfloat16><<<mgrid, kThreads, 0, s>>>(ma);
    else
        dpo::muon::muon_momentum_kernel<float><<<mgrid, kThreads, 0, s>>>(ma);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return mcuda(c, e, "momentum launch");
    dpo::muon::muon_norm_kernel<<<(c->n + 7) / 8, 256, 0, s>>>(c->d_partials, c->chunks, c->n,
                                                               c->hp.ns_eps, c->d_inv_norm);
    if ((e = cudaGetLastError()) != cudaSuccess)
        return mcuda(c, e, "norm launch");

    for (Group &g : c->groups) {
        const int64_t nb = (int64_t)g.mats.size();
        dpo::muon::NormArgsM na{c->d_mats, g.d_mats, c->d_inv_norm, g.x[0],
                                c->hp.ns_steps == 0 ? g.xt : nullptr, g.R, g.W, g.r, g.w,
                                predict ? 1 : 0};
        const dim3 ngrid((unsigned)(g.W / 64), (unsigned)(g.R / 64), (unsigned)nb);
        dpo::muon::muon_normalize_kernel<<<ngrid, kThreads, 0, s>>>(na);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return mcuda(c, e, "normalize launch");
    }
    cudaEvent_t ev_end = nullptr;
    if (c->timing && c->hp.ns_steps > 0) {
        if (c->ev_used + 2 > c->ev_pool.size()) {
            for (int q = 0; q < 2; ++q) {
                cudaEvent_t ev;
                if ((e = cudaEventCreate(&ev)) != cudaSuccess)
                    return mcuda(c, e, "timing event");
                c->ev_pool.push_back(ev);
            }
        }
        if ((e = cudaEventRecord(c->ev_pool[c->ev_used], s)) != cudaSuccess)
            return mcuda(c, e, "timing event record");
        ev_end = c->ev_pool[c->ev_used + 1];
        c->ev_used += 2;
    }
    // Newton-Schulz, per step: A = X X^T, B = c A A + b A, X <- B X + a X.
    // Short launches (c->grouped) take the same product of up to kMaxGroups
    // shape groups in one launch, step by step; long ones run one group's
    // chain after another, one launch per product.
    auto stall_next = [c]() {
        if (c->stall_launches <= 0)
            return 0;
        --c->stall_launches;
        return 1;
    };
    const int n_groups = (int)c->groups.size();
    const int per = c->grouped ? dpo::gemm::kMaxGroups : 1;
    for (int g0 = 0; g0 < n_groups; g0 += per) {
        const int n = std::min(per, n_groups - g0);
        for (int it = 0; it < c->hp.ns_steps; ++it) {
            const bool last = it + 1 == c->hp.ns_steps;
            const int cur = it % 2, nxt = cur ^ 1;
            GemmJob xx[dpo::gemm::kMaxGroups], aa[dpo::gemm::kMaxGroups],
                bx[dpo::gemm::kMaxGroups];
            const int st_xx = stall_next(), st_aa = stall_next(), st_bx = stall_next();
            for (int q = 0; q < n; ++q) {
                Group &g = c->groups[g0 + q];
                const int64_t nb = (int64_t)g.mats.size();
                dpo::gemm::Params p{};
                p.err = c->d_err;
                // A = X X^T
                p.alpha = 1.0f;
                p.k_blocks = (int)(g.W / dpo::gemm::BK);
                p.sym = 1;
                p.stall = st_xx;
                xx[q] = GemmJob{&g.x128[cur], &g.x128[cur], &g.st_a, &g.st_a, p, g.R, g.R, nb};
                // B = c A A + b A
                p.c = g.a;
                p.ldc = g.R;
                p.c_bstride = g.R * g.R;
                p.alpha = c->hp.ns_c;
                p.beta = c->hp.ns_b;
                p.k_blocks = (int)(g.R / dpo::gemm::BK);
                p.stall = st_aa;
                aa[q] = GemmJob{&g.a128, &g.a128, &g.st_b, &g.st_b, p, g.R, g.R, nb};
                // X <- B X + a X (X read MN-major in place of X^T), and at the
                // last step X^T for the tall matrices' output
                p.sym = 0;
                p.trans = last && g.has_tall ? 1 : 0;
                p.c = g.x[cur];
                p.ldc = g.W;
                p.c_bstride = g.R * g.W;
                p.alpha = 1.0f;
                p.beta = c->hp.ns_a;
                p.k_blocks = (int)(g.R / dpo::gemm::BK);
                p.stall = st_bx;
                bx[q] = GemmJob{&g.b128, &g.x_mn[cur], &g.st_x[nxt], &g.st_xt, p, g.R, g.W, nb};
            }
            int rc = launch_gemm(c, xx, n, false, s);
            if (rc == DPO_OK)
                rc = launch_gemm(c, aa, n, false, s);
            if (rc == DPO_OK)
                rc = launch_gemm(c, bx, n, true, s);
            if (rc != DPO_OK)
                return rc;
        }
    }
    if (ev_end != nullptr && (e = cudaEventRecord(ev_end, s)) != cudaSuccess)
        return mcuda(c, e, "timing event record");

    return DPO_OK;
}

}  // namespace

extern "C" int dpo_muon_step(dpo_muon_ctx *c, float lr, void *stream)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (!(lr > 0.0f) || !std::isfinite(lr))
        return mfail(c, DPO_EINVAL, "lr must be positive and finite");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t k = c->k + 1;
    if (c->n == 0 || c->total_elems == 0) {
        if (c->capturable) {   // keep the device counter in step
            dpo::muon::muon_scalars_kernel<<<1, 1, 0, s>>>(c->d_cnt, c->lr_src, lr, 0.0, 0,
                                                           c->d_asc);
            const cudaError_t e = cudaGetLastError();
            return e == cudaSuccess ? DPO_OK : mcuda(c, e, "scalars launch");
        }
        c->k = k;
        return DPO_OK;
    }
    const bool clip = c->hp.max_grad_norm > 0.0f;
    if (clip && c->clip_src != nullptr) {
        const cudaError_t e = dpo::launch_clip_from_sumsq(c->clip_src, c->hp.max_grad_norm,
                                                          c->d_norm_scalars, s);
        if (e != cudaSuccess)
            return mcuda(c, e, "clip-coefficient launch");
    } else if (clip) {
        dpo::NormArgs na{};
        na.table = c->d_norm_table;
        na.pkt_begin = c->d_pkt_begin;
        na.n_tensors = c->n;
        na.total_pkts = c->total_pkts;
        na.partials = c->d_norm_partials;
        na.out = c->d_norm_scalars;
        na.max_norm = c->hp.max_grad_norm;
        const cudaError_t e = dpo::launch_norm(c->grad_dt == DPO_BF16, c->norm_grid, na, s);
        if (e != cudaSuccess)
            return mcuda(c, e, "norm launch");
    }
    int rc = orthogonalize(c, s, false);
    if (rc != DPO_OK)
        return rc;
    cudaError_t e;
    const dim3 mgrid((unsigned)c->chunks, (unsigned)c->n);

    // update, stash, history, weights
    const int64_t t = k - c->phase_k0;   // Alg. 1 iteration within the delayed phase
    dpo::muon::ApplyArgs aa{};
    aa.mats = c->d_mats;
    aa.chunks = c->chunks;
    aa.lr = lr;
    aa.lr_wd = (float)((double)lr * (double)c->hp.weight_decay);
    aa.delayed = c->hp.delay == 1;
    aa.hist = c->ef && c->hp.delay == 1;
    const bool updated = c->hp.correction == DPO_CORR_SAPIPE_UPDATED;
    aa.sapipe = c->hp.correction == DPO_CORR_SAPIPE_SAME || updated;
    aa.keep_hist = updated;
    aa.ef_now = aa.hist && !aa.sapipe && t >= 2 && c->hp.ef_lambda != 0.0f;
    aa.lam = c->hp.ef_lambda;
    if (c->capturable) {   // lr and EF's start from the device counters
        dpo::muon::muon_scalars_kernel<<<1, 1, 0, s>>>(
            c->d_cnt, c->lr_src, lr, (double)c->hp.weight_decay,
            aa.hist && !aa.sapipe && c->hp.ef_lambda != 0.0f ? 1 : 0, c->d_asc);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return mcuda(c, e, "scalars launch");
        aa.dev = c->d_asc;
    }
    const bool st = c->hp.delay == 1;
    if (!st)
        dpo::muon::muon_apply_kernel<dpo::kStashNone><<<mgrid, kThreads, 0, s>>>(aa);
    else if (c->stash_dt == DPO_BF16)
        dpo::muon::muon_apply_kernel<dpo::kStashBF16><<<mgrid, kThreads, 0, s>>>(aa);
    else
        dpo::muon::muon_apply_kernel<dpo::kStashF32><<<mgrid, kThreads, 0, s>>>(aa);
    if ((e = cudaGetLastError()) != cudaSuccess)
        return mcuda(c, e, "apply launch");
    if (updated && aa.hist) {
        // SAPipe-WP updated state: the step once more on the same gradient
        // from the momentum just stored, decaying X_{t+1}, into the history
        if ((rc = orthogonalize(c, s, true)) != DPO_OK)
            return rc;
        dpo::muon::muon_predict_kernel<<<mgrid, kThreads, 0, s>>>(aa);
        if ((e = cudaGetLastError()) != cudaSuccess)
            return mcuda(c, e, "prediction launch");
    }
    if (!c->capturable)
        c->k = k;
    return DPO_OK;
}

namespace {

// A capturable context's counters live on the device: refresh the host copy
// (after all work so far), or write the host copy back.
int mpull(const dpo_muon_ctx *c)
{
    if (!c->capturable)
        return DPO_OK;
    dpo::muon::MuonCounters h{};
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess)
        e = cudaMemcpy(&h, c->d_cnt, sizeof h, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return DPO_ECUDA;
    c->k = h.k;
    c->phase_k0 = h.phase_k0;
    return DPO_OK;
}

int mpush(const dpo_muon_ctx *c, cudaStream_t s)
{
    const dpo::muon::MuonCounters h{c->k, c->phase_k0};
    // pageable source: the call returns once the bytes are staged
    return cudaMemcpyAsync(c->d_cnt, &h, sizeof h, cudaMemcpyHostToDevice, s) == cudaSuccess
               ? DPO_OK
               : DPO_ECUDA;
}

}  // namespace

extern "C" int dpo_muon_set_capturable(dpo_muon_ctx *c, int on, const float *lr_source,
                                       void *stream)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (lr_source != nullptr && reinterpret_cast<uintptr_t>(lr_source) % alignof(float) != 0)
        return mfail(c, DPO_EINVAL, "lr_source must be 4-byte aligned");
    if (on) {
        if (!c->capturable && mpush(c, static_cast<cudaStream_t>(stream)) != DPO_OK)
            return mfail(c, DPO_ECUDA, "writing the device step counters failed");
        c->capturable = true;
        c->lr_src = lr_source;
    } else {
        if (c->capturable && mpull(c) != DPO_OK)
            return mfail(c, DPO_ECUDA, "reading the device step counters failed");
        c->capturable = false;
        c->lr_src = nullptr;
    }
    return DPO_OK;
}

extern "C" int dpo_muon_set_delay(dpo_muon_ctx *c, int delay, void *stream)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (delay != 0 && delay != 1)
        return mfail(c, DPO_EINVAL, "delay must be 0 or 1");
    if (delay == c->hp.delay)
        return DPO_OK;
    if (delay == 1) {
        if (!c->can_delay)
            return mfail(c, DPO_ESTATE,
                         "delayed training needs a stash for every matrix without DPO_SYNC");
        // stash := the current weights, update history := 0: Alg. 1 restarts
        const int rc = launch_init(c, static_cast<cudaStream_t>(stream), 0, 1);
        if (rc != DPO_OK)
            return rc;
        if (mpull(c) != DPO_OK)
            return mfail(c, DPO_ECUDA, "reading the device step counters failed");
        c->phase_k0 = c->k;
        if (c->capturable && mpush(c, static_cast<cudaStream_t>(stream)) != DPO_OK)
            return mfail(c, DPO_ECUDA, "writing the device step counters failed");
    }
    c->hp.delay = delay;
    return DPO_OK;
}

extern "C" int dpo_muon_last_update(const dpo_muon_ctx *c, int i, const void **ptr, int64_t *ld)
{
    if (c == nullptr || ptr == nullptr || ld == nullptr || i < 0 || i >= c->n)
        return DPO_EINVAL;
    *ptr = c->host_mats[i].o;
    *ld = c->host_mats[i].o_ld;
    return DPO_OK;
}

extern "C" int dpo_muon_copy_update(const dpo_muon_ctx *c, int i, void *dst, void *stream)
{
    if (c == nullptr || dst == nullptr || i < 0 || i >= c->n)
        return DPO_EINVAL;
    const DevMat &d = c->host_mats[i];
    if (d.rows * d.cols == 0)
        return DPO_OK;
    const cudaError_t e = cudaMemcpy2DAsync(dst, (size_t)d.cols * 2, d.o, (size_t)d.o_ld * 2,
                                            (size_t)d.cols * 2, (size_t)d.rows,
                                            cudaMemcpyDeviceToDevice,
                                            static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? DPO_OK : DPO_ECUDA;
}

extern "C" int dpo_muon_get_status(dpo_muon_ctx *c, uint32_t *bits)
{
    if (c == nullptr || bits == nullptr)
        return DPO_EINVAL;
    unsigned int v = 0;
    const cudaError_t e = cudaMemcpy(&v, c->d_err, sizeof v, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return mcuda(c, e, "status read");
    *bits = v;
    return DPO_OK;
}

extern "C" int dpo_muon_clear_status(dpo_muon_ctx *c, void *stream)
{
    if (c == nullptr)
        return DPO_EINVAL;
    const cudaError_t e = cudaMemsetAsync(c->d_err, 0, sizeof(unsigned int),
                                          static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? DPO_OK : mcuda(c, e, "status reset");
}

extern "C" int dpo_muon_test_stall(dpo_muon_ctx *c, int launches)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (launches < 0)
        return mfail(c, DPO_EINVAL, "launches must be >= 0");
    c->stall_launches = launches;
    return DPO_OK;
}

extern "C" int dpo_muon_grad_sqnorm(dpo_muon_ctx *c, double *d_sumsq, void *stream)
{
    if (c == nullptr)
        return mfail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (d_sumsq == nullptr || reinterpret_cast<uintptr_t>(d_sumsq) % alignof(double) != 0)
        return mfail(c, DPO_EINVAL, "d_sumsq must be an 8-byte aligned device pointer");
    if (c->total_pkts == 0)
        return DPO_OK;
    dpo::NormArgs na{};
    na.table = c->d_norm_table;
    na.pkt_begin = c->d_pkt_begin;
    na.n_tensors = c->n;
    na.total_pkts = c->total_pkts;
    na.partials = c->d_norm_partials;
    na.out = c->d_norm_scalars;
    na.accum = d_sumsq;
    const cudaError_t e = dpo::launch_norm(c->grad_dt == DPO_BF16, c->norm_grid, na,
                                           static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess)
        return mcuda(c, e, "norm launch");
    return DPO_OK;
}

extern "C" int dpo_muon_set_clip_source(dpo_muon_ctx *c, const double *d_sumsq)
{
    if (c == nullptr)
        return mfail(nullptr, DPO_EINVAL, "ctx is NULL");
    if (d_sumsq != nullptr && reinterpret_cast<uintptr_t>(d_sumsq) % alignof(double) != 0)
        return mfail(c, DPO_EINVAL, "d_sumsq must be 8-byte aligned");
    if (d_sumsq != nullptr && !(c->hp.max_grad_norm > 0.0f))
        return mfail(c, DPO_ESTATE, "a clip source needs max_grad_norm > 0");
    c->clip_src = d_sumsq;
    return DPO_OK;
}

extern "C" int dpo_muon_get_phase_start(const dpo_muon_ctx *c, int64_t *k0)
{
    if (c == nullptr || k0 == nullptr)
        return DPO_EINVAL;
    if (mpull(c) != DPO_OK)
        return DPO_ECUDA;
    *k0 = c->phase_k0;
    return DPO_OK;
}

extern "C" int dpo_muon_set_phase_start(dpo_muon_ctx *c, int64_t k0)
{
    if (c == nullptr)
        return DPO_EINVAL;
    if (mpull(c) != DPO_OK)
        return mfail(c, DPO_ECUDA, "reading the device step counters failed");
    if (k0 < 0 || k0 > c->k)
        return mfail(c, DPO_EINVAL, "phase start must lie in [0, k]");
    c->phase_k0 = k0;
    if (c->capturable && (mpush(c, nullptr) != DPO_OK || cudaDeviceSynchronize() != cudaSuccess))
        return mfail(c, DPO_ECUDA, "writing the device step counters failed");
    return DPO_OK;
}

extern "C" int dpo_muon_get_step(const dpo_muon_ctx *c, int64_t *k)
{
    if (c == nullptr || k == nullptr)
        return DPO_EINVAL;
    if (mpull(c) != DPO_OK)
        return DPO_ECUDA;
    *k = c->k;
    return DPO_OK;
}

extern "C" int dpo_muon_set_step(dpo_muon_ctx *c, int64_t k)
{
    if (c == nullptr || k < 0)
        return DPO_EINVAL;
    if (mpull(c) != DPO_OK)
        return mfail(c, DPO_ECUDA, "reading the device step counters failed");
    c->k = k;
    if (c->phase_k0 > k)
        c->phase_k0 = k;
    if (c->capturable && (mpush(c, nullptr) != DPO_OK || cudaDeviceSynchronize() != cudaSuccess))
        return mfail(c, DPO_ECUDA, "writing the device step counters failed");
    return DPO_OK;
}

extern "C" int dpo_muon_flops(const dpo_muon_ctx *c, double *flops)
{
    if (c == nullptr || flops == nullptr)
        return DPO_EINVAL;
    // the updated-state prediction runs the Newton-Schulz chains a second
    // time (delayed training with history buffers)
    const bool twice = c->hp.correction == DPO_CORR_SAPIPE_UPDATED && c->ef && c->hp.delay == 1;
    *flops = twice ? 2.0 * c->flops : c->flops;
    return DPO_OK;
}

extern "C" int dpo_muon_set_timing(dpo_muon_ctx *c, int on)
{
    if (c == nullptr)
        return DPO_EINVAL;
    c->timing = on != 0;
    return DPO_OK;
}

extern "C" int dpo_muon_get_gemm_time(dpo_muon_ctx *c, double *ms, int64_t *launches)
{
    if (c == nullptr || ms == nullptr || launches == nullptr)
        return DPO_EINVAL;
    double total = 0.0;
    for (size_t q = 0; q + 1 < c->ev_used; q += 2) {
        cudaError_t e = cudaEventSynchronize(c->ev_pool[q + 1]);
        float t = 0.0f;
        if (e == cudaSuccess)
            e = cudaEventElapsedTime(&t, c->ev_pool[q], c->ev_pool[q + 1]);
        if (e != cudaSuccess)
            return mcuda(c, e, "timing event read");
        total += t;
    }
    *ms = total;
    *launches = c->gemm_launches;
    c->ev_used = 0;
    c->gemm_launches = 0;
    return DPO_OK;
}

extern "C" int dpo_muon_workspace_bytes(const dpo_muon_ctx *c, int64_t *bytes)
{
    if (c == nullptr || bytes == nullptr)
        return DPO_EINVAL;
    *bytes = c->ws_bytes;
    return DPO_OK;
}

extern "C" void dpo_muon_destroy(dpo_muon_ctx *c)
{
    free_ctx(c);
}
