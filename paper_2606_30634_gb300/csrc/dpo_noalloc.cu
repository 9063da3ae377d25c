// dpo_noalloc.cu -- global gradient norm and clip coefficient without any
// device allocation (dpo_grad_norm_noalloc in include/dpo.h).
//
// Why it exists: some callers cannot call cudaMalloc. A training framework
// whose caching allocator has already reserved the GPU's memory cannot let a
// library take more behind its back (the call fails, or takes memory the
// framework does not account for), and a latency-critical loop cannot take
// the device-wide synchronization cudaMalloc and cudaFree may imply. dpo_init
// allocates a small device block for its table and norm scratch; this entry
// point gives such callers the same norm and clip coefficient the clipped
// dpo_step computes, over one contiguous gradient buffer, with its scratch in
// a fixed file-scope device array instead.
//
// Scratch: g_noalloc_scratch holds one fp64 partial sum per chunk (at most
// kMaxChunks chunks of at most kChunkElems elements, so at most
// DPO_NOALLOC_MAX_NUMEL elements per call) and the arrival ticket of the
// last-CTA-finishes reduction. Every GPU that loads the library holds it until
// the process exits. All calls share it and it keeps the last call's
// contents: each call clears the ticket before its launch, and calls whose
// kernels overlap on the GPU (different streams, or different host threads,
// on one device) race on it.
//
// Chunking: a buffer is cut into equal chunks, one CTA each, of
// chunk_elems(numel) elements: about numel / kTargetCtas rounded up to a
// multiple of kMinChunk (one full round of the CTA's loads), between
// kMinChunk and kChunkElems. So a gradient of a few million elements still
// spreads over several CTAs per SM, and the largest ones use at most
// kMaxChunks partials. The chunking, and with it the summation order,
// depends only on numel: the result is deterministic.
#include "dpo.h"
#include "dpo_reduce.cuh"

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <math.h>
#include <mutex>

namespace {

using dpo::block_sum;
using dpo::kahan_add;
using dpo::NormUnroll;
using dpo::RawPacket;

constexpr int kThreads = 256;
constexpr int64_t kChunkElems = DPO_NOALLOC_CHUNK_ELEMS;
constexpr int kMaxChunks = DPO_NOALLOC_MAX_CHUNKS;
// one round of a CTA's loads of bf16 packets (two of fp32 ones)
constexpr int64_t kMinChunk =
    (int64_t)kThreads * NormUnroll<__nv_bfloat16>::value * dpo::kPacket;   // 16384
constexpr int64_t kTargetCtas = 1216;   // 8 per SM on a 152-SM GB300
constexpr size_t kTicketOffset = sizeof(double) * kMaxChunks;
constexpr size_t kScratchBytes = kTicketOffset + 256;

static_assert(kChunkElems % kMinChunk == 0, "chunks are whole rounds of loads");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// Elements per chunk for a buffer of numel elements (see the file comment).
int64_t chunk_elems(int64_t numel)
{
    int64_t c = (numel + kTargetCtas - 1) / kTargetCtas;
    c = (c + kMinChunk - 1) / kMinChunk * kMinChunk;
    return c < kMinChunk ? kMinChunk : (c > kChunkElems ? kChunkElems : c);
}

// Device address of g_noalloc_scratch per device, looked up by the first
// call on each device and kept for the life of the process (host code cannot
// use the symbol's name as a device address). This assumes the device's
// primary context lives until exit: after cudaDeviceReset the module may be
// loaded at another address, and the kept one would be stale.
constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_addr[kMaxDevices] = {};

cudaError_t scratch_address(int device, void **out)
{
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_addr[device] == nullptr) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess)
            return e;
        g_addr[device] = p;
    }
    *out = g_addr[device];
    return cudaSuccess;
}

// CTA c sums the squares of chunk c, elements [c chunk, min((c+1) chunk,
// numel)) (8-element packets; each thread issues the loads of its U packets
// of a round before summing them; Kahan fp32 per thread, fp64 block tree),
// stores the partial in the scratch array, and the last CTA to arrive adds
// the partials in chunk order and writes the norm and the clip coefficient
// min(1, max_norm / (norm + 1e-6)). Deterministic for a given numel.
template <class GT>
__global__ void __launch_bounds__(kThreads)
noalloc_sqnorm_kernel(const GT *__restrict__ grad, int64_t numel, int64_t chunk,
                      double max_norm, unsigned char *scratch, double *norm_out,
                      float *clip_out)
{
    __shared__ double red[kThreads / 32];
    __shared__ bool last;
    double *partials = reinterpret_cast<double *>(scratch);
    unsigned int *ticket = reinterpret_cast<unsigned int *>(scratch + kTicketOffset);

    const int64_t lo = (int64_t)blockIdx.x * chunk;
    const int64_t hi = lo + chunk < numel ? lo + chunk : numel;
    const int64_t pkts = hi > lo ? (hi - lo + dpo::kPacket - 1) / dpo::kPacket : 0;
    constexpr int U = NormUnroll<GT>::value;
    float sum = 0.0f, comp = 0.0f;
    for (int64_t base = threadIdx.x; base < pkts; base += (int64_t)kThreads * U) {
        int cnt[U];   // elements of the packet: 8, 1..7 (the buffer's last), 0 (none)
        RawPacket<GT> raw[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t e = lo + (base + (int64_t)u * kThreads) * dpo::kPacket;
            cnt[u] = e < hi ? (hi - e < dpo::kPacket ? (int)(hi - e) : dpo::kPacket) : 0;
        }
#pragma unroll
        for (int u = 0; u < U; ++u)
            if (cnt[u] == dpo::kPacket)
                raw[u].load(grad + lo + (base + (int64_t)u * kThreads) * dpo::kPacket);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            float s = 0.0f;
            if (cnt[u] == dpo::kPacket) {
                s = raw[u].sqsum();
            } else {
                const GT *p = grad + lo + (base + (int64_t)u * kThreads) * dpo::kPacket;
                for (int i = 0; i < cnt[u]; ++i) {
                    const float x = dpo::ld1(p + i);
                    s += x * x;
                }
            }
            kahan_add(sum, comp, s);
        }
    }
    const double cta = block_sum<kThreads>((double)sum - (double)comp, red);
    if (threadIdx.x == 0) {
        partials[blockIdx.x] = cta;
        __threadfence();
        last = (atomicAdd(ticket, 1u) == gridDim.x - 1);
    }
    __syncthreads();
    if (!last)
        return;
    __threadfence();
    double acc = 0.0;
    for (int b = threadIdx.x; b < (int)gridDim.x; b += kThreads)
        acc += __ldcg(partials + b);
    const double total = block_sum<kThreads>(acc, red);
    if (threadIdx.x == 0) {
        const double norm = sqrt(total);
        double coef = max_norm > 0.0 ? max_norm / (norm + 1e-6) : 1.0;
        coef = coef > 1.0 ? 1.0 : coef;   // a NaN norm stays NaN
        *norm_out = norm;
        *clip_out = (float)coef;
        *ticket = 0u;
    }
}

}  // namespace

extern "C" int dpo_grad_norm_noalloc(const void *grad, int64_t numel, dpo_dtype grad_dtype,
                                     float max_grad_norm, double *norm_out, float *clip_out,
                                     void *cuda_stream)
{
    if (grad_dtype != DPO_F32 && grad_dtype != DPO_BF16)
        return DPO_EDTYPE;
    if (numel < 0 || (numel > 0 && grad == nullptr) || norm_out == nullptr ||
        clip_out == nullptr || !isfinite(max_grad_norm))
        return DPO_EINVAL;
    if (numel > DPO_NOALLOC_MAX_NUMEL)
        return DPO_EINVAL;   // more chunks than the static scratch array holds
    if ((reinterpret_cast<uintptr_t>(grad) % 32) != 0 ||
        (reinterpret_cast<uintptr_t>(norm_out) % 8) != 0 ||
        (reinterpret_cast<uintptr_t>(clip_out) % 4) != 0)
        return DPO_EALIGN;

    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kMaxDevices)
        return DPO_ECUDA;
    void *scratch = nullptr;
    if (scratch_address(device, &scratch) != cudaSuccess)
        return DPO_ECUDA;
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    unsigned char *base = static_cast<unsigned char *>(scratch);
    // the ticket must start at zero (a previous call may have been cut short)
    if (cudaMemsetAsync(base + kTicketOffset, 0, sizeof(unsigned int), s) != cudaSuccess)
        return DPO_ECUDA;
    const int64_t chunk = chunk_elems(numel);
    const int grid = numel > 0 ? (int)((numel + chunk - 1) / chunk) : 1;
    if (grad_dtype == DPO_BF16)
        noalloc_sqnorm_kernel<__nv_bfloat16><<<grid, kThreads, 0, s>>>(
            static_cast<const __nv_bfloat16 *>(grad), numel, chunk, (double)max_grad_norm,
            base, norm_out, clip_out);
    else
        noalloc_sqnorm_kernel<float><<<grid, kThreads, 0, s>>>(
            static_cast<const float *>(grad), numel, chunk, (double)max_grad_norm, base,
            norm_out, clip_out);
    return cudaGetLastError() == cudaSuccess ? DPO_OK : DPO_ECUDA;
}
