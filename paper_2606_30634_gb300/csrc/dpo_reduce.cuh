// dpo_reduce.cuh -- the pieces of the deterministic sum of squares that the
// gradient-norm kernels share (grad_sqnorm_kernel over a tensor table in
// dpo_kernels.cu, and the single-buffer kernel of dpo_noalloc.cu): the sum of
// squares of one 8-element packet, Kahan-compensated fp32 accumulation per
// thread, and a fixed warp-shuffle tree over the block in fp64.
#pragma once

#include "dpo_device.cuh"

namespace dpo {
namespace {

// Sum of the squares of elements [e, min(e + 8, numel)) of grad: a full
// packet is one vector load and a fixed pairwise tree; a partial one (the
// last packet of a buffer) adds its elements in order.
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

// One full packet held as loaded (bf16: 16 bytes, fp32: 32 bytes), so that a
// thread can issue the loads of several packets before it sums any of them;
// sqsum() is packet_sqsum's tree for a full packet.
template <class GT> struct RawPacket;

template <> struct RawPacket<__nv_bfloat16> {
    uint4 q;
    __device__ __forceinline__ void load(const __nv_bfloat16 *p)
    {
        q = __ldcs(reinterpret_cast<const uint4 *>(p));
    }
    __device__ __forceinline__ float sqsum() const
    {
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
        float g[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            g[2 * j] = __uint_as_float(w[j] << 16);
            g[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
        }
        return ((g[0] * g[0] + g[1] * g[1]) + (g[2] * g[2] + g[3] * g[3])) +
               ((g[4] * g[4] + g[5] * g[5]) + (g[6] * g[6] + g[7] * g[7]));
    }
};

template <> struct RawPacket<float> {
    float g[8];
    __device__ __forceinline__ void load(const float *p) { ld8(p, g); }
    __device__ __forceinline__ float sqsum() const
    {
        return ((g[0] * g[0] + g[1] * g[1]) + (g[2] * g[2] + g[3] * g[3])) +
               ((g[4] * g[4] + g[5] * g[5]) + (g[6] * g[6] + g[7] * g[7]));
    }
};

// Packets a thread keeps in flight per round of a norm pass: 128 bytes of
// gradient either way (eight bf16 packets, four fp32 packets).
template <class GT> struct NormUnroll { static constexpr int value = 4; };
template <> struct NormUnroll<__nv_bfloat16> { static constexpr int value = 8; };

// Kahan-compensated fp32 accumulation of per-packet sums of squares: the
// compensation keeps a thread's error near one rounding however many
// packets it visits.
__device__ __forceinline__ void kahan_add(float &sum, float &c, float x)
{
    const float y = x - c;
    const float t = sum + y;
    c = (t - sum) - y;
    sum = t;
}

// Sum of x over the NT threads of the block in fp64, in a fixed order
// (shuffle tree within each warp, then over the warps' sums); the result is
// valid in thread 0. red holds NT / 32 doubles of shared memory.
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
    return r;
}

}  // namespace
}  // namespace dpo
