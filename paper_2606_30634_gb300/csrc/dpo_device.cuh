// dpo_device.cuh -- device helpers shared by the kernels of the delayed step:
// packet I/O (fp32 packets as one 256-bit access, bf16 packets as one
// 128-bit access, streaming cache hints) and the per-thread tensor cursor of
// the grid-stride walk over the virtual concatenation of the tensors.
#pragma once

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

}  // namespace
}  // namespace dpo
