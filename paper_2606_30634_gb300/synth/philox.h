/*
 * philox.h -- counter-based random numbers for the seeded synthetic inputs.
 *
 * Philox4x32-10 as defined by Salmon, Moraes, Dror and Shaw, "Parallel
 * Random Numbers: As Easy as 1, 2, 3" (SC'11): a 10-round Feistel-like
 * network on a 128-bit counter under a 64-bit key, with the multipliers
 * 0xD2511F53 / 0xCD9E8D57 and the key schedule (Weyl) constants
 * 0x9E3779B9 / 0xBB67AE85.
 *
 * The same inline functions compile as host C/C++ and as CUDA device code, so
 * the device fill kernels and the host fills that tests and the oracle side use
 * produce bit-identical values. Only integer operations, one int -> float
 * conversion (exact) and one fp32 multiply (IEEE, round to nearest even) are
 * involved. This file holds input generation only, none of the optimizer's
 * arithmetic.
 *
 * Draw for element i of stream s at step k under seed S:
 *   counter = (lo32(i), hi32(i), k, s), key = (lo32(S), hi32(S)).
 * Normal: Irwin-Hall sum of the eight 16-bit halves of the four output
 *   words, centred (integer), times an fp32 scale sigma / (65536 sqrt(2/3)):
 *   mean 0, standard deviation sigma, support +-4.9 sigma.
 * Uniform: top 24 bits of the first output word times 2^-24, in [0, 1).
 */
#ifndef DPO_SYNTH_PHILOX_H
#define DPO_SYNTH_PHILOX_H

#include <stdint.h>
#include <string.h>

#ifdef __CUDACC__
#define SYNTH_HD __host__ __device__ __forceinline__
#else
#define SYNTH_HD static inline
#endif

#define SYNTH_PHILOX_M0 0xD2511F53u
#define SYNTH_PHILOX_M1 0xCD9E8D57u
#define SYNTH_PHILOX_W0 0x9E3779B9u
#define SYNTH_PHILOX_W1 0xBB67AE85u

typedef struct { uint32_t v[4]; } synth_u32x4;

SYNTH_HD void synth_mulhilo32(uint32_t a, uint32_t b, uint32_t *hi, uint32_t *lo)
{
    const uint64_t p = (uint64_t)a * (uint64_t)b;
    *hi = (uint32_t)(p >> 32);
    *lo = (uint32_t)p;
}

SYNTH_HD synth_u32x4 synth_philox4x32_10(synth_u32x4 c, uint32_t k0, uint32_t k1)
{
    for (int r = 0; r < 10; ++r) {
        uint32_t hi0, lo0, hi1, lo1;
        synth_mulhilo32(SYNTH_PHILOX_M0, c.v[0], &hi0, &lo0);
        synth_mulhilo32(SYNTH_PHILOX_M1, c.v[2], &hi1, &lo1);
        synth_u32x4 n;
        n.v[0] = hi1 ^ c.v[1] ^ k0;
        n.v[1] = lo1;
        n.v[2] = hi0 ^ c.v[3] ^ k1;
        n.v[3] = lo0;
        c = n;
        k0 += SYNTH_PHILOX_W0;
        k1 += SYNTH_PHILOX_W1;
    }
    return c;
}

SYNTH_HD synth_u32x4 synth_draw(uint64_t seed, uint32_t stream, uint32_t step, uint64_t i)
{
    synth_u32x4 c;
    c.v[0] = (uint32_t)i;
    c.v[1] = (uint32_t)(i >> 32);
    c.v[2] = step;
    c.v[3] = stream;
    return synth_philox4x32_10(c, (uint32_t)seed, (uint32_t)(seed >> 32));
}

/* Centred Irwin-Hall integer: sum of eight 16-bit halves minus 8 * 32767.5. */
SYNTH_HD int32_t synth_irwin_hall8(synth_u32x4 w)
{
    uint32_t s = 0;
    for (int j = 0; j < 4; ++j)
        s += (w.v[j] & 0xFFFFu) + (w.v[j] >> 16);
    return (int32_t)s - 262140;
}

/* Normal draw: scale is synth_normal_scale(sigma), computed once on the
 * host and passed to both sides as the same fp32 value. */
SYNTH_HD float synth_normal(uint64_t seed, uint32_t stream, uint32_t step, uint64_t i, float scale)
{
    return (float)synth_irwin_hall8(synth_draw(seed, stream, step, i)) * scale;
}

SYNTH_HD float synth_uniform(uint64_t seed, uint32_t stream, uint32_t step, uint64_t i)
{
    return (float)(synth_draw(seed, stream, step, i).v[0] >> 8) * 5.9604644775390625e-08f;
}

/* fp32 -> bf16 bits, round to nearest even (finite inputs: the generator
 * never produces anything else). */
SYNTH_HD uint16_t synth_bf16_bits(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    const uint32_t lsb = (u >> 16) & 1u;
    return (uint16_t)((u + 0x7FFFu + lsb) >> 16);
}

#endif /* DPO_SYNTH_PHILOX_H */
