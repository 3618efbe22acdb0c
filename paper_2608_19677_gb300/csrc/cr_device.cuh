// Device-side building blocks shared by the kernels of this library.
#pragma once

#include <stdint.h>

#define CR_GAMMA 0x9e3779b97f4a7c15ull

// SplitMix64 finaliser (Steele, Lea and Flood, OOPSLA 2014).
__device__ __forceinline__ unsigned long long cr_fmix64(unsigned long long z)
{
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

// Philox4x64-10 (Salmon, Moraes, Dror and Shaw, SC 2011): ten rounds of two
// 64x64->128 multiplies with the published multipliers and Weyl key bumps.
struct cr_u64x4 {
    unsigned long long x, y, z, w;
};

__device__ __forceinline__ cr_u64x4 cr_philox4x64_10(unsigned long long c0, unsigned long long c1,
                                                      unsigned long long c2, unsigned long long c3,
                                                      unsigned long long k0, unsigned long long k1)
{
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const unsigned long long M0 = 0xD2E7470EE14C6C93ull, M1 = 0xCA5A826395121157ull;
        unsigned long long hi0 = __umul64hi(M0, c0), lo0 = M0 * c0;
        unsigned long long hi1 = __umul64hi(M1, c2), lo1 = M1 * c2;
        unsigned long long n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
        k0 += 0x9E3779B97F4A7C15ull;
        k1 += 0xBB67AE8584CAA73Bull;
    }
    cr_u64x4 o = {c0, c1, c2, c3};
    return o;
}

// floor(u * m / 2^64)
__device__ __forceinline__ uint32_t cr_scale(unsigned long long u, unsigned long long m)
{
    return (uint32_t)__umul64hi(u, m);
}

// Jump consistent hash (Lamping and Veach 2014) with the jump evaluated exactly
// in integers: j = floor((b + 1) * 2^31 / d), d = (k >> 33) + 1 in [1, 2^31].
// No 64-bit division: a single-precision estimate of the quotient settles
// j >= R whenever it exceeds R + 2; otherwise it is at most R + 2 <= 8194, and
// one integer step either way (products below 2^46) gives the exact floor.  The
// estimate is the numerator (exact in float) over d rounded to float (relative
// error 2^-24), divided by the fast approximate division (at most 2 ulp for
// divisors below 2^126): relative error below 2^-21, so an error below 0.01
// wherever the estimate is at most R + 2.
__device__ __forceinline__ uint32_t cr_jump_hash(unsigned long long k, uint32_t R)
{
    uint32_t b = 0, j = 0;
    while (j < R) {
        b = j;
        k = k * 2862933555777941757ull + 1ull;
        const uint32_t d = (uint32_t)(k >> 33) + 1u;
        const unsigned long long num = (unsigned long long)(b + 1u) << 31;
        const float est = __fdividef((float)(b + 1u) * 2147483648.0f, (float)d);
        if (est > (float)R + 2.0f) break;  // the exact quotient is above R as well
        uint32_t q = (uint32_t)est;
        if ((unsigned long long)q * d > num)
            --q;
        else if ((unsigned long long)(q + 1u) * d <= num)
            ++q;
        j = q;
    }
    return b;
}

__device__ __forceinline__ unsigned long long cr_warp_sum_u64(unsigned long long v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ unsigned long long cr_warp_min_u64(unsigned long long v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w < v ? w : v;
    }
    return v;
}

__device__ __forceinline__ uint32_t cr_lane() { return threadIdx.x & 31u; }
