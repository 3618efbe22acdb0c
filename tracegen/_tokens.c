/* Host-side token generation for the synthetic traces (input generation only).
 * Same integer map as tracegen.token_values: every intermediate is a
 * non-negative int64 below 2^62, so the result equals the numpy and torch
 * evaluations bit for bit.  Reductions mod 2^31 - 1 use the Mersenne identity
 * 2^31 = 1 (mod 2^31 - 1) instead of a division. */
#include <stdint.h>

#define M31 2147483647LL

/* x mod (2^31 - 1) for 0 <= x < 2^62 */
static int64_t mod_m31(int64_t x)
{
    int64_t r = (x & M31) + (x >> 31); /* < 2^32 */
    r = (r & M31) + (r >> 31);         /* <= 2^31 */
    return r >= M31 ? r - M31 : r;
}

static int32_t token(int64_t stream, int64_t pos, int64_t seed, uint32_t vocab)
{
    int64_t x = mod_m31(stream * 1000003LL + pos * 7919LL + (seed * 104729LL + 12345LL));
    x = mod_m31(x * 48271LL + 11LL);
    x = x ^ (x >> 13);
    x = mod_m31(x * 69621LL + 7LL);
    x = x ^ (x >> 11);
    x = mod_m31(x * 48271LL);
    return (int32_t)((uint32_t)x % vocab);
}

/* Prefix spans of n keys, packed back to back from out[0]: key i's span starts
 * at base + off[i], where base is the position of out[0] in the caller's
 * whole arena (so that chunks of one arena can be filled independently). */
void tg_prefix_tokens(const int64_t *key_ids, const uint32_t *plen, uint64_t n, int64_t seed, int64_t vocab,
                      int32_t *out, uint64_t *off, uint64_t base)
{
    uint64_t o = 0;
    for (uint64_t i = 0; i < n; ++i) {
        off[i] = base + o;
        for (uint32_t j = 0; j < plen[i]; ++j) out[o + j] = token(key_ids[i], (int64_t)j, seed, (uint32_t)vocab);
        o += plen[i];
    }
}
