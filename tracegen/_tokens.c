/* Host-side token generation for the synthetic traces (input generation only).
 * Same integer map as tracegen.token_values: every intermediate is a
 * non-negative int64 below 2^62, so the result equals the numpy and torch
 * evaluations bit for bit. */
#include <stdint.h>

#define M31 2147483647LL

static int32_t token(int64_t stream, int64_t pos, int64_t seed, int64_t vocab)
{
    int64_t x = (stream * 1000003LL + pos * 7919LL + (seed * 104729LL + 12345LL)) % M31;
    x = (x * 48271LL + 11LL) % M31;
    x = x ^ (x >> 13);
    x = (x * 69621LL + 7LL) % M31;
    x = x ^ (x >> 11);
    x = (x * 48271LL) % M31;
    return (int32_t)(x % vocab);
}

/* Prefix spans of n keys, packed back to back: key i's span starts at off[i]. */
void tg_prefix_tokens(const int64_t *key_ids, const uint32_t *plen, uint64_t n, int64_t seed, int64_t vocab,
                      int32_t *out, uint64_t *off)
{
    uint64_t o = 0;
    for (uint64_t i = 0; i < n; ++i) {
        off[i] = o;
        for (uint32_t j = 0; j < plen[i]; ++j) out[o + j] = token(key_ids[i], (int64_t)j, seed, vocab);
        o += plen[i];
    }
}
