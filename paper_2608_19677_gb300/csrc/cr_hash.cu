// a1: prefix-span routing key (cr_hash_prefixes).
//
// The key is the wrapping sum of one SplitMix64-mixed term per 64-bit word
// (two int32 tokens) of the prefix plus a length term, so any partition of the
// words over lanes gives the same result.  One warp hashes one request: lanes
// stride over the span with 16-byte streaming loads (four tokens = two words
// per load, up to eight loads in flight per lane: the next group of four is
// fetched while the current one is mixed), then the warp reduces its partial
// sums; the next request's span descriptor is fetched a request ahead.  The path is an HBM stream of 4*P bytes per request; the per-word mix
// (about two dozen integer instructions) keeps the ALU just under that stream
// rate on sm_103a.
#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

constexpr int kHashBlock = 256;

__device__ __forceinline__ unsigned long long word_term(uint32_t lo, uint32_t hi, unsigned long long k)
{
    unsigned long long w = (unsigned long long)lo | ((unsigned long long)hi << 32);
    return cr_fmix64(w ^ k);
}

// Words [first, nw) of a span starting at `base`, one per lane, scalar loads;
// used for unaligned spans and for the last words of aligned ones.
__device__ __forceinline__ unsigned long long scalar_words(const int32_t *__restrict__ base, uint32_t P,
                                                           uint32_t first, uint32_t nw,
                                                           unsigned long long salt, uint32_t lane)
{
    unsigned long long acc = 0;
    for (uint32_t i = first + lane; i < nw; i += 32) {
        uint32_t lo = (uint32_t)__ldcs(base + 2 * i);
        uint32_t hi = (2 * i + 1 < P) ? (uint32_t)__ldcs(base + 2 * i + 1) : 0u;
        acc += word_term(lo, hi, salt + (unsigned long long)(i + 1) * CR_GAMMA);
    }
    return acc;
}

__device__ __forceinline__ void load4(int4 (&x)[4], const int4 *__restrict__ b4, uint32_t v, uint32_t nvec)
{
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t i = v + 32u * q;
        if (i < nvec)
            x[q] = __ldcs(b4 + i);
        else
            x[q] = make_int4(0, 0, 0, 0);
    }
}

// 64 registers per thread: 32 warps per SM, which measured faster than larger
// unrolls at lower occupancy.
__global__ void __launch_bounds__(kHashBlock, 4)
k_hash_prefixes(const int32_t *__restrict__ tok, const unsigned long long *__restrict__ off,
                const uint32_t *__restrict__ plen, unsigned long long n, unsigned long long salt,
                unsigned long long *__restrict__ out)
{
    const uint32_t lane = cr_lane();
    const unsigned long long nwarps = ((unsigned long long)gridDim.x * blockDim.x) >> 5;
    const unsigned long long G64 = 64ull * CR_GAMMA, G256 = 256ull * CR_GAMMA;
    unsigned long long r = ((unsigned long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    unsigned long long o_next = 0;
    uint32_t P_next = 0;
    if (r < n) {
        o_next = off[r];
        P_next = plen[r];
    }
    for (; r < n; r += nwarps) {
        const unsigned long long o = o_next;
        const uint32_t P = P_next;
        if (r + nwarps < n) {  // the next request's span descriptor is in flight meanwhile
            o_next = off[r + nwarps];
            P_next = plen[r + nwarps];
        }
        const uint32_t nw = (P + 1) >> 1;
        const int32_t *base = tok + o;
        unsigned long long acc = 0;
        if ((o & 3ull) == 0) {
            // 16-byte aligned: vector v holds words 2v and 2v+1.  Two groups of
            // four vectors per lane are in flight: the next group loads while
            // the current one is mixed.
            const uint32_t nvec = P >> 2;
            const int4 *b4 = reinterpret_cast<const int4 *>(base);
            uint32_t v = lane;
            unsigned long long k = salt + (unsigned long long)(2 * lane + 1) * CR_GAMMA;  // key of word 2v
            int4 cur[4];
            load4(cur, b4, v, nvec);
            while (v < nvec) {
                int4 nxt[4];
                load4(nxt, b4, v + 128u, nvec);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    if (v + 32u * q < nvec) {
                        const unsigned long long kq = k + (unsigned long long)q * G64;
                        acc += word_term(cur[q].x, cur[q].y, kq) + word_term(cur[q].z, cur[q].w, kq + CR_GAMMA);
                    }
                }
#pragma unroll
                for (int q = 0; q < 4; ++q) cur[q] = nxt[q];
                v += 128u;
                k += G256;
            }
            acc += scalar_words(base, P, 2 * nvec, nw, salt, lane);
        } else if ((o & 1ull) == 0) {
            // 8-byte aligned: one word per load
            const uint32_t nfull = P >> 1;
            const uint2 *b2 = reinterpret_cast<const uint2 *>(base);
            uint32_t i = lane;
            unsigned long long k = salt + (unsigned long long)(lane + 1) * CR_GAMMA;
            const unsigned long long G32 = 32ull * CR_GAMMA;
            for (; i + 32 < nfull; i += 64, k += G64) {
                uint2 a = __ldcs(b2 + i), b = __ldcs(b2 + i + 32);
                acc += word_term(a.x, a.y, k) + word_term(b.x, b.y, k + G32);
            }
            for (; i < nfull; i += 32, k += G32) {
                uint2 a = __ldcs(b2 + i);
                acc += word_term(a.x, a.y, k);
            }
            acc += scalar_words(base, P, nfull, nw, salt, lane);
        } else {
            acc = scalar_words(base, P, 0, nw, salt, lane);
        }
        acc = cr_warp_sum_u64(acc);
        if (lane == 0) out[r] = cr_fmix64(salt ^ (unsigned long long)P) + acc;
    }
}

}  // namespace

extern "C" int cr_hash_prefixes(cr_ctx *ctx, const int32_t *d_tokens, const uint64_t *d_off,
                                const uint32_t *d_plen, uint64_t n, uint64_t salt, uint64_t *d_key_out)
{
    cr_nvtx_range nv("cr_hash_prefixes");
    if (!ctx) return CR_EINVAL;
    if (n == 0) return CR_OK;
    if (!d_tokens || !d_off || !d_plen || !d_key_out)
        return cr_fail(ctx, CR_EINVAL, "cr_hash_prefixes: NULL pointer");
    const unsigned int warps_per_block = kHashBlock / 32;
    // many more blocks than fit at once (32 per SM): blocks start as others
    // finish, which evens out the widely varying span lengths across the SMs
    unsigned int grid = cr_blocks(n, warps_per_block, (unsigned int)ctx->num_sms * 32u);
    const int pi = cr_prof_begin(ctx, ctx->stream, CR_PROF_HASH);
    CR_LAUNCH(ctx, k_hash_prefixes, grid, kHashBlock, 0, d_tokens, (const unsigned long long *)d_off,
              d_plen, (unsigned long long)n, (unsigned long long)salt, (unsigned long long *)d_key_out);
    cr_prof_end(ctx, ctx->stream, pi);
    return CR_OK;
}
