// a8, a9: shadow replay (cr_shadow_replay).
//
//   partition  stable radix sort of (replica, destination) over every routed
//              request: each (replica, destination) stream in arrival order
//   replay     one warp per stream; the stream's LRU at the LARGEST capacity
//              lives in shared memory (key + access stamp per entry, spread
//              over the lanes).  A hit's depth (1 + entries touched after it)
//              decides the hit at every smaller capacity at once, because LRU
//              caches are nested (Mattson et al. 1970): the cache of capacity c
//              is the c most recent entries of any larger one.
//   state      kept between calls as keys in recency order (most recent first);
//              stamps are re-derived from that order at the start of a call.
#include <stdlib.h>
#include <string.h>

#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

struct replay_caps {
    uint32_t n_caps;
    uint32_t cap[CR_MAX_CAPS];
};

__global__ void k_part_keys(const uint16_t *__restrict__ dest, unsigned long long n, uint32_t n_rep, uint32_t R,
                            int dbits, uint32_t *__restrict__ ck, uint32_t *status)
{
    const unsigned long long total = n * n_rep;
    bool bad = false;
    for (unsigned long long j = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; j < total;
         j += (unsigned long long)gridDim.x * blockDim.x) {
        uint32_t rep = (uint32_t)(j / n);
        uint32_t d = dest[j];
        if (d >= R) {
            bad = true;
            ck[j] = n_rep << dbits;  // sorts after every valid stream: skipped
        } else {
            ck[j] = (rep << dbits) | d;
        }
    }
    if (__any_sync(0xffffffffu, bad) && cr_lane() == 0) atomicOr(status, CR_FLAG_BADDEST);
}

// start[s] = first position of stream s = (rep, r) in the sorted composite keys.
__global__ void k_stream_starts(const uint32_t *__restrict__ sk, unsigned long long m, uint32_t n_rep, uint32_t R,
                                int dbits, uint32_t *__restrict__ start)
{
    const uint32_t ns = n_rep * R;
    for (uint32_t s = blockIdx.x * blockDim.x + threadIdx.x; s <= ns; s += gridDim.x * blockDim.x) {
        uint32_t target = (s == ns) ? (n_rep << dbits) : (((s / R) << dbits) | (s % R));
        unsigned long long lo = 0, hi = m;
        while (lo < hi) {
            unsigned long long mid = (lo + hi) >> 1;
            if (sk[mid] < target)
                lo = mid + 1;
            else
                hi = mid;
        }
        start[s] = (uint32_t)lo;
    }
}

template <int E>  // entries per lane: cmax <= 32 * E
__global__ void k_lru_replay(const replay_caps caps, uint32_t cmax, uint32_t n_rep, uint32_t R,
                             const uint32_t *__restrict__ start, const uint32_t *__restrict__ sval,
                             unsigned long long n, const unsigned long long *__restrict__ keys,
                             const uint32_t *__restrict__ plen, const uint32_t *__restrict__ slen,
                             unsigned long long *__restrict__ st_keys, uint32_t *__restrict__ st_fill,
                             unsigned long long *__restrict__ ctr, uint32_t *status)
{
    extern __shared__ unsigned long long sm[];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
    const uint32_t slots = 32u * E;
    unsigned long long *sk = sm + (size_t)warp * slots;                                     // keys
    uint32_t *ss = reinterpret_cast<uint32_t *>(sm + (size_t)wpb * slots) + (size_t)warp * slots;  // stamps
    const uint32_t stream = blockIdx.x * wpb + warp;
    if (stream >= n_rep * R) return;
    const uint32_t rep = stream / R, r = stream % R;
    const uint32_t b = start[stream], e = start[stream + 1];
    if (b == e) return;

    // load state: rank q (0 = most recent) gets stamp fill - q
    uint32_t fill = st_fill[stream];
    const unsigned long long *gk = st_keys + (unsigned long long)stream * cmax;
    for (uint32_t q = lane; q < fill; q += 32) {
        sk[q] = gk[q];
        ss[q] = fill - q;
    }
    __syncwarp();
    uint32_t clock = fill;

    unsigned long long c_req = 0, c_prompt = 0;
    unsigned long long c_hit[CR_MAX_CAPS], c_hit_tok[CR_MAX_CAPS];
#pragma unroll
    for (int c = 0; c < CR_MAX_CAPS; ++c) c_hit[c] = c_hit_tok[c] = 0;
    const unsigned long long rep_base = (unsigned long long)rep * n;

    for (uint32_t t0 = b; t0 < e; t0 += 32) {
        // stage up to 32 requests of the stream, one per lane
        unsigned long long mykey = 0;
        uint32_t myP = 0, myS = 0;
        if (t0 + lane < e) {
            unsigned long long i = (unsigned long long)sval[t0 + lane] - rep_base;
            mykey = keys[i];
            myP = plen[i];
            myS = slen[i];
        }
        const uint32_t cnt = (e - t0) < 32u ? (e - t0) : 32u;
        for (uint32_t j = 0; j < cnt; ++j) {
            const unsigned long long key = __shfl_sync(0xffffffffu, mykey, j);
            const uint32_t P = __shfl_sync(0xffffffffu, myP, j);
            const uint32_t S = __shfl_sync(0xffffffffu, myS, j);
            // lookup
            int mine = -1;
#pragma unroll
            for (int x = 0; x < E; ++x) {
                uint32_t idx = (uint32_t)x * 32u + lane;
                if (idx < fill && sk[idx] == key) mine = (int)idx;
            }
            const uint32_t hb = __ballot_sync(0xffffffffu, mine >= 0);
            uint32_t depth = 0xffffffffu;
            ++clock;
            if (hb) {
                const uint32_t hl = __ffs(hb) - 1;
                const uint32_t hs = (uint32_t)__shfl_sync(0xffffffffu, mine, hl);
                const uint32_t s_hit = ss[hs];
                uint32_t newer = 0;
#pragma unroll
                for (int x = 0; x < E; ++x) {
                    uint32_t idx = (uint32_t)x * 32u + lane;
                    if (idx < fill && ss[idx] > s_hit) ++newer;
                }
                depth = 1u + __reduce_add_sync(0xffffffffu, newer);
                __syncwarp();
                if (lane == hl) ss[hs] = clock;
            } else if (fill < cmax) {
                if (lane == 0) {
                    sk[fill] = key;
                    ss[fill] = clock;
                }
                ++fill;
            } else {
                // evict the least recent entry (stamps are unique)
                uint32_t lmin = 0xffffffffu, lidx = 0;
#pragma unroll
                for (int x = 0; x < E; ++x) {
                    uint32_t idx = (uint32_t)x * 32u + lane;
                    if (idx < fill && ss[idx] < lmin) {
                        lmin = ss[idx];
                        lidx = idx;
                    }
                }
                const uint32_t wmin = __reduce_min_sync(0xffffffffu, lmin);
                const uint32_t vl = __ffs(__ballot_sync(0xffffffffu, lmin == wmin)) - 1;
                const uint32_t vidx = __shfl_sync(0xffffffffu, lidx, vl);
                __syncwarp();
                if (lane == 0) {
                    sk[vidx] = key;
                    ss[vidx] = clock;
                }
            }
            __syncwarp();
            c_req += 1;
            c_prompt += (unsigned long long)P + S;
#pragma unroll
            for (int c = 0; c < CR_MAX_CAPS; ++c) {
                if (c < (int)caps.n_caps && depth <= caps.cap[c]) {
                    c_hit[c] += 1;
                    c_hit_tok[c] += P;
                }
            }
        }
    }
    if (clock < fill) atomicOr(status, CR_FLAG_OVERFLOW);  // stamp counter wrapped

    // store state in recency order: rank = entries with a newer stamp
    unsigned long long *gkw = st_keys + (unsigned long long)stream * cmax;
#pragma unroll
    for (int x = 0; x < E; ++x) {
        uint32_t idx = (uint32_t)x * 32u + lane;
        if (idx < fill) {
            const uint32_t my = ss[idx];
            uint32_t rank = 0;
            for (uint32_t f = 0; f < fill; ++f) rank += (ss[f] > my) ? 1u : 0u;
            gkw[rank] = sk[idx];
        }
    }
    if (lane == 0) {
        st_fill[stream] = fill;
#pragma unroll
        for (int c = 0; c < CR_MAX_CAPS; ++c) {
            if (c < (int)caps.n_caps) {
                unsigned long long *C =
                    ctr + (((unsigned long long)rep * caps.n_caps + c) * R + r) * CR_CTR_FIELDS;
                C[0] += c_req;
                C[1] += c_hit[c];
                C[2] += c_hit_tok[c];
                C[3] += c_prompt;
                C[4] += c_prompt - c_hit_tok[c];
            }
        }
    }
}

int bits_for(uint64_t v)
{
    int b = 0;
    while (b < 64 && (v >> b) != 0) ++b;
    return b;
}

template <int E>
int launch_replay(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, const uint32_t *start, const uint32_t *sval,
                  uint64_t n, const uint64_t *d_key, const uint32_t *d_plen, const uint32_t *d_slen, uint64_t *d_ctr)
{
    const uint32_t wpb = E >= 16 ? 4 : 8;
    const size_t smem = (size_t)wpb * 32 * E * (sizeof(unsigned long long) + sizeof(uint32_t));
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_replay<E>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    const uint32_t ns = rp->n_rep * rp->R;
    CR_LAUNCH(ctx, k_lru_replay<E>, (ns + wpb - 1) / wpb, wpb * 32, smem, caps, rp->cmax, rp->n_rep, rp->R, start,
              sval, (unsigned long long)n, (const unsigned long long *)d_key, d_plen, d_slen, rp->d_keys, rp->d_fill,
              (unsigned long long *)d_ctr, ctx->d_status);
    return CR_OK;
}

}  // namespace

extern "C" int cr_replay_create(cr_ctx *ctx, uint32_t n_rep, uint32_t R, const uint32_t *caps, uint32_t n_caps,
                                cr_replay **out)
{
    if (!ctx || !out || !caps) return CR_EINVAL;
    *out = nullptr;
    if (n_rep == 0 || n_rep > CR_MAX_REPLICAS) return cr_fail(ctx, CR_EINVAL, "replay: n_rep=%u", n_rep);
    if (R == 0 || R > CR_MAX_R) return cr_fail(ctx, CR_EINVAL, "replay: R=%u", R);
    if (n_caps == 0 || n_caps > CR_MAX_CAPS) return cr_fail(ctx, CR_EINVAL, "replay: n_caps=%u", n_caps);
    uint32_t cmax = 0;
    for (uint32_t c = 0; c < n_caps; ++c) {
        if (caps[c] == 0 || caps[c] > CR_MAX_CAP) return cr_fail(ctx, CR_EINVAL, "replay: cap %u", caps[c]);
        cmax = caps[c] > cmax ? caps[c] : cmax;
    }
    if ((uint64_t)n_rep * R >= (1ull << 31)) return cr_fail(ctx, CR_EINVAL, "replay: too many streams");
    cr_replay *rp = (cr_replay *)calloc(1, sizeof(cr_replay));
    if (!rp) return cr_fail(ctx, CR_ENOMEM, "replay: host allocation failed");
    rp->n_rep = n_rep;
    rp->R = R;
    rp->n_caps = n_caps;
    rp->cmax = cmax;
    memcpy(rp->caps, caps, n_caps * sizeof(uint32_t));
    rp->n_streams = (uint64_t)n_rep * R;
    if (cudaMalloc(&rp->d_keys, rp->n_streams * cmax * sizeof(unsigned long long)) != cudaSuccess ||
        cudaMalloc(&rp->d_fill, rp->n_streams * sizeof(uint32_t)) != cudaSuccess) {
        cudaGetLastError();
        if (rp->d_keys) cudaFree(rp->d_keys);
        free(rp);
        return cr_fail(ctx, CR_ENOMEM, "replay: cannot allocate state");
    }
    *out = rp;
    return cr_replay_reset(ctx, rp);
}

extern "C" int cr_replay_reset(cr_ctx *ctx, cr_replay *rp)
{
    if (!ctx || !rp) return CR_EINVAL;
    CR_CUDA(ctx, cudaMemsetAsync(rp->d_fill, 0, rp->n_streams * sizeof(uint32_t), ctx->stream));
    return CR_OK;
}

extern "C" int cr_replay_destroy(cr_ctx *ctx, cr_replay *rp)
{
    if (!rp) return CR_OK;
    if (ctx) cudaStreamSynchronize(ctx->stream);
    cudaFree(rp->d_keys);
    cudaFree(rp->d_fill);
    free(rp);
    return CR_OK;
}

extern "C" int cr_shadow_replay(cr_ctx *ctx, cr_replay *rp, const uint64_t *d_key, const uint32_t *d_plen,
                                const uint32_t *d_slen, const uint16_t *d_dest, uint64_t n, uint64_t *d_ctr)
{
    if (!ctx || !rp) return CR_EINVAL;
    if (n == 0) return CR_OK;
    if (!d_key || !d_plen || !d_slen || !d_dest || !d_ctr)
        return cr_fail(ctx, CR_EINVAL, "cr_shadow_replay: NULL pointer");
    const uint64_t m = n * rp->n_rep;
    if (n >= (1ull << 31) || m >= 0xffffffffull)
        return cr_fail(ctx, CR_EINVAL, "cr_shadow_replay: n * n_rep must be < 2^32 - 1");
    const int dbits = bits_for(rp->R - 1) ? bits_for(rp->R - 1) : 1;
    const int rbits = bits_for(rp->n_rep);  // rep == n_rep marks a skipped request
    if (dbits + rbits > 32) return cr_fail(ctx, CR_EINVAL, "cr_shadow_replay: composite key too wide");
    void *pk, *ps;
    CR_TRY(cr_scratch(ctx, SCR_REPLAY_IDX, m * sizeof(uint32_t), &pk));
    CR_TRY(cr_scratch(ctx, SCR_REPLAY_START, (rp->n_streams + 1) * sizeof(uint32_t), &ps));
    uint32_t *ck = (uint32_t *)pk, *start = (uint32_t *)ps;
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    CR_LAUNCH(ctx, k_part_keys, cr_blocks(m, 256, gcap), 256, 0, d_dest, (unsigned long long)n, rp->n_rep, rp->R,
              dbits, ck, ctx->d_status);
    const uint32_t *sk = nullptr, *sval = nullptr;
    CR_TRY(cr_radix_sort_u32(ctx, ck, nullptr, m, dbits + rbits, &sk, &sval));
    CR_LAUNCH(ctx, k_stream_starts, cr_blocks(rp->n_streams + 1, 256, gcap), 256, 0, sk, (unsigned long long)m,
              rp->n_rep, rp->R, dbits, start);
    replay_caps caps;
    caps.n_caps = rp->n_caps;
    for (uint32_t c = 0; c < CR_MAX_CAPS; ++c) caps.cap[c] = c < rp->n_caps ? rp->caps[c] : 0;
    const uint32_t E = (rp->cmax + 31) / 32;
    if (E <= 1) return launch_replay<1>(ctx, rp, caps, start, sval, n, d_key, d_plen, d_slen, d_ctr);
    if (E <= 2) return launch_replay<2>(ctx, rp, caps, start, sval, n, d_key, d_plen, d_slen, d_ctr);
    if (E <= 4) return launch_replay<4>(ctx, rp, caps, start, sval, n, d_key, d_plen, d_slen, d_ctr);
    if (E <= 8) return launch_replay<8>(ctx, rp, caps, start, sval, n, d_key, d_plen, d_slen, d_ctr);
    if (E <= 16) return launch_replay<16>(ctx, rp, caps, start, sval, n, d_key, d_plen, d_slen, d_ctr);
    return launch_replay<32>(ctx, rp, caps, start, sval, n, d_key, d_plen, d_slen, d_ctr);
}

extern "C" int cr_replay_export_state(cr_ctx *ctx, const cr_replay *rp, uint32_t rep, uint32_t r,
                                      uint64_t *keys_out, uint32_t *fill_out)
{
    if (!ctx || !rp || !keys_out || !fill_out) return CR_EINVAL;
    if (rep >= rp->n_rep || r >= rp->R) return cr_fail(ctx, CR_EINVAL, "export_state: bad stream");
    const uint64_t s = (uint64_t)rep * rp->R + r;
    uint32_t fill = 0;
    CR_CUDA(ctx, cudaMemcpyAsync(&fill, rp->d_fill + s, sizeof(uint32_t), cudaMemcpyDeviceToHost, ctx->stream));
    CR_TRY(cr_sync(ctx));
    if (fill)
        CR_CUDA(ctx, cudaMemcpyAsync(keys_out, rp->d_keys + s * rp->cmax, fill * sizeof(uint64_t),
                                     cudaMemcpyDeviceToHost, ctx->stream));
    *fill_out = fill;
    return cr_sync(ctx);
}
