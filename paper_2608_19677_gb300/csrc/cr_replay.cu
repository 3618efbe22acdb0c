// a8, a9: shadow replay (cr_shadow_replay).
//
//   partition  one stable counting sort per replica by destination: each
//              (replica, destination) stream's (key, prefix, suffix) records
//              in arrival order
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

struct rec16 {
    unsigned long long key;
    uint32_t P, S;
};

// ---- partition: one stable counting sort per replica, by destination --------
// Tiles of 2048 requests.  k_part_count writes each tile's destination counts
// at [(replica * R + r) * ntiles + tile]; one exclusive scan of that array
// gives every (stream, tile) its output base, in stream-major order.
// k_part_scatter ranks each tile's requests stably and writes their
// (key, prefix, suffix) records straight to their place in stream order.
constexpr int kPartBlock = 256;
constexpr int kPartWarps = kPartBlock / 32;
constexpr int kPartTile = kPartBlock * 8;

__global__ void __launch_bounds__(kPartBlock) k_part_count(const uint16_t *__restrict__ dest, unsigned long long n,
                                                           uint32_t R, uint32_t ntiles, uint32_t *__restrict__ cnt,
                                                           uint32_t *status)
{
    extern __shared__ uint32_t hist[];
    const uint32_t rep = blockIdx.y, tile = blockIdx.x, lane = cr_lane();
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) hist[r] = 0;
    __syncthreads();
    const uint16_t *D = dest + (unsigned long long)rep * n;
    const unsigned long long base = (unsigned long long)tile * kPartTile;
    bool bad = false;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const unsigned long long i = base + (unsigned long long)j * kPartBlock + threadIdx.x;
        uint32_t d = i < n ? D[i] : 0xffffu;
        if (i < n && d >= R) {
            bad = true;
            d = 0xffffu;  // skipped: reported through the status word
        }
        const uint32_t peers = __match_any_sync(0xffffffffu, d);
        if (d != 0xffffu && (peers & ((1u << lane) - 1u)) == 0) atomicAdd(&hist[d], (uint32_t)__popc(peers));
    }
    __syncthreads();
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock)
        cnt[((unsigned long long)rep * R + r) * ntiles + tile] = hist[r];
    if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(status, CR_FLAG_BADDEST);
}

// start[s] = first record of stream s = (replica, r); start[ns] = number of records.
__global__ void k_part_starts(const uint32_t *__restrict__ off, uint32_t ns, uint32_t ntiles,
                              const uint32_t *__restrict__ total, uint32_t *__restrict__ start)
{
    for (uint32_t s = blockIdx.x * blockDim.x + threadIdx.x; s <= ns; s += gridDim.x * blockDim.x)
        start[s] = s < ns ? off[(unsigned long long)s * ntiles] : *total;
}

// Warp w ranks items [256w, 256w+256) of the tile in 8 rounds against
// warp-private counters (u16, destination-major); one pass over the
// destinations turns them into per-warp offsets.
__global__ void __launch_bounds__(kPartBlock) k_part_scatter(const uint16_t *__restrict__ dest, unsigned long long n,
                                                             uint32_t R, uint32_t ntiles,
                                                             const uint32_t *__restrict__ off,
                                                             const unsigned long long *__restrict__ keys,
                                                             const uint32_t *__restrict__ plen,
                                                             const uint32_t *__restrict__ slen,
                                                             rec16 *__restrict__ rec)
{
    extern __shared__ uint16_t wc[];  // [R][8]
    const uint32_t rep = blockIdx.y, tile = blockIdx.x, lane = cr_lane(), warp = threadIdx.x >> 5;
    const uint32_t lt = (1u << lane) - 1u;
    uint4 *wc4 = reinterpret_cast<uint4 *>(wc);
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) wc4[r] = make_uint4(0, 0, 0, 0);
    __syncthreads();
    const uint16_t *D = dest + (unsigned long long)rep * n;
    const unsigned long long base = (unsigned long long)tile * kPartTile + (unsigned long long)warp * 256;
    uint32_t dig[8], rank[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const unsigned long long i = base + (unsigned long long)j * 32 + lane;
        uint32_t d = i < n ? D[i] : 0xffffu;
        if (d >= R) d = 0xffffu;
        const uint32_t peers = __match_any_sync(0xffffffffu, d);
        const uint32_t before = d != 0xffffu ? wc[d * kPartWarps + warp] : 0u;
        rank[j] = before + __popc(peers & lt);
        dig[j] = d;
        __syncwarp();
        if (d != 0xffffu && (peers & lt) == 0) wc[d * kPartWarps + warp] = (uint16_t)(before + __popc(peers));
        __syncwarp();
    }
    __syncthreads();
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) {  // exclusive prefix over the 8 warps
        uint4 v = wc4[r];
        uint16_t c[8];
        memcpy(c, &v, 16);
        uint16_t run = 0;
#pragma unroll
        for (int w = 0; w < kPartWarps; ++w) {
            const uint16_t x = c[w];
            c[w] = run;
            run = (uint16_t)(run + x);
        }
        memcpy(&v, c, 16);
        wc4[r] = v;
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        if (dig[j] == 0xffffu) continue;
        const unsigned long long i = base + (unsigned long long)j * 32 + lane;
        const uint32_t pos = off[((unsigned long long)rep * R + dig[j]) * ntiles + tile] +
                             wc[dig[j] * kPartWarps + warp] + rank[j];
        rec16 rr;
        rr.key = keys[i];
        rr.P = plen[i];
        rr.S = slen[i];
        rec[pos] = rr;
    }
}

// Chunks per stream (an empty stream still gets one work item that carries its state over).
__global__ void k_chunk_counts(const uint32_t *__restrict__ start, uint32_t ns, uint32_t CL, uint32_t *__restrict__ nch)
{
    for (uint32_t s = blockIdx.x * blockDim.x + threadIdx.x; s < ns; s += gridDim.x * blockDim.x) {
        const uint32_t len = start[s + 1] - start[s];
        nch[s] = len ? (len + CL - 1) / CL : 1u;
    }
}

struct replay_state {
    const unsigned long long *keys_in;  // [stream][cmax], most recent first
    const uint32_t *fill_in;
    unsigned long long *keys_out;
    uint32_t *fill_out;
};

// One warp per (stream, chunk).  The LRU state at the chunk's first request is
// rebuilt by walking the stream backwards (and then the state carried in from
// the previous call) collecting distinct keys, most recent first, until cmax
// are found: those are exactly the resident entries of an LRU of capacity
// cmax at that point.  The chunk is then simulated forwards.
template <int E, int NC>  // NC: capacities counted (a compile-time bound on caps.n_caps)
__global__ void __launch_bounds__(E == 1 ? 256 : 128, E == 1 ? 4 : 1)
k_lru_chunks(const replay_caps caps, uint32_t cmax, uint32_t R, uint32_t ns, uint32_t CL,
             const uint32_t *__restrict__ start, const uint32_t *__restrict__ coff, const uint32_t *__restrict__ total,
             const rec16 *__restrict__ rec, const replay_state st, unsigned long long *__restrict__ ctr)
{
    extern __shared__ unsigned long long sm[];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
    const uint32_t slots = 32u * E;
    unsigned long long *sk = sm + (size_t)warp * slots;
    uint32_t *ss = reinterpret_cast<uint32_t *>(sm + (size_t)wpb * slots) + (size_t)warp * slots;
    const uint32_t w = blockIdx.x * wpb + warp;
    if (w >= *total) return;
    // stream of this work item: the last s with coff[s] <= w
    uint32_t lo = 0, hi = ns;
    while (hi - lo > 1) {
        uint32_t mid = (lo + hi) >> 1;
        if (coff[mid] <= w)
            lo = mid;
        else
            hi = mid;
    }
    const uint32_t s = lo, ci = w - coff[s];
    const uint32_t b = start[s], e = start[s + 1];
    const uint32_t p0 = b + ci * CL;
    const uint32_t p1 = (e - p0) < CL ? e : p0 + CL;
    const uint32_t rep = s / R, r = s % R;
    const uint32_t fill_in = st.fill_in[s];
    const unsigned long long *kin = st.keys_in + (unsigned long long)s * cmax;
    const uint32_t lt = (1u << lane) - 1u;

    if (b == e) {  // nothing routed here: carry the state over unchanged
        unsigned long long *kout = st.keys_out + (unsigned long long)s * cmax;
        for (uint32_t q = lane; q < fill_in; q += 32) kout[q] = kin[q];
        if (lane == 0) st.fill_out[s] = fill_in;
        return;
    }

    // ---- state at p0 -------------------------------------------------------
    uint32_t fill = 0;
    if (ci == 0) {
        for (uint32_t q = lane; q < fill_in; q += 32) sk[q] = kin[q];
        fill = fill_in;
    } else {
        const uint32_t back = p0 - b;            // stream positions before the chunk
        const uint32_t vtot = back + fill_in;    // then the carried-in state
        for (uint32_t v0 = 0; v0 < vtot && fill < cmax; v0 += 32) {
            const uint32_t v = v0 + lane;
            const bool valid = v < vtot;
            unsigned long long key = 0;
            if (valid) key = v < back ? rec[p0 - 1 - v].key : kin[v - back];
            const uint32_t peers = __match_any_sync(0xffffffffu, key);
            bool fresh = valid && (peers & lt) == 0;
            for (uint32_t q = 0; q < fill; ++q)
                if (sk[q] == key) fresh = false;
            const uint32_t bal = __ballot_sync(0xffffffffu, fresh);
            const uint32_t rank = __popc(bal & lt);
            __syncwarp();
            if (fresh && fill + rank < cmax) sk[fill + rank] = key;
            fill = min(cmax, fill + (uint32_t)__popc(bal));
            __syncwarp();
        }
    }
    for (uint32_t q = lane; q < fill; q += 32) ss[q] = fill - q;
    __syncwarp();
    uint32_t clock = fill;

    // register copy of the state when it fits one entry per lane
    unsigned long long ek = 0;
    uint32_t es = 0;
    if (E == 1 && lane < fill) {
        ek = sk[lane];
        es = ss[lane];
    }

    unsigned long long my_req = 0, my_prompt = 0;
    unsigned long long my_hit[NC], my_tok[NC];
#pragma unroll
    for (int c = 0; c < NC; ++c) my_hit[c] = my_tok[c] = 0;

    for (uint32_t t0 = p0; t0 < p1; t0 += 32) {
        rec16 mine_rec = {0ull, 0u, 0u};
        if (t0 + lane < p1) {
            mine_rec = rec[t0 + lane];
            my_req += 1;
            my_prompt += (unsigned long long)mine_rec.P + mine_rec.S;
        }
        const uint32_t cnt = (p1 - t0) < 32u ? (p1 - t0) : 32u;
        uint32_t my_depth = 0xffffffffu;  // lanes without a request never count a hit
        for (uint32_t j = 0; j < cnt; ++j) {
            const unsigned long long key = __shfl_sync(0xffffffffu, mine_rec.key, j);
            ++clock;
            uint32_t depth = 0xffffffffu;
            if (E == 1) {
                const bool have = lane < fill;
                const uint32_t hb = __ballot_sync(0xffffffffu, have && ek == key);
                if (hb) {
                    const uint32_t hl = __ffs(hb) - 1;
                    const uint32_t s_hit = __shfl_sync(0xffffffffu, es, hl);
                    depth = 1u + __popc(__ballot_sync(0xffffffffu, have && es > s_hit));
                    if (lane == hl) es = clock;
                } else if (fill < cmax) {
                    if (lane == fill) {
                        ek = key;
                        es = clock;
                    }
                    ++fill;
                } else {
                    const uint32_t mn = __reduce_min_sync(0xffffffffu, have ? es : 0xffffffffu);
                    const uint32_t vl = __ffs(__ballot_sync(0xffffffffu, have && es == mn)) - 1;
                    if (lane == vl) {
                        ek = key;
                        es = clock;
                    }
                }
            } else {
                int mine = -1;
#pragma unroll
                for (int x = 0; x < E; ++x) {
                    const uint32_t idx = (uint32_t)x * 32u + lane;
                    if (idx < fill && sk[idx] == key) mine = (int)idx;
                }
                const uint32_t hb = __ballot_sync(0xffffffffu, mine >= 0);
                if (hb) {
                    const uint32_t hl = __ffs(hb) - 1;
                    const uint32_t hs = (uint32_t)__shfl_sync(0xffffffffu, mine, hl);
                    const uint32_t s_hit = ss[hs];
                    uint32_t newer = 0;
#pragma unroll
                    for (int x = 0; x < E; ++x) {
                        const uint32_t idx = (uint32_t)x * 32u + lane;
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
                    uint32_t lmin = 0xffffffffu, lidx = 0;
#pragma unroll
                    for (int x = 0; x < E; ++x) {
                        const uint32_t idx = (uint32_t)x * 32u + lane;
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
            }
            // the lane that loaded request j keeps its depth
            if (lane == j) my_depth = depth;
        }
        // counters of the group, each lane for its own request
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            if (c < (int)caps.n_caps && my_depth <= caps.cap[c]) {
                my_hit[c] += 1;
                my_tok[c] += mine_rec.P;
            }
        }
    }

    // ---- counters -------------------------------------------------------------
    my_req = cr_warp_sum_u64(my_req);
    my_prompt = cr_warp_sum_u64(my_prompt);
#pragma unroll
    for (int c = 0; c < NC; ++c) {
        if (c < (int)caps.n_caps) {
            const unsigned long long h = cr_warp_sum_u64(my_hit[c]);
            const unsigned long long tk = cr_warp_sum_u64(my_tok[c]);
            if (lane == 0) {
                unsigned long long *C = ctr + (((unsigned long long)rep * caps.n_caps + c) * R + r) * CR_CTR_FIELDS;
                atomicAdd(&C[0], my_req);
                if (h) atomicAdd(&C[1], h);
                if (tk) atomicAdd(&C[2], tk);
                atomicAdd(&C[3], my_prompt);
                atomicAdd(&C[4], my_prompt - tk);
            }
        }
    }

    // ---- the stream's last chunk hands the state to the next call ---------------
    if (p1 == e) {
        unsigned long long *kout = st.keys_out + (unsigned long long)s * cmax;
        if (E == 1) {
            uint32_t rank = 0;
            for (uint32_t q = 0; q < 32; ++q) {
                const uint32_t sq = __shfl_sync(0xffffffffu, es, q);
                if (q < fill && sq > es) ++rank;
            }
            if (lane < fill) kout[rank] = ek;
        } else {
#pragma unroll
            for (int x = 0; x < E; ++x) {
                const uint32_t idx = (uint32_t)x * 32u + lane;
                if (idx < fill) {
                    const uint32_t my = ss[idx];
                    uint32_t rank = 0;
                    for (uint32_t f = 0; f < fill; ++f) rank += (ss[f] > my) ? 1u : 0u;
                    kout[rank] = sk[idx];
                }
            }
        }
        if (lane == 0) st.fill_out[s] = fill;
    }
}

// ---- capacities above 32: linked-list LRU with a hash index -----------------
// One warp per (stream, chunk); lane 0 runs the simulator, the warp helps to
// load and rebuild states.  Shared memory per warp: keys, prev/next links in
// recency order (most recent at the head), a segment id per entry and an
// open-addressing index key -> entry.  With the distinct capacities sorted
// c_0 < c_1 < ... < c_{m-1} = cmax, segment j holds recency positions
// (c_{j-1}, c_j] and B[j] is the entry at position c_j: an access at segment
// s hits every capacity c_j with j >= s (LRU inclusion).  Moving an entry to
// the front shifts the last entry of each earlier segment into the next one,
// so every access costs O(m) pointer updates, independent of cmax.
struct list_caps {
    uint32_t m;                 // distinct capacities
    uint32_t c[CR_MAX_CAPS];    // ascending
    uint32_t out[CR_MAX_CAPS];  // counter index (position in the caller's caps) of c[j]
    uint32_t n_out;             // caller's capacity count
    uint32_t seg_of[CR_MAX_CAPS];  // for each caller index: its segment j
};

constexpr uint16_t kNil = 0xffffu;

struct lru_list {
    unsigned long long *key;
    uint16_t *prev, *next;
    uint8_t *seg;
    uint32_t *tab;  // entry + 1; 0 = empty
    uint32_t mask;
    int tbits;
};

__device__ __forceinline__ uint32_t home_slot(unsigned long long key, int tbits) { return (uint32_t)(key >> (64 - tbits)); }

__device__ __forceinline__ int list_find(const lru_list &L, unsigned long long key)
{
    uint32_t s = home_slot(key, L.tbits);
    for (;;) {
        const uint32_t e = L.tab[s];
        if (e == 0) return -1;
        if (L.key[e - 1] == key) return (int)(e - 1);
        s = (s + 1) & L.mask;
    }
}

__device__ __forceinline__ void list_insert_index(const lru_list &L, unsigned long long key, uint32_t node)
{
    uint32_t s = home_slot(key, L.tbits);
    while (atomicCAS(&L.tab[s], 0u, node + 1) != 0u) s = (s + 1) & L.mask;
}

// Remove the index entry of `node` (key `key`): backward-shift deletion for linear probing.
__device__ __forceinline__ void list_erase_index(const lru_list &L, unsigned long long key, uint32_t node)
{
    uint32_t i = home_slot(key, L.tbits);
    while (L.tab[i] != node + 1) i = (i + 1) & L.mask;
    uint32_t j = i;
    for (;;) {
        j = (j + 1) & L.mask;
        const uint32_t e = L.tab[j];
        if (e == 0) break;
        const uint32_t k = home_slot(L.key[e - 1], L.tbits);
        const bool stays = (i <= j) ? (i < k && k <= j) : (i < k || k <= j);
        if (stays) continue;
        L.tab[i] = e;
        i = j;
    }
    L.tab[i] = 0;
}

template <int NC>
__global__ void __launch_bounds__(128)
k_lru_list(const list_caps lc, uint32_t cmax, uint32_t R, uint32_t ns, uint32_t CL, int tbits,
           const uint32_t *__restrict__ start, const uint32_t *__restrict__ coff, const uint32_t *__restrict__ total,
           const rec16 *__restrict__ rec, const replay_state st, unsigned long long *__restrict__ ctr)
{
    extern __shared__ unsigned long long smw[];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
    const uint32_t tsz = 1u << tbits;
    // per-warp region, 8-byte aligned pieces
    const size_t per_warp = (size_t)cmax * 8 + (size_t)tsz * 4 + (((size_t)cmax * 5 + 7) & ~(size_t)7);
    unsigned char *base = reinterpret_cast<unsigned char *>(smw) + per_warp * warp;
    lru_list L;
    L.key = reinterpret_cast<unsigned long long *>(base);
    L.tab = reinterpret_cast<uint32_t *>(base + (size_t)cmax * 8);
    L.prev = reinterpret_cast<uint16_t *>(base + (size_t)cmax * 8 + (size_t)tsz * 4);
    L.next = L.prev + cmax;
    L.seg = reinterpret_cast<uint8_t *>(L.next + cmax);
    L.mask = tsz - 1;
    L.tbits = tbits;

    const uint32_t w = blockIdx.x * wpb + warp;
    if (w >= *total) return;
    uint32_t lo = 0, hi = ns;
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (coff[mid] <= w)
            lo = mid;
        else
            hi = mid;
    }
    const uint32_t s = lo, ci = w - coff[s];
    const uint32_t b = start[s], e = start[s + 1];
    const uint32_t p0 = b + ci * CL;
    const uint32_t p1 = (e - p0) < CL ? e : p0 + CL;
    const uint32_t rep = s / R, r = s % R;
    const uint32_t fill_in = st.fill_in[s];
    const unsigned long long *kin = st.keys_in + (unsigned long long)s * cmax;
    const uint32_t lt = (1u << lane) - 1u;

    if (b == e) {  // nothing routed here: carry the state over unchanged
        unsigned long long *kout = st.keys_out + (unsigned long long)s * cmax;
        for (uint32_t q = lane; q < fill_in; q += 32) kout[q] = kin[q];
        if (lane == 0) st.fill_out[s] = fill_in;
        return;
    }

    // ---- state at p0, as keys in recency order in L.key[0..fill) ---------------
    for (uint32_t x = lane; x < tsz; x += 32) L.tab[x] = 0;
    __syncwarp();
    uint32_t fill = 0;
    if (ci == 0) {
        for (uint32_t q = lane; q < fill_in; q += 32) {
            L.key[q] = kin[q];
            list_insert_index(L, kin[q], q);
        }
        fill = fill_in;
    } else {
        const uint32_t back = p0 - b;
        const uint32_t vtot = back + fill_in;
        for (uint32_t v0 = 0; v0 < vtot && fill < cmax; v0 += 32) {
            const uint32_t v = v0 + lane;
            const bool valid = v < vtot;
            unsigned long long key = 0;
            if (valid) key = v < back ? rec[p0 - 1 - v].key : kin[v - back];
            const uint32_t peers = __match_any_sync(0xffffffffu, key);
            const bool fresh = valid && (peers & lt) == 0 && list_find(L, key) < 0;
            const uint32_t bal = __ballot_sync(0xffffffffu, fresh);
            const uint32_t rank = __popc(bal & lt);
            __syncwarp();
            if (fresh && fill + rank < cmax) {
                L.key[fill + rank] = key;
                list_insert_index(L, key, fill + rank);
            }
            fill = min(cmax, fill + (uint32_t)__popc(bal));
            __syncwarp();
        }
    }
    // links and segments of the recency order 0..fill-1
    for (uint32_t q = lane; q < fill; q += 32) {
        L.prev[q] = q == 0 ? kNil : (uint16_t)(q - 1);
        L.next[q] = q + 1 == fill ? kNil : (uint16_t)(q + 1);
        uint32_t sg = 0;
        while (sg + 1 < lc.m && q + 1 > lc.c[sg]) ++sg;
        L.seg[q] = (uint8_t)sg;
    }
    __syncwarp();

    unsigned long long my_req = 0, my_prompt = 0;
    unsigned long long hitc[NC], hitt[NC];
#pragma unroll
    for (int j = 0; j < NC; ++j) hitc[j] = hitt[j] = 0;
    // simulator registers (meaningful in lane 0)
    uint32_t head = fill ? 0u : kNil, tail = fill ? fill - 1 : kNil;
    uint32_t B[NC];
#pragma unroll
    for (int j = 0; j < NC; ++j) B[j] = (j + 1 < (int)lc.m && fill >= lc.c[j]) ? lc.c[j] - 1 : kNil;

    for (uint32_t t0 = p0; t0 < p1; t0 += 32) {
        // the warp stages 32 requests; lane 0 simulates them in order
        rec16 mine = {0ull, 0u, 0u};
        if (t0 + lane < p1) {
            mine = rec[t0 + lane];
            my_req += 1;
            my_prompt += (unsigned long long)mine.P + mine.S;
        }
        const uint32_t cnt = (p1 - t0) < 32u ? (p1 - t0) : 32u;
        for (uint32_t jq = 0; jq < cnt; ++jq) {
            const unsigned long long key = __shfl_sync(0xffffffffu, mine.key, jq);
            const uint32_t P = __shfl_sync(0xffffffffu, mine.P, jq);
            if (lane == 0) {
                const int n = list_find(L, key);
                if (n >= 0) {
                    const uint32_t sg = L.seg[n];
#pragma unroll
                    for (int j = 0; j < NC; ++j) {
                        if (j < (int)lc.m && (uint32_t)j >= sg) {
                            hitc[j] += 1;
                            hitt[j] += P;
                        }
                    }
                    if ((uint32_t)n != head) {
                        const uint32_t pn = L.prev[n];
#pragma unroll
                        for (int j = 0; j < NC; ++j) {
                            if (j + 1 < (int)lc.m) {
                                if ((uint32_t)j < sg) {
                                    L.seg[B[j]] = (uint8_t)(j + 1);
                                    B[j] = lc.c[j] == 1 ? (uint32_t)n : L.prev[B[j]];
                                } else if ((uint32_t)j == sg && B[j] == (uint32_t)n) {
                                    B[j] = pn;
                                }
                            }
                        }
                        // unlink n, push it to the front
                        const uint32_t nx = L.next[n];
                        L.next[pn] = (uint16_t)nx;
                        if (nx != kNil)
                            L.prev[nx] = (uint16_t)pn;
                        else
                            tail = pn;
                        L.prev[n] = kNil;
                        L.next[n] = (uint16_t)head;
                        L.prev[head] = (uint16_t)n;
                        head = (uint32_t)n;
                        L.seg[n] = 0;
                    }
                } else {
                    uint32_t node;
                    const uint32_t old_fill = fill;
                    // every resident entry moves back one position
#pragma unroll
                    for (int j = 0; j < NC; ++j) {
                        if (j + 1 < (int)lc.m && B[j] != kNil) {
                            L.seg[B[j]] = (uint8_t)(j + 1);
                            B[j] = L.prev[B[j]];  // kNil when c_j == 1: the new entry, set below
                        }
                    }
                    if (fill == cmax) {
                        node = tail;
                        list_erase_index(L, L.key[node], node);
                        tail = L.prev[node];
                        if (tail != kNil) L.next[tail] = kNil;
                        if (head == node) head = kNil;
                    } else {
                        node = fill++;
                    }
                    L.key[node] = key;
                    L.seg[node] = 0;
                    L.prev[node] = kNil;
                    L.next[node] = (uint16_t)head;
                    if (head != kNil) L.prev[head] = (uint16_t)node;
                    head = node;
                    if (tail == kNil) tail = node;
                    list_insert_index(L, key, node);
#pragma unroll
                    for (int j = 0; j < NC; ++j) {
                        if (j + 1 < (int)lc.m) {
                            if (B[j] == kNil && old_fill >= lc.c[j]) B[j] = node;    // c_j == 1
                            if (old_fill < lc.c[j] && fill == lc.c[j]) B[j] = tail;  // boundary now defined
                        }
                    }
                }
            }
            __syncwarp();
        }
    }

    // ---- counters -------------------------------------------------------------
    my_req = cr_warp_sum_u64(my_req);
    my_prompt = cr_warp_sum_u64(my_prompt);
    if (lane == 0) {
        // hand the state to the next call, most recent first
        if (p1 == e) {
            unsigned long long *kout = st.keys_out + (unsigned long long)s * cmax;
            uint32_t q = 0;
            for (uint32_t x = head; x != kNil; x = L.next[x]) kout[q++] = L.key[x];
            st.fill_out[s] = fill;
        }
        for (uint32_t oi = 0; oi < lc.n_out; ++oi) {
            const uint32_t j = lc.seg_of[oi];
            unsigned long long h = 0, tk = 0;
#pragma unroll
            for (int jj = 0; jj < NC; ++jj)
                if ((uint32_t)jj == j) {
                    h = hitc[jj];
                    tk = hitt[jj];
                }
            unsigned long long *C = ctr + (((unsigned long long)rep * lc.n_out + oi) * R + r) * CR_CTR_FIELDS;
            atomicAdd(&C[0], my_req);
            if (h) atomicAdd(&C[1], h);
            if (tk) atomicAdd(&C[2], tk);
            atomicAdd(&C[3], my_prompt);
            atomicAdd(&C[4], my_prompt - tk);
        }
    }
}

template <int E, int NC>
int launch_replay_nc(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                     const uint32_t *coff, const uint32_t *total, uint64_t m, const rec16 *rec, uint64_t *d_ctr)
{
    const uint32_t wpb = E == 1 ? 8 : 4;
    const size_t smem = (size_t)wpb * 32 * E * (sizeof(unsigned long long) + sizeof(uint32_t));
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_chunks<E, NC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)smem));
    const uint32_t ns = rp->n_rep * rp->R;
    const uint64_t items = (uint64_t)ns + (m + CL - 1) / CL;  // upper bound on work items
    replay_state st;
    st.keys_in = rp->d_keys[rp->cur];
    st.fill_in = rp->d_fill[rp->cur];
    st.keys_out = rp->d_keys[rp->cur ^ 1];
    st.fill_out = rp->d_fill[rp->cur ^ 1];
    CR_LAUNCH(ctx, (k_lru_chunks<E, NC>), (unsigned int)((items + wpb - 1) / wpb), wpb * 32, smem, caps, rp->cmax,
              rp->R, ns, CL, start, coff, total, rec, st, (unsigned long long *)d_ctr);
    rp->cur ^= 1;
    return CR_OK;
}

template <int E>
int launch_replay(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                  const uint32_t *coff, const uint32_t *total, uint64_t m, const rec16 *rec, uint64_t *d_ctr)
{
    if (caps.n_caps == 1) return launch_replay_nc<E, 1>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
    if (caps.n_caps <= 3) return launch_replay_nc<E, 3>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
    return launch_replay_nc<E, CR_MAX_CAPS>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
}

template <int NC>
int launch_list_nc(cr_ctx *ctx, cr_replay *rp, const list_caps &lc, uint32_t CL, int tbits, const uint32_t *start,
                   const uint32_t *coff, const uint32_t *total, uint64_t m, const rec16 *rec, uint64_t *d_ctr)
{
    const uint32_t cmax = rp->cmax, tsz = 1u << tbits;
    const size_t per_warp = (size_t)cmax * 8 + (size_t)tsz * 4 + (((size_t)cmax * 5 + 7) & ~(size_t)7);
    uint32_t wpb = 4;
    while (wpb > 1 && per_warp * wpb > 200 * 1024) wpb >>= 1;
    const size_t smem = per_warp * wpb;
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_list<NC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    const uint32_t ns = rp->n_rep * rp->R;
    const uint64_t items = (uint64_t)ns + (m + CL - 1) / CL;
    replay_state st;
    st.keys_in = rp->d_keys[rp->cur];
    st.fill_in = rp->d_fill[rp->cur];
    st.keys_out = rp->d_keys[rp->cur ^ 1];
    st.fill_out = rp->d_fill[rp->cur ^ 1];
    CR_LAUNCH(ctx, k_lru_list<NC>, (unsigned int)((items + wpb - 1) / wpb), wpb * 32, smem, lc, cmax, rp->R, ns, CL,
              tbits, start, coff, total, rec, st, (unsigned long long *)d_ctr);
    rp->cur ^= 1;
    return CR_OK;
}

int launch_list(cr_ctx *ctx, cr_replay *rp, uint32_t CL, const uint32_t *start, const uint32_t *coff,
                const uint32_t *total, uint64_t m, const rec16 *rec, uint64_t *d_ctr)
{
    list_caps lc;
    memset(&lc, 0, sizeof(lc));
    uint32_t sorted[CR_MAX_CAPS];
    uint32_t ns_ = 0;
    for (uint32_t i = 0; i < rp->n_caps; ++i) {
        bool dup = false;
        for (uint32_t j = 0; j < ns_; ++j) dup |= sorted[j] == rp->caps[i];
        if (!dup) sorted[ns_++] = rp->caps[i];
    }
    for (uint32_t i = 1; i < ns_; ++i)
        for (uint32_t j = i; j > 0 && sorted[j - 1] > sorted[j]; --j) {
            uint32_t t = sorted[j];
            sorted[j] = sorted[j - 1];
            sorted[j - 1] = t;
        }
    lc.m = ns_;
    for (uint32_t j = 0; j < ns_; ++j) lc.c[j] = sorted[j];
    lc.n_out = rp->n_caps;
    for (uint32_t i = 0; i < rp->n_caps; ++i)
        for (uint32_t j = 0; j < ns_; ++j)
            if (sorted[j] == rp->caps[i]) lc.seg_of[i] = j;
    int tbits = 0;
    while ((1u << tbits) < 2 * rp->cmax) ++tbits;
    if (lc.m <= 1) return launch_list_nc<1>(ctx, rp, lc, CL, tbits, start, coff, total, m, rec, d_ctr);
    if (lc.m <= 3) return launch_list_nc<3>(ctx, rp, lc, CL, tbits, start, coff, total, m, rec, d_ctr);
    return launch_list_nc<CR_MAX_CAPS>(ctx, rp, lc, CL, tbits, start, coff, total, m, rec, d_ctr);
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
    for (int b = 0; b < 2; ++b) {
        if (cudaMalloc(&rp->d_keys[b], rp->n_streams * cmax * sizeof(unsigned long long)) != cudaSuccess ||
            cudaMalloc(&rp->d_fill[b], rp->n_streams * sizeof(uint32_t)) != cudaSuccess) {
            cudaGetLastError();
            for (int x = 0; x < 2; ++x) {
                if (rp->d_keys[x]) cudaFree(rp->d_keys[x]);
                if (rp->d_fill[x]) cudaFree(rp->d_fill[x]);
            }
            free(rp);
            return cr_fail(ctx, CR_ENOMEM, "replay: cannot allocate state");
        }
    }
    *out = rp;
    return cr_replay_reset(ctx, rp);
}

extern "C" int cr_replay_reset(cr_ctx *ctx, cr_replay *rp)
{
    if (!ctx || !rp) return CR_EINVAL;
    for (int b = 0; b < 2; ++b)
        CR_CUDA(ctx, cudaMemsetAsync(rp->d_fill[b], 0, rp->n_streams * sizeof(uint32_t), ctx->stream));
    return CR_OK;
}

extern "C" int cr_replay_destroy(cr_ctx *ctx, cr_replay *rp)
{
    if (!rp) return CR_OK;
    if (ctx) cudaStreamSynchronize(ctx->stream);
    for (int b = 0; b < 2; ++b) {
        cudaFree(rp->d_keys[b]);
        cudaFree(rp->d_fill[b]);
    }
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
    const uint32_t R = rp->R, ns = (uint32_t)rp->n_streams;
    const uint32_t ntiles = (uint32_t)((n + kPartTile - 1) / kPartTile);
    const uint64_t ncnt = (uint64_t)ns * ntiles;
    if (ncnt >= 0xffffffffull) return cr_fail(ctx, CR_EINVAL, "cr_shadow_replay: too many (stream, tile) pairs");
    void *pk, *ps, *prec, *pch;
    CR_TRY(cr_scratch(ctx, SCR_REPLAY_IDX, (ncnt + 2) * sizeof(uint32_t), &pk));
    CR_TRY(cr_scratch(ctx, SCR_REPLAY_START, ((size_t)ns + 1) * sizeof(uint32_t), &ps));
    CR_TRY(cr_scratch(ctx, SCR_REPLAY_REC, m * sizeof(rec16), &prec));
    CR_TRY(cr_scratch(ctx, SCR_REPLAY_CHUNK, ((size_t)ns + 2) * sizeof(uint32_t), &pch));
    uint32_t *cnt = (uint32_t *)pk, *nrec = cnt + ncnt, *start = (uint32_t *)ps;
    rec16 *rec = (rec16 *)prec;
    uint32_t *coff = (uint32_t *)pch, *total = coff + ns;
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    const dim3 pgrid(ntiles, rp->n_rep);
    const size_t csmem = (size_t)R * sizeof(uint32_t), ssmem = (size_t)R * kPartWarps * sizeof(uint16_t);
    if (csmem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_part_count, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)csmem));
    if (ssmem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_part_scatter, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ssmem));
    CR_LAUNCH(ctx, k_part_count, pgrid, kPartBlock, csmem, d_dest, (unsigned long long)n, R, ntiles, cnt,
              ctx->d_status);
    CR_TRY(cr_scan_u32(ctx, cnt, cnt, ncnt, nrec));
    CR_LAUNCH(ctx, k_part_starts, cr_blocks((uint64_t)ns + 1, 256, gcap), 256, 0, (const uint32_t *)cnt, ns, ntiles,
              (const uint32_t *)nrec, start);
    CR_LAUNCH(ctx, k_part_scatter, pgrid, kPartBlock, ssmem, d_dest, (unsigned long long)n, R, ntiles,
              (const uint32_t *)cnt, (const unsigned long long *)d_key, d_plen, d_slen, rec);
    replay_caps caps;
    caps.n_caps = rp->n_caps;
    for (uint32_t c = 0; c < CR_MAX_CAPS; ++c) caps.cap[c] = c < rp->n_caps ? rp->caps[c] : 0;
    // chunk length: long enough that rebuilding an LRU state of cmax entries is amortised
    const uint32_t CL = rp->cmax * 16u > 256u ? rp->cmax * 16u : 256u;
    CR_LAUNCH(ctx, k_chunk_counts, cr_blocks(ns, 256, gcap), 256, 0, (const uint32_t *)start, ns, CL, coff);
    CR_TRY(cr_scan_u32(ctx, coff, coff, ns, total));
    const uint32_t E = (rp->cmax + 31) / 32;
    // capacities up to 32: one entry per lane in registers; above: linked list + hash index
    if (E > 1) return launch_list(ctx, rp, CL, start, coff, total, m, rec, d_ctr);
    return launch_replay<1>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
}

extern "C" int cr_replay_export_state(cr_ctx *ctx, const cr_replay *rp, uint32_t rep, uint32_t r,
                                      uint64_t *keys_out, uint32_t *fill_out)
{
    if (!ctx || !rp || !keys_out || !fill_out) return CR_EINVAL;
    if (rep >= rp->n_rep || r >= rp->R) return cr_fail(ctx, CR_EINVAL, "export_state: bad stream");
    const uint64_t s = (uint64_t)rep * rp->R + r;
    uint32_t fill = 0;
    CR_CUDA(ctx, cudaMemcpyAsync(&fill, rp->d_fill[rp->cur] + s, sizeof(uint32_t), cudaMemcpyDeviceToHost,
                                 ctx->stream));
    CR_TRY(cr_sync(ctx));
    if (fill)
        CR_CUDA(ctx, cudaMemcpyAsync(keys_out, rp->d_keys[rp->cur] + s * rp->cmax, fill * sizeof(uint64_t),
                                     cudaMemcpyDeviceToHost, ctx->stream));
    *fill_out = fill;
    return cr_sync(ctx);
}
