// a8, a9: shadow replay (cr_shadow_replay).
//
//   partition  one stable counting sort per replica by destination: each
//              (replica, destination) stream's (key, prefix, suffix) records
//              in arrival order
//   replay     one warp per (stream, chunk); the stream's LRU at the LARGEST
//              capacity lives in shared memory as keys in recency order with
//              a hash index, and 32 requests are simulated per step, one per
//              lane.  A request's depth (its LRU stack distance) decides the
//              hit at every smaller capacity at once, because LRU caches are
//              nested (Mattson et al. 1970): the cache of capacity c is the c
//              most recent entries of any larger one.
//   state      kept between calls as keys in recency order (most recent first).
//   tokens     the byte-aware variant (cr_replay_create_tokens): capacities in
//              prefix tokens, one warp walking each stream (k_lru_tokens).
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

// ---- replay: batched stack distances ------------------------------------------
// One warp per (stream, chunk) holds the LRU of the largest capacity as keys in
// recency order, K[0] most recent, in shared memory, with an open-addressing
// index key -> physical slot (u16, slot + 1, 0 = empty, tombstones for evicted
// keys, rebuilt when a quarter of it is tombstones).  The keys form a ring:
// recency position q (0 = most recent) is slot (H + q) mod cmax.  A batch is
// 32 consecutive requests, one per lane.  The depth of
// request i (its LRU stack distance, Mattson et al. 1970) follows from the
// state before the batch and the batch itself:
//   - key seen earlier in the batch, last at lane j: 1 + the number of
//     distinct keys among lanes (j, i);
//   - first time in the batch, at position d0 before it: d0 + 1 + the number
//     of distinct keys among lanes < i that were deeper than d0 or absent;
//   - absent before the batch: a miss at every capacity.
// A request hits capacity c iff its depth <= c.  The state after the batch is
// the batch's distinct keys by last access (latest first) followed by the
// untouched old keys in their old order, cut at cmax.  Old keys below the
// deepest one the batch touched move (in place); those beyond it all shift by
// the same amount, which moving the head H does, so they stay where they are.
constexpr uint32_t kNone = 0xffffffffu;
constexpr uint16_t kTomb = 0xffffu;  // index slot whose key was evicted

struct lru_index {
    unsigned long long *K;  // [cmax] keys: a ring, recency position q at slot (H + q) mod cmax
    uint16_t *TS;           // [cmax] index slot of the key in each ring slot
    uint16_t *tab;          // [tsz] ring slot + 1; 0 = empty, kTomb = evicted
    uint32_t *bm;           // [32] bitmap of old positions touched by the batch
    uint32_t mask;
    int tbits;
};

__device__ __forceinline__ uint32_t lru_home(unsigned long long key, int tbits) { return (uint32_t)(key >> (64 - tbits)); }

// Ring slot of `key` (kNone if absent); *slot gets its index slot.
__device__ __forceinline__ uint32_t lru_lookup(const lru_index &X, unsigned long long key, uint32_t *slot)
{
    uint32_t s = lru_home(key, X.tbits);
    for (;;) {
        const uint32_t e = X.tab[s];
        if (e == 0) return kNone;
        if (e != kTomb && X.K[e - 1] == key) {
            *slot = s;
            return e - 1;
        }
        s = (s + 1) & X.mask;
    }
}

// Claim an empty or evicted slot for an absent key; returns the slot.
__device__ __forceinline__ uint32_t lru_insert(const lru_index &X, unsigned long long key, uint32_t pos)
{
    unsigned short *t = reinterpret_cast<unsigned short *>(X.tab);
    uint32_t s = lru_home(key, X.tbits);
    for (;;) {
        const unsigned short v = t[s];
        if (v == 0 || v == kTomb) {
            if (atomicCAS(&t[s], v, (unsigned short)(pos + 1)) == v) return s;
            continue;  // lost the slot to another lane: look at it again
        }
        s = (s + 1) & X.mask;
    }
}

__device__ __forceinline__ uint32_t ring_slot(uint32_t H, uint32_t q, uint32_t cmax)
{
    const uint32_t x = H + q;  // H < cmax, q < 2 cmax
    return x >= cmax ? (x - cmax >= cmax ? x - 2 * cmax : x - cmax) : x;
}

// Index of the fill keys from ring slot H on, from scratch (warp-cooperative);
// clears every tombstone.
__device__ __forceinline__ void lru_reindex(const lru_index &X, uint32_t H, uint32_t fill, uint32_t cmax,
                                            uint32_t lane)
{
    uint4 *t4 = reinterpret_cast<uint4 *>(X.tab);
    for (uint32_t x = lane; x < (X.mask + 1) / 8; x += 32) t4[x] = make_uint4(0, 0, 0, 0);
    __syncwarp();
    for (uint32_t q = lane; q < fill; q += 32) {
        const uint32_t ph = ring_slot(H, q, cmax);
        X.TS[ph] = (uint16_t)lru_insert(X, X.K[ph], ph);
    }
    __syncwarp();
}

template <int NC>
__global__ void __launch_bounds__(128)
k_lru_batch(const replay_caps caps, uint32_t cmax, uint32_t R, uint32_t ns, uint32_t CL, int tbits,
            const uint32_t *__restrict__ start, const uint32_t *__restrict__ coff, const uint32_t *__restrict__ total,
            const rec16 *__restrict__ rec, const replay_state st, unsigned long long *__restrict__ ctr)
{
    extern __shared__ uint4 smb[];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
    const uint32_t tsz = 1u << tbits;
    // per-warp region: index (2*tsz bytes), bitmap (128), keys (8*cmax), slots (2*cmax)
    const size_t per_warp = ((size_t)tsz * 2 + 128 + (size_t)cmax * 10 + 15) & ~(size_t)15;
    unsigned char *base = reinterpret_cast<unsigned char *>(smb) + per_warp * warp;
    lru_index X;
    X.tab = reinterpret_cast<uint16_t *>(base);
    X.bm = reinterpret_cast<uint32_t *>(base + (size_t)tsz * 2);
    X.K = reinterpret_cast<unsigned long long *>(base + (size_t)tsz * 2 + 128);
    X.TS = reinterpret_cast<uint16_t *>(base + (size_t)tsz * 2 + 128 + (size_t)cmax * 8);
    X.mask = tsz - 1;
    X.tbits = tbits;

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
    const uint32_t lt = (1u << lane) - 1u, gt = ~(lt | (1u << lane));

    if (b == e) {  // nothing routed here: carry the state over unchanged
        unsigned long long *kout = st.keys_out + (unsigned long long)s * cmax;
        for (uint32_t q = lane; q < fill_in; q += 32) kout[q] = kin[q];
        if (lane == 0) st.fill_out[s] = fill_in;
        return;
    }

    // ---- state at p0 ------------------------------------------------------------
    uint32_t fill = 0;
    if (ci == 0) {
        for (uint32_t q = lane; q < fill_in; q += 32) X.K[q] = kin[q];
        fill = fill_in;
        __syncwarp();
        lru_reindex(X, 0, fill, cmax, lane);
    } else {
        // walk backwards collecting distinct keys, most recent first
        lru_reindex(X, 0, 0, cmax, lane);
        const uint32_t back = p0 - b;
        const uint32_t vtot = back + fill_in;
        for (uint32_t v0 = 0; v0 < vtot && fill < cmax; v0 += 32) {
            const uint32_t v = v0 + lane;
            const bool valid = v < vtot;
            unsigned long long key = 0;
            if (valid) key = v < back ? rec[p0 - 1 - v].key : kin[v - back];
            const uint32_t vm = __ballot_sync(0xffffffffu, valid);
            const uint32_t peers = __match_any_sync(0xffffffffu, key) & vm;
            uint32_t sl;
            const bool fresh = valid && (peers & lt) == 0 && lru_lookup(X, key, &sl) == kNone;
            const uint32_t bal = __ballot_sync(0xffffffffu, fresh);
            const uint32_t pos = fill + __popc(bal & lt);
            __syncwarp();
            if (fresh && pos < cmax) {
                X.K[pos] = key;
                X.TS[pos] = (uint16_t)lru_insert(X, key, pos);
            }
            fill = min(cmax, fill + (uint32_t)__popc(bal));
            __syncwarp();
        }
    }

    unsigned long long my_req = 0, my_prompt = 0;
    unsigned long long my_hit[NC], my_tok[NC];
#pragma unroll
    for (int c = 0; c < NC; ++c) my_hit[c] = my_tok[c] = 0;
    const uint32_t nwords = (cmax + 31) / 32;
    uint32_t tomb = 0;  // tombstones in the index
    uint32_t H = 0;     // ring slot of recency position 0

    rec16 ahead = {0ull, 0u, 0u};  // the next batch's records, loaded one batch early
    if (p0 + lane < p1) ahead = rec[p0 + lane];
    for (uint32_t t0 = p0; t0 < p1; t0 += 32) {
        const uint32_t cnt = (p1 - t0) < 32u ? (p1 - t0) : 32u;
        const bool valid = lane < cnt;
        const rec16 mine = ahead;
        if (t0 + 32u + lane < p1) ahead = rec[t0 + 32u + lane];
        if (valid) {
            my_req += 1;
            my_prompt += (unsigned long long)mine.P + mine.S;
        }
        const uint32_t vm = cnt == 32 ? 0xffffffffu : (1u << cnt) - 1u;
        const uint32_t grp = __match_any_sync(0xffffffffu, mine.key) & vm;
        const uint32_t below = grp & lt, above = grp & gt;
        const bool first = valid && below == 0;
        const uint32_t next = above ? (uint32_t)__ffs(above) - 1u : 32u;
        uint32_t slot0 = kNone, d0 = kNone;
        if (first) {
            const uint32_t ph = lru_lookup(X, mine.key, &slot0);
            if (ph != kNone) d0 = ph >= H ? ph - H : ph + cmax - H;  // recency position
        }
        // lanes that push request i deeper, for every lane at once, by comparing
        // bit-sliced values from the most significant bit down (per bit: lanes
        // still equal keep the ones with the same bit; a lane whose bit is 1
        // where this lane's is 0 is decided greater):
        //   repeat i: lanes whose key does not recur before i (next_l > i);
        //   first i:  first occurrences whose old position is deeper (D_l > D_i)
        const uint32_t D = first ? (d0 < cmax ? d0 : 2047u) : 2047u;  // 2047: absent
        uint32_t gN = 0, eN = 0xffffffffu, gD = 0, eD = 0xffffffffu;
#pragma unroll
        for (int bt = 10; bt >= 0; --bt) {
            const uint32_t BD = __ballot_sync(0xffffffffu, (D >> bt) & 1u);
            const uint32_t MD = 0u - ((D >> bt) & 1u);
            gD |= eD & BD & ~MD;
            eD &= ~(BD ^ MD);
            if (bt <= 5) {
                const uint32_t BN = __ballot_sync(0xffffffffu, (next >> bt) & 1u);
                const uint32_t MN = 0u - ((lane >> bt) & 1u);
                gN |= eN & BN & ~MN;
                eN &= ~(BN ^ MN);
            }
        }
        const uint32_t firstm = __ballot_sync(0xffffffffu, first);
        // repeat: lanes strictly between the previous occurrence and this one
        const uint32_t win = lt & ~((2u << (31u - (uint32_t)__clz(below | 1u))) - 1u);
        const uint32_t dep_rep = 1u + (uint32_t)__popc(gN & win);
        const uint32_t dep_first = d0 < cmax ? d0 + 1u + (uint32_t)__popc(gD & firstm & lt) : kNone;
        const uint32_t depth = !valid ? kNone : (first ? dep_first : dep_rep);
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            if (c < (int)caps.n_caps && depth <= caps.cap[c]) {
                my_hit[c] += 1;
                my_tok[c] += mine.P;
            }
        }

        // ---- state after the batch ------------------------------------------------
        const uint32_t lastm = __ballot_sync(0xffffffffu, valid && above == 0);
        const uint32_t u = (uint32_t)__popc(lastm);
        if (lane < nwords) X.bm[lane] = 0;
        __syncwarp();
        if (d0 != kNone) atomicOr(&X.bm[d0 >> 5], 1u << (d0 & 31));
        __syncwarp();
        const uint32_t wv = lane < nwords ? X.bm[lane] : 0u;
        uint32_t pre = (uint32_t)__popc(wv);  // inclusive prefix over words
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, pre, o);
            if (lane >= (uint32_t)o) pre += y;
        }
        const uint32_t touched = __shfl_sync(0xffffffffu, pre, 31);
        pre -= (uint32_t)__popc(wv);  // exclusive
        // old keys up to the deepest touched one move back (never forward),
        // highest block first, in place; each rewrites its index slot.  Those
        // beyond it shift by delta = u - touched, done by moving the head.
        const uint32_t pmax = __reduce_max_sync(0xffffffffu, d0 != kNone ? d0 + 1u : 0u);  // deepest + 1
        const uint32_t delta = u - touched;
        const uint32_t H2 = H >= delta % cmax ? H - delta % cmax : H + cmax - delta % cmax;
        uint32_t evicted = 0;
        for (int tb = (int)((pmax + 31) / 32) - 1; tb >= 0; --tb) {
            const uint32_t p = (uint32_t)tb * 32u + lane;
            const uint32_t wt = __shfl_sync(0xffffffffu, wv, tb), pt = __shfl_sync(0xffffffffu, pre, tb);
            unsigned long long v = 0;
            uint32_t np = kNone, ts = 0;
            if (p < pmax && !((wt >> lane) & 1u)) {
                const uint32_t ph = ring_slot(H, p, cmax);
                v = X.K[ph];
                ts = X.TS[ph];
                np = p + u - (pt + (uint32_t)__popc(wt & lt));
            }
            __syncwarp();
            if (np < cmax) {
                const uint32_t ph = ring_slot(H2, np, cmax);
                X.K[ph] = v;
                X.TS[ph] = (uint16_t)ts;
                X.tab[ts] = (uint16_t)(ph + 1);
            } else if (np != kNone) {
                X.tab[ts] = kTomb;
                ++evicted;
            }
        }
        // old keys beyond the deepest touched one that the shift pushes past cmax
        {
            const uint32_t from = max(pmax, cmax > delta ? cmax - delta : 0u);
            const uint32_t p = from + lane;
            if (p < fill) {  // at most delta <= 32 of them
                X.tab[X.TS[ring_slot(H, p, cmax)]] = kTomb;
                ++evicted;
            }
        }
        __syncwarp();
        // the batch's distinct keys go to the front; a key already resident keeps
        // its slot (taken from the lane of its first occurrence), a new one claims one
        const uint32_t fl = (uint32_t)__ffs(grp ? grp : 1u) - 1u;
        const uint32_t kslot = __shfl_sync(0xffffffffu, slot0, fl);
        const uint32_t rank = (uint32_t)__popc(lastm & gt);
        if (valid && above == 0) {
            if (kslot != kNone) {
                if (rank < cmax) {
                    const uint32_t ph = ring_slot(H2, rank, cmax);
                    X.K[ph] = mine.key;
                    X.TS[ph] = (uint16_t)kslot;
                    X.tab[kslot] = (uint16_t)(ph + 1);
                } else {
                    X.tab[kslot] = kTomb;
                    ++evicted;
                }
            } else if (rank < cmax) {
                const uint32_t ph = ring_slot(H2, rank, cmax);
                X.K[ph] = mine.key;
                X.TS[ph] = (uint16_t)lru_insert(X, mine.key, ph);
            }
        }
        H = H2;
        fill = min(cmax, fill - touched + u);
        tomb += __reduce_add_sync(0xffffffffu, evicted);
        __syncwarp();
        if (4 * (fill + tomb) > 3 * (X.mask + 1)) {  // too many tombstones: index afresh
            lru_reindex(X, H, fill, cmax, lane);
            tomb = 0;
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
    // ---- the stream's last chunk hands the state to the next call, most recent first
    if (p1 == e) {
        unsigned long long *kout = st.keys_out + (unsigned long long)s * cmax;
        for (uint32_t q = lane; q < fill; q += 32) kout[q] = X.K[ring_slot(H, q, cmax)];
        if (lane == 0) st.fill_out[s] = fill;
    }
}

template <int NC>
int launch_batch_nc(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                    const uint32_t *coff, const uint32_t *total, uint64_t m, const rec16 *rec, uint64_t *d_ctr)
{
    const uint32_t cmax = rp->cmax;
    int tbits = 6;
    while ((1u << tbits) < 4 * cmax) ++tbits;  // index at most a quarter full of live keys
    const size_t per_warp = ((size_t)(1u << tbits) * 2 + 128 + (size_t)cmax * 10 + 15) & ~(size_t)15;
    // warps per block: the most warps per SM that shared memory allows
    const size_t sm_bytes = 227 * 1024;
    uint32_t wpb = 4, best = 0;
    for (uint32_t x = 4; x >= 1; --x) {
        const size_t blk = per_warp * x + 1024;
        const uint32_t nb = blk <= sm_bytes ? (uint32_t)(sm_bytes / blk) : 0u;
        if (nb * x > best) {
            best = nb * x;
            wpb = x;
        }
    }
    const size_t smem = per_warp * wpb;
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_batch<NC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    const uint32_t ns = rp->n_rep * rp->R;
    const uint64_t items = (uint64_t)ns + (m + CL - 1) / CL;  // upper bound on work items
    replay_state st;
    st.keys_in = rp->d_keys[rp->cur];
    st.fill_in = rp->d_fill[rp->cur];
    st.keys_out = rp->d_keys[rp->cur ^ 1];
    st.fill_out = rp->d_fill[rp->cur ^ 1];
    CR_LAUNCH(ctx, k_lru_batch<NC>, (unsigned int)((items + wpb - 1) / wpb), wpb * 32, smem, caps, cmax, rp->R, ns,
              CL, tbits, start, coff, total, rec, st, (unsigned long long *)d_ctr);
    rp->cur ^= 1;
    return CR_OK;
}

int launch_batch(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                 const uint32_t *coff, const uint32_t *total, uint64_t m, const rec16 *rec, uint64_t *d_ctr)
{
    if (caps.n_caps == 1) return launch_batch_nc<1>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
    if (caps.n_caps <= 3) return launch_batch_nc<3>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
    return launch_batch_nc<CR_MAX_CAPS>(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
}

// ---- token-weighted variant ---------------------------------------------------
// Capacities count prefix tokens.  With one prefix length per key, the cache
// of capacity c holds the longest run of most recent prefixes whose tokens fit
// in c (evictions always take the least recent), so one list at the largest
// capacity decides every capacity: a request hits at c iff its key is listed
// and the tokens from the front of the list through the key are <= c.  One
// warp per (replica, destination) stream walks the stream's requests in
// order.  The list holds keys and CUMULATIVE tokens (entry j: the tokens of
// entries 0..j), so a lookup is a ballot plus one read, moving a key to the
// front adds its length to the entries it passes, and eviction is a ballot on
// the tail.  A list of at most 32 prefixes lives in registers (lane j holds
// entry j; the move is a shuffle-up); a longer one lives in shared memory and
// is scanned 32 entries at a time.  Only hits and hit tokens depend on the
// capacity; request and prompt totals are summed once per 32 records.
constexpr int kTokWarps = 4;
constexpr uint32_t kTokMax = CR_MAX_CAP;  // prefixes per list

__device__ __forceinline__ uint32_t sat_add(uint32_t a, uint32_t b)
{
    // a sum past 2^32 - 1 is above every capacity (<= 2^31) and is evicted anyway
    const unsigned long long v = (unsigned long long)a + b;
    return v > 0xffffffffull ? 0xffffffffu : (uint32_t)v;
}

__global__ void __launch_bounds__(kTokWarps * 32) k_lru_tokens(const __grid_constant__ replay_caps caps, uint32_t ns,
                                                               uint32_t R, const uint32_t *__restrict__ start,
                                                               const rec16 *__restrict__ rec,
                                                               unsigned long long *__restrict__ keys_state,
                                                               uint32_t *__restrict__ cum_state,
                                                               uint32_t *__restrict__ fill_state,
                                                               unsigned long long *__restrict__ ctr, uint32_t *status)
{
    extern __shared__ unsigned long long tok_sh[];
    const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const uint32_t s = blockIdx.x * kTokWarps + w;
    if (s >= ns) return;  // whole warps only; the kernel has no block-wide barrier
    unsigned long long *K = tok_sh + (size_t)w * kTokMax;
    uint32_t *Cm = reinterpret_cast<uint32_t *>(tok_sh + (size_t)kTokWarps * kTokMax) + (size_t)w * kTokMax;
    uint32_t capmax = 0;
    for (uint32_t c = 0; c < caps.n_caps; ++c) capmax = caps.cap[c] > capmax ? caps.cap[c] : capmax;
    const uint32_t mycap = lane < caps.n_caps ? caps.cap[lane] : 0u;
    uint32_t f = fill_state[s];
    unsigned long long kr = 0;  // register list: entry `lane`
    uint32_t cr = 0;
    bool inreg = f <= 32;
    if (inreg) {
        if (lane < f) {
            kr = keys_state[(size_t)s * kTokMax + lane];
            cr = cum_state[(size_t)s * kTokMax + lane];
        }
    } else {
        for (uint32_t j = lane; j < f; j += 32) {
            K[j] = keys_state[(size_t)s * kTokMax + j];
            Cm[j] = cum_state[(size_t)s * kTokMax + j];
        }
    }
    __syncwarp();
    unsigned long long c_hit = 0, c_hit_tok = 0, c_prompt = 0;  // lane = capacity (prompt: every lane)
    const uint32_t i0 = start[s], i1 = start[s + 1];
    rec16 nx = {0ull, 0u, 0u};
    if (i0 + lane < i1) nx = rec[i0 + lane];
    for (uint32_t b0 = i0; b0 < i1; b0 += 32) {
        const rec16 cur = nx;
        if (b0 + 32 + lane < i1) nx = rec[b0 + 32 + lane];  // next 32 records in flight
        const uint32_t nb = i1 - b0 < 32 ? i1 - b0 : 32;
        if (lane < nb) c_prompt += (unsigned long long)cur.P + cur.S;
        for (uint32_t q = 0; q < nb; ++q) {
            const unsigned long long x = __shfl_sync(0xffffffffu, cur.key, q);
            const uint32_t P = __shfl_sync(0xffffffffu, cur.P, q);
            bool found;
            uint32_t upto = 0, zx = 0;
            if (inreg) {
                // ---- list in registers (f <= 32) ----
                const unsigned match = __ballot_sync(0xffffffffu, lane < f && kr == x);
                found = match != 0;
                const uint32_t pos = found ? __ffs(match) - 1 : f;
                const uint32_t cprev = __shfl_sync(0xffffffffu, cr, pos == 0 ? 0 : pos - 1);
                if (found) {
                    upto = __shfl_sync(0xffffffffu, cr, pos);
                    zx = upto - (pos ? cprev : 0u);
                }
                // entries [0, pos) move down one place and now follow x
                const unsigned long long kup = __shfl_up_sync(0xffffffffu, kr, 1);
                const uint32_t cup = __shfl_up_sync(0xffffffffu, cr, 1);
                const unsigned long long k31 = __shfl_sync(0xffffffffu, kr, 31);
                const uint32_t c31 = __shfl_sync(0xffffffffu, cr, 31);
                if (lane == 0) {
                    kr = x;
                    cr = P;
                } else if (lane <= pos) {
                    kr = kup;
                    cr = sat_add(cup, P);
                }
                if (!found) ++f;  // f may reach 33: entry 32 is the old entry 31
                const unsigned over = __ballot_sync(0xffffffffu, lane < f && cr > capmax);
                if (over) {
                    f = __ffs(over) - 1;  // the 33rd entry, if any, lies beyond and goes too
                } else if (f == 33) {
                    const uint32_t c32 = sat_add(c31, P);
                    if (c32 > capmax) {
                        f = 32;
                    } else {  // the list outgrows the registers
                        K[lane] = kr;
                        Cm[lane] = cr;
                        if (lane == 0) {
                            K[32] = k31;
                            Cm[32] = c32;
                        }
                        __syncwarp();
                        inreg = false;
                    }
                }
            } else {
                // ---- list in shared memory (f > 32) ----
                uint32_t pos = f;
                for (uint32_t c0 = 0; c0 < f; c0 += 32) {
                    const uint32_t j = c0 + lane;
                    const unsigned match = __ballot_sync(0xffffffffu, j < f && K[j] == x);
                    if (match) {
                        pos = c0 + __ffs(match) - 1;
                        break;
                    }
                }
                found = pos < f;
                if (found) {
                    upto = Cm[pos];
                    zx = upto - (pos ? Cm[pos - 1] : 0u);
                } else {
                    if (f == kTokMax) --f;  // the least recent prefix makes room
                    pos = f;
                    ++f;
                }
                for (int c0 = (int)((pos + 31) / 32) * 32 - 32; c0 >= 0; c0 -= 32) {  // [0, pos) down one
                    const uint32_t j = (uint32_t)c0 + lane;
                    const bool m = j < pos;
                    const unsigned long long k = m ? K[j] : 0ull;
                    const uint32_t cm = m ? Cm[j] : 0u;
                    __syncwarp();
                    if (m) {
                        K[j + 1] = k;
                        Cm[j + 1] = sat_add(cm, P);
                    }
                    __syncwarp();
                }
                if (lane == 0) {
                    K[0] = x;
                    Cm[0] = P;
                }
                __syncwarp();
                // the entries whose sums exceed the largest capacity form a suffix
                for (int c0 = (int)((f + 31) / 32) * 32 - 32; c0 >= 0; c0 -= 32) {
                    const uint32_t j = (uint32_t)c0 + lane;
                    const unsigned over = __ballot_sync(0xffffffffu, j < f && Cm[j] > capmax);
                    if (!over) break;
                    f = (uint32_t)c0 + __ffs(over) - 1;
                }
                if (f <= 32) {  // back to registers
                    kr = lane < f ? K[lane] : 0ull;
                    cr = lane < f ? Cm[lane] : 0u;
                    inreg = true;
                }
                __syncwarp();
            }
            if (found && zx != P && lane == 0) atomicOr(status, CR_FLAG_BADSIZE);
            if (found && upto <= mycap) {  // lanes past n_caps have mycap 0 < upto
                c_hit += 1;
                c_hit_tok += P;
            }
        }
    }
    if (inreg) {
        if (lane < f) {
            keys_state[(size_t)s * kTokMax + lane] = kr;
            cum_state[(size_t)s * kTokMax + lane] = cr;
        }
    } else {
        for (uint32_t j = lane; j < f; j += 32) {
            keys_state[(size_t)s * kTokMax + j] = K[j];
            cum_state[(size_t)s * kTokMax + j] = Cm[j];
        }
    }
    if (lane == 0) fill_state[s] = f;
    for (int o = 16; o > 0; o >>= 1) c_prompt += __shfl_xor_sync(0xffffffffu, c_prompt, o);
    if (lane < caps.n_caps) {
        const uint32_t rep = s / R, r = s - rep * R;
        unsigned long long *C = ctr + (((unsigned long long)rep * caps.n_caps + lane) * R + r) * CR_CTR_FIELDS;
        C[0] += i1 - i0;
        C[1] += c_hit;
        C[2] += c_hit_tok;
        C[3] += c_prompt;
        C[4] += c_prompt - c_hit_tok;
    }
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

extern "C" int cr_replay_create_tokens(cr_ctx *ctx, uint32_t n_rep, uint32_t R, const uint32_t *token_caps,
                                       uint32_t n_caps, cr_replay **out)
{
    if (!ctx || !out || !token_caps) return CR_EINVAL;
    *out = nullptr;
    if (n_rep == 0 || n_rep > CR_MAX_REPLICAS) return cr_fail(ctx, CR_EINVAL, "replay: n_rep=%u", n_rep);
    if (R == 0 || R > CR_MAX_R) return cr_fail(ctx, CR_EINVAL, "replay: R=%u", R);
    if (n_caps == 0 || n_caps > CR_MAX_CAPS) return cr_fail(ctx, CR_EINVAL, "replay: n_caps=%u", n_caps);
    for (uint32_t c = 0; c < n_caps; ++c)
        if (token_caps[c] == 0 || token_caps[c] > (1u << 31))
            return cr_fail(ctx, CR_EINVAL, "replay: token capacity %u outside 1..2^31", token_caps[c]);
    if ((uint64_t)n_rep * R >= (1ull << 31)) return cr_fail(ctx, CR_EINVAL, "replay: too many streams");
    cr_replay *rp = (cr_replay *)calloc(1, sizeof(cr_replay));
    if (!rp) return cr_fail(ctx, CR_ENOMEM, "replay: host allocation failed");
    rp->n_rep = n_rep;
    rp->R = R;
    rp->n_caps = n_caps;
    rp->cmax = kTokMax;
    rp->tokens = 1;
    memcpy(rp->caps, token_caps, n_caps * sizeof(uint32_t));
    rp->n_streams = (uint64_t)n_rep * R;
    if (cudaMalloc(&rp->d_keys[0], rp->n_streams * kTokMax * sizeof(unsigned long long)) != cudaSuccess ||
        cudaMalloc(&rp->d_size, rp->n_streams * kTokMax * sizeof(uint32_t)) != cudaSuccess ||
        cudaMalloc(&rp->d_fill[0], rp->n_streams * sizeof(uint32_t)) != cudaSuccess) {
        cudaGetLastError();
        cr_replay_destroy(ctx, rp);
        return cr_fail(ctx, CR_ENOMEM, "replay: cannot allocate state");
    }
    *out = rp;
    return cr_replay_reset(ctx, rp);
}

extern "C" int cr_replay_reset(cr_ctx *ctx, cr_replay *rp)
{
    if (!ctx || !rp) return CR_EINVAL;
    for (int b = 0; b < 2; ++b)
        if (rp->d_fill[b])
            CR_CUDA(ctx, cudaMemsetAsync(rp->d_fill[b], 0, rp->n_streams * sizeof(uint32_t), ctx->stream));
    return CR_OK;
}

extern "C" int cr_replay_destroy(cr_ctx *ctx, cr_replay *rp)
{
    if (!rp) return CR_OK;
    if (ctx) cudaStreamSynchronize(ctx->stream);
    for (int b = 0; b < 2; ++b) {
        if (rp->d_keys[b]) cudaFree(rp->d_keys[b]);
        if (rp->d_fill[b]) cudaFree(rp->d_fill[b]);
    }
    if (rp->d_size) cudaFree(rp->d_size);
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
    if (rp->tokens) {
        // token-weighted: one warp per stream, its list in shared memory, state updated in place
        const size_t tsmem = (size_t)kTokWarps * kTokMax * (sizeof(unsigned long long) + sizeof(uint32_t));
        if (tsmem > 48 * 1024)
            CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_tokens, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tsmem));
        CR_LAUNCH(ctx, k_lru_tokens, (ns + kTokWarps - 1) / kTokWarps, kTokWarps * 32, tsmem, caps, ns, R,
                  (const uint32_t *)start, (const rec16 *)rec, (unsigned long long *)rp->d_keys[0], rp->d_size,
                  rp->d_fill[0], (unsigned long long *)d_ctr, ctx->d_status);
        return CR_OK;
    }
    // chunk length: long enough that rebuilding an LRU state of cmax entries is amortised
    const uint32_t CL = rp->cmax * 16u > 256u ? rp->cmax * 16u : 256u;
    CR_LAUNCH(ctx, k_chunk_counts, cr_blocks(ns, 256, gcap), 256, 0, (const uint32_t *)start, ns, CL, coff);
    CR_TRY(cr_scan_u32(ctx, coff, coff, ns, total));
    return launch_batch(ctx, rp, caps, CL, start, coff, total, m, rec, d_ctr);
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
