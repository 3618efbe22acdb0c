// a8, a9: shadow replay (cr_shadow_replay).
//
//   partition  one stable counting sort per replica by destination: each
//              (replica, destination) stream's request indices in arrival
//              order; the replay gathers each request's (key, prefix, suffix)
//              record, packed once per call, through them
//   replay     one warp per (stream, chunk); the stream's LRU at the LARGEST
//              capacity lives in shared memory as keys with recency stamps, a
//              bitmap of live stamps and a hash index, and 32 requests are
//              simulated per step, one per lane.  A request's depth (its LRU stack distance) decides the
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

__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t v, uint32_t lane)
{
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= (uint32_t)o) v += y;
    }
    return v;
}

// ---- partition: one stable counting sort per replica, by destination --------
// Tiles of 8192 requests.  k_part_count writes each tile's destination counts
// at [(replica * R + r) * ntiles + tile]; one exclusive scan of that array
// gives every (stream, tile) its output base, in stream-major order.
// k_part_scatter ranks each tile's requests stably (warp-private counters),
// stages their request indices in shared memory in (destination, arrival)
// order, and writes them out so that consecutive threads write consecutive
// positions of a destination's run.  The replay reads each request's
// (key, prefix, suffix) record, packed once per call by k_part_records,
// through these indices.
constexpr int kPartBlock = 256;
constexpr int kPartWarps = kPartBlock / 32;
constexpr int kPartPer = 32;                      // requests per thread
constexpr int kPartTile = kPartBlock * kPartPer;  // 8192
constexpr uint32_t kNoDest = 0xffffu;

// Counts of one tile in u32 bins [R], one shared-memory atomic add per item:
// counting needs no order, so lane l of warp w takes the 32 consecutive items
// 1024 w + 32 l .. + 31, read up front with four 16-byte loads.
__global__ void __launch_bounds__(kPartBlock) k_part_count(const uint16_t *__restrict__ dest, unsigned long long n,
                                                           uint32_t R, uint32_t ntiles, uint32_t *__restrict__ cnt,
                                                           uint32_t *status)
{
    extern __shared__ uint32_t pcb[];  // [R]
    const uint32_t rep = blockIdx.y, tile = blockIdx.x, lane = cr_lane(), warp = threadIdx.x >> 5;
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) pcb[r] = 0;
    __syncthreads();
    const uint16_t *D = dest + (unsigned long long)rep * n;
    const unsigned long long base = (unsigned long long)tile * kPartTile;
    const uint32_t cnt_t = (uint32_t)min((unsigned long long)kPartTile, n - base);
    constexpr uint32_t kPerWarp = kPartTile / kPartWarps;
    const uint32_t first = warp * kPerWarp + lane * 32u;
    uint32_t dv[16];  // two destinations per word
    const bool whole = base + first + 32u <= n && ((base + first) & 7u) == 0 &&
                       ((reinterpret_cast<uintptr_t>(D) & 15u) == 0);
    if (whole) {
        const uint4 *src = reinterpret_cast<const uint4 *>(D + base + first);
#pragma unroll
        for (int x = 0; x < 4; ++x) {
            const uint4 v = src[x];
            dv[4 * x] = v.x;
            dv[4 * x + 1] = v.y;
            dv[4 * x + 2] = v.z;
            dv[4 * x + 3] = v.w;
        }
    } else {
#pragma unroll
        for (int x = 0; x < 16; ++x) {
            const uint32_t i0 = first + 2u * x, i1 = i0 + 1u;
            const uint32_t a = i0 < cnt_t ? D[base + i0] : kNoDest, c = i1 < cnt_t ? D[base + i1] : kNoDest;
            dv[x] = a | (c << 16);
        }
    }
    bool bad = false;
#pragma unroll
    for (uint32_t j = 0; j < (uint32_t)kPartPer; ++j) {
        const uint32_t d = (dv[j >> 1] >> (16 * (j & 1))) & 0xffffu;
        if (first + j < cnt_t) {
            if (d < R)
                atomicAdd(&pcb[d], 1u);
            else
                bad = true;  // skipped: reported through the status word
        }
    }
    __syncthreads();
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) cnt[((unsigned long long)rep * R + r) * ntiles + tile] = pcb[r];
    if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(status, CR_FLAG_BADDEST);
}

// start[s] = first record of stream s = (replica, r); start[ns] = number of records.
__global__ void k_part_starts(const uint32_t *__restrict__ off, uint32_t ns, uint32_t ntiles,
                              const uint32_t *__restrict__ total, uint32_t *__restrict__ start)
{
    for (uint32_t s = blockIdx.x * blockDim.x + threadIdx.x; s <= ns; s += gridDim.x * blockDim.x)
        start[s] = s < ns ? off[(unsigned long long)s * ntiles] : *total;
}

// Shared memory of k_part_scatter: per-warp counters wc[8][R] (u16), the
// tile's destination offsets toff[R] (u32), each item's (destination << 16 |
// rank among its warp's items of that destination) (u32), and the tile's items
// in (destination, arrival) order (u16 item numbers).
__host__ __device__ inline size_t part_scatter_smem(uint32_t R)
{
    return (size_t)R * kPartWarps * 2 + (size_t)R * 4 + (size_t)kPartTile * 6;
}

__global__ void __launch_bounds__(kPartBlock) k_part_scatter(const uint16_t *__restrict__ dest, unsigned long long n,
                                                             uint32_t R, uint32_t ntiles,
                                                             const uint32_t *__restrict__ off,
                                                             uint32_t *__restrict__ out, unsigned long long m)
{
    extern __shared__ uint4 psm[];
    uint16_t *wc = reinterpret_cast<uint16_t *>(psm);                            // [8][R]
    uint32_t *toff = reinterpret_cast<uint32_t *>(wc + (size_t)R * kPartWarps);  // [R]
    uint32_t *spk = toff + R;                                                    // [kPartTile]
    uint16_t *sitem = reinterpret_cast<uint16_t *>(spk + kPartTile);            // [kPartTile]
    __shared__ uint32_t part[kPartBlock];
    __shared__ uint32_t s_valid;
    const uint32_t rep = blockIdx.y, tile = blockIdx.x, lane = cr_lane(), warp = threadIdx.x >> 5;
    const uint32_t lt = (1u << lane) - 1u;
    uint4 *wc4 = reinterpret_cast<uint4 *>(wc);
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) wc4[r] = make_uint4(0, 0, 0, 0);
    __syncthreads();
    const uint16_t *D = dest + (unsigned long long)rep * n;
    const unsigned long long base = (unsigned long long)tile * kPartTile;
    const uint32_t cnt = (uint32_t)min((unsigned long long)kPartTile, n - base);
    // ranks: warp w takes items [1024 w, 1024 w + 1024) of the tile, 32 at a time
    // (lane order is arrival order); all 32 rounds' destinations are read up front.
    // The lanes of a round with equal destinations are found from one ballot per
    // bit of the destination (R stands for "no item").
    constexpr uint32_t kPerWarp = kPartTile / kPartWarps;
    const uint32_t nb = 32u - (uint32_t)__clz(R);
    uint16_t *wcw = wc + (size_t)warp * R;
    uint32_t dv[kPartPer / 2];
#pragma unroll
    for (int x = 0; x < kPartPer / 2; ++x) {
        const uint32_t i0 = warp * kPerWarp + (2u * x) * 32u + lane, i1 = i0 + 32u;
        const uint32_t a = i0 < cnt ? D[base + i0] : kNoDest, c = i1 < cnt ? D[base + i1] : kNoDest;
        dv[x] = a | (c << 16);
    }
#pragma unroll
    for (uint32_t j = 0; j < (uint32_t)kPartPer; ++j) {
        const uint32_t it = warp * kPerWarp + j * 32u + lane;
        uint32_t d = (dv[j >> 1] >> (16 * (j & 1))) & 0xffffu;
        const uint32_t dd = d < R ? d : R;
        if (d >= R) d = kNoDest;
        uint32_t peers = 0xffffffffu;
        for (uint32_t bt = 0; bt < nb; ++bt) {
            const uint32_t bit = (dd >> bt) & 1u;
            const uint32_t B = __ballot_sync(0xffffffffu, bit);
            peers &= bit ? B : ~B;
        }
        const uint32_t before = d != kNoDest ? wcw[d] : 0u;
        spk[it] = (d << 16) | (before + (uint32_t)__popc(peers & lt));
        __syncwarp();
        if (d != kNoDest && (peers & lt) == 0) wcw[d] = (uint16_t)(before + __popc(peers));
        __syncwarp();
    }
    __syncthreads();
    // per destination: exclusive prefix over the 8 warps and its total; then the
    // tile's destination offsets by a block scan over thread-contiguous ranges of R
    const uint32_t per = (R + kPartBlock - 1) / kPartBlock, r0 = threadIdx.x * per;
    uint32_t run = 0;
    for (uint32_t r = r0; r < r0 + per && r < R; ++r) {
        uint16_t acc = 0;
#pragma unroll
        for (int w = 0; w < kPartWarps; ++w) {
            const uint16_t x = wc[(size_t)w * R + r];
            wc[(size_t)w * R + r] = acc;
            acc = (uint16_t)(acc + x);
        }
        toff[r] = acc;  // the destination's total until the scan below
        run += acc;
    }
    part[threadIdx.x] = run;
    __syncthreads();
    if (threadIdx.x < 32) {  // exclusive scan of the 256 partials by one warp
        constexpr int kPer = kPartBlock / 32;
        uint32_t x[kPer], sum = 0;
#pragma unroll
        for (int k = 0; k < kPer; ++k) {
            x[k] = part[threadIdx.x * kPer + k];
            sum += x[k];
        }
        const uint32_t incl = warp_incl_scan(sum, lane);
        uint32_t ex = incl - sum;
#pragma unroll
        for (int k = 0; k < kPer; ++k) {
            part[threadIdx.x * kPer + k] = ex;
            ex += x[k];
        }
        if (threadIdx.x == 31) s_valid = incl;
    }
    __syncthreads();
    run = part[threadIdx.x];
    for (uint32_t r = r0; r < r0 + per && r < R; ++r) {
        const uint32_t t = toff[r];
        toff[r] = run;
        run += t;
    }
    __syncthreads();
    // staging: every valid item at its place in (destination, arrival) order
    for (uint32_t it = threadIdx.x; it < cnt; it += kPartBlock) {
        const uint32_t pk = spk[it];
        const uint32_t d = pk >> 16;
        if (d == kNoDest) continue;
        const uint32_t pos = toff[d] + wc[(size_t)(it / kPerWarp) * R + d] + (pk & 0xffffu);
        sitem[pos] = (uint16_t)it;
    }
    // each destination's output position minus its staging position (mod 2^32), in
    // the counters' space, which the staging no longer needs
    uint32_t *gb = reinterpret_cast<uint32_t *>(wc);  // [R]
    const uint32_t *O = off + (unsigned long long)rep * R * ntiles;
    __syncthreads();
    for (uint32_t r = threadIdx.x; r < R; r += kPartBlock) gb[r] = O[(unsigned long long)r * ntiles + tile] - toff[r];
    __syncthreads();
    // output: consecutive threads write consecutive positions of each destination's run
    const uint32_t valid = s_valid;
    for (uint32_t j = threadIdx.x; j < valid; j += kPartBlock) {
        const uint32_t it = sitem[j];
        const uint32_t d = spk[it] >> 16;
        if (d >= R) continue;  // never: every staged item is valid (guards the writes)
        const uint32_t o = gb[d] + j;
        if (o < m) out[o] = (uint32_t)(base + it);
    }
}

// One (key, prefix, suffix) record per request, read by the replay through the indices.
__global__ void k_part_records(const unsigned long long *__restrict__ keys, const uint32_t *__restrict__ plen,
                               const uint32_t *__restrict__ slen, unsigned long long n, rec16 *__restrict__ recs)
{
    for (unsigned long long i = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (unsigned long long)gridDim.x * blockDim.x) {
        rec16 r;
        r.key = keys[i];
        r.P = plen[i];
        r.S = slen[i];
        recs[i] = r;
    }
}

// The stream of every work item: items coff[s] .. coff[s + 1] - 1 belong to stream s
// (coff[ns] is the total), written at wmap[item].
__global__ void k_item_streams(const uint32_t *__restrict__ coff, uint32_t ns, uint32_t *__restrict__ wmap,
                               uint64_t items_max)
{
    for (uint32_t s = blockIdx.x * blockDim.x + threadIdx.x; s < ns; s += gridDim.x * blockDim.x)
        for (uint32_t w = coff[s]; w < coff[s + 1] && w < items_max; ++w) wmap[w] = s;
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

// ---- replay: batched stack distances over recency stamps -----------------------
// One warp per (stream, chunk) holds the LRU of the LARGEST capacity in shared
// memory.  Each resident key has a slot holding the key and its STAMP, the
// time of its last access, and an entry in an open-addressing index
// key -> slot.  Time advances by one 32-bit word per step of 32 requests (the
// request on lane l of the step at word w has time 32 w + l), and a bitmap
// over the times of a window marks the live stamps: bit t is set iff t is the
// stamp of a resident key.  The recency position of a resident key (0 = most
// recent) is the number of live bits above its stamp, which one warp-wide scan
// of the words' popcounts gives for every lane of a step at once.  Nothing
// moves when a key is accessed: its old bit is cleared and its bit in the new
// word set.  When the window's words are used up, the stamps are renumbered
// 0 .. fill-1 in recency order (compaction).
//
// A step is 32 consecutive requests of the stream, one per lane.  The depth of
// request i (its LRU stack distance, Mattson et al. 1970) follows from the
// state before the step and the step itself:
//   - key seen earlier in the step, last at lane j: 1 + the number of distinct
//     keys among lanes (j, i), at most 31;
//   - first time in the step, at recency position d0 before it: d0 + 1 + the
//     number of distinct keys among lanes < i that were deeper than d0 or
//     absent;
//   - absent before the step: a miss at every capacity.
// A request hits capacity c iff its depth <= c.  The state after the step is
// the step's distinct keys by last access, then the untouched old keys in
// their old order, cut at cmax: when the step brings m new keys and the cache
// would exceed cmax, the oldest untouched keys (the lowest live bits) leave
// and the new keys take their slots.
constexpr uint32_t kNone = 0xffffffffu;
constexpr uint32_t kAbsent = 2047u;    // depth code of a key not resident (above every position < 1024)

constexpr uint32_t kStash = 32;              // index entries that found both buckets full
constexpr uint32_t kDegraded = 0x80000000u;  // stash overflowed: lookups scan the keys
constexpr uint16_t kInStash = 0xffffu;       // TS of a slot whose entry is in the stash

struct stamp_lru {
    unsigned long long *K;    // [cmax] key of each slot
    uint32_t *BM;             // [nw] live-stamp bits, word w = times 32 w .. 32 w + 31
    uint32_t *stash_n;        // stash entries claimed (| kDegraded once it overflowed)
    unsigned long long *bkt;  // [2^nbb] index buckets of four 16-bit entries (0 = empty)
    uint16_t *ST;             // [cmax] stamp of each slot
    uint16_t *T2S;            // [32 nw] slot whose stamp is each time (where the bit is set)
    uint16_t *EV;             // [32] slots the step's evictions freed
    uint16_t *stash;          // [kStash] slot + 1 of keys indexed outside their buckets (0 = free)
    uint16_t *TS;             // [cmax] where each slot's index entry is: bucket << 2 | entry, or kInStash
    uint32_t nbb;             // log2 of the bucket count
};

// Per-warp layout: K at 0 (8-byte entries), BM and the stash count after it, the
// buckets at the next 16-byte boundary (cleared with 16-byte stores), then ST,
// T2S, EV and the stash.
__host__ __device__ inline size_t stamp_bkt_offset(uint32_t cmax, uint32_t nw)
{
    return ((size_t)cmax * 8 + (size_t)(nw + 1) * 4 + 15) & ~(size_t)15;
}

__host__ __device__ inline size_t stamp_lru_bytes(uint32_t cmax, uint32_t nw, uint32_t nbb)
{
    return (stamp_bkt_offset(cmax, nw) + ((size_t)8 << nbb) + (size_t)cmax * 4 + (size_t)nw * 64 + 64 +
            (size_t)kStash * 2 + 15) &
           ~(size_t)15;
}

__device__ __forceinline__ stamp_lru stamp_lru_at(unsigned char *base, uint32_t cmax, uint32_t nw, uint32_t nbb)
{
    stamp_lru X;
    X.K = reinterpret_cast<unsigned long long *>(base);
    X.BM = reinterpret_cast<uint32_t *>(base + (size_t)cmax * 8);
    X.stash_n = X.BM + nw;
    X.bkt = reinterpret_cast<unsigned long long *>(base + stamp_bkt_offset(cmax, nw));
    X.ST = reinterpret_cast<uint16_t *>(X.bkt + (1u << nbb));
    X.T2S = X.ST + cmax;
    X.EV = X.T2S + (size_t)nw * 32;
    X.stash = X.EV + 32;
    X.TS = X.stash + kStash;
    X.nbb = nbb;
    return X;
}

// Index: two candidate buckets of four 16-bit entries per key, each entry
// (5-bit tag << 11) | (slot + 1).  A key goes into the emptier of its buckets
// (the first when equal); a key whose buckets are both full goes to a small
// stash (with at most a quarter of the entries live that is rare); if even the
// stash is full the index is marked degraded and lookups scan every key.
// Entries never move, so concurrent lanes only need compare-and-swap on the
// 64-bit bucket words, and a deleted entry becomes empty (no tombstones).
struct bkt_hash {
    uint32_t b1, b2, tag;
};

__device__ __forceinline__ bkt_hash sl_hash(unsigned long long key, uint32_t nbb)
{
    const unsigned long long h = key * 0x9e3779b97f4a7c15ull;  // an odd multiplier spreads every key bit upwards
    bkt_hash r;
    r.b1 = (uint32_t)(h >> (64 - nbb));
    r.b2 = (uint32_t)(h >> (64 - 2 * nbb)) & ((1u << nbb) - 1u);
    r.tag = (uint32_t)(h >> (59 - 2 * nbb)) & 31u;
    return r;
}

__device__ __forceinline__ uint32_t bkt_entry(unsigned long long w, int p) { return (uint32_t)(w >> (16 * p)) & 0xffffu; }

// Slot of `key`, or kNone (fill: resident keys, scanned only when the index is degraded).
__device__ __forceinline__ uint32_t sl_lookup(const stamp_lru &X, unsigned long long key, uint32_t fill, uint32_t cmax)
{
    const bkt_hash H = sl_hash(key, X.nbb);
    const unsigned long long w1 = X.bkt[H.b1], w2 = X.bkt[H.b2];
#pragma unroll
    for (int p = 0; p < 8; ++p) {
        const uint32_t e = bkt_entry(p < 4 ? w1 : w2, p & 3);
        if (e != 0 && (e >> 11) == H.tag) {
            const uint32_t q = (e & 0x7ffu) - 1u;
            if (q < cmax && X.K[q] == key) return q;
        }
    }
    const uint32_t sn = *X.stash_n;
    if (sn) {
        if (sn & kDegraded) {
            for (uint32_t q = 0; q < fill; ++q)
                if (X.K[q] == key) return q;
            return kNone;
        }
        for (uint32_t i = 0; i < sn && i < kStash; ++i) {
            const uint32_t e = X.stash[i];
            if (e != 0 && e <= cmax && X.K[e - 1] == key) return e - 1;
        }
    }
    return kNone;
}

// Index an absent key held in slot q.  A lost compare-and-swap means another lane
// changed the bucket, so the next look sees it; the bound only guards the loop.
__device__ __forceinline__ void sl_insert(const stamp_lru &X, unsigned long long key, uint32_t q)
{
    const bkt_hash H = sl_hash(key, X.nbb);
    const unsigned long long ent = (unsigned long long)((H.tag << 11) | (q + 1u));
    for (int it = 0; it < 64; ++it) {
        const unsigned long long w1 = X.bkt[H.b1], w2 = X.bkt[H.b2];
        int f1 = -1, f2 = -1, n1 = 0, n2 = 0;
#pragma unroll
        for (int p = 3; p >= 0; --p) {
            if (bkt_entry(w1, p) == 0) {
                f1 = p;
                ++n1;
            }
            if (bkt_entry(w2, p) == 0) {
                f2 = p;
                ++n2;
            }
        }
        uint32_t b;
        unsigned long long w;
        int p;
        if (f1 >= 0 && (n1 >= n2 || f2 < 0)) {
            b = H.b1;
            w = w1;
            p = f1;
        } else if (f2 >= 0) {
            b = H.b2;
            w = w2;
            p = f2;
        } else {
            break;  // both buckets full
        }
        if (atomicCAS(&X.bkt[b], w, w | (ent << (16 * p))) == w) {
            X.TS[q] = (uint16_t)((b << 2) | (uint32_t)p);
            return;
        }
    }
    X.TS[q] = kInStash;
    const uint32_t i = atomicAdd(X.stash_n, 1u);
    if (i < kStash)
        X.stash[i] = (uint16_t)(q + 1u);
    else
        atomicOr(X.stash_n, kDegraded);
}

// Remove the index entry of slot q: its place is recorded in TS[q].
__device__ __forceinline__ void sl_erase(const stamp_lru &X, uint32_t q)
{
    const uint32_t loc = X.TS[q];
    if (loc != kInStash) {
        atomicAnd(&X.bkt[loc >> 2], ~(0xffffull << (16 * (loc & 3u))));
        return;
    }
    const uint32_t sn = *X.stash_n & ~kDegraded;
    for (uint32_t i = 0; i < sn && i < kStash; ++i)
        if (X.stash[i] == q + 1u) {
            X.stash[i] = 0;
            return;
        }
}

// Index of slots 0 .. fill-1 from scratch (warp-cooperative).
__device__ __forceinline__ void sl_reindex(const stamp_lru &X, uint32_t fill, uint32_t lane)
{
    uint4 *t4 = reinterpret_cast<uint4 *>(X.bkt);
    for (uint32_t x = lane; x < (1u << X.nbb) / 2; x += 32) t4[x] = make_uint4(0, 0, 0, 0);
    if (lane == 0) *X.stash_n = 0;
    __syncwarp();
    for (uint32_t q = lane; q < fill; q += 32) sl_insert(X, X.K[q], q);
    __syncwarp();
}

// Stamps for keys K[0 .. fill) held in recency order (K[0] most recent): times
// fill-1 .. 0, bits 0 .. fill-1 set, the next step at the first word above them.
__device__ __forceinline__ void sl_stamps_in_order(const stamp_lru &X, uint32_t fill, uint32_t nw, uint32_t lane,
                                                   uint32_t &wnow, uint32_t &lo)
{
    for (uint32_t q = lane; q < fill; q += 32) {
        const uint32_t t = fill - 1u - q;
        X.ST[q] = (uint16_t)t;
        X.T2S[t] = (uint16_t)q;
    }
    for (uint32_t w = lane; w < nw; w += 32)
        X.BM[w] = 32u * w + 32u <= fill ? 0xffffffffu : (32u * w < fill ? (1u << (fill - 32u * w)) - 1u : 0u);
    wnow = (fill + 31u) / 32u;
    lo = 0;
    __syncwarp();
}


// Position of the k-th (from 0) set bit of w, which has more than k set bits.
__device__ __forceinline__ uint32_t nth_set_bit(uint32_t w, uint32_t k)
{
    uint32_t pos = 0;
#pragma unroll
    for (int sh = 16; sh >= 1; sh >>= 1) {
        const uint32_t lowc = (uint32_t)__popc(w & ((1u << sh) - 1u));
        if (k >= lowc) {
            k -= lowc;
            w >>= sh;
            pos += (uint32_t)sh;
        }
    }
    return pos;
}

// Live stamps below any time of the window: lane l keeps word 32 g + l of every
// group g of 32 words and the number of live bits in the words before it.
template <int NG>
struct live_prefix {
    uint32_t w[NG], ex[NG];
    __device__ __forceinline__ void load(const uint32_t *BM, uint32_t nw, uint32_t lane)
    {
        // both groups' popcounts in one scan: group g in bits 16 g .. 16 g + 15
        // (a group holds at most 1024 live bits, so the halves never carry)
        uint32_t pc = 0;
#pragma unroll
        for (int g = 0; g < NG; ++g) {
            const uint32_t wi = 32u * g + lane;
            w[g] = wi < nw ? BM[wi] : 0u;
            pc |= (uint32_t)__popc(w[g]) << (16 * g);
        }
        const uint32_t incl = warp_incl_scan(pc, lane);
        const uint32_t ex2 = incl - pc;
        ex[0] = ex2 & 0xffffu;
        if (NG > 1) ex[NG - 1] = (ex2 >> 16) + (__shfl_sync(0xffffffffu, incl, 31) & 0xffffu);
    }
    // live stamps < s; every lane of the warp must call it
    __device__ __forceinline__ uint32_t below(uint32_t s) const
    {
        const uint32_t src = (s >> 5) & 31u, g = s >> 10;
        uint32_t e = 0, b = 0;
#pragma unroll
        for (int gg = 0; gg < NG; ++gg) {
            const uint32_t ee = __shfl_sync(0xffffffffu, ex[gg], src), bb = __shfl_sync(0xffffffffu, w[gg], src);
            if (g == (uint32_t)gg) {
                e = ee;
                b = bb;
            }
        }
        return e + (uint32_t)__popc(b & ((1u << (s & 31u)) - 1u));
    }
};

// Renumber the stamps of slots 0 .. fill-1 to 0 .. fill-1 keeping their order.
template <int NG>
__device__ __forceinline__ void sl_compact(const stamp_lru &X, uint32_t fill, uint32_t nw, uint32_t lane,
                                           uint32_t &wnow, uint32_t &lo)
{
    live_prefix<NG> LP;
    LP.load(X.BM, nw, lane);
    for (uint32_t q0 = 0; q0 < fill; q0 += 32) {
        const uint32_t q = q0 + lane;
        const uint32_t nb = LP.below(q < fill ? (uint32_t)X.ST[q] : 0u);
        if (q < fill) {
            X.ST[q] = (uint16_t)nb;
            X.T2S[nb] = (uint16_t)q;
        }
    }
    for (uint32_t w = lane; w < nw; w += 32)
        X.BM[w] = 32u * w + 32u <= fill ? 0xffffffffu : (32u * w < fill ? (1u << (fill - 32u * w)) - 1u : 0u);
    wnow = (fill + 31u) / 32u;
    lo = 0;
    __syncwarp();
}

template <int NC, int NG, bool SMALL>
__global__ void __launch_bounds__(128)
k_lru_stamp(const replay_caps caps, uint32_t cmax, uint32_t nw, uint32_t R, uint32_t ns, uint32_t CL, uint32_t nbb,
            const uint32_t *__restrict__ start, const uint32_t *__restrict__ coff, const uint32_t *__restrict__ total,
            const uint32_t *__restrict__ idx, const rec16 *__restrict__ recs, uint32_t nrec,
            const replay_state st, unsigned long long *__restrict__ ctr,
            uint32_t *status)
{
    extern __shared__ uint4 smb[];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5, wpb = blockDim.x >> 5;
    const size_t per_warp = stamp_lru_bytes(cmax, nw, nbb);
    const stamp_lru X = stamp_lru_at(reinterpret_cast<unsigned char *>(smb) + per_warp * warp, cmax, nw, nbb);

    const uint32_t w = blockIdx.x * wpb + warp;
    if (w >= *total) return;
    const uint32_t s = min(coff[ns + 2 + w], ns - 1u), ci = w - coff[s];  // the item's stream and chunk
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

    // ---- state at p0, in recency order in K[0 .. fill) ------------------------------
    uint32_t fill = 0;
    sl_reindex(X, 0, lane);
    if (ci == 0) {
        // the carried-in keys, eight loads in flight per lane
        for (uint32_t q0 = 0; q0 < fill_in; q0 += 256) {
            unsigned long long kk[8];
#pragma unroll
            for (uint32_t x = 0; x < 8; ++x) {
                const uint32_t q = q0 + 32u * x + lane;
                kk[x] = q < fill_in ? kin[q] : 0ull;
            }
#pragma unroll
            for (uint32_t x = 0; x < 8; ++x) {
                const uint32_t q = q0 + 32u * x + lane;
                if (q < fill_in) {
                    X.K[q] = kk[x];
                    sl_insert(X, kk[x], q);
                }
            }
        }
        fill = fill_in;
    } else {
        // walk backwards collecting distinct keys, most recent first
        const uint32_t back = p0 - b;
        const uint32_t vtot = back + fill_in;
        for (uint32_t v0 = 0; v0 < vtot && fill < cmax; v0 += 32) {
            const uint32_t v = v0 + lane;
            const bool valid = v < vtot;
            unsigned long long key = 0;
            if (valid) key = v < back ? recs[min(idx[p0 - 1 - v], nrec - 1u)].key : kin[v - back];
            const uint32_t vm = __ballot_sync(0xffffffffu, valid);
            const uint32_t peers = __match_any_sync(0xffffffffu, key) & vm;
            const bool fresh = valid && (peers & lt) == 0 && sl_lookup(X, key, fill, cmax) == kNone;
            const uint32_t bal = __ballot_sync(0xffffffffu, fresh);
            const uint32_t pos = fill + __popc(bal & lt);
            __syncwarp();
            if (fresh && pos < cmax) {
                X.K[pos] = key;
                sl_insert(X, key, pos);
            }
            fill = min(cmax, fill + (uint32_t)__popc(bal));
            __syncwarp();
        }
    }
    __syncwarp();
    uint32_t wnow, lo;
    sl_stamps_in_order(X, fill, nw, lane, wnow, lo);

    unsigned long long my_req = 0, my_prompt = 0;
    unsigned long long my_hit[NC], my_tok[NC];
#pragma unroll
    for (int c = 0; c < NC; ++c) my_hit[c] = my_tok[c] = 0;

    // the next step's records are gathered one step early, through request
    // indices read two steps early
    rec16 ahead = {0ull, 0u, 0u};
    if (p0 + lane < p1) {
        const uint32_t ix = idx[p0 + lane];
        (void)CR_DCHECK(ix < nrec, status);
        ahead = recs[min(ix, nrec - 1u)];  // (the bound guards the gather)
    }
    uint32_t ix_next = p0 + 32u + lane < p1 ? idx[p0 + 32u + lane] : 0u;
    for (uint32_t t0 = p0; t0 < p1; t0 += 32) {
        const uint32_t cnt = (p1 - t0) < 32u ? (p1 - t0) : 32u;
        const bool valid = lane < cnt;
        const rec16 mine = ahead;
        if (t0 + 32u + lane < p1) {
            (void)CR_DCHECK(ix_next < nrec, status);
            ahead = recs[min(ix_next, nrec - 1u)];
        }
        ix_next = t0 + 64u + lane < p1 ? idx[t0 + 64u + lane] : 0u;
        if (valid) {
            my_req += 1;
            my_prompt += (unsigned long long)mine.P + mine.S;
        }
        const uint32_t vm = cnt == 32 ? 0xffffffffu : (1u << cnt) - 1u;
        const uint32_t grp = __match_any_sync(0xffffffffu, mine.key) & vm;
        const uint32_t below = grp & lt, above = grp & gt;
        const bool first = valid && below == 0;
        const bool last = valid && above == 0;
        uint32_t slot = first ? sl_lookup(X, mine.key, fill, cmax) : kNone;
        const bool res = slot != kNone;  // first occurrence of a resident key
        uint32_t s_old = res ? (uint32_t)X.ST[slot] : 0u;
        if (s_old >= 32u * nw) {  // never: stamps stay inside the window (guards the bitmap)
            atomicOr(status, CR_FLAG_INTERNAL);
            s_old = 0;
        }

        // recency position at the step's start: live stamps above the key's
        live_prefix<NG> LP;
        LP.load(X.BM, nw, lane);
        const uint32_t bl = LP.below(s_old);
        const uint32_t D = res ? fill - 1u - bl : kAbsent;
        // a first occurrence at old position D is pushed deeper by the step's earlier
        // first occurrences that were deeper or absent: between the absent ones
        // (jlo) and all of them (jhi).  Where that range straddles a capacity the
        // exact count decides the hit: those lanes (a few per step) are counted one
        // at a time against every lane; any count in the range decides the others.
        const uint32_t firstm = __ballot_sync(0xffffffffu, first);
        const uint32_t absm = __ballot_sync(0xffffffffu, first && !res);
        const uint32_t jlo = (uint32_t)__popc(absm & lt), jhi = (uint32_t)__popc(firstm & lt);
        bool amb = false;
#pragma unroll
        for (int c = 0; c < NC; ++c)
            if (c < (int)caps.n_caps && D + 1u + jlo <= caps.cap[c] && caps.cap[c] < D + 1u + jhi) amb = true;
        uint32_t jx = jhi;
        for (uint32_t am = __ballot_sync(0xffffffffu, res && amb); am; am &= am - 1u) {  // uniform
            const uint32_t a = (uint32_t)__ffs(am) - 1u;
            const uint32_t Da = __shfl_sync(0xffffffffu, D, a);
            const uint32_t deeper = __ballot_sync(0xffffffffu, first && (!res || D > Da));
            if (lane == a) jx = (uint32_t)__popc(deeper & lt);
        }
        uint32_t dep_rep = 1u;
        if (SMALL) {
            // a repeat of lane j: 1 + the distinct keys of lanes (j, i), i.e. the lanes
            // there whose key does not recur before i (next occurrence lane > i);
            // compared bit-sliced over the 6-bit next-occurrence lane; only needed
            // below capacity 32 (a repeat's depth is at most 31)
            const uint32_t next = above ? (uint32_t)__ffs(above) - 1u : 32u;
            uint32_t gN = 0, eN = 0xffffffffu;
#pragma unroll
            for (int bt = 5; bt >= 0; --bt) {
                const uint32_t BN = __ballot_sync(0xffffffffu, (next >> bt) & 1u);
                const uint32_t MN = 0u - ((lane >> bt) & 1u);
                gN |= eN & BN & ~MN;
                eN &= ~(BN ^ MN);
            }
            const uint32_t win = lt & ~((2u << (31u - (uint32_t)__clz(below | 1u))) - 1u);
            dep_rep = 1u + (uint32_t)__popc(gN & win);
        }
        const uint32_t dep_first = res ? D + 1u + jx : kNone;
        const uint32_t depth = !valid ? kNone : (first ? dep_first : dep_rep);
#pragma unroll
        for (int c = 0; c < NC; ++c) {
            if (c < (int)caps.n_caps && depth <= caps.cap[c]) {
                my_hit[c] += 1;
                my_tok[c] += mine.P;
            }
        }

        // ---- state after the step ------------------------------------------------------
        const uint32_t lastm = __ballot_sync(0xffffffffu, last);
        const uint32_t u = (uint32_t)__popc(lastm);
        const uint32_t mnew = (uint32_t)__popc(absm);
        if (SMALL && u > cmax) {
            // more distinct keys than the capacity: every old key leaves and the
            // cmax most recently used keys of the step form the cache
            __syncwarp();
            sl_reindex(X, 0, lane);
            for (uint32_t x = lane; x < nw; x += 32) X.BM[x] = 0;
            __syncwarp();
            const uint32_t rk = (uint32_t)__popc(lastm & gt);  // 0 = most recent
            const bool keep = last && rk < cmax;
            const uint32_t keepm = __ballot_sync(0xffffffffu, keep);
            if (keep) {
                const uint32_t t = wnow * 32u + lane;
                X.K[rk] = mine.key;
                sl_insert(X, mine.key, rk);
                X.ST[rk] = (uint16_t)t;
                X.T2S[t] = (uint16_t)rk;
            }
            if (lane == 0) X.BM[wnow] = keepm;
            fill = cmax;
            lo = wnow;
            ++wnow;
        } else {
            // touched keys leave their old time
            if (res) atomicAnd(&X.BM[s_old >> 5], ~(1u << (s_old & 31u)));
            __syncwarp();
            // the oldest untouched keys leave until the cache fits: the lowest live
            // bits, found 32 words at a time from the lowest word that has any
            uint32_t need = fill + mnew > cmax ? fill + mnew - cmax : 0u;
            uint32_t done = 0;
            while (need && lo < wnow) {  // each pass ends the loop or moves lo up
                const uint32_t wd = lo + lane;
                const uint32_t word = wd < wnow ? X.BM[wd] : 0u;
                const uint32_t pc = (uint32_t)__popc(word);
                const uint32_t incl = warp_incl_scan(pc, lane);
                const uint32_t tot = __shfl_sync(0xffffffffu, incl, 31);
                const uint32_t take = min(need, tot);
                uint32_t o = 0;  // the word holding this lane's bit: first lane whose prefix exceeds lane
#pragma unroll
                for (uint32_t stp = 16; stp >= 1; stp >>= 1) {
                    const uint32_t v = __shfl_sync(0xffffffffu, incl, o + stp - 1u);
                    if (v <= lane) o += stp;
                }
                const uint32_t exo = __shfl_sync(0xffffffffu, incl - pc, o & 31u);
                const uint32_t wo = __shfl_sync(0xffffffffu, word, o & 31u);
                const uint32_t olast = __shfl_sync(0xffffffffu, o, (take + 31u) & 31u);
                __syncwarp();
                if (lane < take) {
                    const uint32_t bit = nth_set_bit(wo, lane - exo);
                    uint32_t q = X.T2S[(lo + o) * 32u + bit];
                    atomicAnd(&X.BM[lo + o], ~(1u << bit));
                    if (q < cmax) {
                        sl_erase(X, q);
                    } else {  // never: a live time always maps to a slot (guards the arrays)
                        atomicOr(status, CR_FLAG_INTERNAL);
                        q = 0;
                    }
                    X.EV[done + lane] = (uint16_t)q;
                }
                lo = take == tot ? min(lo + 32u, wnow) : lo + olast;
                need -= take;
                done += take;
                __syncwarp();
            }
            // new keys take the never-used slots, then the freed ones
            if (first && !res) {
                const uint32_t a = (uint32_t)__popc(absm & lt);
                const uint32_t freecnt = cmax - fill;
                const uint32_t q = a < freecnt ? fill + a : (uint32_t)X.EV[a - freecnt];
                X.K[q] = mine.key;
                sl_insert(X, mine.key, q);
                slot = q;
            }
            // every key of the step takes the time of its last access
            const uint32_t fl = (uint32_t)__ffs(grp ? grp : 1u) - 1u;
            const uint32_t ks = __shfl_sync(0xffffffffu, slot, fl);
            if (last) {
                const uint32_t t = wnow * 32u + lane;
                X.ST[ks] = (uint16_t)t;
                X.T2S[t] = (uint16_t)ks;
            }
            if (lane == 0) X.BM[wnow] = lastm;
            fill = min(cmax, fill + mnew);
            ++wnow;
        }
        __syncwarp();
        if (wnow == nw) sl_compact<NG>(X, fill, nw, lane, wnow, lo);
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
        live_prefix<NG> LP;
        LP.load(X.BM, nw, lane);
        for (uint32_t q0 = 0; q0 < fill; q0 += 32) {
            const uint32_t q = q0 + lane;
            const uint32_t nb = LP.below(q < fill ? (uint32_t)X.ST[q] : 0u);
            if (q < fill && nb < fill) kout[fill - 1u - nb] = X.K[q];
        }
        if (lane == 0) st.fill_out[s] = fill;
    }
}

// Words of the stamp window: the cmax stamps a compaction leaves plus at least
// as many steps (and at least 8) before the next one.
inline uint32_t stamp_words(uint32_t cmax)
{
    const uint32_t w0 = (cmax + 31) / 32;
    return w0 + (w0 > 8 ? w0 : 8);
}

template <int NC, int NG, bool SMALL>
int launch_stamp(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                 const uint32_t *coff, const uint32_t *total, uint64_t m, const uint32_t *idx,
                 const rec16 *recs, uint64_t *d_ctr)
{
    const uint32_t cmax = rp->cmax, nw = stamp_words(cmax);
    // warps per block: the most warps per SM that shared memory allows (at most 32
    // blocks and 64 warps per SM, and what the registers allow)
    const size_t sm_bytes = 227 * 1024;
    cudaFuncAttributes fa;
    uint32_t warps_regs = 64;
    if (cudaFuncGetAttributes(&fa, k_lru_stamp<NC, NG, SMALL>) == cudaSuccess && fa.numRegs > 0)
        warps_regs = 65536u / ((((uint32_t)fa.numRegs * 32u + 255u) / 256u) * 256u);
    else
        cudaGetLastError();
    auto fit = [&](uint32_t nb_bits, uint32_t *wpb_out) {
        const size_t pw = stamp_lru_bytes(cmax, nw, nb_bits);
        uint32_t best = 0;
        for (uint32_t x = 4; x >= 1; --x) {
            const size_t blk = pw * x + 1024;
            uint32_t nb = blk <= sm_bytes ? (uint32_t)(sm_bytes / blk) : 0u;
            nb = nb < 32u ? nb : 32u;
            nb = nb < warps_regs / x ? nb : warps_regs / x;
            const uint32_t wps = nb * x < 64u ? nb * x : 64u;
            if (wps > best) {
                best = wps;
                *wpb_out = x;
            }
        }
        return best;
    };
    // index buckets: one per resident key at most (a quarter of the entries live); half
    // as many (half the entries live: a few more probes and inserts) when that fits more
    // warps on an SM, i.e. when the state of the largest capacities bounds the occupancy
    uint32_t nbb = 4;
    while ((1u << nbb) < cmax) ++nbb;
    uint32_t wpb = 1, wpb_half = 1;
    const uint32_t w_full = fit(nbb, &wpb);
    if (nbb > 4 && fit(nbb - 1, &wpb_half) * 10u >= w_full * 11u) {  // at least 10% more warps
        --nbb;
        wpb = wpb_half;
    }
    const size_t per_warp = stamp_lru_bytes(cmax, nw, nbb);
    const size_t smem = per_warp * wpb;
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_stamp<NC, NG, SMALL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)smem));
    const uint32_t ns = rp->n_rep * rp->R;
    const uint64_t items = (uint64_t)ns + (m + CL - 1) / CL;  // upper bound on work items
    replay_state st;
    st.keys_in = rp->d_keys[rp->cur];
    st.fill_in = rp->d_fill[rp->cur];
    st.keys_out = rp->d_keys[rp->cur ^ 1];
    st.fill_out = rp->d_fill[rp->cur ^ 1];
    const int pr = cr_prof_begin(ctx, ctx->stream, CR_PROF_REPLAY);
    CR_LAUNCH(ctx, (k_lru_stamp<NC, NG, SMALL>), (unsigned int)((items + wpb - 1) / wpb), wpb * 32, smem, caps, cmax,
              nw, rp->R, ns, CL, nbb, start, coff, total, idx, recs, (uint32_t)(m / rp->n_rep), st,
              (unsigned long long *)d_ctr,
              ctx->d_status);
    cr_prof_end(ctx, ctx->stream, pr);
    rp->cur ^= 1;
    return CR_OK;
}

template <int NC>
int launch_stamp_nc(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                    const uint32_t *coff, const uint32_t *total, uint64_t m, const uint32_t *idx,
                 const rec16 *recs, uint64_t *d_ctr)
{
    uint32_t cmin = 0xffffffffu;
    for (uint32_t c = 0; c < caps.n_caps; ++c) cmin = caps.cap[c] < cmin ? caps.cap[c] : cmin;
    const bool small = cmin < 32;  // a repeat within a step can miss only below capacity 32
    if (stamp_words(rp->cmax) <= 32)
        return small ? launch_stamp<NC, 1, true>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr)
                     : launch_stamp<NC, 1, false>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr);
    return small ? launch_stamp<NC, 2, true>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr)
                 : launch_stamp<NC, 2, false>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr);
}

int launch_batch(cr_ctx *ctx, cr_replay *rp, const replay_caps &caps, uint32_t CL, const uint32_t *start,
                 const uint32_t *coff, const uint32_t *total, uint64_t m, const uint32_t *idx,
                 const rec16 *recs, uint64_t *d_ctr)
{
    if (caps.n_caps == 1) return launch_stamp_nc<1>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr);
    if (caps.n_caps <= 3) return launch_stamp_nc<3>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr);
    return launch_stamp_nc<CR_MAX_CAPS>(ctx, rp, caps, CL, start, coff, total, m, idx, recs, d_ctr);
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

struct token_state {
    const unsigned long long *keys_in;  // [stream][kTokMax], most recent first
    const uint32_t *cum_in;             // [stream][kTokMax], tokens of entries 0..j
    const uint32_t *fill_in;
    unsigned long long *keys_out;
    uint32_t *cum_out;
    uint32_t *fill_out;
};

__global__ void __launch_bounds__(kTokWarps * 32) k_lru_tokens(const __grid_constant__ replay_caps caps, uint32_t ns,
                                                               uint32_t R, uint32_t CL, const uint32_t *__restrict__ start,
                                                               const uint32_t *__restrict__ coff,
                                                               const uint32_t *__restrict__ total,
                                                               const uint32_t *__restrict__ idx,
                                                               const rec16 *__restrict__ recs, uint32_t nrec,
                                                               const token_state st,
                                                               unsigned long long *__restrict__ ctr, uint32_t *status)
{
    extern __shared__ unsigned long long tok_sh[];
    const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const uint32_t wi = blockIdx.x * kTokWarps + w;
    if (wi >= *total) return;  // whole warps only; the kernel has no block-wide barrier
    // work item -> (stream, chunk)
    const uint32_t s = min(coff[ns + 2 + wi], ns - 1u), ci = wi - coff[s];
    const uint32_t b = start[s], e = start[s + 1];
    unsigned long long *K = tok_sh + (size_t)w * kTokMax;
    uint32_t *Cm = reinterpret_cast<uint32_t *>(tok_sh + (size_t)kTokWarps * kTokMax) + (size_t)w * kTokMax;
    uint32_t capmax = 0;
    for (uint32_t c = 0; c < caps.n_caps; ++c) capmax = caps.cap[c] > capmax ? caps.cap[c] : capmax;
    const uint32_t mycap = lane < caps.n_caps ? caps.cap[lane] : 0u;
    const uint32_t fin = st.fill_in[s];
    const unsigned long long *kin = st.keys_in + (size_t)s * kTokMax;
    const uint32_t *cin = st.cum_in + (size_t)s * kTokMax;
    if (b == e) {  // nothing routed here: carry the state over unchanged
        for (uint32_t j = lane; j < fin; j += 32) {
            st.keys_out[(size_t)s * kTokMax + j] = kin[j];
            st.cum_out[(size_t)s * kTokMax + j] = cin[j];
        }
        if (lane == 0) st.fill_out[s] = fin;
        return;
    }
    const uint32_t i0 = b + ci * CL;
    const uint32_t i1 = (e - i0) < CL ? e : i0 + CL;
    uint32_t f = 0;
    if (ci == 0) {
        f = fin;
        for (uint32_t j = lane; j < f; j += 32) {
            K[j] = kin[j];
            Cm[j] = cin[j];
        }
    } else {
        // the state at i0 is the longest run of most recent distinct prefixes that fits
        // (tokens <= the largest capacity, at most kTokMax of them): walk back over the
        // stream, then over the carried-in list, keeping each key's most recent access
        const uint32_t back = i0 - b;
        uint32_t tot = 0;
        bool stop = false;
        for (uint32_t v0 = 0; v0 < back + fin && !stop; v0 += 32) {
            const uint32_t v = v0 + lane;
            unsigned long long ck = 0;
            uint32_t cp = 0;
            if (v < back) {
                const rec16 rr = recs[min(idx[i0 - 1 - v], nrec - 1u)];
                ck = rr.key;
                cp = rr.P;
            } else if (v < back + fin) {
                const uint32_t j = v - back;
                ck = kin[j];
                cp = cin[j] - (j ? cin[j - 1] : 0u);
            }
            const uint32_t nb = min(32u, back + fin - v0);
            for (uint32_t q = 0; q < nb; ++q) {  // uniform over the warp
                const unsigned long long x = __shfl_sync(0xffffffffu, ck, q);
                const uint32_t P = __shfl_sync(0xffffffffu, cp, q);
                bool seen = false;
                for (uint32_t c0 = 0; c0 < f && !seen; c0 += 32)
                    seen = __ballot_sync(0xffffffffu, c0 + lane < f && K[c0 + lane] == x) != 0;
                if (seen) continue;
                const unsigned long long nt = (unsigned long long)tot + P;
                if (f == kTokMax || nt > capmax) {  // the first distinct prefix that does not fit ends the run
                    stop = true;
                    break;
                }
                tot = (uint32_t)nt;
                if (lane == 0) {
                    K[f] = x;
                    Cm[f] = tot;
                }
                ++f;
                __syncwarp();
            }
        }
    }
    __syncwarp();
    unsigned long long kr = 0;  // register list: entry `lane`
    uint32_t cr = 0;
    bool inreg = f <= 32;
    if (inreg && lane < f) {
        kr = K[lane];
        cr = Cm[lane];
    }
    __syncwarp();
    unsigned long long c_hit = 0, c_hit_tok = 0, c_prompt = 0;  // lane = capacity (prompt: every lane)
    rec16 nx = {0ull, 0u, 0u};
    if (i0 + lane < i1) nx = recs[min(idx[i0 + lane], nrec - 1u)];
    for (uint32_t b0 = i0; b0 < i1; b0 += 32) {
        const rec16 cur = nx;
        if (b0 + 32 + lane < i1) nx = recs[min(idx[b0 + 32 + lane], nrec - 1u)];  // next 32 in flight
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
    if (i1 == e) {  // the stream's last chunk hands the state to the next call
        if (inreg) {
            if (lane < f) {
                st.keys_out[(size_t)s * kTokMax + lane] = kr;
                st.cum_out[(size_t)s * kTokMax + lane] = cr;
            }
        } else {
            for (uint32_t j = lane; j < f; j += 32) {
                st.keys_out[(size_t)s * kTokMax + j] = K[j];
                st.cum_out[(size_t)s * kTokMax + j] = Cm[j];
            }
        }
        if (lane == 0) st.fill_out[s] = f;
    }
    for (int o = 16; o > 0; o >>= 1) c_prompt += __shfl_xor_sync(0xffffffffu, c_prompt, o);
    if (lane < caps.n_caps) {
        const uint32_t rep = s / R, r = s - rep * R;
        unsigned long long *C = ctr + (((unsigned long long)rep * caps.n_caps + lane) * R + r) * CR_CTR_FIELDS;
        atomicAdd(&C[0], (unsigned long long)(i1 - i0));
        if (c_hit) atomicAdd(&C[1], c_hit);
        if (c_hit_tok) atomicAdd(&C[2], c_hit_tok);
        atomicAdd(&C[3], c_prompt);
        atomicAdd(&C[4], c_prompt - c_hit_tok);
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
    for (int x = 0; x < 2; ++x) {  // double-buffered: chunks of a stream read the old state
        if (cudaMalloc(&rp->d_keys[x], rp->n_streams * kTokMax * sizeof(unsigned long long)) != cudaSuccess ||
            cudaMalloc(&rp->d_size[x], rp->n_streams * kTokMax * sizeof(uint32_t)) != cudaSuccess ||
            cudaMalloc(&rp->d_fill[x], rp->n_streams * sizeof(uint32_t)) != cudaSuccess) {
            cudaGetLastError();
            cr_replay_destroy(ctx, rp);
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
    for (int b = 0; b < 2; ++b)
        if (rp->d_size[b]) cudaFree(rp->d_size[b]);
    free(rp);
    return CR_OK;
}

// ---- a8 / a9 as separate calls --------------------------------------------------
// A partitioned input: every (replica, destination) stream's request indices in
// arrival order, the packed records, the streams' starts and their chunking.
struct cr_replay_input {
    uint32_t n_rep, R, tokens;   // shape of the replay it was built for
    uint32_t CL;                 // chunk length of the work items
    uint64_t n, m;               // requests, (request, replica) pairs
    uint32_t ns, ntiles;
    uint32_t *d_idx;             // [m]
    rec16 *d_recs;               // [n]
    uint32_t *d_cnt;             // [ns * ntiles + 2]: tile counts -> offsets, and their total
    uint32_t *d_start;           // [ns + 1]
    uint32_t *d_coff;            // [ns + 2 + items]: work-item offsets, their total, then each item's stream
    uint64_t cap_m, cap_n, cap_cnt, cap_ns, cap_coff;
};

static int grow_u32(cr_ctx *ctx, uint32_t **p, uint64_t *cap, uint64_t need)
{
    if (*cap >= need && *p) return CR_OK;
    if (*p) {
        // the old buffer may still be read by work on any stream (a simulation ordered after
        // the partition by an event): wait for the whole device before freeing it
        CR_CUDA(ctx, cudaDeviceSynchronize());
        cudaFree(*p);
        *p = nullptr;
    }
    const uint64_t c = need + need / 4 + 64;
    if (cudaMalloc((void **)p, c * sizeof(uint32_t)) != cudaSuccess) {
        cudaGetLastError();
        *cap = 0;
        return cr_fail(ctx, CR_ENOMEM, "replay input: cannot allocate %llu words", (unsigned long long)c);
    }
    *cap = c;
    return CR_OK;
}

extern "C" int cr_replay_input_create(cr_ctx *ctx, cr_replay_input **out)
{
    if (!ctx || !out) return CR_EINVAL;
    *out = (cr_replay_input *)calloc(1, sizeof(cr_replay_input));
    return *out ? CR_OK : cr_fail(ctx, CR_ENOMEM, "replay input: host allocation failed");
}

extern "C" int cr_replay_input_destroy(cr_ctx *ctx, cr_replay_input *in)
{
    if (!in) return CR_OK;
    if (ctx) cudaStreamSynchronize(ctx->stream);
    cudaFree(in->d_idx);
    cudaFree(in->d_recs);
    cudaFree(in->d_cnt);
    cudaFree(in->d_start);
    cudaFree(in->d_coff);
    free(in);
    return CR_OK;
}

extern "C" int cr_replay_partition(cr_ctx *ctx, const cr_replay *rp, const uint64_t *d_key, const uint32_t *d_plen,
                                   const uint32_t *d_slen, const uint16_t *d_dest, uint64_t n, cr_replay_input *in)
{
    if (!ctx || !rp || !in) return CR_EINVAL;
    cr_nvtx_range nv("cr_replay_partition");
    const uint64_t m = n * rp->n_rep;
    if (n >= (1ull << 31) || m >= 0xffffffffull)
        return cr_fail(ctx, CR_EINVAL, "cr_replay_partition: n * n_rep must be < 2^32 - 1");
    if (n && (!d_key || !d_plen || !d_slen || !d_dest))
        return cr_fail(ctx, CR_EINVAL, "cr_replay_partition: NULL pointer");
    const uint32_t R = rp->R, ns = (uint32_t)rp->n_streams;
    const uint32_t ntiles = (uint32_t)((n + kPartTile - 1) / kPartTile);
    const uint64_t ncnt = (uint64_t)ns * ntiles;
    if (ncnt >= 0xffffffffull) return cr_fail(ctx, CR_EINVAL, "cr_replay_partition: too many (stream, tile) pairs");
    in->n_rep = rp->n_rep;
    in->R = R;
    in->tokens = (uint32_t)rp->tokens;
    in->n = n;
    in->m = m;
    in->ns = ns;
    in->ntiles = ntiles;
    if (rp->tokens) {
        uint32_t capmax = 0;
        for (uint32_t c = 0; c < rp->n_caps; ++c) capmax = rp->caps[c] > capmax ? rp->caps[c] : capmax;
        // chunks long against the rebuild walk, which reaches back until the largest capacity fills
        in->CL = capmax <= (1u << 16) ? 1024u : (capmax <= (1u << 17) ? 4096u : 16384u);
    } else {
        // long enough that rebuilding an LRU state of cmax entries is amortised
        in->CL = rp->cmax * 16u > 256u ? rp->cmax * 16u : 256u;
    }
    if (n == 0) return CR_OK;
    CR_TRY(grow_u32(ctx, &in->d_idx, &in->cap_m, m));
    CR_TRY(grow_u32(ctx, (uint32_t **)&in->d_recs, &in->cap_n, n * (sizeof(rec16) / sizeof(uint32_t))));
    CR_TRY(grow_u32(ctx, &in->d_cnt, &in->cap_cnt, ncnt + 2));
    CR_TRY(grow_u32(ctx, &in->d_start, &in->cap_ns, (uint64_t)ns + 2));
    const uint64_t items_max = (uint64_t)ns + m / in->CL + 1;  // every stream's chunks, at least one each
    CR_TRY(grow_u32(ctx, &in->d_coff, &in->cap_coff, (uint64_t)ns + 2 + items_max));
    uint32_t *cnt = in->d_cnt, *nrec = cnt + ncnt, *start = in->d_start;
    uint32_t *coff = in->d_coff, *total = coff + ns;
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    const dim3 pgrid(ntiles, rp->n_rep);
    const size_t csmem = (size_t)R * sizeof(uint32_t), ssmem = part_scatter_smem(R);
    if (csmem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_part_count, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)csmem));
    if (ssmem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_part_scatter, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ssmem));
    const int pp = cr_prof_begin(ctx, ctx->stream, CR_PROF_PARTITION);
    CR_LAUNCH(ctx, k_part_records, cr_blocks(n, 256, gcap), 256, 0, (const unsigned long long *)d_key, d_plen, d_slen,
              (unsigned long long)n, in->d_recs);
    CR_LAUNCH(ctx, k_part_count, pgrid, kPartBlock, csmem, d_dest, (unsigned long long)n, R, ntiles, cnt,
              ctx->d_status);
    CR_TRY(cr_scan_u32(ctx, cnt, cnt, ncnt, nrec));
    CR_LAUNCH(ctx, k_part_starts, cr_blocks((uint64_t)ns + 1, 256, gcap), 256, 0, (const uint32_t *)cnt, ns, ntiles,
              (const uint32_t *)nrec, start);
    CR_LAUNCH(ctx, k_part_scatter, pgrid, kPartBlock, ssmem, d_dest, (unsigned long long)n, R, ntiles,
              (const uint32_t *)cnt, in->d_idx, (unsigned long long)m);
    CR_LAUNCH(ctx, k_chunk_counts, cr_blocks(ns, 256, gcap), 256, 0, (const uint32_t *)start, ns, in->CL, coff);
    CR_TRY(cr_scan_u32(ctx, coff, coff, ns, total));
    CR_LAUNCH(ctx, k_item_streams, cr_blocks(ns, 256, gcap), 256, 0, (const uint32_t *)coff, ns, coff + ns + 2,
              items_max);
    cr_prof_end(ctx, ctx->stream, pp);
    return CR_OK;
}

extern "C" int cr_replay_simulate(cr_ctx *ctx, cr_replay *rp, const cr_replay_input *in, uint64_t *d_ctr)
{
    if (!ctx || !rp || !in) return CR_EINVAL;
    cr_nvtx_range nv("cr_replay_simulate");
    if (in->n_rep != rp->n_rep || in->R != rp->R || in->tokens != (uint32_t)rp->tokens)
        return cr_fail(ctx, CR_EINVAL, "cr_replay_simulate: the input was partitioned for another replay shape");
    if (in->n == 0) return CR_OK;
    if (!d_ctr) return cr_fail(ctx, CR_EINVAL, "cr_replay_simulate: d_ctr is NULL");
    const uint32_t R = rp->R, ns = in->ns;
    const uint64_t m = in->m, n = in->n;
    const uint32_t *start = in->d_start, *coff = in->d_coff, *total = in->d_coff + ns;
    replay_caps caps;
    caps.n_caps = rp->n_caps;
    for (uint32_t c = 0; c < CR_MAX_CAPS; ++c) caps.cap[c] = c < rp->n_caps ? rp->caps[c] : 0;
    if (rp->tokens) {
        // token-weighted: one warp per (stream, chunk), its list in registers or shared memory
        const uint32_t TCL = in->CL;
        const size_t tsmem = (size_t)kTokWarps * kTokMax * (sizeof(unsigned long long) + sizeof(uint32_t));
        if (tsmem > 48 * 1024)
            CR_CUDA(ctx, cudaFuncSetAttribute(k_lru_tokens, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tsmem));
        token_state tst;
        tst.keys_in = rp->d_keys[rp->cur];
        tst.cum_in = rp->d_size[rp->cur];
        tst.fill_in = rp->d_fill[rp->cur];
        tst.keys_out = rp->d_keys[rp->cur ^ 1];
        tst.cum_out = rp->d_size[rp->cur ^ 1];
        tst.fill_out = rp->d_fill[rp->cur ^ 1];
        const uint64_t items = (uint64_t)ns + (m + TCL - 1) / TCL;  // upper bound on work items
        const int pt = cr_prof_begin(ctx, ctx->stream, CR_PROF_REPLAY);
        CR_LAUNCH(ctx, k_lru_tokens, (unsigned int)((items + kTokWarps - 1) / kTokWarps), kTokWarps * 32, tsmem,
                  caps, ns, R, TCL, start, coff, total, (const uint32_t *)in->d_idx, (const rec16 *)in->d_recs,
                  (uint32_t)n, tst, (unsigned long long *)d_ctr, ctx->d_status);
        cr_prof_end(ctx, ctx->stream, pt);
        rp->cur ^= 1;
        return CR_OK;
    }
    return launch_batch(ctx, rp, caps, in->CL, start, coff, total, m, in->d_idx, in->d_recs, d_ctr);
}

extern "C" int cr_shadow_replay(cr_ctx *ctx, cr_replay *rp, const uint64_t *d_key, const uint32_t *d_plen,
                                const uint32_t *d_slen, const uint16_t *d_dest, uint64_t n, uint64_t *d_ctr)
{
    if (!ctx || !rp) return CR_EINVAL;
    cr_nvtx_range nv("cr_shadow_replay");
    if (n == 0) return CR_OK;
    if (!d_key || !d_plen || !d_slen || !d_dest || !d_ctr)
        return cr_fail(ctx, CR_EINVAL, "cr_shadow_replay: NULL pointer");
    if (!ctx->replay_in) CR_TRY(cr_replay_input_create(ctx, &ctx->replay_in));
    CR_TRY(cr_replay_partition(ctx, rp, d_key, d_plen, d_slen, d_dest, n, ctx->replay_in));
    return cr_replay_simulate(ctx, rp, ctx->replay_in, d_ctr);
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

extern "C" int cr_replay_import_state(cr_ctx *ctx, cr_replay *rp, uint32_t rep, uint32_t r, const uint64_t *keys,
                                      uint32_t fill)
{
    if (!ctx || !rp || (fill && !keys)) return CR_EINVAL;
    if (rp->tokens) return cr_fail(ctx, CR_EINVAL, "import_state: token-weighted replays keep prefix sizes too");
    if (rep >= rp->n_rep || r >= rp->R) return cr_fail(ctx, CR_EINVAL, "import_state: bad stream");
    if (fill > rp->cmax) return cr_fail(ctx, CR_EINVAL, "import_state: %u keys exceed capacity %u", fill, rp->cmax);
    // the keys of one LRU are distinct
    uint64_t *tmp = (uint64_t *)malloc((size_t)(fill ? fill : 1) * sizeof(uint64_t));
    if (!tmp) return cr_fail(ctx, CR_ENOMEM, "import_state: host allocation failed");
    memcpy(tmp, keys, (size_t)fill * sizeof(uint64_t));
    qsort(tmp, fill, sizeof(uint64_t), [](const void *a, const void *b) {
        const uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
        return x < y ? -1 : (x > y ? 1 : 0);
    });
    int dup = 0;
    for (uint32_t i = 1; i < fill; ++i) dup |= tmp[i] == tmp[i - 1];
    free(tmp);
    if (dup) return cr_fail(ctx, CR_EINVAL, "import_state: a key is listed twice");
    const uint64_t s = (uint64_t)rep * rp->R + r;
    if (fill)
        CR_CUDA(ctx, cudaMemcpyAsync(rp->d_keys[rp->cur] + s * rp->cmax, keys, (size_t)fill * sizeof(uint64_t),
                                     cudaMemcpyHostToDevice, ctx->stream));
    CR_CUDA(ctx, cudaMemcpyAsync(rp->d_fill[rp->cur] + s, &fill, sizeof(uint32_t), cudaMemcpyHostToDevice,
                                 ctx->stream));
    return cr_sync(ctx);  // blocking: the host arrays may be reused when the call returns
}
