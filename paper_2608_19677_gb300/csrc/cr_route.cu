// a7: batched dispatch (cr_route_batch) and the ring of the bounded-load
// comparison policy (cr_ring_*).
//
// Two passes.  k_route_cand runs over every (replica, request) pair at once and
// does all the work that does not depend on the live load: the table probe,
// the Philox draws of power-of-two choices, the ring position of consistent
// hashing with bounded loads, round robin and the jump hash.  Round-robin and
// hash replicas are then finished (their loads are counted by k_route_count);
// every other replica leaves one packed candidate per request.  The
// load-dependent pass then walks each replica's requests in arrival order:
//   - batches longer than a warp: k_route_resolve, one CTA per replica that
//     holds the live load in shared memory; a batch is resolved by all its
//     threads against the batch-start loads, the batch's counts accumulate in
//     a second shared vector and are merged at the boundary;
//   - batches of at most 32 requests (batch_B = 1 is exact sequential
//     dispatch): k_route_resolve_warp, one warp per replica taking
//     S = floor(32 / B) * B requests (whole batches) per step.  Inside a step a
//     request's decision depends on the destinations of the earlier batches of
//     the step; the warp finds them by fixed-point iteration: every lane
//     decides from the step-start loads plus the lanes of earlier batches that
//     currently sit on each candidate (a per-destination lane bitmask in
//     shared memory), until no lane changes.  After iteration t the first t
//     batches are final, so at most S iterations are needed and typically two
//     or three; the result is the sequential one.
#include <stdlib.h>
#include <string.h>

#include <algorithm>

#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

constexpr int kRouteBlock = 1024;
constexpr uint32_t kEmpty = 0xffffffffu;
constexpr size_t kSmemBudget = 200 * 1024;  // dynamic shared memory a resolve CTA may take

// 48 bytes: a replica uses either a plan (CACHEROUTE-type) or a ring (CHWBL).
struct route_desc {
    uint32_t policy;
    int32_t tbits;                    // log2 table slots (plan policies)
    unsigned long long seed;
    union {
        const cr_table_slot *table;      // plan
        const unsigned long long *rpoint;  // ring points
    };
    union {
        const uint16_t *members;         // plan: member lists
        const uint16_t *rowner;          // ring: owner of each point
    };
    union {
        const unsigned long long *n_members;  // plan, device: the sum of k_b
        const uint32_t *rdir;                 // ring: start directory
    };
    uint32_t rM;                      // ring points
    int32_t rdbits;                   // log2 directory entries
};
static_assert(sizeof(route_desc) == 48, "route_desc layout");

struct route_args {
    route_desc d[CR_MAX_REPLICAS];
    uint32_t dep[CR_MAX_REPLICAS];    // load-dependent replicas, one CTA each in the resolve pass
    uint32_t cand[CR_MAX_REPLICAS];   // candidate pass: replica order, costliest policy first
    uint32_t rr_b0[CR_MAX_REPLICAS];  // round robin: (g0 + seed) mod 2^64 mod R
    unsigned long long rr_wrap[CR_MAX_REPLICAS];  // round robin: first i where g0 + seed + i wraps (~0: never)
};

// Candidate encoding, one u32 per (replica, request):
//   kind 0 FIXED  bits 0..15  destination (RR, HASH, and keys with k_b = 1)
//   kind 1 PAIR   bits 0..12  d1, bits 13..25 d2 (power-of-two choices; R <= 8192)
//   kind 2 SET    bits 0..29  table slot of a key with k_b > 1
//   kind 3 RING   bits 0..29  first ring index at or after the key's position
constexpr uint32_t kFixed = 0u << 30, kPair = 1u << 30, kSet = 2u << 30, kRing = 3u << 30,
                   kKindMask = 3u << 30, kLow30 = 0x3fffffffu;

__device__ __forceinline__ uint32_t p2c_pair(unsigned long long seed, uint32_t policy, unsigned long long g,
                                             uint32_t R)
{
    cr_u64x4 u = cr_philox4x64_10(g, 0ull, 0ull, 0ull, seed, (unsigned long long)policy);
    uint32_t d1 = cr_scale(u.x, R);
    uint32_t d2 = d1 + 1u + cr_scale(u.y, (unsigned long long)(R - 1));  // < 2R: one subtraction is mod R
    if (d2 >= R) d2 -= R;
    return kPair | d1 | (d2 << 13);
}

// First ring index whose point is >= h, wrapping to 0 past the last point.
__device__ __forceinline__ uint32_t ring_start(const route_desc &rd, unsigned long long h)
{
    uint32_t j = rd.rdir[h >> (64 - rd.rdbits)];
    while (j < rd.rM && rd.rpoint[j] < h) ++j;
    return j == rd.rM ? 0u : j;
}

// ceil(5 (m + 1) / (4 R)): the per-destination bound at epsilon = 1/4.
__device__ __forceinline__ unsigned long long chwbl_cap(unsigned long long m, uint32_t R)
{
    const unsigned long long den = 4ull * R;
    return (5ull * (m + 1ull) + den - 1ull) / den;
}

// Everything that does not depend on the live load, for every (replica, request).
// A warp takes 32 consecutive requests, reads their keys once and computes the
// candidates of the replicas of its group for them (blockIdx.y = group g of
// gridDim.y: replicas args.cand[g], args.cand[g + G], ..., so every group mixes
// costly and cheap policies; one group when the requests alone fill the GPU);
// round robin and sticky-hash replicas write their destinations directly.
// Plan replicas' table misses queue per warp in shared memory, and the warp draws
// their power-of-two choices 32 at a time, so the Philox rounds run with every lane
// busy.
__global__ void __launch_bounds__(256) k_route_cand(const __grid_constant__ route_args args, uint32_t n_rep,
                                                    const unsigned long long *__restrict__ keys,
                                                    unsigned long long n, unsigned long long g0, uint32_t R,
                                                    uint32_t *__restrict__ cand, uint16_t *__restrict__ dest)
{
    __shared__ unsigned long long q_req[256 / 32][64];  // replica << 40 | request
    const uint32_t lane = threadIdx.x & 31u, lt = (1u << lane) - 1u;
    unsigned long long *Q = q_req[threadIdx.x >> 5];
    uint32_t qn = 0;  // queued, < 32 between rounds
    const unsigned long long stride = (unsigned long long)gridDim.x * blockDim.x;
    for (unsigned long long wb = (unsigned long long)blockIdx.x * blockDim.x + (threadIdx.x & ~31u); wb < n;
         wb += stride) {  // uniform over the warp
        const unsigned long long i = wb + lane;
        const bool valid = i < n;
        const unsigned long long key = valid ? keys[i] : 0ull;
        for (uint32_t x = blockIdx.y; x < n_rep; x += gridDim.y) {  // uniform
            const uint32_t rep = args.cand[x];
            const route_desc &rd = args.d[rep];
            const unsigned long long o = (unsigned long long)rep * n + i;
            switch (rd.policy) {
            case CR_POLICY_RR:
                // (g0 + i + seed) mod 2^64 mod R: before the sum wraps, (b0 + i mod R) mod R
                if (valid) {
                    uint32_t r;
                    if (i < args.rr_wrap[rep] && i < (1ull << 32)) {
                        r = args.rr_b0[rep] + (uint32_t)i % R;
                        if (r >= R) r -= R;
                    } else {
                        r = (uint32_t)((g0 + rd.seed + i) % R);
                    }
                    dest[o] = (uint16_t)r;
                }
                break;
            case CR_POLICY_HASH:
                if (valid) dest[o] = (uint16_t)cr_jump_hash(cr_fmix64(key ^ rd.seed), R);
                break;
            case CR_POLICY_P2C:
                if (valid) cand[o] = p2c_pair(rd.seed, rd.policy, g0 + i, R);
                break;
            case CR_POLICY_CHWBL:
                if (valid) cand[o] = kRing | ring_start(rd, cr_fmix64(key ^ rd.seed));
                break;
            default: {
                uint32_t c = 0xffffffffu;
                if (valid) {
                    const unsigned long long mask = (1ull << rd.tbits) - 1ull;
                    unsigned long long sl = key >> (64 - rd.tbits);
                    for (;;) {
                        const cr_table_slot slot = rd.table[sl];
                        if (slot.koff == kEmpty) break;
                        if (slot.key == key) {
                            c = slot.k == 1 ? (kFixed | slot.m0) : (kSet | (uint32_t)sl);
                            break;
                        }
                        sl = (sl + 1) & mask;
                    }
                    if (c != 0xffffffffu) cand[o] = c;
                }
                const bool miss = valid && c == 0xffffffffu;
                const uint32_t mm = __ballot_sync(0xffffffffu, miss);
                if (miss) Q[qn + (uint32_t)__popc(mm & lt)] = ((unsigned long long)rep << 40) | i;
                qn += (uint32_t)__popc(mm);
                __syncwarp();
                if (qn >= 32u) {
                    const unsigned long long e = Q[qn - 32u + lane];
                    const uint32_t er = (uint32_t)(e >> 40);
                    const unsigned long long j = e & ((1ull << 40) - 1ull);
                    cand[(unsigned long long)er * n + j] = p2c_pair(args.d[er].seed, args.d[er].policy, g0 + j, R);
                    qn -= 32u;
                    __syncwarp();
                }
            }
            }
        }
    }
    if (lane < qn) {
        const unsigned long long e = Q[lane];
        const uint32_t er = (uint32_t)(e >> 40);
        const unsigned long long j = e & ((1ull << 40) - 1ull);
        cand[(unsigned long long)er * n + j] = p2c_pair(args.d[er].seed, args.d[er].policy, g0 + j, R);
    }
}

// Live-load counts of the load-independent replicas.
__global__ void __launch_bounds__(256) k_route_count(const uint16_t *__restrict__ dest, unsigned long long n,
                                                     uint32_t R, unsigned long long *__restrict__ load)
{
    extern __shared__ uint32_t hist[];
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) hist[r] = 0;
    __syncthreads();
    const uint16_t *D = dest + (unsigned long long)blockIdx.y * n;
    for (unsigned long long i = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (unsigned long long)gridDim.x * blockDim.x)
        atomicAdd(&hist[D[i]], 1u);
    __syncthreads();
    unsigned long long *L = load + (unsigned long long)blockIdx.y * R;
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x)
        if (hist[r]) atomicAdd(&L[r], (unsigned long long)hist[r]);
}

// Walk the ring from index j for the first owner whose load is below cap.
// The least-loaded destination always is, so the walk ends within M steps
// unless the load sum has wrapped; then the first owner is taken and the
// overflow flag raised.
template <typename LoadOf>
__device__ __forceinline__ uint32_t ring_walk(const route_desc &rd, const uint16_t *own, uint32_t j,
                                              unsigned long long cap, LoadOf load_of, uint32_t *status)
{
    const uint32_t j0 = j;
    for (uint32_t t = 0; t < rd.rM; ++t) {
        const uint32_t d = own[j];
        if (load_of(d) < cap) return d;
        j = (j + 1 == rd.rM) ? 0u : j + 1;
    }
    atomicOr(status, CR_FLAG_OVERFLOW);
    return own[j0];
}

// Least-loaded member of T(b) = mem[off .. off + k), first member m0 given;
// ties keep the earlier member.  Members are read four at a time.
template <typename LoadOf>
__device__ __forceinline__ uint32_t set_min(const uint16_t *mem, uint32_t off, uint32_t k, uint32_t m0,
                                            LoadOf load_of)
{
    uint32_t best = m0;
    unsigned long long bl = load_of(best);
    uint32_t m = 1;
    for (; m + 4 <= k; m += 4) {
        uint32_t d[4];
        unsigned long long l[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) d[u] = mem[off + m + u];
#pragma unroll
        for (int u = 0; u < 4; ++u) l[u] = load_of(d[u]);
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (l[u] < bl) {
                bl = l[u];
                best = d[u];
            }
    }
    for (; m < k; ++m) {
        const uint32_t d = mem[off + m];
        const unsigned long long l = load_of(d);
        if (l < bl) {
            bl = l;
            best = d;
        }
    }
    return best;
}

// Copy a replica's u16 side array -- a plan's member lists, or a ring's
// owners -- into shared memory when it fits (cap entries); returns the array
// the decisions read.
__device__ __forceinline__ const uint16_t *stage_aux(const route_desc &rd, uint16_t *sm, unsigned long long cap)
{
    const uint16_t *src = rd.policy == CR_POLICY_CHWBL ? rd.rowner : rd.members;
    if (cap == 0 || src == nullptr) return src;
    const unsigned long long nk = rd.policy == CR_POLICY_CHWBL ? rd.rM : (rd.n_members ? *rd.n_members : cap + 1);
    if (nk > cap) return src;
    for (unsigned long long x = threadIdx.x; x < nk; x += blockDim.x) sm[x] = src[x];
    return sm;
}

// One decision against the batch-start loads.  A bounded-load replica's
// candidates are all RING; every other replica's are FIXED, PAIR or SET, so
// the two cases are compiled apart.  m: requests in the load vector the batch
// sees (the bounded-load rule's m).
// Replica classes of the resolution loop, compiled apart: a plan replica's
// candidates are FIXED, PAIR or SET, a power-of-two-choices replica's only PAIR,
// a bounded-load replica's only RING.
constexpr int kResolvePlan = 0, kResolveRing = 1, kResolvePair = 2;

template <int MODE>
__device__ __forceinline__ uint32_t resolve(uint32_t c, const route_desc &rd, const uint16_t *mem,
                                            const unsigned long long *L, unsigned long long m, uint32_t R,
                                            uint32_t *status)
{
    auto load_of = [&](uint32_t d) { return L[d]; };
    if (MODE == kResolveRing) return ring_walk(rd, mem, c & kLow30, chwbl_cap(m, R), load_of, status);
    if (MODE == kResolvePair) {
        const uint32_t d1 = c & 0x1fffu, d2 = (c >> 13) & 0x1fffu;
        return L[d1] <= L[d2] ? d1 : d2;
    }
    const uint32_t kind = c & kKindMask;
    if (kind == kFixed) return c & 0xffffu;
    if (kind == kPair) {
        const uint32_t d1 = c & 0x1fffu, d2 = (c >> 13) & 0x1fffu;
        return L[d1] <= L[d2] ? d1 : d2;
    }
    const cr_table_slot slot = rd.table[c & kLow30];
#ifdef CR_DEBUG_CHECKS
    // the member list of the slot lies inside the plan's members (sum of k_b)
    if (!CR_DCHECK(rd.n_members == nullptr || (unsigned long long)slot.koff + slot.k <= *rd.n_members, status))
        return 0;
#endif
    return set_min(mem, slot.koff, slot.k, slot.m0, load_of);
}

// Candidates are staged in shared memory a whole chunk (a multiple of the
// batch, at most kStage requests) ahead: while chunk c is resolved from one
// buffer, chunk c+1's loads are in flight into registers and land in the other.
constexpr uint32_t kStage = 16384;

// 4-byte asynchronous global -> shared copies (the next chunk lands while this
// one is resolved, without holding registers)
__device__ __forceinline__ void cp_async4(void *smem, const void *gmem)
{
    const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

// Start copying chunk [c1, c1 + CH) of the candidates into buffer nb.
__device__ __forceinline__ void stage_next(uint32_t *nb, const uint32_t *__restrict__ Cd, unsigned long long c1,
                                           unsigned long long n, uint32_t CH)
{
    for (uint32_t q = threadIdx.x; q < CH && c1 + q < n; q += blockDim.x) cp_async4(&nb[q], &Cd[c1 + q]);
}

// Sum of a replica's load vector on entry (the m of the bounded-load rule).
__device__ __forceinline__ unsigned long long block_load_sum(const unsigned long long *L, uint32_t R)
{
    __shared__ unsigned long long s_tot;
    if (threadIdx.x == 0) s_tot = 0;
    __syncthreads();
    unsigned long long t = 0;
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) t += L[r];
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if ((threadIdx.x & 31) == 0 && t) atomicAdd(&s_tot, t);
    __syncthreads();
    return s_tot;
}

// The batch loop of one replica (L already holds its loads; ends with a barrier).
template <int MODE>
__device__ __forceinline__ void resolve_batches(const route_desc &rd, const uint16_t *mem, unsigned long long *L,
                                                uint32_t *delta, uint32_t *cbuf, const uint32_t *__restrict__ Cd,
                                                uint16_t *__restrict__ D, unsigned long long n, uint32_t B,
                                                uint32_t CH, uint32_t R, unsigned long long tot0, uint32_t *status)
{
    const uint32_t tid = threadIdx.x;
    if (CH == 0) {
        // batches longer than the stage: candidates straight from global memory
        for (unsigned long long b0 = 0; b0 < n; b0 += B) {
            const unsigned long long b1 = (b0 + B < n) ? b0 + B : n;
            for (unsigned long long i = b0 + tid; i < b1; i += blockDim.x) {
                const uint32_t d = resolve<MODE>(Cd[i], rd, mem, L, tot0 + b0, R, status);
                if (!CR_DCHECK(d < R, status)) continue;
                D[i] = (uint16_t)d;
                atomicAdd(&delta[d], 1u);
            }
            __syncthreads();
            for (uint32_t r = tid; r < R; r += blockDim.x) {
                L[r] += delta[r];
                delta[r] = 0;
            }
            __syncthreads();
        }
        return;
    }
    for (uint32_t x = tid; x < CH && x < n; x += blockDim.x) cbuf[x] = Cd[x];
    __syncthreads();
    int cur = 0;
    for (unsigned long long c0 = 0; c0 < n; c0 += CH) {
        const unsigned long long c1 = (c0 + CH < n) ? c0 + CH : n;
        stage_next(cbuf + (size_t)(cur ^ 1) * CH, Cd, c1, n, CH);  // next chunk in flight
        const uint32_t *cb = cbuf + (size_t)cur * CH;
        uint16_t *Dc = D + c0;
        const uint32_t len = (uint32_t)(c1 - c0);  // chunk offsets fit 32 bits
        for (uint32_t o0 = 0; o0 < len; o0 += B) {
            const uint32_t o1 = (o0 + B < len) ? o0 + B : len;
            for (uint32_t o = o0 + tid; o < o1; o += blockDim.x) {
                const uint32_t d = resolve<MODE>(cb[o], rd, mem, L, tot0 + c0 + o0, R, status);
                if (!CR_DCHECK(d < R, status)) continue;
                Dc[o] = (uint16_t)d;
                atomicAdd(&delta[d], 1u);
            }
            __syncthreads();
            for (uint32_t r = tid; r < R; r += blockDim.x) {
                L[r] += delta[r];
                delta[r] = 0;
            }
            __syncthreads();
        }
        cp_async_wait_all();
        __syncthreads();
        cur ^= 1;
    }
}

// ---- plan replicas: keys with several members decided once per batch ---------
// Inside a batch every request of a key with k_b > 1 goes to the same member:
// the least loaded of T(b) at the batch start (ties to the earlier member).  So
// the CTA keeps the member lists of those keys in shared memory, collected as
// the staging meets them, and finds each key's member once per batch, at the
// boundary; a request then reads its key's answer.  Loads and batch counts are
// double-buffered so that the answers for batch b + 1 (loads of batch b plus
// its counts) are computed while the loads are being updated, behind the same
// two barriers per batch.
constexpr uint32_t kSetCap = 256;      // keys with k_b > 1 tracked per replica
constexpr uint32_t kSetMapCap = 512;   // open-addressing map: table slot -> key index
constexpr uint32_t kSetPool = 4096;    // member entries of the tracked keys

struct set_cache {
    uint32_t map_slot[kSetMapCap];  // table slot of each map entry, kEmpty when free
    uint16_t map_j[kSetMapCap];     // key index of each map entry
    uint32_t off[kSetCap];          // first member of key j in the pool
    uint16_t k[kSetCap];
    uint16_t res[2][kSetCap];       // least-loaded member of each key, per batch parity
    uint16_t pool[kSetPool];
    uint32_t n, used, ready, overflow;
};

__host__ __device__ inline size_t set_cache_bytes() { return (sizeof(set_cache) + 15) & ~(size_t)15; }

// Shared-memory layout of k_route_resolve: loads [R] u64, counts [R] u32, two
// staging buffers [CH] u32, member lists / ring owners [MC] u16, then (plan
// replicas) the second loads and counts and the key cache, 16-byte aligned.
__host__ __device__ inline size_t resolve_plan_extra_at(uint32_t R, uint32_t CH, unsigned long long MC)
{
    return ((size_t)R * 12 + (size_t)CH * 8 + (size_t)MC * 2 + 15) & ~(size_t)15;
}
__host__ __device__ inline size_t resolve_plan_extra_bytes(uint32_t R)
{
    return (((size_t)R * 12 + 15) & ~(size_t)15) + set_cache_bytes();
}

__device__ __forceinline__ uint32_t set_hash(uint32_t slot) { return (slot * 0x9E3779B1u) >> 23; }  // 9 bits

// Record the key of table slot `slot` (a SET candidate) unless it is known.
__device__ void set_discover(set_cache &S, const route_desc &rd, const uint16_t *mem, uint32_t slot)
{
    uint32_t h = set_hash(slot);
    for (uint32_t it = 0; it < kSetMapCap; ++it, h = (h + 1) & (kSetMapCap - 1)) {
        const uint32_t cur = *(volatile uint32_t *)&S.map_slot[h];
        if (cur == slot) return;
        if (cur != kEmpty) continue;
        const uint32_t prev = atomicCAS(&S.map_slot[h], kEmpty, slot);
        if (prev == slot) return;
        if (prev != kEmpty) continue;
        const uint32_t j = atomicAdd(&S.n, 1u);
        const cr_table_slot ts = rd.table[slot];
        const uint32_t off = atomicAdd(&S.used, (uint32_t)ts.k);
        if (j >= kSetCap || off + ts.k > kSetPool) {
            S.overflow = 1u;
            return;
        }
        for (uint32_t m = 0; m < ts.k; ++m) S.pool[off + m] = mem[(size_t)ts.koff + m];
        S.off[j] = off;
        S.k[j] = ts.k;
        S.map_j[h] = (uint16_t)j;
        return;
    }
    S.overflow = 1u;
}

// Key index of a discovered slot, or kEmpty.
__device__ __forceinline__ uint32_t set_find(const set_cache &S, uint32_t slot)
{
    uint32_t h = set_hash(slot);
    for (uint32_t it = 0; it < kSetMapCap; ++it, h = (h + 1) & (kSetMapCap - 1)) {
        const uint32_t cur = S.map_slot[h];
        if (cur == slot) return S.map_j[h];
        if (cur == kEmpty) return kEmpty;
    }
    return kEmpty;
}

// res[j] for keys j0 .. j1-1: the first member with the least load Lb[m] (+ db[m]),
// one warp per key.
__device__ __forceinline__ void set_results(set_cache &S, uint16_t *res, const unsigned long long *Lb,
                                            const uint32_t *db, uint32_t j0, uint32_t j1)
{
    const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (uint32_t j = j0 + warp; j < j1; j += nw) {
        const uint32_t off = S.off[j], k = S.k[j];
        unsigned long long bl = ~0ull;
        uint32_t bp = 0xffffffffu;
        for (uint32_t p = lane; p < k; p += 32) {
            const uint32_t m = S.pool[off + p];
            const unsigned long long l = Lb[m] + (db ? db[m] : 0u);
            if (l < bl) {  // positions rise within a lane: the first minimum stays
                bl = l;
                bp = p;
            }
        }
        // the lexicographic minimum of (load, position) over the warp, by three 32-bit
        // warp reductions: high word of the load, low word among those, position among those
        const uint32_t hi = (uint32_t)(bl >> 32), lo = (uint32_t)bl;
        const uint32_t mhi = __reduce_min_sync(0xffffffffu, hi);
        const uint32_t mlo = __reduce_min_sync(0xffffffffu, hi == mhi ? lo : 0xffffffffu);
        const uint32_t mp = __reduce_min_sync(0xffffffffu, (hi == mhi && lo == mlo) ? bp : 0xffffffffu);
        if (lane == 0) res[j] = S.pool[off + mp];
    }
}

// The batch loop of a plan replica with staging (CH > 0).  L0/dl0 hold the loads
// and zero counts on entry; returns the buffer (0 or 1) that holds the loads at
// the end.  Falls back to per-request member scans once the cache overflows.
__device__ int resolve_batches_plan(const route_desc &rd, const uint16_t *mem, unsigned long long *L0,
                                    unsigned long long *L1, uint32_t *dl0, uint32_t *dl1, set_cache &S,
                                    uint32_t *cbuf, const uint32_t *__restrict__ Cd, uint16_t *__restrict__ D,
                                    unsigned long long n, uint32_t B, uint32_t CH, uint32_t R, uint32_t *status)
{
    const uint32_t tid = threadIdx.x;
    for (uint32_t x = tid; x < kSetMapCap; x += blockDim.x) S.map_slot[x] = kEmpty;
    if (tid == 0) {
        S.n = 0;
        S.used = 0;
        S.ready = 0;
        S.overflow = 0;
    }
    for (uint32_t r = tid; r < R; r += blockDim.x) dl1[r] = 0;
    __syncthreads();
    for (uint32_t x = tid; x < CH && x < n; x += blockDim.x) {
        const uint32_t c = Cd[x];
        cbuf[x] = c;
        if ((c & kKindMask) == kSet) set_discover(S, rd, mem, c & kLow30);
    }
    __syncthreads();
    if (!S.overflow) set_results(S, S.res[0], L0, nullptr, 0, min(S.n, kSetCap));
    if (tid == 0) S.ready = min(S.n, kSetCap);  // read by nobody before the barrier
    __syncthreads();
    int par = 0, cur = 0;
    for (unsigned long long c0 = 0; c0 < n; c0 += CH) {
        const unsigned long long c1 = (c0 + CH < n) ? c0 + CH : n;
        uint32_t *nb = cbuf + (size_t)(cur ^ 1) * CH;
        stage_next(nb, Cd, c1, n, CH);
        const uint32_t *cb = cbuf + (size_t)cur * CH;
        uint16_t *Dc = D + c0;
        const uint32_t len = (uint32_t)(c1 - c0);
        const bool ovf = S.overflow != 0u;  // uniform: written only while staging
        for (uint32_t o0 = 0; o0 < len; o0 += B) {
            const uint32_t o1 = (o0 + B < len) ? o0 + B : len;
            unsigned long long *Lc = par ? L1 : L0, *Ln = par ? L0 : L1;
            uint32_t *dc = par ? dl1 : dl0, *dn = par ? dl0 : dl1;
            const uint16_t *res = S.res[par];
            for (uint32_t o = o0 + tid; o < o1; o += blockDim.x) {
                const uint32_t c = cb[o], kind = c & kKindMask;
                // FIXED and PAIR without a branch: for FIXED the two fields read are the
                // destination (< R <= 8192) and 0, in range as well; a SET reads entry 0
                const bool two = kind < kSet;
                const uint32_t d1 = two ? (c & 0x1fffu) : 0u, d2 = two ? ((c >> 13) & 0x1fffu) : 0u;
                const bool p1 = Lc[d1] <= Lc[d2];
                uint32_t d = kind == kFixed ? (c & 0xffffu) : (p1 ? d1 : d2);
                if (!two) {
                    const uint32_t j = ovf ? kEmpty : set_find(S, c & kLow30);
                    if (j < kSetCap) {
                        d = res[j];
                    } else {
                        const cr_table_slot slot = rd.table[c & kLow30];
                        auto load_of = [&](uint32_t x) { return Lc[x]; };
                        d = set_min(mem, slot.koff, slot.k, slot.m0, load_of);
                    }
                }
                if (!CR_DCHECK(d < R, status)) continue;
                Dc[o] = (uint16_t)d;
                atomicAdd(&dc[d], 1u);
            }
            __syncthreads();
            for (uint32_t r = tid; r < R; r += blockDim.x) {
                Ln[r] = Lc[r] + dc[r];
                dn[r] = 0;
            }
            if (!ovf) set_results(S, S.res[par ^ 1], Lc, dc, 0, min(S.ready, kSetCap));
            __syncthreads();
            par ^= 1;
        }
        cp_async_wait_all();
        __syncthreads();
        for (uint32_t q = tid; q < CH && c1 + q < n; q += blockDim.x)
            if ((nb[q] & kKindMask) == kSet) set_discover(S, rd, mem, nb[q] & kLow30);
        __syncthreads();
        // keys met for the first time: their answers for the next batch, from its loads
        const uint32_t nn = min(S.n, kSetCap), rd0 = S.ready;
        if (nn > rd0 && !S.overflow) set_results(S, S.res[par], par ? L1 : L0, nullptr, rd0, nn);  // uniform
        __syncthreads();  // every thread has read S.ready
        if (tid == 0) S.ready = S.overflow ? rd0 : nn;
        __syncthreads();
        cur ^= 1;
    }
    return par;
}

__global__ void __launch_bounds__(kRouteBlock) k_route_resolve(const __grid_constant__ route_args args,
                                                               const uint32_t *__restrict__ cand,
                                                               unsigned long long n, uint32_t B, uint32_t CH,
                                                               uint32_t R, unsigned long long *__restrict__ load,
                                                               uint16_t *__restrict__ dest, uint32_t *status,
                                                               unsigned long long MC, int plan_x)
{
    extern __shared__ unsigned long long sh[];
    unsigned long long *L = sh;                              // [R] live load
    uint32_t *delta = reinterpret_cast<uint32_t *>(sh + R);  // [R] this batch
    uint32_t *cbuf = delta + R;                              // [2][CH] staged candidates
    uint16_t *smem_aux = reinterpret_cast<uint16_t *>(cbuf + 2 * (size_t)CH);  // [MC] members or ring owners
    // plan replicas (when the launch reserved it): the second load and count buffers and the key cache
    unsigned char *px = reinterpret_cast<unsigned char *>(sh) + resolve_plan_extra_at(R, CH, MC);
    const uint32_t rep = args.dep[blockIdx.x];
    const route_desc rd = args.d[rep];
    unsigned long long *Lg = load + (unsigned long long)rep * R;
    const uint32_t *Cd = cand + (unsigned long long)rep * n;
    uint16_t *D = dest + (unsigned long long)rep * n;
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) {
        L[r] = Lg[r];
        delta[r] = 0;
    }
    const uint16_t *mem = stage_aux(rd, smem_aux, MC);
    if (rd.policy == CR_POLICY_CHWBL) {  // uniform over the block
        const unsigned long long tot0 = block_load_sum(L, R);
        resolve_batches<kResolveRing>(rd, mem, L, delta, cbuf, Cd, D, n, B, CH, R, tot0, status);
    } else if (rd.policy == CR_POLICY_P2C) {
        __syncthreads();  // orders the copies above
        resolve_batches<kResolvePair>(rd, mem, L, delta, cbuf, Cd, D, n, B, CH, R, 0ull, status);
    } else if (plan_x && CH > 0) {
        __syncthreads();
        unsigned long long *L1 = reinterpret_cast<unsigned long long *>(px);
        uint32_t *dl1 = reinterpret_cast<uint32_t *>(L1 + R);
        set_cache &S = *reinterpret_cast<set_cache *>(px + (((size_t)R * 12 + 15) & ~(size_t)15));
        if (resolve_batches_plan(rd, mem, L, L1, delta, dl1, S, cbuf, Cd, D, n, B, CH, R, status))
            for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) L[r] = L1[r];
        __syncthreads();
    } else {
        __syncthreads();
        resolve_batches<kResolvePlan>(rd, mem, L, delta, cbuf, Cd, D, n, B, CH, R, 0ull, status);
    }
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) Lg[r] = L[r];
}

// ---- batches of at most one warp: one warp per replica ----------------------

constexpr int kWarpChunk = 8;  // steps whose candidates are fetched one chunk ahead

// A candidate with its table slot or first ring owner already fetched.
struct prep_cand {
    uint32_t kind;
    uint32_t a;  // FIXED: destination; PAIR: d1; SET: first member; RING: owner of the first point
    uint32_t b;  // PAIR: d2; SET: member offset; RING: first ring index
    uint32_t k;  // SET: members
};

__device__ __forceinline__ prep_cand prepare(uint32_t c, const route_desc &rd, const uint16_t *own)
{
    prep_cand p;
    p.kind = c & kKindMask;
    p.a = c & 0xffffu;
    p.b = 0;
    p.k = 1;
    if (p.kind == kPair) {
        p.a = c & 0x1fffu;
        p.b = (c >> 13) & 0x1fffu;
    } else if (p.kind == kSet) {
        const cr_table_slot slot = rd.table[c & kLow30];
        p.a = slot.m0;
        p.b = slot.koff;
        p.k = slot.k;
    } else if (p.kind == kRing) {
        p.b = c & kLow30;
        p.a = own[p.b];
    }
    return p;
}

// The decision of one request that sees load L[d] plus the lanes of `earlier`
// currently placed on d.
__device__ __forceinline__ uint32_t decide(const prep_cand &p, const route_desc &rd, const uint16_t *mem,
                                           const unsigned long long *L, const uint32_t *mask, uint32_t earlier,
                                           unsigned long long cap, uint32_t *status)
{
    auto seen = [&](uint32_t d) { return L[d] + (unsigned long long)__popc(mask[d] & earlier); };
    if (p.kind == kFixed) return p.a;
    if (p.kind == kPair) return seen(p.a) <= seen(p.b) ? p.a : p.b;
    if (p.kind == kRing) return seen(p.a) < cap ? p.a : ring_walk(rd, mem, p.b, cap, seen, status);
    return set_min(mem, p.b, p.k, p.a, seen);
}

__global__ void __launch_bounds__(32) k_route_resolve_warp(const __grid_constant__ route_args args,
                                                           const uint32_t *__restrict__ cand, unsigned long long n,
                                                           uint32_t B, uint32_t R,
                                                           unsigned long long *__restrict__ load,
                                                           uint16_t *__restrict__ dest, uint32_t *status,
                                                           unsigned long long MC)
{
    extern __shared__ unsigned long long sh[];
    prep_cand *ps = reinterpret_cast<prep_cand *>(sh);      // [kWarpChunk][32] prepared candidates
    unsigned long long *L = sh + kWarpChunk * 32 * sizeof(prep_cand) / sizeof(unsigned long long);  // [R]
    uint32_t *mask = reinterpret_cast<uint32_t *>(L + R);   // [R] lanes of the step on each destination
    uint16_t *smem_aux = reinterpret_cast<uint16_t *>(mask + R);  // [MC] members or ring owners
    const uint32_t rep = args.dep[blockIdx.x];
    const route_desc &rd = args.d[rep];
    unsigned long long *Lg = load + (unsigned long long)rep * R;
    const uint32_t *Cd = cand + (unsigned long long)rep * n;
    uint16_t *D = dest + (unsigned long long)rep * n;
    const uint32_t lane = threadIdx.x;
    unsigned long long tot = 0;
    for (uint32_t r = lane; r < R; r += 32) {
        const unsigned long long v = Lg[r];
        L[r] = v;
        mask[r] = 0;
        tot += v;
    }
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    const uint16_t *mem = stage_aux(rd, smem_aux, MC);
    __syncwarp();
    const uint32_t S = (32u / B) * B;               // requests per step: whole batches
    const uint32_t bstart = (lane / B) * B;         // first lane of this lane's batch
    const uint32_t earlier = (1u << bstart) - 1u;   // lanes of the earlier batches of the step
    const uint32_t bit = 1u << lane;
    const bool several = S > B;
    const bool ring = rd.policy == CR_POLICY_CHWBL;  // only its decisions read the cap
    const unsigned long long CHR = (unsigned long long)S * kWarpChunk;
    uint32_t cn[kWarpChunk];
#pragma unroll
    for (int q = 0; q < kWarpChunk; ++q) {
        const unsigned long long i = (unsigned long long)q * S + lane;
        cn[q] = (lane < S && i < n) ? Cd[i] : 0u;  // 0 = FIXED 0: inactive lanes read nothing
    }
    for (unsigned long long c0 = 0; c0 < n; c0 += CHR) {
        // each lane prepares (and later reads) only its own entries: no barrier needed
#pragma unroll
        for (int q = 0; q < kWarpChunk; ++q) ps[q * 32 + lane] = prepare(cn[q], rd, mem);
#pragma unroll
        for (int q = 0; q < kWarpChunk; ++q) {
            const unsigned long long i = c0 + CHR + (unsigned long long)q * S + lane;
            cn[q] = (lane < S && i < n) ? Cd[i] : 0u;
        }
#pragma unroll 1
        for (int q = 0; q < kWarpChunk; ++q) {
            const unsigned long long s0 = c0 + (unsigned long long)q * S;
            if (s0 >= n) break;  // uniform over the warp
            const unsigned long long i = s0 + lane;
            const bool active = lane < S && i < n;
            const unsigned long long cap = ring ? chwbl_cap(tot + bstart, R) : 0ull;
            const prep_cand pq = ps[q * 32 + lane];
            uint32_t d = decide(pq, rd, mem, L, mask, 0u, cap, status);
            if (!CR_DCHECK(d < R, status)) d = 0;
            if (active) atomicOr(&mask[d], bit);
            __syncwarp();
            if (several) {
                // fixed point: after iteration t the first t batches of the step are final
                for (uint32_t it = 0;; ++it) {
                    uint32_t nd = active ? decide(pq, rd, mem, L, mask, earlier, cap, status) : d;
                    if (!CR_DCHECK(nd < R, status)) nd = 0;
                    const uint32_t moved = __ballot_sync(0xffffffffu, nd != d);
                    if (!moved) break;
                    if (it >= S) {  // unreachable: S iterations always settle the step
                        if (lane == 0) atomicOr(status, CR_FLAG_TIMEOUT);
                        break;
                    }
                    if (nd != d) {
                        atomicAnd(&mask[d], ~bit);
                        atomicOr(&mask[nd], bit);
                        d = nd;
                    }
                    __syncwarp();
                }
            }
            if (active) {
                const uint32_t mk = mask[d];
                if ((mk & (0u - mk)) == bit) L[d] += (unsigned long long)__popc(mk);  // lowest lane adds
                D[i] = (uint16_t)d;
            }
            __syncwarp();
            if (active) mask[d] = 0;
            __syncwarp();
            const unsigned long long left = n - s0;
            tot += left < S ? left : S;
        }
    }
    for (uint32_t r = lane; r < R; r += 32) Lg[r] = L[r];
}

// ---- ring construction ------------------------------------------------------

__global__ void __launch_bounds__(256) k_ring_points(unsigned long long seed, unsigned long long M,
                                                     unsigned long long *__restrict__ pt)
{
    for (unsigned long long k = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; k < M;
         k += (unsigned long long)gridDim.x * blockDim.x)
        pt[k] = cr_fmix64(seed + (k + 1ull) * CR_GAMMA);  // SplitMix64 output k
}

// Sorted points (stable: equal points keep ascending owner) -> point and owner arrays.
__global__ void __launch_bounds__(256) k_ring_finish(const unsigned long long *__restrict__ ks,
                                                     const uint32_t *__restrict__ pos, unsigned long long M,
                                                     uint32_t V, unsigned long long *__restrict__ pt,
                                                     uint16_t *__restrict__ ow)
{
    for (unsigned long long j = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; j < M;
         j += (unsigned long long)gridDim.x * blockDim.x) {
        pt[j] = ks[j];
        ow[j] = (uint16_t)(pos[j] / V);
    }
}

// dir[t] = first ring index whose point is >= t << (64 - dbits) (M if none).
__global__ void __launch_bounds__(256) k_ring_dir(const unsigned long long *__restrict__ pt, unsigned long long M,
                                                  int dbits, uint32_t *__restrict__ dir)
{
    const unsigned long long nd = 1ull << dbits;
    for (unsigned long long t = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; t < nd;
         t += (unsigned long long)gridDim.x * blockDim.x) {
        const unsigned long long h = t << (64 - dbits);
        unsigned long long lo = 0, hi = M;
        while (lo < hi) {
            const unsigned long long mid = (lo + hi) >> 1;
            if (pt[mid] < h)
                lo = mid + 1;
            else
                hi = mid;
        }
        dir[t] = (uint32_t)lo;
    }
}

}  // namespace

static int ring_fill(cr_ctx *ctx, cr_ring *g, uint64_t seed)
{
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    const unsigned long long M = g->M;
    const unsigned long long *ks = nullptr;
    const uint32_t *pos = nullptr;
    CR_LAUNCH(ctx, k_ring_points, cr_blocks(M, 256, gcap), 256, 0, (unsigned long long)seed, M, g->d_point);
    CR_TRY(cr_radix_sort_u64(ctx, g->d_point, nullptr, M, 64, &ks, &pos));
    CR_LAUNCH(ctx, k_ring_finish, cr_blocks(M, 256, gcap), 256, 0, ks, pos, M, g->V, g->d_point, g->d_owner);
    CR_LAUNCH(ctx, k_ring_dir, cr_blocks(1ull << g->dbits, 256, gcap), 256, 0, (const unsigned long long *)g->d_point,
              M, (int)g->dbits, g->d_dir);
    return CR_OK;
}

extern "C" int cr_ring_create(cr_ctx *ctx, uint32_t R, uint32_t vnodes, uint64_t seed, cr_ring **out)
{
    if (!ctx || !out) return CR_EINVAL;
    *out = nullptr;
    if (R == 0 || R > CR_MAX_R) return cr_fail(ctx, CR_EINVAL, "cr_ring_create: R=%u outside 1..%u", R, CR_MAX_R);
    if (vnodes == 0 || vnodes > CR_MAX_VNODES)
        return cr_fail(ctx, CR_EINVAL, "cr_ring_create: vnodes=%u outside 1..%u", vnodes, CR_MAX_VNODES);
    const uint64_t M = (uint64_t)R * vnodes;
    int dbits = 1;
    while ((1ull << dbits) < M) ++dbits;
    cr_ring *g = (cr_ring *)calloc(1, sizeof(cr_ring));
    if (!g) return cr_fail(ctx, CR_ENOMEM, "cr_ring_create: host allocation failed");
    g->R = R;
    g->V = vnodes;
    g->M = M;
    g->dbits = (uint32_t)dbits;
    if (cudaMalloc(&g->d_point, M * sizeof(unsigned long long)) != cudaSuccess ||
        cudaMalloc(&g->d_owner, M * sizeof(uint16_t)) != cudaSuccess ||
        cudaMalloc(&g->d_dir, (1ull << dbits) * sizeof(uint32_t)) != cudaSuccess) {
        cudaGetLastError();
        cr_ring_destroy(ctx, g);
        return cr_fail(ctx, CR_ENOMEM, "cr_ring_create: device allocation of %llu points failed",
                       (unsigned long long)M);
    }
    const int st = ring_fill(ctx, g, seed);
    if (st != CR_OK) {
        cr_ring_destroy(ctx, g);
        return st;
    }
    *out = g;
    return CR_OK;
}

extern "C" int cr_ring_destroy(cr_ctx *ctx, cr_ring *g)
{
    if (!g) return CR_OK;
    if (ctx) cudaStreamSynchronize(ctx->stream);
    if (g->d_point) cudaFree(g->d_point);
    if (g->d_owner) cudaFree(g->d_owner);
    if (g->d_dir) cudaFree(g->d_dir);
    free(g);
    return CR_OK;
}

extern "C" int cr_ring_export(cr_ctx *ctx, const cr_ring *g, uint64_t *point, uint16_t *owner)
{
    if (!ctx || !g) return CR_EINVAL;
    if (point)
        CR_CUDA(ctx, cudaMemcpyAsync(point, g->d_point, g->M * sizeof(uint64_t), cudaMemcpyDeviceToHost, ctx->stream));
    if (owner)
        CR_CUDA(ctx, cudaMemcpyAsync(owner, g->d_owner, g->M * sizeof(uint16_t), cudaMemcpyDeviceToHost, ctx->stream));
    return cr_sync(ctx);
}

static int launch_resolve(cr_ctx *ctx, cudaStream_t rs, const route_args &args, const uint32_t *cand, uint64_t n,
                          uint32_t batch_B, uint32_t R, uint64_t mc, uint32_t n_dep, uint64_t *d_load,
                          uint16_t *d_dest);

extern "C" int cr_route_batch(cr_ctx *ctx, const cr_plan *const *plans, const cr_replica *reps, uint32_t n_rep,
                              uint32_t R, const uint64_t *d_key, uint64_t n, uint64_t first_req_index,
                              uint32_t batch_B, uint64_t *d_load, uint16_t *d_dest)
{
    if (!ctx) return CR_EINVAL;
    cr_nvtx_range nv("cr_route_batch");
    if (R == 0 || R > CR_MAX_R) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: R=%u outside 1..%u", R, CR_MAX_R);
    if (n_rep == 0 || n_rep > CR_MAX_REPLICAS || !reps)
        return cr_fail(ctx, CR_EINVAL, "cr_route_batch: n_rep=%u outside 1..%u", n_rep, CR_MAX_REPLICAS);
    if (batch_B == 0) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: batch_B must be >= 1");
    if (n >= (1ull << 40)) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: n >= 2^40");
    if (!d_load) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: d_load is NULL");
    if (n > 0 && (!d_key || !d_dest)) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: NULL key or dest");
    route_args args;
    memset(&args, 0, sizeof(args));
    uint64_t mc = 0;  // largest u16 side array: a plan's member lists or a ring's owners
    for (uint32_t i = 0; i < n_rep; ++i) {
        route_desc &d = args.d[i];
        d.policy = reps[i].policy;
        d.seed = reps[i].seed;
        if (reps[i].policy > CR_POLICY_CHWBL || reps[i].reserved != 0)
            return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u has policy %u", i, reps[i].policy);
        if (reps[i].policy <= CR_POLICY_CR_NOREPL) {
            const cr_plan *p = plans ? plans[i] : nullptr;
            if (!p || !p->built)
                return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u needs a built plan", i);
            if (p->R != R)
                return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u plan has R=%u, call has R=%u", i, p->R, R);
            int bits = 0;
            while ((1ull << bits) < p->table_slots) ++bits;
            if (bits > 30) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: plan table too large");
            d.tbits = bits;
            d.table = p->d_table;
            d.members = p->d_members;
            d.n_members = &p->d_info->sum_k;
            mc = std::max<uint64_t>(mc, (uint64_t)p->R * p->W);  // sum of k_b <= C = R W
        } else if (reps[i].policy == CR_POLICY_CHWBL) {
            const cr_ring *g = reps[i].ring;
            if (!g) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u needs a ring", i);
            if (g->R != R)
                return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u ring has R=%u, call has R=%u", i, g->R, R);
            d.rpoint = g->d_point;
            d.rowner = g->d_owner;
            d.rdir = g->d_dir;
            d.rM = (uint32_t)g->M;
            d.rdbits = (int32_t)g->dbits;
            mc = std::max<uint64_t>(mc, g->M);
        }
    }
    if (n == 0) return CR_OK;
    // replicas whose choices depend on the live load
    uint32_t n_dep = 0;
    for (uint32_t i = 0; i < n_rep; ++i)
        if (reps[i].policy != CR_POLICY_RR && reps[i].policy != CR_POLICY_HASH) args.dep[n_dep++] = i;
    // candidate rows, costliest policy first, so that the grid's last wave holds cheap rows
    // (per request: jump hash ~8 jumps, Philox ~10 rounds, plan probe + Philox for misses,
    // ring lookup, round robin)
    {
        auto cost = [&](uint32_t p) {
            return p == CR_POLICY_HASH ? 0 : p == CR_POLICY_P2C ? 1 : p <= CR_POLICY_CR_NOREPL ? 2
                 : p == CR_POLICY_CHWBL ? 3 : 4;
        };
        uint32_t k = 0;
        for (uint32_t c = 0; c <= 4; ++c)
            for (uint32_t i = 0; i < n_rep; ++i)
                if ((uint32_t)cost(reps[i].policy) == c) args.cand[k++] = i;
    }
    // split routing: the candidates scratch is free once the last resolution has read it
    const cudaStream_t rs = ctx->resolve_stream ? ctx->resolve_stream : ctx->stream;
    const bool split = rs != ctx->stream;
    if (split && ctx->resolve_recorded) CR_CUDA(ctx, cudaStreamWaitEvent(ctx->stream, ctx->ev_resolve, 0));
    void *pc;
    CR_TRY(cr_scratch(ctx, SCR_ROUTE_DESC, (size_t)n * n_rep * sizeof(uint32_t), &pc));
    uint32_t *cand = (uint32_t *)pc;
    const int pcand = cr_prof_begin(ctx, ctx->stream, CR_PROF_ROUTE_CAND);
    for (uint32_t i = 0; i < n_rep; ++i) {
        const uint64_t base = (uint64_t)first_req_index + reps[i].seed;  // wraps mod 2^64 as the policy does
        args.rr_b0[i] = (uint32_t)(base % R);
        args.rr_wrap[i] = base ? 0ull - base : ~0ull;
    }
    // request blocks; replica groups only as many as it takes to reach ~16 blocks per SM
    const unsigned int cbx = cr_blocks(n, 256, (unsigned int)ctx->num_sms * 32u);
    const unsigned int want = (unsigned int)ctx->num_sms * 16u;
    unsigned int cgy = (want + cbx - 1) / cbx;
    cgy = cgy < 1 ? 1 : (cgy > n_rep ? n_rep : cgy);
    CR_LAUNCH(ctx, k_route_cand, dim3(cbx, cgy), 256, 0, args, n_rep,
              (const unsigned long long *)d_key, (unsigned long long)n, (unsigned long long)first_req_index, R, cand,
              d_dest);
    cr_prof_end(ctx, ctx->stream, pcand);
    // load counts of RR / HASH replicas (their choices never read the load)
    for (uint32_t i = 0; i < n_rep; ++i) {
        if (reps[i].policy != CR_POLICY_RR && reps[i].policy != CR_POLICY_HASH) continue;
        uint32_t j = i;
        while (j + 1 < n_rep && (reps[j + 1].policy == CR_POLICY_RR || reps[j + 1].policy == CR_POLICY_HASH)) ++j;
        dim3 grid(cr_blocks(n, 256, 64), j - i + 1);
        CR_LAUNCH(ctx, k_route_count, grid, 256, (size_t)R * sizeof(uint32_t), d_dest + (uint64_t)i * n,
                  (unsigned long long)n, R, (unsigned long long *)d_load + (uint64_t)i * R);
        i = j;
    }
    if (split) {  // the resolution (and the caller's later readers) follow everything above
        CR_CUDA(ctx, cudaEventRecord(ctx->ev_cand, ctx->stream));
        CR_CUDA(ctx, cudaStreamWaitEvent(rs, ctx->ev_cand, 0));
    }
    if (n_dep) {
        const int pr = cr_prof_begin(ctx, rs, CR_PROF_ROUTE_RESOLVE);
        CR_TRY(launch_resolve(ctx, rs, args, cand, n, batch_B, R, mc, n_dep, d_load, d_dest));
        cr_prof_end(ctx, rs, pr);
    }
    if (split) {
        CR_CUDA(ctx, cudaEventRecord(ctx->ev_resolve, rs));
        ctx->resolve_recorded = 1;
    }
    return CR_OK;
}

// The load-dependent resolution of every dependent replica, enqueued on stream rs.
static int launch_resolve(cr_ctx *ctx, cudaStream_t rs, const route_args &args, const uint32_t *cand, uint64_t n,
                          uint32_t batch_B, uint32_t R, uint64_t mc, uint32_t n_dep, uint64_t *d_load,
                          uint16_t *d_dest)
{
    // member lists and ring owners go to shared memory when they fit beside the loads
    auto with_members = [&](size_t base, uint64_t *MC) {
        *MC = (mc && base + mc * sizeof(uint16_t) <= kSmemBudget) ? mc : 0;
        return base + *MC * sizeof(uint16_t);
    };
    uint64_t MC;
    if (batch_B <= 32) {
        const size_t smem = with_members(kWarpChunk * 32 * sizeof(prep_cand) +
                                             (size_t)R * (sizeof(unsigned long long) + sizeof(uint32_t)), &MC);
        if (smem > 48 * 1024)
            CR_CUDA(ctx, cudaFuncSetAttribute(k_route_resolve_warp, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smem));
        CR_LAUNCH_ON(ctx, rs, k_route_resolve_warp, n_dep, 32, smem, args, (const uint32_t *)cand, (unsigned long long)n,
                  batch_B, R, (unsigned long long *)d_load, d_dest, ctx->d_status, (unsigned long long)MC);
        return CR_OK;
    }
    // staging chunk: a whole number of batches, at most kStage requests
    uint32_t CH = batch_B <= kStage ? (kStage / batch_B) * batch_B : 0u;  // 0: no staging
    const size_t loads = (size_t)R * (sizeof(unsigned long long) + sizeof(uint32_t));
    // plan replicas take the second load and count buffers and the key cache when they
    // fit beside a stage of at least one batch (the stage shrinks by whole batches)
    bool any_plan = false;
    for (uint32_t i = 0; i < n_dep; ++i) any_plan |= args.d[args.dep[i]].policy <= CR_POLICY_CR_NOREPL;
    const size_t px = resolve_plan_extra_bytes(R);
    int plan_x = 0;
    if (any_plan && CH) {
        uint32_t ch = CH;
        while (ch >= batch_B && loads + (size_t)ch * 8 + 16 + px > kSmemBudget) ch -= batch_B;
        if (ch >= batch_B) {
            CH = ch;
            plan_x = 1;
        }
    }
    size_t smem;
    if (plan_x) {
        const size_t fixed = loads + (size_t)CH * 8 + 16 + px;
        MC = (mc && fixed + mc * sizeof(uint16_t) <= kSmemBudget) ? mc : 0;
        smem = resolve_plan_extra_at(R, CH, MC) + px;
    } else {
        smem = with_members(loads + 2ull * CH * sizeof(uint32_t), &MC);
    }
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_route_resolve, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    CR_LAUNCH_ON(ctx, rs, k_route_resolve, n_dep, kRouteBlock, smem, args, (const uint32_t *)cand, (unsigned long long)n,
              batch_B, CH, R, (unsigned long long *)d_load, d_dest, ctx->d_status, (unsigned long long)MC, plan_x);
    return CR_OK;
}
