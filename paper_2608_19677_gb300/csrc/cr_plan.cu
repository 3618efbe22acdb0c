// a2..a6: per-interval plan construction (Eq. 1 and Algorithm 1).
//
//   histogram   warp-aggregated counts in an L2-resident open-addressing table,
//               occupied slots compacted to (b, lambda_b)
//   order       (lambda desc, key asc): for intervals of up to 524,288 requests
//               one CTA sorts only the admission candidates (the keys whose count
//               reaches the C-th largest, C = R*W); above, device-wide radix
//               passes sort every key
//   per plan    k_b (Eq. 1), inclusive scan of k_b, admission cut, admitted
//               arrays, cold-tail total and initial loads (small intervals: every
//               plan in one launch, one CTA each), placement (LPT: one warp per
//               plan, warp argmin over per-lane minima, runs of equal-count
//               single-copy keys placed at once; RANDOM: one warp per key,
//               Fisher-Yates steps in shared memory), then the device hash table
//               b -> (offset, k_b, first member) used by dispatch.
// No host synchronisation: sizes known only on the device (U, S, n_adm) are
// read by the kernels, and grids are sized from host-side upper bounds.
#include <stdlib.h>
#include <string.h>

#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

constexpr uint32_t kEmpty = 0xffffffffu;
constexpr unsigned long long kLoadLimit = 1ull << 47;

__global__ void k_plan_reset(cr_plan_info_dev *info, unsigned long long n)
{
    info->n = n;
    info->U = 0;
    info->S = 0;
    info->adm_lam = 0;
    info->n_adm = 0;
    info->sum_k = 0;
    info->cold = 0;
    info->max_k = 0;
    info->special = 0;
}

// ---- histogram: counts in an L2-resident open-addressing table ----------
// Slots hold (key, count); an empty slot holds the key 2^64-1, so requests
// whose key is 2^64-1 itself are counted apart in info->special.
constexpr unsigned long long kEmptyKey = ~0ull;

__global__ void k_hist_insert(const unsigned long long *__restrict__ keys, uint64_t n,
                              unsigned long long *__restrict__ tkey, uint32_t *__restrict__ tcnt, int bits,
                              cr_plan_info_dev *info)
{
    const unsigned long long mask = (1ull << bits) - 1ull;
    const uint32_t lane = cr_lane();
    const uint32_t lt = (1u << lane) - 1u;
    for (uint64_t base = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) & ~31ull; base < n;
         base += (uint64_t)gridDim.x * blockDim.x) {
        const uint64_t i = base + lane;
        const bool valid = i < n;
        const unsigned long long key = valid ? keys[i] : kEmptyKey;
        const uint32_t vmask = __ballot_sync(0xffffffffu, valid);
        const uint32_t peers = __match_any_sync(0xffffffffu, key) & vmask;
        if (!valid || (peers & lt) != 0) continue;  // one leader per distinct key in the warp
        const uint32_t c = __popc(peers);
        if (key == kEmptyKey) {
            atomicAdd(&info->special, (unsigned long long)c);
            continue;
        }
        unsigned long long sl = key >> (64 - bits);
        for (;;) {
            unsigned long long cur = tkey[sl];
            if (cur == kEmptyKey) {
                cur = atomicCAS(&tkey[sl], kEmptyKey, key);
                if (cur == kEmptyKey) cur = key;
            }
            if (cur == key) {
                atomicAdd(&tcnt[sl], c);
                break;
            }
            sl = (sl + 1) & mask;  // at least twice as many slots as keys
        }
    }
}

// Occupied slots -> a dense list (order immaterial: it is sorted next).
// Occupied slots appended to a dense list (order free: the list is sorted next).
// A warp takes 8 x 32 consecutive slots and claims their places with one atomic:
// one atomic per 32 slots on the single counter serialised the launch.
constexpr int kCompactRounds = 8;
__global__ void k_hist_compact(const unsigned long long *__restrict__ tkey, const uint32_t *__restrict__ tcnt,
                               uint64_t slots, unsigned long long *__restrict__ lkey, uint32_t *__restrict__ lcnt,
                               cr_plan_info_dev *info)
{
    const uint32_t lane = cr_lane(), lt = (1u << lane) - 1u;
    constexpr uint64_t kSpan = 32ull * kCompactRounds;
    const uint64_t w0 = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint64_t nwarps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
    for (uint64_t base = w0 * kSpan; base < slots; base += nwarps * kSpan) {
        unsigned long long k[kCompactRounds];
        uint32_t bal[kCompactRounds], tot = 0;
#pragma unroll
        for (int r = 0; r < kCompactRounds; ++r) {
            const uint64_t s = base + 32ull * r + lane;
            k[r] = s < slots ? tkey[s] : kEmptyKey;
            bal[r] = __ballot_sync(0xffffffffu, k[r] != kEmptyKey);
            tot += (uint32_t)__popc(bal[r]);
        }
        if (!tot) continue;
        unsigned long long at = 0;
        if (lane == 0) at = atomicAdd(&info->U, (unsigned long long)tot);
        at = __shfl_sync(0xffffffffu, at, 0);
#pragma unroll
        for (int r = 0; r < kCompactRounds; ++r) {
            if (k[r] != kEmptyKey) {
                const unsigned long long pos = at + (uint32_t)__popc(bal[r] & lt);
                lkey[pos] = k[r];
                lcnt[pos] = tcnt[base + 32ull * r + lane];
            }
            at += (uint32_t)__popc(bal[r]);
        }
    }
    if (blockIdx.x == 0 && threadIdx.x == 0 && info->special) {
        // the key 2^64-1 was counted apart; it joins the list last
        const unsigned long long pos = atomicAdd(&info->U, 1ull);
        lkey[pos] = kEmptyKey;
        lcnt[pos] = (uint32_t)info->special;
    }
}

// ---- one-CTA stable LSD radix sort of the U distinct keys --------------------
// 1024 threads, 8-bit digits.  All passes' digit histograms are taken in one
// sweep.  A pass walks tiles of 4096 items; warp w owns items [128w, 128w+128)
// of a tile, ranks them in 4 rounds with __match_any_sync against warp-private
// digit counters, and one cross-warp prefix per digit turns the counters into
// offsets.  The next tile's items are loaded while the current one is ranked.
constexpr int kSmallBlock = 1024;
constexpr int kSmallWarps = kSmallBlock / 32;
constexpr int kSmallTile = kSmallBlock * 4;

struct small_sort_smem {
    uint32_t hist[8][256];             // digit counts of every pass, then running bases
    uint32_t wcnt[256][kSmallWarps + 1];  // per-warp digit counters of the current tile, digit-major
                                          // (row padded to 33 words: a warp reading one digit of every
                                          // warp, or every digit of one warp, hits 32 distinct banks)
};

template <typename K>
__device__ void cta_histograms(const K *kin, uint32_t n, int npass, small_sort_smem &sm)
{
    for (uint32_t x = threadIdx.x; x < 8 * 256; x += kSmallBlock) (&sm.hist[0][0])[x] = 0;
    __syncthreads();
    const uint32_t lt = (1u << cr_lane()) - 1u;
    for (uint32_t i0 = 0; i0 < n; i0 += kSmallBlock) {  // warp-uniform trip count
        const uint32_t i = i0 + threadIdx.x;
        const bool valid = i < n;
        const K key = valid ? kin[i] : (K)0;
        for (int p = 0; p < npass; ++p) {
            // one atomic per distinct digit in the warp: skewed digits do not serialise
            const uint32_t d = valid ? ((uint32_t)(key >> (8 * p)) & 0xffu) : 256u;
            const uint32_t peers = __match_any_sync(0xffffffffu, d);
            if (valid && (peers & lt) == 0) atomicAdd(&sm.hist[p][d], (uint32_t)__popc(peers));
        }
    }
    __syncthreads();
    // exclusive scan of each pass's 256 counts (warp p scans pass p, 8 digits per lane)
    const uint32_t warp = threadIdx.x >> 5, lane = cr_lane();
    if (warp < (uint32_t)npass) {
        uint32_t v[8], sum = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            v[j] = sm.hist[warp][lane * 8 + j];
            sum += v[j];
        }
        uint32_t inc = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            uint32_t u = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= (uint32_t)o) inc += u;
        }
        uint32_t run = inc - sum;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            sm.hist[warp][lane * 8 + j] = run;
            run += v[j];
        }
    }
    __syncthreads();
}

template <typename K>
__device__ void cta_radix_pass(const K *kin, const uint32_t *vin, K *kout, uint32_t *vout, uint32_t n, int pass,
                               small_sort_smem &sm)
{
    const uint32_t tid = threadIdx.x, lane = cr_lane(), warp = tid >> 5;
    const uint32_t lt = (1u << lane) - 1u;
    const int shift = 8 * pass;
    uint32_t *base = sm.hist[pass];
    K k[4];
    uint32_t v[4];
    auto load_tile = [&](uint32_t t0) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t i = t0 + warp * 128 + j * 32 + lane;
            if (i < n) {
                k[j] = kin[i];
                v[j] = vin ? vin[i] : i;
            }
        }
    };
    load_tile(0);
    for (uint32_t t0 = 0; t0 < n; t0 += kSmallTile) {
        K ck[4];
        uint32_t cv[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            ck[j] = k[j];
            cv[j] = v[j];
        }
        if (t0 + kSmallTile < n) load_tile(t0 + kSmallTile);
        for (uint32_t x = lane; x < 256; x += 32) sm.wcnt[x][warp] = 0;
        __syncwarp();
        uint32_t rank[4], dig[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t i = t0 + warp * 128 + j * 32 + lane;
            const bool valid = i < n;
            const uint32_t d = valid ? ((uint32_t)(ck[j] >> shift) & 0xffu) : 256u;
            const uint32_t peers = __match_any_sync(0xffffffffu, d);
            const uint32_t before = valid ? sm.wcnt[d][warp] : 0u;
            rank[j] = before + __popc(peers & lt);
            dig[j] = d;
            __syncwarp();
            if (valid && (peers & lt) == 0) sm.wcnt[d][warp] = before + __popc(peers);
            __syncwarp();
        }
        __syncthreads();
        // per digit, exclusive prefix over the warps (warp w scans digits 8w..8w+7)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const uint32_t dd = warp * 8 + j;
            const uint32_t c = sm.wcnt[dd][lane];
            uint32_t inc = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                uint32_t u = __shfl_up_sync(0xffffffffu, inc, o);
                if (lane >= (uint32_t)o) inc += u;
            }
            const uint32_t b0 = base[dd];
            sm.wcnt[dd][lane] = b0 + inc - c;
            __syncwarp();
            if (lane == 31) base[dd] = b0 + inc;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (dig[j] < 256u) {
                const uint32_t pos = sm.wcnt[dig[j]][warp] + rank[j];
                kout[pos] = ck[j];
                vout[pos] = cv[j];
            }
        }
        __syncthreads();
    }
}

// Sorts the U distinct (key, count) pairs: key ascending into (ukey, ucnt), then
// stably by (n - count) into `order` = admission order (count desc, key asc).
// Stable LSD sort of U (key, count) pairs in one CTA: by key (8 passes), the
// sorted pairs written to ukey/ucnt, then by n - count (ceil(cbits/8) passes)
// giving order = positions in ukey/ucnt by (count desc, key asc).  The pairs
// start in (ki, vi) and ping-pong with (ko, vo).
__device__ __forceinline__ void small_sort(small_sort_smem &sm, uint32_t U, unsigned long long n, int cbits,
                                           unsigned long long *ki, uint32_t *vi, unsigned long long *ko,
                                           uint32_t *vo, unsigned long long *__restrict__ ukey,
                                           unsigned long long *__restrict__ ucnt, uint32_t *s32A, uint32_t *s32B,
                                           uint32_t *o32A, uint32_t *o32B, uint32_t *__restrict__ order)
{
    cta_histograms<unsigned long long>(ki, U, 8, sm);
    for (int pass = 0; pass < 8; ++pass) {
        cta_radix_pass<unsigned long long>(ki, vi, ko, vo, U, pass, sm);
        unsigned long long *tk = ki; ki = ko; ko = tk;
        uint32_t *tv = vi; vi = vo; vo = tv;
    }
    for (uint32_t u = threadIdx.x; u < U; u += kSmallBlock) {
        ukey[u] = ki[u];
        ucnt[u] = vi[u];
        s32A[u] = (uint32_t)(n - vi[u]);
    }
    __syncthreads();
    const int cpass = (cbits + 7) / 8;
    uint32_t *si = s32A, *so = s32B, *oi = nullptr, *oo = o32A;
    cta_histograms<uint32_t>(si, U, cpass, sm);
    for (int pass = 0; pass < cpass; ++pass) {
        cta_radix_pass<uint32_t>(si, oi, so, oo, U, pass, sm);
        uint32_t *t = si; si = so; so = t;
        oi = oo;
        oo = (oo == o32A) ? o32B : o32A;
    }
    for (uint32_t u = threadIdx.x; u < U; u += kSmallBlock) order[u] = oi ? oi[u] : u;
}

__global__ void __launch_bounds__(kSmallBlock) k_plan_sort(const cr_plan_info_dev *info, unsigned long long n,
                                                           int cbits, unsigned long long *kA, uint32_t *vA,
                                                           unsigned long long *kB, uint32_t *vB,
                                                           unsigned long long *__restrict__ ukey,
                                                           unsigned long long *__restrict__ ucnt, uint32_t *s32A,
                                                           uint32_t *s32B, uint32_t *o32A, uint32_t *o32B,
                                                           uint32_t *__restrict__ order)
{
    __shared__ small_sort_smem sm;
    small_sort(sm, (uint32_t)info->U, n, cbits, kA, vA, kB, vB, ukey, ucnt, s32A, s32B, o32A, o32B, order);
}

// Admission reads only the first keys of the (count desc, key asc) order: at
// most C = R*W of them, since every k_b >= 1.  One CTA finds the count lam_C
// of the C-th largest count (two-level radix select over the counts), moves
// the keys with count >= lam_C (ties at lam_C included) to the front, sorts
// only those, and writes the other keys after them in table order.  order then
// covers the S candidates, every key admission can reach; the plan's per-key
// arrays still hold all U keys.
__device__ __forceinline__ void select_from_top(const uint32_t *hist, uint32_t nbk, unsigned long long want,
                                                uint32_t *res)
{
    // lane l sums buckets [nbk - (l+1) per, nbk - l per): lane 0 holds the top
    const uint32_t lane = cr_lane(), per = (nbk + 31) / 32;
    const int hi = (int)nbk - (int)(lane * per), lo = hi - (int)per;
    unsigned long long c = 0;
    for (int b = hi - 1; b >= lo && b >= 0; --b) c += hist[b];
    unsigned long long inc = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= (uint32_t)o) inc += y;
    }
    const bool here = inc >= want && inc - c < want;
    if (here) {
        unsigned long long run = inc - c;  // counted in buckets above this lane's chunk
        for (int b = hi - 1; b >= lo && b >= 0; --b) {
            if (run + hist[b] >= want) {
                res[0] = (uint32_t)b;
                res[1] = (uint32_t)run;
                break;
            }
            run += hist[b];
        }
    }
}

__global__ void __launch_bounds__(kSmallBlock) k_plan_topk(cr_plan_info_dev *info, unsigned long long n, int cbits,
                                                           unsigned long long cmax, unsigned long long *kA,
                                                           uint32_t *vA, unsigned long long *kB, uint32_t *vB,
                                                           unsigned long long *__restrict__ ukey,
                                                           unsigned long long *__restrict__ ucnt, uint32_t *s32A,
                                                           uint32_t *s32B, uint32_t *o32A, uint32_t *o32B,
                                                           uint32_t *__restrict__ order)
{
    __shared__ small_sort_smem sm;
    __shared__ uint32_t res[4];
    __shared__ uint32_t wtot[2][kSmallWarps];
    const uint32_t U = (uint32_t)info->U;
    const uint32_t tid = threadIdx.x, lane = cr_lane(), warp = tid >> 5, lt = (1u << lane) - 1u;
    if (U <= cmax) {  // every key is a candidate
        small_sort(sm, U, n, cbits, kA, vA, kB, vB, ukey, ucnt, s32A, s32B, o32A, o32B, order);
        if (tid == 0) info->S = U;
        return;
    }
    uint32_t *h1 = &sm.hist[0][0], *h2 = h1 + 1024;
    const int nb = 64 - __clzll(n);  // counts are <= n < 2^nb
    const int s1 = nb > 10 ? nb - 10 : 0;
    const uint32_t nb1 = 1u << (nb - s1), nb2 = 1u << s1;
    for (uint32_t x = tid; x < 2048; x += kSmallBlock) h1[x] = 0;
    __syncthreads();
    const uint32_t Ur = (U + kSmallBlock - 1) / kSmallBlock * kSmallBlock;
    for (uint32_t u = tid; u < Ur; u += kSmallBlock) {  // level 1: high bits of the count
        const uint32_t b = u < U ? (vA[u] >> s1) : 0xffffffffu;
        const uint32_t peers = __match_any_sync(0xffffffffu, b);
        if (b != 0xffffffffu && (peers & lt) == 0) atomicAdd(&h1[b], (uint32_t)__popc(peers));
    }
    __syncthreads();
    if (warp == 0) select_from_top(h1, nb1, cmax, res);
    __syncthreads();
    const uint32_t b1 = res[0], above1 = res[1];
    for (uint32_t u = tid; u < Ur; u += kSmallBlock) {  // level 2: low bits inside bucket b1
        const uint32_t v = u < U ? vA[u] : 0u;
        const uint32_t b = (u < U && (v >> s1) == b1) ? (v & (nb2 - 1u)) : 0xffffffffu;
        const uint32_t peers = __match_any_sync(0xffffffffu, b);
        if (b != 0xffffffffu && (peers & lt) == 0) atomicAdd(&h2[b], (uint32_t)__popc(peers));
    }
    __syncthreads();
    if (warp == 0) select_from_top(h2, nb2, cmax - above1, res + 2);
    __syncthreads();
    const uint32_t thr = (b1 << s1) | res[2];
    const uint32_t S = above1 + res[3] + h2[res[2]];
    // stable partition: candidates to (kB, vB)[0..S), the rest to ukey/ucnt[S..U)
    uint32_t run_c = 0, run_o = 0;
    for (uint32_t base = 0; base < U; base += kSmallBlock) {
        const uint32_t u = base + tid;
        const bool valid = u < U;
        const unsigned long long key = valid ? kA[u] : 0ull;
        const uint32_t cnt = valid ? vA[u] : 0u;
        const bool cand = valid && cnt >= thr;
        const uint32_t bc = __ballot_sync(0xffffffffu, cand), bo = __ballot_sync(0xffffffffu, valid && !cand);
        if (lane == 0) {
            wtot[0][warp] = __popc(bc);
            wtot[1][warp] = __popc(bo);
        }
        __syncthreads();
        uint32_t pc = 0, po = 0, tc = 0, to = 0;
        for (uint32_t w = 0; w < kSmallWarps; ++w) {
            const uint32_t a = wtot[0][w], o = wtot[1][w];
            if (w < warp) {
                pc += a;
                po += o;
            }
            tc += a;
            to += o;
        }
        if (cand) {
            const uint32_t pos = run_c + pc + __popc(bc & lt);
            kB[pos] = key;
            vB[pos] = cnt;
        } else if (valid) {
            const uint32_t pos = S + run_o + po + __popc(bo & lt);
            ukey[pos] = key;
            ucnt[pos] = cnt;
        }
        run_c += tc;
        run_o += to;
        __syncthreads();
    }
    small_sort(sm, S, n, cbits, kB, vB, kA, vA, ukey, ucnt, s32A, s32B, o32A, o32B, order);
    if (tid == 0) info->S = S;
}
// Intervals of up to this many requests sort their histogram in one CTA (one
// launch, one SM, so the planner barely touches the SMs the overlapped main
// stream uses); larger ones in device-wide radix passes.
constexpr uint64_t kPlanSortOneCta = 524288;

// Large histograms (multi-CTA passes): after the key sort, the per-key output
// and the count-descending sort key n - count.
__global__ void k_plan_sorted_keys(const cr_plan_info_dev *info, unsigned long long n,
                                   const unsigned long long *__restrict__ k, const uint32_t *__restrict__ c,
                                   unsigned long long *__restrict__ ukey, unsigned long long *__restrict__ ucnt,
                                   uint32_t *__restrict__ s32)
{
    const unsigned long long U = info->U;
    for (uint64_t u = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; u < U; u += (uint64_t)gridDim.x * blockDim.x) {
        ukey[u] = k[u];
        ucnt[u] = c[u];
        s32[u] = (uint32_t)(n - c[u]);
    }
}

__global__ void k_plan_copy_order(cr_plan_info_dev *info, const uint32_t *__restrict__ src,
                                  uint32_t *__restrict__ order)
{
    const unsigned long long U = info->U;
    if (blockIdx.x == 0 && threadIdx.x == 0) info->S = U;  // every key ordered
    for (uint64_t u = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; u < U; u += (uint64_t)gridDim.x * blockDim.x)
        order[u] = src[u];
}

// Eq. 1: k_b = min(R, max(1, ceil(lambda * den / num))); NOREPL: 1.
__device__ __forceinline__ uint32_t eq1_kb(unsigned long long lam, unsigned long long num, unsigned long long den,
                                           uint32_t R)
{
    unsigned long long a = lam * den;
    unsigned long long k = a / num + ((a % num) != 0ull);
    if (k < 1ull) k = 1ull;
    if (k > R) k = R;
    return (uint32_t)k;
}

__global__ void k_plan_kb(const uint32_t *__restrict__ order, const unsigned long long *__restrict__ ucnt,
                          uint64_t n, const cr_plan_info_dev *info, unsigned long long num, unsigned long long den,
                          uint32_t R, int norepl, unsigned long long *__restrict__ kk)
{
    const unsigned long long S = info->S;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < S; a += (uint64_t)gridDim.x * blockDim.x)
        kk[a] = norepl ? 1ull : eq1_kb(ucnt[order[a]], num, den, R);
}

// Admission: the longest prefix of the order whose inclusive k-sum stays <= C.
__global__ void k_plan_admit(const unsigned long long *__restrict__ kscan, cr_plan_info_dev *info,
                             unsigned long long C)
{
    const unsigned long long S = info->S;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < S; a += (uint64_t)gridDim.x * blockDim.x) {
        if (kscan[a] <= C && (a + 1 == S || kscan[a + 1] > C)) {
            info->n_adm = a + 1;
            info->sum_k = kscan[a];
        }
    }
}

__global__ void k_plan_fill(const uint32_t *__restrict__ order, const unsigned long long *__restrict__ ukey,
                            const unsigned long long *__restrict__ ucnt, const unsigned long long *__restrict__ kscan,
                            cr_plan_info_dev *info, unsigned long long *__restrict__ adm_key,
                            unsigned long long *__restrict__ adm_cnt, uint32_t *__restrict__ adm_k,
                            uint32_t *__restrict__ koff)
{
    const unsigned long long na = info->n_adm;
    unsigned long long lam = 0;
    uint32_t kmax = 0;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < na; a += (uint64_t)gridDim.x * blockDim.x) {
        uint32_t u = order[a];
        {
            uint32_t k = (uint32_t)(kscan[a] - (a ? kscan[a - 1] : 0ull));
            adm_key[a] = ukey[u];
            adm_cnt[a] = ucnt[u];
            adm_k[a] = k;
            koff[a] = (uint32_t)(kscan[a] - k);
            kmax = k > kmax ? k : kmax;
            if (a + 1 == na) koff[na] = (uint32_t)kscan[a];
            lam += ucnt[u];
        }
    }
    lam = cr_warp_sum_u64(lam);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
    if (cr_lane() == 0) {
        if (lam) atomicAdd(&info->adm_lam, lam);
        if (kmax) atomicMax(&info->max_k, (unsigned long long)kmax);
    }
}

// Admission for every plan of a build in one launch (intervals sorted by one
// CTA, whose admission candidates are few): one 1024-thread CTA per plan clears
// its table, runs Eq. 1 and the inclusive k-sum over the candidates tile by
// tile (a block scan), admits the prefix that fits C (Algorithm 1 admission
// step; it stops at the first tile with a key that does not fit), writes the
// admitted arrays, the cold tail n - admitted requests and the initial loads.
struct admit_job {
    cr_plan_info_dev *info;
    const unsigned long long *init_load;
    unsigned long long *load, *adm_key, *adm_cnt;
    uint32_t *adm_k, *koff;
    uint4 *table;
    unsigned long long table_slots, C, num, den;
    unsigned long long *ukey_out, *ucnt_out;  // copy of the histogram, or null
    uint32_t R;
    int norepl;
};

struct admit_jobs {
    admit_job j[16];
};

__device__ __forceinline__ unsigned long long warp_incl_scan_u64(unsigned long long x, uint32_t lane)
{
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= (uint32_t)o) x += y;
    }
    return x;
}

__global__ void __launch_bounds__(kSmallBlock) k_plan_admit_cta(const __grid_constant__ admit_jobs jobs,
                                                                const cr_plan_info_dev *info0,
                                                                const uint32_t *__restrict__ order,
                                                                const unsigned long long *__restrict__ ukey,
                                                                const unsigned long long *__restrict__ ucnt,
                                                                unsigned long long n, uint32_t *status)
{
    const admit_job J = jobs.j[blockIdx.x];
    __shared__ unsigned long long wsum[kSmallWarps], wlam[kSmallWarps];
    __shared__ uint32_t wkmax[kSmallWarps];
    __shared__ unsigned long long s_cold;
    const uint32_t tid = threadIdx.x, lane = cr_lane(), warp = tid >> 5;
    for (unsigned long long x = tid; x < J.table_slots; x += kSmallBlock)
        J.table[x] = make_uint4(0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu);  // all slots empty
    if (J.ukey_out) {
        const unsigned long long U = info0->U;
        for (unsigned long long x = tid; x < U; x += kSmallBlock) {
            J.ukey_out[x] = ukey[x];
            J.ucnt_out[x] = ucnt[x];
        }
    }
    const unsigned long long S = info0->S;
    unsigned long long carry = 0, n_adm = 0, lam = 0;
    uint32_t kmax = 0;
    for (unsigned long long base = 0; base < S; base += kSmallBlock) {
        const unsigned long long a = base + tid;
        const bool valid = a < S;
        const uint32_t u = valid ? order[a] : 0u;
        const unsigned long long cnt = valid ? ucnt[u] : 0ull;
        const uint32_t k = !valid ? 0u : (J.norepl ? 1u : eq1_kb(cnt, J.num, J.den, J.R));
        const unsigned long long x = warp_incl_scan_u64(k, lane);
        if (lane == 31) wsum[warp] = x;
        __syncthreads();
        if (warp == 0) wsum[lane] = warp_incl_scan_u64(wsum[lane], lane);
        __syncthreads();
        const unsigned long long ks = carry + x + (warp ? wsum[warp - 1] : 0ull);
        const bool adm = valid && ks <= J.C;  // ks grows with a: the admitted keys are a prefix
        const unsigned long long nt = (unsigned long long)__syncthreads_count(adm);
        if (adm) {
            J.adm_key[a] = ukey[u];
            J.adm_cnt[a] = cnt;
            J.adm_k[a] = k;
            J.koff[a] = (uint32_t)(ks - k);
            lam += cnt;
            kmax = k > kmax ? k : kmax;
            if (a + 1 == base + nt) {  // the last admitted key so far
                J.koff[a + 1] = (uint32_t)ks;
                J.info->sum_k = ks;
            }
        }
        n_adm += nt;
        const unsigned long long tile = wsum[kSmallWarps - 1];
        __syncthreads();
        if (nt < (S - base < kSmallBlock ? S - base : (unsigned long long)kSmallBlock)) break;
        carry += tile;
    }
    lam = cr_warp_sum_u64(lam);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
    if (lane == 0) {
        wlam[warp] = lam;
        wkmax[warp] = kmax;
    }
    __syncthreads();
    if (tid == 0) {
        unsigned long long L = 0;
        uint32_t km = 0;
        for (int w = 0; w < kSmallWarps; ++w) {
            L += wlam[w];
            km = wkmax[w] > km ? wkmax[w] : km;
        }
        cr_plan_info_dev *I = J.info;
        I->n = n;
        I->U = info0->U;
        I->S = S;
        I->special = info0->special;
        I->n_adm = n_adm;
        if (n_adm == 0) {
            I->sum_k = 0;
            J.koff[0] = 0;
        }
        I->max_k = km;
        I->adm_lam = L;
        I->cold = n - L;
        s_cold = n - L;
    }
    __syncthreads();
    const unsigned long long share = s_cold / J.R;
    for (uint32_t r = tid; r < J.R; r += kSmallBlock) {
        const unsigned long long v = J.init_load ? J.init_load[r] : share;
        if (v >= kLoadLimit) atomicOr(status, CR_FLAG_OVERFLOW);
        J.load[r] = v;
    }
}

// Cold tail: every request of a key that was not admitted (n - admitted).
__global__ void k_plan_init_load(cr_plan_info_dev *info, const unsigned long long *__restrict__ init_load,
                                 uint32_t R, unsigned long long *__restrict__ load, uint32_t *status)
{
    const unsigned long long cold = info->n - info->adm_lam;
    if (blockIdx.x == 0 && threadIdx.x == 0) info->cold = cold;
    const unsigned long long share = cold / R;
    for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
        unsigned long long v = init_load ? init_load[r] : share;
        if (v >= kLoadLimit) atomicOr(status, CR_FLAG_OVERFLOW);
        load[r] = v;
    }
}

// LPT placement (Algorithm 1 placement loop) on one warp.  Lane l owns the
// destinations r = l, l+32, ... (their loads and "taken" flags are touched by
// no other lane) and caches the smallest packed key (L[r] << 16 | r) among its
// untaken ones; packing makes (L, r) order a plain integer order (L < 2^47 is
// enforced, r < 2^13).  Each job is one warp minimum of the 32 cached keys,
// taken with two redux.sync reductions (high word, then low word).
__device__ __forceinline__ unsigned long long lane_min(const unsigned long long *L, const unsigned char *taken,
                                                       uint32_t R, uint32_t lane)
{
    unsigned long long m = ~0ull;
    for (uint32_t r = lane; r < R; r += 32) {
        if (taken[r]) continue;
        const unsigned long long v = (L[r] << 16) | r;
        m = v < m ? v : m;
    }
    return m;
}

__device__ __forceinline__ unsigned long long warp_min_u64(unsigned long long v)
{
    const uint32_t hi = __reduce_min_sync(0xffffffffu, (uint32_t)(v >> 32));
    const uint32_t lo = __reduce_min_sync(0xffffffffu, (uint32_t)(v >> 32) == hi ? (uint32_t)v : 0xffffffffu);
    return ((unsigned long long)hi << 32) | lo;
}

__global__ void __launch_bounds__(32) k_plan_lpt(const cr_plan_info_dev *info,
                                                 const unsigned long long *__restrict__ adm_cnt,
                                                 const uint32_t *__restrict__ adm_k,
                                                 const uint32_t *__restrict__ koff, uint32_t R,
                                                 unsigned long long *__restrict__ load_g,
                                                 uint16_t *__restrict__ members,
                                                 unsigned long long *__restrict__ jobs, uint32_t *status)
{
    extern __shared__ unsigned long long smem_u64[];
    unsigned long long *L = smem_u64;                                  // [R]
    unsigned char *taken = reinterpret_cast<unsigned char *>(L + R);   // [R]
    const uint32_t lane = cr_lane();
    for (uint32_t r = lane; r < R; r += 32) {
        L[r] = load_g[r];
        taken[r] = 0;
    }
    unsigned long long m = lane_min(L, taken, R, lane);
    const unsigned long long na = info->n_adm;
    bool overflow = false;
    // the admitted keys' (lambda, k, offset) are staged 32 at a time, one per lane,
    // and broadcast with shuffles: no global-memory latency on the sequential chain
    unsigned long long st_lam = 0;
    uint32_t st_k = 0, st_off = 0;
    for (unsigned long long a = 0; a < na; ++a) {
        const uint32_t slot = (uint32_t)(a & 31ull);
        if (slot == 0) {
            const unsigned long long ia = a + lane;
            if (ia < na) {
                st_lam = adm_cnt[ia];
                st_k = adm_k[ia];
                st_off = koff[ia];
            }
        }
        const uint32_t k = __shfl_sync(0xffffffffu, st_k, slot);
        const uint32_t base = __shfl_sync(0xffffffffu, st_off, slot);
        const unsigned long long lam = __shfl_sync(0xffffffffu, st_lam, slot);
        const unsigned long long q = k == 1 ? lam : lam / k, rem = k == 1 ? 0ull : lam % k;
        bool took = false;
        for (uint32_t s = 0; s < k; ++s) {
            const unsigned long long best = warp_min_u64(m);
            const uint32_t br = (uint32_t)(best & 0xffffu);
            const unsigned long long job = q + (s < rem ? 1ull : 0ull);
            if (lane == 0) {
                members[base + s] = (uint16_t)br;
                jobs[base + s] = job;
            }
            if ((br & 31u) == lane) {
                // a chosen destination is not eligible again for this key
                if (k > 1) {
                    taken[br] = 1;
                    took = true;
                }
                const unsigned long long nl = L[br] + job;
                if (nl >= kLoadLimit) overflow = true;
                L[br] = nl;
                m = lane_min(L, taken, R, lane);
            }
        }
        if (took) {  // release this key's destinations for the next key
            for (uint32_t r = lane; r < R; r += 32) taken[r] = 0;
            m = lane_min(L, taken, R, lane);
        }
    }
    for (uint32_t r = lane; r < R; r += 32) load_g[r] = L[r];
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(status, CR_FLAG_OVERFLOW);
}

// Slot-capped LPT (per-destination budget of W replicas; this library's
// reading of a byte-aware placement): as k_plan_lpt, but a destination that
// holds W replicas is no longer eligible, and a key gets
// k = min(k_b, destinations with a free slot) replicas (at least one: the
// aggregate admission leaves a free slot for every admitted key).  Member
// offsets are written compactly, adm_k receives the placed counts and
// info->sum_k their sum.
__device__ __forceinline__ unsigned long long lane_min_capped(const unsigned long long *L,
                                                              const unsigned char *taken, const uint32_t *slots,
                                                              uint32_t W, uint32_t R, uint32_t lane)
{
    unsigned long long m = ~0ull;
    for (uint32_t r = lane; r < R; r += 32) {
        if (taken[r] || slots[r] >= W) continue;
        const unsigned long long v = (L[r] << 16) | r;
        m = v < m ? v : m;
    }
    return m;
}

__global__ void __launch_bounds__(32) k_plan_lpt_capped(cr_plan_info_dev *info,
                                                        const unsigned long long *__restrict__ adm_cnt,
                                                        uint32_t *__restrict__ adm_k, uint32_t *__restrict__ koff,
                                                        uint32_t R, uint32_t W, unsigned long long *__restrict__ load_g,
                                                        uint16_t *__restrict__ members,
                                                        unsigned long long *__restrict__ jobs, uint32_t *status)
{
    extern __shared__ unsigned long long smem_u64[];
    unsigned long long *L = smem_u64;                                      // [R]
    uint32_t *slots = reinterpret_cast<uint32_t *>(L + R);                 // [R] replicas held
    unsigned char *taken = reinterpret_cast<unsigned char *>(slots + R);   // [R]
    const uint32_t lane = cr_lane();
    for (uint32_t r = lane; r < R; r += 32) {
        L[r] = load_g[r];
        slots[r] = 0;
        taken[r] = 0;
    }
    __syncwarp();
    unsigned long long m = lane_min_capped(L, taken, slots, W, R, lane);
    const unsigned long long na = info->n_adm;
    uint32_t free_dest = R;  // destinations with a free slot (uniform over the warp)
    uint32_t pos = 0;        // compact member offset
    bool overflow = false;
    unsigned long long st_lam = 0;
    uint32_t st_k = 0;
    for (unsigned long long a = 0; a < na; ++a) {
        const uint32_t slot = (uint32_t)(a & 31ull);
        if (slot == 0) {
            const unsigned long long ia = a + lane;
            if (ia < na) {
                st_lam = adm_cnt[ia];
                st_k = adm_k[ia];
            }
        }
        const uint32_t kb = __shfl_sync(0xffffffffu, st_k, slot);
        const unsigned long long lam = __shfl_sync(0xffffffffu, st_lam, slot);
        const uint32_t k = kb < free_dest ? kb : free_dest;
        if (lane == 0) {
            koff[a] = pos;
            adm_k[a] = k;
        }
        if (k == 0) continue;
        const unsigned long long q = lam / k, rem = lam % k;
        bool took = false;
        for (uint32_t s = 0; s < k; ++s) {
            const unsigned long long best = warp_min_u64(m);
            const uint32_t br = (uint32_t)(best & 0xffffu);
            const unsigned long long job = q + (s < rem ? 1ull : 0ull);
            if (lane == 0) {
                members[pos + s] = (uint16_t)br;
                jobs[pos + s] = job;
            }
            bool filled = false;
            if ((br & 31u) == lane) {
                if (k > 1) {
                    taken[br] = 1;
                    took = true;
                }
                const unsigned long long nl = L[br] + job;
                if (nl >= kLoadLimit) overflow = true;
                L[br] = nl;
                filled = ++slots[br] == W;
                m = lane_min_capped(L, taken, slots, W, R, lane);
            }
            free_dest -= __shfl_sync(0xffffffffu, filled ? 1u : 0u, br & 31u);
        }
        if (took) {  // release this key's destinations for the next key
            for (uint32_t r = lane; r < R; r += 32) taken[r] = 0;
            m = lane_min_capped(L, taken, slots, W, R, lane);
        }
        pos += k;
    }
    if (lane == 0) {
        koff[na] = pos;
        info->sum_k = pos;
    }
    for (uint32_t r = lane; r < R; r += 32) load_g[r] = L[r];
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(status, CR_FLAG_OVERFLOW);
}

// LPT for R <= 32: lane i holds the i-th smallest packed key (L << 16 | r), so
// T(b) for a key with k_b = k is lanes 0..k-1.  After a single-copy job the
// grown key is re-inserted with one ballot and one shuffle; after a replicated
// key the warp is re-sorted with a bitonic network.
__device__ __forceinline__ unsigned long long warp_bitonic_sort(unsigned long long x)
{
    const uint32_t lane = cr_lane();
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const unsigned long long y = __shfl_xor_sync(0xffffffffu, x, stride);
            const bool up = (lane & size) == 0;
            const bool lower = (lane & stride) == 0;
            const unsigned long long lo = x < y ? x : y, hi = x < y ? y : x;
            x = (lower == up) ? lo : hi;
        }
    }
    return x;
}

__device__ __forceinline__ void lpt32_body(const cr_plan_info_dev *info,
                                                   const unsigned long long *__restrict__ adm_cnt,
                                                   const uint32_t *__restrict__ adm_k,
                                                   const uint32_t *__restrict__ koff, uint32_t R,
                                                   unsigned long long *__restrict__ load_g,
                                                   uint16_t *__restrict__ members,
                                                   unsigned long long *__restrict__ jobs, uint32_t *status)
{
    const uint32_t lane = cr_lane();
    unsigned long long key = lane < R ? ((load_g[lane] << 16) | lane) : ~0ull;
    key = warp_bitonic_sort(key);
    const unsigned long long na = info->n_adm;
    bool overflow = false;
    unsigned long long st_lam = 0;
    uint32_t st_k = 0, st_off = 0;
    for (unsigned long long a = 0; a < na; ++a) {
        const uint32_t slot = (uint32_t)(a & 31ull);
        if (slot == 0) {
            const unsigned long long ia = a + lane;
            if (ia < na) {
                st_lam = adm_cnt[ia];
                st_k = adm_k[ia];
                st_off = koff[ia];
            }
        }
        const uint32_t k = __shfl_sync(0xffffffffu, st_k, slot);
        const uint32_t base = __shfl_sync(0xffffffffu, st_off, slot);
        const unsigned long long lam = __shfl_sync(0xffffffffu, st_lam, slot);
        if (k == 1) {
            const unsigned long long nk = __shfl_sync(0xffffffffu, key, 0) + (lam << 16);
            if (lane == 0) {
                members[base] = (uint16_t)(key & 0xffffu);
                jobs[base] = lam;
                if ((nk >> 16) >= kLoadLimit) overflow = true;
            }
            // lanes 1..pos hold keys below the grown one: shift them down one lane
            const uint32_t below = __ballot_sync(0xffffffffu, lane > 0 && key < nk);
            const uint32_t pos = __popc(below);
            const unsigned long long up = __shfl_down_sync(0xffffffffu, key, 1);
            key = lane < pos ? up : (lane == pos ? nk : key);
        } else {
            const unsigned long long q = lam / k, rem = lam % k;
            if (lane < k) {
                const unsigned long long job = q + (lane < rem ? 1ull : 0ull);
                members[base + lane] = (uint16_t)(key & 0xffffu);
                jobs[base + lane] = job;
                key += job << 16;
                if ((key >> 16) >= kLoadLimit) overflow = true;
            }
            key = warp_bitonic_sort(key);
        }
    }
    if (lane < R) load_g[key & 0xffffu] = key >> 16;
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(status, CR_FLAG_OVERFLOW);
}

__global__ void __launch_bounds__(32) k_plan_lpt32(const cr_plan_info_dev *info,
                                                   const unsigned long long *__restrict__ adm_cnt,
                                                   const uint32_t *__restrict__ adm_k,
                                                   const uint32_t *__restrict__ koff, uint32_t R,
                                                   unsigned long long *__restrict__ load_g,
                                                   uint16_t *__restrict__ members,
                                                   unsigned long long *__restrict__ jobs, uint32_t *status)
{
    lpt32_body(info, adm_cnt, adm_k, koff, R, load_g, members, jobs, status);
}

// Placement jobs of several plans in one launch (the block index picks the plan).
struct place_job {
    const cr_plan_info_dev *info;
    const unsigned long long *adm_cnt;
    const uint32_t *adm_k, *koff;
    unsigned long long *load, *jobs;
    uint16_t *members;
    unsigned long long seed, epoch;
    uint32_t R;
};

struct place_jobs {
    place_job j[16];
};

__global__ void __launch_bounds__(32) k_plan_lpt32_multi(const __grid_constant__ place_jobs pj, uint32_t *status)
{
    const place_job &J = pj.j[blockIdx.x];
    lpt32_body(J.info, J.adm_cnt, J.adm_k, J.koff, J.R, J.load, J.members, J.jobs, status);
}

// LPT for 32 < R <= 1024, all LPT plans of one build at once (one warp per
// plan).  Lane l holds the packed keys of destinations l, l+32, ... in NE
// registers and their minimum; a job is one warp minimum (two redux.sync),
// then the owner lane updates the chosen register and recomputes its minimum
// with a tree over registers.  Destinations chosen earlier for the same key
// are masked out by a per-lane bit set.
struct lpt_job {
    const cr_plan_info_dev *info;
    const unsigned long long *adm_cnt;
    const uint32_t *adm_k, *koff;
    unsigned long long *load;
    uint16_t *members;
    unsigned long long *jobs;
    uint32_t R;
};

struct lpt_jobs {
    lpt_job j[16];
};

template <int NE>
__device__ __forceinline__ unsigned long long reg_min(const unsigned long long (&v)[NE], uint32_t taken)
{
    unsigned long long t[NE];
#pragma unroll
    for (int j = 0; j < NE; ++j) t[j] = ((taken >> j) & 1u) ? ~0ull : v[j];
#pragma unroll
    for (int w = NE / 2; w > 0; w >>= 1) {
#pragma unroll
        for (int j = 0; j < w; ++j) t[j] = t[j + w] < t[j] ? t[j + w] : t[j];
    }
    return t[0];
}

// Runs of keys with k_b = 1 and equal λ = q (Algorithm 1's loop over such a
// run, done at once).  Each greedy pick is a current minimum (L_r, r) and
// raising it by q keeps later picks no smaller, so the m picks are the m
// smallest pairs (L_r + j q, r), j >= 0.  With L_r = q l_r + f_r (0 <= f_r < q)
// pair (r, j) sorts by (l_r + j, f_r, r): picks come in rounds t = l_r + j,
// each visiting {r : l_r <= t} in (f_r, r) order.  Between two consecutive
// distinct levels l the visited set is fixed, so that stretch of rounds cycles
// through it.  Cost: one pass over R per distinct level reached, plus the
// output writes, instead of one warp minimum per key.
struct lpt_run_smem {
    uint16_t order[1024];  // destinations by (f_r, r)
    uint16_t cyc[1024];    // destinations visited in the current stretch, in that order
    uint32_t lev[1024];    // l_r
    uint32_t add[1024];    // jobs given to r in this run; first q buckets reused for the sort
};

template <int NE>
__device__ __forceinline__ bool lpt_equal_run(unsigned long long (&v)[NE], uint32_t R, unsigned long long q,
                                              unsigned long long m, uint32_t base, uint16_t *__restrict__ members,
                                              unsigned long long *__restrict__ jobs, lpt_run_smem &S,
                                              bool &overflow)
{
    const uint32_t lane = cr_lane(), lt = (1u << lane) - 1u;
    if (q == 0 || q > 1024) return false;
    unsigned long long lmax = 0;
#pragma unroll
    for (int j = 0; j < NE; ++j)
        if (lane + 32u * j < R) lmax = max(lmax, v[j] >> 16);
    if (~cr_warp_min_u64(~lmax) >= (1ull << 31)) return false;  // levels in 32 bits
    const uint32_t q32 = (uint32_t)q;
    // counting sort by phase f_r, stable in r
    for (uint32_t x = lane; x < q32; x += 32) S.add[x] = 0;
    __syncwarp();
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        const uint32_t r = lane + 32u * j;
        if (r < R) {
            const uint32_t L = (uint32_t)(v[j] >> 16);
            S.lev[r] = L / q32;
            atomicAdd(&S.add[L % q32], 1u);
        }
    }
    __syncwarp();
    {
        const uint32_t per = (q32 + 31) / 32, x0 = lane * per;
        uint32_t run = 0;
        for (uint32_t x = x0; x < x0 + per && x < q32; ++x) run += S.add[x];
        uint32_t inc = run;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= (uint32_t)o) inc += y;
        }
        uint32_t off = inc - run;
        __syncwarp();
        for (uint32_t x = x0; x < x0 + per && x < q32; ++x) {
            const uint32_t c = S.add[x];
            S.add[x] = off;
            off += c;
        }
    }
    __syncwarp();
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        const uint32_t r = lane + 32u * j;
        const uint32_t f = r < R ? (uint32_t)(v[j] >> 16) % q32 : 0xffffffffu;
        const uint32_t peers = __match_any_sync(0xffffffffu, f);
        const uint32_t at = r < R ? S.add[f] : 0u;
        __syncwarp();
        if (r < R) {
            S.order[at + __popc(peers & lt)] = (uint16_t)r;
            if ((peers & lt) == 0) S.add[f] = at + __popc(peers);
        }
        __syncwarp();
    }
    for (uint32_t x = lane; x < R; x += 32) S.add[x] = 0;
    __syncwarp();
    // stretches of rounds between consecutive distinct levels
    uint32_t T = 0xffffffffu;
#pragma unroll
    for (int j = 0; j < NE; ++j)
        if (lane + 32u * j < R) T = min(T, S.lev[lane + 32u * j]);
    T = __reduce_min_sync(0xffffffffu, T);
    unsigned long long left = m, done = 0;
    while (left) {
        uint32_t n_in = 0, nxt = 0xffffffffu;
#pragma unroll
        for (int j = 0; j < NE; ++j) {
            const uint32_t r = lane + 32u * j;
            if (r < R) {
                const uint32_t l = S.lev[r];
                n_in += l <= T ? 1u : 0u;
                if (l > T) nxt = min(nxt, l);
            }
        }
        n_in = __reduce_add_sync(0xffffffffu, n_in);
        nxt = __reduce_min_sync(0xffffffffu, nxt);
        unsigned long long cnt = left;
        if (nxt != 0xffffffffu && (unsigned long long)n_in * (nxt - T) < left)
            cnt = (unsigned long long)n_in * (nxt - T);
        const unsigned long long full = cnt / n_in;
        const uint32_t part = (uint32_t)(cnt % n_in);
        uint32_t seen = 0;
        for (uint32_t p0 = 0; p0 < R; p0 += 32) {
            const uint32_t p = p0 + lane;
            const uint32_t r = p < R ? S.order[p] : 0u;
            const bool in = p < R && S.lev[r] <= T;
            const uint32_t bal = __ballot_sync(0xffffffffu, in);
            if (in) {
                const uint32_t k = seen + __popc(bal & lt);
                S.cyc[k] = (uint16_t)r;
                S.add[r] += (uint32_t)full + (k < part ? 1u : 0u);
            }
            seen += __popc(bal);
        }
        __syncwarp();
        unsigned long long i = lane, ci = lane % n_in;
        const uint32_t step = 32u % n_in;
        for (; i < cnt; i += 32) {
            members[base + done + i] = S.cyc[ci];
            jobs[base + done + i] = q;
            ci += step;
            if (ci >= n_in) ci -= n_in;
        }
        __syncwarp();
        done += cnt;
        left -= cnt;
        T = nxt;
    }
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        const uint32_t r = lane + 32u * j;
        if (r < R) {
            v[j] += ((unsigned long long)S.add[r] * q) << 16;
            if ((v[j] >> 16) >= kLoadLimit) overflow = true;
        }
    }
    __syncwarp();
    return true;
}

// LPT for R <= 32 uses the sorted-lane kernel (fastest per key) unless the slot
// budget admits this many keys or more: long admission lists reach the long
// runs of equal counts in the tail, which the register kernel places at once.
constexpr uint64_t kLptRunsFrom = 512;

template <int NE>
__global__ void __launch_bounds__(32) k_plan_lpt_reg(const __grid_constant__ lpt_jobs jobs_in, uint32_t *status)
{
    const lpt_job J = jobs_in.j[blockIdx.x];
    const uint32_t lane = cr_lane(), R = J.R;
    unsigned long long v[NE];
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        const uint32_t r = lane + 32u * j;
        v[j] = r < R ? ((J.load[r] << 16) | r) : ~0ull;
    }
    uint32_t taken = 0;
    unsigned long long m = reg_min<NE>(v, 0u);
    const unsigned long long na = J.info->n_adm;
    bool overflow = false;
    unsigned long long st_lam = 0;
    uint32_t st_k = 0, st_off = 0;
    __shared__ lpt_run_smem S;
    unsigned long long stage = 0;  // first key of the 32 staged in st_*
    for (unsigned long long a = 0; a < na; ++a) {
        if (a == 0 || a - stage >= 32) {
            stage = a;
            const unsigned long long ia = a + lane;
            if (ia < na) {
                st_lam = J.adm_cnt[ia];
                st_k = J.adm_k[ia];
                st_off = J.koff[ia];
            }
            // a run of >= 32 keys with k = 1 and equal λ starts here: place it at once
            const uint32_t k0 = __shfl_sync(0xffffffffu, st_k, 0);
            const unsigned long long l0 = __shfl_sync(0xffffffffu, st_lam, 0);
            const unsigned long long l31 = __shfl_sync(0xffffffffu, st_lam, 31);
            if (k0 == 1 && a + 31 < na && l31 == l0) {
                // end of the run: first index after a whose λ differs (λ is non-increasing)
                unsigned long long lo = a + 31, hi = na;  // adm_cnt[lo] == l0; answer in (lo, hi]
                while (hi - lo > 1) {
                    const unsigned long long span = hi - lo;
                    const unsigned long long pr = lo + 1 + (span - 1) * lane / 32;  // 32 probes in (lo, hi)
                    const bool differs = J.adm_cnt[pr] != l0;
                    const uint32_t bl = __ballot_sync(0xffffffffu, differs);
                    if (!bl) {
                        lo = __shfl_sync(0xffffffffu, pr, 31);
                    } else {
                        const uint32_t f = __ffs(bl) - 1;
                        hi = __shfl_sync(0xffffffffu, pr, f);
                        if (f > 0) lo = __shfl_sync(0xffffffffu, pr, f - 1);
                    }
                }
                const unsigned long long runm = hi - a;
                const uint32_t base0 = __shfl_sync(0xffffffffu, st_off, 0);
                if (lpt_equal_run<NE>(v, R, l0, runm, base0, J.members, J.jobs, S, overflow)) {
                    a = hi - 1;      // the loop's ++a moves to the first key after the run
                    stage = a + 1 - 32;  // forces a restage at hi
                    m = reg_min<NE>(v, 0u);
                    continue;
                }
            }
        }
        const uint32_t slot = (uint32_t)(a - stage);
        const uint32_t k = __shfl_sync(0xffffffffu, st_k, slot);
        const uint32_t base = __shfl_sync(0xffffffffu, st_off, slot);
        const unsigned long long lam = __shfl_sync(0xffffffffu, st_lam, slot);
        const unsigned long long q = k == 1 ? lam : lam / k, rem = k == 1 ? 0ull : lam % k;
        for (uint32_t s = 0; s < k; ++s) {
            const unsigned long long best = warp_min_u64(m);
            const uint32_t br = (uint32_t)(best & 0xffffu);
            const unsigned long long job = q + (s < rem ? 1ull : 0ull);
            if (lane == 0) {
                J.members[base + s] = (uint16_t)br;
                J.jobs[base + s] = job;
            }
            if ((br & 31u) == lane) {
                const uint32_t jj = br >> 5;
#pragma unroll
                for (int j = 0; j < NE; ++j)
                    if (j == (int)jj) v[j] += job << 16;
                if (((best >> 16) + job) >= kLoadLimit) overflow = true;
                if (k > 1) taken |= 1u << jj;
                m = reg_min<NE>(v, taken);
            }
        }
        if (k > 1) {  // release this key's destinations for the next key
            taken = 0;
            m = reg_min<NE>(v, 0u);
        }
    }
#pragma unroll
    for (int j = 0; j < NE; ++j) {
        const uint32_t r = lane + 32u * j;
        if (r < R) J.load[r] = v[j] >> 16;
    }
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(status, CR_FLAG_OVERFLOW);
}

// RANDOM placement: T(b) = the first k_b entries of a Fisher-Yates shuffle of
// 0..R-1 (step s swaps position s with s + floor(u R_s / 2^64), R_s = R - s).
// A key with k_b = 1 needs no array: its member is the first draw itself, so
// every lane of a warp places one such key.  Keys with k_b > 1 are shuffled by
// the warp's lane 0 over a shared-memory array that is never reset: an entry
// counts only when its stamp equals the key being placed, otherwise position x
// holds x.  Every key therefore costs O(k_b), not O(R).
constexpr int kRandWarps = 4;

__device__ __forceinline__ void random_body(const cr_plan_info_dev *info,
                                                                 const unsigned long long *__restrict__ adm_cnt,
                                                                 const uint32_t *__restrict__ adm_k,
                                                                 const uint32_t *__restrict__ koff, uint32_t R,
                                                                 unsigned long long seed, unsigned long long epoch,
                                                                 unsigned long long *__restrict__ load_g,
                                                                 uint16_t *__restrict__ members,
                                                                 unsigned long long *__restrict__ jobs,
                                                                 uint32_t *status, uint16_t *perm_all)
{
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5;
    const uint32_t Rp = (R + 1u) & ~1u;                                  // keeps the stamps 4-byte aligned
    uint16_t *val = perm_all + (size_t)warp * Rp * 3;                  // [R] values of touched positions
    uint32_t *stamp = reinterpret_cast<uint32_t *>(val + Rp);           // [R] key (+1) that touched each
    for (uint32_t r = lane; r < R; r += 32) stamp[r] = 0;
    __syncwarp();
    const unsigned long long na = info->n_adm;
    const unsigned long long nw = (unsigned long long)gridDim.x * kRandWarps;
    for (unsigned long long a0 = ((unsigned long long)blockIdx.x * kRandWarps + warp) * 32; a0 < na; a0 += nw * 32) {
        const unsigned long long a = a0 + lane;
        const bool live = a < na;
        const uint32_t k = live ? adm_k[a] : 0u;
        if (live && k == 1) {
            const cr_u64x4 u = cr_philox4x64_10(a, 0ull, 1ull, epoch, seed, (unsigned long long)CR_POLICY_CR_NOLPT);
            const uint32_t m = cr_scale(u.x, (unsigned long long)R);
            const unsigned long long lam = adm_cnt[a];
            members[koff[a]] = (uint16_t)m;
            jobs[koff[a]] = lam;
            const unsigned long long old = atomicAdd(&load_g[m], lam);
            if (old + lam >= kLoadLimit) atomicOr(status, CR_FLAG_OVERFLOW);
        }
        for (unsigned mk = __ballot_sync(0xffffffffu, live && k > 1); mk; mk &= mk - 1) {  // uniform
            const uint32_t src = (uint32_t)__ffs(mk) - 1u;
            const unsigned long long b = a0 + src;
            const uint32_t kb = __shfl_sync(0xffffffffu, k, src), base = koff[b];
            const unsigned long long lam = adm_cnt[b];
            const unsigned long long q = lam / kb, rem = lam % kb;
            const uint32_t tag = (uint32_t)b + 1u;
            if (lane == 0) {
                for (uint32_t s2 = 0; s2 < kb; ++s2) {
                    const cr_u64x4 u = cr_philox4x64_10(b, s2, 1ull, epoch, seed, (unsigned long long)CR_POLICY_CR_NOLPT);
                    const uint32_t t = s2 + cr_scale(u.x, (unsigned long long)(R - s2));
                    const uint32_t vs = stamp[s2] == tag ? val[s2] : s2;
                    const uint32_t vt = stamp[t] == tag ? val[t] : t;
                    val[t] = (uint16_t)vs;
                    stamp[t] = tag;
                    val[s2] = (uint16_t)vt;
                    stamp[s2] = tag;
                    members[base + s2] = (uint16_t)vt;  // later steps only swap positions above s2
                }
            }
            __syncwarp();
            for (uint32_t s2 = lane; s2 < kb; s2 += 32) {
                const unsigned long long job = q + (s2 < rem ? 1ull : 0ull);
                const uint32_t m = val[s2];
                jobs[base + s2] = job;
                const unsigned long long old = atomicAdd(&load_g[m], job);
                if (old + job >= kLoadLimit) atomicOr(status, CR_FLAG_OVERFLOW);
            }
            __syncwarp();
        }
    }
}

__global__ void __launch_bounds__(kRandWarps * 32) k_plan_random(const cr_plan_info_dev *info,
                                                                 const unsigned long long *__restrict__ adm_cnt,
                                                                 const uint32_t *__restrict__ adm_k,
                                                                 const uint32_t *__restrict__ koff, uint32_t R,
                                                                 unsigned long long seed, unsigned long long epoch,
                                                                 unsigned long long *__restrict__ load_g,
                                                                 uint16_t *__restrict__ members,
                                                                 unsigned long long *__restrict__ jobs,
                                                                 uint32_t *status)
{
    extern __shared__ uint16_t perm_all[];
    random_body(info, adm_cnt, adm_k, koff, R, seed, epoch, load_g, members, jobs, status, perm_all);
}

__global__ void __launch_bounds__(kRandWarps * 32) k_plan_random_multi(const __grid_constant__ place_jobs pj,
                                                                       uint32_t *status)
{
    extern __shared__ uint16_t perm_all[];
    const place_job &J = pj.j[blockIdx.y];
    random_body(J.info, J.adm_cnt, J.adm_k, J.koff, J.R, J.seed, J.epoch, J.load, J.members, J.jobs, status,
                perm_all);
}

__device__ __forceinline__ void table_body(const cr_plan_info_dev *info, const unsigned long long *__restrict__ adm_key,
                               const uint32_t *__restrict__ adm_k, const uint32_t *__restrict__ koff,
                               const uint16_t *__restrict__ members, cr_table_slot *__restrict__ table,
                               int bits)
{
    const unsigned long long na = info->n_adm;
    const unsigned long long mask = (1ull << bits) - 1ull;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < na; a += (uint64_t)gridDim.x * blockDim.x) {
        if (adm_k[a] == 0) continue;  // a key placed on no destination has no entry
        const unsigned long long key = adm_key[a];
        unsigned long long s = key >> (64 - bits);
        for (;;) {
            uint32_t prev = atomicCAS(&table[s].koff, kEmpty, koff[a]);
            if (prev == kEmpty) {
                table[s].key = key;
                table[s].k = (uint16_t)adm_k[a];
                table[s].m0 = members[koff[a]];
                break;
            }
            s = (s + 1) & mask;  // the table has at least twice as many slots as keys
        }
    }
}

__global__ void k_table_insert(const cr_plan_info_dev *info, const unsigned long long *__restrict__ adm_key,
                               const uint32_t *__restrict__ adm_k, const uint32_t *__restrict__ koff,
                               const uint16_t *__restrict__ members, cr_table_slot *__restrict__ table,
                               int bits)
{
    table_body(info, adm_key, adm_k, koff, members, table, bits);
}

struct table_job {
    const cr_plan_info_dev *info;
    const unsigned long long *adm_key;
    const uint32_t *adm_k, *koff;
    const uint16_t *members;
    cr_table_slot *table;
    int bits;
};

struct table_jobs {
    table_job j[16];
};

// Tables of several plans in one launch (blockIdx.y picks the plan).
__global__ void k_table_insert_multi(const __grid_constant__ table_jobs tj)
{
    const table_job &J = tj.j[blockIdx.y];
    table_body(J.info, J.adm_key, J.adm_k, J.koff, J.members, J.table, J.bits);
}

template <typename T>
int ensure(cr_ctx *ctx, T **p, uint64_t *cap, uint64_t need)
{
    if (*p && *cap >= need) return CR_OK;
    if (*p) cudaFree(*p);
    *p = nullptr;
    uint64_t c = need < 16 ? 16 : need + need / 4;
    if (cudaMalloc((void **)p, c * sizeof(T)) != cudaSuccess) {
        cudaGetLastError();
        *p = nullptr;
        *cap = 0;
        return cr_fail(ctx, CR_ENOMEM, "plan: cannot allocate %llu elements", (unsigned long long)c);
    }
    *cap = c;
    return CR_OK;
}

int bits_for(uint64_t v)  // smallest b with v < 2^b
{
    int b = 0;
    while (b < 64 && (v >> b) != 0) ++b;
    return b;
}

struct plan_caps {
    uint64_t n, adm, mem, load;
};

int plan_reserve(cr_ctx *ctx, cr_plan *p, uint64_t n, uint32_t R, uint32_t W)
{
    const uint64_t C = (uint64_t)R * W;
    const uint64_t adm = n < C ? n : C;
    uint64_t mem = C;
    if (n * (uint64_t)R < mem) mem = n * (uint64_t)R;
    if (p->cap_n < n + 1 || !p->d_ukey) {
        uint64_t c0 = 0, c1 = 0;
        if (p->d_ukey) cudaFree(p->d_ukey), p->d_ukey = nullptr;
        if (p->d_ucnt) cudaFree(p->d_ucnt), p->d_ucnt = nullptr;
        CR_TRY(ensure(ctx, &p->d_ukey, &c0, n + 1));
        CR_TRY(ensure(ctx, &p->d_ucnt, &c1, n + 1));
        p->cap_n = c0 < c1 ? c0 : c1;
    }
    if (p->cap_adm < adm + 1 || !p->d_adm_key) {
        uint64_t c[4] = {0, 0, 0, 0};
        if (p->d_adm_key) cudaFree(p->d_adm_key), p->d_adm_key = nullptr;
        if (p->d_adm_cnt) cudaFree(p->d_adm_cnt), p->d_adm_cnt = nullptr;
        if (p->d_adm_k) cudaFree(p->d_adm_k), p->d_adm_k = nullptr;
        if (p->d_koff) cudaFree(p->d_koff), p->d_koff = nullptr;
        CR_TRY(ensure(ctx, &p->d_adm_key, &c[0], adm + 1));
        CR_TRY(ensure(ctx, &p->d_adm_cnt, &c[1], adm + 1));
        CR_TRY(ensure(ctx, &p->d_adm_k, &c[2], adm + 1));
        CR_TRY(ensure(ctx, &p->d_koff, &c[3], adm + 1));
        p->cap_adm = c[0];
        for (int i = 1; i < 4; ++i) p->cap_adm = c[i] < p->cap_adm ? c[i] : p->cap_adm;
    }
    if (p->cap_mem < mem + 1 || !p->d_members) {
        uint64_t c0 = 0, c1 = 0;
        if (p->d_members) cudaFree(p->d_members), p->d_members = nullptr;
        if (p->d_jobs) cudaFree(p->d_jobs), p->d_jobs = nullptr;
        CR_TRY(ensure(ctx, &p->d_members, &c0, mem + 1));
        CR_TRY(ensure(ctx, &p->d_jobs, &c1, mem + 1));
        p->cap_mem = c0 < c1 ? c0 : c1;
    }
    if (p->R < R || !p->d_load) {
        uint64_t c = 0;
        if (p->d_load) cudaFree(p->d_load), p->d_load = nullptr;
        CR_TRY(ensure(ctx, &p->d_load, &c, (uint64_t)R));
    }
    uint64_t slots = 16;
    while (slots < 2 * (adm + 1)) slots <<= 1;
    if (p->table_slots < slots || !p->d_table) {
        if (p->d_table) cudaFree(p->d_table), p->d_table = nullptr;
        uint64_t c = 0;
        CR_TRY(ensure(ctx, &p->d_table, &c, slots));
        p->table_slots = slots;
    } else {
        slots = p->table_slots;
    }
    if (!p->d_info) {
        uint64_t c = 0;
        CR_TRY(ensure(ctx, &p->d_info, &c, 1));
    }
    p->R = R;
    p->W = W;
    return CR_OK;
}

}  // namespace

extern "C" int cr_plan_create(cr_ctx *ctx, cr_plan **out)
{
    if (!ctx || !out) return CR_EINVAL;
    cr_plan *p = (cr_plan *)calloc(1, sizeof(cr_plan));
    if (!p) return cr_fail(ctx, CR_ENOMEM, "cr_plan_create: host allocation failed");
    *out = p;
    return CR_OK;
}

extern "C" int cr_plan_destroy(cr_ctx *ctx, cr_plan *p)
{
    if (!p) return CR_OK;
    if (ctx) cudaStreamSynchronize(ctx->stream);
    void *bufs[] = {p->d_ukey, p->d_ucnt, p->d_adm_key, p->d_adm_cnt, p->d_adm_k, p->d_koff,
                    p->d_members, p->d_jobs, p->d_load, p->d_table, p->d_info};
    for (void *b : bufs)
        if (b) cudaFree(b);
    free(p);
    return CR_OK;
}

static int check_params(cr_ctx *ctx, const cr_plan_params *pp)
{
    if (pp->R == 0 || pp->R > CR_MAX_R) return cr_fail(ctx, CR_EINVAL, "plan: R=%u outside 1..%u", pp->R, CR_MAX_R);
    if (pp->W == 0) return cr_fail(ctx, CR_EINVAL, "plan: W must be >= 1");
    if ((uint64_t)pp->R * pp->W >= 0xffffffffull) return cr_fail(ctx, CR_EINVAL, "plan: C = R*W must be < 2^32-1");
    if (pp->qcap_num == 0 || pp->qcap_den == 0 || pp->qcap_den >= (1ull << 32))
        return cr_fail(ctx, CR_EINVAL, "plan: q_cap needs num >= 1 and 1 <= den < 2^32");
    if (pp->variant > CR_VARIANT_SLOTCAP || pp->reserved != 0)
        return cr_fail(ctx, CR_EINVAL, "plan: bad variant %u or reserved field", pp->variant);
    return CR_OK;
}

static int build_plans(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
                       uint32_t n_plans, cr_plan *const *plans);

extern "C" int cr_build_plans(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
                              uint32_t n_plans, cr_plan *const *plans)
{
    if (!ctx) return CR_EINVAL;
    cr_nvtx_range nv("cr_build_plans");
    const int pi = cr_prof_begin(ctx, ctx->stream, CR_PROF_PLAN);
    const int st = build_plans(ctx, d_key, n, params, n_plans, plans);
    cr_prof_end(ctx, ctx->stream, pi);
    return st;
}

static int build_plans(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
                       uint32_t n_plans, cr_plan *const *plans)
{
    if (!ctx) return CR_EINVAL;
    if (!params || !plans || n_plans == 0) return cr_fail(ctx, CR_EINVAL, "cr_build_plans: no plans");
    if (n >= (1ull << 32) - 1) return cr_fail(ctx, CR_EINVAL, "cr_build_plans: n >= 2^32-1");
    if (n > 0 && !d_key) return cr_fail(ctx, CR_EINVAL, "cr_build_plans: d_key is NULL");
    for (uint32_t j = 0; j < n_plans; ++j) {
        if (!plans[j]) return cr_fail(ctx, CR_EINVAL, "cr_build_plans: plan %u is NULL", j);
        for (uint32_t i = 0; i < j; ++i)
            if (plans[i] == plans[j]) return cr_fail(ctx, CR_EINVAL, "cr_build_plans: plan %u repeated", j);
        CR_TRY(check_params(ctx, &params[j]));
    }
    for (uint32_t j = 0; j < n_plans; ++j) {
        CR_TRY(plan_reserve(ctx, plans[j], n, params[j].R, params[j].W));
        plans[j]->n = n;
        plans[j]->qnum = params[j].qcap_num;
        plans[j]->qden = params[j].qcap_den;
        plans[j]->variant = params[j].variant;
        plans[j]->built = 1;
        if (j == 0 || n == 0 || n > kPlanSortOneCta)  // small intervals: the admission CTA writes every field
            CR_LAUNCH(ctx, k_plan_reset, 1, 1, 0, plans[j]->d_info, (unsigned long long)n);
    }
    cr_plan *p0 = plans[0];
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    const unsigned int grid_n = cr_blocks(n, 256, gcap);

    // ---- shared histogram and admission order ------------------------------
    const uint32_t *order = nullptr;
    if (n > 0) {
        uint64_t slots = 1024;
        while (slots < 2 * n) slots <<= 1;
        const int tbits = bits_for(slots - 1);
        void *ptk, *ptc, *pk0, *pk1, *pv0, *pv1, *po;
        CR_TRY(cr_scratch(ctx, SCR_PLAN_A, slots * sizeof(unsigned long long), &ptk));
        CR_TRY(cr_scratch(ctx, SCR_PLAN_B, slots * sizeof(uint32_t) + 16, &ptc));
        CR_TRY(cr_scratch(ctx, SCR_SORT_K0, n * sizeof(unsigned long long), &pk0));
        CR_TRY(cr_scratch(ctx, SCR_SORT_K1, n * sizeof(unsigned long long), &pk1));
        CR_TRY(cr_scratch(ctx, SCR_SORT_V0, n * sizeof(uint32_t), &pv0));
        CR_TRY(cr_scratch(ctx, SCR_SORT_V1, n * sizeof(uint32_t), &pv1));
        CR_TRY(cr_scratch(ctx, SCR_PLAN_C, (2 * n + 1) * sizeof(uint32_t), &po));
        unsigned long long *tkey = (unsigned long long *)ptk;
        uint32_t *tcnt = (uint32_t *)ptc;
        CR_CUDA(ctx, cudaMemsetAsync(tkey, 0xff, slots * sizeof(unsigned long long), ctx->stream));
        CR_CUDA(ctx, cudaMemsetAsync(tcnt, 0, slots * sizeof(uint32_t), ctx->stream));
        CR_LAUNCH(ctx, k_hist_insert, grid_n, 256, 0, (const unsigned long long *)d_key, n, tkey, tcnt, tbits,
                  p0->d_info);
        CR_LAUNCH(ctx, k_hist_compact, cr_blocks(slots, 256, gcap), 256, 0, (const unsigned long long *)tkey,
                  (const uint32_t *)tcnt, slots, (unsigned long long *)pk0, (uint32_t *)pv0, p0->d_info);
        // the (n - count) keys and the order ping-pong through the now idle table memory
        uint32_t *s32A = (uint32_t *)ptk, *s32B = s32A + n, *o32B = (uint32_t *)ptc;
        uint32_t *ord = (uint32_t *)po;
        if (n <= kPlanSortOneCta) {
            // admission candidates only: the largest slot budget of the build bounds how far it reaches
            unsigned long long cmax = 0;
            for (uint32_t j = 0; j < n_plans; ++j) {
                const unsigned long long c = (unsigned long long)params[j].R * params[j].W;
                cmax = c > cmax ? c : cmax;
            }
            CR_LAUNCH(ctx, k_plan_topk, 1, kSmallBlock, 0, p0->d_info, (unsigned long long)n, bits_for(n), cmax,
                      (unsigned long long *)pk0, (uint32_t *)pv0, (unsigned long long *)pk1, (uint32_t *)pv1,
                      p0->d_ukey, p0->d_ucnt, s32A, s32B, ord + n, o32B, ord);
        } else {
            // the same two sorts in device-wide passes, the key count read on the device
            const unsigned long long *dU = &p0->d_info->U;
            int in1 = 0;
            CR_TRY(cr_radix_pairs_u64_dev(ctx, (unsigned long long *)pk0, (uint32_t *)pv0, (unsigned long long *)pk1,
                                          (uint32_t *)pv1, n, dU, 0ull, 64, 0, &in1));
            CR_LAUNCH(ctx, k_plan_sorted_keys, grid_n, 256, 0, (const cr_plan_info_dev *)p0->d_info,
                      (unsigned long long)n, (const unsigned long long *)(in1 ? pk1 : pk0),
                      (const uint32_t *)(in1 ? pv1 : pv0), p0->d_ukey, p0->d_ucnt, s32A);
            uint32_t *o32A = (uint32_t *)pv0;  // free again after the key sort's results were copied out
            CR_TRY(cr_radix_pairs_u32_dev(ctx, s32A, o32A, s32B, o32B, n, dU, 0ull, bits_for(n), 1, &in1));
            CR_LAUNCH(ctx, k_plan_copy_order, grid_n, 256, 0, p0->d_info,
                      (const uint32_t *)(in1 ? o32B : o32A), ord);
        }
        order = ord;
    }

    // ---- per plan -------------------------------------------------------------
    // LPT placements with 32 < R <= 1024 are collected and run together, one
    // warp per plan, followed by their tables.
    lpt_jobs lj;
    uint32_t n_lj = 0, lj_maxR = 0, deferred[16];
    const bool fused = n > 0 && n <= kPlanSortOneCta;  // small intervals: batched launches throughout
    const bool tables_later = fused;
    auto table_insert = [&](uint32_t j) -> int {
        cr_plan *p = plans[j];
        const uint64_t C = (uint64_t)params[j].R * params[j].W;
        const int bits = bits_for(p->table_slots - 1);
        const uint64_t adm = n < C ? n : C;
        CR_LAUNCH(ctx, k_table_insert, cr_blocks(adm, 256, gcap), 256, 0, (const cr_plan_info_dev *)p->d_info,
                  (const unsigned long long *)p->d_adm_key, (const uint32_t *)p->d_adm_k,
                  (const uint32_t *)p->d_koff, (const uint16_t *)p->d_members, p->d_table, bits);
        return CR_OK;
    };
    auto flush_lpt = [&]() -> int {
        if (!n_lj) return CR_OK;
        const uint32_t ne = (lj_maxR + 31) / 32;
        if (ne <= 1)
            CR_LAUNCH(ctx, k_plan_lpt_reg<1>, n_lj, 32, 0, lj, ctx->d_status);
        else if (ne <= 2)
            CR_LAUNCH(ctx, k_plan_lpt_reg<2>, n_lj, 32, 0, lj, ctx->d_status);
        else if (ne <= 4)
            CR_LAUNCH(ctx, k_plan_lpt_reg<4>, n_lj, 32, 0, lj, ctx->d_status);
        else if (ne <= 8)
            CR_LAUNCH(ctx, k_plan_lpt_reg<8>, n_lj, 32, 0, lj, ctx->d_status);
        else if (ne <= 16)
            CR_LAUNCH(ctx, k_plan_lpt_reg<16>, n_lj, 32, 0, lj, ctx->d_status);
        else
            CR_LAUNCH(ctx, k_plan_lpt_reg<32>, n_lj, 32, 0, lj, ctx->d_status);
        if (!tables_later)
            for (uint32_t x = 0; x < n_lj; ++x) CR_TRY(table_insert(deferred[x]));
        n_lj = 0;
        lj_maxR = 0;
        return CR_OK;
    };
    // small intervals: admission of every plan in one launch, one CTA per plan
    if (fused) {
        for (uint32_t j0 = 0; j0 < n_plans; j0 += 16) {
            admit_jobs aj;
            const uint32_t nj = n_plans - j0 < 16 ? n_plans - j0 : 16;
            for (uint32_t x = 0; x < nj; ++x) {
                cr_plan *p = plans[j0 + x];
                const cr_plan_params &pp = params[j0 + x];
                admit_job &J = aj.j[x];
                J.info = p->d_info;
                J.init_load = (const unsigned long long *)pp.d_init_load;
                J.load = p->d_load;
                J.adm_key = p->d_adm_key;
                J.adm_cnt = p->d_adm_cnt;
                J.adm_k = p->d_adm_k;
                J.koff = p->d_koff;
                J.table = reinterpret_cast<uint4 *>(p->d_table);
                J.table_slots = p->table_slots;
                J.C = (unsigned long long)pp.R * pp.W;
                J.num = pp.qcap_num;
                J.den = pp.qcap_den;
                J.R = pp.R;
                J.norepl = pp.variant == CR_VARIANT_NOREPL ? 1 : 0;
                J.ukey_out = j0 + x > 0 ? p->d_ukey : nullptr;  // every plan keeps the histogram
                J.ucnt_out = j0 + x > 0 ? p->d_ucnt : nullptr;
            }
            CR_LAUNCH(ctx, k_plan_admit_cta, nj, kSmallBlock, 0, aj, (const cr_plan_info_dev *)p0->d_info, order,
                      (const unsigned long long *)p0->d_ukey, (const unsigned long long *)p0->d_ucnt,
                      (unsigned long long)n, ctx->d_status);
        }
        // placements: random and single-warp LPT plans batched per launch
        place_jobs rj, l32;
        uint32_t nr = 0, n32 = 0, rmaxR = 0;
        uint64_t radm = 0;
        auto flush_random = [&]() -> int {
            if (!nr) return CR_OK;
            const size_t smem = (size_t)kRandWarps * (rmaxR + 1) * 3 * sizeof(uint16_t);
            if (smem > 48 * 1024)
                CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_random_multi, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  (int)smem));
            CR_LAUNCH(ctx, k_plan_random_multi, dim3(cr_blocks(radm, kRandWarps * 32, gcap), nr), kRandWarps * 32, smem,
                      rj, ctx->d_status);
            nr = 0;
            rmaxR = 0;
            radm = 0;
            return CR_OK;
        };
        auto flush_l32 = [&]() -> int {
            if (!n32) return CR_OK;
            CR_LAUNCH(ctx, k_plan_lpt32_multi, n32, 32, 0, l32, ctx->d_status);
            n32 = 0;
            return CR_OK;
        };
        for (uint32_t j = 0; j < n_plans; ++j) {
            cr_plan *p = plans[j];
            const cr_plan_params &pp = params[j];
            const uint64_t C = (uint64_t)pp.R * pp.W;
            place_job J;
            J.info = p->d_info;
            J.adm_cnt = p->d_adm_cnt;
            J.adm_k = p->d_adm_k;
            J.koff = p->d_koff;
            J.load = p->d_load;
            J.jobs = p->d_jobs;
            J.members = p->d_members;
            J.seed = pp.seed;
            J.epoch = pp.epoch;
            J.R = pp.R;
            if (pp.variant == CR_VARIANT_SLOTCAP) {
                const size_t smem = (size_t)pp.R * (sizeof(unsigned long long) + sizeof(uint32_t) + 1) + 16;
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_lpt_capped, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                CR_LAUNCH(ctx, k_plan_lpt_capped, 1, 32, smem, p->d_info, (const unsigned long long *)p->d_adm_cnt,
                          p->d_adm_k, p->d_koff, pp.R, pp.W, p->d_load, p->d_members, p->d_jobs, ctx->d_status);
            } else if (pp.variant == CR_VARIANT_RANDOM) {
                rj.j[nr++] = J;
                rmaxR = pp.R > rmaxR ? pp.R : rmaxR;
                radm = (n < C ? n : C) > radm ? (n < C ? n : C) : radm;
                if (nr == 16) CR_TRY(flush_random());
            } else if (pp.R <= 32 && C < kLptRunsFrom) {
                l32.j[n32++] = J;
                if (n32 == 16) CR_TRY(flush_l32());
            } else if (pp.R <= 1024) {
                lpt_job &jb = lj.j[n_lj++];
                jb.info = p->d_info;
                jb.adm_cnt = p->d_adm_cnt;
                jb.adm_k = p->d_adm_k;
                jb.koff = p->d_koff;
                jb.load = p->d_load;
                jb.members = p->d_members;
                jb.jobs = p->d_jobs;
                jb.R = pp.R;
                lj_maxR = pp.R > lj_maxR ? pp.R : lj_maxR;
                deferred[n_lj - 1] = j;
                if (n_lj == 16) CR_TRY(flush_lpt());
            } else {
                const size_t smem = (size_t)pp.R * (sizeof(unsigned long long) + 1) + 16;
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_lpt, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                CR_LAUNCH(ctx, k_plan_lpt, 1, 32, smem, (const cr_plan_info_dev *)p->d_info,
                          (const unsigned long long *)p->d_adm_cnt, (const uint32_t *)p->d_adm_k,
                          (const uint32_t *)p->d_koff, pp.R, p->d_load, p->d_members, p->d_jobs, ctx->d_status);
            }
        }
        CR_TRY(flush_random());
        CR_TRY(flush_l32());
        CR_TRY(flush_lpt());
        // tables of every plan, batched per launch
        for (uint32_t j0 = 0; j0 < n_plans; j0 += 16) {
            table_jobs tj;
            const uint32_t nj = n_plans - j0 < 16 ? n_plans - j0 : 16;
            uint64_t adm = 0;
            for (uint32_t x = 0; x < nj; ++x) {
                cr_plan *p = plans[j0 + x];
                const uint64_t C = (uint64_t)params[j0 + x].R * params[j0 + x].W;
                adm = (n < C ? n : C) > adm ? (n < C ? n : C) : adm;
                table_job &T = tj.j[x];
                T.info = p->d_info;
                T.adm_key = p->d_adm_key;
                T.adm_k = p->d_adm_k;
                T.koff = p->d_koff;
                T.members = p->d_members;
                T.table = p->d_table;
                T.bits = bits_for(p->table_slots - 1);
            }
            CR_LAUNCH(ctx, k_table_insert_multi, dim3(cr_blocks(adm, 256, gcap), nj), 256, 0, tj);
        }
        return CR_OK;
    }
    // large intervals (and empty ones): plan by plan.  Eq. 1 and the admission depend only
    // on (R, W, q_cap, single copy or not): a plan equal in those to an earlier one of the
    // build (the random placements of several seeds, say) copies its admitted arrays and
    // counters instead of recomputing them.
    auto same_admission = [&](uint32_t a, uint32_t b) {
        const cr_plan_params &x = params[a], &y = params[b];
        return x.R == y.R && x.W == y.W && x.qcap_num == y.qcap_num && x.qcap_den == y.qcap_den &&
               (x.variant == CR_VARIANT_NOREPL) == (y.variant == CR_VARIANT_NOREPL);
    };
    for (uint32_t j = 0; j < n_plans; ++j) {
        cr_plan *p = plans[j];
        const cr_plan_params &pp = params[j];
        const uint64_t C = (uint64_t)pp.R * pp.W;
        uint32_t src = j;
        for (uint32_t i = 0; i < j && src == j; ++i)
            if (same_admission(i, j)) src = i;
        if (j > 0 && n > 0) {
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_ukey, p0->d_ukey, n * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_ucnt, p0->d_ucnt, n * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(&p->d_info->U, &p0->d_info->U, 2 * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));  // U and S
        }
        CR_CUDA(ctx, cudaMemsetAsync(p->d_table, 0xff, p->table_slots * sizeof(cr_table_slot), ctx->stream));
        if (n > 0 && src != j) {
            const cr_plan *q = plans[src];
            const uint64_t na = n < C ? n : C;  // a bound on the admitted keys
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_info, q->d_info, sizeof(cr_plan_info_dev), cudaMemcpyDeviceToDevice,
                                         ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_adm_key, q->d_adm_key, na * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_adm_cnt, q->d_adm_cnt, na * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_adm_k, q->d_adm_k, na * sizeof(uint32_t), cudaMemcpyDeviceToDevice,
                                         ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_koff, q->d_koff, (na + 1) * sizeof(uint32_t), cudaMemcpyDeviceToDevice,
                                         ctx->stream));
        } else if (n > 0) {
            void *pk;
            CR_TRY(cr_scratch(ctx, SCR_PLAN_B, (n + 2) * sizeof(unsigned long long), &pk));
            unsigned long long *kk = (unsigned long long *)pk;
            CR_LAUNCH(ctx, k_plan_kb, grid_n, 256, 0, order, (const unsigned long long *)p->d_ucnt, n,
                      (const cr_plan_info_dev *)p->d_info, (unsigned long long)pp.qcap_num,
                      (unsigned long long)pp.qcap_den, pp.R, pp.variant == CR_VARIANT_NOREPL ? 1 : 0, kk);
            CR_TRY(cr_scan_u64_inclusive(ctx, kk, kk, n));
            CR_LAUNCH(ctx, k_plan_admit, grid_n, 256, 0, (const unsigned long long *)kk, p->d_info,
                      (unsigned long long)C);
            CR_LAUNCH(ctx, k_plan_fill, grid_n, 256, 0, order, (const unsigned long long *)p->d_ukey,
                      (const unsigned long long *)p->d_ucnt, (const unsigned long long *)kk, p->d_info,
                      p->d_adm_key, p->d_adm_cnt, p->d_adm_k, p->d_koff);
        }
        CR_LAUNCH(ctx, k_plan_init_load, cr_blocks(pp.R, 256, gcap), 256, 0, p->d_info,
                  (const unsigned long long *)pp.d_init_load, pp.R, p->d_load, ctx->d_status);
        if (n > 0) {
            if (pp.variant == CR_VARIANT_SLOTCAP) {
                const size_t smem = (size_t)pp.R * (sizeof(unsigned long long) + sizeof(uint32_t) + 1) + 16;
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_lpt_capped, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                CR_LAUNCH(ctx, k_plan_lpt_capped, 1, 32, smem, p->d_info, (const unsigned long long *)p->d_adm_cnt,
                          p->d_adm_k, p->d_koff, pp.R, pp.W, p->d_load, p->d_members, p->d_jobs, ctx->d_status);
            } else if (pp.variant == CR_VARIANT_RANDOM) {
                size_t smem = (size_t)kRandWarps * (pp.R + 1) * 3 * sizeof(uint16_t);
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_random, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                uint64_t adm = n < C ? n : C;
                CR_LAUNCH(ctx, k_plan_random, cr_blocks(adm, kRandWarps * 32, gcap), kRandWarps * 32, smem,
                          (const cr_plan_info_dev *)p->d_info, (const unsigned long long *)p->d_adm_cnt,
                          (const uint32_t *)p->d_adm_k, (const uint32_t *)p->d_koff, pp.R,
                          (unsigned long long)pp.seed, (unsigned long long)pp.epoch, p->d_load, p->d_members,
                          p->d_jobs, ctx->d_status);
            } else {
                size_t smem = (size_t)pp.R * (sizeof(unsigned long long) + 1) + 16;
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_lpt, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                if (pp.R <= 32 && C < kLptRunsFrom)
                    CR_LAUNCH(ctx, k_plan_lpt32, 1, 32, 0, (const cr_plan_info_dev *)p->d_info,
                              (const unsigned long long *)p->d_adm_cnt, (const uint32_t *)p->d_adm_k,
                              (const uint32_t *)p->d_koff, pp.R, p->d_load, p->d_members, p->d_jobs,
                              ctx->d_status);
                else if (pp.R <= 1024) {
                    lpt_job &jb = lj.j[n_lj++];
                    jb.info = p->d_info;
                    jb.adm_cnt = p->d_adm_cnt;
                    jb.adm_k = p->d_adm_k;
                    jb.koff = p->d_koff;
                    jb.load = p->d_load;
                    jb.members = p->d_members;
                    jb.jobs = p->d_jobs;
                    jb.R = pp.R;
                    lj_maxR = pp.R > lj_maxR ? pp.R : lj_maxR;
                    deferred[n_lj - 1] = j;
                    if (n_lj == 16) CR_TRY(flush_lpt());
                    continue;
                } else
                CR_LAUNCH(ctx, k_plan_lpt, 1, 32, smem, (const cr_plan_info_dev *)p->d_info,
                          (const unsigned long long *)p->d_adm_cnt, (const uint32_t *)p->d_adm_k,
                          (const uint32_t *)p->d_koff, pp.R, p->d_load, p->d_members, p->d_jobs, ctx->d_status);
            }
            CR_TRY(table_insert(j));
        }
    }
    return flush_lpt();
}

extern "C" int cr_build_plan(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
                             cr_plan *plan)
{
    return cr_build_plans(ctx, d_key, n, params, 1, &plan);
}

extern "C" int cr_plan_get_info(cr_ctx *ctx, const cr_plan *p, cr_plan_info *out)
{
    if (!ctx || !p || !out) return CR_EINVAL;
    if (!p->built) return cr_fail(ctx, CR_EINVAL, "plan was never built");
    cr_plan_info_dev d;
    CR_CUDA(ctx, cudaMemcpyAsync(&d, p->d_info, sizeof(d), cudaMemcpyDeviceToHost, ctx->stream));
    CR_TRY(cr_sync(ctx));
    out->n = d.n;
    out->U = d.U;
    out->n_adm = d.n_adm;
    out->sum_k = d.sum_k;
    out->cold = d.cold;
    out->max_k = d.max_k;
    out->R = p->R;
    out->W = p->W;
    return CR_OK;
}

__global__ void k_gather_u64(const unsigned long long *__restrict__ src, const uint32_t *__restrict__ idx,
                             unsigned long long n, unsigned long long *__restrict__ out)
{
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x)
        out[i] = src[idx[i]];
}

extern "C" int cr_plan_export(cr_ctx *ctx, const cr_plan *p, uint64_t *ukey, uint64_t *ucnt, uint64_t *adm_key,
                              uint64_t *adm_cnt, uint32_t *adm_k, uint32_t *koff, uint16_t *members,
                              uint64_t *jobs, uint64_t *load)
{
    cr_plan_info info;
    CR_TRY(cr_plan_get_info(ctx, p, &info));
    cudaStream_t s = ctx->stream;
    cr_plan_info_dev d;
    CR_CUDA(ctx, cudaMemcpyAsync(&d, p->d_info, sizeof(d), cudaMemcpyDeviceToHost, s));
    CR_TRY(cr_sync(ctx));
    const unsigned long long *sk = (const unsigned long long *)p->d_ukey, *sc = (const unsigned long long *)p->d_ucnt;
    if ((ukey || ucnt) && d.U && d.S < d.U) {
        // only the admission candidates are in key order: sort the whole histogram by key
        const unsigned long long *ks;
        const uint32_t *pos;
        CR_TRY(cr_radix_sort_u64(ctx, (const unsigned long long *)p->d_ukey, nullptr, d.U, 64, &ks, &pos));
        void *pc;
        CR_TRY(cr_scratch(ctx, SCR_PLAN_A, d.U * sizeof(unsigned long long), &pc));
        CR_LAUNCH(ctx, k_gather_u64, cr_blocks(d.U, 256, (unsigned int)ctx->num_sms * 8u), 256, 0,
                  (const unsigned long long *)p->d_ucnt, pos, (unsigned long long)d.U, (unsigned long long *)pc);
        sk = ks;
        sc = (const unsigned long long *)pc;
    }
    if (ukey && info.U) CR_CUDA(ctx, cudaMemcpyAsync(ukey, sk, info.U * 8, cudaMemcpyDeviceToHost, s));
    if (ucnt && info.U) CR_CUDA(ctx, cudaMemcpyAsync(ucnt, sc, info.U * 8, cudaMemcpyDeviceToHost, s));
    if (adm_key && info.n_adm)
        CR_CUDA(ctx, cudaMemcpyAsync(adm_key, p->d_adm_key, info.n_adm * 8, cudaMemcpyDeviceToHost, s));
    if (adm_cnt && info.n_adm)
        CR_CUDA(ctx, cudaMemcpyAsync(adm_cnt, p->d_adm_cnt, info.n_adm * 8, cudaMemcpyDeviceToHost, s));
    if (adm_k && info.n_adm)
        CR_CUDA(ctx, cudaMemcpyAsync(adm_k, p->d_adm_k, info.n_adm * 4, cudaMemcpyDeviceToHost, s));
    if (koff) {
        if (info.n_adm)
            CR_CUDA(ctx, cudaMemcpyAsync(koff, p->d_koff, (info.n_adm + 1) * 4, cudaMemcpyDeviceToHost, s));
        else
            koff[0] = 0;
    }
    if (members && info.sum_k)
        CR_CUDA(ctx, cudaMemcpyAsync(members, p->d_members, info.sum_k * 2, cudaMemcpyDeviceToHost, s));
    if (jobs && info.sum_k)
        CR_CUDA(ctx, cudaMemcpyAsync(jobs, p->d_jobs, info.sum_k * 8, cudaMemcpyDeviceToHost, s));
    if (load) CR_CUDA(ctx, cudaMemcpyAsync(load, p->d_load, (uint64_t)info.R * 8, cudaMemcpyDeviceToHost, s));
    return cr_sync(ctx);
}

// ---- allocation-free key histogram (cr_key_histogram_noalloc) ---------------
// Some callers cannot allocate device memory when they call in: a process whose
// device memory is owned and handed out by another runtime's pool, or a
// latency-critical path where a cudaMalloc (which may synchronise the device)
// is not acceptable.  For them the histogram of the plan builder runs with its
// scratch in this file-scope array, sized for at most CR_NOALLOC_MAX_KEYS keys.
// Every GPU that loads the library holds the array until the process exits.
// Layout: table keys | table counts | sort keys (2 buffers) | sort values
// (2 buffers) | order (2 buffers) | info.
namespace {
constexpr uint64_t kNaSlots = 2ull * CR_NOALLOC_MAX_KEYS;  // power of two, >= 2n
constexpr uint64_t kNaN = CR_NOALLOC_MAX_KEYS;
constexpr size_t kNaOffTcnt = kNaSlots * 8;
constexpr size_t kNaOffKA = kNaOffTcnt + kNaSlots * 4;
constexpr size_t kNaOffKB = kNaOffKA + kNaN * 8;
constexpr size_t kNaOffVA = kNaOffKB + kNaN * 8;
constexpr size_t kNaOffVB = kNaOffVA + kNaN * 4;
constexpr size_t kNaOffOrd = kNaOffVB + kNaN * 4;
constexpr size_t kNaOffInfo = kNaOffOrd + (2 * kNaN + 64) * 4;
constexpr size_t kNaBytes = kNaOffInfo + 256;
}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNaBytes];

namespace {
constexpr int kNaMaxDevices = 64;
void *g_noalloc_ptr[kNaMaxDevices];  // device address of g_noalloc_scratch, per device

__global__ void k_copy_u(const cr_plan_info_dev *info, unsigned long long *out) { *out = info->U; }
}  // namespace

extern "C" int cr_key_histogram_noalloc(const uint64_t *d_key, uint64_t n, uint64_t *d_ukey, uint64_t *d_ucnt,
                                        uint64_t *d_U, void *cuda_stream)
{
    if (n > CR_NOALLOC_MAX_KEYS)
        return cr_fail(NULL, CR_EINVAL, "cr_key_histogram_noalloc: n=%llu exceeds CR_NOALLOC_MAX_KEYS=%d",
                       (unsigned long long)n, CR_NOALLOC_MAX_KEYS);
    if (!d_U || (n > 0 && (!d_key || !d_ukey || !d_ucnt)))
        return cr_fail(NULL, CR_EINVAL, "cr_key_histogram_noalloc: NULL pointer");
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNaMaxDevices) {
        cudaGetLastError();
        return cr_fail(NULL, CR_ECUDA, "cr_key_histogram_noalloc: no usable current device");
    }
    if (!g_noalloc_ptr[dev]) {
        // once per device, with that device current: the array's device address
        void *p = NULL;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) {
            cudaGetLastError();
            return cr_fail(NULL, CR_ECUDA, "cr_key_histogram_noalloc: cudaGetSymbolAddress: %s",
                           cudaGetErrorString(e));
        }
        g_noalloc_ptr[dev] = p;
    }
    cudaStream_t s = (cudaStream_t)cuda_stream;
    unsigned char *base = (unsigned char *)g_noalloc_ptr[dev];
    cr_plan_info_dev *info = (cr_plan_info_dev *)(base + kNaOffInfo);
    k_plan_reset<<<1, 1, 0, s>>>(info, (unsigned long long)n);
    if (n > 0) {
        uint64_t slots = 1024;
        while (slots < 2 * n) slots <<= 1;
        int tbits = 0;
        while ((1ull << tbits) < slots) ++tbits;
        unsigned long long *tkey = (unsigned long long *)base;
        uint32_t *tcnt = (uint32_t *)(base + kNaOffTcnt);
        unsigned long long *kA = (unsigned long long *)(base + kNaOffKA), *kB = (unsigned long long *)(base + kNaOffKB);
        uint32_t *vA = (uint32_t *)(base + kNaOffVA), *vB = (uint32_t *)(base + kNaOffVB);
        uint32_t *ord = (uint32_t *)(base + kNaOffOrd);
        int nsm = 1;
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
        const unsigned int grid = cr_blocks(n, 256, (unsigned int)nsm * 8u);
        if (cudaMemsetAsync(tkey, 0xff, slots * sizeof(unsigned long long), s) != cudaSuccess ||
            cudaMemsetAsync(tcnt, 0, slots * sizeof(uint32_t), s) != cudaSuccess) {
            cudaGetLastError();
            return cr_fail(NULL, CR_ECUDA, "cr_key_histogram_noalloc: clearing the table failed");
        }
        k_hist_insert<<<grid, 256, 0, s>>>((const unsigned long long *)d_key, n, tkey, tcnt, tbits, info);
        k_hist_compact<<<cr_blocks(slots, 256, (unsigned int)nsm * 8u), 256, 0, s>>>(tkey, tcnt, slots, kA, vA, info);
        uint32_t *s32A = (uint32_t *)tkey, *s32B = s32A + n;
        k_plan_sort<<<1, kSmallBlock, 0, s>>>(info, (unsigned long long)n, bits_for(n), kA, vA, kB, vB,
                                              (unsigned long long *)d_ukey, (unsigned long long *)d_ucnt, s32A,
                                              s32B, ord + n, tcnt, ord);
    }
    k_copy_u<<<1, 1, 0, s>>>(info, (unsigned long long *)d_U);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return cr_fail(NULL, CR_ECUDA, "cr_key_histogram_noalloc: launch failed: %s", cudaGetErrorString(e));
    return CR_OK;
}

// ---- plan import (a table computed elsewhere, e.g. exported earlier) --------
namespace {
struct imp_ent {
    unsigned long long key, cnt;
};
int cmp_imp(const void *a, const void *b)
{
    const unsigned long long x = ((const imp_ent *)a)->key, y = ((const imp_ent *)b)->key;
    return x < y ? -1 : (x > y ? 1 : 0);
}
}  // namespace

extern "C" int cr_plan_import(cr_ctx *ctx, cr_plan *p, uint32_t R, uint32_t W, uint64_t n_adm, const uint64_t *adm_key,
                              const uint64_t *adm_cnt, const uint32_t *adm_k, const uint16_t *members,
                              const uint64_t *jobs, const uint64_t *load)
{
    if (!ctx || !p) return CR_EINVAL;
    cr_nvtx_range nv("cr_plan_import");
    if (R == 0 || R > CR_MAX_R || W == 0) return cr_fail(ctx, CR_EINVAL, "cr_plan_import: R=%u W=%u", R, W);
    const uint64_t C = (uint64_t)R * W;
    if (n_adm > C) return cr_fail(ctx, CR_EINVAL, "cr_plan_import: %llu keys exceed C = R*W", (unsigned long long)n_adm);
    if (n_adm && (!adm_key || !adm_cnt || !adm_k || !members))
        return cr_fail(ctx, CR_EINVAL, "cr_plan_import: NULL array");
    // host checks: every k in 1..R, sum of k <= C, members < R and distinct per key, keys distinct
    uint64_t sum_k = 0, max_k = 0, adm_lam = 0;
    for (uint64_t a = 0; a < n_adm; ++a) {
        if (adm_k[a] == 0 || adm_k[a] > R)
            return cr_fail(ctx, CR_EINVAL, "cr_plan_import: key %llu has k=%u", (unsigned long long)a, adm_k[a]);
        sum_k += adm_k[a];
        max_k = adm_k[a] > max_k ? adm_k[a] : max_k;
        adm_lam += adm_cnt[a];
    }
    if (sum_k > C) return cr_fail(ctx, CR_EINVAL, "cr_plan_import: sum of k exceeds C = R*W");
    uint32_t *koff = (uint32_t *)malloc((n_adm + 1) * sizeof(uint32_t));
    imp_ent *srt = (imp_ent *)malloc((n_adm + 1) * sizeof(imp_ent));
    uint8_t *seen = (uint8_t *)calloc(R, 1);
    int bad = !koff || !srt || !seen;
    if (!bad) {
        koff[0] = 0;
        for (uint64_t a = 0; a < n_adm && !bad; ++a) {
            koff[a + 1] = koff[a] + adm_k[a];
            for (uint32_t j = koff[a]; j < koff[a + 1]; ++j) {
                if (members[j] >= R || seen[members[j]]) bad = 2;
                else seen[members[j]] = 1;
            }
            for (uint32_t j = koff[a]; j < koff[a + 1]; ++j)
                if (members[j] < R) seen[members[j]] = 0;
            srt[a].key = adm_key[a];
            srt[a].cnt = adm_cnt[a];
        }
        if (!bad) {
            qsort(srt, n_adm, sizeof(imp_ent), cmp_imp);
            for (uint64_t a = 1; a < n_adm; ++a)
                if (srt[a].key == srt[a - 1].key) bad = 3;
        }
    }
    int st = CR_OK;
    if (bad == 1) st = cr_fail(ctx, CR_ENOMEM, "cr_plan_import: host allocation failed");
    else if (bad == 2) st = cr_fail(ctx, CR_EINVAL, "cr_plan_import: a member is >= R or repeated within a key");
    else if (bad == 3) st = cr_fail(ctx, CR_EINVAL, "cr_plan_import: a key is listed twice");
    if (st == CR_OK) st = plan_reserve(ctx, p, n_adm, R, W);
    if (st == CR_OK) {
        cudaStream_t s = ctx->stream;
        // the histogram of an imported plan is its admitted keys, ascending
        unsigned long long *hk = (unsigned long long *)malloc((n_adm + 1) * 16);
        if (!hk) st = cr_fail(ctx, CR_ENOMEM, "cr_plan_import: host allocation failed");
        for (uint64_t a = 0; hk && a < n_adm; ++a) {
            hk[a] = srt[a].key;
            hk[n_adm + 1 + a] = srt[a].cnt;
        }
        cr_plan_info_dev d;
        memset(&d, 0, sizeof(d));
        d.n = adm_lam;
        d.U = n_adm;
        d.S = n_adm;
        d.n_adm = n_adm;
        d.sum_k = sum_k;
        d.max_k = max_k;
        d.adm_lam = adm_lam;
        auto up = [&](void *dst, const void *src, size_t bytes) -> int {
            if (bytes && cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, s) != cudaSuccess)
                return cr_fail(ctx, CR_ECUDA, "cr_plan_import: copy failed");
            return CR_OK;
        };
        if (st == CR_OK) st = up(p->d_ukey, hk, n_adm * 8);
        if (st == CR_OK) st = up(p->d_ucnt, hk + n_adm + 1, n_adm * 8);
        if (st == CR_OK) st = up(p->d_adm_key, adm_key, n_adm * 8);
        if (st == CR_OK) st = up(p->d_adm_cnt, adm_cnt, n_adm * 8);
        if (st == CR_OK) st = up(p->d_adm_k, adm_k, n_adm * 4);
        if (st == CR_OK) st = up(p->d_koff, koff, (n_adm + 1) * 4);
        if (st == CR_OK) st = up(p->d_members, members, sum_k * 2);
        if (st == CR_OK && jobs) st = up(p->d_jobs, jobs, sum_k * 8);
        if (st == CR_OK && !jobs && sum_k && cudaMemsetAsync(p->d_jobs, 0, sum_k * 8, s) != cudaSuccess)
            st = cr_fail(ctx, CR_ECUDA, "cr_plan_import: memset failed");
        if (st == CR_OK && load) st = up(p->d_load, load, (size_t)R * 8);
        if (st == CR_OK && !load && cudaMemsetAsync(p->d_load, 0, (size_t)R * 8, s) != cudaSuccess)
            st = cr_fail(ctx, CR_ECUDA, "cr_plan_import: memset failed");
        if (st == CR_OK) st = up(p->d_info, &d, sizeof(d));
        if (st == CR_OK && cudaMemsetAsync(p->d_table, 0xff, p->table_slots * sizeof(cr_table_slot), s) != cudaSuccess)
            st = cr_fail(ctx, CR_ECUDA, "cr_plan_import: memset failed");
        if (st == CR_OK && n_adm) {
            const int bits = bits_for(p->table_slots - 1);
            CR_LAUNCH(ctx, k_table_insert, cr_blocks(n_adm, 256, (unsigned int)ctx->num_sms * 8u), 256, 0,
                      (const cr_plan_info_dev *)p->d_info, (const unsigned long long *)p->d_adm_key,
                      (const uint32_t *)p->d_adm_k, (const uint32_t *)p->d_koff, (const uint16_t *)p->d_members,
                      p->d_table, bits);
        }
        if (st == CR_OK) {
            p->n = adm_lam;
            p->qnum = 1;
            p->qden = 1;
            p->variant = CR_VARIANT_LPT;
            p->built = 1;
            st = cr_sync(ctx);  // the host arrays may be reused as soon as the call returns
        }
        free(hk);
    }
    free(koff);
    free(srt);
    free(seen);
    return st;
}
