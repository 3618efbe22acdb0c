// a2..a6: per-interval plan construction (Eq. 1 and Algorithm 1).
//
//   histogram   radix sort of the interval's keys, run-length encoding -> (b, lambda_b)
//   order       stable radix sort of (n - lambda_b): lambda descending, key ascending
//   per plan    k_b (Eq. 1), inclusive scan of k_b, admission cut, admitted arrays,
//               cold-tail total, placement (LPT: one warp, sequential over admitted
//               keys, warp argmin over cached per-lane minima; RANDOM: one warp per
//               key, Fisher-Yates steps in shared memory), then the device hash
//               table b -> (offset, k_b, first member) used by dispatch.
// No host synchronisation: sizes known only on the device (U, n_adm) are read
// by the kernels, and grids are sized from host-side upper bounds.
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
    info->n_adm = 0;
    info->sum_k = 0;
    info->cold = 0;
    info->max_k = 0;
}

__global__ void k_rle_flags(const unsigned long long *__restrict__ s, uint64_t n, uint32_t *__restrict__ flag)
{
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x)
        flag[i] = (i == 0 || s[i] != s[i - 1]) ? 1u : 0u;
}

// pos = exclusive scan of flags; every run head writes its key and position.
__global__ void k_rle_heads(const unsigned long long *__restrict__ s, const uint32_t *__restrict__ pos, uint64_t n,
                            unsigned long long *__restrict__ ukey, uint32_t *__restrict__ head,
                            cr_plan_info_dev *info)
{
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x) {
        bool h = (i == 0 || s[i] != s[i - 1]);
        if (h) {
            ukey[pos[i]] = s[i];
            head[pos[i]] = (uint32_t)i;
        }
        if (i == n - 1) {
            unsigned long long U = (unsigned long long)pos[i] + (h ? 1ull : 0ull);
            info->U = U;
            head[U] = (uint32_t)n;
        }
    }
}

// lambda_b and the sort key (n - lambda_b); entries at u >= U sort last with key n.
__global__ void k_rle_counts(const uint32_t *__restrict__ head, uint64_t n, const cr_plan_info_dev *info,
                             unsigned long long *__restrict__ ucnt, uint32_t *__restrict__ sortkey)
{
    const unsigned long long U = info->U;
    for (uint64_t u = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n; u += (uint64_t)gridDim.x * blockDim.x) {
        if (u < U) {
            uint32_t c = head[u + 1] - head[u];
            ucnt[u] = c;
            sortkey[u] = (uint32_t)(n - c);
        } else {
            sortkey[u] = (uint32_t)n;
        }
    }
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
    const unsigned long long U = info->U;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < U; a += (uint64_t)gridDim.x * blockDim.x)
        kk[a] = norepl ? 1ull : eq1_kb(ucnt[order[a]], num, den, R);
}

// Admission: the longest prefix of the order whose inclusive k-sum stays <= C.
__global__ void k_plan_admit(const unsigned long long *__restrict__ kscan, cr_plan_info_dev *info,
                             unsigned long long C)
{
    const unsigned long long U = info->U;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < U; a += (uint64_t)gridDim.x * blockDim.x) {
        if (kscan[a] <= C && (a + 1 == U || kscan[a + 1] > C)) {
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
    const unsigned long long U = info->U, na = info->n_adm;
    unsigned long long cold = 0;
    uint32_t kmax = 0;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < U; a += (uint64_t)gridDim.x * blockDim.x) {
        uint32_t u = order[a];
        if (a < na) {
            uint32_t k = (uint32_t)(kscan[a] - (a ? kscan[a - 1] : 0ull));
            adm_key[a] = ukey[u];
            adm_cnt[a] = ucnt[u];
            adm_k[a] = k;
            koff[a] = (uint32_t)(kscan[a] - k);
            kmax = k > kmax ? k : kmax;
            if (a + 1 == na) koff[na] = (uint32_t)kscan[a];
        } else {
            cold += ucnt[u];
        }
    }
    cold = cr_warp_sum_u64(cold);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
    if (cr_lane() == 0) {
        if (cold) atomicAdd(&info->cold, cold);
        if (kmax) atomicMax(&info->max_k, (unsigned long long)kmax);
    }
}

__global__ void k_plan_init_load(const cr_plan_info_dev *info, const unsigned long long *__restrict__ init_load,
                                 uint32_t R, unsigned long long *__restrict__ load, uint32_t *status)
{
    const unsigned long long share = info->cold / R;
    for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
        unsigned long long v = init_load ? init_load[r] : share;
        if (v >= kLoadLimit) atomicOr(status, CR_FLAG_OVERFLOW);
        load[r] = v;
    }
}

// LPT placement (Algorithm 1 placement loop) on one warp.  Lane l owns the
// destinations r = l, l+32, ...; it caches the smallest (L[r], r) among its
// untaken ones.  Each job is one warp argmin over the 32 cached minima.
__device__ __forceinline__ void lane_min(const unsigned long long *L, const unsigned char *taken, uint32_t R,
                                         uint32_t lane, unsigned long long &mL, uint32_t &mr)
{
    mL = ~0ull;
    mr = 0xffffffffu;  // no eligible destination on this lane
    for (uint32_t r = lane; r < R; r += 32) {
        if (taken[r]) continue;
        unsigned long long v = L[r];
        if (mr == 0xffffffffu || v < mL) {  // r ascending: ties keep the lower index
            mL = v;
            mr = r;
        }
    }
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
    __syncwarp();
    unsigned long long mL;
    uint32_t mr;
    lane_min(L, taken, R, lane, mL, mr);
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
        for (uint32_t s = 0; s < k; ++s) {
            // warp argmin of (L, r) over the lanes' cached minima
            unsigned long long bL = mL;
            uint32_t br = mr;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                unsigned long long oL = __shfl_xor_sync(0xffffffffu, bL, o);
                uint32_t orr = __shfl_xor_sync(0xffffffffu, br, o);
                if (oL < bL || (oL == bL && orr < br)) {
                    bL = oL;
                    br = orr;
                }
            }
            const unsigned long long job = q + (s < rem ? 1ull : 0ull);
            if (lane == 0) {
                members[base + s] = (uint16_t)br;
                jobs[base + s] = job;
            }
            if ((br & 31u) == lane) {
                // a chosen destination is not eligible again for this key
                if (k > 1) taken[br] = 1;
                unsigned long long nl = L[br] + job;
                if (nl >= kLoadLimit) overflow = true;
                L[br] = nl;
                lane_min(L, taken, R, lane, mL, mr);
            }
            __syncwarp();
        }
        if (k > 1) {
            // release this key's destinations for the next key
            bool dirty = false;
            for (uint32_t s = 0; s < k; ++s) {
                uint32_t m = members[base + s];
                if ((m & 31u) == lane) {
                    taken[m] = 0;
                    dirty = true;
                }
            }
            __syncwarp();
            if (dirty) lane_min(L, taken, R, lane, mL, mr);
            __syncwarp();
        }
    }
    for (uint32_t r = lane; r < R; r += 32) load_g[r] = L[r];
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(status, CR_FLAG_OVERFLOW);
}

// RANDOM placement: one warp per admitted key; the first k steps of a
// Fisher-Yates shuffle of 0..R-1 held in shared memory.
constexpr int kRandWarps = 4;

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
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5;
    uint16_t *perm = perm_all + (size_t)warp * R;
    const unsigned long long na = info->n_adm;
    const unsigned long long nw = (unsigned long long)gridDim.x * kRandWarps;
    for (unsigned long long a = (unsigned long long)blockIdx.x * kRandWarps + warp; a < na; a += nw) {
        const uint32_t k = adm_k[a], base = koff[a];
        const unsigned long long lam = adm_cnt[a];
        const unsigned long long q = lam / k, rem = lam % k;
        for (uint32_t r = lane; r < R; r += 32) perm[r] = (uint16_t)r;
        __syncwarp();
        if (lane == 0) {
            for (uint32_t s = 0; s < k; ++s) {
                cr_u64x4 u = cr_philox4x64_10(a, s, 1ull, epoch, seed, (unsigned long long)CR_POLICY_CR_NOLPT);
                uint32_t t = s + cr_scale(u.x, (unsigned long long)(R - s));
                uint16_t tmp = perm[s];
                perm[s] = perm[t];
                perm[t] = tmp;
            }
        }
        __syncwarp();
        for (uint32_t s = lane; s < k; s += 32) {
            const unsigned long long job = q + (s < rem ? 1ull : 0ull);
            uint16_t m = perm[s];
            members[base + s] = m;
            jobs[base + s] = job;
            unsigned long long old = atomicAdd(&load_g[m], job);
            if (old + job >= kLoadLimit) atomicOr(status, CR_FLAG_OVERFLOW);
        }
        __syncwarp();
    }
}

__global__ void k_table_insert(const cr_plan_info_dev *info, const unsigned long long *__restrict__ adm_key,
                               const uint32_t *__restrict__ adm_k, const uint32_t *__restrict__ koff,
                               const uint16_t *__restrict__ members, cr_table_slot *__restrict__ table,
                               int bits)
{
    const unsigned long long na = info->n_adm;
    const unsigned long long mask = (1ull << bits) - 1ull;
    for (uint64_t a = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; a < na; a += (uint64_t)gridDim.x * blockDim.x) {
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
    if (pp->variant > CR_VARIANT_NOREPL || pp->reserved != 0)
        return cr_fail(ctx, CR_EINVAL, "plan: bad variant %u or reserved field", pp->variant);
    return CR_OK;
}

extern "C" int cr_build_plans(cr_ctx *ctx, const uint64_t *d_key, uint64_t n, const cr_plan_params *params,
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
        plans[j]->built = 1;
        CR_LAUNCH(ctx, k_plan_reset, 1, 1, 0, plans[j]->d_info, (unsigned long long)n);
    }
    cr_plan *p0 = plans[0];
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    const unsigned int grid_n = cr_blocks(n, 256, gcap);

    // ---- shared histogram and admission order ------------------------------
    const uint32_t *order = nullptr;
    if (n > 0) {
        const unsigned long long *sorted = nullptr;
        CR_TRY(cr_radix_sort_u64(ctx, (const unsigned long long *)d_key, nullptr, n, 64, &sorted, nullptr));
        void *pa, *pb, *pc;
        CR_TRY(cr_scratch(ctx, SCR_PLAN_A, (n + 1) * sizeof(uint32_t), &pa));
        CR_TRY(cr_scratch(ctx, SCR_PLAN_B, (n + 2) * sizeof(uint32_t), &pb));
        CR_TRY(cr_scratch(ctx, SCR_PLAN_C, (n + 1) * sizeof(uint32_t), &pc));
        uint32_t *flag = (uint32_t *)pa, *head = (uint32_t *)pb, *skey = (uint32_t *)pc;
        CR_LAUNCH(ctx, k_rle_flags, grid_n, 256, 0, sorted, n, flag);
        CR_TRY(cr_scan_u32(ctx, flag, flag, n, nullptr));
        CR_LAUNCH(ctx, k_rle_heads, grid_n, 256, 0, sorted, flag, n, p0->d_ukey, head, p0->d_info);
        CR_LAUNCH(ctx, k_rle_counts, grid_n, 256, 0, head, n, (const cr_plan_info_dev *)p0->d_info, p0->d_ucnt,
                  skey);
        const uint32_t *sk_sorted = nullptr;
        CR_TRY(cr_radix_sort_u32(ctx, skey, nullptr, n, bits_for(n), &sk_sorted, &order));
        // `order` lives in radix scratch until the next sort; nothing below sorts.
    }

    // ---- per plan -------------------------------------------------------------
    for (uint32_t j = 0; j < n_plans; ++j) {
        cr_plan *p = plans[j];
        const cr_plan_params &pp = params[j];
        const uint64_t C = (uint64_t)pp.R * pp.W;
        if (j > 0 && n > 0) {
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_ukey, p0->d_ukey, n * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(p->d_ucnt, p0->d_ucnt, n * sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
            CR_CUDA(ctx, cudaMemcpyAsync(&p->d_info->U, &p0->d_info->U, sizeof(unsigned long long),
                                         cudaMemcpyDeviceToDevice, ctx->stream));
        }
        CR_CUDA(ctx, cudaMemsetAsync(p->d_table, 0xff, p->table_slots * sizeof(cr_table_slot), ctx->stream));
        if (n > 0) {
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
        CR_LAUNCH(ctx, k_plan_init_load, cr_blocks(pp.R, 256, gcap), 256, 0, (const cr_plan_info_dev *)p->d_info,
                  (const unsigned long long *)pp.d_init_load, pp.R, p->d_load, ctx->d_status);
        if (n > 0) {
            if (pp.variant == CR_VARIANT_RANDOM) {
                size_t smem = (size_t)kRandWarps * pp.R * sizeof(uint16_t);
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_random, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                uint64_t adm = n < C ? n : C;
                CR_LAUNCH(ctx, k_plan_random, cr_blocks(adm, kRandWarps, gcap), kRandWarps * 32, smem,
                          (const cr_plan_info_dev *)p->d_info, (const unsigned long long *)p->d_adm_cnt,
                          (const uint32_t *)p->d_adm_k, (const uint32_t *)p->d_koff, pp.R,
                          (unsigned long long)pp.seed, (unsigned long long)pp.epoch, p->d_load, p->d_members,
                          p->d_jobs, ctx->d_status);
            } else {
                size_t smem = (size_t)pp.R * (sizeof(unsigned long long) + 1) + 16;
                if (smem > 48 * 1024)
                    CR_CUDA(ctx, cudaFuncSetAttribute(k_plan_lpt, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)smem));
                CR_LAUNCH(ctx, k_plan_lpt, 1, 32, smem, (const cr_plan_info_dev *)p->d_info,
                          (const unsigned long long *)p->d_adm_cnt, (const uint32_t *)p->d_adm_k,
                          (const uint32_t *)p->d_koff, pp.R, p->d_load, p->d_members, p->d_jobs, ctx->d_status);
            }
            int bits = bits_for(p->table_slots - 1);
            uint64_t adm = n < C ? n : C;
            CR_LAUNCH(ctx, k_table_insert, cr_blocks(adm, 256, gcap), 256, 0, (const cr_plan_info_dev *)p->d_info,
                      (const unsigned long long *)p->d_adm_key, (const uint32_t *)p->d_adm_k,
                      (const uint32_t *)p->d_koff, (const uint16_t *)p->d_members, p->d_table, bits);
        }
    }
    return CR_OK;
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

extern "C" int cr_plan_export(cr_ctx *ctx, const cr_plan *p, uint64_t *ukey, uint64_t *ucnt, uint64_t *adm_key,
                              uint64_t *adm_cnt, uint32_t *adm_k, uint32_t *koff, uint16_t *members,
                              uint64_t *jobs, uint64_t *load)
{
    cr_plan_info info;
    CR_TRY(cr_plan_get_info(ctx, p, &info));
    cudaStream_t s = ctx->stream;
    if (ukey && info.U) CR_CUDA(ctx, cudaMemcpyAsync(ukey, p->d_ukey, info.U * 8, cudaMemcpyDeviceToHost, s));
    if (ucnt && info.U) CR_CUDA(ctx, cudaMemcpyAsync(ucnt, p->d_ucnt, info.U * 8, cudaMemcpyDeviceToHost, s));
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
