// f2: difference of two plans (replanning under drift; supplement "Replanning
// Under Drift", replan table: cache churn = 1 - Jaccard of consecutive
// assignment sets, count churn = share of keys whose k_b changes).
//
// The assignment set of a plan is its set of (key, destination) pairs.  Pass 1
// takes every admitted key of plan a, one warp per key: it looks the key up in
// b's device table; for a key admitted by both, the warp marks b's members in
// a per-warp bitmap of R bits in shared memory and counts a's members found
// there (|T_a(key) & T_b(key)|), then clears the bits it set.  Pass 2 takes
// every admitted key of b and counts only the keys a did not admit.
//
// Count churn is taken over every key of either plan's histogram, with k_b
// from Eq. 1 of that plan's rate (k_b is defined for every key, admitted or
// not; a key absent from an interval has lambda = 0, so k_b = 1): each plan's
// histogram goes into an open-addressing table (key -> k_b), and each side's
// keys are looked up in the other's.  All counts are integers accumulated
// with 64-bit atomics.
#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

constexpr uint32_t kEmptySlot = 0xffffffffu;
constexpr int kDiffWarps = 8;

enum { D_COMMON = 0, D_PAIRS_COMMON, D_K_CHANGED, D_SET_CHANGED, D_HIST_KEYS, D_HIST_KB_CHANGED, D_NUM };

struct hist_slot {  // 16 bytes; used = 0 marks an empty slot
    unsigned long long key;
    uint32_t kb;
    uint32_t used;
};

struct hist_side {  // a plan's histogram and the q_cap of its Eq. 1
    const unsigned long long *ukey, *ucnt;
    const unsigned long long *U;  // device
    unsigned long long num, den;
    uint32_t R;
    int norepl;
};

// Eq. 1: k_b = min(R, max(1, ceil(lambda / q_cap))), q_cap = num / den; 1 for single-copy plans.
__device__ __forceinline__ uint32_t hist_kb(const hist_side &h, unsigned long long lam)
{
    if (h.norepl) return 1u;
    const unsigned long long a = lam * h.den;  // lambda < 2^32, den < 2^32
    unsigned long long k = a / h.num + ((a % h.num) != 0ull);
    if (k < 1ull) k = 1ull;
    if (k > h.R) k = h.R;
    return (uint32_t)k;
}

__global__ void __launch_bounds__(256) k_diff_hist_table(hist_side h, hist_slot *__restrict__ tab, int tbits)
{
    const unsigned long long U = *h.U, mask = (1ull << tbits) - 1ull;
    for (unsigned long long u = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; u < U;
         u += (unsigned long long)gridDim.x * blockDim.x) {
        const unsigned long long key = h.ukey[u];
        unsigned long long sl = key >> (64 - tbits);
        while (atomicCAS(&tab[sl].used, 0u, 1u) != 0u) sl = (sl + 1) & mask;  // keys are distinct
        tab[sl].key = key;
        tab[sl].kb = hist_kb(h, h.ucnt[u]);
    }
}

// Keys of side h looked up in the other side's table.  Pass 1 counts every key
// of h; pass 2 only the keys the other side does not hold (k_b = 1 there).
__global__ void __launch_bounds__(256) k_diff_hist_cmp(hist_side h, const hist_slot *__restrict__ other, int tbits,
                                                       int count_found, unsigned long long *ctr)
{
    const unsigned long long U = *h.U, mask = (1ull << tbits) - 1ull;
    unsigned long long keys = 0, changed = 0;
    for (unsigned long long u = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; u < U;
         u += (unsigned long long)gridDim.x * blockDim.x) {
        const unsigned long long key = h.ukey[u];
        unsigned long long sl = key >> (64 - tbits);
        uint32_t ko = 0;
        for (;;) {
            const hist_slot s = other[sl];
            if (!s.used) break;
            if (s.key == key) {
                ko = s.kb;
                break;
            }
            sl = (sl + 1) & mask;
        }
        if (ko != 0 && !count_found) continue;
        const uint32_t kh = hist_kb(h, h.ucnt[u]);
        ++keys;
        changed += kh != (ko != 0 ? ko : 1u);
    }
    for (int o = 16; o > 0; o >>= 1) {
        keys += __shfl_xor_sync(0xffffffffu, keys, o);
        changed += __shfl_xor_sync(0xffffffffu, changed, o);
    }
    if ((threadIdx.x & 31) == 0) {
        if (keys) atomicAdd(&ctr[D_HIST_KEYS], keys);
        if (changed) atomicAdd(&ctr[D_HIST_KB_CHANGED], changed);
    }
}

struct diff_keys {  // the plan whose admitted keys are walked
    const unsigned long long *adm_key;
    const uint32_t *adm_k;
    const uint32_t *koff;
    const uint16_t *members;
    const unsigned long long *n_adm;  // device
};

struct diff_table {  // the plan whose table is probed
    const cr_table_slot *table;
    const uint16_t *members;
    int tbits;
};

__global__ void __launch_bounds__(kDiffWarps * 32) k_plan_diff(diff_keys a, diff_table b, uint32_t words,
                                                               int count_common, unsigned long long *ctr)
{
    extern __shared__ uint32_t bm[];  // [kDiffWarps][words] member bitmaps, kept all-zero between keys
    const uint32_t lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    uint32_t *mine = bm + (size_t)wib * words;
    for (uint32_t x = lane; x < words; x += 32) mine[x] = 0;
    __syncwarp();
    const unsigned long long n = *a.n_adm;
    const unsigned long long mask = (1ull << b.tbits) - 1ull;
    unsigned long long common = 0, pairs_common = 0, k_changed = 0, set_changed = 0;
    for (unsigned long long e = (unsigned long long)blockIdx.x * kDiffWarps + wib; e < n;
         e += (unsigned long long)gridDim.x * kDiffWarps) {
        const unsigned long long key = a.adm_key[e];
        const uint32_t ka = a.adm_k[e], oa = a.koff[e];
        // every lane probes the same slots (one L2 line per probe)
        unsigned long long sl = key >> (64 - b.tbits);
        uint32_t kb = 0, ob = 0;
        for (;;) {
            const cr_table_slot slot = b.table[sl];
            if (slot.koff == kEmptySlot) break;
            if (slot.key == key) {
                kb = slot.k;
                ob = slot.koff;
                break;
            }
            sl = (sl + 1) & mask;
        }
        if (kb == 0) {  // admitted by a only: k_b 0 vs ka, empty set vs T_a
            ++k_changed;
            ++set_changed;
            continue;
        }
        if (!count_common) continue;
        for (uint32_t m = lane; m < kb; m += 32) {
            const uint32_t d = b.members[ob + m];
            atomicOr(&mine[d >> 5], 1u << (d & 31));
        }
        __syncwarp();
        uint32_t inter = 0;
        for (uint32_t m = lane; m < ka; m += 32) {
            const uint32_t d = a.members[oa + m];
            inter += (mine[d >> 5] >> (d & 31)) & 1u;
        }
        for (int o = 16; o > 0; o >>= 1) inter += __shfl_xor_sync(0xffffffffu, inter, o);
        __syncwarp();
        for (uint32_t m = lane; m < kb; m += 32) mine[b.members[ob + m] >> 5] = 0;
        __syncwarp();
        ++common;
        pairs_common += inter;
        k_changed += ka != kb;
        set_changed += !(ka == kb && inter == ka);
    }
    if (lane == 0) {
        if (common) atomicAdd(&ctr[D_COMMON], common);
        if (pairs_common) atomicAdd(&ctr[D_PAIRS_COMMON], pairs_common);
        if (k_changed) atomicAdd(&ctr[D_K_CHANGED], k_changed);
        if (set_changed) atomicAdd(&ctr[D_SET_CHANGED], set_changed);
    }
}

int table_bits(const cr_plan *p)
{
    int bits = 0;
    while ((1ull << bits) < p->table_slots) ++bits;
    return bits;
}

}  // namespace

extern "C" int cr_plan_diff(cr_ctx *ctx, const cr_plan *a, const cr_plan *b, cr_plan_diff_counts *out)
{
    if (!ctx || !out) return CR_EINVAL;
    if (!a || !b || !a->built || !b->built) return cr_fail(ctx, CR_EINVAL, "cr_plan_diff: both plans must be built");
    if (a->R != b->R) return cr_fail(ctx, CR_EINVAL, "cr_plan_diff: plans have R=%u and R=%u", a->R, b->R);
    // scratch: counters, then one histogram table per plan (>= 2 slots per request)
    uint64_t slots = 16;
    while (slots < 2 * ((a->n > b->n ? a->n : b->n) + 1)) slots <<= 1;
    int hbits = 0;
    while ((1ull << hbits) < slots) ++hbits;
    const size_t ctr_bytes = 256, tab_bytes = slots * sizeof(hist_slot);
    void *pc;
    CR_TRY(cr_scratch(ctx, SCR_DIFF, ctr_bytes + 2 * tab_bytes, &pc));
    unsigned long long *ctr = (unsigned long long *)pc;
    hist_slot *tabs[2] = {(hist_slot *)((char *)pc + ctr_bytes), (hist_slot *)((char *)pc + ctr_bytes + tab_bytes)};
    CR_CUDA(ctx, cudaMemsetAsync(pc, 0, ctr_bytes + 2 * tab_bytes, ctx->stream));
    const uint32_t words = (a->R + 31) / 32;
    const size_t smem = (size_t)kDiffWarps * words * sizeof(uint32_t);
    const unsigned int gcap = (unsigned int)ctx->num_sms * 8u;
    for (int pass = 0; pass < 2; ++pass) {
        const cr_plan *x = pass == 0 ? a : b, *y = pass == 0 ? b : a;
        diff_keys dk{x->d_adm_key, x->d_adm_k, x->d_koff, x->d_members, &x->d_info->n_adm};
        diff_table dt{y->d_table, y->d_members, table_bits(y)};
        CR_LAUNCH(ctx, k_plan_diff, cr_blocks(x->cap_adm, kDiffWarps, gcap), kDiffWarps * 32, smem, dk, dt, words,
                  pass == 0 ? 1 : 0, ctr);
    }
    const cr_plan *side[2] = {a, b};
    hist_side hs[2];
    for (int i = 0; i < 2; ++i) {
        const cr_plan *p = side[i];
        hs[i] = hist_side{p->d_ukey, p->d_ucnt, &p->d_info->U, p->qnum, p->qden, p->R,
                          p->variant == CR_VARIANT_NOREPL ? 1 : 0};
        CR_LAUNCH(ctx, k_diff_hist_table, cr_blocks(p->n, 256, gcap), 256, 0, hs[i], tabs[i], hbits);
    }
    for (int i = 0; i < 2; ++i)
        CR_LAUNCH(ctx, k_diff_hist_cmp, cr_blocks(side[i]->n, 256, gcap), 256, 0, hs[i], (const hist_slot *)tabs[i ^ 1],
                  hbits, i == 0 ? 1 : 0, ctr);
    unsigned long long h[D_NUM];
    cr_plan_info_dev ia, ib;
    CR_CUDA(ctx, cudaMemcpyAsync(h, ctr, sizeof(h), cudaMemcpyDeviceToHost, ctx->stream));
    CR_CUDA(ctx, cudaMemcpyAsync(&ia, a->d_info, sizeof(ia), cudaMemcpyDeviceToHost, ctx->stream));
    CR_CUDA(ctx, cudaMemcpyAsync(&ib, b->d_info, sizeof(ib), cudaMemcpyDeviceToHost, ctx->stream));
    CR_TRY(cr_sync(ctx));
    out->keys_a = ia.n_adm;
    out->keys_b = ib.n_adm;
    out->keys_common = h[D_COMMON];
    out->pairs_a = ia.sum_k;
    out->pairs_b = ib.sum_k;
    out->pairs_common = h[D_PAIRS_COMMON];
    out->adm_k_changed = h[D_K_CHANGED];
    out->adm_set_changed = h[D_SET_CHANGED];
    out->hist_keys = h[D_HIST_KEYS];
    out->hist_kb_changed = h[D_HIST_KB_CHANGED];
    return CR_OK;
}
