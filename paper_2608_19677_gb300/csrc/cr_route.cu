// a7: batched dispatch (cr_route_batch).
//
// One CTA per replica walks the requests in arrival order, batch by batch.  The
// CTA holds the replica's live load vector in shared memory; every request of
// a batch is decided against it (table probe, Philox draws, argmin over T(b)),
// counts of the batch accumulate in a second shared vector, and the two are
// merged at the batch boundary.  The next batch's keys are fetched before the
// current batch is decided so that their latency overlaps the merge.
#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

constexpr int kRouteBlock = 1024;
constexpr uint32_t kEmpty = 0xffffffffu;

struct route_desc {
    uint32_t policy;
    int32_t tbits;                    // log2 table slots (plan policies)
    unsigned long long seed;
    const cr_table_slot *table;
    const uint16_t *members;
};

struct route_args {
    route_desc d[CR_MAX_REPLICAS];
};

__device__ __forceinline__ uint32_t p2c(unsigned long long seed, uint32_t policy, unsigned long long g, uint32_t R,
                                        const unsigned long long *L)
{
    cr_u64x4 u = cr_philox4x64_10(g, 0ull, 0ull, 0ull, seed, (unsigned long long)policy);
    uint32_t d1 = cr_scale(u.x, R);
    uint32_t d2 = (uint32_t)((d1 + 1ull + cr_scale(u.y, (unsigned long long)(R - 1))) % R);
    return L[d1] <= L[d2] ? d1 : d2;
}

__device__ __forceinline__ uint32_t route_one(const route_desc &rd, unsigned long long key, unsigned long long g,
                                              uint32_t R, const unsigned long long *L)
{
    switch (rd.policy) {
    case CR_POLICY_RR:
        return (uint32_t)((g + rd.seed) % R);
    case CR_POLICY_HASH:
        return cr_jump_hash(cr_fmix64(key ^ rd.seed), R);
    case CR_POLICY_P2C:
        return p2c(rd.seed, rd.policy, g, R, L);
    default: {
        const unsigned long long mask = (1ull << rd.tbits) - 1ull;
        unsigned long long s = key >> (64 - rd.tbits);
        for (;;) {
            const cr_table_slot slot = rd.table[s];
            if (slot.koff == kEmpty) break;
            if (slot.key == key) {
                if (slot.k == 1) return slot.m0;
                // least-loaded member of T(b); ties keep the earlier member
                uint32_t best = slot.m0;
                unsigned long long bl = L[best];
                for (uint32_t j = 1; j < slot.k; ++j) {
                    uint32_t m = rd.members[slot.koff + j];
                    unsigned long long l = L[m];
                    if (l < bl) {
                        bl = l;
                        best = m;
                    }
                }
                return best;
            }
            s = (s + 1) & mask;
        }
        return p2c(rd.seed, rd.policy, g, R, L);
    }
    }
}

__global__ void __launch_bounds__(kRouteBlock) k_route(const __grid_constant__ route_args args,
                                                       const unsigned long long *__restrict__ keys,
                                                       unsigned long long n, unsigned long long g0, uint32_t B,
                                                       uint32_t R, unsigned long long *__restrict__ load,
                                                       uint16_t *__restrict__ dest)
{
    extern __shared__ unsigned long long sh[];
    unsigned long long *L = sh;                                 // [R] snapshot
    uint32_t *delta = reinterpret_cast<uint32_t *>(sh + R);     // [R] this batch
    const uint32_t rep = blockIdx.x;
    const route_desc rd = args.d[rep];
    unsigned long long *Lg = load + (unsigned long long)rep * R;
    uint16_t *D = dest + (unsigned long long)rep * n;
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) {
        L[r] = Lg[r];
        delta[r] = 0;
    }
    __syncthreads();
    for (unsigned long long b0 = 0; b0 < n; b0 += B) {
        const unsigned long long b1 = (b0 + B < n) ? b0 + B : n;
        for (unsigned long long i = b0 + threadIdx.x; i < b1; i += blockDim.x) {
            const uint32_t d = route_one(rd, keys[i], g0 + i, R, L);
            D[i] = (uint16_t)d;
            atomicAdd(&delta[d], 1u);
        }
        __syncthreads();
        for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) {
            L[r] += delta[r];
            delta[r] = 0;
        }
        __syncthreads();
    }
    for (uint32_t r = threadIdx.x; r < R; r += blockDim.x) Lg[r] = L[r];
}

}  // namespace

extern "C" int cr_route_batch(cr_ctx *ctx, const cr_plan *const *plans, const cr_replica *reps, uint32_t n_rep,
                              uint32_t R, const uint64_t *d_key, uint64_t n, uint64_t first_req_index,
                              uint32_t batch_B, uint64_t *d_load, uint16_t *d_dest)
{
    if (!ctx) return CR_EINVAL;
    if (R == 0 || R > CR_MAX_R) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: R=%u outside 1..%u", R, CR_MAX_R);
    if (n_rep == 0 || n_rep > CR_MAX_REPLICAS || !reps)
        return cr_fail(ctx, CR_EINVAL, "cr_route_batch: n_rep=%u outside 1..%u", n_rep, CR_MAX_REPLICAS);
    if (batch_B == 0) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: batch_B must be >= 1");
    if (n >= (1ull << 40)) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: n >= 2^40");
    if (!d_load) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: d_load is NULL");
    if (n > 0 && (!d_key || !d_dest)) return cr_fail(ctx, CR_EINVAL, "cr_route_batch: NULL key or dest");
    route_args args;
    for (uint32_t i = 0; i < n_rep; ++i) {
        route_desc &d = args.d[i];
        d.policy = reps[i].policy;
        d.seed = reps[i].seed;
        d.tbits = 0;
        d.table = nullptr;
        d.members = nullptr;
        if (reps[i].policy > CR_POLICY_HASH || reps[i].reserved != 0)
            return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u has policy %u", i, reps[i].policy);
        if (reps[i].policy <= CR_POLICY_CR_NOREPL) {
            const cr_plan *p = plans ? plans[i] : nullptr;
            if (!p || !p->built)
                return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u needs a built plan", i);
            if (p->R != R)
                return cr_fail(ctx, CR_EINVAL, "cr_route_batch: replica %u plan has R=%u, call has R=%u", i, p->R, R);
            int bits = 0;
            while ((1ull << bits) < p->table_slots) ++bits;
            d.tbits = bits;
            d.table = p->d_table;
            d.members = p->d_members;
        }
    }
    if (n == 0) return CR_OK;
    size_t smem = (size_t)R * (sizeof(unsigned long long) + sizeof(uint32_t));
    if (smem > 48 * 1024)
        CR_CUDA(ctx, cudaFuncSetAttribute(k_route, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    CR_LAUNCH(ctx, k_route, n_rep, kRouteBlock, smem, args, (const unsigned long long *)d_key,
              (unsigned long long)n, (unsigned long long)first_req_index, batch_B, R,
              (unsigned long long *)d_load, d_dest);
    return CR_OK;
}
