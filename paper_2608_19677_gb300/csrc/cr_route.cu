// a7: batched dispatch (cr_route_batch).
//
// Two passes.  k_route_cand runs over every (replica, request) pair at once and
// does all the work that does not depend on the live load: the table probe,
// the Philox draws of power-of-two choices, round robin and the jump hash.
// Round-robin and hash replicas are then finished (their loads are counted by
// k_route_count); every other replica leaves one packed candidate per request.
// k_route_resolve then walks each load-dependent replica's requests in arrival
// order, batch by batch, on one CTA that holds the replica's live load in
// shared memory: a decision is one or two shared-memory reads, the batch's
// counts accumulate in a second shared vector and are merged at the boundary.
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
    uint32_t dep[CR_MAX_REPLICAS];    // load-dependent replicas, one CTA each in the resolve pass
};

// Candidate encoding, one u32 per (replica, request):
//   kind 0 FIXED  bits 0..15  destination (RR, HASH, and keys with k_b = 1)
//   kind 1 PAIR   bits 0..12  d1, bits 13..25 d2 (power-of-two choices; R <= 8192)
//   kind 2 SET    bits 0..29  table slot of a key with k_b > 1
constexpr uint32_t kFixed = 0u << 30, kPair = 1u << 30, kSet = 2u << 30, kKindMask = 3u << 30;

__device__ __forceinline__ uint32_t p2c_pair(unsigned long long seed, uint32_t policy, unsigned long long g,
                                             uint32_t R)
{
    cr_u64x4 u = cr_philox4x64_10(g, 0ull, 0ull, 0ull, seed, (unsigned long long)policy);
    uint32_t d1 = cr_scale(u.x, R);
    uint32_t d2 = (uint32_t)((d1 + 1ull + cr_scale(u.y, (unsigned long long)(R - 1))) % R);
    return kPair | d1 | (d2 << 13);
}

// Everything that does not depend on the live load, for every (replica, request).
// Load-independent replicas (RR, HASH) write their destinations directly.
__global__ void __launch_bounds__(256) k_route_cand(const __grid_constant__ route_args args, uint32_t n_rep,
                                                    const unsigned long long *__restrict__ keys,
                                                    unsigned long long n, unsigned long long g0, uint32_t R,
                                                    uint32_t *__restrict__ cand, uint16_t *__restrict__ dest)
{
    const unsigned long long total = n * n_rep;
    for (unsigned long long j = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; j < total;
         j += (unsigned long long)gridDim.x * blockDim.x) {
        const uint32_t rep = (uint32_t)(j / n);
        const unsigned long long i = j - (unsigned long long)rep * n;
        const route_desc &rd = args.d[rep];
        const unsigned long long g = g0 + i;
        switch (rd.policy) {
        case CR_POLICY_RR:
            dest[j] = (uint16_t)((g + rd.seed) % R);
            break;
        case CR_POLICY_HASH:
            dest[j] = (uint16_t)cr_jump_hash(cr_fmix64(keys[i] ^ rd.seed), R);
            break;
        case CR_POLICY_P2C:
            cand[j] = p2c_pair(rd.seed, rd.policy, g, R);
            break;
        default: {
            const unsigned long long key = keys[i];
            const unsigned long long mask = (1ull << rd.tbits) - 1ull;
            unsigned long long sl = key >> (64 - rd.tbits);
            uint32_t c = 0xffffffffu;
            for (;;) {
                const cr_table_slot slot = rd.table[sl];
                if (slot.koff == kEmpty) break;
                if (slot.key == key) {
                    c = slot.k == 1 ? (kFixed | slot.m0) : (kSet | (uint32_t)sl);
                    break;
                }
                sl = (sl + 1) & mask;
            }
            cand[j] = c != 0xffffffffu ? c : p2c_pair(rd.seed, rd.policy, g, R);
        }
        }
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

// Sequential part: one CTA per load-dependent replica walks the batches.
__device__ __forceinline__ uint32_t resolve(uint32_t c, const route_desc &rd, const unsigned long long *L)
{
    const uint32_t kind = c & kKindMask;
    if (kind == kFixed) return c & 0xffffu;
    if (kind == kPair) {
        const uint32_t d1 = c & 0x1fffu, d2 = (c >> 13) & 0x1fffu;
        return L[d1] <= L[d2] ? d1 : d2;
    }
    const cr_table_slot slot = rd.table[c & 0x3fffffffu];
    uint32_t best = slot.m0;
    unsigned long long bl = L[best];
    for (uint32_t m = 1; m < slot.k; ++m) {
        const uint32_t d = rd.members[slot.koff + m];
        const unsigned long long l = L[d];
        if (l < bl) {  // ties keep the earlier member
            bl = l;
            best = d;
        }
    }
    return best;
}

// Candidates are staged in shared memory a whole chunk (a multiple of the
// batch, at most kStage requests) ahead: while chunk c is resolved from one
// buffer, chunk c+1's loads are in flight into registers and land in the other.
constexpr uint32_t kStage = 16384;
constexpr int kStageRegs = kStage / kRouteBlock;  // 16

__global__ void __launch_bounds__(kRouteBlock) k_route_resolve(const __grid_constant__ route_args args,
                                                               const uint32_t *__restrict__ cand,
                                                               unsigned long long n, uint32_t B, uint32_t CH,
                                                               uint32_t R, unsigned long long *__restrict__ load,
                                                               uint16_t *__restrict__ dest)
{
    extern __shared__ unsigned long long sh[];
    unsigned long long *L = sh;                              // [R] live load
    uint32_t *delta = reinterpret_cast<uint32_t *>(sh + R);  // [R] this batch
    uint32_t *cbuf = delta + R;                              // [2][CH] staged candidates
    const uint32_t rep = args.dep[blockIdx.x];
    const route_desc rd = args.d[rep];
    unsigned long long *Lg = load + (unsigned long long)rep * R;
    const uint32_t *Cd = cand + (unsigned long long)rep * n;
    uint16_t *D = dest + (unsigned long long)rep * n;
    const uint32_t tid = threadIdx.x;
    for (uint32_t r = tid; r < R; r += blockDim.x) {
        L[r] = Lg[r];
        delta[r] = 0;
    }
    if (CH == 0) {
        // batches longer than the stage: candidates straight from global memory
        __syncthreads();
        for (unsigned long long b0 = 0; b0 < n; b0 += B) {
            const unsigned long long b1 = (b0 + B < n) ? b0 + B : n;
            for (unsigned long long i = b0 + tid; i < b1; i += blockDim.x) {
                const uint32_t d = resolve(Cd[i], rd, L);
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
        for (uint32_t r = tid; r < R; r += blockDim.x) Lg[r] = L[r];
        return;
    }
    for (uint32_t x = tid; x < CH && x < n; x += blockDim.x) cbuf[x] = Cd[x];
    __syncthreads();
    int cur = 0;
    for (unsigned long long c0 = 0; c0 < n; c0 += CH) {
        const unsigned long long c1 = (c0 + CH < n) ? c0 + CH : n;
        // next chunk in flight
        uint32_t nx[kStageRegs];
#pragma unroll
        for (int q = 0; q < kStageRegs; ++q) {
            const unsigned long long i = c1 + (unsigned long long)q * blockDim.x + tid;
            nx[q] = (q * blockDim.x + tid < CH && i < n) ? Cd[i] : 0u;
        }
        const uint32_t *cb = cbuf + (size_t)cur * CH;
        for (unsigned long long b0 = c0; b0 < c1; b0 += B) {
            const unsigned long long b1 = (b0 + B < c1) ? b0 + B : c1;
            for (unsigned long long i = b0 + tid; i < b1; i += blockDim.x) {
                const uint32_t d = resolve(cb[i - c0], rd, L);
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
        uint32_t *nb = cbuf + (size_t)(cur ^ 1) * CH;
#pragma unroll
        for (int q = 0; q < kStageRegs; ++q)
            if (q * blockDim.x + tid < CH) nb[q * blockDim.x + tid] = nx[q];
        __syncthreads();
        cur ^= 1;
    }
    for (uint32_t r = tid; r < R; r += blockDim.x) Lg[r] = L[r];
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
    for (uint32_t i = 0; i < n_rep; ++i)
        if (args.d[i].policy <= CR_POLICY_CR_NOREPL && args.d[i].tbits > 30)
            return cr_fail(ctx, CR_EINVAL, "cr_route_batch: plan table too large");
    // replicas whose choices depend on the live load
    uint32_t n_dep = 0;
    for (uint32_t i = 0; i < n_rep; ++i)
        if (reps[i].policy != CR_POLICY_RR && reps[i].policy != CR_POLICY_HASH) args.dep[n_dep++] = i;
    void *pc;
    CR_TRY(cr_scratch(ctx, SCR_ROUTE_DESC, (size_t)n * n_rep * sizeof(uint32_t), &pc));
    uint32_t *cand = (uint32_t *)pc;
    const unsigned int gcap = (unsigned int)ctx->num_sms * 16u;
    CR_LAUNCH(ctx, k_route_cand, cr_blocks(n * n_rep, 256, gcap), 256, 0, args, n_rep,
              (const unsigned long long *)d_key, (unsigned long long)n, (unsigned long long)first_req_index, R, cand,
              d_dest);
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
    if (n_dep) {
        // staging chunk: a whole number of batches, at most kStage requests
        const uint32_t CH = batch_B <= kStage ? (kStage / batch_B) * batch_B : 0u;  // 0: no staging
        size_t smem = (size_t)R * (sizeof(unsigned long long) + sizeof(uint32_t)) + 2ull * CH * sizeof(uint32_t);
        if (smem > 48 * 1024)
            CR_CUDA(ctx, cudaFuncSetAttribute(k_route_resolve, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smem));
        CR_LAUNCH(ctx, k_route_resolve, n_dep, kRouteBlock, smem, args, (const uint32_t *)cand,
                  (unsigned long long)n, batch_B, CH, R, (unsigned long long *)d_load, d_dest);
    }
    return CR_OK;
}
