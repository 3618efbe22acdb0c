// Device-wide scan and stable LSD radix sort.
//
// Radix sort: 8-bit digits, three launches per pass and no inter-block waits:
//   upsweep   per-tile digit counts, written digit-major [256][ntiles]
//   scan      exclusive scan of those counts = each tile's output base per digit
//   downsweep each tile ranks its items stably (arrival order = round, warp,
//             lane; warp peers found with __match_any_sync) and scatters them.
// Scan: reduce-then-scan over 4096-element blocks, recursing on the partials.
#include "cr_device.cuh"
#include "cr_internal.cuh"

namespace {

constexpr int kSortBlock = 256;
constexpr int kSortItems = 8;
constexpr int kSortTile = kSortBlock * kSortItems;  // 2048 items per tile
constexpr int kScanBlock = 1024;
constexpr int kScanItems = 4;
constexpr int kScanTile = kScanBlock * kScanItems;  // 4096 elements per block

// ---------------------------------------------------------------- scan ----
template <typename T>
__device__ __forceinline__ T warp_incl_scan(T v)
{
    const uint32_t lane = cr_lane();
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        T u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= (uint32_t)o) v += u;
    }
    return v;
}

// Exclusive scan of one value per thread across a 1024-thread block; returns
// the exclusive prefix and writes the block total to *total.
template <typename T>
__device__ __forceinline__ T block_excl_scan(T v, T *total)
{
    __shared__ T warp_sums[32];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5;
    T inc = warp_incl_scan(v);
    if (lane == 31) warp_sums[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        T s = warp_sums[lane];  // 1024 threads: 32 warps, every lane has a warp sum
        T si = warp_incl_scan(s);
        warp_sums[lane] = si - s;
        if (lane == 31) *total = si;
    }
    __syncthreads();
    T r = warp_sums[warp] + inc - v;
    __syncthreads();
    return r;
}

template <typename T>
__global__ void __launch_bounds__(kScanBlock) k_scan_reduce(const T *__restrict__ in, uint64_t n,
                                                            T *__restrict__ partial)
{
    __shared__ T tot;
    const uint64_t base = (uint64_t)blockIdx.x * kScanTile;
    T s = 0;
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
        uint64_t i = base + (uint64_t)j * kScanBlock + threadIdx.x;
        if (i < n) s += in[i];
    }
    block_excl_scan<T>(s, &tot);
    if (threadIdx.x == 0) partial[blockIdx.x] = tot;
}

// Scan one 4096-element block (blocked arrangement: thread t owns 4 consecutive
// elements), adding the block's offset from `partial` (exclusive) if given.
template <typename T>
__global__ void __launch_bounds__(kScanBlock) k_scan_block(const T *__restrict__ in, T *__restrict__ out,
                                                           uint64_t n, const T *__restrict__ partial,
                                                           int inclusive, T *__restrict__ total_out)
{
    __shared__ T tot;
    const uint64_t base = (uint64_t)blockIdx.x * kScanTile + (uint64_t)threadIdx.x * kScanItems;
    T x[kScanItems];
    T s = 0;
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
        x[j] = (base + j < n) ? in[base + j] : (T)0;
        s += x[j];
    }
    T pre = block_excl_scan<T>(s, &tot);
    if (partial) pre += partial[blockIdx.x];
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
        T nx = pre + x[j];
        if (base + j < n) out[base + j] = inclusive ? nx : pre;
        pre = nx;
    }
    if (total_out && threadIdx.x == kScanBlock - 1 && blockIdx.x == gridDim.x - 1) *total_out = pre;
}

// Elements of partial sums needed below a scan of n elements (all levels).
static uint64_t scan_partials_size(uint64_t n)
{
    uint64_t total = 0;
    uint64_t m = (n + kScanTile - 1) / kScanTile;
    while (m > 1) {
        total += m + 32;
        m = (m + kScanTile - 1) / kScanTile;
    }
    return total;
}

template <typename T>
int scan_rec(cr_ctx *ctx, const T *in, T *out, uint64_t n, int inclusive, T *d_total, T *partials)
{
    uint64_t nb = (n + kScanTile - 1) / kScanTile;
    if (nb == 1) {
        CR_LAUNCH(ctx, k_scan_block<T>, 1, kScanBlock, 0, in, out, n, (const T *)nullptr, inclusive, d_total);
        return CR_OK;
    }
    T *partial = partials;
    CR_LAUNCH(ctx, k_scan_reduce<T>, (unsigned int)nb, kScanBlock, 0, in, n, partial);
    CR_TRY(scan_rec<T>(ctx, partial, partial, nb, 0, (T *)nullptr, partials + nb + 32));
    CR_LAUNCH(ctx, k_scan_block<T>, (unsigned int)nb, kScanBlock, 0, in, out, n, (const T *)partial, inclusive,
              d_total);
    return CR_OK;
}

template <typename T>
int scan_impl(cr_ctx *ctx, const T *in, T *out, uint64_t n, int inclusive, T *d_total)
{
    if (n == 0) return CR_OK;
    void *p = nullptr;
    CR_TRY(cr_scratch(ctx, SCR_SCAN, (size_t)(scan_partials_size(n) + 32) * sizeof(T), &p));
    return scan_rec<T>(ctx, in, out, n, inclusive, d_total, reinterpret_cast<T *>(p));
}

// ---------------------------------------------------------- radix sort ----
// n_dev (optional): the item count in device memory; n is then an upper bound
// that sized the grid and the histogram, and tiles past the count stay empty.
// A count <= skip_le makes the pass a no-op (another path sorts those).
template <typename K>
__global__ void __launch_bounds__(kSortBlock) k_radix_upsweep(const K *__restrict__ keys, uint64_t n, int shift,
                                                              uint32_t ntiles, uint32_t *__restrict__ hist,
                                                              const unsigned long long *n_dev,
                                                              unsigned long long skip_le)
{
    if (n_dev && *n_dev <= skip_le) return;
    if (n_dev && *n_dev < n) n = *n_dev;
    __shared__ uint32_t cnt[256];
    cnt[threadIdx.x] = 0;
    __syncthreads();
    const uint64_t base = (uint64_t)blockIdx.x * kSortTile;
#pragma unroll
    for (int j = 0; j < kSortItems; ++j) {
        uint64_t i = base + (uint64_t)j * kSortBlock + threadIdx.x;
        if (i < n) atomicAdd(&cnt[(uint32_t)(keys[i] >> shift) & 0xffu], 1u);
    }
    __syncthreads();
    hist[(uint64_t)threadIdx.x * ntiles + blockIdx.x] = cnt[threadIdx.x];
}

template <typename K>
__global__ void __launch_bounds__(kSortBlock) k_radix_downsweep(const K *__restrict__ kin,
                                                                const uint32_t *__restrict__ vin,
                                                                K *__restrict__ kout, uint32_t *__restrict__ vout,
                                                                uint64_t n, int shift, uint32_t ntiles,
                                                                const uint32_t *__restrict__ offs,
                                                                const unsigned long long *n_dev,
                                                                unsigned long long skip_le)
{
    if (n_dev && *n_dev <= skip_le) return;
    if (n_dev && *n_dev < n) n = *n_dev;
    constexpr int kWarps = kSortBlock / 32;
    __shared__ uint32_t base_s[256];
    __shared__ uint32_t wcnt[kWarps][257];
    const uint32_t lane = cr_lane(), warp = threadIdx.x >> 5;
    base_s[threadIdx.x] = offs[(uint64_t)threadIdx.x * ntiles + blockIdx.x];
    uint32_t run = 0;  // items of digit threadIdx.x already placed in this tile
    const uint64_t tbase = (uint64_t)blockIdx.x * kSortTile;
    const uint32_t lt_mask = (1u << lane) - 1u;
    for (int j = 0; j < kSortItems; ++j) {
        for (int w = 0; w < kWarps; ++w) wcnt[w][threadIdx.x] = 0;
        if (threadIdx.x == 0)
            for (int w = 0; w < kWarps; ++w) wcnt[w][256] = 0;
        __syncthreads();
        const uint64_t i = tbase + (uint64_t)j * kSortBlock + threadIdx.x;
        const bool valid = i < n;
        K key = valid ? kin[i] : (K)0;
        uint32_t d = valid ? ((uint32_t)(key >> shift) & 0xffu) : 256u;
        uint32_t peers = __match_any_sync(0xffffffffu, d);
        uint32_t rank = __popc(peers & lt_mask);
        if (rank == 0) wcnt[warp][d] = __popc(peers);
        __syncthreads();
        {
            uint32_t dd = threadIdx.x;
            for (int w = 0; w < kWarps; ++w) {
                uint32_t c = wcnt[w][dd];
                wcnt[w][dd] = run;
                run += c;
            }
        }
        __syncthreads();
        if (valid) {
            uint32_t pos = base_s[d] + wcnt[warp][d] + rank;
            kout[pos] = key;
            if (vout) vout[pos] = vin ? vin[i] : (uint32_t)i;
        }
        __syncthreads();
    }
}

template <typename K>
int radix_impl(cr_ctx *ctx, const K *k_in, const uint32_t *v_in, uint64_t n, int bits, const K **k_out,
               const uint32_t **v_out, int kslot0, int kslot1)
{
    const int want_vals = v_out != nullptr;
    *k_out = k_in;
    if (v_out) *v_out = v_in;
    if (n == 0 || bits <= 0) return CR_OK;
    if (n >= (1ull << 32)) return cr_fail(ctx, CR_EINVAL, "radix sort: n >= 2^32");
    const uint32_t ntiles = (uint32_t)((n + kSortTile - 1) / kSortTile);
    void *kb0, *kb1, *vb0 = nullptr, *vb1 = nullptr, *hist;
    CR_TRY(cr_scratch(ctx, kslot0, n * sizeof(K), &kb0));
    CR_TRY(cr_scratch(ctx, kslot1, n * sizeof(K), &kb1));
    if (want_vals) {
        CR_TRY(cr_scratch(ctx, SCR_SORT_V0, n * sizeof(uint32_t), &vb0));
        CR_TRY(cr_scratch(ctx, SCR_SORT_V1, n * sizeof(uint32_t), &vb1));
    }
    CR_TRY(cr_scratch(ctx, SCR_SORT_HIST, (size_t)256 * ntiles * sizeof(uint32_t), &hist));
    const K *ksrc = k_in;
    const uint32_t *vsrc = v_in;
    int pass = 0;
    for (int shift = 0; shift < bits; shift += 8, ++pass) {
        K *kdst = reinterpret_cast<K *>((pass & 1) ? kb1 : kb0);
        uint32_t *vdst = want_vals ? reinterpret_cast<uint32_t *>((pass & 1) ? vb1 : vb0) : nullptr;
        CR_LAUNCH(ctx, k_radix_upsweep<K>, ntiles, kSortBlock, 0, ksrc, n, shift, ntiles, (uint32_t *)hist,
                  (const unsigned long long *)nullptr, 0ull);
        CR_TRY(scan_impl<uint32_t>(ctx, (const uint32_t *)hist, (uint32_t *)hist, (uint64_t)256 * ntiles, 0,
                                   (uint32_t *)nullptr));
        CR_LAUNCH(ctx, k_radix_downsweep<K>, ntiles, kSortBlock, 0, ksrc, vsrc, kdst, vdst, n, shift, ntiles,
                  (const uint32_t *)hist, (const unsigned long long *)nullptr, 0ull);
        ksrc = kdst;
        vsrc = vdst;
    }
    *k_out = ksrc;
    if (v_out) *v_out = vsrc;
    return CR_OK;
}

// (key, value) pairs ping-ponged between caller buffers 0 and 1, bits
// [0, bits) in 8-bit passes; the item count is read from n_dev (<= n_max).
// With iota the input values are not read: they are the items' positions.
template <typename K>
int radix_pairs_dev(cr_ctx *ctx, K *k0, uint32_t *v0, K *k1, uint32_t *v1, uint64_t n_max,
                    const unsigned long long *n_dev, unsigned long long skip_le, int bits, int iota, int *in1)
{
    *in1 = 0;
    if (n_max == 0 || bits <= 0) return CR_OK;
    if (n_max >= (1ull << 32)) return cr_fail(ctx, CR_EINVAL, "radix sort: n >= 2^32");
    const uint32_t ntiles = (uint32_t)((n_max + kSortTile - 1) / kSortTile);
    void *hist;
    CR_TRY(cr_scratch(ctx, SCR_SORT_HIST, (size_t)256 * ntiles * sizeof(uint32_t), &hist));
    int cur = 0;
    for (int shift = 0; shift < bits; shift += 8) {
        K *ks = cur ? k1 : k0, *kd = cur ? k0 : k1;
        const uint32_t *vs = (shift == 0 && iota) ? nullptr : (cur ? v1 : v0);
        uint32_t *vd = cur ? v0 : v1;
        CR_LAUNCH(ctx, k_radix_upsweep<K>, ntiles, kSortBlock, 0, (const K *)ks, n_max, shift, ntiles,
                  (uint32_t *)hist, n_dev, skip_le);
        CR_TRY(scan_impl<uint32_t>(ctx, (const uint32_t *)hist, (uint32_t *)hist, (uint64_t)256 * ntiles, 0,
                                   (uint32_t *)nullptr));
        CR_LAUNCH(ctx, k_radix_downsweep<K>, ntiles, kSortBlock, 0, (const K *)ks, vs, kd, vd, n_max, shift, ntiles,
                  (const uint32_t *)hist, n_dev, skip_le);
        cur ^= 1;
    }
    *in1 = cur;
    return CR_OK;
}

}  // namespace

int cr_radix_pairs_u64_dev(cr_ctx *ctx, unsigned long long *k0, uint32_t *v0, unsigned long long *k1, uint32_t *v1,
                           uint64_t n_max, const unsigned long long *n_dev, unsigned long long skip_le, int bits,
                           int iota, int *in1)
{
    return radix_pairs_dev<unsigned long long>(ctx, k0, v0, k1, v1, n_max, n_dev, skip_le, bits, iota, in1);
}

int cr_radix_pairs_u32_dev(cr_ctx *ctx, uint32_t *k0, uint32_t *v0, uint32_t *k1, uint32_t *v1, uint64_t n_max,
                           const unsigned long long *n_dev, unsigned long long skip_le, int bits, int iota,
                           int *in1)
{
    return radix_pairs_dev<uint32_t>(ctx, k0, v0, k1, v1, n_max, n_dev, skip_le, bits, iota, in1);
}

int cr_scan_u32(cr_ctx *ctx, const uint32_t *in, uint32_t *out, uint64_t n, uint32_t *d_total)
{
    return scan_impl<uint32_t>(ctx, in, out, n, 0, d_total);
}

int cr_scan_u64_inclusive(cr_ctx *ctx, const unsigned long long *in, unsigned long long *out, uint64_t n)
{
    return scan_impl<unsigned long long>(ctx, in, out, n, 1, (unsigned long long *)nullptr);
}

int cr_radix_sort_u64(cr_ctx *ctx, const unsigned long long *k_in, const uint32_t *v_in, uint64_t n, int bits,
                      const unsigned long long **k_out, const uint32_t **v_out)
{
    return radix_impl<unsigned long long>(ctx, k_in, v_in, n, bits, k_out, v_out, SCR_SORT_K0, SCR_SORT_K1);
}

int cr_radix_sort_u32(cr_ctx *ctx, const uint32_t *k_in, const uint32_t *v_in, uint64_t n, int bits,
                      const uint32_t **k_out, const uint32_t **v_out)
{
    return radix_impl<uint32_t>(ctx, k_in, v_in, n, bits, k_out, v_out, SCR_SORT_K0, SCR_SORT_K1);
}
