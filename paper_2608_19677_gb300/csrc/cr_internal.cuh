// Internal declarations of the CUDA library (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdint.h>
#include <stdio.h>

#include <nvtx3/nvToolsExt.h>

#include "cacheroute.h"

// NVTX range over one C ABI call (free unless a profiler is attached).
struct cr_nvtx_range {
    explicit cr_nvtx_range(const char *name) { nvtxRangePushA(name); }
    ~cr_nvtx_range() { nvtxRangePop(); }
};

// ---- device error flags (a bitmask in device memory, read by cr_sync) ------
#define CR_FLAG_OVERFLOW 1u  // a load reached 2^47, or a stamp counter overflowed
#define CR_FLAG_BADDEST 2u   // a destination index >= R reached the replay
#define CR_FLAG_TIMEOUT 4u   // a bounded wait gave up
#define CR_FLAG_BADSIZE 8u   // token-weighted replay: a key came back with another prefix length
#define CR_FLAG_INTERNAL 16u // a kernel found its own state inconsistent and skipped the access
#define CR_FLAG_BOUNDS 32u   // debug build: an index outside its array was skipped

// Debug build (compiled with -DCR_DEBUG_CHECKS, see buildlib.py): data-dependent
// indices are checked before use; a failing check raises CR_FLAG_BOUNDS in the
// status word and the caller skips the access.  In the normal build the check
// is the constant true and costs nothing.
#ifdef CR_DEBUG_CHECKS
#define CR_DCHECK(ok, status) ((ok) || (atomicOr((status), CR_FLAG_BOUNDS), false))
#else
#define CR_DCHECK(ok, status) (true)
#endif

// ---- scratch slots owned by the context ------------------------------------
enum cr_scratch_slot {
    SCR_SORT_K0 = 0,   // radix-sort keys (ping)
    SCR_SORT_K1,       // radix-sort keys (pong)
    SCR_SORT_V0,       // radix-sort values (ping)
    SCR_SORT_V1,       // radix-sort values (pong)
    SCR_SORT_HIST,     // per-tile digit counts / offsets
    SCR_SCAN,          // block partials of the device-wide scan
    SCR_PLAN_A,        // plan-build temporaries
    SCR_PLAN_B,
    SCR_PLAN_C,
    SCR_REPLAY_IDX,    // partitioned request indices
    SCR_REPLAY_START,  // per-stream start offsets
    SCR_REPLAY_REC,    // request indices in stream order
    SCR_REPLAY_RECS,   // (key, prefix, suffix) record of each request
    SCR_REPLAY_CHUNK,  // per-stream chunk counts -> offsets, and their total
    SCR_ROUTE_DESC,    // per-replica route descriptors
    SCR_DIFF,          // plan-difference counters
    SCR_NUM
};

// ---- per-launch timing of selected kernels (cr_profile_enable) ---------------
struct cr_prof {
    uint32_t cap, used;  // event pairs available / recorded
    cudaEvent_t *ev;     // [2 cap]: start, end of each timed launch
    uint8_t *tag;        // [cap]: CR_PROF_* of each
};

struct cr_ctx {
    cr_prof prof;
    cr_replay_input *replay_in;  // partition of cr_shadow_replay (library-owned)
    int device;
    int num_sms;
    cudaStream_t stream;
    uint32_t *d_status;          // CR_FLAG_* bits
    uint64_t launches;
    void *scratch[SCR_NUM];
    size_t scratch_bytes[SCR_NUM];
    char msg[320];
    // routing split over two streams (cr_set_resolve_stream): the load-dependent
    // resolution runs on resolve_stream, after ev_cand; ev_resolve marks its end
    cudaStream_t resolve_stream;     // NULL: everything on `stream`
    cudaEvent_t ev_cand, ev_resolve;
    int resolve_recorded;            // ev_resolve has been recorded at least once
};

// Plan: every array lives on the device; capacities are host-side upper bounds.
struct cr_plan_info_dev {
    unsigned long long n, U;
    unsigned long long S;        // admission candidates ordered by (count desc, key asc): order[0..S)
    unsigned long long n_adm, sum_k, cold, max_k, special;
    unsigned long long adm_lam;  // requests of the admitted keys
};

struct cr_table_slot {               // 16 bytes: one sector-aligned probe
    unsigned long long key;
    uint32_t koff;                   // 0xffffffff = empty
    uint16_t k;
    uint16_t m0;                     // first member (the destination when k == 1)
};

struct cr_plan {
    uint32_t R, W;
    uint64_t cap_n;                  // capacity for histogram arrays (>= n)
    uint64_t cap_adm;                // capacity for admitted arrays (>= min(n, C))
    uint64_t cap_mem;                // capacity for member arrays (>= C)
    uint64_t table_slots;            // power of two
    uint64_t n;                      // requests of the last build (host copy)
    unsigned long long *d_ukey, *d_ucnt;
    unsigned long long *d_adm_key, *d_adm_cnt;
    uint32_t *d_adm_k, *d_koff;
    uint16_t *d_members;
    unsigned long long *d_jobs, *d_load;
    cr_table_slot *d_table;
    cr_plan_info_dev *d_info;
    uint64_t qnum, qden;             // q_cap = qnum / qden of the last build
    uint32_t variant;                // CR_VARIANT_* of the last build
    int built;
};

// Ring of the bounded-load policy: R*V points ascending, their owners, and a
// directory dir[t] = first ring index whose point is >= t << (64 - dbits).
struct cr_ring {
    uint32_t R, V, dbits;
    uint64_t M;
    unsigned long long *d_point;
    uint16_t *d_owner;
    uint32_t *d_dir;
};

struct cr_replay {
    uint32_t n_rep, R, n_caps, cmax;  // cmax: largest capacity, or CR_MAX_CAP entries in token mode
    int tokens;                       // capacities in prefix tokens (one state buffer, d_size used)
    uint32_t *d_size[2];             // token mode: [stream][cmax] tokens of the listed keys up to each one
    uint32_t caps[CR_MAX_CAPS];
    uint64_t n_streams;              // n_rep * R
    unsigned long long *d_keys[2];   // [stream][cmax], most recent first; double-buffered
    uint32_t *d_fill[2];             // [stream]
    int cur;                         // buffer holding the current state
};

// ---- host helpers (cr_api.cu) ----------------------------------------------
int cr_fail(cr_ctx *ctx, int code, const char *fmt, ...);
int cr_scratch(cr_ctx *ctx, int slot, size_t bytes, void **out);
int cr_check_launch(cr_ctx *ctx, const char *what);

#define CR_TRY(expr)                 \
    do {                             \
        int _st = (expr);            \
        if (_st != CR_OK) return _st; \
    } while (0)

#define CR_CUDA(ctx, expr)                                                              \
    do {                                                                                \
        cudaError_t _e = (expr);                                                        \
        if (_e != cudaSuccess)                                                          \
            return cr_fail((ctx), CR_ECUDA, "%s: %s", #expr, cudaGetErrorString(_e));   \
    } while (0)

// Launch on the context's stream and account for it.
#define CR_LAUNCH(ctx, kern, grid, block, smem, ...)                       \
    do {                                                                   \
        kern<<<(grid), (block), (smem), (ctx)->stream>>>(__VA_ARGS__);     \
        (ctx)->launches++;                                                 \
        CR_TRY(cr_check_launch((ctx), #kern));                             \
    } while (0)

// Launch on a given stream of the context (e.g. its resolve stream) and account for it.
#define CR_LAUNCH_ON(ctx, st, kern, grid, block, smem, ...)                \
    do {                                                                   \
        kern<<<(grid), (block), (smem), (st)>>>(__VA_ARGS__);              \
        (ctx)->launches++;                                                 \
        CR_TRY(cr_check_launch((ctx), #kern));                             \
    } while (0)

// Bracket work enqueued on `st` with a timed event pair when profiling is on;
// returns the pair's index (or -1) for cr_prof_end.
static inline int cr_prof_begin(cr_ctx *ctx, cudaStream_t st, int tag)
{
    cr_prof &P = ctx->prof;
    if (!P.ev || P.used >= P.cap) return -1;
    const uint32_t i = P.used++;
    P.tag[i] = (uint8_t)tag;
    cudaEventRecord(P.ev[2 * i], st);
    return (int)i;
}
static inline void cr_prof_end(cr_ctx *ctx, cudaStream_t st, int i)
{
    if (i >= 0) cudaEventRecord(ctx->prof.ev[2 * i + 1], st);
}

static inline unsigned int cr_blocks(uint64_t work, unsigned int per_block, unsigned int cap)
{
    uint64_t b = (work + per_block - 1) / per_block;
    if (b < 1) b = 1;
    if (b > cap) b = cap;
    return (unsigned int)b;
}

// ---- sort and scan primitives (cr_sort.cu) -----------------------------------
// Stable LSD radix sort of keys (and optional u32 values) on bits [0, bits).
// Input in (k_in, v_in); the sorted result is returned through *k_out/*v_out,
// which point at either the input buffers or the context's ping-pong scratch.
int cr_radix_sort_u64(cr_ctx *ctx, const unsigned long long *k_in, const uint32_t *v_in, uint64_t n,
                      int bits, const unsigned long long **k_out, const uint32_t **v_out);
int cr_radix_sort_u32(cr_ctx *ctx, const uint32_t *k_in, const uint32_t *v_in, uint64_t n, int bits,
                      const uint32_t **k_out, const uint32_t **v_out);
// Exclusive scan of u32 counts into u32 offsets (in place allowed); total to *d_total if non-null.
// Radix sort of (key, value) pairs by bits [0, bits), ping-ponging between the
// caller's buffers 0 and 1; the item count is read from n_dev (grid sized by
// n_max); a count <= skip_le leaves everything untouched.  With iota the
// values start as the items' positions.  *in1 tells whether the result ended
// in buffers 1.
int cr_radix_pairs_u64_dev(cr_ctx *ctx, unsigned long long *k0, uint32_t *v0, unsigned long long *k1, uint32_t *v1,
                           uint64_t n_max, const unsigned long long *n_dev, unsigned long long skip_le, int bits,
                           int iota, int *in1);
int cr_radix_pairs_u32_dev(cr_ctx *ctx, uint32_t *k0, uint32_t *v0, uint32_t *k1, uint32_t *v1, uint64_t n_max,
                           const unsigned long long *n_dev, unsigned long long skip_le, int bits, int iota,
                           int *in1);
int cr_scan_u32(cr_ctx *ctx, const uint32_t *in, uint32_t *out, uint64_t n, uint32_t *d_total);
// Inclusive scan of u64 values.
int cr_scan_u64_inclusive(cr_ctx *ctx, const unsigned long long *in, unsigned long long *out, uint64_t n);
